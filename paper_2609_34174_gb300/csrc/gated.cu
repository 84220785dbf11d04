// gated.cu -- the scans with the paper's general gates (Sec. 3 "Observation",
// Eq. 2): per-token step sizes eta_t and retention alpha_t with decay centred at
// the slow weights,
//
//     W_{t+1} = W0 + alpha_t (W_t - W0) - eta_t ghat_t x_t^T,       W at t = 0 is W0,
//
// read before each write: y_t = W_t x_t (Eq. 3), gin_t = W_t^T gout_t (Eq. 4).
// alpha_t = 0 resets the fast weights to W0 (a document boundary).
//
// Two kernels:
//   prescale_kernel  eta_t only (alpha = 1): the writes eta_t ghat_t x_t^T are the
//                    plain writes of ghat'_t = eta_t ghat_t, so the chunked kernels
//                    run on ghat' with eta = 1.  One elementwise pass into the
//                    workspace (rounded to the input dtype, like ghat itself).
//   chunk_decay_kernel  with alpha_t, bf16 64 x 64 maps: the recurrence in chunks
//                    of 64 tokens, the within-chunk decays as plain products of
//                    the alphas, contractions on bf16 mma.sync fragments.
//   serial_kernel    with alpha_t, any other shape: the recurrence token by token,
//                    exactly as Eq. 2 states it.  Each CTA holds a 64-wide slice of
//                    W - W0 and of W0 for one unit; the forward slices W by rows
//                    (outputs are rows), the costate by columns.
#include <cuda_bf16.h>

#include "scan_common.cuh"

namespace gl {
namespace gated {

constexpr int kTile = 64;       // output indices per CTA
constexpr int kThreads = 256;   // 4 threads per output index

template <bool BF16>
__device__ __forceinline__ float ld(const void* p, long long i) {
    if constexpr (BF16)
        return __bfloat162float(static_cast<const __nv_bfloat16*>(p)[i]);
    else
        return static_cast<const float*>(p)[i];
}

template <bool BF16>
__device__ __forceinline__ void st(void* p, long long i, float v) {
    if constexpr (BF16)
        static_cast<__nv_bfloat16*>(p)[i] = __float2bfloat16_rn(v);
    else
        static_cast<float*>(p)[i] = v;
}

constexpr int kFlatThreads = 256;

// The same scaling for a contiguous input: piece v (16 bytes) belongs to token
// v / vpr at the same offset in and out.  Each thread keeps four pieces in flight.
template <bool BF16>
__global__ void __launch_bounds__(kFlatThreads)
    prescale_flat_kernel(const void* __restrict__ g, const float* __restrict__ eta,
                         void* __restrict__ out, int n, int vpr) {
    const uint4* in = static_cast<const uint4*>(g);
    uint4* o = static_cast<uint4*>(out);
    const int stride = gridDim.x * kFlatThreads;
    for (int v0 = blockIdx.x * kFlatThreads + threadIdx.x; v0 < n; v0 += 4 * stride) {
        uint4 x[4];
        float e[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const int v = v0 + k * stride;
            if (v < n) {
                x[k] = __ldcs(in + v);
                e[k] = __ldg(eta + v / vpr);
            }
        }
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const int v = v0 + k * stride;
            if (v >= n) continue;
            uint4 y;
            if constexpr (BF16) {
                const __nv_bfloat162* pi = reinterpret_cast<const __nv_bfloat162*>(&x[k]);
                __nv_bfloat162* po = reinterpret_cast<__nv_bfloat162*>(&y);
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const float2 f = __bfloat1622float2(pi[i]);
                    po[i] = __floats2bfloat162_rn(e[k] * f.x, e[k] * f.y);
                }
            } else {
                y = make_uint4(__float_as_uint(e[k] * __uint_as_float(x[k].x)),
                               __float_as_uint(e[k] * __uint_as_float(x[k].y)),
                               __float_as_uint(e[k] * __uint_as_float(x[k].z)),
                               __float_as_uint(e[k] * __uint_as_float(x[k].w)));
            }
            o[v] = y;
        }
    }
}

// ghat'[l,b,t,h,:] = eta_t[l,b,t,h] * ghat[l,b,t,h,:], written contiguous.  One
// thread per 16-byte piece of a token row (w a multiple of 16 bytes / element).
template <bool BF16>
__global__ void prescale_kernel(const void* __restrict__ g, TokStr gs, const float* __restrict__ eta,
                                void* __restrict__ out, int L, int B, int T, int H, int w) {
    constexpr int kPer = BF16 ? 8 : 4;  // elements per 16 bytes
    const int vpr = w / kPer;           // pieces per token row
    const long long tokens = (long long)L * B * T * H;
    const long long n = tokens * vpr;
    for (long long v = (long long)blockIdx.x * blockDim.x + threadIdx.x; v < n;
         v += (long long)gridDim.x * blockDim.x) {
        const long long tok = v / vpr;
        const int f = (int)(v - tok * vpr) * kPer;
        const int h = (int)(tok % H);
        const long long r = tok / H;
        const int t = (int)(r % T);
        const long long r2 = r / T;
        const int b = (int)(r2 % B);
        const int l = (int)(r2 / B);
        const long long src = (long long)l * gs.s[0] + (long long)b * gs.s[1] + (long long)t * gs.s[2] +
                              (long long)h * gs.s[3] + f;
        const float e = eta[tok];
        uint4 in;
        if constexpr (BF16)
            in = *reinterpret_cast<const uint4*>(static_cast<const __nv_bfloat16*>(g) + src);
        else
            in = *reinterpret_cast<const uint4*>(static_cast<const float*>(g) + src);
        uint4 o;
        if constexpr (BF16) {
            const __nv_bfloat162* pi = reinterpret_cast<const __nv_bfloat162*>(&in);
            __nv_bfloat162* po = reinterpret_cast<__nv_bfloat162*>(&o);
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const float2 x = __bfloat1622float2(pi[k]);
                po[k] = __floats2bfloat162_rn(e * x.x, e * x.y);
            }
            *reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(out) + tok * w + f) = o;
        } else {
            const float* pi = reinterpret_cast<const float*>(&in);
            float* po = reinterpret_cast<float*>(&o);
#pragma unroll
            for (int k = 0; k < 4; ++k) po[k] = e * pi[k];
            *reinterpret_cast<uint4*>(static_cast<float*>(out) + tok * w + f) = o;
        }
    }
}

// One CTA: unit (l, b, h) and a tile of 64 output indices.
//   forward  (COSTATE = false): outputs are rows m of W [m][d]; q = x (length d),
//            a = ghat (row-indexed), bvec = x (column-indexed)
//   costate  (COSTATE = true):  outputs are columns d of W; q = g_out (length m),
//            a = x (column-indexed), bvec = ghat (row-indexed)
// Held per CTA (fp32): W0t[i][j] = W0 entry and Dt[i][j] = (W_t - W0) entry for
// output i of the tile and input j (J = d forward, m costate).  Thread 4i+p owns
// entries (i, j) with j = p mod 4: it both reads and writes exactly those, so a
// token needs one barrier (its staged vectors, double-buffered).  The next
// token's vectors are loaded into registers while this token is computed.
template <bool COSTATE, bool BF16>
__global__ void __launch_bounds__(kThreads)
    serial_kernel(GatedParams p) {
    extern __shared__ float sm[];
    const int J = COSTATE ? p.dout : p.din;   // inputs of the read (at most kThreads)
    const int NO = COSTATE ? p.din : p.dout;  // outputs of the read
    // rows padded to J + 4 floats: the 8 rows x 4 parts a warp touches then fall in
    // 32 distinct banks (row stride = 4 banks)
    const int JS = J + 4;
    float* W0t = sm;                          // [64][JS]
    float* Dt = W0t + kTile * JS;             // [64][JS]
    float* stage = Dt + kTile * JS;           // 2 x { q [J], b [J], a [64], eta, alpha }
    const int sstride = 2 * J + kTile + 2;

    const int tiles = (NO + kTile - 1) / kTile;
    const int tile = blockIdx.x % tiles;
    const int unit = blockIdx.x / tiles;
    const int h = unit % p.H;
    const int l = unit / (p.H * p.B);
    const int b = (unit / p.H) % p.B;
    const int o0 = tile * kTile;
    const float* w0 = p.W0 + (size_t)(l * p.H + h) * p.din * p.dout;  // [dout][din]

    for (int e = threadIdx.x; e < kTile * J; e += kThreads) {
        const int i = e / J, j = e - i * J;
        const int o = o0 + i;
        float w = 0.0f;
        if (o < NO) w = COSTATE ? w0[(size_t)j * p.din + o] : w0[(size_t)o * p.din + j];
        W0t[i * JS + j] = w;
        Dt[i * JS + j] = 0.0f;
    }
    // what this thread stages: q[tid], b[tid] (tid < J), a[tid] (tid < 64), gates (tid 0)
    const int tid = threadIdx.x;
    auto fetch = [&](int t, float& qv, float& bv, float& av, float& ev, float& alv) {
        const long long xo = tok_off(p.x_s, l, b, t, h);
        const long long go = tok_off(p.g_s, l, b, t, h);
        const long long qo = tok_off(p.q_s, l, b, t, h);
        if (tid < J) {
            qv = ld<BF16>(p.q, qo + tid);
            bv = COSTATE ? ld<BF16>(p.g, go + tid) : ld<BF16>(p.x, xo + tid);
        }
        if (tid < kTile) {
            const int o = o0 + tid;
            av = o < NO ? (COSTATE ? ld<BF16>(p.x, xo + o) : ld<BF16>(p.g, go + o)) : 0.0f;
        }
        if (tid == 0) {
            const long long tok = ((long long)l * p.B + b) * p.T * p.H + (long long)t * p.H + h;
            ev = p.eta[tok];
            alv = p.alpha ? p.alpha[tok] : 1.0f;
        }
    };
    auto put = [&](int buf, float qv, float bv, float av, float ev, float alv) {
        float* s = stage + buf * sstride;
        if (tid < J) {
            s[tid] = qv;
            s[J + tid] = bv;
        }
        if (tid < kTile) s[2 * J + tid] = av;
        if (tid == 0) {
            s[2 * J + kTile] = ev;
            s[2 * J + kTile + 1] = alv;
        }
    };
    // register ring of the next kAhead tokens' vectors (slots indexed by t mod kAhead)
    constexpr int kAhead = 4;
    float qv[kAhead], bv[kAhead], av[kAhead], ev[kAhead], alv[kAhead];
#pragma unroll
    for (int u = 0; u < kAhead; ++u) {
        qv[u] = bv[u] = av[u] = ev[u] = 0.0f;
        alv[u] = 1.0f;
        if (u < p.T) fetch(u, qv[u], bv[u], av[u], ev[u], alv[u]);
    }
    if (p.T > 0) put(0, qv[0], bv[0], av[0], ev[0], alv[0]);
    const int i_own = threadIdx.x >> 2;  // output index of this thread's group of 4
    const int part = threadIdx.x & 3;
    const int o = o0 + i_own;
    float* w_row = W0t + i_own * JS;
    float* d_row = Dt + i_own * JS;
    for (int t0 = 0; t0 < p.T; t0 += kAhead) {
#pragma unroll
        for (int u = 0; u < kAhead; ++u) {
            const int t = t0 + u;
            if (t >= p.T) break;
            __syncthreads();  // token t staged; token t-1's buffer no longer read
            const float* s = stage + (t & 1) * sstride;
            const float* q = s;
            const float* bw = s + J;
            const float a_i = s[2 * J + i_own];
            const float eta = s[2 * J + kTile], alpha = s[2 * J + kTile + 1];
            // read before write: out_i = sum_j (W0 + D)[i][j] q_j, then
            // write D[i][j] = alpha D[i][j] - eta a_i b_j on the same entries
            float acc = 0.0f;
            for (int j = part; j < J; j += 4) {
                const float dv = d_row[j];
                acc += (w_row[j] + dv) * q[j];
                d_row[j] = alpha * dv - eta * a_i * bw[j];
            }
            acc += __shfl_xor_sync(0xffffffffu, acc, 1);
            acc += __shfl_xor_sync(0xffffffffu, acc, 2);
            if (part == 0 && o < NO) {
                const EpiParams& e = p.epi;
                const long long oo = tok_off(e.out_str, l, b, t, h) + o;
                float v = acc;
                if (e.zin) v *= act_df(e.act, ld<BF16>(e.zin, tok_off(e.z_str, l, b, t, h) + o));
                st<BF16>(e.out, oo, v);
                if (e.out2) st<BF16>(e.out2, tok_off(e.out2_str, l, b, t, h) + o, act_f(e.act, acc));
            }
            // stage token t+1 (fetched kAhead-1 tokens ago), then refill this slot
            const int un = (u + 1) % kAhead;
            if (t + 1 < p.T) put((t + 1) & 1, qv[un], bv[un], av[un], ev[un], alv[un]);
            if (t + kAhead < p.T) fetch(t + kAhead, qv[u], bv[u], av[u], ev[u], alv[u]);
        }
    }
}

// The same recurrence for bf16 reads of at most kRegJ inputs, with the state in
// registers: thread 4i+p owns the entries (i, j) of output i for the contiguous
// inputs j in [16p, 16p + 16) and holds W0 and D for them in registers.  The
// per-token vectors (q, b, the tile's a, eta_t, alpha_t) arrive by cp.async in
// blocks of kBlk tokens, one block ahead, so the CTA synchronises once per block
// instead of once per token, and no state ever goes through shared memory.
constexpr int kRegJ = 64;
constexpr int kBlk = 16;
constexpr int kTokBytes = 3 * 128 + 16;  // q, b, a (64 bf16 each), eta and alpha (+ pad)

__device__ __forceinline__ void cpa16(uint32_t dst, const void* src, bool valid) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src),
                 "r"(valid ? 16 : 0)
                 : "memory");
}
__device__ __forceinline__ void cpa4(uint32_t dst, const void* src, bool valid) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"(dst), "l"(src),
                 "r"(valid ? 4 : 0)
                 : "memory");
}
__device__ __forceinline__ void cpa_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cpa_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

template <bool COSTATE>
__global__ void __launch_bounds__(kThreads)
    serial_reg_kernel(GatedParams p) {
    __shared__ __align__(16) unsigned char buf[2][kBlk * kTokBytes];
    constexpr int JP = kRegJ / 4;            // entries per thread
    const int J = COSTATE ? p.dout : p.din;  // a multiple of 16, at most kRegJ
    const int NO = COSTATE ? p.din : p.dout;
    const int tiles = (NO + kTile - 1) / kTile;
    const int tile = blockIdx.x % tiles;
    const int unit = blockIdx.x / tiles;
    const int h = unit % p.H;
    const int l = unit / (p.H * p.B);
    const int b = (unit / p.H) % p.B;
    const int o0 = tile * kTile;
    const float* w0 = p.W0 + (size_t)(l * p.H + h) * p.din * p.dout;  // [dout][din]
    const int tid = threadIdx.x;
    const int i_own = tid >> 2, part = tid & 3;
    const int o = o0 + i_own;
    const int j0 = part * JP;
    float w[JP], d[JP];
#pragma unroll
    for (int k = 0; k < JP; ++k) {
        const int j = j0 + k;
        w[k] = (o < NO && j < J) ? (COSTATE ? w0[(size_t)j * p.din + o] : w0[(size_t)o * p.din + j])
                                 : 0.0f;
        d[k] = 0.0f;
    }
    // token-0 positions of the vectors and their steps per token
    const __nv_bfloat16* X = static_cast<const __nv_bfloat16*>(p.x) + tok_off(p.x_s, l, b, 0, h);
    const __nv_bfloat16* G = static_cast<const __nv_bfloat16*>(p.g) + tok_off(p.g_s, l, b, 0, h);
    const __nv_bfloat16* Qb = static_cast<const __nv_bfloat16*>(p.q) + tok_off(p.q_s, l, b, 0, h);
    const __nv_bfloat16* Bb = COSTATE ? G : X;
    const __nv_bfloat16* Ab = (COSTATE ? X : G) + o0;
    const long long qst = p.q_s[2], bst = COSTATE ? p.g_s[2] : p.x_s[2],
                    ast = COSTATE ? p.x_s[2] : p.g_s[2];
    const long long gate0 = ((long long)l * p.B + b) * p.T * p.H + h;
    // stage tokens [kBlk k, kBlk k + kBlk) into buffer k & 1: 24 pieces of 16 bytes per
    // token (q, b, a: 8 each) plus the two gates; zeros past T, J or the tile
    auto stage = [&](int k) {
        const uint32_t base = (uint32_t)__cvta_generic_to_shared(buf[k & 1]);
        for (int pc = tid; pc < kBlk * 24; pc += kThreads) {
            const int u = pc / 24, kind = pc - u * 24, t = k * kBlk + u;
            const int sub = kind & 7;
            const uint32_t dst = base + u * kTokBytes + kind * 16;
            // a zero-filled piece reads nothing; it is given a valid address all the same
            if (kind < 8) {
                const bool ok = t < p.T && sub * 8 < J;
                cpa16(dst, ok ? Qb + (long long)t * qst + sub * 8 : Qb, ok);
            } else if (kind < 16) {
                const bool ok = t < p.T && sub * 8 < J;
                cpa16(dst, ok ? Bb + (long long)t * bst + sub * 8 : Qb, ok);
            } else {
                const bool ok = t < p.T && o0 + sub * 8 < NO;
                cpa16(dst, ok ? Ab + (long long)t * ast + sub * 8 : Qb, ok);
            }
        }
        if (tid < 2 * kBlk) {
            const int u = tid >> 1, t = k * kBlk + u;
            const float* src = (tid & 1) ? p.alpha : p.eta;
            const bool ok = t < p.T && src != nullptr;
            cpa4(base + u * kTokBytes + 384 + (tid & 1) * 4, ok ? src + gate0 + (long long)t * p.H : p.eta,
                 ok);
        }
        cpa_commit();
    };
    const int n_blk = (p.T + kBlk - 1) / kBlk;
    if (n_blk > 0) stage(0);
    for (int k = 0; k < n_blk; ++k) {
        if (k + 1 < n_blk) {
            stage(k + 1);
            cpa_wait<1>();
        } else {
            cpa_wait<0>();
        }
        __syncthreads();  // block k staged by every thread
        const unsigned char* bk = buf[k & 1];
        const int nt = min(kBlk, p.T - k * kBlk);
        for (int u = 0; u < nt; ++u) {
            const int t = k * kBlk + u;
            const unsigned char* tk = bk + u * kTokBytes;
            const uint4 q0 = *reinterpret_cast<const uint4*>(tk + j0 * 2);
            const uint4 q1 = *reinterpret_cast<const uint4*>(tk + j0 * 2 + 16);
            const uint4 b0 = *reinterpret_cast<const uint4*>(tk + 128 + j0 * 2);
            const uint4 b1 = *reinterpret_cast<const uint4*>(tk + 128 + j0 * 2 + 16);
            const float a_i = __bfloat162float(reinterpret_cast<const __nv_bfloat16*>(tk + 256)[i_own]);
            const float eta = *reinterpret_cast<const float*>(tk + 384);
            const float alpha = p.alpha ? *reinterpret_cast<const float*>(tk + 388) : 1.0f;
            const float ea = eta * a_i;
            const uint32_t qw[8] = {q0.x, q0.y, q0.z, q0.w, q1.x, q1.y, q1.z, q1.w};
            const uint32_t bw[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
            // read before write: out_i = sum_j (W0 + D)[i][j] q_j, then
            // D[i][j] = alpha D[i][j] - eta a_i b_j on the same entries
            float ac[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
            for (int k2 = 0; k2 < JP / 2; ++k2) {
                const float2 qf = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&qw[k2]));
                const float2 bf = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&bw[k2]));
                const int kk = 2 * k2;
                ac[kk & 3] = fmaf(w[kk] + d[kk], qf.x, ac[kk & 3]);
                ac[(kk + 1) & 3] = fmaf(w[kk + 1] + d[kk + 1], qf.y, ac[(kk + 1) & 3]);
                d[kk] = fmaf(alpha, d[kk], -ea * bf.x);
                d[kk + 1] = fmaf(alpha, d[kk + 1], -ea * bf.y);
            }
            float acc = (ac[0] + ac[1]) + (ac[2] + ac[3]);
            acc += __shfl_xor_sync(0xffffffffu, acc, 1);
            acc += __shfl_xor_sync(0xffffffffu, acc, 2);
            if (part == 0 && o < NO) {
                const EpiParams& e = p.epi;
                const long long oo = tok_off(e.out_str, l, b, t, h) + o;
                float v = acc;
                if (e.zin) v *= act_df(e.act, ld<true>(e.zin, tok_off(e.z_str, l, b, t, h) + o));
                st<true>(e.out, oo, v);
                if (e.out2) st<true>(e.out2, tok_off(e.out2_str, l, b, t, h) + o, act_f(e.act, acc));
            }
        }
        __syncthreads();  // block k read: its buffer may take block k + 2
    }
}

// ---------------------------------------------------------------------------
// Chunked retention scan for bf16 maps of 64 x 64.  In the orientation shared by
// both reads (o_t = (B0 + S_t) q_t with writes S <- alpha_s S - eta_s v_s k_s^T):
//   forward  q = k = x, v = ghat, B0 = W0,   S = W - W0
//   costate  q = gout, k = ghat, v = x, B0 = W0^T, S = (W - W0)^T
// Eq. 2 unrolled over a chunk of kC tokens from the state S at its first token:
//
//   o_t = B0 q_t + a_t S q_t - sum_{s<t} E_ts (k_s . q_t) v_s
//   S'  = a_end S - sum_s w_s v_s k_s^T
//
// with a_t = prod_{r<t} alpha_r, E_ts = eta_s prod_{s<r<t} alpha_r, w_s = eta_s
// prod_{r>s} alpha_r and a_end the product of all the chunk's alphas (indices
// local to the chunk; tokens past T carry alpha = 1, eta = 0).  The decays are
// products of alphas, never ratios, so a reset (alpha = 0) and underflow give
// exact zeros.  They are assembled from 8-token pieces: sig_s (alphas after s to
// the end of its piece), pi_t (alphas from the start of t's piece up to t) and
// the piece products tp_j.
//
// One CTA per unit walks its chunks in order.  Warp w reads tokens [16w, 16w+16)
// of the chunk and owns rows [16w, 16w+16) of S, which stay in fp32 accumulator
// registers from chunk to chunk; a bf16 copy in shared memory is the B operand of
// the next chunk's read.  Tiles are 64 rows of 128 bytes, 16-byte pieces swizzled
// by the row (piece ^ (row & 7)) so that every ldmatrix phase is conflict free.
namespace cdec {

constexpr int kC = 64;                 // tokens per chunk
constexpr int kThr = 128;              // 4 warps
constexpr int kTileB = kC * 64 * 2;    // one bf16 tile [64][64]

template <bool COSTATE>
__host__ __device__ constexpr int buf_bytes() {            // q, v (, k) tiles and alpha, eta of one chunk
    return (COSTATE ? 3 : 2) * kTileB + 2 * kC * 4;
}
template <bool COSTATE>
__host__ __device__ constexpr size_t smem_bytes() {        // B0, S copy, two chunk buffers, decay tables
    return 2 * kTileB + 2 * buf_bytes<COSTATE>() + (2 * kC + 8) * 4;
}

__device__ __forceinline__ uint32_t swz(int row, int piece) {
    return (uint32_t)(row * 128 + ((piece ^ (row & 7)) << 4));
}
// The fragment loads read shared memory (memory clobber: they stay between the
// barriers and stores around them); the MMAs are pure register operations, free
// to be scheduled between the loads.
__device__ __forceinline__ void ldsm4(uint32_t a, uint32_t (&r)[4]) {
    asm("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
        : "r"(a)
        : "memory");
}
__device__ __forceinline__ void ldsm4t(uint32_t a, uint32_t (&r)[4]) {
    asm("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
        : "r"(a)
        : "memory");
}
// d += a b: a 16 x 16 (row), b 16 x 8 (col), bf16 in, fp32 accumulate
__device__ __forceinline__ void mma(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
        "{%8,%9}, {%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t pack(float lo, float hi) {
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&v);
}
__device__ __forceinline__ uint32_t scale2(uint32_t u, float a, float b) {
    const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u));
    return pack(f.x * a, f.y * b);
}
// B fragments of two 8-column tiles [n0, n0+16) for the k-step [k0, k0+16):
// from a tile stored [n][k] (k contiguous) ...
__device__ __forceinline__ void ld_b_nk(uint32_t tile, int n0, int k0, int lane, uint32_t (&r)[4]) {
    ldsm4(tile + swz(n0 + (lane & 7) + ((lane >> 4) << 3), (k0 >> 3) + ((lane >> 3) & 1)), r);
}
// ... or stored [k][n] (n contiguous)
__device__ __forceinline__ void ld_b_kn(uint32_t tile, int n0, int k0, int lane, uint32_t (&r)[4]) {
    ldsm4t(tile + swz(k0 + (lane & 7) + (((lane >> 3) & 1) << 3), (n0 >> 3) + (lane >> 4)), r);
}

template <bool COSTATE>
__global__ void __launch_bounds__(kThr, 3) chunk_decay_kernel(GatedParams p) {
    extern __shared__ __align__(128) unsigned char smc[];
    constexpr int kBufB = buf_bytes<COSTATE>();
    constexpr int kGateOff = (COSTATE ? 3 : 2) * kTileB;
    unsigned char* B0s = smc;                          // B0 [v][q], bf16
    unsigned char* Sbs = smc + kTileB;                 // S [v][k], bf16 copy
    unsigned char* bufs = smc + 2 * kTileB;            // 2 x { q, v (, k), alpha, eta }
    float* sig = reinterpret_cast<float*>(bufs + 2 * kBufB);
    float* pim = sig + kC;
    float* tpr = pim + kC;
    const uint32_t sB0 = (uint32_t)__cvta_generic_to_shared(B0s);
    const uint32_t sS = (uint32_t)__cvta_generic_to_shared(Sbs);

    const int unit = blockIdx.x;
    const int h = unit % p.H;
    const int b = (unit / p.H) % p.B;
    const int l = unit / (p.H * p.B);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, g = lane >> 2, cq = lane & 3;

    using bf = __nv_bfloat16;
    const bf* X = static_cast<const bf*>(p.x) + tok_off(p.x_s, l, b, 0, h);
    const bf* G = static_cast<const bf*>(p.g) + tok_off(p.g_s, l, b, 0, h);
    const bf* Qp = static_cast<const bf*>(p.q) + tok_off(p.q_s, l, b, 0, h);
    const bf* Vp = COSTATE ? X : G;
    const bf* Kp = COSTATE ? G : X;
    const long long qst = p.q_s[2], vst = COSTATE ? p.x_s[2] : p.g_s[2], kst = COSTATE ? p.g_s[2] : p.x_s[2];
    const long long gate0 = ((long long)l * p.B + b) * p.T * p.H + h;

    // B0 as bf16 [v][q]; S starts at zero (the fast weights begin at W0)
    const float* w0 = p.W0 + (size_t)(l * p.H + h) * 64 * 64;  // [dout][din]
    for (int e = tid; e < 64 * 32; e += kThr) {
        const int m = e >> 5, k = (e & 31) * 2;
        const float v0 = COSTATE ? w0[k * 64 + m] : w0[m * 64 + k];
        const float v1 = COSTATE ? w0[(k + 1) * 64 + m] : w0[m * 64 + k + 1];
        const uint32_t off = swz(m, k >> 3) + (k & 7) * 2;
        *reinterpret_cast<uint32_t*>(B0s + off) = pack(v0, v1);
        *reinterpret_cast<uint32_t*>(Sbs + off) = 0u;
    }

    // chunk c's rows and gates into buffer c & 1 (zeros, alpha = 1, eta = 0 past T)
    auto stage = [&](int c) {
        unsigned char* bb = bufs + (c & 1) * kBufB;
        const uint32_t sb = (uint32_t)__cvta_generic_to_shared(bb);
        const int c0 = c * kC;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int pc = tid + i * kThr;
            const int row = pc >> 3, piece = pc & 7;
            const bool ok = c0 + row < p.T;
            const long long t = ok ? c0 + row : 0;
            const uint32_t off = swz(row, piece);
            cpa16(sb + off, Qp + t * qst + piece * 8, ok);
            cpa16(sb + kTileB + off, Vp + t * vst + piece * 8, ok);
            if (COSTATE) cpa16(sb + 2 * kTileB + off, Kp + t * kst + piece * 8, ok);
        }
        const int t = c0 + (tid & 63);
        if (t < p.T)
            cpa4(sb + kGateOff + tid * 4, (tid < 64 ? p.alpha : p.eta) + gate0 + (long long)t * p.H, true);
        else
            reinterpret_cast<float*>(bb + kGateOff)[tid] = tid < 64 ? 1.0f : 0.0f;
        cpa_commit();
    };

    float sacc[8][4];
#pragma unroll
    for (int n = 0; n < 8; ++n) sacc[n][0] = sacc[n][1] = sacc[n][2] = sacc[n][3] = 0.0f;
    const int n_chunks = (p.T + kC - 1) / kC;
    stage(0);
    for (int c = 0; c < n_chunks; ++c) {
        cpa_wait<0>();
        __syncthreads();  // chunk c staged, the S copy of chunk c-1 written, chunk c-1 read
        if (c + 1 < n_chunks) stage(c + 1);
        unsigned char* bb = bufs + (c & 1) * kBufB;
        const uint32_t sQ = (uint32_t)__cvta_generic_to_shared(bb);
        const uint32_t sV = sQ + kTileB;
        const uint32_t sK = COSTATE ? sQ + 2 * kTileB : sQ;
        const float* al = reinterpret_cast<const float*>(bb + kGateOff);
        const float* et = al + kC;

        if (tid < kC) {  // decay pieces
            float sg = 1.0f, pp = 1.0f;
            for (int r = tid + 1; r <= (tid | 7); ++r) sg *= al[r];
            for (int r = tid & ~7; r < tid; ++r) pp *= al[r];
            sig[tid] = sg;
            pim[tid] = pp;
        } else if (tid < kC + 8) {
            const int j = tid - kC;
            float tp = 1.0f;
            for (int r = 0; r < 8; ++r) tp *= al[8 * j + r];
            tpr[j] = tp;
        }

        // this warp's Q fragments, reloaded where used (fewer live registers)
        auto ldq = [&](int kk, uint32_t (&q)[4]) { ldsm4(sQ + swz(16 * warp + (lane & 15), 2 * kk + (lane >> 4)), q); };
        // P = Q K^T over the column tiles at or before this warp's tokens
        float pacc[8][4];
#pragma unroll
        for (int n = 0; n < 8; ++n) pacc[n][0] = pacc[n][1] = pacc[n][2] = pacc[n][3] = 0.0f;
        // (k-steps outside, column tiles inside: consecutive MMAs use different
        // accumulators)
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
            uint32_t q[4];
            ldq(kk, q);
#pragma unroll
            for (int jp = 0; jp < 4; ++jp) {
                if (jp <= warp) {
                    uint32_t r[4];
                    ld_b_nk(sK, 16 * jp, 16 * kk, lane, r);
                    mma(pacc[2 * jp], q, r[0], r[1]);
                    mma(pacc[2 * jp + 1], q, r[2], r[3]);
                }
            }
        }
        // the carried fast weights: o = Q S^T (scaled by a_t below)
        float oacc[8][4];
#pragma unroll
        for (int n = 0; n < 8; ++n) oacc[n][0] = oacc[n][1] = oacc[n][2] = oacc[n][3] = 0.0f;
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
            uint32_t q[4];
            ldq(kk, q);
#pragma unroll
            for (int jp = 0; jp < 4; ++jp) {
                uint32_t r[4];
                ld_b_nk(sS, 16 * jp, 16 * kk, lane, r);
                mma(oacc[2 * jp], q, r[0], r[1]);
                mma(oacc[2 * jp + 1], q, r[2], r[3]);
            }
        }
        __syncthreads();  // decay pieces ready; every read of the S copy done

        float tp[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) tp[j] = tpr[j];
        // eta_s sig_s for this thread's columns s = 8j + 2cq + e (reads and write)
        float se[8][2];
#pragma unroll
        for (int j = 0; j < 8; ++j)
#pragma unroll
            for (int e = 0; e < 2; ++e) se[j][e] = et[8 * j + 2 * cq + e] * sig[8 * j + 2 * cq + e];
        // P'_ts = -E_ts P_ts (zero for s >= t); a_t for this thread's two tokens
        float a_row[2];
#pragma unroll
        for (int hr = 0; hr < 2; ++hr) {
            const int t = 16 * warp + g + 8 * hr;
            const int jt = t >> 3;
            float dd[2];  // columns in t's own piece: the alphas strictly between s and t
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                const int s = 8 * jt + 2 * cq + e;
                float d = s < t ? et[s] : 0.0f;
                for (int r = s + 1; r < t; ++r) d *= al[r];
                dd[e] = d;
            }
            float tau = pim[t];  // alphas in [8j + 8, t) for the piece j being scaled
#pragma unroll
            for (int j = 7; j >= 0; --j) {
                const bool below = j < jt;
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                    const float dec = below ? se[j][e] * tau : (j == jt ? dd[e] : 0.0f);
                    pacc[j][2 * hr + e] *= -dec;
                }
                tau = below ? tau * tp[j] : tau;
            }
            a_row[hr] = tau;
        }
#pragma unroll
        for (int n = 0; n < 8; ++n) {
            oacc[n][0] *= a_row[0];
            oacc[n][1] *= a_row[0];
            oacc[n][2] *= a_row[1];
            oacc[n][3] *= a_row[1];
        }
        // + B0 q_t
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
            uint32_t q[4];
            ldq(kk, q);
#pragma unroll
            for (int jp = 0; jp < 4; ++jp) {
                uint32_t r[4];
                ld_b_nk(sB0, 16 * jp, 16 * kk, lane, r);
                mma(oacc[2 * jp], q, r[0], r[1]);
                mma(oacc[2 * jp + 1], q, r[2], r[3]);
            }
        }
        // + P' V (P' carries the minus sign)
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
            if (kk <= warp) {
                const uint32_t pa[4] = {pack(pacc[2 * kk][0], pacc[2 * kk][1]),
                                        pack(pacc[2 * kk][2], pacc[2 * kk][3]),
                                        pack(pacc[2 * kk + 1][0], pacc[2 * kk + 1][1]),
                                        pack(pacc[2 * kk + 1][2], pacc[2 * kk + 1][3])};
#pragma unroll
                for (int jp = 0; jp < 4; ++jp) {
                    uint32_t r[4];
                    ld_b_kn(sV, 16 * jp, 16 * kk, lane, r);
                    mma(oacc[2 * jp], pa, r[0], r[1]);
                    mma(oacc[2 * jp + 1], pa, r[2], r[3]);
                }
            }
        }
        // epilogue: rows of this thread's two tokens, two adjacent columns per tile
        const EpiParams& ep = p.epi;
        if (!ep.out2 && !ep.zin) {
#pragma unroll
            for (int hr = 0; hr < 2; ++hr) {
                const int t = c * kC + 16 * warp + g + 8 * hr;
                if (t < p.T) {
                    bf* orow = static_cast<bf*>(ep.out) + tok_off(ep.out_str, l, b, t, h) + 2 * cq;
#pragma unroll
                    for (int n = 0; n < 8; ++n)
                        *reinterpret_cast<uint32_t*>(orow + 8 * n) = pack(oacc[n][2 * hr], oacc[n][2 * hr + 1]);
                }
            }
        } else {
#pragma unroll
        for (int hr = 0; hr < 2; ++hr) {
            const int t = c * kC + 16 * warp + g + 8 * hr;
            if (t < p.T) {
                bf* orow = static_cast<bf*>(ep.out) + tok_off(ep.out_str, l, b, t, h);
                bf* o2row = ep.out2 ? static_cast<bf*>(ep.out2) + tok_off(ep.out2_str, l, b, t, h) : nullptr;
                const bf* zrow = ep.zin ? static_cast<const bf*>(ep.zin) + tok_off(ep.z_str, l, b, t, h) : nullptr;
#pragma unroll
                for (int n = 0; n < 8; ++n) {
                    const int col = 8 * n + 2 * cq;
                    float v0 = oacc[n][2 * hr], v1 = oacc[n][2 * hr + 1];
                    if (o2row)
                        *reinterpret_cast<__nv_bfloat162*>(o2row + col) =
                            __floats2bfloat162_rn(act_f(ep.act, v0), act_f(ep.act, v1));
                    if (zrow) {
                        const float2 z = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(zrow + col));
                        v0 *= act_df(ep.act, z.x);
                        v1 *= act_df(ep.act, z.y);
                    }
                    *reinterpret_cast<__nv_bfloat162*>(orow + col) = __floats2bfloat162_rn(v0, v1);
                }
            }
        }
        }
        // the write: S <- a_end S - sum_s w_s v_s k_s^T, w_s = eta_s sig_s prod_{pieces after s} tp
        float sfx[8];
        sfx[7] = 1.0f;
#pragma unroll
        for (int j = 6; j >= 0; --j) sfx[j] = sfx[j + 1] * tp[j + 1];
        const float a_end = sfx[0] * tp[0];
#pragma unroll
        for (int n = 0; n < 8; ++n) {
            sacc[n][0] *= a_end;
            sacc[n][1] *= a_end;
            sacc[n][2] *= a_end;
            sacc[n][3] *= a_end;
        }
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
            // A = (w o V)^T rows [16 warp, +16), tokens [16 kk, +16), from V stored [s][v]
            uint32_t va[4];
            ldsm4t(sV + swz(16 * kk + (lane & 7) + ((lane >> 4) << 3), 2 * warp + ((lane >> 3) & 1)), va);
            const float w00 = -se[2 * kk][0] * sfx[2 * kk], w01 = -se[2 * kk][1] * sfx[2 * kk];
            const float w10 = -se[2 * kk + 1][0] * sfx[2 * kk + 1], w11 = -se[2 * kk + 1][1] * sfx[2 * kk + 1];
            va[0] = scale2(va[0], w00, w01);
            va[1] = scale2(va[1], w00, w01);
            va[2] = scale2(va[2], w10, w11);
            va[3] = scale2(va[3], w10, w11);
#pragma unroll
            for (int jp = 0; jp < 4; ++jp) {
                uint32_t r[4];
                ld_b_kn(sK, 16 * jp, 16 * kk, lane, r);
                mma(sacc[2 * jp], va, r[0], r[1]);
                mma(sacc[2 * jp + 1], va, r[2], r[3]);
            }
        }
        // bf16 copy of this warp's rows of S for the next chunk's read
        const int m = 16 * warp + g;
#pragma unroll
        for (int n = 0; n < 8; ++n) {
            *reinterpret_cast<uint32_t*>(Sbs + swz(m, n) + cq * 4) = pack(sacc[n][0], sacc[n][1]);
            *reinterpret_cast<uint32_t*>(Sbs + swz(m + 8, n) + cq * 4) = pack(sacc[n][2], sacc[n][3]);
        }
    }
}

template <bool COSTATE>
cudaError_t launch(const GatedParams& p, int blocks, cudaStream_t stream) {
    auto kern = chunk_decay_kernel<COSTATE>;
    const size_t smem = smem_bytes<COSTATE>();
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e == cudaSuccess)  // room for the CTAs the registers allow
        e = cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
    if (e != cudaSuccess) return e;
    kern<<<blocks, kThr, smem, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace cdec

template <bool COSTATE>
cudaError_t launch_serial_reg(const GatedParams& p, int blocks, cudaStream_t stream) {
    serial_reg_kernel<COSTATE><<<blocks, kThreads, 0, stream>>>(p);
    return cudaGetLastError();
}

template <bool COSTATE, bool BF16>
cudaError_t launch_serial(const GatedParams& p, int blocks, size_t smem, cudaStream_t stream) {
    auto kern = serial_kernel<COSTATE, BF16>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    kern<<<blocks, kThreads, smem, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace gated

size_t gated_serial_smem(int din, int dout, bool costate) {
    const int J = costate ? dout : din;
    return sizeof(float) * ((size_t)2 * gated::kTile * (J + 4) + 2 * (2 * (size_t)J + gated::kTile + 2));
}

// The register kernel reads 16-byte pieces of bf16 rows: widths a multiple of 16,
// the read at most kRegJ wide, every token row 16-byte aligned.
static bool serial_reg_ok(const GatedParams& p, bool costate, bool bf16) {
    const int J = costate ? p.dout : p.din;
    if (!bf16 || J > gated::kRegJ || J % 16 != 0) return false;
    const void* ptrs[3] = {p.x, p.g, p.q};
    const long long* strs[3] = {p.x_s, p.g_s, p.q_s};
    for (int k = 0; k < 3; ++k) {
        if ((reinterpret_cast<uintptr_t>(ptrs[k]) & 15u) != 0) return false;
        for (int i = 0; i < 4; ++i)
            if (strs[k][i] % 8 != 0) return false;
    }
    return true;
}

// The chunked kernel stages 16-byte pieces of 64-wide bf16 token rows and stores
// pairs of bf16 outputs: W 64 x 64, alpha_t given, rows 16-byte aligned, the
// epilogue tensors 4-byte aligned with even strides.
static bool chunk_decay_ok(const GatedParams& p, bool costate, bool bf16) {
    if (!bf16 || p.din != 64 || p.dout != 64 || !p.alpha || !p.eta || p.T <= 0) return false;
    if (!serial_reg_ok(p, costate, bf16)) return false;
    const void* ep[3] = {p.epi.out, p.epi.out2, p.epi.zin};
    const long long* es[3] = {p.epi.out_str, p.epi.out2_str, p.epi.z_str};
    for (int k = 0; k < 3; ++k) {
        if (!ep[k]) continue;
        if ((reinterpret_cast<uintptr_t>(ep[k]) & 3u) != 0) return false;
        for (int i = 0; i < 4; ++i)
            if (es[k][i] % 2 != 0) return false;
    }
    return true;
}

// Retention scans (alpha_t given): the chunked kernel where the shape allows it,
// else a token-serial kernel (registers for bf16 reads of at most 64 inputs,
// shared memory otherwise).
cudaError_t launch_gated_serial(const GatedParams& p, bool costate, bool bf16, cudaStream_t stream) {
    const int NO = costate ? p.din : p.dout;
    const int tiles = (NO + gated::kTile - 1) / gated::kTile;
    const long long blocks = (long long)p.L * p.B * p.H * tiles;
    const size_t smem = gated_serial_smem(p.din, p.dout, costate);
    if (blocks <= 0) return cudaSuccess;
    if (chunk_decay_ok(p, costate, bf16))  // one CTA per unit (tiles == 1)
        return costate ? gated::cdec::launch<true>(p, (int)blocks, stream)
                       : gated::cdec::launch<false>(p, (int)blocks, stream);
    if (serial_reg_ok(p, costate, bf16))  // the state fits in registers
        return costate ? gated::launch_serial_reg<true>(p, (int)blocks, stream)
                       : gated::launch_serial_reg<false>(p, (int)blocks, stream);
    if (costate)
        return bf16 ? gated::launch_serial<true, true>(p, (int)blocks, smem, stream)
                    : gated::launch_serial<true, false>(p, (int)blocks, smem, stream);
    return bf16 ? gated::launch_serial<false, true>(p, (int)blocks, smem, stream)
                : gated::launch_serial<false, false>(p, (int)blocks, smem, stream);
}

cudaError_t launch_gated_prescale(const void* g, const TokStr& gs, const float* eta, void* out, int L,
                                  int B, int T, int H, int w, bool bf16, cudaStream_t stream) {
    const long long n = (long long)L * B * T * H * (w / (bf16 ? 8 : 4));
    if (n <= 0) return cudaSuccess;
    // contiguous rows (the output's own layout) and 32-bit piece indices: the flat
    // kernel, four independent 16-byte pieces per thread and pass
    const bool contig = gs.s[3] == w && gs.s[2] == (long long)H * w &&
                        gs.s[1] == (long long)T * H * w && gs.s[0] == (long long)B * T * H * w;
    if (contig && n < (1ll << 31) - 4 * (long long)gated::kFlatThreads * 152 * 8) {
        const int grid = 152 * 8;
        if (bf16)
            gated::prescale_flat_kernel<true><<<grid, gated::kFlatThreads, 0, stream>>>(
                g, eta, out, (int)n, w / 8);
        else
            gated::prescale_flat_kernel<false><<<grid, gated::kFlatThreads, 0, stream>>>(
                g, eta, out, (int)n, w / 4);
        return cudaGetLastError();
    }
    long long blocks = (n + 255) / 256;
    if (blocks > 152 * 16) blocks = 152 * 16;
    if (bf16)
        gated::prescale_kernel<true><<<(int)blocks, 256, 0, stream>>>(g, gs, eta, out, L, B, T, H, w);
    else
        gated::prescale_kernel<false><<<(int)blocks, 256, 0, stream>>>(g, gs, eta, out, L, B, T, H, w);
    return cudaGetLastError();
}

}  // namespace gl
