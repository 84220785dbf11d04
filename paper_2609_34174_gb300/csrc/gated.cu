// gated.cu -- the scans with the paper's general gates (Sec. 3 "Observation",
// Eq. 2): per-token step sizes eta_t and retention alpha_t with decay centred at
// the slow weights,
//
//     W_{t+1} = W0 + alpha_t (W_t - W0) - eta_t ghat_t x_t^T,       W at t = 0 is W0,
//
// read before each write: y_t = W_t x_t (Eq. 3), gin_t = W_t^T gout_t (Eq. 4).
// alpha_t = 0 resets the fast weights to W0 (a document boundary).
//
// Two kernels (bf16 64 x 64 maps with alpha_t run the tensor-core kernel of
// scan_decay_tc.cu):
//   prescale_kernel  eta_t only (alpha = 1): the writes eta_t ghat_t x_t^T are the
//                    plain writes of ghat'_t = eta_t ghat_t, so the chunked kernels
//                    run on ghat' with eta = 1.  One elementwise pass into the
//                    workspace (rounded to the input dtype, like ghat itself).
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

// Retention scans (alpha_t given) that the tensor-core kernel (scan_decay_tc.cu)
// does not take: a token-serial kernel (registers for bf16 reads of at most 64
// inputs, shared memory otherwise).
cudaError_t launch_gated_serial(const GatedParams& p, bool costate, bool bf16, cudaStream_t stream) {
    const int NO = costate ? p.din : p.dout;
    const int tiles = (NO + gated::kTile - 1) / gated::kTile;
    const long long blocks = (long long)p.L * p.B * p.H * tiles;
    const size_t smem = gated_serial_smem(p.din, p.dout, costate);
    if (blocks <= 0) return cudaSuccess;
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
