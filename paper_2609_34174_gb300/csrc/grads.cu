// grads.cu -- per-token reductions for the outer gradients through the reads.
//
// With the writes detached and per-token step sizes learned (Sec. 3, practical
// architecture and training), the read y_t = W_t x_t is linear in every eta_s, and
//     dL/deta_s = -ghat_s . r_s,   r_s = sum_{t>s} (x_t . x_s) dL/dy_t,
// the anti-causal (suffix) read of the same writes.  For the costate read
// gin_t = W_t^T g_t the same holds with dL/deta_s = -x_s . r_s and
// r_s = sum_{t>s} (g_t . ghat_s) dL/dgin_t.  The suffix read runs in the scan
// kernels (reverse mode); this file holds the final row dot.  With retention alpha_t
// the gate derivatives take the state of the retention scan at every chunk start,
// forwards and over the inputs reversed in time (the reversed copies and the
// per-chunk combination are here).
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "scan_common.cuh"

namespace gl {
namespace grads {

constexpr int kThreads = 256;

template <bool BF16>
__device__ __forceinline__ float ld(const void* p, long long i) {
    if constexpr (BF16)
        return __bfloat162float(static_cast<const __nv_bfloat16*>(p)[i]);
    else
        return static_cast<const float*>(p)[i];
}

// 8 bf16 or 4 fp32 values of one 16-byte piece, as floats; returns the count.
template <bool BF16>
__device__ __forceinline__ int ld16(const void* p, long long i, float* f) {
    const uint4 v = *reinterpret_cast<const uint4*>(static_cast<const char*>(p) + i * (BF16 ? 2 : 4));
    if constexpr (BF16) {
        const __nv_bfloat16* h = reinterpret_cast<const __nv_bfloat16*>(&v);
#pragma unroll
        for (int k = 0; k < 8; ++k) f[k] = __bfloat162float(h[k]);
        return 8;
    } else {
        f[0] = __uint_as_float(v.x);
        f[1] = __uint_as_float(v.y);
        f[2] = __uint_as_float(v.z);
        f[3] = __uint_as_float(v.w);
        return 4;
    }
}

// out[l][b][t][h] = scale * sum_j a[l,b,t,h,j] * r[l,b,t,h,j], or with SQ the squared
// distance scale * sum_j (a - r)^2 (the consistency term of Eq. 5).  A group of
// `lanes` lanes (a power of two up to 32) takes one token row in 16-byte pieces when
// `vec`, else element by element with a whole warp per row.
template <bool BF16, bool SQ>
__global__ void __launch_bounds__(kThreads)
    rowdot_kernel(const void* __restrict__ a, TokStr as, const void* __restrict__ r, TokStr rs,
                  float* __restrict__ out, int L, int B, int T, int H, int w, float scale, int vec,
                  int lanes) {
    const long long rows = (long long)L * B * T * H;
    const int lane = threadIdx.x & 31;
    const int LR = vec ? lanes : 32;
    const int sub = lane / LR, cl = lane - sub * LR;
    const long long row = ((long long)blockIdx.x * (kThreads / 32) + (threadIdx.x >> 5)) * (32 / LR) + sub;
    const bool live = row < rows;
    long long t = live ? row : 0;
    const int h = (int)(t % H);
    t /= H;
    const int tt = (int)(t % T);
    t /= T;
    const int b = (int)(t % B);
    const int l = (int)(t / B);
    const long long ao = tok_off(as.s, l, b, tt, h), ro = tok_off(rs.s, l, b, tt, h);
    float acc = 0.f;
    if (live) {
        if (vec) {
            constexpr int kPer = BF16 ? 8 : 4;
            for (int j = cl * kPer; j < w; j += LR * kPer) {
                float fa[8], fr[8];
                ld16<BF16>(a, ao + j, fa);
                ld16<BF16>(r, ro + j, fr);
#pragma unroll
                for (int k = 0; k < kPer; ++k) {
                    if constexpr (SQ) {
                        const float dlt = fa[k] - fr[k];
                        acc = fmaf(dlt, dlt, acc);
                    } else {
                        acc = fmaf(fa[k], fr[k], acc);
                    }
                }
            }
        } else {
            for (int j = cl; j < w; j += 32) {
                if constexpr (SQ) {
                    const float dlt = ld<BF16>(a, ao + j) - ld<BF16>(r, ro + j);
                    acc = fmaf(dlt, dlt, acc);
                } else {
                    acc = fmaf(ld<BF16>(a, ao + j), ld<BF16>(r, ro + j), acc);
                }
            }
        }
    }
    for (int o = LR >> 1; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if (live && cl == 0) out[row] = scale * acc;
}

// ---------------------------------------------------------------------------
// Gate derivatives with retention (alpha_t).  The decayed suffix state is the state
// of the forward retention scan over the inputs reversed in time; its inputs are
// copied reversed, after T_pad - T zero rows, so that the reversed chunks of 128
// tokens are the original chunks in reverse order.

// out[l][b][T_pad-1-t][h][:] = in[l][b][t][h][:], in with element strides s, out
// contiguous with T_pad tokens; one thread per 16-byte piece.
__global__ void __launch_bounds__(kThreads)
    flip_rows_kernel(const void* __restrict__ in, TokStr s, void* __restrict__ out, int L, int B,
                     int T, int T_pad, int H, int pieces, int elem) {
    const long long n = (long long)L * B * T * H * pieces;
    for (long long v = (long long)blockIdx.x * kThreads + threadIdx.x; v < n;
         v += (long long)gridDim.x * kThreads) {
        const int pc = (int)(v % pieces);
        long long r = v / pieces;
        const int h = (int)(r % H);
        r /= H;
        const int t = (int)(r % T);
        r /= T;
        const int b = (int)(r % B);
        const int l = (int)(r / B);
        const long long src = tok_off(s.s, l, b, t, h) * elem + (long long)pc * 16;
        const long long dst = ((((long long)l * B + b) * T_pad + (T_pad - 1 - t)) * H + h) * pieces * 16 +
                              (long long)pc * 16;
        *reinterpret_cast<uint4*>(static_cast<char*>(out) + dst) =
            *reinterpret_cast<const uint4*>(static_cast<const char*>(in) + src);
    }
}

// Per-token gates [L][B][T][H] reversed into [L][B][T_pad][H]: the T_pad - T leading
// entries are pad, the others in (or fill where in == nullptr).
__global__ void __launch_bounds__(kThreads)
    flip_gates_kernel(const float* __restrict__ in, float fill, float pad, float* __restrict__ out,
                      int LB, int T, int T_pad, int H) {
    const long long n = (long long)LB * T_pad * H;
    for (long long v = (long long)blockIdx.x * kThreads + threadIdx.x; v < n;
         v += (long long)gridDim.x * kThreads) {
        const int h = (int)(v % H);
        const long long r = v / H;
        const int tau = (int)(r % T_pad);
        const long long lb = r / T_pad;
        const int t = T_pad - 1 - tau;
        out[v] = t >= T ? pad : (in ? in[(lb * T + t) * H + h] : fill);
    }
}

constexpr int kGC = 128;              // tokens per chunk (the retention kernel's)
constexpr int kGW = 64;               // map width (64 x 64 maps)
constexpr int kGRow = kGW * 2;        // bytes of a bf16 token row
constexpr int kGateSmem = (2 * kGW * kGW + kGC * kGC + 4 * kGC + 32) * 4 + 4 * kGC * kGRow;

// 16 bf16 values (32 bytes) of a shared-memory row as floats.
__device__ __forceinline__ void ld_row16(const __nv_bfloat16* p, float* f) {
#pragma unroll
    for (int q = 0; q < 2; ++q) {
        const uint4 v = reinterpret_cast<const uint4*>(p)[q];
        const __nv_bfloat16* hb = reinterpret_cast<const __nv_bfloat16*>(&v);
#pragma unroll
        for (int k = 0; k < 8; ++k) f[8 * q + k] = __bfloat162float(hb[k]);
    }
}

// One CTA per (unit, chunk of 128 tokens) of a 64 x 64 map.  With D_t = W_t - W0 and
// the read's pair (a, b) (forward: a = u, b = x; costate: a = g_out, b = u), S the
// state D at the chunk's first token and Rt the decayed suffix state at its last
// token c1 - 1, every token j of the chunk gets
//   dlog_alpha_j = alpha_j (P_j Q_j <S, Rt> + P_j sum_{s>j} G(j,s) v_s
//                           + Q_j sum_{i<j} (-eta_i) E(i,j) w_i + sum_{i<j<s} (-eta_i) E(i,j) G(j,s) M_is)
//   deta_j       = -(Q_j w_j + sum_{s>j} G(j,s) M_js)
// over tokens i, s of the chunk, with P_j, Q_j the alphas of the chunk before and
// after j, E(i,j) and G(j,s) those strictly between, v_s = a_s^T S b_s,
// w_i = ghat_i^T Rt x_i and M_is = (a_s . ghat_i)(x_i . b_s).  Tokens past T have
// alpha = 1, eta = 0 and zero rows.  S and Rt are fp32 [64][64] as the retention
// kernel's state warps hold them (row k: x index, column l: ghat index).  fp32
// throughout.
__global__ void __launch_bounds__(kThreads)
    gate_chunk_kernel(const __nv_bfloat16* __restrict__ x, TokStr xs, const __nv_bfloat16* __restrict__ gh,
                      TokStr gs, const __nv_bfloat16* __restrict__ a, TokStr as_,
                      const __nv_bfloat16* __restrict__ b, TokStr bs, const float* __restrict__ eta,
                      const float* __restrict__ alpha, const float* __restrict__ Sd,
                      const float* __restrict__ Rd, float* __restrict__ dlog_alpha,
                      float* __restrict__ deta, int B, int T, int H, int nch) {
    extern __shared__ float4 gsm4[];
    float* S = reinterpret_cast<float*>(gsm4);  // [64][64]
    float* Rt = S + kGW * kGW;                  // [64][64]
    float* Nm = Rt + kGW * kGW;                 // [128][128]  N_{i,j}
    float* v = Nm + kGC * kGC;
    float* w = v + kGC;
    float* et = w + kGC;
    float* al = et + kGC;
    float* red = al + kGC;                      // [32]
    __nv_bfloat16* tx = reinterpret_cast<__nv_bfloat16*>(red + 32);  // [128][64] each
    __nv_bfloat16* tg = tx + kGC * kGW;
    __nv_bfloat16* ta = tg + kGC * kGW;
    __nv_bfloat16* tb = ta + kGC * kGW;
    const int tid = threadIdx.x, lane = tid & 31;
    const long long unit = blockIdx.x / nch;
    const int c = (int)(blockIdx.x % nch);
    const int h = (int)(unit % H);
    const long long lb = unit / H;
    const int bb = (int)(lb % B);
    const int l = (int)(lb / B);
    const int c0 = c * kGC;
    // ---- states and token rows
    const float4* s4 = reinterpret_cast<const float4*>(Sd + (unit * nch + c) * (long long)(kGW * kGW));
    const float4* r4 = reinterpret_cast<const float4*>(Rd + (unit * nch + (nch - 1 - c)) * (long long)(kGW * kGW));
    for (int i = tid; i < kGW * kGW / 4; i += kThreads) {
        reinterpret_cast<float4*>(S)[i] = s4[i];
        reinterpret_cast<float4*>(Rt)[i] = r4[i];
    }
    const __nv_bfloat16* src[4] = {x, gh, a, b};
    const TokStr* str[4] = {&xs, &gs, &as_, &bs};
    __nv_bfloat16* dst[4] = {tx, tg, ta, tb};
    for (int e = tid; e < 4 * kGC * 8; e += kThreads) {
        const int which = e / (kGC * 8), r = (e / 8) % kGC, pc = e % 8;
        const int t = c0 + r;
        uint4 val = make_uint4(0u, 0u, 0u, 0u);
        if (t < T) val = *reinterpret_cast<const uint4*>(src[which] + tok_off(str[which]->s, l, bb, t, h) + pc * 8);
        reinterpret_cast<uint4*>(dst[which] + r * kGW)[pc] = val;
    }
    for (int r = tid; r < kGC; r += kThreads) {
        const int t = c0 + r;
        const long long gi = (lb * T + t) * H + h;
        et[r] = t < T ? eta[gi] : 0.0f;
        al[r] = t < T ? (alpha ? alpha[gi] : 1.0f) : 1.0f;
        Nm[r * kGC + kGC - 1] = 0.0f;  // N_{i,127}: no later token in the chunk
    }
    __syncthreads();
    // ---- <S, Rt>
    float kp = 0.0f;
    for (int i = tid; i < kGW * kGW; i += kThreads) kp = fmaf(S[i], Rt[i], kp);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) kp += __shfl_xor_sync(0xffffffffu, kp, o);
    if (lane == 0) red[tid >> 5] = kp;
    // ---- v_s = a_s^T S b_s and w_i = ghat_i^T Rt x_i: token pairs, half the rows k each
    {
        const int tok = tid >> 1, hh = tid & 1;
        float av[kGW], gv[kGW];
#pragma unroll
        for (int q = 0; q < kGW / 16; ++q) {
            ld_row16(ta + tok * kGW + 16 * q, av + 16 * q);
            ld_row16(tg + tok * kGW + 16 * q, gv + 16 * q);
        }
        float vs = 0.0f, wi = 0.0f;
#pragma unroll 4
        for (int k = hh * 32; k < hh * 32 + 32; ++k) {
            float sa = 0.0f, rg = 0.0f;
#pragma unroll
            for (int q = 0; q < kGW; ++q) {
                sa = fmaf(S[k * kGW + q], av[q], sa);
                rg = fmaf(Rt[k * kGW + q], gv[q], rg);
            }
            vs = fmaf(__bfloat162float(tb[tok * kGW + k]), sa, vs);
            wi = fmaf(__bfloat162float(tx[tok * kGW + k]), rg, wi);
        }
        vs += __shfl_xor_sync(0xffffffffu, vs, 1);
        wi += __shfl_xor_sync(0xffffffffu, wi, 1);
        if (hh == 0) {
            v[tok] = vs;
            w[tok] = wi;
        }
    }
    // ---- N_{i,j} = sum_{s>j} G(j,s) M_is, row i by a token pair (half the features each)
    {
        const int i = tid >> 1, hh = tid & 1;
        float gi[32], xi[32];
        ld_row16(tg + i * kGW + 32 * hh, gi);
        ld_row16(tg + i * kGW + 32 * hh + 16, gi + 16);
        ld_row16(tx + i * kGW + 32 * hh, xi);
        ld_row16(tx + i * kGW + 32 * hh + 16, xi + 16);
        float nrun = 0.0f;
#pragma unroll 1
        for (int s2 = kGC - 1; s2 >= 1; --s2) {
            float as2[32], bs2[32];
            ld_row16(ta + s2 * kGW + 32 * hh, as2);
            ld_row16(ta + s2 * kGW + 32 * hh + 16, as2 + 16);
            ld_row16(tb + s2 * kGW + 32 * hh, bs2);
            ld_row16(tb + s2 * kGW + 32 * hh + 16, bs2 + 16);
            float d1 = 0.0f, d2 = 0.0f;
#pragma unroll
            for (int q = 0; q < 32; ++q) {
                d1 = fmaf(as2[q], gi[q], d1);
                d2 = fmaf(bs2[q], xi[q], d2);
            }
            d1 += __shfl_xor_sync(0xffffffffu, d1, 1);
            d2 += __shfl_xor_sync(0xffffffffu, d2, 1);
            if (s2 > i) {
                nrun = fmaf(al[s2], nrun, d1 * d2);  // N_{i,s2-1} = M_{i,s2} + alpha_{s2} N_{i,s2}
                if (hh == 0) Nm[i * kGC + s2 - 1] = nrun;
            }
        }
    }
    __syncthreads();
    // ---- per token j: the four terms
    if (tid < kGC) {
        const int j = tid;
        float kappa = 0.0f;
#pragma unroll
        for (int q = 0; q < kThreads / 32; ++q) kappa += red[q];
        float P = 1.0f, Q = 1.0f;
        for (int r = 0; r < j; ++r) P *= al[r];
        for (int r = j + 1; r < kGC; ++r) Q *= al[r];
        float t2 = 0.0f, g = 1.0f;
        for (int s2 = j + 1; s2 < kGC; ++s2) {
            t2 = fmaf(g, v[s2], t2);
            g *= al[s2];
        }
        float t3 = 0.0f, t4j = 0.0f, e = 1.0f;
        for (int i = j - 1; i >= 0; --i) {
            const float ne = -et[i] * e;
            t3 = fmaf(ne, w[i], t3);
            t4j = fmaf(ne, Nm[i * kGC + j], t4j);
            e *= al[i];
        }
        const int t = c0 + j;
        if (t < T) {
            const long long gi = (lb * T + t) * H + h;
            dlog_alpha[gi] = al[j] * (P * Q * kappa + P * t2 + Q * t3 + t4j);
            deta[gi] = -(Q * w[j] + Nm[j * kGC + j]);
        }
    }
}

}  // namespace grads

cudaError_t launch_flip_rows(const void* in, const TokStr& s, void* out, int L, int B, int T, int T_pad,
                             int H, int w, int elem, cudaStream_t stream) {
    const int pieces = w * elem / 16;
    const long long n = (long long)L * B * T * H * pieces;
    if (n <= 0) return cudaSuccess;
    const long long grid = (n + grads::kThreads - 1) / grads::kThreads;
    grads::flip_rows_kernel<<<(int)(grid < 152 * 16 ? grid : 152 * 16), grads::kThreads, 0, stream>>>(
        in, s, out, L, B, T, T_pad, H, pieces, elem);
    return cudaGetLastError();
}

cudaError_t launch_flip_gates(const float* in, float fill, float pad, float* out, int L, int B, int T,
                              int T_pad, int H, cudaStream_t stream) {
    const long long n = (long long)L * B * T_pad * H;
    if (n <= 0) return cudaSuccess;
    const long long grid = (n + grads::kThreads - 1) / grads::kThreads;
    grads::flip_gates_kernel<<<(int)(grid < 152 * 16 ? grid : 152 * 16), grads::kThreads, 0, stream>>>(
        in, fill, pad, out, L * B, T, T_pad, H);
    return cudaGetLastError();
}

// The per-chunk gate derivatives of 64 x 64 bf16 maps (gate_chunk_kernel).
cudaError_t launch_gate_chunks(const void* x, const TokStr& xs, const void* gh, const TokStr& gs,
                               const void* a, const TokStr& as, const void* b, const TokStr& bs,
                               const float* eta, const float* alpha, const float* Sd, const float* Rd,
                               float* dlog_alpha, float* deta, int L, int B, int T, int H,
                               cudaStream_t stream) {
    const int nch = (T + grads::kGC - 1) / grads::kGC;
    const long long blocks = (long long)L * B * H * nch;
    if (blocks <= 0) return cudaSuccess;
    if (blocks > 0x7FFFFFFF) return cudaErrorInvalidValue;
    cudaError_t e = cudaFuncSetAttribute(grads::gate_chunk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         grads::kGateSmem);
    if (e != cudaSuccess) return e;
    using bf = __nv_bfloat16;
    grads::gate_chunk_kernel<<<(int)blocks, grads::kThreads, grads::kGateSmem, stream>>>(
        static_cast<const bf*>(x), xs, static_cast<const bf*>(gh), gs, static_cast<const bf*>(a), as,
        static_cast<const bf*>(b), bs, eta, alpha, Sd, Rd, dlog_alpha, deta, B, T, H, nch);
    return cudaGetLastError();
}

cudaError_t launch_rowdot(const void* a, const TokStr& as, const void* r, const TokStr& rs,
                          float* out, int L, int B, int T, int H, int w, float scale, bool bf16,
                          cudaStream_t stream, bool sqdist) {
    const long long rows = (long long)L * B * T * H;
    // 16-byte pieces when every row starts on a 16-byte boundary
    const int per = bf16 ? 8 : 4, elem = bf16 ? 2 : 4;
    bool vec = w % per == 0 && (reinterpret_cast<uintptr_t>(a) & 15u) == 0 &&
               (reinterpret_cast<uintptr_t>(r) & 15u) == 0;
    for (int i = 0; i < 4; ++i) vec = vec && (as.s[i] * elem) % 16 == 0 && (rs.s[i] * elem) % 16 == 0;
    int lanes = 32;
    if (vec) {
        const int pieces = w / per;
        lanes = 1;
        while (lanes < pieces && lanes < 32) lanes <<= 1;
    }
    const long long rows_per_cta = (long long)(grads::kThreads / 32) * (vec ? 32 / lanes : 1);
    const long long grid = (rows + rows_per_cta - 1) / rows_per_cta;
    if (grid <= 0 || grid > 0x7FFFFFFF) return cudaErrorInvalidValue;
    auto kern = bf16 ? (sqdist ? grads::rowdot_kernel<true, true> : grads::rowdot_kernel<true, false>)
                     : (sqdist ? grads::rowdot_kernel<false, true> : grads::rowdot_kernel<false, false>);
    kern<<<(int)grid, grads::kThreads, 0, stream>>>(a, as, r, rs, out, L, B, T, H, w, scale,
                                                    vec ? 1 : 0, lanes);
    return cudaGetLastError();
}

}  // namespace gl
