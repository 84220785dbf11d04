// grads.cu -- per-token reductions for the outer gradients through the reads.
//
// With the writes detached and per-token step sizes learned (Sec. 3, practical
// architecture and training), the read y_t = W_t x_t is linear in every eta_s, and
//     dL/deta_s = -ghat_s . r_s,   r_s = sum_{t>s} (x_t . x_s) dL/dy_t,
// the anti-causal (suffix) read of the same writes.  For the costate read
// gin_t = W_t^T g_t the same holds with dL/deta_s = -x_s . r_s and
// r_s = sum_{t>s} (g_t . ghat_s) dL/dgin_t.  The suffix read runs in the scan
// kernels (reverse mode); this file holds the final row dot.  With retention alpha_t
// the gate derivatives take the states at every chunk boundary, carried here from
// per-chunk aggregates; the aggregates and the per-chunk expansion are in
// gate_grads_tc.cu.
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
// Gate derivatives with retention (alpha_t): the states at every chunk boundary from
// the per-chunk aggregates, in place (fp32 [unit][nch][64][64], one thread per entry
// and unit):
//   VS[c] <- D at chunk c's first token:  D_0 = 0,  D_{c+1} = A_c D_c + Vt_c
//   UR[c] <- R at chunk c's last token:   R_{nch-1} = 0,  R_c = Ut_{c+1} + A_{c+1} R_{c+1}
// (the chunk map of Eq. 2, S -> a S + U, carried forwards and, for the decayed suffix
// state, backwards).
// One thread: two float4s of one unit (entries 4e..4e+3 and 4e+2048..4e+2051), with
// loads two chunks ahead: four 16-byte loads in flight per thread.
__global__ void __launch_bounds__(kThreads)
    gate_state_scan_kernel(float* __restrict__ VS, float* __restrict__ UR, const float* __restrict__ Ad,
                           long long units, int nch) {
    const long long e = (long long)blockIdx.x * kThreads + threadIdx.x;  // one of 512 per unit
    if (e >= units * 512) return;
    const long long unit = e >> 9;
    const long long off = unit * nch * 1024ll + (e & 511);
    const float* a = Ad + unit * nch;
    auto carry = [&](float4* P, bool forward) {
        float4 s0 = make_float4(0.f, 0.f, 0.f, 0.f), s1 = s0;
        auto at = [&](int c) { return (long long)(forward ? c : nch - 1 - c) * 1024; };
        float4 n0 = P[at(0)], n1 = P[at(0) + 512];
        float4 m0 = s0, m1 = s0;
        if (nch > 1) {
            m0 = P[at(1)];
            m1 = P[at(1) + 512];
        }
        for (int c = 0; c < nch; ++c) {
            const float4 c0 = n0, c1 = n1;
            n0 = m0;
            n1 = m1;
            if (c + 2 < nch) {
                m0 = P[at(c + 2)];
                m1 = P[at(c + 2) + 512];
            }
            P[at(c)] = s0;
            P[at(c) + 512] = s1;
            const float ac = a[forward ? c : nch - 1 - c];
            s0 = make_float4(fmaf(ac, s0.x, c0.x), fmaf(ac, s0.y, c0.y), fmaf(ac, s0.z, c0.z), fmaf(ac, s0.w, c0.w));
            s1 = make_float4(fmaf(ac, s1.x, c1.x), fmaf(ac, s1.y, c1.y), fmaf(ac, s1.z, c1.z), fmaf(ac, s1.w, c1.w));
        }
    };
    carry(reinterpret_cast<float4*>(VS) + off, true);
    carry(reinterpret_cast<float4*>(UR) + off, false);
}

}  // namespace grads

cudaError_t launch_gate_state_scan(float* VS, float* UR, const float* Ad, long long units, int nch,
                                   cudaStream_t stream) {
    const long long n = units * 512;  // pairs of float4 entries
    if (n <= 0 || nch <= 0) return cudaSuccess;
    const long long grid = (n + grads::kThreads - 1) / grads::kThreads;
    if (grid > 0x7FFFFFFF) return cudaErrorInvalidValue;
    grads::gate_state_scan_kernel<<<(int)grid, grads::kThreads, 0, stream>>>(VS, UR, Ad, units, nch);
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
