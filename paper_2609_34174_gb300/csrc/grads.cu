// grads.cu -- per-token reductions for the outer gradients through the reads.
//
// With the writes detached and per-token step sizes learned (Sec. 3, practical
// architecture and training), the read y_t = W_t x_t is linear in every eta_s, and
//     dL/deta_s = -ghat_s . r_s,   r_s = sum_{t>s} (x_t . x_s) dL/dy_t,
// the anti-causal (suffix) read of the same writes.  For the costate read
// gin_t = W_t^T g_t the same holds with dL/deta_s = -x_s . r_s and
// r_s = sum_{t>s} (g_t . ghat_s) dL/dgin_t.  The suffix read runs in the scan
// kernels (reverse mode); this file holds the final row dot.
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

// out[l][b][t][h] = scale * sum_j a[l,b,t,h,j] * r[l,b,t,h,j]; one warp per token row.
template <bool BF16>
__global__ void __launch_bounds__(kThreads)
    rowdot_kernel(const void* __restrict__ a, TokStr as, const void* __restrict__ r, TokStr rs,
                  float* __restrict__ out, int L, int B, int T, int H, int w, float scale) {
    const long long rows = (long long)L * B * T * H;
    const long long row = (long long)blockIdx.x * (kThreads / 32) + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (row >= rows) return;  // warp-uniform
    long long t = row;
    const int h = (int)(t % H);
    t /= H;
    const int tt = (int)(t % T);
    t /= T;
    const int b = (int)(t % B);
    const int l = (int)(t / B);
    const long long ao = tok_off(as.s, l, b, tt, h), ro = tok_off(rs.s, l, b, tt, h);
    float acc = 0.f;
    for (int j = lane; j < w; j += 32) acc = fmaf(ld<BF16>(a, ao + j), ld<BF16>(r, ro + j), acc);
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if (lane == 0) out[row] = scale * acc;
}

}  // namespace grads

cudaError_t launch_rowdot(const void* a, const TokStr& as, const void* r, const TokStr& rs,
                          float* out, int L, int B, int T, int H, int w, float scale, bool bf16,
                          cudaStream_t stream) {
    const long long rows = (long long)L * B * T * H;
    const long long grid = (rows + grads::kThreads / 32 - 1) / (grads::kThreads / 32);
    if (grid <= 0 || grid > 0x7FFFFFFF) return cudaErrorInvalidValue;
    if (bf16)
        grads::rowdot_kernel<true><<<(int)grid, grads::kThreads, 0, stream>>>(a, as, r, rs, out, L, B,
                                                                               T, H, w, scale);
    else
        grads::rowdot_kernel<false><<<(int)grid, grads::kThreads, 0, stream>>>(a, as, r, rs, out, L,
                                                                                B, T, H, w, scale);
    return cudaGetLastError();
}

}  // namespace gl
