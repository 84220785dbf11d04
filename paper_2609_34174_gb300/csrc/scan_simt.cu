// scan_simt.cu -- fp32 chunked token scan on the CUDA cores (FFMA).
//
// The same computation as the tensor-core kernel (Sec. 3, Eqs. 3-4; Appendix C),
//     o_t = B0 q_t - eta * sum_{s<t} (k_s . q_t) v_s,
// for fp32 inputs, where the 1e-5 relative accuracy asked of fp32 rules out
// TF32 tensor-core products.  One CTA owns one (unit, 32-wide output tile) and
// walks the tokens in chunks of 32:
//     O_c = Q_c S_c^T - eta * strict_lower(Q_c K_c^T) V_c,
//     S_{c+1}^T = S_c^T - eta * K_c^T V_c,
// with the state S^T (dq x 32) resident in shared memory in fp32.
#include "scan_common.cuh"

namespace gl {

constexpr int kSimtChunk = 32;
constexpr int kSimtNv = 32;
constexpr int kSimtThreads = 256;

template <typename T>
__device__ __forceinline__ float ld_as_f32(const T* p);
template <>
__device__ __forceinline__ float ld_as_f32<float>(const float* p) { return *p; }
template <>
__device__ __forceinline__ float ld_as_f32<__nv_bfloat16>(const __nv_bfloat16* p) {
    return __bfloat162float(*p);
}

template <typename T>
__device__ __forceinline__ void st_from_f32(T* p, float v);
template <>
__device__ __forceinline__ void st_from_f32<float>(float* p, float v) { *p = v; }
template <>
__device__ __forceinline__ void st_from_f32<__nv_bfloat16>(__nv_bfloat16* p, float v) {
    *p = __float2bfloat16_rn(v);
}

// Shared memory: Q, K [32][dq], V [32][32], scores [32][33], S^T [dq][32].
// REV walks the chunks from the last to the first and mixes in the strictly LATER
// tokens of each chunk: the anti-causal read sum_{s>t} (k_s . q_t) v_s of the same
// writes (outer gradients through the reads).  W0 may be null (no base matrix).
template <typename T, bool REV>
__global__ void __launch_bounds__(kSimtThreads) simt_scan_kernel(const SimtScanParams p) {
    extern __shared__ float sm[];
    const int dq = p.dq;
    float* Qs = sm;
    float* Ks = Qs + kSimtChunk * dq;
    float* Vs = Ks + kSimtChunk * dq;
    float* Sc = Vs + kSimtChunk * kSimtNv;
    float* ST = Sc + kSimtChunk * (kSimtChunk + 1);

    const int n_tiles = (p.dv + kSimtNv - 1) / kSimtNv;
    const int j = blockIdx.x % n_tiles;
    const int u = blockIdx.x / n_tiles;
    const int h = u % p.H;
    const int b = (u / p.H) % p.B;
    const int l = u / (p.H * p.B);
    const int v0 = j * kSimtNv;
    const int tid = threadIdx.x;
    const T* q = static_cast<const T*>(p.q);
    const T* k = static_cast<const T*>(p.k);
    const T* v = static_cast<const T*>(p.v);

    // S^T[q][c] = B0[v0 + c][q]
    const float* w0 = p.W0 + (size_t)(l * p.H + h) * p.dq * p.dv;
    for (int i = tid; i < dq * kSimtNv; i += kSimtThreads) {
        const int qi = i / kSimtNv, c = i % kSimtNv;
        float w = 0.0f;
        if (p.W0 && v0 + c < p.dv)
            w = p.w0_transposed ? w0[(size_t)qi * p.dv + v0 + c] : w0[(size_t)(v0 + c) * dq + qi];
        ST[i] = w;
    }

    const int n_ch = (p.T + kSimtChunk - 1) / kSimtChunk;
    for (int ci = 0; ci < n_ch; ++ci) {
        const int t0 = (REV ? n_ch - 1 - ci : ci) * kSimtChunk;
        __syncthreads();
        for (int i = tid; i < kSimtChunk * dq; i += kSimtThreads) {
            const int r = i / dq, c = i % dq, t = t0 + r;
            float a = 0.0f, bb = 0.0f;
            if (t < p.T) {
                a = ld_as_f32(q + tok_off(p.q_str, l, b, t, h) + c);
                bb = ld_as_f32(k + tok_off(p.k_str, l, b, t, h) + c);
            }
            Qs[i] = a;
            Ks[i] = bb;
        }
        for (int i = tid; i < kSimtChunk * kSimtNv; i += kSimtThreads) {
            const int r = i / kSimtNv, c = i % kSimtNv, t = t0 + r;
            float a = 0.0f;
            if (t < p.T && v0 + c < p.dv) a = ld_as_f32(v + tok_off(p.v_str, l, b, t, h) + v0 + c);
            Vs[i] = a;
        }
        __syncthreads();
        // scores of the strictly earlier (REV: later) tokens of this chunk, scaled by -eta
        for (int i = tid; i < kSimtChunk * kSimtChunk; i += kSimtThreads) {
            const int r = i / kSimtChunk, s = i % kSimtChunk;
            float acc = 0.0f;
            if (REV ? s > r : s < r)
                for (int c = 0; c < dq; ++c) acc = fmaf(Qs[r * dq + c], Ks[s * dq + c], acc);
            Sc[r * (kSimtChunk + 1) + s] = -p.eta * acc;
        }
        __syncthreads();
        // outputs: state read plus intra-chunk causal mix
        for (int i = tid; i < kSimtChunk * kSimtNv; i += kSimtThreads) {
            const int r = i / kSimtNv, c = i % kSimtNv, t = t0 + r;
            float acc = 0.0f;
            for (int qi = 0; qi < dq; ++qi) acc = fmaf(Qs[r * dq + qi], ST[qi * kSimtNv + c], acc);
            for (int s = REV ? r + 1 : 0; s < (REV ? kSimtChunk : r); ++s)
                acc = fmaf(Sc[r * (kSimtChunk + 1) + s], Vs[s * kSimtNv + c], acc);
            if (t < p.T && v0 + c < p.dv) {
                const EpiParams& e = p.epi;
                float o = acc;
                if (e.zin)
                    o *= act_df(e.act, ld_as_f32(static_cast<const T*>(e.zin) +
                                                 tok_off(e.z_str, l, b, t, h) + v0 + c));
                st_from_f32(static_cast<T*>(e.out) + tok_off(e.out_str, l, b, t, h) + v0 + c, o);
                if (e.out2)
                    st_from_f32(static_cast<T*>(e.out2) + tok_off(e.out2_str, l, b, t, h) + v0 + c,
                                act_f(e.act, o));
            }
        }
        __syncthreads();
        // state update S^T -= eta * K^T V
        for (int i = tid; i < dq * kSimtNv; i += kSimtThreads) {
            const int qi = i / kSimtNv, c = i % kSimtNv;
            float acc = 0.0f;
            for (int s = 0; s < kSimtChunk; ++s) acc = fmaf(Ks[s * dq + qi], Vs[s * kSimtNv + c], acc);
            ST[i] = fmaf(-p.eta, acc, ST[i]);
        }
    }
}

size_t simt_smem_bytes(int dq) {
    return sizeof(float) * ((size_t)2 * kSimtChunk * dq + kSimtChunk * kSimtNv +
                            kSimtChunk * (kSimtChunk + 1) + (size_t)dq * kSimtNv);
}

template <typename T, bool REV>
static cudaError_t launch_simt_t(const SimtScanParams& p, int grid, size_t smem, cudaStream_t stream) {
    const cudaError_t e = cudaFuncSetAttribute(simt_scan_kernel<T, REV>,
                                               cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    simt_scan_kernel<T, REV><<<grid, kSimtThreads, smem, stream>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_simt_scan(const SimtScanParams& p, bool bf16, bool rev, cudaStream_t stream) {
    const int n_tiles = (p.dv + kSimtNv - 1) / kSimtNv;
    const long long grid = (long long)p.L * p.B * p.H * n_tiles;
    if (grid <= 0 || grid > 0x7FFFFFFF) return cudaErrorInvalidValue;
    const size_t smem = simt_smem_bytes(p.dq);
    if (bf16)
        return rev ? launch_simt_t<__nv_bfloat16, true>(p, (int)grid, smem, stream)
                   : launch_simt_t<__nv_bfloat16, false>(p, (int)grid, smem, stream);
    return rev ? launch_simt_t<float, true>(p, (int)grid, smem, stream)
               : launch_simt_t<float, false>(p, (int)grid, smem, stream);
}

}  // namespace gl
