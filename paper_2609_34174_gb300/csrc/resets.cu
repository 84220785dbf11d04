// resets.cu -- gate arrays for packed documents.
//
// Sequences packed from several documents reset the fast state at every
// document start: a read excludes every write made before the most recent
// document start (Appendix C, the scan reads; Appendix E, packed rows).  In the
// gates of Eq. 2,
//
//     W_{t+1} = W0 + alpha_t (W_t - W0) - eta_t ghat_t x_t^T,
//
// a document starting at token s > 0 is alpha_{s-1} = 0 and eta_{s-1} = 0: the
// previous document's fast weights go back to W0 and its last write, which no
// read of that document sees, is dropped, so the read at s sees W0.  This file
// folds per-token document starts into the gate arrays; the gated scans then run
// unchanged.
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>

#include "../../include/gradlev.h"

namespace {

constexpr int kThreads = 256;

// One thread per gate entry (l, b, t, h) of the [L][B][T][H] arrays, grid-stride.
__global__ void document_gates_kernel(const uint8_t* __restrict__ doc_start, float eta,
                                      const float* eta_t, const float* alpha_t, float* eta_out,
                                      float* alpha_out, long long n, int B, int T, int H) {
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n;
         i += (long long)gridDim.x * blockDim.x) {
        const long long th = i / H;            // (l, b, t) index
        const int t = (int)(th % T);
        const int b = (int)((th / T) % B);
        const bool last = t + 1 < T && doc_start[(long long)b * T + t + 1] != 0;
        const float e = eta_t ? eta_t[i] : eta;
        const float a = alpha_t ? alpha_t[i] : 1.0f;
        eta_out[i] = last ? 0.0f : e;
        alpha_out[i] = last ? 0.0f : a;
    }
}

bool aligned4(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 3u) == 0; }

}  // namespace

extern "C" {

int gradlev_document_gates(const gradlev_desc* desc, const uint8_t* doc_start, float eta,
                           const float* eta_t, const float* alpha_t, float* eta_out,
                           float* alpha_out, gradlev_stream_t stream) {
    if (!desc) return GRADLEV_ERR_INVALID_ARG;
    const gradlev_desc& d = *desc;
    if (d.L < 0 || d.B < 0 || d.T < 0 || d.H < 0 || d.reserved != 0) return GRADLEV_ERR_INVALID_ARG;
    const long long n = (long long)d.L * d.B * d.T * d.H;
    if (n == 0) return GRADLEV_OK;
    if (!doc_start || !eta_out || !alpha_out) return GRADLEV_ERR_INVALID_ARG;
    if (!eta_t && !std::isfinite(eta)) return GRADLEV_ERR_INVALID_ARG;
    const void* f32[4] = {eta_t, alpha_t, eta_out, alpha_out};
    for (const void* p : f32)
        if (p && !aligned4(p)) return GRADLEV_ERR_INVALID_ARG;
    long long blocks = (n + kThreads - 1) / kThreads;
    if (blocks > 152 * 8) blocks = 152 * 8;
    document_gates_kernel<<<(int)blocks, kThreads, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
        doc_start, eta, eta_t, alpha_t, eta_out, alpha_out, n, d.B, d.T, d.H);
    return cudaGetLastError() == cudaSuccess ? GRADLEV_OK : GRADLEV_ERR_CUDA;
}

}  // extern "C"
