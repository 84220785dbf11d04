// scan_common.cuh -- definitions shared by the scan kernels and the host layer.
//
// Both GradLev scans are one computation (Sec. 3, Eqs. 3-4; Appendix C):
//
//     o_t = B0 q_t - eta * sum_{s<t} (k_s . q_t) v_s,
//
// an exclusive causal "linear attention" with an additive base matrix B0:
//   forward scan  (Eq. 3): q = k = x, v = ghat, B0 = W0      (dq = d_in,  dv = d_out)
//   costate scan  (Eq. 4): q = g_out, k = ghat, v = x, B0 = W0^T (dq = d_out, dv = d_in)
// The running state is S_t^T = B0^T - eta * sum_{s<t} k_s v_s^T  (dq x dv).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace gl {

enum Act : int { ACT_NONE = 0, ACT_GELU_TANH = 1, ACT_GELU_ERF = 2, ACT_TANH = 3 };

// sigma and sigma' in fp32 from their formulas (tanh-approximate GELU, exact
// GELU, tanh), calling CUDA's tanhf / erff / expf.
__device__ __forceinline__ float act_f(int act, float z) {
    const float k0 = 0.7978845608028654f;  // sqrt(2/pi)
    switch (act) {
    case ACT_GELU_TANH: return 0.5f * z * (1.0f + tanhf(k0 * (z + 0.044715f * z * z * z)));
    case ACT_GELU_ERF: return 0.5f * z * (1.0f + erff(z * 0.7071067811865476f));
    case ACT_TANH: return tanhf(z);
    default: return z;
    }
}

__device__ __forceinline__ float act_df(int act, float z) {
    const float k0 = 0.7978845608028654f;
    switch (act) {
    case ACT_GELU_TANH: {
        float th = tanhf(k0 * (z + 0.044715f * z * z * z));
        float du = k0 * (1.0f + 3.0f * 0.044715f * z * z);
        return 0.5f * (1.0f + th) + 0.5f * z * (1.0f - th * th) * du;
    }
    case ACT_GELU_ERF: {
        float cdf = 0.5f * (1.0f + erff(z * 0.7071067811865476f));
        float pdf = expf(-0.5f * z * z) * 0.3989422804014327f;
        return cdf + z * pdf;
    }
    case ACT_TANH: {
        float th = tanhf(z);
        return 1.0f - th * th;
    }
    default: return 1.0f;
    }
}

// Element offset of token (l, b, t, h) in a [L][B][T][H][w] tensor with the
// given element strides of (L, B, T, H).
__host__ __device__ __forceinline__ long long tok_off(const long long (&s)[4], int l, int b, int t,
                                                      int h) {
    return (long long)l * s[0] + (long long)b * s[1] + (long long)t * s[2] + (long long)h * s[3];
}

// Epilogue outputs shared by all kernels.
struct EpiParams {
    void* out;            // [L][B][T][H][dv], the scan result (bf16 or f32)
    long long out_str[4];
    void* out2;           // optional sigma(out) (forward MLP fusion), same layout
    long long out2_str[4];
    const void* zin;      // optional preactivation: out = sigma'(z) (.) result (costate)
    long long z_str[4];
    int act;
    // optional per-token dot (suffix read only): dot_out[l][b][t][h] +=
    // dot_scale * (result row . dot_a row), fp32 [L][B][T][H] contiguous
    const void* dot_a;
    long long dot_a_str[4];
    float* dot_out;
    float dot_scale;
    // optional consistency term (fused pass, costate read): cons_out[l][b][t][h] =
    // cons_scale * ||cons_p row - result row||^2, fp32 [L][B][T][H] contiguous
    const void* cons_p;
    long long cons_str[4];
    float* cons_out;
    float cons_scale;
};

// Parameters of the tensor-core scan kernel (bf16, dq in {64, 128}, dv % 64 == 0).
struct TcScanParams {
    int L, B, T, H;
    int dq, dv;
    int n_tiles;          // dv / 64 output tiles per unit
    int seg_len;          // tokens per segment (multiple of 128)
    int n_seg;            // segments per (unit, tile)
    int n_items;          // units * n_tiles * n_seg
    int n_ut;             // units * n_tiles: items per segment index (segment-major order)
    float eta;
    // State units of the chunk kernel: lam = -eta (1 when eta = 0), inv_lam = 1 / lam,
    // mu = -eta / lam (1, or 0 when eta = 0).
    float lam, inv_lam, mu;
    int w0_transposed;    // 0: B0 = W0 ([dv][dq], forward); 1: B0 = W0^T (W0 is [dq][dv])
    const float* W0;      // [L][H][rows][cols] fp32 contiguous
    EpiParams epi;
    unsigned int* ctrl;   // [0] work ticket, [1] error bits
    unsigned int* flags;  // [n_items] look-back status: 0 none, 1 aggregate, 2 inclusive
    unsigned long long lookback_limit_ns;  // bound on a look-back wait (4 s)
    int test_skip_publish;  // failure tests only: this item never publishes (-1: none)
    float* agg;           // [n_items][dq][64] segment aggregate  sum_s k_s v_s^T
    float* incl;          // [n_items][dq][64] inclusive prefix of the aggregates
    // retention kernel only: per-token gates, fp32 [L][B][T][H] contiguous, and the
    // alpha product of each segment (aggregate pass, [n_items])
    const float* g_eta;
    const float* g_alpha;  // null: alpha = 1
    float* seg_a;
};

// Parameters of the wide-layer passes (bf16, dq % 128 == 0, dv % 64 == 0): the
// scan split at segment boundaries into three GEMM-shaped passes.
struct SegGemmParams {
    int L, B, T, H;
    int dq, dv;
    int seg_len;             // Ls, tokens per segment (multiple of 128)
    int n_seg;               // segments per unit
    int n_tiles;             // output tiles of the pass being launched
    float eta;
    int w0_transposed;       // as in TcScanParams
    const float* W0;
    __nv_bfloat16* sbuf;     // [U][n_seg][dq][dv]  S_k^T at every segment start
    __nv_bfloat16* pbuf;     // [U][n_seg][Ls][Ls]  -eta * strict_lower(Q_k K_k^T)
    EpiParams epi;
    unsigned int* ctrl;      // [1] error bits
};

// Parameters of the fp32 SIMT scan kernel.
struct SimtScanParams {
    int L, B, T, H;
    int dq, dv;
    float eta;
    int w0_transposed;
    const float* W0;
    const void* q; long long q_str[4];
    const void* k; long long k_str[4];
    const void* v; long long v_str[4];
    EpiParams epi;
};

// Element strides of (L, B, T, H) of a token tensor.
struct TokStr {
    long long s[4];
};

// Parameters of the gated token-serial kernel (gated.cu).
struct GatedParams {
    int L, B, T, H, din, dout;
    const float* W0;       // [L][H][dout][din]
    const float* eta;      // [L][B][T][H] per-token step sizes
    const float* alpha;    // [L][B][T][H] retention, or null (= 1)
    const void* x; long long x_s[4];   // layer inputs (the writes' right factor)
    const void* g; long long g_s[4];   // proposals ghat (the writes' left factor)
    const void* q; long long q_s[4];   // read vector: x (forward) or g_out (costate)
    EpiParams epi;
};

// Parameters of the deployment kernels (decode.cu): one token per unit, fast
// weights held as Delta = W - W0 in fp32 between calls (Sec. 3, deployment).
struct DecodeParams {
    int L, B, H;
    int din, dout;         // columns (d_in) and rows (d_out) of every matrix
    int cpr;               // din / 4: 16-byte pieces per matrix row
    int lanes;             // lanes sharing one row: 32, or the power of two >= cpr below 32
    int rows;              // matrix rows per CTA tile
    int n_rt;              // row tiles per unit
    int n_strips;          // column strips of 32 pieces (write kernel)
    const float* W0;       // [L][H][dout][din]
    float* delta;          // [L][B][H][dout][din]
    const void* x; long long x_s[4];   // [L][B][1][H][din]
    const void* g; long long g_s[4];   // [L][B][1][H][dout] (write: the true costate)
    const float* eta;      // [L][B][H] (write)
    const float* alpha;    // [L][B][H] or null (write)
    EpiParams epi;         // read: out = y, out2 = sigma(y); write: out = g_in, zin = z
    float* part;           // write with g_in over several row tiles: [U][n_rt][din]
    unsigned int* cnt;     // ... and its arrival counters [U][n_strips], zero on entry
};

// Error bits written to ctrl[1].
constexpr unsigned int kErrWaitTimeout = 1u;
constexpr unsigned int kErrLookbackTimeout = 2u;

}  // namespace gl
