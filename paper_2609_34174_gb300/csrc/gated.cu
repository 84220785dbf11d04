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
//   serial_kernel    with alpha_t: the recurrence token by token, exactly as Eq. 2
//                    states it.  Each CTA holds a 64-wide slice of W - W0 and of W0
//                    in shared memory (fp32) for one unit; the forward slices W by
//                    rows (outputs are rows), the costate by columns.  This is also
//                    the token-serial deployment update used for decoding.
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

// ghat'[l,b,t,h,:] = eta_t[l,b,t,h] * ghat[l,b,t,h,:], written contiguous.
template <bool BF16>
__global__ void prescale_kernel(const void* __restrict__ g, TokStr gs, const float* __restrict__ eta,
                                void* __restrict__ out, int L, int B, int T, int H, int w) {
    const long long n = (long long)L * B * T * H * w;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (long long)gridDim.x * blockDim.x) {
        const long long tok = i / w;
        const int f = (int)(i - tok * w);
        const int h = (int)(tok % H);
        long long r = tok / H;
        const int t = (int)(r % T);
        r /= T;
        const int b = (int)(r % B);
        const int l = (int)(r / B);
        const long long src = (long long)l * gs.s[0] + (long long)b * gs.s[1] + (long long)t * gs.s[2] +
                              (long long)h * gs.s[3] + f;
        st<BF16>(out, i, eta[tok] * ld<BF16>(g, src));
    }
}

// One CTA: unit (l, b, h) and a tile of 64 output indices.
//   forward  (COSTATE = false): outputs are rows m of W [m][d]; q = x (length d),
//            a = ghat (row-indexed), bvec = x (column-indexed)
//   costate  (COSTATE = true):  outputs are columns d of W; q = g_out (length m),
//            a = x (column-indexed), bvec = ghat (row-indexed)
// Held per CTA (fp32): Wt[i][j] = W0 entry and Dt[i][j] = (W_t - W0) entry for output
// i of the tile and input j (J = d forward, m costate).
template <bool COSTATE, bool BF16>
__global__ void __launch_bounds__(kThreads)
    serial_kernel(GatedParams p) {
    extern __shared__ float sm[];
    const int J = COSTATE ? p.dout : p.din;   // inputs of the read
    const int NO = COSTATE ? p.din : p.dout;  // outputs of the read
    float* W0t = sm;                          // [64][J]
    float* Dt = W0t + kTile * J;              // [64][J]
    float* qv = Dt + kTile * J;               // [J]  read vector
    float* bv = qv + J;                       // [J]  write vector on the input side
    float* av = bv + J;                       // [64] write vector on the output side
    float* gate = av + kTile;                 // [2]  eta_t, alpha_t

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
        W0t[e] = w;
        Dt[e] = 0.0f;
    }
    const int i_own = threadIdx.x >> 2;  // output index of this thread's group of 4
    const int part = threadIdx.x & 3;
    for (int t = 0; t < p.T; ++t) {
        const long long tok = ((long long)l * p.B + b) * p.T * p.H + (long long)t * p.H + h;
        // stage this token's vectors
        const long long xo = tok_off(p.x_s, l, b, t, h);
        const long long go = tok_off(p.g_s, l, b, t, h);
        const long long qo = tok_off(p.q_s, l, b, t, h);
        for (int j = threadIdx.x; j < J; j += kThreads) {
            qv[j] = ld<BF16>(p.q, qo + j);
            bv[j] = COSTATE ? ld<BF16>(p.g, go + j) : ld<BF16>(p.x, xo + j);
        }
        for (int i = threadIdx.x; i < kTile; i += kThreads) {
            const int o = o0 + i;
            av[i] = o < NO ? (COSTATE ? ld<BF16>(p.x, xo + o) : ld<BF16>(p.g, go + o)) : 0.0f;
        }
        if (threadIdx.x == 0) {
            gate[0] = p.eta[tok];
            gate[1] = p.alpha ? p.alpha[tok] : 1.0f;
        }
        __syncthreads();
        // read before write: out_i = sum_j (W0 + D)[i][j] q_j
        float acc = 0.0f;
        const float* w_row = W0t + i_own * J;
        const float* d_row = Dt + i_own * J;
        for (int j = part; j < J; j += 4) acc += (w_row[j] + d_row[j]) * qv[j];
        acc += __shfl_xor_sync(0xffffffffu, acc, 1);
        acc += __shfl_xor_sync(0xffffffffu, acc, 2);
        const int o = o0 + i_own;
        if (part == 0 && o < NO) {
            const EpiParams& e = p.epi;
            const long long oo = tok_off(e.out_str, l, b, t, h) + o;
            float v = acc;
            if (e.zin) {
                const long long zo = tok_off(e.z_str, l, b, t, h) + o;
                v *= act_df(e.act, ld<BF16>(e.zin, zo));
            }
            st<BF16>(e.out, oo, v);
            if (e.out2) st<BF16>(e.out2, tok_off(e.out2_str, l, b, t, h) + o, act_f(e.act, acc));
        }
        // every read of D for this token is done before the write
        __syncthreads();
        // write: D = alpha D - eta a b^T
        const float eta = gate[0], alpha = gate[1];
        for (int e = threadIdx.x; e < kTile * J; e += kThreads) {
            const int i = e / J, j = e - i * J;
            Dt[e] = alpha * Dt[e] - eta * av[i] * bv[j];
        }
        __syncthreads();
    }
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
    return sizeof(float) * ((size_t)2 * gated::kTile * J + 2 * (size_t)J + gated::kTile + 2);
}

cudaError_t launch_gated_serial(const GatedParams& p, bool costate, bool bf16, cudaStream_t stream) {
    const int NO = costate ? p.din : p.dout;
    const int tiles = (NO + gated::kTile - 1) / gated::kTile;
    const long long blocks = (long long)p.L * p.B * p.H * tiles;
    const size_t smem = gated_serial_smem(p.din, p.dout, costate);
    if (blocks <= 0) return cudaSuccess;
    if (costate)
        return bf16 ? gated::launch_serial<true, true>(p, (int)blocks, smem, stream)
                    : gated::launch_serial<true, false>(p, (int)blocks, smem, stream);
    return bf16 ? gated::launch_serial<false, true>(p, (int)blocks, smem, stream)
                : gated::launch_serial<false, false>(p, (int)blocks, smem, stream);
}

cudaError_t launch_gated_prescale(const void* g, const TokStr& gs, const float* eta, void* out, int L,
                                  int B, int T, int H, int w, bool bf16, cudaStream_t stream) {
    const long long n = (long long)L * B * T * H * w;
    if (n <= 0) return cudaSuccess;
    long long blocks = (n + 255) / 256;
    if (blocks > 152 * 16) blocks = 152 * 16;
    if (bf16)
        gated::prescale_kernel<true><<<(int)blocks, 256, 0, stream>>>(g, gs, eta, out, L, B, T, H, w);
    else
        gated::prescale_kernel<false><<<(int)blocks, 256, 0, stream>>>(g, gs, eta, out, L, B, T, H, w);
    return cudaGetLastError();
}

}  // namespace gl
