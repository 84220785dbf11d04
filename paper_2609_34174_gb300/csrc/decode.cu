// decode.cu -- the deployment kernels: one token per unit, the fast weights kept
// between calls as Delta = W - W0 in fp32 (Sec. 3: at deployment the proposal
// network is removed and every map updates from its own costates once the target
// has been scored; Appendix A: the deployed MLP writes its true costates).
//
//   read   y     = (W0 + Delta) x                                 (optional sigma(y))
//   write  g_in  = sigma'(z) (.) (W0 + Delta)^T g                 (optional; before the write)
//          Delta <- alpha Delta - eta g x^T                        (Eq. 2, decay centred at W0)
//
// Both are streaming passes over Delta (fp32, 4 d_out d_in bytes per unit) and
// bound by HBM bandwidth.  Layout choices:
//   * CTA (row tile, batch row) of one (layer, head): the B units that share W0
//     are adjacent in the launch order, so W0 is fetched from HBM about once and
//     served from L2 to the other rows;
//   * every access is a 16-byte piece of a matrix row; a warp covers 32 pieces
//     (512 contiguous bytes) of one row, or several short rows at once;
//   * the write forms the column sums of g_in inside each (row tile, column strip)
//     tile and combines the tiles deterministically: the last CTA of a strip to
//     finish (an arrival counter) adds the partial sums in tile order.  No CTA
//     waits for another.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "scan_common.cuh"

namespace gl {
namespace dec {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
// rows whose loads a lane of the write issues together (without / with the g_in read)
constexpr int kRowBatch = 4;
constexpr int kRowBatchGin = 1;

template <bool BF16>
__device__ __forceinline__ float ld_tok(const void* p, long long i) {
    if constexpr (BF16)
        return __bfloat162float(static_cast<const __nv_bfloat16*>(p)[i]);
    else
        return static_cast<const float*>(p)[i];
}

template <bool BF16>
__device__ __forceinline__ void st_tok(void* p, long long i, float v) {
    if constexpr (BF16)
        static_cast<__nv_bfloat16*>(p)[i] = __float2bfloat16_rn(v);
    else
        static_cast<float*>(p)[i] = v;
}

// Delta streams through once per call: read it with an evict-first hint so that
// W0, which the other batch rows read again, keeps its place in L2.
__device__ __forceinline__ float4 ld_stream(const float4* p) { return __ldcs(p); }

__device__ __forceinline__ float4 f4add(float4 a, float4 b) {
    return make_float4(a.x + b.x, a.y + b.y, a.z + b.z, a.w + b.w);
}

template <bool BF16>
__device__ __forceinline__ float4 ld_x4(const void* x, long long o) {
    if constexpr (BF16) {
        const uint2 r = *reinterpret_cast<const uint2*>(static_cast<const __nv_bfloat16*>(x) + o);
        const float2 a = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&r.x));
        const float2 b = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&r.y));
        return make_float4(a.x, a.y, b.x, b.y);
    } else {
        return *reinterpret_cast<const float4*>(static_cast<const float*>(x) + o);
    }
}

// y = (W0 + Delta) x.  grid = (n_rt * B, L * H).
// A group of `lanes` lanes owns a row; each lane takes CPL pieces of it per
// segment and NR rows at a time, and issues all 2 * NR * CPL loads of W0 and
// Delta (plus its pieces of x) before the first multiply, so that enough bytes
// are in flight to cover the memory latency without staging in shared memory.
template <bool BF16, int CPL, int NR>
__global__ void __launch_bounds__(kThreads) read_kernel(const DecodeParams p) {
    const int b = blockIdx.x % p.B, rt = blockIdx.x / p.B;
    const int lh = blockIdx.y, l = lh / p.H, h = lh - l * p.H;
    const long long u = ((long long)l * p.B + b) * p.H + h;
    const long long xo = tok_off(p.x_s, l, b, 0, h);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int LR = p.lanes, rpw = 32 / LR, sub = lane / LR, cl = lane - sub * LR;
    const size_t mat = (size_t)p.dout * p.cpr;
    const float4* W = reinterpret_cast<const float4*>(p.W0) + (size_t)lh * mat;
    const float4* D = reinterpret_cast<const float4*>(p.delta) + (size_t)u * mat;
    const int r0 = rt * p.rows, r1 = min(p.dout, r0 + p.rows);
    const long long yo = tok_off(p.epi.out_str, l, b, 0, h);
    const long long ao = tok_off(p.epi.out2_str, l, b, 0, h);
    const int seg = LR * CPL;  // pieces of a row per segment
    // the loop bounds depend on the warp only, so every lane reaches the shuffles
    for (int base = r0 + warp * rpw * NR; base < r1; base += kWarps * rpw * NR) {
        float acc[NR];
#pragma unroll
        for (int q = 0; q < NR; ++q) acc[q] = 0.f;
        for (int c0 = cl; c0 - cl < p.cpr; c0 += seg) {
            float4 xv[CPL], w[NR][CPL], dl[NR][CPL];
#pragma unroll
            for (int k = 0; k < CPL; ++k) {
                const int c = c0 + k * LR;
                xv[k] = c < p.cpr ? ld_x4<BF16>(p.x, xo + 4ll * c) : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
                for (int q = 0; q < NR; ++q) {
                    const int row = base + q * rpw + sub;
                    if (c < p.cpr && row < r1) {
                        w[q][k] = __ldg(W + (size_t)row * p.cpr + c);
                        dl[q][k] = ld_stream(D + (size_t)row * p.cpr + c);
                    } else {
                        w[q][k] = make_float4(0.f, 0.f, 0.f, 0.f);
                        dl[q][k] = w[q][k];
                    }
                }
            }
#pragma unroll
            for (int q = 0; q < NR; ++q)
#pragma unroll
                for (int k = 0; k < CPL; ++k) {
                    acc[q] = fmaf(w[q][k].x + dl[q][k].x, xv[k].x, acc[q]);
                    acc[q] = fmaf(w[q][k].y + dl[q][k].y, xv[k].y, acc[q]);
                    acc[q] = fmaf(w[q][k].z + dl[q][k].z, xv[k].z, acc[q]);
                    acc[q] = fmaf(w[q][k].w + dl[q][k].w, xv[k].w, acc[q]);
                }
        }
#pragma unroll
        for (int q = 0; q < NR; ++q) {
            float a = acc[q];
            for (int o = LR >> 1; o > 0; o >>= 1) a += __shfl_xor_sync(0xffffffffu, a, o);
            const int row = base + q * rpw + sub;
            if (cl == 0 && row < r1) {
                st_tok<BF16>(p.epi.out, yo + row, a);
                if (p.epi.out2) st_tok<BF16>(p.epi.out2, ao + row, act_f(p.epi.act, a));
            }
        }
    }
}

// g_in for the four columns of piece c: apply sigma'(z) when fused, store.
template <bool BF16>
__device__ __forceinline__ void store_gin(const DecodeParams& p, int l, int b, int h, int c,
                                          float4 v) {
    const long long oo = tok_off(p.epi.out_str, l, b, 0, h) + 4ll * c;
    float r[4] = {v.x, v.y, v.z, v.w};
    if (p.epi.zin) {
        const long long zo = tok_off(p.epi.z_str, l, b, 0, h) + 4ll * c;
#pragma unroll
        for (int k = 0; k < 4; ++k) r[k] *= act_df(p.epi.act, ld_tok<BF16>(p.epi.zin, zo + k));
    }
#pragma unroll
    for (int k = 0; k < 4; ++k) st_tok<BF16>(p.epi.out, oo + k, r[k]);
}

// grid = (n_rt * n_strips * B, L * H).  A CTA owns rows [r0, r1) and the column
// pieces [32 s, 32 s + 32) of one unit's Delta.
template <bool BF16, bool GIN, int RB>
__global__ void __launch_bounds__(kThreads) write_kernel(const DecodeParams p) {
    __shared__ float4 red[kThreads];
    __shared__ unsigned int s_last;
    int bx = blockIdx.x;
    const int b = bx % p.B;
    bx /= p.B;
    const int s = bx % p.n_strips, rt = bx / p.n_strips;
    const int lh = blockIdx.y, l = lh / p.H, h = lh - l * p.H;
    const long long u = ((long long)l * p.B + b) * p.H + h;

    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int LR = p.lanes, rpw = 32 / LR, sub = lane / LR, cl = lane - sub * LR;
    const int c = s * 32 + cl;  // this lane's 16-byte piece of every row it visits
    const bool col = c < p.cpr;
    float4 xv = make_float4(0.f, 0.f, 0.f, 0.f);
    if (col) {
        const long long xo = tok_off(p.x_s, l, b, 0, h) + 4ll * c;
        xv = make_float4(ld_tok<BF16>(p.x, xo), ld_tok<BF16>(p.x, xo + 1),
                         ld_tok<BF16>(p.x, xo + 2), ld_tok<BF16>(p.x, xo + 3));
    }
    const float eta = p.eta[u];
    const float alpha = p.alpha ? p.alpha[u] : 1.0f;
    const long long go = tok_off(p.g_s, l, b, 0, h);
    const size_t mat = (size_t)p.dout * p.cpr;
    float4* D = reinterpret_cast<float4*>(p.delta) + (size_t)u * mat;
    const float4* W = reinterpret_cast<const float4*>(p.W0) + (size_t)lh * mat;
    const int r0 = rt * p.rows, r1 = min(p.dout, r0 + p.rows);

    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    if (col) {
        // RB rows at a time: every load of the batch is issued before its stores
        const int step = kWarps * rpw;
        for (int row0 = r0 + warp * rpw + sub; row0 < r1; row0 += RB * step) {
            float4 dl[RB], w[RB];
            float gi[RB];
#pragma unroll
            for (int q = 0; q < RB; ++q) {
                const int row = row0 + q * step;
                if (row < r1) {
                    gi[q] = ld_tok<BF16>(p.g, go + row);
                    dl[q] = ld_stream(D + (size_t)row * p.cpr + c);
                    if constexpr (GIN) w[q] = __ldg(W + (size_t)row * p.cpr + c);
                }
            }
#pragma unroll
            for (int q = 0; q < RB; ++q) {
                const int row = row0 + q * step;
                if (row < r1) {
                    if constexpr (GIN) {
                        // the costate read uses the weights before this token's write
                        acc.x = fmaf(gi[q], w[q].x + dl[q].x, acc.x);
                        acc.y = fmaf(gi[q], w[q].y + dl[q].y, acc.y);
                        acc.z = fmaf(gi[q], w[q].z + dl[q].z, acc.z);
                        acc.w = fmaf(gi[q], w[q].w + dl[q].w, acc.w);
                    }
                    const float eg = -eta * gi[q];
                    __stcs(D + (size_t)row * p.cpr + c,
                           make_float4(fmaf(eg, xv.x, alpha * dl[q].x), fmaf(eg, xv.y, alpha * dl[q].y),
                                       fmaf(eg, xv.z, alpha * dl[q].z), fmaf(eg, xv.w, alpha * dl[q].w)));
                }
            }
        }
    }
    if constexpr (!GIN) {
        return;
    } else {
        // column sums of this tile: lanes that share piece c, over warps and sub-rows
        red[threadIdx.x] = acc;
        __syncthreads();
        const int npc = min(32, p.cpr - s * 32);  // pieces in this strip
        const int pc = threadIdx.x;               // piece owned by threads below npc
        float4 sum = make_float4(0.f, 0.f, 0.f, 0.f);
        if (pc < npc) {
            for (int w = 0; w < kWarps; ++w)
                for (int q = 0; q < rpw; ++q) sum = f4add(sum, red[w * 32 + q * LR + pc]);
        }
        if (p.n_rt == 1) {
            if (pc < npc) store_gin<BF16>(p, l, b, h, s * 32 + pc, sum);
            return;
        }
        float4* part = reinterpret_cast<float4*>(p.part);
        if (pc < npc) part[((size_t)u * p.n_rt + rt) * p.cpr + s * 32 + pc] = sum;
        __threadfence();
        __syncthreads();
        if (threadIdx.x == 0) {
            const unsigned int prev = atomicAdd(&p.cnt[(size_t)u * p.n_strips + s], 1u);
            s_last = prev == (unsigned int)(p.n_rt - 1) ? 1u : 0u;
        }
        __syncthreads();
        if (!s_last) return;
        __threadfence();
        // the last tile of this strip adds all partial sums: warp w takes tiles
        // w, w + 8, ...; then the warps are added in order (a fixed order)
        float4 t = make_float4(0.f, 0.f, 0.f, 0.f);
        if (lane < npc) {
            const float4* pp = part + (size_t)u * p.n_rt * p.cpr + s * 32 + lane;
            for (int k = warp; k < p.n_rt; k += kWarps) t = f4add(t, __ldcg(pp + (size_t)k * p.cpr));
        }
        __syncthreads();
        red[threadIdx.x] = t;
        __syncthreads();
        if (pc < npc) {
            float4 v = red[pc];
            for (int w = 1; w < kWarps; ++w) v = f4add(v, red[w * 32 + pc]);
            store_gin<BF16>(p, l, b, h, s * 32 + pc, v);
        }
    }
}

}  // namespace dec

// Pieces per lane per segment (CPL) and rows per lane (NR) of the read, chosen by
// measurement: a lane keeps 8 to 16 loads of W0 and Delta in flight, and the
// register count stays low enough for several CTAs per SM.  cpr < 32 gives one
// piece per lane (lanes >= cpr).
int decode_read_cpl(int cpr, int lanes) {
    if (cpr <= lanes) return 1;
    const int per = (cpr + lanes - 1) / lanes;
    return per >= 4 ? 4 : per >= 2 ? 2 : 1;
}

template <bool BF16>
cudaError_t launch_read_t(const DecodeParams& p, dim3 grid, cudaStream_t stream) {
    switch (decode_read_cpl(p.cpr, p.lanes)) {
    case 1: dec::read_kernel<BF16, 1, 4><<<grid, dec::kThreads, 0, stream>>>(p); break;
    case 2: dec::read_kernel<BF16, 2, 4><<<grid, dec::kThreads, 0, stream>>>(p); break;
    default: dec::read_kernel<BF16, 4, 1><<<grid, dec::kThreads, 0, stream>>>(p); break;
    }
    return cudaGetLastError();
}

cudaError_t launch_decode_read(const DecodeParams& p, bool bf16, cudaStream_t stream) {
    const dim3 grid((unsigned)(p.n_rt * p.B), (unsigned)(p.L * p.H));
    return bf16 ? launch_read_t<true>(p, grid, stream) : launch_read_t<false>(p, grid, stream);
}

cudaError_t launch_decode_write(const DecodeParams& p, bool bf16, bool gin, cudaStream_t stream) {
    const dim3 grid((unsigned)(p.n_rt * p.n_strips * p.B), (unsigned)(p.L * p.H));
    constexpr int rb = dec::kRowBatch, rbg = dec::kRowBatchGin;
    if (bf16) {
        if (gin)
            dec::write_kernel<true, true, rbg><<<grid, dec::kThreads, 0, stream>>>(p);
        else
            dec::write_kernel<true, false, rb><<<grid, dec::kThreads, 0, stream>>>(p);
    } else {
        if (gin)
            dec::write_kernel<false, true, rbg><<<grid, dec::kThreads, 0, stream>>>(p);
        else
            dec::write_kernel<false, false, rb><<<grid, dec::kThreads, 0, stream>>>(p);
    }
    return cudaGetLastError();
}

}  // namespace gl
