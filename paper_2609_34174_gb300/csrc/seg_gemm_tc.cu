// seg_gemm_tc.cu -- the scans for wide layers (hundreds to thousands of features,
// e.g. the 512 -> 2048 -> 512 MLP of Appendix A) as three tensor-core passes over
// segments of the sequence.
//
// At these widths the running state S^T (dq x dv fp32: 4 MB at 512 x 2048) does
// not fit one SM, so the chunk recurrence of scan_tc.cu gives way to the
// associativity of the additive write scan (Sec. 3, Eq. 2; Appendix C).  Each
// unit's tokens are cut into segments of Ls tokens; with Q_k, K_k, V_k the rows
// of segment k,
//
//   state pass   S_k^T = B0^T - eta * sum_{j<k} K_j^T V_j            (bf16, dq x dv)
//   score pass   P_k   = -eta * strict_lower(Q_k K_k^T)             (bf16, Ls x Ls)
//   output pass  O_k   = Q_k S_k^T + P_k V_k     (+ sigma / sigma' fused on the way out)
//
// which is Eq. 3 (forward: q = k = x, v = g_hat, B0 = W0) and Eq. 4 (costate:
// q = g_out, k = g_hat, v = x, B0 = W0^T) with the exclusive sum over s < t split
// at the segment start.  Each pass is a persistent warp-specialised kernel: a TMA
// producer warp, a tcgen05.mma issuer warp that owns the tensor memory, and eight
// epilogue warps that read the fp32 accumulator out of TMEM (warp w reads lanes
// 32*(w%4)..+31; warps 2-5 take the left half of the tile's columns and warps
// 6-9 the right half).
//
// Operand tiles are 128B-swizzled [rows][64 bf16] atoms written by TMA:
//   K-major  (A = Q or P; B = K in the score pass): 128 rows x 64 K, 16 KB
//   MN-major (A = K^T in the state pass; B = V, S^T): 64 K-rows x 64 M/N per atom,
//            8 KB, atoms of one operand 8 KB apart (the descriptor's LBO).
#include <cuda.h>

#include "scan_common.cuh"
#include "sm103_ptx.cuh"

namespace gl {
namespace sg {

constexpr int kWarps = 10;   // producer, MMA issuer, eight epilogue warps
constexpr int kEpiWarps = 8;
constexpr int kThreads = kWarps * 32;
constexpr int kStages = 4;
constexpr int kAtom = 8192;                         // [64 rows][64 bf16]
constexpr int kTileA = 16384;                       // A of one K-block
constexpr int kStageBytes = kTileA + 4 * kAtom;     // A + B up to 256 wide
constexpr int kBarOff = kStages * kStageBytes;
constexpr int kSmemBytes = kBarOff + 1024 + 1024;   // barriers + alignment slack
constexpr uint32_t kTmemCols = 512;                 // two accumulators of up to 256 columns
static_assert(kSmemBytes <= 232448, "shared memory budget exceeded");

// K-step offsets in descriptor units (16 B): a K-major step moves 32 B along the
// swizzled 128-byte row; an MN-major step moves 16 K-rows (2 KB).
__host__ __device__ constexpr uint32_t kstep(int kk) { return (uint32_t)((kk * 32) >> 4); }
__host__ __device__ constexpr uint32_t mnstep(int kk) { return (uint32_t)((kk * 2048) >> 4); }

enum Mode : int { STATE = 0, SCORE = 1, OUT = 2 };

struct Tile {
    int u, l, b, h;   // unit and its (layer, batch, head)
    int k;            // segment
    int r, c;         // row block (128 query tokens) / column block of the score tile
    int mi, ni;       // state rows block (128 of dq) / output column block (BN of dv)
};

template <int MODE, int BN>
__device__ __forceinline__ Tile decode(int tile, const SegGemmParams& p) {
    Tile t;
    t.k = t.r = t.c = t.mi = t.ni = 0;
    const int R = p.seg_len / 128;
    if (MODE == STATE) {
        const int nN = p.dv / BN, nM = p.dq / 128;
        t.ni = tile % nN;
        const int q = tile / nN;
        t.mi = q % nM;
        t.u = q / nM;
    } else if (MODE == SCORE) {
        const int NL = R * (R + 1) / 2;  // lower-triangular blocks incl. the diagonal
        const int li = tile % NL;
        const int q = tile / NL;
        t.k = q % p.n_seg;
        t.u = q / p.n_seg;
        int rr = 0;
        while ((rr + 1) * (rr + 2) / 2 <= li) ++rr;
        t.r = rr;
        t.c = li - rr * (rr + 1) / 2;
    } else {
        const int nN = p.dv / BN;
        t.ni = tile % nN;
        int q = tile / nN;
        t.r = q % R;
        q /= R;
        t.k = q % p.n_seg;
        t.u = q / p.n_seg;
    }
    t.h = t.u % p.H;
    const int lb = t.u / p.H;
    t.b = lb % p.B;
    t.l = lb / p.B;
    return t;
}

__device__ __forceinline__ void raise_error(const SegGemmParams& p, volatile int* abort_flag) {
    atomicOr(p.ctrl + 1, kErrWaitTimeout);
    if (abort_flag) *abort_flag = 1;
}

__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag) {
    const int lane = threadIdx.x & 31;
    int ok = 1;
    if (lane == 0) ok = mbar_wait(bar, parity, abort_flag) ? 1 : 0;
    ok = __shfl_sync(0xffffffffu, ok, 0);
    __syncwarp();
    return ok != 0;
}

__device__ __forceinline__ void drain(uint64_t* bar, uint32_t parity) {
    const uint64_t t0 = globaltimer_ns();
    while (!mbar_try_wait(bar, parity)) {
        if (globaltimer_ns() - t0 > 200000000ull) break;  // 0.2 s
    }
}

__device__ __forceinline__ void store_bf16x32(__nv_bfloat16* dst, const float (&v)[32]) {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        uint4 w;
        w.x = pack_bf16x2(v[8 * q + 0], v[8 * q + 1]);
        w.y = pack_bf16x2(v[8 * q + 2], v[8 * q + 3]);
        w.z = pack_bf16x2(v[8 * q + 4], v[8 * q + 5]);
        w.w = pack_bf16x2(v[8 * q + 6], v[8 * q + 7]);
        *reinterpret_cast<uint4*>(dst + 8 * q) = w;
    }
}

// One persistent pass.  Tensor maps by mode:
//   STATE  a = K (64-token box), b = V (64-token box)
//   SCORE  a = Q (128-token box), b = K (128-token box)
//   OUT    a = Q (128-token box), b = S^T workspace, a2 = P workspace, b2 = V (64-token box)
template <int MODE, int BN>
__global__ void __launch_bounds__(kThreads, 1)
    seg_gemm_kernel(const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_b,
                    const __grid_constant__ CUtensorMap tm_a2,
                    const __grid_constant__ CUtensorMap tm_b2, const SegGemmParams p) {
    constexpr int NS = kStages;
    constexpr int NB = (MODE == SCORE) ? 2 : BN / 64;  // B atoms per stage
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~static_cast<uintptr_t>(1023));
    const uint32_t sbase = smem_u32(smem);
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kBarOff);
    uint64_t* full = bars;           // [NS]
    uint64_t* empty = bars + 8;      // [NS]
    uint64_t* acc_full = bars + 16;  // [2]
    uint64_t* acc_free = bars + 18;  // [2]
    int* misc = reinterpret_cast<int*>(bars + 24);
    volatile int* abort_flag = misc;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(misc + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int i = 0; i < NS; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&acc_full[i], 1);
            mbar_init(&acc_free[i], kEpiWarps);
        }
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, kTmemCols);
        tmem_relinquish();
        tc_fence_before();
    }
    if (warp == 0 && lane == 0) {
        prefetch_tmap(&tm_a);
        prefetch_tmap(&tm_b);
        if (MODE == OUT) {
            prefetch_tmap(&tm_a2);
            prefetch_tmap(&tm_b2);
        }
    }
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    const int Ls = p.seg_len;

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            uint32_t n = 0;
            bool ok = true;
            auto stage = [&](uint32_t bytes) -> int {
                const int s = n % NS;
                if (!mbar_wait(&empty[s], ((n / NS) & 1) ^ 1, abort_flag)) {
                    raise_error(p, abort_flag);
                    ok = false;
                    return -1;
                }
                mbar_arrive_expect_tx(&full[s], bytes);
                ++n;
                return s;
            };
            for (int tile = blockIdx.x; tile < p.n_tiles && ok; tile += gridDim.x) {
                const Tile t = decode<MODE, BN>(tile, p);
                if (MODE == STATE) {
                    for (int k = 0; k + 1 < p.n_seg && ok; ++k) {
                        for (int kb = 0; kb < Ls / 64 && ok; ++kb) {
                            const int s = stage(2 * kAtom + NB * kAtom);
                            if (s < 0) break;
                            uint8_t* st = smem + s * kStageBytes;
                            const int t0 = k * Ls + kb * 64;
                            tma_load_5d(st, &tm_a, &full[s], t.mi * 128, t.h, t0, t.b, t.l);
                            tma_load_5d(st + kAtom, &tm_a, &full[s], t.mi * 128 + 64, t.h, t0, t.b, t.l);
#pragma unroll
                            for (int j = 0; j < NB; ++j)
                                tma_load_5d(st + kTileA + j * kAtom, &tm_b, &full[s], t.ni * BN + j * 64,
                                            t.h, t0, t.b, t.l);
                        }
                    }
                } else if (MODE == SCORE) {
                    for (int kb = 0; kb < p.dq / 64 && ok; ++kb) {
                        const int s = stage(2 * kTileA);
                        if (s < 0) break;
                        uint8_t* st = smem + s * kStageBytes;
                        tma_load_5d(st, &tm_a, &full[s], kb * 64, t.h, t.k * Ls + t.r * 128, t.b, t.l);
                        tma_load_5d(st + kTileA, &tm_b, &full[s], kb * 64, t.h, t.k * Ls + t.c * 128,
                                    t.b, t.l);
                    }
                } else {
                    const int us = t.u * p.n_seg + t.k;
                    for (int kb = 0; kb < p.dq / 64 && ok; ++kb) {
                        const int s = stage(kTileA + NB * kAtom);
                        if (s < 0) break;
                        uint8_t* st = smem + s * kStageBytes;
                        tma_load_5d(st, &tm_a, &full[s], kb * 64, t.h, t.k * Ls + t.r * 128, t.b, t.l);
#pragma unroll
                        for (int j = 0; j < NB; ++j)
                            tma_load_3d(st + kTileA + j * kAtom, &tm_b, &full[s], t.ni * BN + j * 64,
                                        kb * 64, us);
                    }
                    for (int sb = 0; sb < 2 * (t.r + 1) && ok; ++sb) {
                        const int s = stage(kTileA + NB * kAtom);
                        if (s < 0) break;
                        uint8_t* st = smem + s * kStageBytes;
                        tma_load_3d(st, &tm_a2, &full[s], sb * 64, t.r * 128, us);
#pragma unroll
                        for (int j = 0; j < NB; ++j)
                            tma_load_5d(st + kTileA + j * kAtom, &tm_b2, &full[s], t.ni * BN + j * 64,
                                        t.h, t.k * Ls + sb * 64, t.b, t.l);
                    }
                }
            }
            // Every issued load lands before the CTA may exit.
            if (*abort_flag) {
                for (int s = 0; s < NS; ++s) {
                    if (n > (uint32_t)s) {
                        const uint32_t last = ((n - 1 - s) / NS) * NS + s;
                        drain(&full[s], (last / NS) & 1);
                    }
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------- MMA issuer
        if (lane == 0) {
            constexpr uint32_t ID_ST = idesc_bf16(128, BN, true, true);    // K^T V
            constexpr uint32_t ID_SC = idesc_bf16(128, 128, false, false); // Q K^T
            constexpr uint32_t ID_OUT = idesc_bf16(128, BN, false, true);  // Q S^T, P V
            uint32_t n = 0, g = 0;
            int it = 0;
            bool ok = true;
            // One K-block of 64: four K=16 MMAs from stage n, then release the stage.
            auto kblock = [&](uint32_t dcol, uint32_t idesc, bool a_mn, bool b_mn,
                              bool first) -> bool {
                const int s = n % NS;
                if (!mbar_wait(&full[s], (n / NS) & 1, abort_flag)) return false;
                tc_fence_after();
                const uint32_t st = sbase + s * kStageBytes;
                const uint32_t a_lo = sdesc_lo(st, a_mn ? kAtom : 16);
                const uint32_t b_lo = sdesc_lo(st + kTileA, b_mn ? kAtom : 16);
#pragma unroll
                for (int kk = 0; kk < 4; ++kk)
                    mma_bf16_ss(tmem + dcol, sdesc_from_lo(a_lo + (a_mn ? mnstep(kk) : kstep(kk))),
                                sdesc_from_lo(b_lo + (b_mn ? mnstep(kk) : kstep(kk))), idesc,
                                (first && kk == 0) ? 0u : 1u);
                mma_commit(&empty[s]);
                ++n;
                return true;
            };
            for (int tile = blockIdx.x; tile < p.n_tiles && ok; tile += gridDim.x, ++it) {
                const Tile t = decode<MODE, BN>(tile, p);
                if (MODE == STATE) {
                    // One accumulator carries the running sum across the segments; each
                    // segment waits until the epilogue has read the previous value.
                    for (int k = 0; k + 1 < p.n_seg && ok; ++k, ++g) {
                        if (!(ok = mbar_wait(&acc_free[0], (g & 1) ^ 1, abort_flag))) break;
                        tc_fence_after();
                        for (int kb = 0; kb < Ls / 64 && ok; ++kb)
                            ok = kblock(0, ID_ST, true, true, k == 0 && kb == 0);
                        if (ok) mma_commit(&acc_full[0]);
                    }
                } else {
                    const uint32_t buf = it & 1;
                    if (!(ok = mbar_wait(&acc_free[buf], ((it >> 1) & 1) ^ 1, abort_flag))) break;
                    tc_fence_after();
                    const uint32_t dcol = buf * 256;
                    if (MODE == SCORE) {
                        for (int kb = 0; kb < p.dq / 64 && ok; ++kb)
                            ok = kblock(dcol, ID_SC, false, false, kb == 0);
                    } else {
                        for (int kb = 0; kb < p.dq / 64 && ok; ++kb)
                            ok = kblock(dcol, ID_OUT, false, true, kb == 0);
                        for (int sb = 0; sb < 2 * (t.r + 1) && ok; ++sb)
                            ok = kblock(dcol, ID_OUT, false, true, false);
                    }
                    if (ok) mma_commit(&acc_full[buf]);
                }
            }
            if (!ok) raise_error(p, abort_flag);
        }
    } else {
        // --------------------------------------------------------- epilogue
        const int q4 = warp & 3;
        const int half = (warp - 2) >> 2;
        const int row = q4 * 32 + lane;
        const uint32_t lane_off = static_cast<uint32_t>(q4 * 32) << 16;
        const float eta = p.eta;
        constexpr int W = (MODE == SCORE) ? 128 : BN;  // accumulator columns of a tile
        constexpr int HW = W / 2;                       // columns this warp handles
        const int cb = half * HW;                       // first of them
        uint32_t e = 0;
        int it = 0;
        for (int tile = blockIdx.x; tile < p.n_tiles; tile += gridDim.x, ++it) {
            const Tile t = decode<MODE, BN>(tile, p);
            bool ok = true;
            if (MODE == STATE) {
                // B0^T for this tile goes to TMEM columns 256.. once (the accumulator
                // uses columns 0..BN-1), and is also segment 0's starting state.
                const int dq_row = t.mi * 128 + row;
                const float* w0 = p.W0 + (size_t)(t.l * p.H + t.h) * p.dq * p.dv;
                const uint32_t b0_t = tmem + lane_off + 256;
                __nv_bfloat16* dst0 = p.sbuf + ((size_t)(t.u * p.n_seg) * p.dq + dq_row) * p.dv + t.ni * BN;
#pragma unroll 1
                for (int c0 = cb; c0 < cb + HW; c0 += 32) {
                    float a[32];
                    const int col0 = t.ni * BN + c0;
                    if (p.w0_transposed) {
                        const float* src = w0 + (size_t)dq_row * p.dv + col0;  // W0 [dq][dv]
#pragma unroll
                        for (int j = 0; j < 32; j += 4) {
                            const float4 b = *reinterpret_cast<const float4*>(src + j);
                            a[j] = b.x;
                            a[j + 1] = b.y;
                            a[j + 2] = b.z;
                            a[j + 3] = b.w;
                        }
                    } else {
#pragma unroll
                        for (int j = 0; j < 32; ++j)  // W0 [dv][dq]: column dq_row
                            a[j] = w0[(size_t)(col0 + j) * p.dq + dq_row];
                    }
                    uint32_t r[32];
#pragma unroll
                    for (int j = 0; j < 32; ++j) r[j] = __float_as_uint(a[j]);
                    tmem_st32_async(b0_t + c0, r);
                    store_bf16x32(dst0 + c0, a);
                }
                tmem_wait_st();
                for (int k = 1; k < p.n_seg; ++k) {
                    if (!warp_wait(&acc_full[0], e & 1, abort_flag)) {
                        raise_error(p, abort_flag);
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    __nv_bfloat16* dst = p.sbuf + ((size_t)(t.u * p.n_seg + k) * p.dq + dq_row) * p.dv +
                                         t.ni * BN;
#pragma unroll 1
                    for (int c0 = cb; c0 < cb + HW; c0 += 32) {
                        float a[32], b[32];
                        tmem_ld32(tmem + lane_off + c0, a);
                        if (c0 + 32 == cb + HW) {
                            // last accumulator read of this segment: let the next one start
                            tc_fence_before();
                            __syncwarp();
                            if (lane == 0) mbar_arrive(&acc_free[0]);
                        }
                        tmem_ld32(b0_t + c0, b);
#pragma unroll
                        for (int j = 0; j < 32; ++j) a[j] = b[j] - eta * a[j];
                        store_bf16x32(dst + c0, a);
                    }
                    ++e;
                }
            } else {
                const uint32_t buf = it & 1;
                if (!warp_wait(&acc_full[buf], (it >> 1) & 1, abort_flag)) {
                    raise_error(p, abort_flag);
                    break;
                }
                tc_fence_after();
                const uint32_t acc = tmem + lane_off + buf * 256;
                if (MODE == SCORE) {
                    const int t_seg = t.r * 128 + row;
                    __nv_bfloat16* dst = p.pbuf + ((size_t)(t.u * p.n_seg + t.k) * Ls + t_seg) * Ls +
                                         t.c * 128;
#pragma unroll 1
                    for (int c0 = cb; c0 < cb + HW; c0 += 32) {
                        float a[32];
                        tmem_ld32(acc + c0, a);
                        const int s0 = t.c * 128 + c0;
#pragma unroll
                        for (int j = 0; j < 32; ++j) a[j] = (s0 + j < t_seg) ? -eta * a[j] : 0.0f;
                        store_bf16x32(dst + c0, a);
                    }
                } else {
                    const EpiParams& ep = p.epi;
                    const int tok = t.k * Ls + t.r * 128 + row;
                    const bool valid = tok < p.T;
#pragma unroll 1
                    for (int c0 = cb; c0 < cb + HW; c0 += 32) {
                        float a[32];
                        tmem_ld32(acc + c0, a);
                        if (!valid) continue;
                        const int col0 = t.ni * BN + c0;
                        if (ep.zin) {
                            const __nv_bfloat16* zp = static_cast<const __nv_bfloat16*>(ep.zin) +
                                                      tok_off(ep.z_str, t.l, t.b, tok, t.h) + col0;
#pragma unroll
                            for (int q = 0; q < 4; ++q) {
                                const uint4 zz = *reinterpret_cast<const uint4*>(zp + 8 * q);
                                const __nv_bfloat16* zb = reinterpret_cast<const __nv_bfloat16*>(&zz);
#pragma unroll
                                for (int i = 0; i < 8; ++i)
                                    a[8 * q + i] *= act_df(ep.act, __bfloat162float(zb[i]));
                            }
                        }
                        if (ep.out2) {
                            float h[32];
#pragma unroll
                            for (int j = 0; j < 32; ++j) h[j] = act_f(ep.act, a[j]);
                            store_bf16x32(static_cast<__nv_bfloat16*>(ep.out2) +
                                              tok_off(ep.out2_str, t.l, t.b, tok, t.h) + col0,
                                          h);
                        }
                        store_bf16x32(static_cast<__nv_bfloat16*>(ep.out) +
                                          tok_off(ep.out_str, t.l, t.b, tok, t.h) + col0,
                                      a);
                    }
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&acc_free[buf]);
            }
            if (!ok) break;
        }
    }

    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

template <int MODE, int BN>
cudaError_t launch(const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& a2,
                   const CUtensorMap& b2, const SegGemmParams& p, int grid, cudaStream_t stream) {
    auto kern = seg_gemm_kernel<MODE, BN>;
    cudaError_t err =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
    if (err != cudaSuccess) return err;
    kern<<<grid, kThreads, kSmemBytes, stream>>>(a, b, a2, b2, p);
    return cudaGetLastError();
}

}  // namespace sg

// mode: 0 state, 1 score, 2 output.  bn: output tile width (64, 128 or 256).
cudaError_t launch_seg_gemm(int mode, int bn, const CUtensorMap& a, const CUtensorMap& b,
                            const CUtensorMap& a2, const CUtensorMap& b2, const SegGemmParams& p,
                            int grid, cudaStream_t stream) {
    if (mode == sg::SCORE) return sg::launch<sg::SCORE, 128>(a, b, a2, b2, p, grid, stream);
    if (mode == sg::STATE) {
        if (bn == 256) return sg::launch<sg::STATE, 256>(a, b, a2, b2, p, grid, stream);
        if (bn == 128) return sg::launch<sg::STATE, 128>(a, b, a2, b2, p, grid, stream);
        if (bn == 64) return sg::launch<sg::STATE, 64>(a, b, a2, b2, p, grid, stream);
    }
    if (mode == sg::OUT) {
        if (bn == 256) return sg::launch<sg::OUT, 256>(a, b, a2, b2, p, grid, stream);
        if (bn == 128) return sg::launch<sg::OUT, 128>(a, b, a2, b2, p, grid, stream);
        if (bn == 64) return sg::launch<sg::OUT, 64>(a, b, a2, b2, p, grid, stream);
    }
    return cudaErrorInvalidValue;
}

int seg_gemm_grid(int tiles, int sms) { return tiles < sms ? tiles : sms; }

}  // namespace gl
