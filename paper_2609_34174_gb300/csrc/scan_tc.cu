// scan_tc.cu -- tensor-core (tcgen05) chunked token scan for sm_103a.
//
// Computes, for every unit and every token t (Sec. 3, Eqs. 3-4; Appendix C):
//     o_t = B0 q_t - eta * sum_{s<t} (k_s . q_t) v_s
// in chunks of C = 128 tokens.  With the running state at the start of chunk c
//     S_c^T = B0^T - eta * Z_c,   Z_c = sum_{s < cC} k_s v_s^T   (dq x dv, fp32),
// the chunk's outputs are (all products on the tensor cores, fp32 accumulate)
//     O_c = Q_c S_c^T  +  P_c V_c,      P_c = -eta * strict_lower(Q_c K_c^T)
// and the state advances by Z_{c+1} = Z_c + K_c^T V_c.
//
// Work decomposition.  One item = (unit, 64-wide output tile, token segment).
// A persistent CTA per SM takes items in ticket order.  Segments after the first
// need the state carried in from the earlier segments of their unit; that carry
// is a decoupled look-back over per-segment aggregates sum_{s in seg} k_s v_s^T
// (the additive scan is associative, Sec. 3 "Observation", Eq. 2).  A segment
// that has successors first streams its keys/values once to form its aggregate
// (phase 1), publishes it, looks back, publishes its inclusive prefix, then runs
// the full chunk loop (phase 2, which re-reads the same tiles, mostly from L2).
//
// Warp roles (14 warps, one CTA per SM):
//   warp 0      TMA producer: tickets, item queue, chunk tiles into a stage ring
//   warp 1      TMEM allocator and single-thread tcgen05.mma issuer
//   warps 2-5   score -> P: TMEM score tile, causal mask, scale by -eta, bf16 into smem
//   warps 6-9   output epilogue: TMEM O tile, optional activation, bf16 stores
//   warps 10-13 state: fp32 state rows in registers, dZ from TMEM, S^T tile into smem,
//               look-back carry
//
// Tensor memory (512 columns): score x2 (128 each), O x2 (64), dZ x2 (64).
#include <cuda.h>

#include "scan_common.cuh"
#include "sm103_ptx.cuh"

namespace gl {

constexpr int kChunk = 128;
constexpr int kTile = 16384;  // one [128 rows][64 bf16] 128B-swizzled tile
constexpr int kWarps = 14;
constexpr int kThreads = kWarps * 32;
constexpr int kWarpO0 = 6, kWarpZ0 = 10;  // score->P warps are 2..5
constexpr int kItemConsumers = 1 + 4 + 4 + 4;  // MMA thread + lane 0 of every other role warp

// TMEM column map.
constexpr uint32_t kTmemCols = 512;
__host__ __device__ constexpr uint32_t col_sc(uint32_t i) { return i * 128u; }
__host__ __device__ constexpr uint32_t col_o(uint32_t i) { return 256u + i * 64u; }
__host__ __device__ constexpr uint32_t col_dz(uint32_t i) { return 384u + i * 64u; }

template <int DQ, bool COSTATE>
struct TcLayout {
    static constexpr int kQkBlocks = DQ / 64;
    static constexpr int kQOff = 0;
    static constexpr int kKOff = COSTATE ? kQkBlocks * kTile : 0;
    static constexpr int kVOff = kKOff + kQkBlocks * kTile;
    static constexpr int kStageBytes = kVOff + kTile;
    // Stage count: fill what is left of the 227 KB opt-in budget after P, the two
    // S^T tiles, the barrier block and the alignment slack.
    static constexpr int kFixed = 2 * kTile + 2 * DQ * 128;
    static constexpr int kStages0 = (232448 - kFixed - 1024 - 1024) / kStageBytes;
    static constexpr int kStages = kStages0 > 4 ? 4 : kStages0;
    static constexpr int kPOff = kStages * kStageBytes;
    static constexpr int kStOff = kPOff + 2 * kTile;
    static constexpr int kStBytes = DQ * 128;
    static constexpr int kBarOff = kStOff + 2 * kStBytes;
    static constexpr int kBarBytes = 1024;
    static constexpr int kSmemBytes = kBarOff + kBarBytes + 1024;  // + alignment slack
    // Bytes one stage receives in each pass.
    static constexpr uint32_t kTxPass1 = (kQkBlocks + 1) * kTile;
    static constexpr uint32_t kTxPass2 = ((COSTATE ? 2 : 1) * kQkBlocks + 1) * kTile;
    static_assert(kStages >= 2, "not enough shared memory for two stages");
    static_assert(kSmemBytes <= 232448, "shared memory budget exceeded");
};

struct Item {
    int l, b, h, j, k;
    int t_begin, t_end, nch;
    bool phase1;
};

__device__ __forceinline__ Item decode_item(int item, const TcScanParams& p) {
    Item I;
    I.k = item % p.n_seg;
    int r = item / p.n_seg;
    I.j = r % p.n_tiles;
    int u = r / p.n_tiles;
    I.h = u % p.H;
    int lb = u / p.H;
    I.b = lb % p.B;
    I.l = lb / p.B;
    I.t_begin = I.k * p.seg_len;
    I.t_end = min(p.T, I.t_begin + p.seg_len);
    I.nch = (I.t_end - I.t_begin + kChunk - 1) / kChunk;
    I.phase1 = (p.n_seg > 1) && (I.k < p.n_seg - 1);
    return I;
}

__device__ __forceinline__ void raise_error(const TcScanParams& p, unsigned int bits,
                                            volatile int* abort_flag) {
    atomicOr(p.ctrl + 1, bits);
    if (abort_flag) *abort_flag = 1;
}

// Wait ignoring the abort flag (used only to drain in-flight async work).
__device__ __forceinline__ void mbar_drain(uint64_t* bar, uint32_t parity) {
    uint64_t t0 = globaltimer_ns();
    while (!mbar_try_wait(bar, parity)) {
        if (globaltimer_ns() - t0 > 200000000ull) break;  // 0.2 s
    }
}

// Warp-level wait: lane 0 polls the barrier, the result is broadcast and the
// warp is reconverged (the tcgen05.ld that follow are .sync.aligned).
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag) {
    const int lane = threadIdx.x & 31;
    int ok = 1;
    if (lane == 0) ok = mbar_wait(bar, parity, abort_flag) ? 1 : 0;
    ok = __shfl_sync(0xffffffffu, ok, 0);
    __syncwarp();
    return ok != 0;
}

template <int DQ, bool COSTATE>
__global__ void __launch_bounds__(kThreads, 1)
    tc_scan_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                   const __grid_constant__ CUtensorMap tm_v, const TcScanParams p) {
    using Lay = TcLayout<DQ, COSTATE>;
    constexpr int NS = Lay::kStages;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~static_cast<uintptr_t>(1023));
    const uint32_t sbase = smem_u32(smem);

    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + Lay::kBarOff);
    uint64_t* full = bars;                 // [NS]
    uint64_t* empty = bars + 8;            // [NS]
    uint64_t* sc_full = bars + 16;         // [2]
    uint64_t* sc_free = bars + 18;         // [2]
    uint64_t* o_full = bars + 20;          // [2]
    uint64_t* o_free = bars + 22;          // [2]
    uint64_t* dz_full = bars + 24;         // [2]
    uint64_t* dz_free = bars + 26;         // [2]
    uint64_t* st_ready = bars + 28;        // [2]
    uint64_t* st_free = bars + 30;         // [2]
    uint64_t* item_full = bars + 32;       // [2]
    uint64_t* item_empty = bars + 34;      // [2]
    uint64_t* p_ready = bars + 36;
    uint64_t* p_free = bars + 37;
    uint64_t* z_pub = bars + 38;           // state warps: all rows written before a flag
    uint64_t* z_lb = bars + 39;            // state warps: look-back result broadcast
    uint64_t* z_ack = bars + 40;           // state warps: broadcast consumed
    uint64_t* drain = bars + 41;
    int* misc = reinterpret_cast<int*>(bars + 48);
    volatile int* abort_flag = misc + 0;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(misc + 1);
    volatile int* item_slot = misc + 2;    // [2]
    volatile unsigned int* lb_word = reinterpret_cast<volatile unsigned int*>(misc + 4);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    constexpr int kZActiveWarps = DQ / 32;

    if (threadIdx.x == 0) {
        for (int i = 0; i < NS; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&sc_full[i], 1);
            mbar_init(&sc_free[i], 4);
            mbar_init(&o_full[i], 1);
            mbar_init(&o_free[i], 4);
            mbar_init(&dz_full[i], 1);
            mbar_init(&dz_free[i], 4);
            mbar_init(&st_ready[i], 4);
            mbar_init(&st_free[i], 1);
            mbar_init(&item_full[i], 1);
            mbar_init(&item_empty[i], kItemConsumers);
        }
        mbar_init(p_ready, 4);
        mbar_init(p_free, 1);
        mbar_init(z_pub, kZActiveWarps);
        mbar_init(z_lb, 1);
        mbar_init(z_ack, kZActiveWarps);
        mbar_init(drain, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, kTmemCols);
        tmem_relinquish();
        tc_fence_before();
    }
    if (warp == 0 && lane == 0) {
        prefetch_tmap(&tm_q);
        prefetch_tmap(&tm_k);
        prefetch_tmap(&tm_v);
    }
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            uint32_t n = 0;
            for (int it = 0;; ++it) {
                const int slot = it & 1;
                if (!mbar_wait(&item_empty[slot], ((it >> 1) & 1) ^ 1, abort_flag)) {
                    raise_error(p, kErrWaitTimeout, abort_flag);
                    break;
                }
                int item = static_cast<int>(atomicAdd(p.ctrl, 1u));
                if (item >= p.n_items) item = -1;
                item_slot[slot] = item;
                mbar_arrive(&item_full[slot]);
                if (item < 0) break;
                const Item I = decode_item(item, p);
                bool ok = true;
                for (int pass = I.phase1 ? 1 : 2; pass <= 2 && ok; ++pass) {
                    for (int c = 0; c < I.nch; ++c, ++n) {
                        const int s = n % NS;
                        if (!mbar_wait(&empty[s], ((n / NS) & 1) ^ 1, abort_flag)) {
                            raise_error(p, kErrWaitTimeout, abort_flag);
                            ok = false;
                            break;
                        }
                        uint8_t* st = smem + s * Lay::kStageBytes;
                        const int t0 = I.t_begin + c * kChunk;
                        mbar_arrive_expect_tx(&full[s], pass == 1 ? Lay::kTxPass1 : Lay::kTxPass2);
                        if (COSTATE && pass == 2) {
#pragma unroll
                            for (int kb = 0; kb < Lay::kQkBlocks; ++kb)
                                tma_load_5d(st + Lay::kQOff + kb * kTile, &tm_q, &full[s], kb * 64,
                                            I.h, t0, I.b, I.l);
                        }
#pragma unroll
                        for (int kb = 0; kb < Lay::kQkBlocks; ++kb)
                            tma_load_5d(st + Lay::kKOff + kb * kTile, &tm_k, &full[s], kb * 64, I.h,
                                        t0, I.b, I.l);
                        tma_load_5d(st + Lay::kVOff, &tm_v, &full[s], I.j * 64, I.h, t0, I.b, I.l);
                    }
                }
                if (!ok) break;
            }
            // Drain: every issued load has landed before the CTA can exit.
            if (*abort_flag) {
                for (int s = 0; s < NS; ++s) {
                    if (n > (uint32_t)s) {
                        uint32_t last = ((n - 1 - s) / NS) * NS + s;
                        mbar_drain(&full[s], (last / NS) & 1);
                    }
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------- MMA issuer
        if (lane == 0) {
            constexpr uint32_t ID_SC = idesc_bf16(128, 128, false, false);
            constexpr uint32_t ID_O = idesc_bf16(128, 64, false, true);
            constexpr uint32_t ID_DZ = idesc_bf16(128, 64, true, true);
            const uint32_t p_addr = sbase + Lay::kPOff;
            uint32_t n = 0, c2 = 0, dzc = 0;
            bool ok = true;
            // dZ += K^T V over one stage (A = K^T: MN-major, 64-wide M blocks 16 KB apart;
            // for DQ = 64 the second M block is the V tile, whose rows land in unused lanes).
            auto issue_dz = [&](int s, uint32_t dcol, bool first) {
                const uint32_t st = sbase + s * Lay::kStageBytes;
#pragma unroll
                for (int kk = 0; kk < kChunk / 16; ++kk) {
                    uint64_t a = sdesc_sw128(st + Lay::kKOff + kk * 2048, kTile, 1024);
                    uint64_t b = sdesc_sw128(st + Lay::kVOff + kk * 2048, kTile, 1024);
                    mma_bf16_ss(tmem + dcol, a, b, ID_DZ, (first && kk == 0) ? 0u : 1u);
                }
            };
            auto wait_or_fail = [&](uint64_t* bar, uint32_t par) -> bool {
                if (mbar_wait(bar, par, abort_flag)) return true;
                raise_error(p, kErrWaitTimeout, abort_flag);
                return false;
            };
            for (int it = 0; ok; ++it) {
                const int slot = it & 1;
                if (!wait_or_fail(&item_full[slot], (it >> 1) & 1)) break;
                const int item = item_slot[slot];
                mbar_arrive(&item_empty[slot]);
                if (item < 0) break;
                const Item I = decode_item(item, p);
                if (I.phase1) {
                    const uint32_t b = dzc & 1;
                    if (!wait_or_fail(&dz_free[b], ((dzc >> 1) & 1) ^ 1)) break;
                    tc_fence_after();
                    for (int c = 0; c < I.nch; ++c, ++n) {
                        const int s = n % NS;
                        if (!(ok = wait_or_fail(&full[s], (n / NS) & 1))) break;
                        tc_fence_after();
                        issue_dz(s, col_dz(b), c == 0);
                        mma_commit(&empty[s]);
                    }
                    if (!ok) break;
                    mma_commit(&dz_full[b]);
                    ++dzc;
                }
                // Phase 2.  front(c): score and dZ of chunk c; back(c): O of chunk c.
                const uint32_t n0 = n;
                auto front = [&](int c) -> bool {
                    const uint32_t nn = n0 + c;
                    const int s = nn % NS;
                    if (!wait_or_fail(&full[s], (nn / NS) & 1)) return false;
                    const uint32_t cc = c2 + c, sb = cc & 1;
                    if (!wait_or_fail(&sc_free[sb], ((cc >> 1) & 1) ^ 1)) return false;
                    tc_fence_after();
                    const uint32_t st = sbase + s * Lay::kStageBytes;
#pragma unroll
                    for (int kk = 0; kk < DQ / 16; ++kk) {
                        const uint32_t off = (kk >> 2) * kTile + (kk & 3) * 32;
                        uint64_t a = sdesc_sw128(st + Lay::kQOff + off, 16, 1024);
                        uint64_t b = sdesc_sw128(st + Lay::kKOff + off, 16, 1024);
                        mma_bf16_ss(tmem + col_sc(sb), a, b, ID_SC, kk > 0 ? 1u : 0u);
                    }
                    mma_commit(&sc_full[sb]);
                    if (c < I.nch - 1) {
                        const uint32_t b = dzc & 1;
                        if (!wait_or_fail(&dz_free[b], ((dzc >> 1) & 1) ^ 1)) return false;
                        tc_fence_after();
                        issue_dz(s, col_dz(b), true);
                        mma_commit(&dz_full[b]);
                        ++dzc;
                    }
                    return true;
                };
                if (!(ok = front(0))) break;
                for (int c = 0; c < I.nch && ok; ++c) {
                    if (c + 1 < I.nch && !(ok = front(c + 1))) break;
                    const uint32_t nn = n0 + c;
                    const int s = nn % NS;
                    const uint32_t cc = c2 + c, ob = cc & 1, oph = (cc >> 1) & 1;
                    if (!(ok = wait_or_fail(&o_free[ob], oph ^ 1))) break;
                    if (!(ok = wait_or_fail(&st_ready[ob], oph))) break;
                    tc_fence_after();
                    const uint32_t st = sbase + s * Lay::kStageBytes;
                    const uint32_t st_tile = sbase + Lay::kStOff + ob * Lay::kStBytes;
                    // O = Q S^T  (B = S^T tile [dq][64]: MN-major)
#pragma unroll
                    for (int kk = 0; kk < DQ / 16; ++kk) {
                        const uint32_t off = (kk >> 2) * kTile + (kk & 3) * 32;
                        uint64_t a = sdesc_sw128(st + Lay::kQOff + off, 16, 1024);
                        uint64_t b = sdesc_sw128(st_tile + kk * 2048, kTile, 1024);
                        mma_bf16_ss(tmem + col_o(ob), a, b, ID_O, kk > 0 ? 1u : 0u);
                    }
                    mma_commit(&st_free[ob]);
                    if (!(ok = wait_or_fail(p_ready, cc & 1))) break;
                    tc_fence_after();
                    // O += P V  (A = P [128][128] K-major, B = V [128 tokens][64]: MN-major)
#pragma unroll
                    for (int kk = 0; kk < kChunk / 16; ++kk) {
                        const uint32_t off = (kk >> 2) * kTile + (kk & 3) * 32;
                        uint64_t a = sdesc_sw128(p_addr + off, 16, 1024);
                        uint64_t b = sdesc_sw128(st + Lay::kVOff + kk * 2048, kTile, 1024);
                        mma_bf16_ss(tmem + col_o(ob), a, b, ID_O, 1u);
                    }
                    mma_commit(&o_full[ob]);
                    mma_commit(p_free);
                    mma_commit(&empty[s]);
                }
                n = n0 + I.nch;
                c2 += I.nch;
            }
            // Every MMA has completed before TMEM is released.
            mma_commit(drain);
            mbar_drain(drain, 0);
        }
    } else if (warp < kWarpO0) {
        // ------------------------------------------------------ score -> P
        const int q4 = warp & 3;
        const int row = q4 * 32 + lane;
        const uint32_t lane_off = static_cast<uint32_t>(q4 * 32) << 16;
        const uint32_t p_addr = sbase + Lay::kPOff;
        const float neg_eta = -p.eta;
        uint32_t c2 = 0;
        for (int it = 0;; ++it) {
            const int slot = it & 1;
            if (!warp_wait(&item_full[slot], (it >> 1) & 1, abort_flag)) {
                raise_error(p, kErrWaitTimeout, abort_flag);
                break;
            }
            const int item = item_slot[slot];
            __syncwarp();
            if (lane == 0) mbar_arrive(&item_empty[slot]);
            if (item < 0) break;
            const Item I = decode_item(item, p);
            bool ok = true;
            for (int c = 0; c < I.nch; ++c, ++c2) {
                const uint32_t sb = c2 & 1;
                if (!warp_wait(&sc_full[sb], (c2 >> 1) & 1, abort_flag) ||
                    !warp_wait(p_free, (c2 & 1) ^ 1, abort_flag)) {
                    raise_error(p, kErrWaitTimeout, abort_flag);
                    ok = false;
                    break;
                }
                tc_fence_after();
#pragma unroll 1
                for (int piece = 0; piece < 4; ++piece) {
                    uint32_t w[16];
                    if (piece <= q4) {
                        float v[32];
                        tmem_ld32(tmem + col_sc(sb) + lane_off + piece * 32, v);
#pragma unroll
                        for (int i = 0; i < 16; ++i) {
                            const int s0 = piece * 32 + 2 * i;
                            float a = (s0 < row) ? neg_eta * v[2 * i] : 0.0f;
                            float b2 = (s0 + 1 < row) ? neg_eta * v[2 * i + 1] : 0.0f;
                            w[i] = pack_bf16x2(a, b2);
                        }
                    } else {
#pragma unroll
                        for (int i = 0; i < 16; ++i) w[i] = 0u;
                    }
                    const uint32_t blk = p_addr + (piece >> 1) * kTile;
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        const uint32_t chunk = (piece & 1) * 4 + q;
                        st_shared_v4(blk + sw128_off(row, chunk), w[4 * q], w[4 * q + 1],
                                     w[4 * q + 2], w[4 * q + 3]);
                    }
                }
                tc_fence_before();
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) {
                    mbar_arrive(&sc_free[sb]);
                    mbar_arrive(p_ready);
                }
            }
            if (!ok) break;
        }
    } else if (warp < kWarpZ0) {
        // ------------------------------------------------- output epilogue
        const int q4 = warp & 3;
        const int row = q4 * 32 + lane;
        const uint32_t lane_off = static_cast<uint32_t>(q4 * 32) << 16;
        const EpiParams& e = p.epi;
        uint32_t c2 = 0;
        for (int it = 0;; ++it) {
            const int slot = it & 1;
            if (!warp_wait(&item_full[slot], (it >> 1) & 1, abort_flag)) {
                raise_error(p, kErrWaitTimeout, abort_flag);
                break;
            }
            const int item = item_slot[slot];
            __syncwarp();
            if (lane == 0) mbar_arrive(&item_empty[slot]);
            if (item < 0) break;
            const Item I = decode_item(item, p);
            bool ok = true;
            for (int c = 0; c < I.nch; ++c, ++c2) {
                const uint32_t ob = c2 & 1;
                if (!warp_wait(&o_full[ob], (c2 >> 1) & 1, abort_flag)) {
                    raise_error(p, kErrWaitTimeout, abort_flag);
                    ok = false;
                    break;
                }
                tc_fence_after();
                float v[64];
                {
                    float a[32];
                    tmem_ld32(tmem + col_o(ob) + lane_off, a);
#pragma unroll
                    for (int i = 0; i < 32; ++i) v[i] = a[i];
                    tmem_ld32(tmem + col_o(ob) + lane_off + 32, a);
#pragma unroll
                    for (int i = 0; i < 32; ++i) v[32 + i] = a[i];
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&o_free[ob]);
                const int t = I.t_begin + c * kChunk + row;
                if (t < I.t_end) {
                    const int col0 = I.j * 64;
                    if (e.zin) {
                        const __nv_bfloat16* zp = static_cast<const __nv_bfloat16*>(e.zin) +
                                                  tok_off(e.z_str, I.l, I.b, t, I.h) + col0;
#pragma unroll
                        for (int q = 0; q < 8; ++q) {
                            uint4 zz = *reinterpret_cast<const uint4*>(zp + 8 * q);
                            const __nv_bfloat16* zb = reinterpret_cast<const __nv_bfloat16*>(&zz);
#pragma unroll
                            for (int i = 0; i < 8; ++i)
                                v[8 * q + i] *= act_df(e.act, __bfloat162float(zb[i]));
                        }
                    }
                    __nv_bfloat16* op = static_cast<__nv_bfloat16*>(e.out) +
                                        tok_off(e.out_str, I.l, I.b, t, I.h) + col0;
#pragma unroll
                    for (int q = 0; q < 8; ++q) {
                        uint4 w;
                        w.x = pack_bf16x2(v[8 * q + 0], v[8 * q + 1]);
                        w.y = pack_bf16x2(v[8 * q + 2], v[8 * q + 3]);
                        w.z = pack_bf16x2(v[8 * q + 4], v[8 * q + 5]);
                        w.w = pack_bf16x2(v[8 * q + 6], v[8 * q + 7]);
                        *reinterpret_cast<uint4*>(op + 8 * q) = w;
                    }
                    if (e.out2) {
                        __nv_bfloat16* op2 = static_cast<__nv_bfloat16*>(e.out2) +
                                             tok_off(e.out2_str, I.l, I.b, t, I.h) + col0;
#pragma unroll
                        for (int q = 0; q < 8; ++q) {
                            uint4 w;
                            w.x = pack_bf16x2(act_f(e.act, v[8 * q + 0]), act_f(e.act, v[8 * q + 1]));
                            w.y = pack_bf16x2(act_f(e.act, v[8 * q + 2]), act_f(e.act, v[8 * q + 3]));
                            w.z = pack_bf16x2(act_f(e.act, v[8 * q + 4]), act_f(e.act, v[8 * q + 5]));
                            w.w = pack_bf16x2(act_f(e.act, v[8 * q + 6]), act_f(e.act, v[8 * q + 7]));
                            *reinterpret_cast<uint4*>(op2 + 8 * q) = w;
                        }
                    }
                }
            }
            if (!ok) break;
        }
    } else {
        // ------------------------------------------------------------ state
        const int q4 = warp & 3;
        const int row = q4 * 32 + lane;         // contraction index q of this thread's state row
        const bool active = row < DQ;           // warp-uniform
        const bool leader = (q4 == 0) && (lane == 0);
        const uint32_t lane_off = static_cast<uint32_t>(q4 * 32) << 16;
        const float eta = p.eta;
        uint32_t c2 = 0, dzc = 0, pubc = 0, lbc = 0;
        float st[64];
        const size_t blk = (size_t)DQ * 64;
        for (int it = 0;; ++it) {
            const int slot = it & 1;
            if (!warp_wait(&item_full[slot], (it >> 1) & 1, abort_flag)) {
                raise_error(p, kErrWaitTimeout, abort_flag);
                break;
            }
            const int item = item_slot[slot];
            __syncwarp();
            if (lane == 0) mbar_arrive(&item_empty[slot]);
            if (item < 0) break;
            const Item I = decode_item(item, p);
            bool ok = true;
            // Publish this item's look-back status once every active state thread's
            // rows are globally visible: all arrive and all wait (a full barrier),
            // then the leader releases the flag.
            auto publish = [&](unsigned int flag) -> bool {
                __threadfence();
                __syncwarp();
                if (lane == 0) mbar_arrive(z_pub);
                const bool okp = warp_wait(z_pub, pubc & 1, abort_flag);
                ++pubc;
                if (!okp) {
                    raise_error(p, kErrWaitTimeout, abort_flag);
                    return false;
                }
                if (leader) st_release_gpu(p.flags + item, flag);
                return true;
            };
            // ---- phase 1: this segment's aggregate sum_{s in seg} k_s v_s^T.  The
            // first segment's aggregate is already its inclusive prefix (flag 2);
            // later segments publish the aggregate (flag 1) and look back.
            if (I.phase1) {
                const uint32_t b = dzc & 1;
                if (!warp_wait(&dz_full[b], (dzc >> 1) & 1, abort_flag)) {
                    raise_error(p, kErrWaitTimeout, abort_flag);
                    break;
                }
                tc_fence_after();
                if (active) {
                    float* dst = (I.k == 0 ? p.incl : p.agg) + (size_t)item * blk + (size_t)row * 64;
                    float a[32];
#pragma unroll
                    for (int h = 0; h < 2; ++h) {
                        tmem_ld32(tmem + col_dz(b) + lane_off + h * 32, a);
#pragma unroll
                        for (int i = 0; i < 32; i += 4)
                            *reinterpret_cast<float4*>(dst + h * 32 + i) =
                                make_float4(a[i], a[i + 1], a[i + 2], a[i + 3]);
                    }
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&dz_free[b]);
                ++dzc;
                if (active && !publish(I.k == 0 ? 2u : 1u)) break;
            }
            // ---- look-back: E = sum of the earlier segments' aggregates, stopping at
            // the nearest inclusive prefix.  The leader walks the flags; one broadcast
            // (count << 1 | ends-at-inclusive) tells every state thread what to sum.
#pragma unroll
            for (int i = 0; i < 64; ++i) st[i] = 0.0f;
            if (active && I.k > 0) {
                if (leader) {
                    unsigned int word = 0xFFFFFFFFu;
                    unsigned int cnt = 0;
                    const uint64_t t0 = globaltimer_ns();
                    bool timed_out = false;
                    for (int pred = item - 1, kk = I.k - 1; kk >= 0 && !timed_out; --pred, --kk) {
                        unsigned int f;
                        while ((f = ld_acquire_gpu(p.flags + pred)) == 0u) {
                            if (globaltimer_ns() - t0 > kWaitLimitNs) {
                                timed_out = true;
                                break;
                            }
                            __nanosleep(64);
                        }
                        if (timed_out) break;
                        ++cnt;
                        if (f == 2u) {
                            word = (cnt << 1) | 1u;
                            break;
                        }
                    }
                    if (timed_out) {
                        word = 0xFFFFFFFFu;
                        raise_error(p, kErrLookbackTimeout, nullptr);
                    }
                    // the previous broadcast has been read by every state thread
                    if (!mbar_wait(z_ack, (lbc & 1) ^ 1, abort_flag))
                        raise_error(p, kErrWaitTimeout, abort_flag);
                    *lb_word = word;
                    mbar_arrive(z_lb);
                }
                if (!warp_wait(z_lb, lbc & 1, abort_flag)) {
                    raise_error(p, kErrWaitTimeout, abort_flag);
                    break;
                }
                const unsigned int word = *lb_word;
                __syncwarp();
                if (lane == 0) mbar_arrive(z_ack);
                ++lbc;
                if (word != 0xFFFFFFFFu) {
                    const int cnt = static_cast<int>(word >> 1);
                    const bool ends_incl = (word & 1u) != 0;
                    __threadfence();
                    for (int i = 0; i < cnt; ++i) {
                        const int pred = item - 1 - i;
                        const float* src = ((i == cnt - 1 && ends_incl) ? p.incl : p.agg) +
                                           (size_t)pred * blk + (size_t)row * 64;
#pragma unroll
                        for (int e4 = 0; e4 < 64; e4 += 4) {
                            float4 a = __ldcg(reinterpret_cast<const float4*>(src + e4));
                            st[e4] += a.x;
                            st[e4 + 1] += a.y;
                            st[e4 + 2] += a.z;
                            st[e4 + 3] += a.w;
                        }
                    }
                }
            }
            // ---- publish the inclusive prefix E + aggregate (flag 2)
            if (active && I.phase1 && I.k > 0) {
                const float* own = p.agg + (size_t)item * blk + (size_t)row * 64;
                float* dst = p.incl + (size_t)item * blk + (size_t)row * 64;
#pragma unroll
                for (int i = 0; i < 64; i += 4) {
                    float4 a = __ldcg(reinterpret_cast<const float4*>(own + i));
                    *reinterpret_cast<float4*>(dst + i) =
                        make_float4(st[i] + a.x, st[i + 1] + a.y, st[i + 2] + a.z, st[i + 3] + a.w);
                }
                if (!publish(2u)) break;
            }
            // ---- starting state S^T row = B0^T row - eta * E
            if (active) {
                const float* w0 = p.W0 + (size_t)(I.l * p.H + I.h) * p.dq * p.dv;
                const int v0 = I.j * 64;
                if (p.w0_transposed) {
                    const float* r = w0 + (size_t)row * p.dv + v0;  // W0 [dq][dv]
#pragma unroll
                    for (int i = 0; i < 64; i += 4) {
                        float4 a = *reinterpret_cast<const float4*>(r + i);
                        st[i] = a.x - eta * st[i];
                        st[i + 1] = a.y - eta * st[i + 1];
                        st[i + 2] = a.z - eta * st[i + 2];
                        st[i + 3] = a.w - eta * st[i + 3];
                    }
                } else {
#pragma unroll
                    for (int i = 0; i < 64; ++i)  // W0 [dv][dq]: column `row`
                        st[i] = w0[(size_t)(v0 + i) * p.dq + row] - eta * st[i];
                }
            }
            // ---- phase 2: S^T tile for every chunk, state advanced by dZ
            for (int c = 0; c < I.nch; ++c, ++c2) {
                const uint32_t sb = c2 & 1;
                if (!warp_wait(&st_free[sb], ((c2 >> 1) & 1) ^ 1, abort_flag)) {
                    raise_error(p, kErrWaitTimeout, abort_flag);
                    ok = false;
                    break;
                }
                if (active) {
                    const uint32_t tile = sbase + Lay::kStOff + sb * Lay::kStBytes;
#pragma unroll
                    for (int q = 0; q < 8; ++q)
                        st_shared_v4(tile + sw128_off(row, q), pack_bf16x2(st[8 * q], st[8 * q + 1]),
                                     pack_bf16x2(st[8 * q + 2], st[8 * q + 3]),
                                     pack_bf16x2(st[8 * q + 4], st[8 * q + 5]),
                                     pack_bf16x2(st[8 * q + 6], st[8 * q + 7]));
                    fence_proxy_async_smem();
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(&st_ready[sb]);
                if (c < I.nch - 1) {
                    const uint32_t b = dzc & 1;
                    if (!warp_wait(&dz_full[b], (dzc >> 1) & 1, abort_flag)) {
                        raise_error(p, kErrWaitTimeout, abort_flag);
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    if (active) {
                        float a[32];
#pragma unroll
                        for (int h = 0; h < 2; ++h) {
                            tmem_ld32(tmem + col_dz(b) + lane_off + h * 32, a);
#pragma unroll
                            for (int i = 0; i < 32; ++i) st[h * 32 + i] -= eta * a[i];
                        }
                    }
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&dz_free[b]);
                    ++dzc;
                }
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

// ------------------------------------------------------------------ host side
template <int DQ, bool COSTATE>
static cudaError_t launch_one(const CUtensorMap& q, const CUtensorMap& k, const CUtensorMap& v,
                              const TcScanParams& p, int grid, cudaStream_t stream) {
    using Lay = TcLayout<DQ, COSTATE>;
    auto kern = tc_scan_kernel<DQ, COSTATE>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         Lay::kSmemBytes);
    if (e != cudaSuccess) return e;
    kern<<<grid, kThreads, Lay::kSmemBytes, stream>>>(q, k, v, p);
    return cudaGetLastError();
}

cudaError_t launch_tc_scan(const CUtensorMap& q, const CUtensorMap& k, const CUtensorMap& v,
                           const TcScanParams& p, bool costate, int grid, cudaStream_t stream) {
    if (p.dq == 64)
        return costate ? launch_one<64, true>(q, k, v, p, grid, stream)
                       : launch_one<64, false>(q, k, v, p, grid, stream);
    if (p.dq == 128)
        return costate ? launch_one<128, true>(q, k, v, p, grid, stream)
                       : launch_one<128, false>(q, k, v, p, grid, stream);
    return cudaErrorInvalidValue;
}

}  // namespace gl
