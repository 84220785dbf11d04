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
// A persistent CTA per SM takes items in ticket order, segment-major (segment k of
// every (unit, tile) pair before any segment k+1).  Segments after the first
// need the state carried in from the earlier segments of their unit; that carry
// is a decoupled look-back over per-segment aggregates sum_{s in seg} k_s v_s^T
// (the additive scan is associative, Sec. 3 "Observation", Eq. 2).  A segment
// that has successors first streams its keys/values once to form its aggregate
// (phase 1) and publishes it, then later looks back, publishes its inclusive prefix
// and runs the full chunk loop (phase 2, which re-reads the same tiles).  A CTA runs phase 1 of the item it has just taken BEFORE phase 2 of
// its previous item, so an aggregate is published right after its ticket is
// taken and successors in other CTAs rarely wait in their look-back.
//
// Warp roles (15 warps, 16 for the suffix read, whose numbers are in brackets;
// one CTA per SM):
//   warp 14 [0]   TMA producer: tickets, item queue, chunk tiles into a stage ring
//   warp 1 [14]   lane 0 issues the "front" MMAs of every chunk (score Q K^T and
//                 state increment K^T V), up to two chunks ahead; warp 1 allocates TMEM
//   warp 0 [15]   lane 0 issues the "back" MMAs (O = Q S^T, then O += P V); the two
//                 issuers run independent in-order loops, so the output product of
//                 chunk c never waits behind the score of chunk c+1
//   warps 2-5   score -> P: TMEM score tile, causal mask, bf16 P written back over
//               the same TMEM columns (the PV product reads its A operand from
//               tensor memory, so P never touches shared memory).  P is left
//               unscaled: the state is kept in units of lam = -eta, so the S^T tile
//               carries the factor and the epilogue multiplies O by lam once.
//   warps 6-9   output epilogue: TMEM O tile -> bf16 staging tile in shared memory ->
//               one TMA tensor store per chunk (whole 128-byte rows, no scattered
//               per-thread stores competing with the other roles for the LSU path)
//   warps 10-13 state: fp32 state rows in registers, dZ from TMEM, S^T tile into smem,
//               look-back carry.  With 64-wide keys only warps 10-11... hold state
//               rows (lanes 0..63); the two warps whose lanes are 64..127 then build
//               the second half of P for those rows instead.
//
// Tensor memory (512 columns): score/P x2 (128 each), O x2 (64), dZ x2 (64).
//
// Every MMA operand descriptor is built once per stage; a K-step only adds a
// compile-time constant to its low word, which keeps the single issuing thread
// ahead of the tensor pipe.
#include <cuda.h>

#include "scan_common.cuh"
#include "sm103_ptx.cuh"

namespace gl {

constexpr int kChunk = 128;
constexpr int kTile = 16384;  // one [128 rows][64 bf16] 128B-swizzled tile
constexpr int kWarps = 15;
constexpr int kThreads = kWarps * 32;
constexpr int kWarpO0 = 6, kWarpZ0 = 10;  // score->P warps are 2..5
// The MMA issuers sit on the SM sub-partitions (warp % 4) whose P warps build the
// half-masked rows: 0 and 1 for the causal reads, 2 and 3 for the suffix read (REV),
// which adds a 16th warp for its back issuer; warp 1 then only allocates tensor memory.
// The producer, a few instructions a chunk, takes a sub-partition left over.  A warp
// issuing ALU work every cycle on an issuer's sub-partition slows its MMAs.
template <bool REV> struct Roles {
    static constexpr int kProd = REV ? 0 : 14, kFront = REV ? 14 : 1, kBack = REV ? 15 : 0;
    static constexpr int kThreads = (REV ? 16 : 15) * 32;
};
constexpr int kItemConsumers = 2 + 4 + 4 + 4;  // two MMA issuers + lane 0 of every other role warp
constexpr int kRing = 4;                        // item queue depth

// TMEM column map.
constexpr uint32_t kTmemCols = 512;
__host__ __device__ constexpr uint32_t col_sc(uint32_t i) { return i * 128u; }
__host__ __device__ constexpr uint32_t col_o(uint32_t i) { return 256u + i * 64u; }
__host__ __device__ constexpr uint32_t col_dz(uint32_t i) { return 384u + i * 64u; }

// Stage layout [q | k | v] (costate), [qk | v] (forward).  The reverse read with one
// q/k tile puts v first, [v | qk]: the dZ product's A operand then starts one block
// before k in both reverse layouts, which places K^T in TMEM lanes 64..127.
// FUSED (both reads in one pass, 64-wide maps): [x | ghat | g_out].  The forward read
// takes q = k = x, v = ghat; the costate read q = g_out, k = ghat, v = x; the
// writes (state increment) are those of the forward orientation, x^T ghat.
template <int DQ, bool COSTATE, bool REV = false, bool FUSED = false>
struct TcLayout {
    static constexpr int kQkBlocks = DQ / 64;
    static constexpr bool kVFirst = REV && !COSTATE;
    static constexpr int kQOff = FUSED ? 0 : (kVFirst ? kTile : 0);
    static constexpr int kKOff = FUSED ? 0 : (COSTATE ? kQkBlocks * kTile : kQOff);
    static constexpr int kVOff = FUSED ? kTile : (kVFirst ? 0 : kKOff + kQkBlocks * kTile);
    static constexpr int kGOff = 2 * kTile;  // FUSED: the g_out tile
    static constexpr int kStageBytes =
        FUSED ? 3 * kTile : ((COSTATE ? 2 : 1) * kQkBlocks + 1) * kTile;
    // Stage ring: what is left of the 227 KB opt-in budget after the two S^T
    // tiles, the two output staging tiles, the barrier block and the alignment
    // slack (at most 6 stages).
    // REV: one more tile for the ring of dotted tiles (with the two idle staging tiles)
    static constexpr int kExtraA = REV ? kTile : 0;
    static constexpr int kAvail = 232448 - 2 * DQ * 128 - 2 * kTile - kExtraA - 1024 - 1024;
    static constexpr int kStages0 = kAvail / kStageBytes;
    static constexpr int kStages = kStages0 > 6 ? 6 : kStages0;
    static constexpr int kOOff = kStages * kStageBytes;  // two [128 t][64] output tiles
    static constexpr int kStOff = kOOff + 2 * kTile;
    static constexpr int kStBytes = DQ * 128;
    static constexpr int kAOff = kStOff + 2 * kStBytes;
    static constexpr int kBarOff = kAOff + kExtraA;
    static constexpr int kBarBytes = 1024;
    static constexpr int kSmemBytes = kBarOff + kBarBytes + 1024;  // + alignment slack
    // Bytes one stage receives in each pass.
    static constexpr uint32_t kTxPass1 = (kQkBlocks + 1) * kTile;
    static constexpr uint32_t kTxPass2 = kStageBytes;
    static_assert(kStages >= 2, "not enough shared memory for two stages");
    static_assert(kSmemBytes <= 232448, "shared memory budget exceeded");
};

struct Item {
    int l, b, h, j, k;
    int t_begin, t_end, nch;
    bool phase1;
};

// Items are numbered segment-major: every (unit, tile) pair's segment k comes
// before any segment k+1, so segment k's predecessor is item - n_ut and a
// look-back mostly finds inclusive prefixes published by earlier waves.
// REV (the anti-causal suffix read) numbers segments from the end of the sequence:
// segment k covers [T - (k+1) seg_len, T - k seg_len), clipped at token 0.
template <bool REV>
__device__ __forceinline__ Item decode_item(int item, const TcScanParams& p) {
    Item I;
    I.k = item / p.n_ut;
    int r = item - I.k * p.n_ut;
    I.j = r % p.n_tiles;
    int u = r / p.n_tiles;
    I.h = u % p.H;
    int lb = u / p.H;
    I.b = lb % p.B;
    I.l = lb / p.B;
    if constexpr (REV) {
        I.t_end = p.T - I.k * p.seg_len;
        I.t_begin = max(0, I.t_end - p.seg_len);
    } else {
        I.t_begin = I.k * p.seg_len;
        I.t_end = min(p.T, I.t_begin + p.seg_len);
    }
    I.nch = (I.t_end - I.t_begin + kChunk - 1) / kChunk;
    I.phase1 = (p.n_seg > 1) && (I.k < p.n_seg - 1);
    return I;
}

// First token of chunk c of an item: chunks run forward from the segment start, or
// (REV) backward from its end, so that a reverse item's lowest chunk may start
// before token 0 (its missing rows load as zeros and are not stored).
template <bool REV>
__device__ __forceinline__ int chunk_t0(const Item& I, int c) {
    return REV ? I.t_end - (c + 1) * kChunk : I.t_begin + c * kChunk;
}

// One 64-wide bf16 output row written straight to global memory: a TMA store may
// not start at a negative coordinate, so a reverse chunk that begins before token 0
// is stored row by row.
__device__ __noinline__ void epi_store_row(const EpiParams& e, long long o_off, const float* v) {
    __nv_bfloat16* op = static_cast<__nv_bfloat16*>(e.out) + o_off;
    for (int q = 0; q < 8; ++q) {
        uint4 w;
        w.x = pack_bf16x2(v[8 * q + 0], v[8 * q + 1]);
        w.y = pack_bf16x2(v[8 * q + 2], v[8 * q + 3]);
        w.z = pack_bf16x2(v[8 * q + 4], v[8 * q + 5]);
        w.w = pack_bf16x2(v[8 * q + 6], v[8 * q + 7]);
        *reinterpret_cast<uint4*>(op + 8 * q) = w;
    }
}

// Out of line: cold code inside the role loops spreads their instruction fetch.
__device__ __noinline__ void raise_error(const TcScanParams& p, unsigned int bits,
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

// v *= sigma'(z) for one 64-wide output row piece (costate MLP fusion).
__device__ __noinline__ void epi_apply_dact(const EpiParams& e, long long z_off, float* v) {
    const __nv_bfloat16* zp = static_cast<const __nv_bfloat16*>(e.zin) + z_off;
    for (int q = 0; q < 8; ++q) {
        const uint4 zz = *reinterpret_cast<const uint4*>(zp + 8 * q);
        const __nv_bfloat16* zb = reinterpret_cast<const __nv_bfloat16*>(&zz);
#pragma unroll
        for (int i = 0; i < 8; ++i) v[8 * q + i] *= act_df(e.act, __bfloat162float(zb[i]));
    }
}

// out2 = sigma(v) for one 64-wide output row piece (forward MLP fusion).
__device__ __noinline__ void epi_store_act(const EpiParams& e, long long o_off, const float* v) {
    __nv_bfloat16* op2 = static_cast<__nv_bfloat16*>(e.out2) + o_off;
    for (int q = 0; q < 8; ++q) {
        uint4 w;
        w.x = pack_bf16x2(act_f(e.act, v[8 * q + 0]), act_f(e.act, v[8 * q + 1]));
        w.y = pack_bf16x2(act_f(e.act, v[8 * q + 2]), act_f(e.act, v[8 * q + 3]));
        w.z = pack_bf16x2(act_f(e.act, v[8 * q + 4]), act_f(e.act, v[8 * q + 5]));
        w.w = pack_bf16x2(act_f(e.act, v[8 * q + 6]), act_f(e.act, v[8 * q + 7]));
        *reinterpret_cast<uint4*>(op2 + 8 * q) = w;
    }
}

// e.cons_out[idx] = e.cons_scale * ||p row - v||^2 for one 64-wide output row piece:
// the per-token consistency term between a proposal and the reconstructed costate
// (Sec. 3, Eq. 5; Appendix A).
__device__ __noinline__ void epi_consistency(const EpiParams& e, long long p_off, const float* v,
                                             long long idx) {
    const __nv_bfloat16* pp = static_cast<const __nv_bfloat16*>(e.cons_p) + p_off;
    float acc = 0.f;
    for (int q = 0; q < 8; ++q) {
        const uint4 pv = *reinterpret_cast<const uint4*>(pp + 8 * q);
        const __nv_bfloat16* pb = reinterpret_cast<const __nv_bfloat16*>(&pv);
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            const float dlt = __bfloat162float(pb[i]) - v[8 * q + i];
            acc = fmaf(dlt, dlt, acc);
        }
    }
    e.cons_out[idx] = e.cons_scale * acc;
}

// K-step offsets (in the 16-byte units of a descriptor's low word).
// K-major operand, 64-wide K blocks 16 KB apart: step kk starts 32 B further in
// its 128-byte swizzled row, and every 4 steps moves to the next block.
__host__ __device__ constexpr uint32_t kmaj_step(int kk) {
    return (uint32_t)(((kk >> 2) * kTile + (kk & 3) * 32) >> 4);
}
// MN-major operand: step kk starts 16 rows (two 8-row groups of 1024 B) further.
__host__ __device__ constexpr uint32_t mnmaj_step(int kk) { return (uint32_t)((kk * 2048) >> 4); }

// FUSED runs the forward and the costate read of one 64-wide map in a single pass
// over the shared writes (Sec. 3, steps 2 and 3): per chunk two jobs, the forward
// read (score, P and O buffers 0, stored through tm_o) and the costate read (buffers
// 1, stored through tm_o2), one S'^T tile and one state update.  Maps: tm_q = x,
// tm_k = ghat, tm_v = g_out.
template <int DQ, bool COSTATE, bool REV, bool FUSED, bool DOT>
__global__ void __launch_bounds__(Roles<REV>::kThreads, 1)
    tc_scan_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                   const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_o,
                   const __grid_constant__ CUtensorMap tm_o2, const TcScanParams p) {
    using Lay = TcLayout<DQ, COSTATE, REV, FUSED>;
    static_assert(!FUSED || (DQ == 64 && !COSTATE && !REV), "the fused pass is built for 64-wide maps");
    constexpr int kJobs = FUSED ? 2 : 1;  // reads per chunk
    // The suffix read and the fused pass carry more code (the per-row dot, two reads'
    // epilogues): their MMA K steps stay rolled loops, which eases instruction fetch
    // (c5: suffix read with dot 1.24 -> 1.10 ms, fused 1.29 -> 1.26 ms); the plain
    // causal reads measured faster fully unrolled.
    constexpr int kMmaUnroll = (REV || FUSED) ? 1 : 8;
    // DOT: a suffix read reduced to its per-row dot alone (no rows stored, no
    // activation): its epilogue compiles to the dot, with no staging or store code.
    constexpr bool kDotOnly = REV && DOT;
    constexpr int NS = Lay::kStages;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~static_cast<uintptr_t>(1023));
    const uint32_t sbase = smem_u32(smem);

    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + Lay::kBarOff);
    uint64_t* full = bars;                 // [NS]
    uint64_t* empty = bars + 8;            // [NS]
    uint64_t* sc_full = bars + 16;         // [2] score in TMEM (front commit)
    uint64_t* sc_free = bars + 18;         // [2] score/P buffer reusable (back commit after PV)
    uint64_t* o_full = bars + 20;          // [2]
    uint64_t* o_free = bars + 22;          // [2]
    uint64_t* dz_full = bars + 24;         // [2]
    uint64_t* dz_free = bars + 26;         // [2]
    uint64_t* st_ready = bars + 28;        // [2]
    uint64_t* st_free = bars + 30;         // [2]
    uint64_t* item_full = bars + 48;       // [kRing]
    uint64_t* item_empty = bars + 52;      // [kRing]
    uint64_t* p_ready = bars + 36;         // [2] P written over the score buffer (P warps)
    uint64_t* o_staged = bars + 44;        // [2] output tile staged by all 4 epilogue warps
    uint64_t* o_buf_free = bars + 46;      // [2] output staging tile read by its TMA store
    uint64_t* a_full = bars + 60;          // [3] (REV, dot) tile of the dotted tensor landed
    uint64_t* a_empty = bars + 63;         // [3] (REV, dot) its dot formed
    uint64_t* z_pub = bars + 40;           // state warps: all rows written before a flag
    uint64_t* z_lb = bars + 41;            // state warps: look-back result broadcast
    uint64_t* z_ack = bars + 42;           // state warps: broadcast consumed
    uint64_t* drain = bars + 38;
    uint64_t* drain2 = bars + 39;
    uint64_t* p1_seen = bars + 34;         // every phase-1 stage of an item consumed
    int* misc = reinterpret_cast<int*>(bars + 56);
    volatile int* abort_flag = misc + 0;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(misc + 1);
    volatile unsigned int* lb_word = reinterpret_cast<volatile unsigned int*>(misc + 2);
    volatile int* item_slot = misc + 4;    // [kRing]

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    // (REV, dot) the ring of dotted tiles: the two output staging tiles, which a dot
    // read leaves idle, and one more
    auto a_tile = [&](uint32_t k) -> uint8_t* {
        return smem + (k < 2 ? Lay::kOOff + k * kTile : Lay::kAOff);
    };
    constexpr int kZActiveWarps = DQ / 32;          // state warps holding rows
    constexpr int kPHelpers = 4 - kZActiveWarps;    // state-slot warps building P half 1
    // REV (64-wide, separate q and k tiles) keeps the state rows in TMEM lanes 64..127,
    // so that the spare state-slot warps reach lanes 0..63, the rows whose P needs both
    // halves once the mask is reversed.
    static_assert(!REV || DQ == 64, "the reverse read is built for 64-wide q and k");

    if (threadIdx.x == 0) {
        for (int i = 0; i < NS; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 2);  // released by both MMA issuers
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&sc_full[i], 1);
            mbar_init(&sc_free[i], 1);
            mbar_init(&p_ready[i], 4 + kPHelpers);
            mbar_init(&o_staged[i], 4);
            mbar_init(&o_buf_free[i], 1);
            mbar_init(&o_full[i], 1);
            mbar_init(&o_free[i], 4);
            mbar_init(&dz_full[i], 1);
            mbar_init(&dz_free[i], kZActiveWarps);
            mbar_init(&st_ready[i], kZActiveWarps);
            mbar_init(&st_free[i], 1);
        }
        for (int i = 0; i < kRing; ++i) {
            mbar_init(&item_full[i], 1);
            mbar_init(&item_empty[i], kItemConsumers);
        }
        mbar_init(z_pub, kZActiveWarps);
        mbar_init(z_lb, 1);
        mbar_init(z_ack, kZActiveWarps);
        mbar_init(drain, 1);
        mbar_init(drain2, 1);
        mbar_init(p1_seen, 1);
        if constexpr (REV) {
            for (int i = 0; i < 3; ++i) {
                mbar_init(&a_full[i], 1);
                mbar_init(&a_empty[i], 4);  // the four epilogue warps
            }
        }
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, kTmemCols);
        tmem_relinquish();
        tc_fence_before();
    }
    if (warp == Roles<REV>::kProd && lane == 0) {
        prefetch_tmap(&tm_q);
        prefetch_tmap(&tm_k);
        prefetch_tmap(&tm_v);
        prefetch_tmap(&tm_o);
        if constexpr (FUSED) prefetch_tmap(&tm_o2);
    }
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == Roles<REV>::kProd) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            uint32_t n = 0, an = 0;
            bool ok = true;
            const bool dot = REV && p.epi.dot_out != nullptr;
            // Stream the stages of one pass of an item into the ring.
            auto load_pass = [&](const Item& I, int pass) {
                for (int c = 0; c < I.nch && ok; ++c, ++n) {
                    const int s = n % NS;
                    if (!mbar_wait(&empty[s], ((n / NS) & 1) ^ 1, abort_flag)) {
                        raise_error(p, kErrWaitTimeout, abort_flag);
                        ok = false;
                        break;
                    }
                    uint8_t* st = smem + s * Lay::kStageBytes;
                    const int t0 = chunk_t0<REV>(I, c);
                    mbar_arrive_expect_tx(&full[s], pass == 1 ? Lay::kTxPass1 : Lay::kTxPass2);
                    if constexpr (FUSED) {
                        tma_load_5d(st + Lay::kQOff, &tm_q, &full[s], 0, I.h, t0, I.b, I.l);
                        tma_load_5d(st + Lay::kVOff, &tm_k, &full[s], 0, I.h, t0, I.b, I.l);
                        if (pass == 2)
                            tma_load_5d(st + Lay::kGOff, &tm_v, &full[s], 0, I.h, t0, I.b, I.l);
                        continue;
                    }
                    if (COSTATE && pass == 2) {
#pragma unroll
                        for (int kb = 0; kb < Lay::kQkBlocks; ++kb)
                            tma_load_5d(st + Lay::kQOff + kb * kTile, &tm_q, &full[s], kb * 64, I.h,
                                        t0, I.b, I.l);
                    }
#pragma unroll
                    for (int kb = 0; kb < Lay::kQkBlocks; ++kb)
                        tma_load_5d(st + Lay::kKOff + kb * kTile, &tm_k, &full[s], kb * 64, I.h, t0,
                                    I.b, I.l);
                    tma_load_5d(st + Lay::kVOff, &tm_v, &full[s], I.j * 64, I.h, t0, I.b, I.l);
                    if (dot && pass == 2) {
                        // the dotted tensor's tile, through its own three-deep ring
                        const uint32_t k = an % 3;
                        if (!mbar_wait(&a_empty[k], ((an / 3) & 1) ^ 1, abort_flag)) {
                            raise_error(p, kErrWaitTimeout, abort_flag);
                            ok = false;
                            break;
                        }
                        mbar_arrive_expect_tx(&a_full[k], kTile);
                        tma_load_5d(a_tile(k), &tm_o, &a_full[k], I.j * 64, I.h, t0, I.b, I.l);
                        ++an;
                    }
                }
            };
            // Stage order: P1(i0), P1(i1), P2(i0), P1(i2), P2(i1), ...: phase 1 of a new
            // item is loaded before phase 2 of the previous one.
            int pending = -1;
            for (int it = 0; ok; ++it) {
                const int slot = it % kRing;
                if (!mbar_wait(&item_empty[slot], ((it / kRing) & 1) ^ 1, abort_flag)) {
                    raise_error(p, kErrWaitTimeout, abort_flag);
                    break;
                }
                int item = static_cast<int>(atomicAdd(p.ctrl, 1u));
                if (item >= p.n_items) item = -1;
                item_slot[slot] = item;
                mbar_arrive(&item_full[slot]);
                if (item >= 0) {
                    const Item I = decode_item<REV>(item, p);
                    if (I.phase1) load_pass(I, 1);
                }
                if (pending >= 0) load_pass(decode_item<REV>(pending, p), 2);
                pending = item;
                if (item < 0) break;
            }
            // Drain: every issued load has landed before the CTA can exit.
            if (*abort_flag) {
                for (int s = 0; s < NS; ++s) {
                    if (n > (uint32_t)s) {
                        uint32_t last = ((n - 1 - s) / NS) * NS + s;
                        mbar_drain(&full[s], (last / NS) & 1);
                    }
                }
                for (uint32_t k = 0; k < 3; ++k) {
                    if (an > k) {
                        const uint32_t last = ((an - 1 - k) / 3) * 3 + k;
                        mbar_drain(&a_full[k], (last / 3) & 1);
                    }
                }
            }
        }
    } else if (warp == Roles<REV>::kFront) {
        // ------------------------------------------------- front MMA issuer
        if (lane == 0) {
            constexpr uint32_t ID_SC = idesc_bf16(128, 128, false, false);  // Q K^T
            constexpr uint32_t ID_DZ = idesc_bf16(128, 64, true, true);     // K^T V
            uint32_t n = 0, c2 = 0, dzc = 0;
            bool ok = true;
            auto wait_or_fail = [&](uint64_t* bar, uint32_t par) -> bool {
                if (__builtin_expect(mbar_wait(bar, par, abort_flag), 1)) return true;
                raise_error(p, kErrWaitTimeout, abort_flag);
                return false;
            };
            // dZ += K^T V over one stage.  A = K^T is MN-major with 64-wide M blocks
            // 16 KB apart; for DQ = 64 the second M block is the V tile, whose rows
            // land in TMEM lanes 64..127 that nobody reads.
            auto issue_dz = [&](uint32_t st, uint32_t dcol, bool first) {
                // REV: A starts one block before k, so K^T lands in lanes 64..127
                const uint32_t a_lo = sdesc_lo(st + (REV ? Lay::kKOff - kTile : Lay::kKOff), kTile);
                const uint32_t b_lo = sdesc_lo(st + Lay::kVOff, kTile);
#pragma unroll kMmaUnroll
                for (int kk = 0; kk < kChunk / 16; ++kk)
                    mma_bf16_ss(tmem + dcol, sdesc_from_lo(a_lo + mnmaj_step(kk)),
                                sdesc_from_lo(b_lo + mnmaj_step(kk)), ID_DZ,
                                (first && kk == 0) ? 0u : 1u);
            };
            int pending = -1;
            for (int it = 0; ok; ++it) {
                const int slot = it % kRing;
                if (!wait_or_fail(&item_full[slot], (it / kRing) & 1)) break;
                const int item = item_slot[slot];
                mbar_arrive(&item_empty[slot]);
                // phase 1 of the new item: its segment aggregate sum K^T V
                if (item >= 0) {
                    const Item I = decode_item<REV>(item, p);
                    if (I.phase1) {
                        const uint32_t b = dzc & 1;
                        if (!(ok = wait_or_fail(&dz_free[b], ((dzc >> 1) & 1) ^ 1))) break;
                        tc_fence_after();
                        for (int c = 0; c < I.nch; ++c, ++n) {
                            const int s = n % NS;
                            if (!(ok = wait_or_fail(&full[s], (n / NS) & 1))) break;
                            tc_fence_after();
                            issue_dz(sbase + s * Lay::kStageBytes, col_dz(b), c == 0);
                            mma_commit(&empty[s]);
                            mma_commit(&empty[s]);  // the back issuer skips phase-1 stages
                        }
                        if (!ok) break;
                        mma_commit(&dz_full[b]);
                        ++dzc;
                        // every phase-1 stage of this item has been consumed: the back
                        // issuer, which skips them, may now wait on the full barriers
                        // after them (see there)
                        mma_commit(p1_seen);
                    }
                }
                // phase 2 of the previous item: score and dZ of every chunk (dZ of the
                // last chunk is not needed)
                if (pending >= 0) {
                    const Item I = decode_item<REV>(pending, p);
                    for (int c = 0; c < I.nch; ++c, ++n, ++c2) {
                        const int s = n % NS;
                        if (!(ok = wait_or_fail(&full[s], (n / NS) & 1))) break;
                        const uint32_t sb = c2 & 1;
                        // the score/P buffer is free once the PV product two chunks back is done
                        if (!(ok = wait_or_fail(&sc_free[sb], ((c2 >> 1) & 1) ^ 1))) break;
                        tc_fence_after();
                        const uint32_t st = sbase + s * Lay::kStageBytes;
                        const uint32_t q_lo = sdesc_lo(st + Lay::kQOff, 16);
                        const uint32_t k_lo = sdesc_lo(st + Lay::kKOff, 16);
#pragma unroll kMmaUnroll
                        for (int kk = 0; kk < DQ / 16; ++kk)
                            mma_bf16_ss(tmem + col_sc(sb), sdesc_from_lo(q_lo + kmaj_step(kk)),
                                        sdesc_from_lo(k_lo + kmaj_step(kk)), ID_SC, kk > 0 ? 1u : 0u);
                        mma_commit(&sc_full[sb]);
                        if constexpr (FUSED) {
                            // the costate read of the same chunk: score G Ghat^T into buffer 1
                            ++c2;
                            const uint32_t sb2 = c2 & 1;
                            if (!(ok = wait_or_fail(&sc_free[sb2], ((c2 >> 1) & 1) ^ 1))) break;
                            tc_fence_after();
                            const uint32_t g_lo = sdesc_lo(st + Lay::kGOff, 16);
                            const uint32_t h_lo = sdesc_lo(st + Lay::kVOff, 16);
#pragma unroll kMmaUnroll
                            for (int kk = 0; kk < DQ / 16; ++kk)
                                mma_bf16_ss(tmem + col_sc(sb2), sdesc_from_lo(g_lo + kmaj_step(kk)),
                                            sdesc_from_lo(h_lo + kmaj_step(kk)), ID_SC, kk > 0 ? 1u : 0u);
                            mma_commit(&sc_full[sb2]);
                        }
                        if (c < I.nch - 1) {
                            const uint32_t b = dzc & 1;
                            if (!(ok = wait_or_fail(&dz_free[b], ((dzc >> 1) & 1) ^ 1))) break;
                            tc_fence_after();
                            issue_dz(st, col_dz(b), true);
                            mma_commit(&dz_full[b]);
                            ++dzc;
                        }
                        mma_commit(&empty[s]);
                    }
                }
                pending = item;
                if (item < 0) break;
            }
            // Every MMA this thread issued has completed before TMEM is released.
            mma_commit(drain);
            mbar_drain(drain, 0);
        }
    } else if (warp == Roles<REV>::kBack) {
        // -------------------------------------------------- back MMA issuer
        if (lane == 0) {
            constexpr uint32_t ID_O = idesc_bf16(128, 64, false, true);  // Q S^T, P V
            uint32_t n = 0, c2 = 0, p1c = 0;
            bool ok = true;
            auto wait_or_fail = [&](uint64_t* bar, uint32_t par) -> bool {
                if (__builtin_expect(mbar_wait(bar, par, abort_flag), 1)) return true;
                raise_error(p, kErrWaitTimeout, abort_flag);
                return false;
            };
            int pending = -1;
            for (int it = 0; ok; ++it) {
                const int slot = it % kRing;
                if (!wait_or_fail(&item_full[slot], (it / kRing) & 1)) break;
                const int item = item_slot[slot];
                mbar_arrive(&item_empty[slot]);
                // The new item's phase-1 stages precede the previous item's phase 2 and
                // are consumed and released by the front issuer alone.  A ring slot whose
                // phase-1 load this issuer never waited for can still be a phase behind,
                // and a parity wait on it would then pass for the wrong round (and read
                // the slot before its phase-2 tile lands); so the front issuer's p1_seen
                // (its phase-1 products complete) comes first.  p1_seen cannot run two
                // phases ahead of this wait: between two phase-1 passes the ring holds the
                // phase-2 stages of a full segment (512 tokens or more; the shorter last
                // segments take the highest tickets, after every phase-1 item), and the
                // front issuer needs one of their slots, freed only by this issuer.
                if (item >= 0) {
                    const Item In = decode_item<REV>(item, p);
                    if (In.phase1) {
                        if (!(ok = wait_or_fail(p1_seen, p1c & 1))) break;
                        ++p1c;
                        n += In.nch;
                    }
                }
                if (FUSED && pending >= 0) {
                    // Both reads of a chunk: O_y = X S'^T and O_g = G S' from one S'^T tile
                    // (read MN-major for the forward, K-major for the costate), each
                    // followed by its P V product.  Each direction owns one O and one score
                    // buffer, used once per chunk; the S'^T tiles alternate by chunk.
                    constexpr uint32_t ID_OK = idesc_bf16(128, 64, false, false);  // G S'
                    const Item I = decode_item<REV>(pending, p);
                    for (int c = 0; c < I.nch; ++c, ++n, c2 += 2) {
                        const int s = n % NS;
                        const uint32_t cc = c2 >> 1;  // chunks of this CTA so far
                        const uint32_t sbb = cc & 1, sph = (cc >> 1) & 1, oph = cc & 1;
                        if (!(ok = wait_or_fail(&full[s], (n / NS) & 1))) break;
                        if (!(ok = wait_or_fail(&st_ready[sbb], sph))) break;
                        const uint32_t st = sbase + s * Lay::kStageBytes;
                        const uint32_t tile = sbase + Lay::kStOff + sbb * Lay::kStBytes;
                        // direction 0 (forward) completes before direction 1 waits for its
                        // O buffer, so the forward P V is never held up by the costate
                        // epilogue of the previous chunk
#pragma unroll 1
                        for (int dir = 0; dir < 2; ++dir) {
                            if (!(ok = wait_or_fail(&o_free[dir], oph ^ 1))) break;
                            tc_fence_after();
                            if (dir == 0) {
                                const uint32_t x_lo = sdesc_lo(st + Lay::kQOff, 16);
                                const uint32_t s_mn = sdesc_lo(tile, kTile);
#pragma unroll kMmaUnroll
                                for (int kk = 0; kk < DQ / 16; ++kk)
                                    mma_bf16_ss(tmem + col_o(0), sdesc_from_lo(x_lo + kmaj_step(kk)),
                                                sdesc_from_lo(s_mn + mnmaj_step(kk)), ID_O,
                                                kk > 0 ? 1u : 0u);
                            } else {
                                const uint32_t g_lo = sdesc_lo(st + Lay::kGOff, 16);
                                const uint32_t s_k = sdesc_lo(tile, 16);
#pragma unroll kMmaUnroll
                                for (int kk = 0; kk < DQ / 16; ++kk)
                                    mma_bf16_ss(tmem + col_o(1), sdesc_from_lo(g_lo + kmaj_step(kk)),
                                                sdesc_from_lo(s_k + kmaj_step(kk)), ID_OK,
                                                kk > 0 ? 1u : 0u);
                                mma_commit(&st_free[sbb]);  // both reads of the tile issued
                            }
                            if (!(ok = wait_or_fail(&p_ready[dir], oph))) break;
                            tc_fence_after();
                            // forward: V = ghat; costate: V = x (both MN-major [128 t][64])
                            const uint32_t v_lo = sdesc_lo(st + (dir == 0 ? Lay::kVOff : Lay::kQOff), kTile);
#pragma unroll kMmaUnroll
                            for (int kk = 0; kk < kChunk / 16; ++kk)
                                mma_bf16_ts(tmem + col_o(dir),
                                            tmem + col_sc(dir) + (kk < 4 ? kk * 8 : 64 + (kk - 4) * 8),
                                            sdesc_from_lo(v_lo + mnmaj_step(kk)), ID_O, 1u);
                            mma_commit(&o_full[dir]);
                            mma_commit(&sc_free[dir]);
                        }
                        if (!ok) break;
                        mma_commit(&empty[s]);
                    }
                } else if (pending >= 0) {
                    const Item I = decode_item<REV>(pending, p);
                    for (int c = 0; c < I.nch; ++c, ++n, ++c2) {
                        const int s = n % NS;
                        const uint32_t ob = c2 & 1, oph = (c2 >> 1) & 1;
                        if (!(ok = wait_or_fail(&full[s], (n / NS) & 1))) break;
                        if (!(ok = wait_or_fail(&o_free[ob], oph ^ 1))) break;
                        if (!(ok = wait_or_fail(&st_ready[ob], oph))) break;
                        tc_fence_after();
                        const uint32_t st = sbase + s * Lay::kStageBytes;
                        // O = Q S^T  (B = S^T tile [dq][64]: MN-major)
                        const uint32_t q_lo = sdesc_lo(st + Lay::kQOff, 16);
                        const uint32_t s_lo = sdesc_lo(sbase + Lay::kStOff + ob * Lay::kStBytes, kTile);
#pragma unroll kMmaUnroll
                        for (int kk = 0; kk < DQ / 16; ++kk)
                            mma_bf16_ss(tmem + col_o(ob), sdesc_from_lo(q_lo + kmaj_step(kk)),
                                        sdesc_from_lo(s_lo + mnmaj_step(kk)), ID_O, kk > 0 ? 1u : 0u);
                        mma_commit(&st_free[ob]);
                        if (!(ok = wait_or_fail(&p_ready[ob], oph))) break;
                        tc_fence_after();
                        // O += P V  (A = P in TMEM over the score buffer: tokens s < 64 in
                        // columns 0..31, s >= 64 in columns 64..95; B = V [128 t][64]: MN-major)
                        const uint32_t v_lo = sdesc_lo(st + Lay::kVOff, kTile);
#pragma unroll kMmaUnroll
                        for (int kk = 0; kk < kChunk / 16; ++kk)
                            mma_bf16_ts(tmem + col_o(ob),
                                        tmem + col_sc(ob) + (kk < 4 ? kk * 8 : 64 + (kk - 4) * 8),
                                        sdesc_from_lo(v_lo + mnmaj_step(kk)), ID_O, 1u);
                        mma_commit(&o_full[ob]);
                        mma_commit(&sc_free[ob]);
                        mma_commit(&empty[s]);
                    }
                }
                pending = item;
                if (item < 0) break;
            }
            mma_commit(drain2);
            mbar_drain(drain2, 0);
        }
    } else if (REV && warp == 1) {
        // the suffix read's issuers are warps 14 and 15: this warp only allocates TMEM
    } else if (warp < kWarpO0 ||
               (warp >= kWarpZ0 && (REV ? (warp & 3) < 2 : (warp & 3) >= kZActiveWarps))) {
        // ------------------------------------------------------ score -> P
        // Warps 2-5 build P; with 64-wide keys the two state-slot warps whose
        // lanes (64..127) hold no state rows build the second half of P for them.
        const bool helper = warp >= kWarpZ0;
        const int q4 = warp & 3;
        const int row = q4 * 32 + lane;
        const uint32_t lane_off = static_cast<uint32_t>(q4 * 32) << 16;
        uint32_t c2 = 0;
        for (int it = 0;; ++it) {
            const int slot = it % kRing;
            if (!warp_wait(&item_full[slot], (it / kRing) & 1, abort_flag)) {
                raise_error(p, kErrWaitTimeout, abort_flag);
                break;
            }
            const int item = item_slot[slot];
            __syncwarp();
            if (lane == 0) mbar_arrive(&item_empty[slot]);
            if (item < 0) break;
            const Item I = decode_item<REV>(item, p);
            bool ok = true;
            for (int c = 0; c < kJobs * I.nch; ++c, ++c2) {
                const uint32_t sb = c2 & 1;
                if (!warp_wait(&sc_full[sb], (c2 >> 1) & 1, abort_flag)) {
                    raise_error(p, kErrWaitTimeout, abort_flag);
                    ok = false;
                    break;
                }
                tc_fence_after();
                // Rows of this warp are 32*q4 .. 32*q4+31, so only columns s < 32*(q4+1)
                // survive the strict causal mask.  P row t packs (s, s+1) pairs as
                // bf16x2: tokens s < 64 into columns s/2 (0..31), tokens s >= 64 into
                // columns 64 + (s-64)/2 (64..95), each written only after the same
                // warp has read the score columns it overwrites.  Rows below 64 have
                // an all-zero second half; with 64-wide keys the second half of rows
                // 64..127 is built by the two spare state-slot warps.
                const uint32_t base = tmem + col_sc(sb) + lane_off;
#pragma unroll 1
                for (int half = 0; half < 2; ++half) {
                    // REV keeps tokens s > t: rows >= 64 have an all-zero first half, and
                    // rows < 64 (whose lanes no helper warp can reach) build both halves
                    const bool mine =
                        REV ? (q4 < 2 ? (half == 0 ? !helper : helper) : !helper)
                            : (half == 0 ? !helper : (q4 < 2 ? !helper : (helper || kPHelpers == 0)));
                    if (!mine) continue;
                    if ((REV ? (half == 0 && q4 >= 2) : (half == 1 && q4 < 2)) || p.mu == 0.0f) {
                        // rows < 64: tokens >= 64 all masked; eta = 0: no P at all
                        tmem_zero32_async(base + half * 64);
                        continue;
                    }
#pragma unroll 1
                    for (int sub = 0; sub < 2; ++sub) {
                        float v[32];
                        uint32_t w[16];
                        tmem_ld32(base + half * 64 + sub * 32, v);
#pragma unroll
                        for (int i = 0; i < 16; ++i) {
                            const int s0 = half * 64 + sub * 32 + 2 * i;
                            if constexpr (REV)
                                w[i] = pack_bf16x2(s0 > row ? v[2 * i] : 0.0f,
                                                   s0 + 1 > row ? v[2 * i + 1] : 0.0f);
                            else
                                w[i] = pack_bf16x2(s0 < row ? v[2 * i] : 0.0f,
                                                   s0 + 1 < row ? v[2 * i + 1] : 0.0f);
                        }
                        tmem_st16_async(base + half * 64 + sub * 16, w);
                    }
                }
                tmem_wait_st();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&p_ready[sb]);
            }
            if (!ok) break;
        }
    } else if (warp < kWarpZ0) {
        // ------------------------------------------------- output epilogue
        const int q4 = warp & 3;
        const int row = q4 * 32 + lane;
        const uint32_t lane_off = static_cast<uint32_t>(q4 * 32) << 16;
        const bool storer = (warp == kWarpO0) && (lane == 0);  // issues the TMA stores
        const EpiParams& e = p.epi;
        uint32_t c2 = 0;
        // (REV, dot) each chunk's tile of the dotted tensor arrives through the producer's
        // three-deep ring (no rows are stored)
        uint32_t ae = 0;
        for (int it = 0;; ++it) {
            const int slot = it % kRing;
            if (!warp_wait(&item_full[slot], (it / kRing) & 1, abort_flag)) {
                raise_error(p, kErrWaitTimeout, abort_flag);
                break;
            }
            const int item = item_slot[slot];
            __syncwarp();
            if (lane == 0) mbar_arrive(&item_empty[slot]);
            if (item < 0) break;
            const Item I = decode_item<REV>(item, p);
            bool ok = true;
            for (int jb = 0; jb < kJobs * I.nch; ++jb, ++c2) {
                // FUSED: job 2c is chunk c's forward read (y), job 2c+1 its costate read
                const int c = FUSED ? (jb >> 1) : jb;
                const int dir = FUSED ? (jb & 1) : 0;
                const uint32_t ob = c2 & 1, oph = (c2 >> 1) & 1;
                if (!warp_wait(&o_full[ob], oph, abort_flag)) {
                    raise_error(p, kErrWaitTimeout, abort_flag);
                    ok = false;
                    break;
                }
                tc_fence_after();
                float v[64];
                tmem_ld64(tmem + col_o(ob) + lane_off, v);
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&o_free[ob]);
                // O = lam * (Q S'^T + L(Q K^T) V); a suffix read reduced to its per-row dot
                // alone takes lam into the dot's scale instead
                constexpr bool dot_only = kDotOnly;
                if (!dot_only) {
#pragma unroll
                    for (int i = 0; i < 64; ++i) v[i] *= p.lam;
                }
                const int t0 = chunk_t0<REV>(I, c);
                const int t = t0 + row;
                const int col0 = I.j * 64;
                const bool valid = REV ? (t >= I.t_begin && t < I.t_end) : t < I.t_end;
                // The activation paths (MLP layers only) run out of line, so the hot
                // loop of the plain scans stays small in the instruction cache.
                if (!kDotOnly && e.zin && valid) {
                    float tmp[64];
#pragma unroll
                    for (int i = 0; i < 64; ++i) tmp[i] = v[i];
                    epi_apply_dact(e, tok_off(e.z_str, I.l, I.b, t, I.h) + col0, tmp);
#pragma unroll
                    for (int i = 0; i < 64; ++i) v[i] = tmp[i];
                }
                if (!kDotOnly && e.out2 && valid) {
                    float tmp[64];
#pragma unroll
                    for (int i = 0; i < 64; ++i) tmp[i] = v[i];
                    epi_store_act(e, tok_off(e.out2_str, I.l, I.b, t, I.h) + col0, tmp);
                }
                if constexpr (FUSED) {
                    // consistency term of the costate read against the given proposals
                    if (dir == 1 && e.cons_out && valid) {
                        float tmp[64];
#pragma unroll
                        for (int i = 0; i < 64; ++i) tmp[i] = v[i];
                        epi_consistency(e, tok_off(e.cons_str, I.l, I.b, t, I.h) + col0, tmp,
                                        (((long long)I.l * p.B + I.b) * p.T + t) * p.H + I.h);
                    }
                }
                // (REV) dot_out[t] (+)= dot_scale * (row . a row) over this 64-wide tile.
                // The tile of a (TMA, 128B-swizzled like an output tile) lets each lane
                // read its own row without bank conflicts.
                auto row_dot = [&]() -> bool {
                    const uint32_t ak = ae % 3;
                    if (!warp_wait(&a_full[ak], (ae / 3) & 1, abort_flag)) {
                        raise_error(p, kErrWaitTimeout, abort_flag);
                        return false;
                    }
                    const uint32_t atile = smem_u32(a_tile(ak));
                    float acc = 0.f;
#pragma unroll
                    for (int q = 0; q < 8; ++q) {
                        const uint4 a4 = ld_shared_v4(atile + sw128_off(row, q));
                        const __nv_bfloat16* hb = reinterpret_cast<const __nv_bfloat16*>(&a4);
#pragma unroll
                        for (int i = 0; i < 8; ++i) acc = fmaf(v[8 * q + i], __bfloat162float(hb[i]), acc);
                    }
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&a_empty[ak]);
                    ++ae;
                    if (valid) {
                        float* dst = e.dot_out + (((long long)I.l * p.B + I.b) * p.T + t) * p.H + I.h;
                        const float sc = dot_only ? e.dot_scale * p.lam : e.dot_scale;
                        if (p.n_tiles > 1)
                            atomicAdd(dst, sc * acc);
                        else
                            *dst = sc * acc;
                    }
                    return true;
                };
                if constexpr (kDotOnly) {
                    if (!row_dot()) {
                        ok = false;
                        break;
                    }
                    continue;  // no rows staged or stored
                }
                // Stage the bf16 row in the 128B-swizzled output tile (the TMA store
                // clips rows past the end of the sequence).
                if (!warp_wait(&o_buf_free[ob], oph ^ 1, abort_flag)) {
                    raise_error(p, kErrWaitTimeout, abort_flag);
                    ok = false;
                    break;
                }
                const uint32_t otile = sbase + Lay::kOOff + ob * kTile;
                // (REV only) a chunk starting before token 0 is stored row by row, and a
                // suffix read reduced to a per-token dot stores no rows at all
                const bool direct = REV && (t0 < 0 || e.out == nullptr);
                if constexpr (REV) {
                    if (e.dot_out && !row_dot()) {
                        ok = false;
                        break;
                    }
                }
                if (direct) {
                    if (valid && e.out) {
                        float tmp[64];  // a copy, so that v itself stays in registers
#pragma unroll
                        for (int i = 0; i < 64; ++i) tmp[i] = v[i];
                        epi_store_row(e, tok_off(e.out_str, I.l, I.b, t, I.h) + col0, tmp);
                    }
                } else {
#pragma unroll
                for (int q = 0; q < 8; ++q)
                    st_shared_v4(otile + sw128_off(row, q), pack_bf16x2(v[8 * q], v[8 * q + 1]),
                                 pack_bf16x2(v[8 * q + 2], v[8 * q + 3]),
                                 pack_bf16x2(v[8 * q + 4], v[8 * q + 5]),
                                 pack_bf16x2(v[8 * q + 6], v[8 * q + 7]));
                }
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) mbar_arrive(&o_staged[ob]);
                if (storer) {
                    if (!mbar_wait(&o_staged[ob], oph, abort_flag)) {
                        raise_error(p, kErrWaitTimeout, abort_flag);
                        ok = false;
                    } else {
                        if (!direct)
                            tma_store_5d(dir ? &tm_o2 : &tm_o, smem + Lay::kOOff + ob * kTile, col0,
                                         I.h, t0, I.b, I.l);
                        bulk_commit_group();
                        // the previous chunk's store (other tile) has finished reading
                        bulk_wait_group_read<1>();
                        if (c2 > 0) mbar_arrive(&o_buf_free[ob ^ 1]);
                    }
                }
                if (!__shfl_sync(0xffffffffu, ok ? 1 : 0, 0)) {
                    ok = false;
                    break;
                }
            }
            if (!ok) break;
        }
        if (storer) bulk_wait_group_all();
    } else {
        const int q4 = warp & 3;
        {
        // ------------------------------------------------------------ state
        const int row = q4 * 32 + lane;         // TMEM lane of this thread's state row
        const int srow = REV ? row - 64 : row;  // contraction index q of that row
        const bool active = REV ? row >= 64 : row < DQ;  // warp-uniform
        constexpr int kLeadQ4 = REV ? 2 : 0;    // lane quarter of the lead state warp
        const bool leader = (q4 == kLeadQ4) && (lane == 0);
        const uint32_t lane_off = static_cast<uint32_t>(q4 * 32) << 16;
        // The state is kept in units of lam = -eta (1 when eta = 0): the rows hold
        // S' = S / lam, so the S^T tile carries the -eta of P and the update is
        // S' += mu * dZ with mu = -eta / lam (1, or 0 when eta = 0).
        uint32_t c2 = 0, dzc = 0, pubc = 0, lbc = 0;
        float st[64];
        const size_t blk = (size_t)DQ * 64;
        int pending = -1;
        for (int it = 0;; ++it) {
            const int slot = it % kRing;
            if (!warp_wait(&item_full[slot], (it / kRing) & 1, abort_flag)) {
                raise_error(p, kErrWaitTimeout, abort_flag);
                break;
            }
            const int new_item = item_slot[slot];
            __syncwarp();
            if (lane == 0) mbar_arrive(&item_empty[slot]);
            bool ok = true;
            // Publish an item's look-back status once every active state thread's
            // rows are globally visible: all arrive and all wait (a full barrier),
            // then the leader releases the flag.
            auto publish = [&](int item, unsigned int flag) -> bool {
                __threadfence();
                __syncwarp();
                if (lane == 0) mbar_arrive(z_pub);
                const bool okp = warp_wait(z_pub, pubc & 1, abort_flag);
                ++pubc;
                if (!okp) {
                    raise_error(p, kErrWaitTimeout, abort_flag);
                    return false;
                }
                // (failure tests only: one item may be told never to publish)
                if (leader && item != p.test_skip_publish) st_release_gpu(p.flags + item, flag);
                return true;
            };
            // ---- phase 1 of the newly taken item (before phase 2 of the previous one)
            if (new_item >= 0) {
                const int item = new_item;
                const Item I = decode_item<REV>(item, p);
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
                        float* dst = (I.k == 0 ? p.incl : p.agg) + (size_t)item * blk + (size_t)srow * 64;
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
                    if (active && !publish(item, I.k == 0 ? 2u : 1u)) break;
                }
            }
            // ---- look-back and phase 2 of the previous item
            if (pending >= 0) {
                const int item = pending;
                const Item I = decode_item<REV>(item, p);
                const int n_ut = p.n_ut;
                const int r_ut = item - I.k * n_ut;
                // ---- look-back: E = sum of the earlier segments' aggregates, stopping at
                // the nearest inclusive prefix.  The lead state warp polls up to 32
                // predecessor flags at once (lane i: segment k-1-i) and a ballot finds
                // the nearest inclusive prefix; one broadcast (count << 1 |
                // ends-at-inclusive) tells every state thread what to sum.
#pragma unroll
                for (int i = 0; i < 64; ++i) st[i] = 0.0f;
                if (active && I.k > 0) {
                    if (q4 == kLeadQ4) {
                        // predecessor segment sk of this (unit, tile) is item sk * n_ut + r_ut
                        int total = 0, base_pred = I.k - 1, remaining = I.k;
                        bool found = false, timed_out = false;
                        const uint64_t t0 = globaltimer_ns();
                        while (!found && !timed_out && remaining > 0) {
                            const int n = remaining < 32 ? remaining : 32;
                            unsigned int f = 1u;
                            if (lane < n) {
                                while ((f = ld_acquire_gpu(p.flags + (base_pred - lane) * n_ut + r_ut)) == 0u) {
                                    if (globaltimer_ns() - t0 > p.lookback_limit_ns) {
                                        f = 0xFFFFFFFFu;
                                        break;
                                    }
                                    __nanosleep(32);
                                }
                            }
                            if (__ballot_sync(0xffffffffu, f == 0xFFFFFFFFu)) {
                                timed_out = true;
                                break;
                            }
                            const unsigned int incl = __ballot_sync(0xffffffffu, lane < n && f == 2u);
                            if (incl) {
                                total += __ffs(incl);  // up to and including the nearest inclusive
                                found = true;
                            } else {
                                total += n;
                                base_pred -= n;
                                remaining -= n;
                            }
                        }
                        if (lane == 0) {
                            unsigned int word = ((unsigned int)total << 1) | (found ? 1u : 0u);
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
                        __syncwarp();
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
                            const int pred = (I.k - 1 - i) * n_ut + r_ut;
                            const float* src = ((i == cnt - 1 && ends_incl) ? p.incl : p.agg) +
                                               (size_t)pred * blk + (size_t)srow * 64;
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
                    const float* own = p.agg + (size_t)item * blk + (size_t)srow * 64;
                    float* dst = p.incl + (size_t)item * blk + (size_t)srow * 64;
    #pragma unroll
                    for (int i = 0; i < 64; i += 4) {
                        float4 a = __ldcg(reinterpret_cast<const float4*>(own + i));
                        *reinterpret_cast<float4*>(dst + i) =
                            make_float4(st[i] + a.x, st[i + 1] + a.y, st[i + 2] + a.z, st[i + 3] + a.w);
                    }
                    if (!publish(item, 2u)) break;
                }
                // ---- starting state S'^T row = (B0^T row - eta * E) / lam (REV: no base)
                if (REV && active) {
    #pragma unroll
                    for (int i = 0; i < 64; ++i) st[i] *= p.mu;
                } else if (active) {
                    const float* w0 = p.W0 + (size_t)(I.l * p.H + I.h) * p.dq * p.dv;
                    const int v0 = I.j * 64;
                    if (p.w0_transposed) {
                        const float* r = w0 + (size_t)row * p.dv + v0;  // W0 [dq][dv]
    #pragma unroll
                        for (int i = 0; i < 64; i += 4) {
                            float4 a = *reinterpret_cast<const float4*>(r + i);
                            st[i] = a.x * p.inv_lam + p.mu * st[i];
                            st[i + 1] = a.y * p.inv_lam + p.mu * st[i + 1];
                            st[i + 2] = a.z * p.inv_lam + p.mu * st[i + 2];
                            st[i + 3] = a.w * p.inv_lam + p.mu * st[i + 3];
                        }
                    } else {
    #pragma unroll
                        for (int i = 0; i < 64; ++i)  // W0 [dv][dq]: column `row`
                            st[i] = w0[(size_t)(v0 + i) * p.dq + row] * p.inv_lam + p.mu * st[i];
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
                            st_shared_v4(tile + sw128_off(srow, q), pack_bf16x2(st[8 * q], st[8 * q + 1]),
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
                                for (int i = 0; i < 32; ++i) st[h * 32 + i] += p.mu * a[i];
                            }
                        }
                        tc_fence_before();
                        __syncwarp();
                        if (lane == 0) mbar_arrive(&dz_free[b]);
                        ++dzc;
                    }
                }
            }
            if (!ok) break;
            pending = new_item;
            if (new_item < 0) break;
        }
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
template <int DQ, bool COSTATE, bool REV, bool FUSED = false, bool DOT = false>
static cudaError_t launch_one(const CUtensorMap& q, const CUtensorMap& k, const CUtensorMap& v,
                              const CUtensorMap& o, const TcScanParams& p, int grid,
                              cudaStream_t stream, const CUtensorMap* o2 = nullptr) {
    using Lay = TcLayout<DQ, COSTATE, REV, FUSED>;
    auto kern = tc_scan_kernel<DQ, COSTATE, REV, FUSED, DOT>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         Lay::kSmemBytes);
    if (e != cudaSuccess) return e;
    kern<<<grid, Roles<REV>::kThreads, Lay::kSmemBytes, stream>>>(q, k, v, o, o2 ? *o2 : o, p);
    return cudaGetLastError();
}

cudaError_t launch_tc_scan(const CUtensorMap& q, const CUtensorMap& k, const CUtensorMap& v,
                           const CUtensorMap& o, const TcScanParams& p, bool costate, int grid,
                           cudaStream_t stream) {
    if (p.dq == 64)
        return costate ? launch_one<64, true, false>(q, k, v, o, p, grid, stream)
                       : launch_one<64, false, false>(q, k, v, o, p, grid, stream);
    if (p.dq == 128)
        return costate ? launch_one<128, true, false>(q, k, v, o, p, grid, stream)
                       : launch_one<128, false, false>(q, k, v, o, p, grid, stream);
    return cudaErrorInvalidValue;
}

// Both reads of 64-wide maps in one pass: q = x, k = ghat, v = g_out; o = y, o2 = g_in.
cudaError_t launch_tc_fused(const CUtensorMap& x, const CUtensorMap& ghat, const CUtensorMap& gout,
                            const CUtensorMap& y, const CUtensorMap& gin, const TcScanParams& p,
                            int grid, cudaStream_t stream) {
    if (p.dq != 64 || p.dv != 64) return cudaErrorInvalidValue;
    return launch_one<64, false, false, true>(x, ghat, gout, y, p, grid, stream, &gin);
}

// The anti-causal suffix read r_t = sum_{s>t} (k_s . q_t) v_s (no base matrix) on the
// 64-wide kernel: shared_qk when q and k are one tensor (one tile per chunk).
cudaError_t launch_tc_suffix(const CUtensorMap& q, const CUtensorMap& k, const CUtensorMap& v,
                             const CUtensorMap& o, const TcScanParams& p, bool shared_qk, int grid,
                             cudaStream_t stream) {
    if (p.dq != 64) return cudaErrorInvalidValue;
    const bool dot_only = p.epi.dot_out && !p.epi.out && !p.epi.zin && !p.epi.out2;
    if (dot_only)
        return shared_qk ? launch_one<64, false, true, false, true>(q, k, v, o, p, grid, stream)
                         : launch_one<64, true, true, false, true>(q, k, v, o, p, grid, stream);
    return shared_qk ? launch_one<64, false, true>(q, k, v, o, p, grid, stream)
                     : launch_one<64, true, true>(q, k, v, o, p, grid, stream);
}

}  // namespace gl
