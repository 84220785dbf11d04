// scan_decay_tc.cu -- tensor-core (tcgen05) chunked scan with retention, for bf16
// maps of 64 x 64: Eq. 2 with per-token step sizes eta_t and retention alpha_t and
// the decay centred at the slow weights,
//
//     W_{t+1} = W0 + alpha_t (W_t - W0) - eta_t ghat_t x_t^T,     W_0 = W0,
//
// read before each write (Sec. 3, "Observation"; Eqs. 3-4; Appendix C).  In the
// orientation shared by both reads, with S the fast weights minus W0 (transposed so
// that rows are the read's contraction index q):
//   forward  q = k = x, v = ghat, B0 = W0,   S^T = (W - W0)^T   [d][m]
//   costate  q = g_out, k = ghat, v = x, B0 = W0^T, S^T = (W - W0) [m][d]
// and over a chunk of C = 128 tokens from the state S at its first token,
//
//   o_t = B0 q_t + a_t S q_t - sum_{s<t} E_ts (k_s . q_t) v_s
//   S'  = a_end S - sum_s w_s v_s k_s^T
//
// with a_t = prod_{r<t} alpha_r, E_ts = eta_s prod_{s<r<t} alpha_r,
// w_s = eta_s prod_{r>s} alpha_r and a_end the product of the chunk's alphas
// (indices local to the chunk; tokens past T carry alpha = 1, eta = 0).  The decays
// are plain products of alphas, never ratios or logarithms, so a reset (alpha = 0)
// and underflow give exact zeros and any real alpha is valid.  They are assembled
// from 8-token pieces: sig_s (alphas after s to the end of its piece), pim_t (alphas
// from the start of t's piece up to t) and the piece products tp_j, so that for s in
// an earlier piece than t, E_ts = (eta_s sig_s) * pim_t * prod_{js<i<jt} tp_i.
//
// The read lands in one 128-column TMEM accumulator X:
//   X  = Q [B0^T | S^T]         one N = 128 product: B0^T (per unit) and the chunk's
//                               S^T are the two 64-wide halves of the B operand
//   X[:, 0:64] += P' V          P'_ts = -E_ts (q_t . k_s), built over the score
// and the epilogue forms o_t = X_t[0:64] + a_t X_t[64:128] in fp32.  The state
// update is dZ = K^T (W V), with the rows of V scaled by -w_s into a shared-memory
// tile, then S' = a_end S + dZ in the state warps (fp32 rows).  TMEM holds two chunk
// buffers (score, then P' and dZ in its columns) and two X accumulators, so the
// issuers work on chunk c + 1 while the epilogue drains chunk c.
//
// Warp roles (16 warps), with the rings and bounded waits of the chunk kernel of
// scan_tc.cu:
//   warp 14     TMA producer (stage = [q | k | v], or [qk | v] forward)
//   warp 1      front MMA issuer: the score Q K^T of chunk c + 1, then (P' of chunk
//               c built, so its score columns are free) dZ of chunk c into them
//   warp 0      back MMA issuer: X of chunk c, then (P' ready) P' V
//               (each group's K steps back to back on one accumulator)
//   warp 15     gate factors of each chunk from alpha_t and eta_t, in registers and
//               shuffles, into a ring of three blocks one or two chunks ahead
//   warps 2-5   P' over score columns 0..63 (rows 0..63 also zero 64..127)
//   warps 10-11 P' over columns 64..127 of rows 64..127
//   (warps 4-5 and 10-11, whose P' rows are the shorter ones, then write the chunk's
//   W V rows 0..63 and 64..127)
//   warps 6-9   the epilogue (TMEM -> o_t -> bf16 staging -> TMA store)
//   warps 12-13 state rows, B0^T and S^T tiles, S' = a_end S + dZ
// One work item is one unit, or one segment of a few long units (its chunks run in
// order in one CTA; the segments' start states come from an aggregate pass and the
// carry kernel below).
#include <cuda.h>

#include "scan_common.cuh"
#include "sm103_ptx.cuh"

namespace gl {
namespace dec {

constexpr int kChunk = 128;
constexpr int kTile = 16384;   // [128 rows][64 bf16], 128-byte swizzle
constexpr int kStTile = 8192;  // [64 rows][64 bf16]
constexpr int kWarps = 16;
constexpr int kThreads = kWarps * 32;
// Both MMA issuers sit on sub-partitions 0 and 1 (warp % 4), whose P warps build the
// half-masked rows: a warp issuing ALU work every cycle on an issuer's sub-partition
// slows its MMAs by 1.7x, one on another sub-partition not at all.  The TMA producer
// issues a few instructions a chunk and takes sub-partition 2.
constexpr int kWarpO0 = 6, kWarpZ0 = 10, kWarpBack = 0, kWarpProd = 14, kWarpGate = 15;
constexpr int kRing = 4;
constexpr int kItemConsumers = 2 + 4 + 4 + 2 + 2 + 1;
constexpr uint32_t kTmemCols = 512;
// TMEM columns: two chunk buffers of 128 (the fp32 score; then P' packed in columns
// 0..31 (tokens s < 64) and 96..127 (s >= 64), and the state update dZ of the same
// chunk in columns 32..95) and two X accumulators of 128.
__host__ __device__ constexpr uint32_t col_sc(uint32_t i) { return i * 128u; }
constexpr uint32_t kDzCol = 32, kPhiCol = 96;
__host__ __device__ constexpr uint32_t col_x(uint32_t i) { return 256u + i * 128u; }

// Gate block of one chunk (floats), written by the gate warp: per token alpha, eta,
// -eta_s sig_s, pim_t, a_t and w_t; the products between pieces
// tpm[j][jt] = prod_{j<i<jt} tp_i (0 for j >= jt) and a_end.
constexpr int kGbAl = 0, kGbEt = 128, kGbNse = 256, kGbPim = 384, kGbA = 512, kGbW = 640;
constexpr int kGbTpm = 768, kGbEnd = 1024;
constexpr int kGbFloats = 1032;  // a multiple of 8 floats: every block 32-byte aligned
constexpr int kGbBytes = kGbFloats * 4;
constexpr int kGbRing = 3;

template <bool COSTATE>
struct DLayout {
    static constexpr int kQOff = 0;
    static constexpr int kKOff = COSTATE ? kTile : 0;
    static constexpr int kVOff = COSTATE ? 2 * kTile : kTile;
    static constexpr int kStageBytes = (COSTATE ? 3 : 2) * kTile;
    // fixed regions: the output staging tile, the B0^T tile followed by the two S^T
    // tiles (the N = 128 operand [B0^T | S^T] of buffer i has its halves
    // (i + 1) * kStTile apart), the W V tile, the ring of gate blocks, barriers
    static constexpr int kFixed = kTile + 2 * kStTile + kStTile + kTile + kGbRing * kGbBytes;
    static constexpr int kAvail = 232448 - kFixed - 1024 - 1024;
    static constexpr int kStages0 = kAvail / kStageBytes;
    static constexpr int kStages = kStages0 > 6 ? 6 : kStages0;
    static constexpr int kOOff = kStages * kStageBytes;
    static constexpr int kB0Off = kOOff + kTile;
    static constexpr int kStOff = kB0Off + kStTile;
    static constexpr int kWvOff = kStOff + 2 * kStTile;
    static constexpr int kGfOff = kWvOff + kTile;
    static constexpr int kBarOff = kGfOff + kGbRing * kGbBytes;
    static constexpr int kSmemBytes = kBarOff + 1024 + 1024;
    static_assert(kStages >= 3, "a chunk and the next chunk's score hold two stages");
    static_assert(kSmemBytes <= 232448, "shared memory budget exceeded");
    static_assert(kGfOff % 32 == 0 && kBarOff % 8 == 0, "alignment");
};

// One work item: segment k (tokens [t_begin, t_end)) of one unit.  Items are
// segment-major: item = k * n_ut + unit, with n_ut the number of units.
struct Item {
    int l, b, h, k, t_begin, t_end, nch;
};

__device__ __forceinline__ Item decode_unit(int item, const TcScanParams& p) {
    Item I;
    const int unit = item % p.n_ut;
    I.k = item / p.n_ut;
    I.h = unit % p.H;
    const int lb = unit / p.H;
    I.b = lb % p.B;
    I.l = lb / p.B;
    I.t_begin = I.k * p.seg_len;
    I.t_end = min(p.T, I.t_begin + p.seg_len);
    I.nch = (I.t_end - I.t_begin + kChunk - 1) / kChunk;
    return I;
}

// Out of line, like the slow half of every wait: sixteen warps run different role
// loops, instruction fetch is the first stall, and cold code inside a hot loop spreads
// it over more cache lines.  For the same reason the MMA issuers keep their K steps as
// rolled loops.
__device__ __noinline__ void raise_error(const TcScanParams& p, unsigned int bits,
                                         volatile int* abort_flag) {
    atomicOr(p.ctrl + 1, bits);
    if (abort_flag) *abort_flag = 1;
}

__device__ __forceinline__ void mbar_drain(uint64_t* bar, uint32_t parity) {
    uint64_t t0 = globaltimer_ns();
    while (!mbar_try_wait(bar, parity)) {
        if (globaltimer_ns() - t0 > 200000000ull) break;  // 0.2 s
    }
}

// One non-blocking probe of a barrier phase.
__device__ __forceinline__ bool test_probe(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}\n"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}
// The bounded wait, out of line so that the kernel's many wait sites share one copy
// (instruction-cache footprint).  Up to 64 non-blocking probes first: a thread parked
// by the suspending wait resumes a few thousand cycles after a thread-side arrival,
// which on the hand-offs between roles here costs more than the spin's issue slots.
__device__ __noinline__ bool wait_slow(uint64_t* bar, uint32_t parity, volatile int* abort_flag) {
    for (int i = 0; i < 64; ++i)
        if (test_probe(bar, parity)) return true;
    return mbar_wait(bar, parity, abort_flag);
}
__device__ __forceinline__ bool bwait(uint64_t* bar, uint32_t parity, volatile int* abort_flag) {
    return __builtin_expect(test_probe(bar, parity), 1) || wait_slow(bar, parity, abort_flag);
}

__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag) {
    const int lane = threadIdx.x & 31;
    int ok = 1;
    if (lane == 0) ok = bwait(bar, parity, abort_flag) ? 1 : 0;
    ok = __shfl_sync(0xffffffffu, ok, 0);
    __syncwarp();
    return ok != 0;
}

__host__ __device__ constexpr uint32_t kmaj_step(int kk) {
    return (uint32_t)(((kk >> 2) * kTile + (kk & 3) * 32) >> 4);
}
__host__ __device__ constexpr uint32_t mnmaj_step(int kk) { return (uint32_t)((kk * 2048) >> 4); }

__device__ __forceinline__ float4 lds4(const float* p) { return *reinterpret_cast<const float4*>(p); }

// v *= sigma'(z) / out2 = sigma(v) for one 64-wide output row (MLP layer fusion).
__device__ __noinline__ void epi_apply_dact(const EpiParams& e, long long z_off, float* v) {
    const __nv_bfloat16* zp = static_cast<const __nv_bfloat16*>(e.zin) + z_off;
    for (int q = 0; q < 8; ++q) {
        const uint4 zz = *reinterpret_cast<const uint4*>(zp + 8 * q);
        const __nv_bfloat16* zb = reinterpret_cast<const __nv_bfloat16*>(&zz);
#pragma unroll
        for (int i = 0; i < 8; ++i) v[8 * q + i] *= act_df(e.act, __bfloat162float(zb[i]));
    }
}
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

// -E_ts for the tokens s = 8 jt + i of t's own piece: -eta_s prod_{s<r<t} alpha_r for
// s < t, else 0.
__device__ __forceinline__ void same_piece_decays(const float* gb, int row, float (&ndd)[8]) {
    const int jt = row >> 3, it = row & 7;
    const float4 a0 = lds4(gb + kGbAl + 8 * jt), a1 = lds4(gb + kGbAl + 8 * jt + 4);
    const float4 e0 = lds4(gb + kGbEt + 8 * jt), e1 = lds4(gb + kGbEt + 8 * jt + 4);
    const float al[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
    const float et[8] = {e0.x, e0.y, e0.z, e0.w, e1.x, e1.y, e1.z, e1.w};
    float run = 1.0f;
#pragma unroll
    for (int i = 7; i >= 0; --i) {
        const bool lt = i < it;
        ndd[i] = lt ? -et[i] * run : 0.0f;
        run = lt ? run * al[i] : run;
    }
}

// Two 32-column loads of this thread's TMEM lane (32x32b shape, as tmem_ld32) with
// one wait: columns ta .. ta+31 into a, tb .. tb+31 into b.
__device__ __forceinline__ void tmem_ld32_pair(uint32_t ta, uint32_t tb, float (&a)[32], float (&b)[32]) {
    uint32_t r[64];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
        "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%64];\n\t"
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%32, %33, %34, %35, %36, %37, %38, %39, %40, %41, %42, %43, %44, %45, %46, %47, "
        "%48, %49, %50, %51, %52, %53, %54, %55, %56, %57, %58, %59, %60, %61, %62, %63}, [%65];\n\t"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
          "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
          "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
          "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
          "=r"(r[31]), "=r"(r[32]), "=r"(r[33]), "=r"(r[34]), "=r"(r[35]), "=r"(r[36]),
          "=r"(r[37]), "=r"(r[38]), "=r"(r[39]), "=r"(r[40]), "=r"(r[41]), "=r"(r[42]),
          "=r"(r[43]), "=r"(r[44]), "=r"(r[45]), "=r"(r[46]), "=r"(r[47]), "=r"(r[48]),
          "=r"(r[49]), "=r"(r[50]), "=r"(r[51]), "=r"(r[52]), "=r"(r[53]), "=r"(r[54]),
          "=r"(r[55]), "=r"(r[56]), "=r"(r[57]), "=r"(r[58]), "=r"(r[59]), "=r"(r[60]),
          "=r"(r[61]), "=r"(r[62]), "=r"(r[63])
        : "r"(ta), "r"(tb)
        : "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) {
        a[i] = __uint_as_float(r[i]);
        b[i] = __uint_as_float(r[32 + i]);
    }
}

// P'_ts = -E_ts (q_t . k_s) over the 64 score columns of pieces pb .. pb+7 of this
// lane's row: the fp32 scores at TMEM columns rd .. rd+63 become 32 packed bf16
// columns at wr (stores issued, not waited), two pieces per step.  Pieces 0..7
// (wr = rd) go in increasing order, pieces 8..15 (wr = rd + 32) in decreasing
// order, so that no packed store reaches a score column still to be read.  One copy
// of the code serves every P warp.
__device__ __forceinline__ void build_p64(uint32_t rd, uint32_t wr, const float* gb, int row, float pim,
                                          int pb) {
    const int jt = row >> 3;
    const int jmax = (row | 31) >> 3;  // the last piece of this warp's rows
    float ndd[8];
    same_piece_decays(gb, row, ndd);
#pragma unroll 1
    for (int mi = 0; mi < 4; ++mi) {
        const int m = pb == 0 ? mi : 3 - mi;
        if (pb + 2 * m > jmax) {  // after every row of the warp: masked
            const uint32_t z[8] = {0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u};
            tmem_st8_async(wr + 8 * m, z);
            continue;
        }
        float v[16];
        tmem_ld16(rd + 16 * m, v);
        uint32_t w[8];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int j = pb + 2 * m + h;
            const float tau = pim * gb[kGbTpm + 16 * j + jt];  // 0 unless j < jt
            const float4 s0 = lds4(gb + kGbNse + 8 * j);
            const float4 s1 = lds4(gb + kGbNse + 8 * j + 4);
            float e[8] = {s0.x * tau, s0.y * tau, s0.z * tau, s0.w * tau,
                          s1.x * tau, s1.y * tau, s1.z * tau, s1.w * tau};
            const bool same = j == jt;
#pragma unroll
            for (int i = 0; i < 8; ++i) e[i] = same ? ndd[i] : e[i];
#pragma unroll
            for (int i = 0; i < 4; ++i)
                w[4 * h + i] = pack_bf16x2(e[2 * i] * v[8 * h + 2 * i], e[2 * i + 1] * v[8 * h + 2 * i + 1]);
        }
        tmem_st8_async(wr + 8 * m, w);
    }
}

template <bool COSTATE, bool AGG>
__global__ void __launch_bounds__(kThreads, 1)
    decay_scan_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                      const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_o,
                      const TcScanParams p) {
    using Lay = DLayout<COSTATE>;
    constexpr int NS = Lay::kStages;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~static_cast<uintptr_t>(1023));
    const uint32_t sbase = smem_u32(smem);
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + Lay::kBarOff);
    uint64_t* full = bars;                 // [NS] stage landed
    uint64_t* empty = bars + 8;            // [NS] stage read by both MMA issuers
    uint64_t* sc_full = bars + 16;         // [2] score in TMEM
    uint64_t* sc_free = bars + 18;         // [2] score/P' buffer reusable
    uint64_t* o_full = bars + 20;          // [2] X of the chunk complete
    uint64_t* o_free = bars + 22;          // [2] X read by the epilogue
    uint64_t* dz_full = bars + 24;         // [2] dZ of the chunk in its buffer (or none)
    uint64_t* dz_free = bars + 26;         // [2] dZ read by the state warps
    uint64_t* st_ready = bars + 28;        // [2]
    uint64_t* st_free = bars + 30;         // [2]
    uint64_t* gf_full = bars + 32;         // [3] gate block of a chunk written
    uint64_t* gf_free = bars + 35;         // [3] gate block read by every user
    uint64_t* p_ready = bars + 38;         // [2] P' in TMEM
    uint64_t* b0_ready = bars + 40;        // B0^T tile of the current unit written
    uint64_t* b0_free = bars + 41;         // B0^T tile no longer read
    uint64_t* drain = bars + 42;           // [2]
    uint64_t* o_staged = bars + 44;        // [2]
    uint64_t* o_buf_free = bars + 46;      // the staging tile read by its store
    uint64_t* wv_ready = bars + 61;        // [2] a W V tile written
    uint64_t* wv_free = bars + 63;         // [2] a W V tile read by the dZ product
    uint64_t* item_full = bars + 49;       // [kRing]
    uint64_t* item_empty = bars + 53;      // [kRing]
    int* misc = reinterpret_cast<int*>(bars + 57);
    volatile int* abort_flag = misc + 0;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(misc + 1);
    volatile int* item_slot = misc + 4;    // [kRing]
    float* gfb = reinterpret_cast<float*>(smem + Lay::kGfOff);  // [kGbRing][kGbFloats]

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    // The n-th W V tile: the aggregate pass, which stores no outputs, alternates it
    // with the output staging tile, so that W V of chunk c + 1 is written while the
    // state update of chunk c reads the other; the scan keeps one tile.
    auto wv_buf = [](uint32_t n) -> uint32_t { return AGG ? (n & 1) : 0u; };
    auto wv_par = [](uint32_t n) -> uint32_t { return AGG ? ((n >> 1) & 1) : (n & 1); };

    if (threadIdx.x == 0) {
        for (int i = 0; i < NS; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], AGG ? 1 : 2);  // both issuers (the front one alone in AGG)
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&sc_full[i], 1);
            mbar_init(&sc_free[i], 1);
            mbar_init(&p_ready[i], 6);  // warps 2-5 and the two helpers
            mbar_init(&o_staged[i], 4);
            mbar_init(&o_full[i], 1);
            mbar_init(&o_free[i], 4);
            mbar_init(&dz_full[i], 1);
            mbar_init(&dz_free[i], 2);   // the two state warps
            mbar_init(&st_ready[i], 2);
            mbar_init(&st_free[i], 1);
        }
        for (int i = 0; i < kRing; ++i) {
            mbar_init(&item_full[i], 1);
            mbar_init(&item_empty[i], kItemConsumers);
        }
        for (int i = 0; i < kGbRing; ++i) {
            mbar_init(&gf_full[i], 1);
            // warps 2-5, the helpers, the state warps and (outputs only) the epilogue
            mbar_init(&gf_free[i], AGG ? 4 + 2 + 2 : 4 + 2 + 2 + 4);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&wv_ready[i], 4);  // warps 4-5 and the two helpers
            mbar_init(&wv_free[i], 1);
        }
        mbar_init(o_buf_free, 1);
        mbar_init(b0_ready, 2);
        mbar_init(b0_free, 1);
        mbar_init(drain, 1);  // [2] one per issuer
        mbar_init(drain + 1, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, kTmemCols);
        tmem_relinquish();
        tc_fence_before();
    }
    if (warp == kWarpProd && lane == 0) {
        prefetch_tmap(&tm_q);
        prefetch_tmap(&tm_k);
        prefetch_tmap(&tm_v);
        prefetch_tmap(&tm_o);
    }
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    // next item from the ring (every role warp reads every slot in order)
    auto take_item = [&](int it, int& item) -> bool {
        const int slot = it % kRing;
        if (!warp_wait(&item_full[slot], (it / kRing) & 1, abort_flag)) {
            raise_error(p, kErrWaitTimeout, abort_flag);
            return false;
        }
        item = item_slot[slot];
        __syncwarp();
        if (lane == 0) mbar_arrive(&item_empty[slot]);
        return true;
    };

    if (warp == kWarpProd) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            uint32_t n = 0;
            bool ok = true;
            for (int it = 0; ok; ++it) {
                const int slot = it % kRing;
                if (!bwait(&item_empty[slot], ((it / kRing) & 1) ^ 1, abort_flag)) {
                    raise_error(p, kErrWaitTimeout, abort_flag);
                    break;
                }
                int item = static_cast<int>(atomicAdd(p.ctrl, 1u));
                if (item >= p.n_items) item = -1;
                item_slot[slot] = item;
                mbar_arrive(&item_full[slot]);
                if (item < 0) break;
                const Item I = decode_unit(item, p);
                for (int c = 0; c < I.nch; ++c, ++n) {
                    const int s = n % NS;
                    if (!bwait(&empty[s], ((n / NS) & 1) ^ 1, abort_flag)) {
                        raise_error(p, kErrWaitTimeout, abort_flag);
                        ok = false;
                        break;
                    }
                    uint8_t* st = smem + s * Lay::kStageBytes;
                    const int t0 = I.t_begin + c * kChunk;
                    // the aggregate pass reads no queries
                    mbar_arrive_expect_tx(&full[s], (COSTATE && AGG) ? Lay::kStageBytes - kTile : Lay::kStageBytes);
                    if (COSTATE && !AGG) tma_load_5d(st + Lay::kQOff, &tm_q, &full[s], 0, I.h, t0, I.b, I.l);
                    tma_load_5d(st + Lay::kKOff, &tm_k, &full[s], 0, I.h, t0, I.b, I.l);
                    tma_load_5d(st + Lay::kVOff, &tm_v, &full[s], 0, I.h, t0, I.b, I.l);
                }
            }
            if (*abort_flag) {  // every issued load has landed before the CTA exits
                for (int s = 0; s < NS; ++s) {
                    if (n > (uint32_t)s) {
                        const uint32_t last = ((n - 1 - s) / NS) * NS + s;
                        mbar_drain(&full[s], (last / NS) & 1);
                    }
                }
            }
        }
    } else if (warp == 1 || warp == kWarpBack) {
        // ------------------------------------------- MMA issuers: warp 1 the score
        // of chunk c + 1 and dZ of chunk c, warp 0 X and P' V of chunk c
        const bool front = warp == 1;
        if (lane == 0) {
            constexpr uint32_t ID_SC = idesc_bf16(128, 128, false, false);  // Q K^T
            constexpr uint32_t ID_DZ = idesc_bf16(128, 64, true, true);     // K^T (W V)
            constexpr uint32_t ID_X = idesc_bf16(128, 128, false, true);    // Q [B0^T | S^T]
            constexpr uint32_t ID_PV = idesc_bf16(128, 64, false, true);    // P' V
            const uint32_t wv = sbase + Lay::kWvOff;
            uint32_t n = 0, c2 = 0, dzc = 0, ucnt = 0;
            bool ok = true;
            auto wait_or_fail = [&](uint64_t* bar, uint32_t par) -> bool {
                if (__builtin_expect(bwait(bar, par, abort_flag), 1)) return true;
                raise_error(p, kErrWaitTimeout, abort_flag);
                return false;
            };
            // dZ = K^T (W V) of the chunk in stage sp (chunk counter cc) into columns
            // 32..95 of its buffer, which its P warps have read: A = K^T (MN-major,
            // 64-wide M blocks 16 KB apart; the second block's rows land in TMEM lanes
            // 64..127, unread)
            auto issue_dz = [&](int sp, uint32_t cc) -> bool {
                const uint32_t wb = wv_buf(dzc);
                if (!wait_or_fail(&wv_ready[wb], wv_par(dzc))) return false;
                tc_fence_after();
                const uint32_t a_lo = sdesc_lo(sbase + sp * Lay::kStageBytes + Lay::kKOff, kTile);
                const uint32_t b_lo = sdesc_lo(wb ? sbase + Lay::kOOff : wv, kTile);
#pragma unroll 1
                for (int kk = 0; kk < kChunk / 16; ++kk)
                    mma_bf16_ss(tmem + col_sc(cc & 1) + kDzCol, sdesc_from_lo(a_lo + mnmaj_step(kk)),
                                sdesc_from_lo(b_lo + mnmaj_step(kk)), ID_DZ, kk > 0 ? 1u : 0u);
                mma_commit(&dz_full[cc & 1]);
                mma_commit(&wv_free[wb]);
                ++dzc;
                return true;
            };
            // the score Q K^T of the chunk with stage counter nn and chunk counter cc,
            // once its buffer's previous chunk is done (P' V read, dZ taken)
            auto issue_score = [&](uint32_t nn, uint32_t cc) -> bool {
                const int s = static_cast<int>(nn % NS);
                const uint32_t sb = cc & 1;
                if (!wait_or_fail(&full[s], (nn / NS) & 1)) return false;
                if (!wait_or_fail(&sc_free[sb], ((cc >> 1) & 1) ^ 1)) return false;
                if (!wait_or_fail(&dz_free[sb], ((cc >> 1) & 1) ^ 1)) return false;
                tc_fence_after();
                const uint32_t st = sbase + s * Lay::kStageBytes;
                const uint32_t q_lo = sdesc_lo(st + Lay::kQOff, 16);
                const uint32_t k_lo = sdesc_lo(st + Lay::kKOff, 16);
#pragma unroll 1
                for (int kk = 0; kk < 4; ++kk)
                    mma_bf16_ss(tmem + col_sc(sb), sdesc_from_lo(q_lo + kmaj_step(kk)),
                                sdesc_from_lo(k_lo + kmaj_step(kk)), ID_SC, kk > 0 ? 1u : 0u);
                mma_commit(&sc_full[sb]);
                return true;
            };
            for (int it = 0; ok; ++it) {
                const int slot = it % kRing;
                if (!wait_or_fail(&item_full[slot], (it / kRing) & 1)) break;
                const int item = item_slot[slot];
                mbar_arrive(&item_empty[slot]);
                if (item < 0) break;
                const Item I = decode_unit(item, p);
                if (AGG) {  // the segment's aggregate: the state update of every chunk
                    if (!front) continue;
                    for (int c = 0; c < I.nch; ++c, ++n, ++c2) {
                        const int s = n % NS;
                        if (!(ok = wait_or_fail(&full[s], (n / NS) & 1))) break;
                        if (!(ok = wait_or_fail(&dz_free[c2 & 1], ((c2 >> 1) & 1) ^ 1))) break;
                        if (!(ok = issue_dz(s, c2))) break;
                        mma_commit(&empty[s]);
                    }
                    continue;
                }
                if (front) {
                    if (!(ok = issue_score(n, c2))) break;
                    for (int c = 0; c < I.nch; ++c, ++n, ++c2) {
                        const int s = n % NS;
                        const uint32_t sb = c2 & 1, ph = (c2 >> 1) & 1;
                        // the next chunk's score, then this chunk's state update (an
                        // item's last chunk has none: its barrier completes empty)
                        if (c + 1 < I.nch && !(ok = issue_score(n + 1, c2 + 1))) break;
                        if (!(ok = wait_or_fail(&p_ready[sb], ph))) break;
                        if (c + 1 < I.nch) {
                            if (!(ok = issue_dz(s, c2))) break;
                        } else {
                            mma_commit(&dz_full[sb]);
                        }
                        mma_commit(&empty[s]);
                    }
                    continue;
                }
                if (!(ok = wait_or_fail(b0_ready, ucnt & 1))) break;
                for (int c = 0; c < I.nch; ++c, ++n, ++c2) {
                    const int s = n % NS;
                    const uint32_t sb = c2 & 1, ph = (c2 >> 1) & 1;
                    const uint32_t st = sbase + s * Lay::kStageBytes;
                    if (!(ok = wait_or_fail(&full[s], (n / NS) & 1))) break;
                    // X = Q [B0^T | S^T]: an MN-major B whose two 64-wide N blocks are
                    // the B0^T tile and this chunk's S^T tile, (sb + 1) * kStTile apart
                    if (!(ok = wait_or_fail(&o_free[sb], ph ^ 1))) break;
                    if (!(ok = wait_or_fail(&st_ready[sb], ph))) break;
                    tc_fence_after();
                    const uint32_t q_lo = sdesc_lo(st + Lay::kQOff, 16);
                    const uint32_t b_lo = sdesc_lo(sbase + Lay::kB0Off, kStTile * (sb + 1));
#pragma unroll 1
                    for (int kk = 0; kk < 4; ++kk)
                        mma_bf16_ss(tmem + col_x(sb), sdesc_from_lo(q_lo + kmaj_step(kk)),
                                    sdesc_from_lo(b_lo + mnmaj_step(kk)), ID_X, kk > 0 ? 1u : 0u);
                    mma_commit(&st_free[sb]);
                    // X[:, 0:64] += P' V  (P' in the chunk buffer: tokens s < 64 in
                    // columns 0..31, s >= 64 in columns 96..127)
                    if (!(ok = wait_or_fail(&p_ready[sb], ph))) break;
                    tc_fence_after();
                    const uint32_t v_lo = sdesc_lo(st + Lay::kVOff, kTile);
#pragma unroll 1
                    for (int kk = 0; kk < kChunk / 16; ++kk)
                        mma_bf16_ts(tmem + col_x(sb),
                                    tmem + col_sc(sb) + (kk < 4 ? kk * 8 : kPhiCol + (kk - 4) * 8),
                                    sdesc_from_lo(v_lo + mnmaj_step(kk)), ID_PV, 1u);
                    mma_commit(&o_full[sb]);
                    mma_commit(&sc_free[sb]);
                    mma_commit(&empty[s]);
                }
                if (!ok) break;
                mma_commit(b0_free);  // every product of this unit that reads B0^T issued
                ++ucnt;
            }
            mma_commit(front ? drain : drain + 1);
            mbar_drain(front ? drain : drain + 1, 0);
        }
    } else if (warp == kWarpGate) {
        // ------------------------------------------------------- gate factors
        // Lane l takes tokens 4l .. 4l+3 of each chunk, so piece j (8 tokens) is lanes
        // 2j and 2j+1.  Products inside a lane, then across the lane pair, then over the
        // 16 pieces by shuffles; every factor is a plain product of alphas.
        uint32_t cc = 0;
        bool ok = true;
        for (int it = 0; ok; ++it) {
            int item;
            if (!take_item(it, item) || item < 0) break;
            const Item I = decode_unit(item, p);
            const long long gbase = ((long long)I.l * p.B + I.b) * p.T * p.H + I.h;
            // this lane's gates of chunk c (alpha = 1, eta = 0 past the segment)
            auto load = [&](int c, float (&al)[4], float (&et)[4]) {
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int tg = I.t_begin + c * kChunk + 4 * lane + i;
                    const bool in = tg < I.t_end;
                    const long long gi = gbase + (long long)(in ? tg : 0) * p.H;
                    al[i] = in ? (p.g_alpha ? __ldg(p.g_alpha + gi) : 1.0f) : 1.0f;
                    et[i] = in ? __ldg(p.g_eta + gi) : 0.0f;
                }
            };
            float nal[4], net[4];
            load(0, nal, net);
            for (int c = 0; c < I.nch; ++c, ++cc) {
                float al[4], et[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    al[i] = nal[i];
                    et[i] = net[i];
                }
                if (c + 1 < I.nch) load(c + 1, nal, net);
                // inside the lane: alphas before / after each token
                const float pre[4] = {1.0f, al[0], al[0] * al[1], al[0] * al[1] * al[2]};
                const float suf[4] = {al[1] * al[2] * al[3], al[2] * al[3], al[3], 1.0f};
                const float prod = pre[3] * al[3];
                const float other = __shfl_xor_sync(0xffffffffu, prod, 1);
                const bool hi = lane & 1;  // second half of the piece
                const float tp = hi ? other * prod : prod * other;
                // inclusive prefix / suffix of the piece products (pieces are lane pairs)
                float incl = tp, sincl = tp;
#pragma unroll
                for (int o = 2; o < 32; o <<= 1) {
                    const float u = __shfl_up_sync(0xffffffffu, incl, o);
                    const float d = __shfl_down_sync(0xffffffffu, sincl, o);
                    if (lane >= o) incl = u * incl;
                    if (lane + o < 32) sincl = sincl * d;
                }
                float before = __shfl_up_sync(0xffffffffu, incl, 2);   // pieces before j
                float after = __shfl_down_sync(0xffffffffu, sincl, 2); // pieces after j
                if (lane < 2) before = 1.0f;
                if (lane >= 30) after = 1.0f;
                const float a_end = __shfl_sync(0xffffffffu, incl, 31);
                const uint32_t k = cc % kGbRing;
                if (!warp_wait(&gf_free[k], ((cc / kGbRing) & 1) ^ 1, abort_flag)) {
                    raise_error(p, kErrWaitTimeout, abort_flag);
                    ok = false;
                    break;
                }
                float* gb = gfb + k * kGbFloats;
                float pim[4], nse[4], at[4], wt[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    pim[i] = hi ? other * pre[i] : pre[i];  // alphas before t in its piece
                    const float sig = hi ? suf[i] : suf[i] * other;  // after s in its piece
                    const float es = et[i] * sig;
                    nse[i] = -es;
                    at[i] = before * pim[i];
                    wt[i] = es * after;
                }
                const int t4 = 4 * lane;
                *reinterpret_cast<float4*>(gb + kGbAl + t4) = make_float4(al[0], al[1], al[2], al[3]);
                *reinterpret_cast<float4*>(gb + kGbEt + t4) = make_float4(et[0], et[1], et[2], et[3]);
                *reinterpret_cast<float4*>(gb + kGbNse + t4) = make_float4(nse[0], nse[1], nse[2], nse[3]);
                *reinterpret_cast<float4*>(gb + kGbPim + t4) = make_float4(pim[0], pim[1], pim[2], pim[3]);
                *reinterpret_cast<float4*>(gb + kGbA + t4) = make_float4(at[0], at[1], at[2], at[3]);
                *reinterpret_cast<float4*>(gb + kGbW + t4) = make_float4(wt[0], wt[1], wt[2], wt[3]);
                // tpm[j][jt] = prod_{j<i<jt} tp_i (0 for j >= jt): lane l fills column
                // jt = l / 2, rows 8 (l % 2) .. +7
                {
                    float tpa[16];
#pragma unroll
                    for (int i = 0; i < 16; ++i) tpa[i] = __shfl_sync(0xffffffffu, tp, 2 * i);
                    const int jc = lane >> 1, j0 = 8 * (lane & 1);
                    float run = 1.0f;
#pragma unroll
                    for (int j = 15; j >= 0; --j) {
                        const bool lt = j < jc;
                        const float val = lt ? run : 0.0f;
                        run = lt ? run * tpa[j] : run;
                        if (j >= j0 && j < j0 + 8) gb[kGbTpm + 16 * j + jc] = val;
                    }
                }
                if (lane == 0) gb[kGbEnd] = a_end;
                __syncwarp();
                if (lane == 0) mbar_arrive(&gf_full[k]);
            }
        }
    } else if (warp < kWarpO0 || warp == kWarpZ0 || warp == kWarpZ0 + 1) {
        // ---------------------------------------------------- P' and the W V rows
        // Warps 2-5 own token rows row = 32 (warp & 3) + lane of each chunk: P' over
        // columns 0..63 (rows < 64 also zero columns 64..127).  The two helpers build
        // P' over columns 64..127 of rows 64..127.  Then warps 4-5 (whose P' rows are
        // half masked) and the helpers write the chunk's W V rows -w_t v_t (rows
        // 0..63 and 64..127), which the state update dZ of the same chunk reads.
        const bool helper = warp >= kWarpZ0;
        const int q4 = warp & 3;
        const int row = q4 * 32 + lane;
        const uint32_t lane_off = static_cast<uint32_t>(q4 * 32) << 16;
        const bool wv_writer = helper || q4 < 2;  // W V row wv_row = row
        const int wv_row = row;
        uint32_t c2 = 0, wvn = 0;
        bool ok = true;
        for (int it = 0; ok; ++it) {
            int item;
            if (!take_item(it, item) || item < 0) break;
            const Item I = decode_unit(item, p);
            for (int c = 0; c < I.nch; ++c, ++c2) {
                const uint32_t sb = c2 & 1;
                const int s = static_cast<int>(c2 % NS);  // ring slot: every stage is a chunk
                const uint32_t st = sbase + s * Lay::kStageBytes;
                const uint32_t gk = c2 % kGbRing;
                const float* gb = gfb + gk * kGbFloats;
                if (!warp_wait(&gf_full[gk], (c2 / kGbRing) & 1, abort_flag) ||
                    !warp_wait(&full[s], (c2 / NS) & 1, abort_flag) ||
                    (!AGG && !warp_wait(&sc_full[sb], (c2 >> 1) & 1, abort_flag))) {
                    raise_error(p, kErrWaitTimeout, abort_flag);
                    ok = false;
                    break;
                }
                if (!AGG) {  // the aggregate pass forms no outputs
                tc_fence_after();
                const uint32_t base = tmem + col_sc(sb) + lane_off;
                const float pim_t = gb[kGbPim + row];
                // ---- P'_ts = -E_ts (q_t . k_s): warps 2-5 for s < 64, the helpers for
                // s >= 64 (rows 64..127)
                build_p64(helper ? base + 64 : base, helper ? base + kPhiCol : base, gb, row, pim_t,
                          helper ? 8 : 0);
                if (!helper && q4 < 2) tmem_zero32_async(base + kPhiCol);  // tokens >= 64 all masked
                tmem_wait_st();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&p_ready[sb]);
                }
                if (wv_writer && (AGG || c < I.nch - 1)) {
                    // ---- the chunk's W V row -w_t v_t (an item's last chunk needs none
                    // unless its state at the segment end is the aggregate)
                    const uint32_t wb = wv_buf(wvn);
                    if (!warp_wait(&wv_free[wb], wv_par(wvn) ^ 1, abort_flag)) {
                        raise_error(p, kErrWaitTimeout, abort_flag);
                        ok = false;
                        break;
                    }
                    const float w = -gb[kGbW + wv_row];
                    const uint32_t vt = st + Lay::kVOff;
                    const uint32_t wvt = sbase + (wb ? Lay::kOOff : Lay::kWvOff);
#pragma unroll 1
                    for (int q = 0; q < 8; q += 2) {
                        const uint4 a0 = ld_shared_v4(vt + sw128_off(wv_row, q));
                        const uint4 a1 = ld_shared_v4(vt + sw128_off(wv_row, q + 1));
                        const __nv_bfloat162* h0 = reinterpret_cast<const __nv_bfloat162*>(&a0);
                        const __nv_bfloat162* h1 = reinterpret_cast<const __nv_bfloat162*>(&a1);
                        uint32_t o0[4], o1[4];
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            const float2 f0 = __bfloat1622float2(h0[i]);
                            const float2 f1 = __bfloat1622float2(h1[i]);
                            o0[i] = pack_bf16x2(w * f0.x, w * f0.y);
                            o1[i] = pack_bf16x2(w * f1.x, w * f1.y);
                        }
                        st_shared_v4(wvt + sw128_off(wv_row, q), o0[0], o0[1], o0[2], o0[3]);
                        st_shared_v4(wvt + sw128_off(wv_row, q + 1), o1[0], o1[1], o1[2], o1[3]);
                    }
                    fence_proxy_async_smem();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&wv_ready[wb]);
                    ++wvn;
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(&gf_free[gk]);  // this warp's reads of the block are done
            }
        }
    } else if (warp < kWarpZ0) {
        // ------------------------------------------------- output epilogue
        const int q4 = warp & 3;
        const int row = q4 * 32 + lane;
        const uint32_t lane_off = static_cast<uint32_t>(q4 * 32) << 16;
        const bool storer = (warp == kWarpO0) && (lane == 0);
        const EpiParams& e = p.epi;
        uint32_t c2 = 0;
        bool ok = true;
        for (int it = 0; ok; ++it) {
            int item;
            if (!take_item(it, item) || item < 0) break;
            if (AGG) continue;  // no outputs in the aggregate pass
            const Item I = decode_unit(item, p);
            for (int c = 0; c < I.nch; ++c, ++c2) {
                const uint32_t ob = c2 & 1, oph = (c2 >> 1) & 1;
                const uint32_t gk = c2 % kGbRing;
                if (!warp_wait(&o_full[ob], oph, abort_flag) ||
                    !warp_wait(&gf_full[gk], (c2 / kGbRing) & 1, abort_flag)) {
                    raise_error(p, kErrWaitTimeout, abort_flag);
                    ok = false;
                    break;
                }
                tc_fence_after();
                // o_t = X_t[0:64] + a_t X_t[64:128]
                const float a_t = gfb[gk * kGbFloats + kGbA + row];
                __syncwarp();
                if (lane == 0) mbar_arrive(&gf_free[gk]);
                const uint32_t xt = tmem + col_x(ob) + lane_off;
                const int t0 = I.t_begin + c * kChunk;
                const int t = t0 + row;
                const bool valid = t < p.T;
                const uint32_t otile = sbase + Lay::kOOff;
                if (!e.zin && !e.out2) {
                    // plain result: 16 columns at a time from TMEM into the staging tile
                    if (!warp_wait(o_buf_free, (c2 & 1) ^ 1, abort_flag)) {
                        raise_error(p, kErrWaitTimeout, abort_flag);
                        ok = false;
                        break;
                    }
#pragma unroll 1
                    for (int m = 0; m < 2; ++m) {  // 32 output columns per TMEM round trip
                        float u[32], z[32];
                        tmem_ld32_pair(xt + 32 * m, xt + 64 + 32 * m, u, z);
#pragma unroll
                        for (int i = 0; i < 32; ++i) u[i] = fmaf(a_t, z[i], u[i]);
#pragma unroll
                        for (int h = 0; h < 4; ++h)
                            st_shared_v4(otile + sw128_off(row, 4 * m + h), pack_bf16x2(u[8 * h], u[8 * h + 1]),
                                         pack_bf16x2(u[8 * h + 2], u[8 * h + 3]),
                                         pack_bf16x2(u[8 * h + 4], u[8 * h + 5]),
                                         pack_bf16x2(u[8 * h + 6], u[8 * h + 7]));
                    }
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&o_free[ob]);
                } else {
                float v[64];
                tmem_ld64(xt, v);
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    float z[32];
                    tmem_ld32(xt + 64 + 32 * h, z);
#pragma unroll
                    for (int i = 0; i < 32; ++i) v[32 * h + i] = fmaf(a_t, z[i], v[32 * h + i]);
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&o_free[ob]);
                if (e.zin && valid) {
                    float tmp[64];
#pragma unroll
                    for (int i = 0; i < 64; ++i) tmp[i] = v[i];
                    epi_apply_dact(e, tok_off(e.z_str, I.l, I.b, t, I.h), tmp);
#pragma unroll
                    for (int i = 0; i < 64; ++i) v[i] = tmp[i];
                }
                if (e.out2 && valid) {
                    float tmp[64];
#pragma unroll
                    for (int i = 0; i < 64; ++i) tmp[i] = v[i];
                    epi_store_act(e, tok_off(e.out2_str, I.l, I.b, t, I.h), tmp);
                }
                // one staging tile: the previous chunk's store has read it
                if (!warp_wait(o_buf_free, (c2 & 1) ^ 1, abort_flag)) {
                    raise_error(p, kErrWaitTimeout, abort_flag);
                    ok = false;
                    break;
                }
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
                    if (!bwait(&o_staged[ob], oph, abort_flag)) {
                        raise_error(p, kErrWaitTimeout, abort_flag);
                        ok = false;
                    } else {
                        // rows past the end of the sequence are clipped by the store
                        tma_store_5d(&tm_o, smem + Lay::kOOff, 0, I.h, t0, I.b, I.l);
                        bulk_commit_group();
                        bulk_wait_group_read<0>();  // the store has read the tile
                        mbar_arrive(o_buf_free);
                    }
                }
                if (!__shfl_sync(0xffffffffu, ok ? 1 : 0, 0)) {
                    ok = false;
                    break;
                }
            }
        }
        if (storer) bulk_wait_group_all();
    } else {
        // ------------------------------------------------------------ state
        // Warps 12-13: row q = 32 (warp & 3) + lane of S^T (fp32, registers), the
        // bf16 B0^T tile once per item, the bf16 S^T tile per chunk, and the decayed
        // update S' = a_end S + dZ.  A segment after the first starts from the carried
        // state of the earlier segments; the aggregate pass starts from zero and
        // writes its end state and alpha product instead of tiles.
        const int q4 = warp & 3;
        const int row = q4 * 32 + lane;
        const uint32_t lane_off = static_cast<uint32_t>(q4 * 32) << 16;
        uint32_t c2 = 0, ucnt = 0;
        float st[64];
        bool ok = true;
        auto put_row = [&](uint32_t tile) {
#pragma unroll
            for (int q = 0; q < 8; ++q)
                st_shared_v4(tile + sw128_off(row, q), pack_bf16x2(st[8 * q], st[8 * q + 1]),
                             pack_bf16x2(st[8 * q + 2], st[8 * q + 3]),
                             pack_bf16x2(st[8 * q + 4], st[8 * q + 5]),
                             pack_bf16x2(st[8 * q + 6], st[8 * q + 7]));
            fence_proxy_async_smem();
            __syncwarp();
        };
        // S' = a_end S + dZ with the chunk's product from its TMEM buffer (chunk
        // counter cc); an item's last chunk has no product (use = false) but its
        // barriers still turn
        auto advance = [&](uint32_t cc, float a_end, bool use) -> bool {
            const uint32_t b = cc & 1;
            if (!warp_wait(&dz_full[b], (cc >> 1) & 1, abort_flag)) return false;
            if (use) {
                tc_fence_after();
                float a[32];
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    tmem_ld32(tmem + col_sc(b) + kDzCol + lane_off + h * 32, a);
#pragma unroll
                    for (int i = 0; i < 32; ++i) st[h * 32 + i] = fmaf(a_end, st[h * 32 + i], a[i]);
                }
                tc_fence_before();
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&dz_free[b]);
            return true;
        };
        for (int it = 0; ok; ++it) {
            int item;
            if (!take_item(it, item) || item < 0) break;
            const Item I = decode_unit(item, p);
            if (AGG) {
#pragma unroll
                for (int i = 0; i < 64; ++i) st[i] = 0.0f;
                float prod = 1.0f;
                for (int c = 0; c < I.nch; ++c, ++c2) {
                    const uint32_t gk = c2 % kGbRing;
                    if (!warp_wait(&gf_full[gk], (c2 / kGbRing) & 1, abort_flag)) {
                        ok = false;
                        break;
                    }
                    const float a_end = gfb[gk * kGbFloats + kGbEnd];
                    if (!advance(c2, a_end, true)) {
                        ok = false;
                        break;
                    }
                    prod *= a_end;
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&gf_free[gk]);
                }
                if (!ok) {
                    raise_error(p, kErrWaitTimeout, abort_flag);
                    break;
                }
                float* dst = p.agg + (size_t)item * 64 * 64 + (size_t)row * 64;
#pragma unroll
                for (int i = 0; i < 64; i += 4)
                    *reinterpret_cast<float4*>(dst + i) = make_float4(st[i], st[i + 1], st[i + 2], st[i + 3]);
                if (row == 0) p.seg_a[item] = prod;
                continue;
            }
            if (!warp_wait(b0_free, (ucnt & 1) ^ 1, abort_flag)) {
                raise_error(p, kErrWaitTimeout, abort_flag);
                break;
            }
            // B0^T row q: forward B0 = W0 ([m][d], column q), costate B0 = W0^T (row q)
            const float* w0 = p.W0 + (size_t)(I.l * p.H + I.h) * 64 * 64;
            if (p.w0_transposed) {
#pragma unroll
                for (int i = 0; i < 64; i += 4) {
                    const float4 a = *reinterpret_cast<const float4*>(w0 + (size_t)row * 64 + i);
                    st[i] = a.x;
                    st[i + 1] = a.y;
                    st[i + 2] = a.z;
                    st[i + 3] = a.w;
                }
            } else {
#pragma unroll
                for (int i = 0; i < 64; ++i) st[i] = w0[(size_t)i * 64 + row];
            }
            put_row(sbase + Lay::kB0Off);
            if (lane == 0) mbar_arrive(b0_ready);
            ++ucnt;
            if (I.k > 0) {  // the carried state at the segment's first token
                const float* src = p.incl + (size_t)item * 64 * 64 + (size_t)row * 64;
#pragma unroll
                for (int i = 0; i < 64; i += 4) {
                    const float4 a = *reinterpret_cast<const float4*>(src + i);
                    st[i] = a.x;
                    st[i + 1] = a.y;
                    st[i + 2] = a.z;
                    st[i + 3] = a.w;
                }
            } else {
#pragma unroll
                for (int i = 0; i < 64; ++i) st[i] = 0.0f;  // the fast weights start at W0
            }
            for (int c = 0; c < I.nch; ++c, ++c2) {
                const uint32_t sb = c2 & 1, ph = (c2 >> 1) & 1;
                if (!warp_wait(&st_free[sb], ph ^ 1, abort_flag)) {
                    raise_error(p, kErrWaitTimeout, abort_flag);
                    ok = false;
                    break;
                }
                put_row(sbase + Lay::kStOff + sb * kStTile);
                if (lane == 0) mbar_arrive(&st_ready[sb]);
                const uint32_t gk = c2 % kGbRing;
                if (!warp_wait(&gf_full[gk], (c2 / kGbRing) & 1, abort_flag)) {
                    raise_error(p, kErrWaitTimeout, abort_flag);
                    ok = false;
                    break;
                }
                const float a_end = gfb[gk * kGbFloats + kGbEnd];
                if (!advance(c2, a_end, c < I.nch - 1)) {
                    raise_error(p, kErrWaitTimeout, abort_flag);
                    ok = false;
                    break;
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(&gf_free[gk]);
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

template <bool COSTATE, bool AGG>
static cudaError_t launch_dec(const CUtensorMap& q, const CUtensorMap& k, const CUtensorMap& v,
                              const CUtensorMap& o, const TcScanParams& p, int grid,
                              cudaStream_t stream) {
    using Lay = DLayout<COSTATE>;
    auto kern = decay_scan_kernel<COSTATE, AGG>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         Lay::kSmemBytes);
    if (e != cudaSuccess) return e;
    kern<<<grid, kThreads, Lay::kSmemBytes, stream>>>(q, k, v, o, p);
    return cudaGetLastError();
}

}  // namespace dec

// Carried start states of the segments: for each unit and segment k,
// incl[k] = P_{k-1} with P_{-1} = 0 and P_k = a_k P_{k-1} + agg_k (the affine
// composition of the segments' transforms S -> a S + U).  One thread per state
// entry and unit, walking the segments in order.
__global__ void __launch_bounds__(256)
    decay_carry_kernel(const float* __restrict__ agg, const float* __restrict__ seg_a,
                       float* __restrict__ incl, int n_ut, int n_seg) {
    const long long i = (long long)blockIdx.x * 256 + threadIdx.x;
    if (i >= (long long)n_ut * 4096) return;
    const int unit = (int)(i >> 12), e = (int)(i & 4095);
    float P = 0.0f;
    for (int k = 0; k < n_seg; ++k) {
        const size_t item = (size_t)k * n_ut + unit;
        incl[item * 4096 + e] = P;
        if (k < n_seg - 1) P = fmaf(seg_a[item], P, agg[item * 4096 + e]);
    }
}

// The retention scan of 64 x 64 bf16 maps on the tensor cores.  With p.n_seg > 1
// every unit is cut into segments of p.seg_len tokens: an aggregate pass over all
// but the last segment of each unit (p.agg, p.seg_a), the carry of the start states
// (p.incl), then the scan of every (segment, unit) item from its start state.
cudaError_t launch_tc_decay(const CUtensorMap& q, const CUtensorMap& k, const CUtensorMap& v,
                            const CUtensorMap& o, const TcScanParams& p, bool costate, int grid,
                            cudaStream_t stream) {
    if (p.dq != 64 || p.dv != 64 || !p.g_eta) return cudaErrorInvalidValue;
    if (p.n_seg > 1) {
        if (!p.agg || !p.incl || !p.seg_a) return cudaErrorInvalidValue;
        TcScanParams pa = p;
        pa.n_items = (p.n_seg - 1) * p.n_ut;
        const int ga = pa.n_items < grid ? pa.n_items : grid;
        cudaError_t e = costate ? dec::launch_dec<true, true>(q, k, v, o, pa, ga, stream)
                                : dec::launch_dec<false, true>(q, k, v, o, pa, ga, stream);
        if (e != cudaSuccess) return e;
        const long long n = (long long)p.n_ut * 4096;
        decay_carry_kernel<<<(unsigned)((n + 255) / 256), 256, 0, stream>>>(p.agg, p.seg_a, p.incl,
                                                                                 p.n_ut, p.n_seg);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
        // a fresh work ticket for the scan (the error word stays)
        if ((e = cudaMemsetAsync(p.ctrl, 0, sizeof(unsigned int), stream)) != cudaSuccess) return e;
    }
    return costate ? dec::launch_dec<true, false>(q, k, v, o, p, grid, stream)
                   : dec::launch_dec<false, false>(q, k, v, o, p, grid, stream);
}

}  // namespace gl
