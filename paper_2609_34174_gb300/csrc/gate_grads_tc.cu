// gate_grads_tc.cu -- the per-chunk expansion of the gate derivatives (Sec. 3,
// practical architecture and training; Eq. 2 with retention), 64 x 64 bf16 maps, on
// tcgen05.
//
// With D_t = W_t - W0 and the read's pair (a, b) (forward read: a = u, b = x;
// costate read: a = g_out, b = u, u the read's upstream gradient), S the state D at
// a chunk's first token and Rt = sum_{s>c1-1} prod_{c1-1<r<s} alpha_r a_s b_s^T the
// decayed suffix state at its last token c1 - 1, every token j of the chunk gets
//   dlog_alpha_j = alpha_j (P_j Q_j <S, Rt> + P_j sum_{s>j} G(j,s) v_s
//                           + Q_j sum_{i<j} (-eta_i) E(i,j) w_i
//                           + sum_{i<j} (-eta_i) E(i,j) N_{i,j})
//   deta_j       = -(Q_j w_j + N_{j,j})
// over tokens i, s of the chunk, where P_j, Q_j are the products of the chunk's
// alphas before and after j, E(i,j) and G(j,s) those strictly between,
//   v_s = a_s^T S b_s,  w_i = ghat_i^T Rt x_i,  M_is = (a_s . ghat_i)(x_i . b_s),
//   N_{i,j} = sum_{s>j} G(j,s) M_is      (N_{i,j} = M_{i,j+1} + alpha_{j+1} N_{i,j+1}).
// The products run on the tensor cores from TMA tiles (bf16 inputs, fp32
// accumulators in TMEM):
//   Y  = A S^T   (v_s = Y_s . b_s)        Y2 = Ghat Rt^T   (w_i = Y2_i . x_i)
//   G1 = Ghat A^T, G2 = X B^T             (M = G1 (.) G2, elementwise)
// with S and Rt rounded to bf16 for their products.  One CTA of 128 threads per
// (unit, chunk); thread r owns token row r (TMEM lane r).  Tokens past T are zero
// rows (TMA fill) with alpha = 1 and eta = 0.  S and Rt of every chunk come from
// per-chunk aggregates (gate_agg_tc_kernel) carried over the chunks by
// gate_state_scan_kernel (grads.cu).
#include <cuda.h>

#include "scan_common.cuh"
#include "sm103_ptx.cuh"

namespace gl {
namespace ggtc {

constexpr int kC = 128;                  // tokens per chunk (the retention kernel's)
constexpr int kTile = 16384;             // [128 rows][64 bf16], 128-byte swizzle
constexpr int kStT = 8192;               // [64 rows][64 bf16]
constexpr int kThreads = 128;
constexpr int kX = 0, kG = kTile, kA = 2 * kTile, kB = 3 * kTile;
constexpr int kS = 4 * kTile;            // S^T, then Rt^T (bf16); afterwards N^T
constexpr int kR = kS + kStT;
constexpr int kN = kS;                   // N^T bf16 [128][128], written after the state products
constexpr int kV = kN + kC * kC * 2;     // v, w, eta, alpha fp32 [128] each, red[4]
constexpr int kScan = kV + 4 * kC * 4 + 16;  // two affine scans, (A, B) [2][128] each
constexpr int kBar = kScan + 4 * kC * 4;
constexpr int kSmem = kBar + 64 + 1024;  // + slack for the 1024-byte alignment
constexpr uint32_t kTmemCols = 256;

// Element (j, i) of N^T: row j (a column of N), column i swizzled by the row so that
// both the row pass (fixed j, i = thread) and the column pass (fixed i, j = thread)
// are free of bank conflicts.
__device__ __forceinline__ int nidx(int j, int i) { return j * kC + (i ^ ((2 * j) & (kC - 1))); }

__device__ __forceinline__ bool wait_bar(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                         unsigned int* err) {
    if (mbar_wait(bar, parity, abort_flag)) return true;
    atomicOr(err, kErrWaitTimeout);
    return false;
}

__global__ void __launch_bounds__(kThreads, 2)
    gate_chunk_tc_kernel(const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_g,
                         const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_b,
                         const float* __restrict__ eta, const float* __restrict__ alpha,
                         const float* __restrict__ Sd, const float* __restrict__ Rd,
                         float* __restrict__ dlog_alpha, float* __restrict__ deta, int B, int T, int H,
                         int nch, unsigned int* err) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~static_cast<uintptr_t>(1023));
    const uint32_t sb = smem_u32(smem);
    float* v = reinterpret_cast<float*>(smem + kV);
    float* w = v + kC;
    float* et = w + kC;
    float* al = et + kC;
    float* red = al + kC;  // [4]
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kBar);
    uint64_t* tma_bar = bars;
    uint64_t* mma_bar = bars + 1;
    uint32_t* tslot = reinterpret_cast<uint32_t*>(bars + 2);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(bars + 3);
    __nv_bfloat16* NT = reinterpret_cast<__nv_bfloat16*>(smem + kN);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const long long unit = blockIdx.x / nch;
    const int c = (int)(blockIdx.x % nch);
    const int h = (int)(unit % H);
    const long long lb = unit / H;
    const int b = (int)(lb % B);
    const int l = (int)(lb / B);
    const int c0 = c * kC;

    if (warp == 0) {
        tmem_alloc(tslot, kTmemCols);
        tmem_relinquish();
    }
    if (tid == 0) {
        mbar_init(tma_bar, 1);
        mbar_init(mma_bar, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tslot;
    if (tid == 0) {
        mbar_arrive_expect_tx(tma_bar, 4 * kTile);
        tma_load_5d(smem + kX, &tm_x, tma_bar, 0, h, c0, b, l);
        tma_load_5d(smem + kG, &tm_g, tma_bar, 0, h, c0, b, l);
        tma_load_5d(smem + kA, &tm_a, tma_bar, 0, h, c0, b, l);
        tma_load_5d(smem + kB, &tm_b, tma_bar, 0, h, c0, b, l);
    }
    // ---- the states as bf16 K-major tiles (S^T rows k by threads 0-63, Rt^T by 64-127)
    const float* s_src = Sd + (unit * nch + c) * (long long)(64 * 64);
    const float* r_src = Rd + (unit * nch + c) * (long long)(64 * 64);
    {
        const int k = tid & 63;
        const float* src = (tid < 64 ? s_src : r_src) + k * 64;
        const uint32_t tile = sb + (tid < 64 ? kS : kR);
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            const float4 lo = *reinterpret_cast<const float4*>(src + 8 * q);
            const float4 hi = *reinterpret_cast<const float4*>(src + 8 * q + 4);
            st_shared_v4(tile + sw128_off(k, q), pack_bf16x2(lo.x, lo.y), pack_bf16x2(lo.z, lo.w),
                         pack_bf16x2(hi.x, hi.y), pack_bf16x2(hi.z, hi.w));
        }
    }
    // ---- gates of the chunk's tokens, <S, Rt> in fp32
    {
        const int t = c0 + tid;
        const long long gi = (lb * T + t) * H + h;
        et[tid] = t < T ? eta[gi] : 0.0f;
        al[tid] = t < T ? (alpha ? alpha[gi] : 1.0f) : 1.0f;
        float kp = 0.0f;
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            const float4 s4 = reinterpret_cast<const float4*>(s_src)[tid * 8 + q];
            const float4 r4 = reinterpret_cast<const float4*>(r_src)[tid * 8 + q];
            kp = fmaf(s4.x, r4.x, fmaf(s4.y, r4.y, fmaf(s4.z, r4.z, fmaf(s4.w, r4.w, kp))));
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) kp += __shfl_xor_sync(0xffffffffu, kp, o);
        if (lane == 0) red[warp] = kp;
    }
    fence_proxy_async_smem();
    __syncthreads();
    constexpr uint32_t ID64 = idesc_bf16(128, 64, false, false);
    constexpr uint32_t ID128 = idesc_bf16(128, 128, false, false);
    const uint32_t x_lo = sdesc_lo(sb + kX, 16), g_lo = sdesc_lo(sb + kG, 16);
    const uint32_t a_lo = sdesc_lo(sb + kA, 16), b_lo = sdesc_lo(sb + kB, 16);
    bool ok = true;
    if (tid == 0) {
        if (wait_bar(tma_bar, 0, abort_flag, err)) {
            tc_fence_after();
            const uint32_t s_lo = sdesc_lo(sb + kS, 16), r_lo = sdesc_lo(sb + kR, 16);
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)  // Y = A S^T into columns 0..63
                mma_bf16_ss(tmem, sdesc_from_lo(a_lo + 2 * kk), sdesc_from_lo(s_lo + 2 * kk), ID64, kk > 0 ? 1u : 0u);
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)  // Y2 = Ghat Rt^T into columns 64..127
                mma_bf16_ss(tmem + 64, sdesc_from_lo(g_lo + 2 * kk), sdesc_from_lo(r_lo + 2 * kk), ID64,
                            kk > 0 ? 1u : 0u);
            mma_commit(mma_bar);
        }
    }
    ok = wait_bar(mma_bar, 0, abort_flag, err);
    tc_fence_after();
    const uint32_t lane_base = tmem + (static_cast<uint32_t>(warp * 32) << 16);
    // ---- v_s = Y_s . b_s and w_i = Y2_i . x_i (thread = token row)
    {
        float vs = 0.0f, wi = 0.0f;
#pragma unroll 1
        for (int hf = 0; hf < 2; ++hf) {
            float y[32], y2[32];
            tmem_ld32(lane_base + 32 * hf, y);
            tmem_ld32(lane_base + 64 + 32 * hf, y2);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const uint4 bq = ld_shared_v4(sb + kB + sw128_off(tid, 4 * hf + q));
                const uint4 xq = ld_shared_v4(sb + kX + sw128_off(tid, 4 * hf + q));
                const __nv_bfloat162* bh = reinterpret_cast<const __nv_bfloat162*>(&bq);
                const __nv_bfloat162* xh = reinterpret_cast<const __nv_bfloat162*>(&xq);
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const float2 bf = __bfloat1622float2(bh[e]);
                    const float2 xf = __bfloat1622float2(xh[e]);
                    vs = fmaf(y[8 * q + 2 * e], bf.x, fmaf(y[8 * q + 2 * e + 1], bf.y, vs));
                    wi = fmaf(y2[8 * q + 2 * e], xf.x, fmaf(y2[8 * q + 2 * e + 1], xf.y, wi));
                }
            }
        }
        v[tid] = vs;
        w[tid] = wi;
    }
    tc_fence_before();
    __syncthreads();
    if (tid == 0 && ok) {
        tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)  // G1 = Ghat A^T into columns 0..127
            mma_bf16_ss(tmem, sdesc_from_lo(g_lo + 2 * kk), sdesc_from_lo(a_lo + 2 * kk), ID128, kk > 0 ? 1u : 0u);
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)  // G2 = X B^T into columns 128..255
            mma_bf16_ss(tmem + 128, sdesc_from_lo(x_lo + 2 * kk), sdesc_from_lo(b_lo + 2 * kk), ID128,
                        kk > 0 ? 1u : 0u);
        mma_commit(mma_bar);
    }
    ok = wait_bar(mma_bar, 1, abort_flag, err) && ok;
    tc_fence_after();
    // ---- row i: N_{i,s-1} = M_is + alpha_s N_{i,s} for s > i, into N^T (bf16)
    {
        const int i = tid;
        NT[nidx(kC - 1, i)] = __float2bfloat16_rn(0.0f);  // N_{i,127}: no later token
        float nrun = 0.0f;
        // blocks of 32 columns s; none after a row of this warp below blk = warp
        // (warp-uniform, so the TMEM loads stay collective)
#pragma unroll 1
        for (int blk = 3; blk >= warp; --blk) {
            float g1[32], g2[32];
            tmem_ld32(lane_base + 32 * blk, g1);
            tmem_ld32(lane_base + 128 + 32 * blk, g2);
#pragma unroll
            for (int q = 31; q >= 0; --q) {
                const int s = 32 * blk + q;
                if (s >= 1 && s > i) {
                    nrun = fmaf(al[s], nrun, g1[q] * g2[q]);
                    NT[nidx(s - 1, i)] = __float2bfloat16_rn(nrun);
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    // ---- token j: the four terms.  Two scans of affine maps x -> A x + B over the
    // chunk (Hillis-Steele, 7 steps): the prefix of g_i = (alpha_i, -eta_i w_i) gives
    // P_j and t3_j = sum_{i<j} (-eta_i) E(i,j) w_i; the suffix of f_s = (alpha_s, v_s)
    // gives Q_j and t2_j = sum_{s>j} G(j,s) v_s.
    {
        const int j = tid;
        const float kappa = (red[0] + red[1]) + (red[2] + red[3]);
        float* pa = reinterpret_cast<float*>(smem + kScan);
        float* pb = pa + kC;
        float* sa = pb + kC;
        float* sbv = sa + kC;
        float ap = al[j], bp = -et[j] * w[j];  // inclusive prefix g_j o ... o g_0
        float as = al[j], bs = v[j];           // inclusive suffix f_j o ... o f_127
#pragma unroll 1
        for (int o = 1; o < kC; o <<= 1) {
            pa[j] = ap;
            pb[j] = bp;
            sa[j] = as;
            sbv[j] = bs;
            __syncthreads();
            if (j >= o) {  // (A, B) o (A', B') = (A A', A B' + B)
                bp = fmaf(ap, pb[j - o], bp);
                ap *= pa[j - o];
            }
            if (j + o < kC) {
                bs = fmaf(as, sbv[j + o], bs);
                as *= sa[j + o];
            }
            __syncthreads();
        }
        pa[j] = ap;
        pb[j] = bp;
        sa[j] = as;
        sbv[j] = bs;
        __syncthreads();
        const float P = j > 0 ? pa[j - 1] : 1.0f, t3 = j > 0 ? pb[j - 1] : 0.0f;
        const float Q = j + 1 < kC ? sa[j + 1] : 1.0f, t2 = j + 1 < kC ? sbv[j + 1] : 0.0f;
        float t4 = 0.0f, e = 1.0f;
        for (int i = j - 1; i >= 0; --i) {
            t4 = fmaf(-et[i] * e, __bfloat162float(NT[nidx(j, i)]), t4);
            e *= al[i];
        }
        const int t = c0 + j;
        if (t < T) {
            const long long gi = (lb * T + t) * H + h;
            dlog_alpha[gi] = al[j] * (P * Q * kappa + P * t2 + Q * t3 + t4);
            deta[gi] = -(Q * w[j] + __bfloat162float(NT[nidx(j, j)]));
        }
    }
    __syncthreads();
    if (tid == 0 && *abort_flag) {  // no copy in flight at exit (bounded: 0.2 s)
        const uint64_t t0 = globaltimer_ns();
        while (!mbar_try_wait(tma_bar, 0) && globaltimer_ns() - t0 < 200000000ull) {
        }
    }
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

// Chunk aggregates (one CTA of 128 threads per (unit, chunk)), in the S^T layout
// [k][l] of the states (k: x index, l: ghat index):
//   Vt_c = X^T (w (.) Ghat),  w_i = -eta_i prod_{i<r<c1} alpha_r   (D_{c+1} = A_c D_c + V_c)
//   Ut_c = B^T (p (.) A),     p_s = prod_{c0<=r<s} alpha_r          (R_c = U_{c+1} + A_{c+1} R_{c+1})
// and A_c, the product of the chunk's alphas.  Both products run with M = 128 over
// an MN-major A operand whose second 64-row block is the next tile in shared
// memory; those accumulator rows (TMEM lanes 64..127) are never read.
constexpr int kAggSmem = 6 * kTile + 4 * kC * 4 + 64 + 1024;

__global__ void __launch_bounds__(kThreads, 2)
    gate_agg_tc_kernel(const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_g,
                       const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_b,
                       const float* __restrict__ eta, const float* __restrict__ alpha, float* __restrict__ Vd,
                       float* __restrict__ Ud, float* __restrict__ Ad, int B, int T, int H, int nch,
                       unsigned int* err) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~static_cast<uintptr_t>(1023));
    const uint32_t sb = smem_u32(smem);
    // tiles: X | Ghat | B | A | w Ghat | p A  (X and B are each followed by a tile)
    constexpr int oX = 0, oG = kTile, oB = 2 * kTile, oA = 3 * kTile, oWG = 4 * kTile, oPA = 5 * kTile;
    float* sp = reinterpret_cast<float*>(smem + 6 * kTile);  // prefix products [128]
    float* ss = sp + kC;                                      // suffix products [128]
    float* sal = ss + kC;
    float* set = sal + kC;
    uint64_t* bars = reinterpret_cast<uint64_t*>(set + kC);
    uint64_t* tma_bar = bars;
    uint64_t* mma_bar = bars + 1;
    uint32_t* tslot = reinterpret_cast<uint32_t*>(bars + 2);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(bars + 3);

    const int tid = threadIdx.x, warp = tid >> 5;
    const long long unit = blockIdx.x / nch;
    const int c = (int)(blockIdx.x % nch);
    const int h = (int)(unit % H);
    const long long lb = unit / H;
    const int b = (int)(lb % B);
    const int l = (int)(lb / B);
    const int c0 = c * kC;
    if (warp == 0) {
        tmem_alloc(tslot, 128);
        tmem_relinquish();
    }
    if (tid == 0) {
        mbar_init(tma_bar, 1);
        mbar_init(mma_bar, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tslot;
    if (tid == 0) {
        mbar_arrive_expect_tx(tma_bar, 4 * kTile);
        tma_load_5d(smem + oX, &tm_x, tma_bar, 0, h, c0, b, l);
        tma_load_5d(smem + oG, &tm_g, tma_bar, 0, h, c0, b, l);
        tma_load_5d(smem + oB, &tm_b, tma_bar, 0, h, c0, b, l);
        tma_load_5d(smem + oA, &tm_a, tma_bar, 0, h, c0, b, l);
    }
    // ---- prefix / suffix products of the chunk's alphas (Hillis-Steele, 7 steps)
    const int t = c0 + tid;
    const long long gi = (lb * T + t) * H + h;
    const float a_own = t < T ? (alpha ? alpha[gi] : 1.0f) : 1.0f;
    set[tid] = t < T ? eta[gi] : 0.0f;
    float pr = a_own, su = a_own;  // inclusive
#pragma unroll 1
    for (int o = 1; o < kC; o <<= 1) {
        sp[tid] = pr;
        ss[tid] = su;
        __syncthreads();
        if (tid >= o) pr *= sp[tid - o];
        if (tid + o < kC) su *= ss[tid + o];
        __syncthreads();
    }
    sp[tid] = pr;
    ss[tid] = su;
    __syncthreads();
    const float p_ex = tid > 0 ? sp[tid - 1] : 1.0f;       // alphas before tid
    const float q_ex = tid + 1 < kC ? ss[tid + 1] : 1.0f;  // alphas after tid
    const float wgt = -set[tid] * q_ex;
    // ---- the scaled rows w Ghat and p A (thread = token row)
    bool ok = wait_bar(tma_bar, 0, abort_flag, err);
#pragma unroll 1
    for (int q = 0; q < 8; ++q) {
        const uint4 g4 = ld_shared_v4(sb + oG + sw128_off(tid, q));
        const uint4 a4 = ld_shared_v4(sb + oA + sw128_off(tid, q));
        const __nv_bfloat162* gh2 = reinterpret_cast<const __nv_bfloat162*>(&g4);
        const __nv_bfloat162* ah2 = reinterpret_cast<const __nv_bfloat162*>(&a4);
        uint32_t og[4], oa[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float2 gf = __bfloat1622float2(gh2[e]);
            const float2 af = __bfloat1622float2(ah2[e]);
            og[e] = pack_bf16x2(wgt * gf.x, wgt * gf.y);
            oa[e] = pack_bf16x2(p_ex * af.x, p_ex * af.y);
        }
        st_shared_v4(sb + oWG + sw128_off(tid, q), og[0], og[1], og[2], og[3]);
        st_shared_v4(sb + oPA + sw128_off(tid, q), oa[0], oa[1], oa[2], oa[3]);
    }
    fence_proxy_async_smem();
    __syncthreads();
    if (tid == 0 && ok) {
        tc_fence_after();
        constexpr uint32_t ID = idesc_bf16(128, 64, true, true);
        const uint32_t x_lo = sdesc_lo(sb + oX, kTile), b_lo = sdesc_lo(sb + oB, kTile);
        const uint32_t wg_lo = sdesc_lo(sb + oWG, kTile), pa_lo = sdesc_lo(sb + oPA, kTile);
#pragma unroll
        for (int kk = 0; kk < kC / 16; ++kk)  // Vt = X^T (w Ghat) into columns 0..63
            mma_bf16_ss(tmem, sdesc_from_lo(x_lo + kk * 128), sdesc_from_lo(wg_lo + kk * 128), ID, kk > 0 ? 1u : 0u);
#pragma unroll
        for (int kk = 0; kk < kC / 16; ++kk)  // Ut = B^T (p A) into columns 64..127
            mma_bf16_ss(tmem + 64, sdesc_from_lo(b_lo + kk * 128), sdesc_from_lo(pa_lo + kk * 128), ID,
                        kk > 0 ? 1u : 0u);
        mma_commit(mma_bar);
    }
    ok = wait_bar(mma_bar, 0, abort_flag, err) && ok;
    tc_fence_after();
    if (warp < 2) {  // rows k = 0..63 of both accumulators
        const uint32_t lane_base = tmem + (static_cast<uint32_t>(warp * 32) << 16);
        const long long blk = (unit * nch + c) * (long long)(64 * 64) + tid * 64;
#pragma unroll 1
        for (int hf = 0; hf < 2; ++hf) {
            float vv[32], uu[32];
            tmem_ld32(lane_base + 32 * hf, vv);
            tmem_ld32(lane_base + 64 + 32 * hf, uu);
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                reinterpret_cast<float4*>(Vd + blk + 32 * hf)[q] =
                    make_float4(vv[4 * q], vv[4 * q + 1], vv[4 * q + 2], vv[4 * q + 3]);
                reinterpret_cast<float4*>(Ud + blk + 32 * hf)[q] =
                    make_float4(uu[4 * q], uu[4 * q + 1], uu[4 * q + 2], uu[4 * q + 3]);
            }
        }
    } else {
        // keep the warps' TMEM access shape uniform: nothing to read in lanes 64..127
    }
    if (tid == kC - 1) Ad[unit * nch + c] = sp[kC - 1];
    tc_fence_before();
    __syncthreads();
    if (tid == 0 && *abort_flag) {  // no copy in flight at exit (bounded: 0.2 s)
        const uint64_t t0 = globaltimer_ns();
        while (!mbar_try_wait(tma_bar, 0) && globaltimer_ns() - t0 < 200000000ull) {
        }
    }
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, 128);
    }
}

}  // namespace ggtc

cudaError_t launch_gate_aggregates_tc(const CUtensorMap& x, const CUtensorMap& g, const CUtensorMap& a,
                                      const CUtensorMap& b, const float* eta, const float* alpha, float* Vd,
                                      float* Ud, float* Ad, int L, int B, int T, int H, unsigned int* err,
                                      cudaStream_t stream) {
    const int nch = (T + ggtc::kC - 1) / ggtc::kC;
    const long long blocks = (long long)L * B * H * nch;
    if (blocks <= 0) return cudaSuccess;
    if (blocks > 0x7FFFFFFF) return cudaErrorInvalidValue;
    cudaError_t e = cudaFuncSetAttribute(ggtc::gate_agg_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         ggtc::kAggSmem);
    if (e != cudaSuccess) return e;
    ggtc::gate_agg_tc_kernel<<<(int)blocks, ggtc::kThreads, ggtc::kAggSmem, stream>>>(
        x, g, a, b, eta, alpha, Vd, Ud, Ad, B, T, H, nch, err);
    return cudaGetLastError();
}

cudaError_t launch_gate_chunks_tc(const CUtensorMap& x, const CUtensorMap& g, const CUtensorMap& a,
                                  const CUtensorMap& b, const float* eta, const float* alpha, const float* Sd,
                                  const float* Rd, float* dlog_alpha, float* deta, int L, int B, int T, int H,
                                  unsigned int* err, cudaStream_t stream) {
    const int nch = (T + ggtc::kC - 1) / ggtc::kC;
    const long long blocks = (long long)L * B * H * nch;
    if (blocks <= 0) return cudaSuccess;
    if (blocks > 0x7FFFFFFF) return cudaErrorInvalidValue;
    cudaError_t e = cudaFuncSetAttribute(ggtc::gate_chunk_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         ggtc::kSmem);
    if (e != cudaSuccess) return e;
    ggtc::gate_chunk_tc_kernel<<<(int)blocks, ggtc::kThreads, ggtc::kSmem, stream>>>(
        x, g, a, b, eta, alpha, Sd, Rd, dlog_alpha, deta, B, T, H, nch, err);
    return cudaGetLastError();
}

}  // namespace gl
