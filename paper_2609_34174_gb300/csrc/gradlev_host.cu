// gradlev_host.cu -- the C ABI of include/gradlev.h: argument validation, work
// planning, TMA descriptor creation and kernel launch.  No compute happens on
// the host and there is no host fallback: a call either launches its kernels on
// the caller's stream or returns an error without launching anything.
#include <cuda.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#include <mutex>

#include "../../include/gradlev.h"
#include "scan_common.cuh"

namespace gl {
cudaError_t launch_tc_scan(const CUtensorMap& q, const CUtensorMap& k, const CUtensorMap& v,
                           const CUtensorMap& o, const TcScanParams& p, bool costate, int grid,
                           cudaStream_t stream);
cudaError_t launch_simt_scan(const SimtScanParams& p, bool bf16, bool rev, cudaStream_t stream);
cudaError_t launch_tc_suffix(const CUtensorMap& q, const CUtensorMap& k, const CUtensorMap& v,
                             const CUtensorMap& o, const TcScanParams& p, bool shared_qk, int grid,
                             cudaStream_t stream);
cudaError_t launch_rowdot(const void* a, const TokStr& as, const void* r, const TokStr& rs,
                          float* out, int L, int B, int T, int H, int w, float scale, bool bf16,
                          cudaStream_t stream, bool sqdist = false);
cudaError_t launch_tc_decay(const CUtensorMap& q, const CUtensorMap& k, const CUtensorMap& v,
                            const CUtensorMap& o, const TcScanParams& p, bool costate, int grid,
                            cudaStream_t stream);
cudaError_t launch_gate_state_scan(float* VS, float* UR, const float* Ad, long long units, int nch,
                                   cudaStream_t stream);
cudaError_t launch_gate_aggregates_tc(const CUtensorMap& x, const CUtensorMap& g, const CUtensorMap& a,
                                      const CUtensorMap& b, const float* eta, const float* alpha, float* Vd,
                                      float* Ud, float* Ad, int L, int B, int T, int H, unsigned int* err,
                                      cudaStream_t stream);
cudaError_t launch_gate_chunks_tc(const CUtensorMap& x, const CUtensorMap& g, const CUtensorMap& a,
                                  const CUtensorMap& b, const float* eta, const float* alpha, const float* Sd,
                                  const float* Rd, float* dlog_alpha, float* deta, int L, int B, int T, int H,
                                  unsigned int* err, cudaStream_t stream);
cudaError_t launch_tc_fused(const CUtensorMap& x, const CUtensorMap& ghat, const CUtensorMap& gout,
                            const CUtensorMap& y, const CUtensorMap& gin, const TcScanParams& p,
                            int grid, cudaStream_t stream);
cudaError_t launch_seg_gemm(int mode, int bn, const CUtensorMap& a, const CUtensorMap& b,
                            const CUtensorMap& a2, const CUtensorMap& b2, const SegGemmParams& p,
                            int grid, cudaStream_t stream);
size_t simt_smem_bytes(int dq);
size_t gated_serial_smem(int din, int dout, bool costate);
cudaError_t launch_gated_serial(const GatedParams& p, bool costate, bool bf16, cudaStream_t stream);
cudaError_t launch_gated_prescale(const void* g, const TokStr& gs, const float* eta, void* out, int L,
                                  int B, int T, int H, int w, bool bf16, cudaStream_t stream);
cudaError_t launch_decode_read(const DecodeParams& p, bool bf16, cudaStream_t stream);
cudaError_t launch_decode_write(const DecodeParams& p, bool bf16, bool gin, cudaStream_t stream);
}  // namespace gl

namespace {

using gl::TcScanParams;

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(ptr);
    });
    return fn;
}

constexpr int kMaxDevices = 64;

struct DevInfo {
    int sms = 0;
    int major = 0, minor = 0;
    bool ok = false;
};

bool device_info(DevInfo* out) {
    static DevInfo cache[kMaxDevices];
    static std::mutex mu;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return false;
    std::lock_guard<std::mutex> g(mu);
    if (!cache[dev].ok) {
        DevInfo d;
        if (cudaDeviceGetAttribute(&d.sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&d.major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&d.minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess)
            return false;
        d.ok = true;
        cache[dev] = d;
    }
    *out = cache[dev];
    return true;
}

// Resolved token tensor: pointer plus element strides of (L, B, T, H).
struct Tok {
    void* data = nullptr;
    long long s[4] = {0, 0, 0, 0};
};

bool resolve(const gradlev_desc& d, const gradlev_tensor* t, int width, Tok* out, bool required) {
    if (!t) return !required;
    // an empty sequence (T = 0) has no storage: a null pointer is then accepted, and
    // every caller returns before it launches anything
    if (!t->data) return !required || d.T == 0;
    out->data = t->data;
    bool zero = true;
    for (int i = 0; i < 4; ++i) zero = zero && t->stride[i] == 0;
    if (zero) {
        out->s[3] = width;
        out->s[2] = (long long)d.H * width;
        out->s[1] = (long long)d.T * d.H * width;
        out->s[0] = (long long)d.B * d.T * d.H * width;
    } else {
        const int dims[4] = {d.L, d.B, d.T, d.H};
        // natural contiguous strides, used for size-1 dimensions (never indexed)
        const long long nat[4] = {(long long)d.B * d.T * d.H * width, (long long)d.T * d.H * width,
                                  (long long)d.H * width, (long long)width};
        for (int i = 0; i < 4; ++i) {
            if (t->stride[i] < 0) return false;
            if (t->stride[i] == 0 && dims[i] > 1) return false;
            out->s[i] = dims[i] == 1 ? nat[i] : t->stride[i];
        }
        if (d.H > 1 && out->s[3] < width) return false;  // rows of one token must not overlap
    }
    return true;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// The tensor-core path moves 16-byte pieces: base and every stride must keep
// each 64-element row piece 16-byte aligned, and TMA needs strides < 2^40 bytes.
bool tc_layout_ok(const Tok& t, int elem) {
    if (!t.data) return true;
    if (!aligned16(t.data)) return false;
    for (int i = 0; i < 4; ++i) {
        long long bytes = t.s[i] * elem;
        if (bytes % 16 != 0 || bytes >= (1ll << 40)) return false;
    }
    return true;
}

// Segment plan of the tensor-core path: enough (unit, tile, segment) items to
// keep every SM busy, with segments of at least 512 tokens.
struct Plan {
    int n_tiles = 0, seg_len = 0, n_seg = 1, n_items = 0;
    size_t ws_bytes = 0;
    // workspace layout
    size_t off_flags = 0, off_agg = 0, off_incl = 0, zero_bytes = 0;
};

constexpr int kChunk = 128;

size_t round_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

Plan plan_tc(const gradlev_desc& d, int dq, int dv, int sms) {
    Plan pl;
    pl.n_tiles = dv / 64;
    const long long units = (long long)d.L * d.B * d.H * pl.n_tiles;
    const long long nsm = sms > 0 ? sms : 148;
    // Segment count: with fewer (unit, tile) pairs than two per SM and a long
    // sequence, split it so every SM gets work.  Pick the count that minimises
    // the chunks the busiest SM processes: waves x chunks per segment, with the
    // phase-1 re-stream of every segment but the last (about 0.55 of a full chunk)
    // and a look-back (about 0.7 of a chunk) per item.  Ties go to fewer segments.
    long long best_seg = ((long long)d.T + kChunk - 1) / kChunk * kChunk;
    if (units < 2 * nsm && d.T > 1024) {
        const long long max_seg = (d.T + 511) / 512;
        double best = 1e300;
        for (long long n = 1; n <= max_seg; ++n) {
            long long seg = ((long long)d.T + n - 1) / n;
            seg = (seg + kChunk - 1) / kChunk * kChunk;
            const long long n_eff = ((long long)d.T + seg - 1) / seg;
            const long long waves = (units * n_eff + nsm - 1) / nsm;
            const double chunks = (double)(seg / kChunk);
            const double p1 = n_eff > 1 ? 0.55 * (double)(n_eff - 1) / (double)n_eff : 0.0;
            const double cost = (double)waves * (chunks * (1.0 + p1) + (n_eff > 1 ? 0.7 : 0.0));
            if (cost < best * (1.0 - 1e-9)) {
                best = cost;
                best_seg = seg;
            }
        }
    }
    long long seg = best_seg;
    if (seg < kChunk) seg = kChunk;
    pl.seg_len = (int)seg;
    pl.n_seg = (int)(((long long)d.T + seg - 1) / seg);
    if (pl.n_seg < 1) pl.n_seg = 1;
    pl.n_items = (int)(units * pl.n_seg);
    pl.off_flags = 256;
    pl.off_agg = round_up(pl.off_flags + sizeof(unsigned int) * (size_t)pl.n_items, 256);
    pl.zero_bytes = pl.off_agg;
    size_t blk = sizeof(float) * (size_t)dq * 64;
    if (pl.n_seg > 1) {
        pl.off_incl = pl.off_agg + blk * (size_t)pl.n_items;
        pl.ws_bytes = pl.off_incl + blk * (size_t)pl.n_items;
    } else {
        pl.off_incl = pl.off_agg;
        pl.ws_bytes = pl.off_agg;
    }
    return pl;
}

bool tc_shape_ok(const gradlev_desc& d, int dq, int dv) {
    return d.dtype == GRADLEV_BF16 && (dq == 64 || dq == 128) && dv % 64 == 0 && dv > 0;
}

// The chunk kernel keeps its running state in units of lambda = -eta (it holds
// S / lambda, so that the masked score needs no scaling and the output is
// multiplied by lambda once).  That needs 1 / lambda and W0 / lambda to stay
// well inside fp32: |eta| within [2^-64, 2^64] (or eta = 0, which keeps lambda = 1).
// Any other finite eta runs on the CUDA-core kernel, which scales by eta directly.
bool tc_eta_ok(float eta) {
    const float a = fabsf(eta);
    return eta == 0.0f || (a >= 0x1p-64f && a <= 0x1p64f);
}

constexpr int kSimtMaxDq = 256;

bool simt_shape_ok(const gradlev_desc& d, int dq) {
    (void)d;
    return dq >= 1 && dq <= kSimtMaxDq;
}

bool desc_ok(const gradlev_desc* d) {
    if (!d) return false;
    if (d->L < 1 || d->B < 1 || d->H < 1 || d->T < 0 || d->d_in < 1 || d->d_out < 1) return false;
    if (d->dtype != GRADLEV_F32 && d->dtype != GRADLEV_BF16) return false;
    if (d->reserved != 0) return false;
    long long units = (long long)d->L * d->B * d->H;
    if (units > (1ll << 30) || d->d_in > (1 << 20) || d->d_out > (1 << 20)) return false;
    return true;
}

bool make_tmap(CUtensorMap* m, const gradlev_desc& d, const Tok& t, int width, int box_t = kChunk) {
    EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    const cuuint64_t dims[5] = {(cuuint64_t)width, (cuuint64_t)d.H, (cuuint64_t)d.T, (cuuint64_t)d.B,
                                (cuuint64_t)d.L};
    // byte strides of dims 1..4; a size-1 dimension gets a harmless valid stride
    cuuint64_t strides[4];
    const long long s[4] = {t.s[3], t.s[2], t.s[1], t.s[0]};
    const int sizes[4] = {d.H, d.T, d.B, d.L};
    for (int i = 0; i < 4; ++i) {
        long long b = s[i] * 2;
        if (sizes[i] == 1 && b == 0) b = 16;
        strides[i] = (cuuint64_t)b;
    }
    const cuuint32_t box[5] = {64, 1, (cuuint32_t)box_t, 1, 1};
    const cuuint32_t estr[5] = {1, 1, 1, 1, 1};
    CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, t.data, dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

// 3-D bf16 map over a contiguous workspace tensor [n2][n1][n0] with a {64, box1, 1} box.
bool make_tmap_3d(CUtensorMap* m, void* base, long long n0, long long n1, long long n2, int box1) {
    EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    const cuuint64_t dims[3] = {(cuuint64_t)n0, (cuuint64_t)n1, (cuuint64_t)n2};
    const cuuint64_t strides[2] = {(cuuint64_t)(n0 * 2), (cuuint64_t)(n0 * n1 * 2)};
    const cuuint32_t box[3] = {64, (cuuint32_t)box1, 1};
    const cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, base, dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

// Wide layers (dq a multiple of 128 and at least 256): the scan split at segment
// boundaries into a state pass, a score pass and an output pass (seg_gemm_tc.cu).
struct SegPlan {
    int seg_len = 0, n_seg = 0, bn = 0;
    long long tiles_state = 0, tiles_score = 0, tiles_out = 0;
    size_t off_sbuf = 0, off_pbuf = 0, ws_bytes = 0;
};

bool seg_shape_ok(const gradlev_desc& d, int dq, int dv) {
    return d.dtype == GRADLEV_BF16 && dq >= 256 && dq % 128 == 0 && dv % 64 == 0 && dv > 0;
}

SegPlan plan_seg(const gradlev_desc& d, int dq, int dv) {
    SegPlan sp;
    const long long T = d.T > 0 ? d.T : 1;
    long long ls = (T + kChunk - 1) / kChunk * kChunk;
    if (ls > 1024) ls = 1024;  // measured best on 512 -> 2048 -> 512 (1024 vs 512: 4-6% faster)
    sp.seg_len = (int)ls;
    sp.n_seg = (int)((T + ls - 1) / ls);
    sp.bn = dv % 256 == 0 ? 256 : (dv % 128 == 0 ? 128 : 64);
    const long long U = (long long)d.L * d.B * d.H;
    const long long R = ls / kChunk;
    sp.tiles_state = U * (dq / 128) * (dv / sp.bn);
    sp.tiles_score = U * sp.n_seg * (R * (R + 1) / 2);
    sp.tiles_out = U * sp.n_seg * R * (dv / sp.bn);
    sp.off_sbuf = 1024;
    sp.off_pbuf = round_up(sp.off_sbuf + (size_t)U * sp.n_seg * dq * dv * 2, 1024);
    sp.ws_bytes = sp.off_pbuf + (size_t)U * sp.n_seg * ls * ls * 2;
    return sp;
}

void fill_epi(gl::EpiParams* e, const Tok& out, const Tok& out2, const Tok& z, int act) {
    e->out = out.data;
    e->out2 = out2.data;
    e->zin = z.data;
    e->act = act;
    for (int i = 0; i < 4; ++i) {
        e->out_str[i] = out.s[i];
        e->out2_str[i] = out2.s[i];
        e->z_str[i] = z.s[i];
    }
}

// Shared driver of both scans.  Roles (Sec. 3, Eqs. 3-4):
//   forward:  q = k = x, v = g_hat, B0 = W0     (dq = d_in,  dv = d_out)
//   costate:  q = g_out, k = g_hat, v = x, B0 = W0^T (dq = d_out, dv = d_in)
// With dry set, every argument check runs and nothing is launched.
int run_scan(const gradlev_desc* desc, bool costate, const gradlev_tensor* x,
             const gradlev_tensor* g_hat, const float* W0, float eta, const gradlev_tensor* g_out,
             int act, const gradlev_tensor* out, const gradlev_tensor* out2,
             const gradlev_tensor* z, void* ws, size_t ws_bytes, cudaStream_t stream,
             bool dry = false) {
    if (!desc_ok(desc)) return GRADLEV_ERR_INVALID_ARG;
    const gradlev_desc& d = *desc;
    if (!W0 || !isfinite(eta)) return GRADLEV_ERR_INVALID_ARG;
    if (act < GRADLEV_ACT_NONE || act > GRADLEV_ACT_TANH) return GRADLEV_ERR_INVALID_ARG;
    const int din = d.d_in, dout = d.d_out;
    Tok tx, tg, tgo, to, to2, tz;
    if (!resolve(d, x, din, &tx, true) || !resolve(d, g_hat, dout, &tg, true) ||
        !resolve(d, out, costate ? din : dout, &to, true))
        return GRADLEV_ERR_INVALID_ARG;
    if (costate) {
        if (!resolve(d, g_out, dout, &tgo, true) || !resolve(d, z, din, &tz, false))
            return GRADLEV_ERR_INVALID_ARG;
        if (tz.data && act == GRADLEV_ACT_NONE) return GRADLEV_ERR_INVALID_ARG;
    } else {
        if (!resolve(d, out2, dout, &to2, false)) return GRADLEV_ERR_INVALID_ARG;
        if (to2.data && act == GRADLEV_ACT_NONE) return GRADLEV_ERR_INVALID_ARG;
    }
    DevInfo dev;
    if (!device_info(&dev)) return GRADLEV_ERR_CUDA;
    if (!(dev.major == 10 && dev.minor == 3)) return GRADLEV_ERR_UNSUPPORTED;
    if (d.T == 0) return GRADLEV_OK;

    const int dq = costate ? dout : din;
    const int dv = costate ? din : dout;
    const Tok& tq = costate ? tgo : tx;
    const Tok& tk = costate ? tg : tx;
    const Tok& tv = costate ? tx : tg;
    const int elem = d.dtype == GRADLEV_BF16 ? 2 : 4;

    if (tc_shape_ok(d, dq, dv) && tc_eta_ok(eta) && tc_layout_ok(tq, 2) && tc_layout_ok(tk, 2) &&
        tc_layout_ok(tv, 2) && tc_layout_ok(to, 2) && tc_layout_ok(to2, 2) && tc_layout_ok(tz, 2)) {
        Plan pl = plan_tc(d, dq, dv, dev.sms);
        if (!ws || ws_bytes < pl.ws_bytes) return GRADLEV_ERR_WORKSPACE;
        if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return GRADLEV_ERR_WORKSPACE;
        CUtensorMap mq, mk, mv, mo;
        if (!make_tmap(&mq, d, tq, dq) || !make_tmap(&mk, d, tk, dq) || !make_tmap(&mv, d, tv, dv) ||
            !make_tmap(&mo, d, to, dv))
            return GRADLEV_ERR_UNSUPPORTED;
        TcScanParams p;
        memset(&p, 0, sizeof(p));
        p.L = d.L;
        p.B = d.B;
        p.T = d.T;
        p.H = d.H;
        p.dq = dq;
        p.dv = dv;
        p.n_tiles = pl.n_tiles;
        p.seg_len = pl.seg_len;
        p.n_seg = pl.n_seg;
        p.n_items = pl.n_items;
        p.n_ut = pl.n_items / pl.n_seg;
        // A look-back wait is bounded by 4 s.  Failure tests (host-side fault
        // injection, no GPU fault) can make one item skip its publish and shorten
        // the bound, so that its successors' waits expire, the kernel writes
        // the error word and returns, and the host reports GRADLEV_ERR_TIMEOUT.
        p.lookback_limit_ns = 4000000000ull;
        p.test_skip_publish = -1;
        if (const char* v = getenv("GRADLEV_TEST_SKIP_PUBLISH")) p.test_skip_publish = atoi(v);
        if (const char* v = getenv("GRADLEV_TEST_LOOKBACK_LIMIT_MS"))
            p.lookback_limit_ns = 1000000ull * (unsigned long long)atoi(v);
        p.eta = eta;
        p.lam = eta != 0.0f ? -eta : 1.0f;
        p.inv_lam = 1.0f / p.lam;
        p.mu = eta != 0.0f ? 1.0f : 0.0f;
        p.w0_transposed = costate ? 1 : 0;
        p.W0 = W0;
        fill_epi(&p.epi, to, to2, tz, act);
        uint8_t* wsb = static_cast<uint8_t*>(ws);
        p.ctrl = reinterpret_cast<unsigned int*>(wsb);
        p.flags = reinterpret_cast<unsigned int*>(wsb + pl.off_flags);
        p.agg = reinterpret_cast<float*>(wsb + pl.off_agg);
        p.incl = reinterpret_cast<float*>(wsb + pl.off_incl);
        if (dry) return GRADLEV_OK;
        if (cudaMemsetAsync(ws, 0, pl.zero_bytes, stream) != cudaSuccess) return GRADLEV_ERR_CUDA;
        const int grid = pl.n_items < dev.sms ? pl.n_items : dev.sms;
        if (gl::launch_tc_scan(mq, mk, mv, mo, p, costate, grid, stream) != cudaSuccess)
            return GRADLEV_ERR_CUDA;
        return GRADLEV_OK;
    }
    if (seg_shape_ok(d, dq, dv) && tc_layout_ok(tq, 2) && tc_layout_ok(tk, 2) &&
        tc_layout_ok(tv, 2) && tc_layout_ok(to, 2) && tc_layout_ok(to2, 2) && tc_layout_ok(tz, 2)) {
        SegPlan sp = plan_seg(d, dq, dv);
        const long long lim = 0x7fffffffll;
        if (sp.tiles_state > lim || sp.tiles_score > lim || sp.tiles_out > lim ||
            (long long)d.L * d.B * d.H * sp.n_seg > lim)
            return GRADLEV_ERR_UNSUPPORTED;
        if (!ws || ws_bytes < sp.ws_bytes) return GRADLEV_ERR_WORKSPACE;
        if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return GRADLEV_ERR_WORKSPACE;
        if (!aligned16(W0)) return GRADLEV_ERR_INVALID_ARG;
        uint8_t* wsb = static_cast<uint8_t*>(ws);
        const long long us = (long long)d.L * d.B * d.H * sp.n_seg;
        CUtensorMap mq, mk, mk64, mv64, msb, mpb;
        if (!make_tmap(&mq, d, tq, dq) || !make_tmap(&mk, d, tk, dq) ||
            !make_tmap(&mk64, d, tk, dq, 64) || !make_tmap(&mv64, d, tv, dv, 64) ||
            !make_tmap_3d(&msb, wsb + sp.off_sbuf, dv, dq, us, 64) ||
            !make_tmap_3d(&mpb, wsb + sp.off_pbuf, sp.seg_len, sp.seg_len, us, kChunk))
            return GRADLEV_ERR_UNSUPPORTED;
        gl::SegGemmParams p;
        memset(&p, 0, sizeof(p));
        p.L = d.L;
        p.B = d.B;
        p.T = d.T;
        p.H = d.H;
        p.dq = dq;
        p.dv = dv;
        p.seg_len = sp.seg_len;
        p.n_seg = sp.n_seg;
        p.eta = eta;
        p.w0_transposed = costate ? 1 : 0;
        p.W0 = W0;
        p.sbuf = reinterpret_cast<__nv_bfloat16*>(wsb + sp.off_sbuf);
        p.pbuf = reinterpret_cast<__nv_bfloat16*>(wsb + sp.off_pbuf);
        fill_epi(&p.epi, to, to2, tz, act);
        p.ctrl = reinterpret_cast<unsigned int*>(wsb);
        if (dry) return GRADLEV_OK;
        if (cudaMemsetAsync(ws, 0, 256, stream) != cudaSuccess) return GRADLEV_ERR_CUDA;
        const long long tiles[3] = {sp.tiles_state, sp.tiles_score, sp.tiles_out};
        for (int mode = 0; mode < 3; ++mode) {
            p.n_tiles = (int)tiles[mode];
            const int grid = p.n_tiles < dev.sms ? p.n_tiles : dev.sms;
            if (grid < 1) continue;
            cudaError_t e;
            if (mode == 0)
                e = gl::launch_seg_gemm(0, sp.bn, mk64, mv64, mk64, mv64, p, grid, stream);
            else if (mode == 1)
                e = gl::launch_seg_gemm(1, sp.bn, mq, mk, mq, mk, p, grid, stream);
            else
                e = gl::launch_seg_gemm(2, sp.bn, mq, msb, mpb, mv64, p, grid, stream);
            if (e != cudaSuccess) return GRADLEV_ERR_CUDA;
        }
        return GRADLEV_OK;
    }
    if (simt_shape_ok(d, dq)) {
        // CUDA-core path: fp32 (exact fp32 FMA), or bf16 shapes the tensor-core
        // tiling does not cover.  Needs only element alignment.
        const Tok* all[6] = {&tq, &tk, &tv, &to, &to2, &tz};
        for (const Tok* t : all)
            if (t->data && (reinterpret_cast<uintptr_t>(t->data) % elem) != 0)
                return GRADLEV_ERR_UNSUPPORTED;
        if ((reinterpret_cast<uintptr_t>(W0) & 3u) != 0) return GRADLEV_ERR_INVALID_ARG;
        if (ws && (reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return GRADLEV_ERR_WORKSPACE;
        if (dry) return GRADLEV_OK;
        if (ws) {
            if (ws_bytes >= 256 && cudaMemsetAsync(ws, 0, 256, stream) != cudaSuccess)
                return GRADLEV_ERR_CUDA;
        }
        gl::SimtScanParams p;
        memset(&p, 0, sizeof(p));
        p.L = d.L;
        p.B = d.B;
        p.T = d.T;
        p.H = d.H;
        p.dq = dq;
        p.dv = dv;
        p.eta = eta;
        p.w0_transposed = costate ? 1 : 0;
        p.W0 = W0;
        p.q = tq.data;
        p.k = tk.data;
        p.v = tv.data;
        for (int i = 0; i < 4; ++i) {
            p.q_str[i] = tq.s[i];
            p.k_str[i] = tk.s[i];
            p.v_str[i] = tv.s[i];
        }
        fill_epi(&p.epi, to, to2, tz, act);
        if (gl::launch_simt_scan(p, d.dtype == GRADLEV_BF16, false, stream) != cudaSuccess)
            return GRADLEV_ERR_CUDA;
        return GRADLEV_OK;
    }
    return GRADLEV_ERR_UNSUPPORTED;
}

// Both reads of a map in one call (Sec. 3, steps 2 and 3): y_t = W_t x_t and
// g_in_t = W_t^T g_out_t over the same writes, with the optional per-token
// consistency term cons_t = ||p_t - g_in_t||^2 / d_in against proposals p (Eq. 5).
// 64 x 64 bf16 maps run the single-pass kernel; other shapes run the forward and
// the costate scan one after the other (every check of both passes first).
int run_fused(const gradlev_desc* desc, const gradlev_tensor* x, const gradlev_tensor* g_hat,
              const float* W0, float eta, const gradlev_tensor* g_out, const gradlev_tensor* y,
              const gradlev_tensor* g_in, const gradlev_tensor* cons_p, float* cons, void* ws,
              size_t ws_bytes, cudaStream_t stream) {
    if (!desc_ok(desc)) return GRADLEV_ERR_INVALID_ARG;
    const gradlev_desc& d = *desc;
    if (!W0 || !isfinite(eta)) return GRADLEV_ERR_INVALID_ARG;
    const int din = d.d_in, dout = d.d_out;
    Tok tx, tg, tgo, ty, tgi, tp;
    if (!resolve(d, x, din, &tx, true) || !resolve(d, g_hat, dout, &tg, true) ||
        !resolve(d, g_out, dout, &tgo, true) || !resolve(d, y, dout, &ty, true) ||
        !resolve(d, g_in, din, &tgi, true) || !resolve(d, cons_p, din, &tp, false))
        return GRADLEV_ERR_INVALID_ARG;
    const bool want_cons = tp.data != nullptr && d.T > 0;
    if ((cons_p && cons_p->data) != (cons != nullptr)) return GRADLEV_ERR_INVALID_ARG;
    if (cons && (reinterpret_cast<uintptr_t>(cons) & 3u) != 0) return GRADLEV_ERR_INVALID_ARG;
    DevInfo dev;
    if (!device_info(&dev)) return GRADLEV_ERR_CUDA;
    if (!(dev.major == 10 && dev.minor == 3)) return GRADLEV_ERR_UNSUPPORTED;
    if (d.T == 0) return GRADLEV_OK;
    const bool bf16 = d.dtype == GRADLEV_BF16;
    if (bf16 && din == 64 && dout == 64 && tc_eta_ok(eta) && tc_layout_ok(tx, 2) &&
        tc_layout_ok(tg, 2) && tc_layout_ok(tgo, 2) && tc_layout_ok(ty, 2) && tc_layout_ok(tgi, 2) &&
        tc_layout_ok(tp, 2)) {
        Plan pl = plan_tc(d, 64, 64, dev.sms);
        if (!ws || ws_bytes < pl.ws_bytes) return GRADLEV_ERR_WORKSPACE;
        if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return GRADLEV_ERR_WORKSPACE;
        CUtensorMap mx, mg, mgo, my, mgi;
        if (!make_tmap(&mx, d, tx, 64) || !make_tmap(&mg, d, tg, 64) || !make_tmap(&mgo, d, tgo, 64) ||
            !make_tmap(&my, d, ty, 64) || !make_tmap(&mgi, d, tgi, 64))
            return GRADLEV_ERR_UNSUPPORTED;
        TcScanParams p;
        memset(&p, 0, sizeof(p));
        p.L = d.L;
        p.B = d.B;
        p.T = d.T;
        p.H = d.H;
        p.dq = 64;
        p.dv = 64;
        p.n_tiles = pl.n_tiles;
        p.seg_len = pl.seg_len;
        p.n_seg = pl.n_seg;
        p.n_items = pl.n_items;
        p.n_ut = pl.n_items / pl.n_seg;
        p.lookback_limit_ns = 4000000000ull;
        p.test_skip_publish = -1;
        if (const char* v = getenv("GRADLEV_TEST_SKIP_PUBLISH")) p.test_skip_publish = atoi(v);
        if (const char* v = getenv("GRADLEV_TEST_LOOKBACK_LIMIT_MS"))
            p.lookback_limit_ns = 1000000ull * (unsigned long long)atoi(v);
        p.eta = eta;
        p.lam = eta != 0.0f ? -eta : 1.0f;
        p.inv_lam = 1.0f / p.lam;
        p.mu = eta != 0.0f ? 1.0f : 0.0f;
        p.w0_transposed = 0;  // the state in the forward orientation, W0^T rows
        p.W0 = W0;
        const Tok none;
        fill_epi(&p.epi, ty, none, none, GRADLEV_ACT_NONE);
        if (want_cons) {
            p.epi.cons_p = tp.data;
            for (int i = 0; i < 4; ++i) p.epi.cons_str[i] = tp.s[i];
            p.epi.cons_out = cons;
            p.epi.cons_scale = 1.0f / (float)din;
        }
        uint8_t* wsb = static_cast<uint8_t*>(ws);
        p.ctrl = reinterpret_cast<unsigned int*>(wsb);
        p.flags = reinterpret_cast<unsigned int*>(wsb + pl.off_flags);
        p.agg = reinterpret_cast<float*>(wsb + pl.off_agg);
        p.incl = reinterpret_cast<float*>(wsb + pl.off_incl);
        if (cudaMemsetAsync(ws, 0, pl.zero_bytes, stream) != cudaSuccess) return GRADLEV_ERR_CUDA;
        const int grid = pl.n_items < dev.sms ? pl.n_items : dev.sms;
        if (gl::launch_tc_fused(mx, mg, mgo, my, mgi, p, grid, stream) != cudaSuccess)
            return GRADLEV_ERR_CUDA;
        return GRADLEV_OK;
    }
    // Other shapes: check both passes before launching either.
    int rc = run_scan(desc, false, x, g_hat, W0, eta, nullptr, GRADLEV_ACT_NONE, y, nullptr, nullptr,
                      ws, ws_bytes, stream, true);
    if (rc == GRADLEV_OK)
        rc = run_scan(desc, true, x, g_hat, W0, eta, g_out, GRADLEV_ACT_NONE, g_in, nullptr, nullptr,
                      ws, ws_bytes, stream, true);
    if (rc != GRADLEV_OK) return rc;
    rc = run_scan(desc, false, x, g_hat, W0, eta, nullptr, GRADLEV_ACT_NONE, y, nullptr, nullptr, ws,
                  ws_bytes, stream);
    if (rc == GRADLEV_OK)
        rc = run_scan(desc, true, x, g_hat, W0, eta, g_out, GRADLEV_ACT_NONE, g_in, nullptr, nullptr,
                      ws, ws_bytes, stream);
    if (rc != GRADLEV_OK || !want_cons) return rc;
    gl::TokStr ps, gs;
    for (int i = 0; i < 4; ++i) {
        ps.s[i] = tp.s[i];
        gs.s[i] = tgi.s[i];
    }
    if (gl::launch_rowdot(tp.data, ps, tgi.data, gs, cons, d.L, d.B, d.T, d.H, din, 1.0f / (float)din,
                          bf16, stream, true) != cudaSuccess)
        return GRADLEV_ERR_CUDA;
    return GRADLEV_OK;
}

size_t ws_bytes_for(const gradlev_desc& d, int dq, int dv, int sms) {
    size_t b = 256;
    if (tc_shape_ok(d, dq, dv)) {
        Plan pl = plan_tc(d, dq, dv, sms);
        if (pl.ws_bytes > b) b = pl.ws_bytes;
    } else if (seg_shape_ok(d, dq, dv)) {
        SegPlan sp = plan_seg(d, dq, dv);
        if (sp.ws_bytes > b) b = sp.ws_bytes;
    }
    return b;
}

// Gated scans (Eq. 2 with per-token eta_t and optional retention alpha_t).
constexpr int kGatedSerialMaxWidth = 256;

size_t gated_ws_bytes(const gradlev_desc& d, int sms) {
    const size_t a = ws_bytes_for(d, d.d_in, d.d_out, sms);
    const size_t b = ws_bytes_for(d, d.d_out, d.d_in, sms);
    const size_t base = round_up(a > b ? a : b, 256);
    const size_t elem = d.dtype == GRADLEV_BF16 ? 2 : 4;
    return base + (size_t)d.L * d.B * d.T * d.H * d.d_out * elem;
}

// The retention scan of 64 x 64 bf16 maps on the tensor cores (scan_decay_tc.cu): one
// work item per unit, or per segment of a few long units.  q, k, v are the read's
// orientation (forward: x, x, ghat; costate: g_out, ghat, x).
int run_decay_tc(const gradlev_desc& d, bool costate, const Tok& tq, const Tok& tk, const Tok& tv,
                 const Tok& to, const Tok& to2, const Tok& tz, int act, const float* W0,
                 const float* eta_t, const float* alpha_t, void* ws, size_t ws_bytes, int sms,
                 cudaStream_t stream) {
    CUtensorMap mq, mk, mv, mo;
    if (!make_tmap(&mq, d, tq, 64) || !make_tmap(&mk, d, tk, 64) || !make_tmap(&mv, d, tv, 64) ||
        !make_tmap(&mo, d, to, 64))
        return GRADLEV_ERR_UNSUPPORTED;
    const long long units = (long long)d.L * d.B * d.H;
    gl::TcScanParams p;
    memset(&p, 0, sizeof(p));
    p.L = d.L;
    p.B = d.B;
    p.T = d.T;
    p.H = d.H;
    p.dq = 64;
    p.dv = 64;
    p.n_tiles = 1;
    // Few long units: cut each into segments (multiples of 128 tokens, at least
    // 512) so that about four waves of items fill the SMs; the segments' states
    // are carried through an aggregate pass (scan_decay_tc.cu).
    int n_seg = 1;
    long long seg_len = d.T;
    if (units < 2ll * sms && d.T > 1024) {
        const long long want = (4ll * sms + units - 1) / units;
        seg_len = (((d.T + want - 1) / want) + 127) / 128 * 128;
        if (seg_len < 512) seg_len = 512;
        n_seg = (int)((d.T + seg_len - 1) / seg_len);
        if (n_seg < 2) {
            n_seg = 1;
            seg_len = d.T;
        }
    }
    p.seg_len = (int)seg_len;
    p.n_seg = n_seg;
    p.n_items = (int)(units * n_seg);
    p.n_ut = (int)units;
    if (n_seg > 1) {
        // the segment states go where the eta-only path keeps its scaled proposals
        // (d_out * elem >= 128 bytes per token-unit, against at most 64 here)
        const size_t a = ws_bytes_for(d, d.d_in, d.d_out, sms);
        const size_t bb = ws_bytes_for(d, d.d_out, d.d_in, sms);
        uint8_t* base = static_cast<uint8_t*>(ws) + round_up(a > bb ? a : bb, 256);
        const size_t blk = (size_t)p.n_items * 64 * 64 * sizeof(float);
        p.agg = reinterpret_cast<float*>(base);
        p.incl = reinterpret_cast<float*>(base + blk);
        p.seg_a = reinterpret_cast<float*>(base + 2 * blk);
        if (static_cast<size_t>(base - static_cast<uint8_t*>(ws)) + 2 * blk +
                round_up((size_t)p.n_items * sizeof(float), 256) > ws_bytes)
            return GRADLEV_ERR_WORKSPACE;
    }
    p.lam = 1.0f;
    p.inv_lam = 1.0f;
    p.mu = 1.0f;
    p.w0_transposed = costate ? 1 : 0;
    p.W0 = W0;
    p.g_eta = eta_t;
    p.g_alpha = alpha_t;
    fill_epi(&p.epi, to, to2, tz, act);
    p.ctrl = static_cast<unsigned int*>(ws);
    if (cudaMemsetAsync(ws, 0, 256, stream) != cudaSuccess) return GRADLEV_ERR_CUDA;
    const int grid = p.n_items < sms ? p.n_items : sms;
    if (gl::launch_tc_decay(mq, mk, mv, mo, p, costate, grid, stream) != cudaSuccess)
        return GRADLEV_ERR_CUDA;
    return GRADLEV_OK;
}

int run_gated(const gradlev_desc* desc, bool costate, const gradlev_tensor* x,
              const gradlev_tensor* g_hat, const float* W0, const float* eta_t,
              const float* alpha_t, const gradlev_tensor* g_out, int act, const gradlev_tensor* out,
              const gradlev_tensor* out2, const gradlev_tensor* z, void* ws, size_t ws_bytes,
              cudaStream_t stream) {
    if (!desc_ok(desc)) return GRADLEV_ERR_INVALID_ARG;
    const gradlev_desc& d = *desc;
    if (!W0 || (!eta_t && d.T > 0) || (reinterpret_cast<uintptr_t>(eta_t) & 3u) ||
        (alpha_t && (reinterpret_cast<uintptr_t>(alpha_t) & 3u)))
        return GRADLEV_ERR_INVALID_ARG;
    if (act < GRADLEV_ACT_NONE || act > GRADLEV_ACT_TANH) return GRADLEV_ERR_INVALID_ARG;
    DevInfo dev;
    if (!device_info(&dev)) return GRADLEV_ERR_CUDA;
    if (!(dev.major == 10 && dev.minor == 3)) return GRADLEV_ERR_UNSUPPORTED;
    if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return GRADLEV_ERR_WORKSPACE;
    if (ws_bytes < gated_ws_bytes(d, dev.sms)) return GRADLEV_ERR_WORKSPACE;
    if (d.T == 0) return GRADLEV_OK;
    const bool bf16 = d.dtype == GRADLEV_BF16;
    Tok tx, tg;
    if (!resolve(d, x, d.d_in, &tx, true) || !resolve(d, g_hat, d.d_out, &tg, true))
        return GRADLEV_ERR_INVALID_ARG;
    if (!alpha_t) {
        // eta_t only: scale the writes' proposals, then the ungated scan with eta = 1.
        // The scaling pass moves 16-byte pieces of each token row.
        if (d.d_out % (bf16 ? 8 : 4) != 0 || !tc_layout_ok(tg, bf16 ? 2 : 4))
            return GRADLEV_ERR_UNSUPPORTED;
        const size_t a = ws_bytes_for(d, d.d_in, d.d_out, dev.sms);
        const size_t b = ws_bytes_for(d, d.d_out, d.d_in, dev.sms);
        const size_t base = round_up(a > b ? a : b, 256);
        void* gp = static_cast<uint8_t*>(ws) + base;
        gl::TokStr gs;
        for (int i = 0; i < 4; ++i) gs.s[i] = tg.s[i];
        if (gl::launch_gated_prescale(tg.data, gs, eta_t, gp, d.L, d.B, d.T, d.H, d.d_out, bf16,
                                      stream) != cudaSuccess)
            return GRADLEV_ERR_CUDA;
        gradlev_tensor gpt;
        gpt.data = gp;
        for (int i = 0; i < 4; ++i) gpt.stride[i] = 0;
        return run_scan(desc, costate, x, &gpt, W0, 1.0f, g_out, act, out, out2, z, ws, base, stream);
    }
    // with retention: the tensor-core chunked kernel for 64 x 64 bf16 maps whose
    // tensors a TMA map can describe, else the kernels of gated.cu
    const int J = costate ? d.d_out : d.d_in;
    if (J > kGatedSerialMaxWidth) return GRADLEV_ERR_UNSUPPORTED;
    Tok tgo, to, to2, tz;
    if (!resolve(d, out, costate ? d.d_in : d.d_out, &to, true)) return GRADLEV_ERR_INVALID_ARG;
    if (costate) {
        if (!resolve(d, g_out, d.d_out, &tgo, true) || !resolve(d, z, d.d_in, &tz, false))
            return GRADLEV_ERR_INVALID_ARG;
        if (tz.data && act == GRADLEV_ACT_NONE) return GRADLEV_ERR_INVALID_ARG;
    } else {
        if (!resolve(d, out2, d.d_out, &to2, false)) return GRADLEV_ERR_INVALID_ARG;
        if (to2.data && act == GRADLEV_ACT_NONE) return GRADLEV_ERR_INVALID_ARG;
    }
    const int elem = bf16 ? 2 : 4;
    const Tok* all[6] = {&tx, &tg, &tgo, &to, &to2, &tz};
    for (const Tok* t : all)
        if (t->data && (reinterpret_cast<uintptr_t>(t->data) % elem) != 0) return GRADLEV_ERR_UNSUPPORTED;
    if ((reinterpret_cast<uintptr_t>(W0) & 3u) != 0) return GRADLEV_ERR_INVALID_ARG;
    if (bf16 && d.d_in == 64 && d.d_out == 64 && tc_layout_ok(tx, 2) && tc_layout_ok(tg, 2) &&
        (!costate || tc_layout_ok(tgo, 2)) && tc_layout_ok(to, 2) && tc_layout_ok(to2, 2) &&
        tc_layout_ok(tz, 2)) {
        // 64 x 64 bf16 maps: the chunked retention scan on the tensor cores
        return run_decay_tc(d, costate, costate ? tgo : tx, costate ? tg : tx, costate ? tx : tg, to, to2,
                            tz, act, W0, eta_t, alpha_t, ws, ws_bytes, dev.sms, stream);
    }
    if (cudaMemsetAsync(ws, 0, 256, stream) != cudaSuccess) return GRADLEV_ERR_CUDA;
    gl::GatedParams p;
    memset(&p, 0, sizeof(p));
    p.L = d.L;
    p.B = d.B;
    p.T = d.T;
    p.H = d.H;
    p.din = d.d_in;
    p.dout = d.d_out;
    p.W0 = W0;
    p.eta = eta_t;
    p.alpha = alpha_t;
    p.x = tx.data;
    p.g = tg.data;
    p.q = costate ? tgo.data : tx.data;
    for (int i = 0; i < 4; ++i) {
        p.x_s[i] = tx.s[i];
        p.g_s[i] = tg.s[i];
        p.q_s[i] = costate ? tgo.s[i] : tx.s[i];
    }
    fill_epi(&p.epi, to, to2, tz, act);
    if (gl::launch_gated_serial(p, costate, bf16, stream) != cudaSuccess) return GRADLEV_ERR_CUDA;
    return GRADLEV_OK;
}

// Suffix (anti-causal) read r_s = sum_{t>s} (k_t . q_s) v_t: d_in is the width of q
// and k, d_out the width of v and r.  The scan kernels run in reverse with no base
// matrix and eta = -1: the tensor-core kernel for bf16 with 64-wide q and k, the
// CUDA-core kernel otherwise.
bool suffix_tc_shape(const gradlev_desc& d) {
    return d.dtype == GRADLEV_BF16 && d.d_in == 64 && d.d_out % 64 == 0;
}

int dev_sms_or_default() {
    DevInfo dev;
    return device_info(&dev) ? dev.sms : 160;
}

bool same_tensor(const Tok& a, const Tok& b) {
    if (a.data != b.data) return false;
    for (int i = 0; i < 4; ++i)
        if (a.s[i] != b.s[i]) return false;
    return true;
}

size_t suffix_ws_bytes(const gradlev_desc& d, int sms) {
    return suffix_tc_shape(d) ? plan_tc(d, 64, d.d_out, sms).ws_bytes : 0;
}

// With dot_out, the tensor-core path reduces every result row to the per-token
// dot_out[t] = dot_scale * (r_t . a_t) in its epilogue and stores no r (r may then be
// null); *fused tells whether it did (else r holds the read and no dot was formed).
int run_suffix_impl(const gradlev_desc* desc, const gradlev_tensor* q, const gradlev_tensor* k,
                    const gradlev_tensor* v, const gradlev_tensor* r, const Tok* dot_a,
                    float* dot_out, float dot_scale, bool* fused, void* ws, size_t ws_bytes,
                    cudaStream_t stream) {
    if (fused) *fused = false;
    if (!desc_ok(desc)) return GRADLEV_ERR_INVALID_ARG;
    const gradlev_desc& d = *desc;
    Tok tq, tk, tv, tr;
    if (!resolve(d, q, d.d_in, &tq, true) || !resolve(d, k, d.d_in, &tk, true) ||
        !resolve(d, v, d.d_out, &tv, true) || !resolve(d, r, d.d_out, &tr, dot_out == nullptr))
        return GRADLEV_ERR_INVALID_ARG;
    DevInfo dev;
    if (!device_info(&dev)) return GRADLEV_ERR_CUDA;
    if (!(dev.major == 10 && dev.minor == 3)) return GRADLEV_ERR_UNSUPPORTED;
    const size_t need = suffix_ws_bytes(d, dev.sms);
    if (ws_bytes < need || (need && (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0)))
        return GRADLEV_ERR_WORKSPACE;
    if (d.T == 0) return GRADLEV_OK;
    const int elem = d.dtype == GRADLEV_BF16 ? 2 : 4;
    const Tok* all[4] = {&tq, &tk, &tv, &tr};
    for (const Tok* t : all)
        if ((reinterpret_cast<uintptr_t>(t->data) % elem) != 0) return GRADLEV_ERR_UNSUPPORTED;
    // the dotted rows arrive through the output tensor map: no r is stored then
    const bool dot_ok = dot_out && dot_a && !tr.data && tc_layout_ok(*dot_a, 2);
    if (suffix_tc_shape(d) && tc_layout_ok(tq, 2) && tc_layout_ok(tk, 2) && tc_layout_ok(tv, 2) &&
        tc_layout_ok(tr, 2) && (dot_out == nullptr || dot_ok) && (tr.data || dot_ok)) {
        const Plan pl = plan_tc(d, 64, d.d_out, dev.sms);
        CUtensorMap mq, mk, mv, mo;
        if (!make_tmap(&mq, d, tq, 64) || !make_tmap(&mk, d, tk, 64) ||
            !make_tmap(&mv, d, tv, d.d_out) || !make_tmap(&mo, d, dot_ok ? *dot_a : tr, d.d_out))
            return GRADLEV_ERR_UNSUPPORTED;
        TcScanParams p;
        memset(&p, 0, sizeof(p));
        p.L = d.L;
        p.B = d.B;
        p.T = d.T;
        p.H = d.H;
        p.dq = 64;
        p.dv = d.d_out;
        p.n_tiles = pl.n_tiles;
        p.seg_len = pl.seg_len;
        p.n_seg = pl.n_seg;
        p.n_items = pl.n_items;
        p.n_ut = pl.n_items / pl.n_seg;
        p.lookback_limit_ns = 4000000000ull;
        p.test_skip_publish = -1;
        p.eta = -1.0f;  // + sum over the later tokens
        p.lam = 1.0f;
        p.inv_lam = 1.0f;
        p.mu = 1.0f;
        p.W0 = nullptr;  // the suffix read has no base matrix
        Tok none;
        fill_epi(&p.epi, tr, none, none, GRADLEV_ACT_NONE);
        if (dot_out) {
            p.epi.dot_a = dot_a->data;
            for (int i = 0; i < 4; ++i) p.epi.dot_a_str[i] = dot_a->s[i];
            p.epi.dot_out = dot_out;
            p.epi.dot_scale = dot_scale;
            // several 64-wide tiles add their partial dots
            if (pl.n_tiles > 1 &&
                cudaMemsetAsync(dot_out, 0, sizeof(float) * (size_t)d.L * d.B * d.T * d.H, stream) !=
                    cudaSuccess)
                return GRADLEV_ERR_CUDA;
            if (fused) *fused = true;
        }
        uint8_t* wsb = static_cast<uint8_t*>(ws);
        p.ctrl = reinterpret_cast<unsigned int*>(wsb);
        p.flags = reinterpret_cast<unsigned int*>(wsb + pl.off_flags);
        p.agg = reinterpret_cast<float*>(wsb + pl.off_agg);
        p.incl = reinterpret_cast<float*>(wsb + pl.off_incl);
        if (cudaMemsetAsync(ws, 0, pl.zero_bytes, stream) != cudaSuccess) return GRADLEV_ERR_CUDA;
        const int grid = pl.n_items < dev.sms ? pl.n_items : dev.sms;
        if (gl::launch_tc_suffix(mq, mk, mv, mo, p, same_tensor(tq, tk), grid, stream) != cudaSuccess)
            return GRADLEV_ERR_CUDA;
        return GRADLEV_OK;
    }
    if (!simt_shape_ok(d, d.d_in) || !tr.data) return GRADLEV_ERR_UNSUPPORTED;
    gl::SimtScanParams p;
    memset(&p, 0, sizeof(p));
    p.L = d.L;
    p.B = d.B;
    p.T = d.T;
    p.H = d.H;
    p.dq = d.d_in;
    p.dv = d.d_out;
    p.eta = -1.0f;
    p.W0 = nullptr;
    p.q = tq.data;
    p.k = tk.data;
    p.v = tv.data;
    for (int i = 0; i < 4; ++i) {
        p.q_str[i] = tq.s[i];
        p.k_str[i] = tk.s[i];
        p.v_str[i] = tv.s[i];
    }
    Tok none;
    fill_epi(&p.epi, tr, none, none, GRADLEV_ACT_NONE);
    if (gl::launch_simt_scan(p, d.dtype == GRADLEV_BF16, true, stream) != cudaSuccess)
        return GRADLEV_ERR_CUDA;
    return GRADLEV_OK;
}

// Step-size gradients of one map's read (read 0: forward y = W x; read 1: costate
// gin = W^T g_out): deta_s = -a_s . r_s, r the suffix read of the upstream gradient.
gradlev_desc suffix_desc(const gradlev_desc& d, int read) {
    gradlev_desc s = d;
    if (read == 1) {
        s.d_in = d.d_out;
        s.d_out = d.d_in;
    }
    return s;
}

size_t eta_grad_ws_bytes(const gradlev_desc& d, int read, int sms) {
    const gradlev_desc s = suffix_desc(d, read);
    const size_t elem = d.dtype == GRADLEV_BF16 ? 2 : 4;
    return round_up(suffix_ws_bytes(s, sms), 256) +
           round_up((size_t)d.L * d.B * d.T * d.H * s.d_out * elem, 256);
}

int run_eta_grad(const gradlev_desc* desc, int read, const gradlev_tensor* x,
                 const gradlev_tensor* g_hat, const gradlev_tensor* g_out,
                 const gradlev_tensor* upstream, float* deta, void* ws, size_t ws_bytes,
                 cudaStream_t stream) {
    if (!desc_ok(desc) || (read != 0 && read != 1) || (!deta && desc->T > 0) ||
        (reinterpret_cast<uintptr_t>(deta) & 3u))
        return GRADLEV_ERR_INVALID_ARG;
    const gradlev_desc& d = *desc;
    const gradlev_desc sd = suffix_desc(d, read);
    const int sms = dev_sms_or_default();
    if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0 ||
        ws_bytes < eta_grad_ws_bytes(d, read, sms))
        return GRADLEV_ERR_WORKSPACE;
    Tok tx, tg, tu;
    if (!resolve(d, x, d.d_in, &tx, true) || !resolve(d, g_hat, d.d_out, &tg, true) ||
        !resolve(d, upstream, read == 0 ? d.d_out : d.d_in, &tu, true))
        return GRADLEV_ERR_INVALID_ARG;
    if (read == 1 && (!g_out || (!g_out->data && d.T > 0))) return GRADLEV_ERR_INVALID_ARG;
    if (d.T == 0) return GRADLEV_OK;
    const size_t base = round_up(suffix_ws_bytes(sd, sms), 256);
    gradlev_tensor rt;
    rt.data = static_cast<uint8_t*>(ws) + base;
    for (int i = 0; i < 4; ++i) rt.stride[i] = 0;
    const Tok& ta = read == 0 ? tg : tx;
    // forward read: q = k = x, v = dL/dy;  costate read: q = ghat, k = g_out, v = dL/dgin.
    // The tensor-core path forms the dot in its epilogue; otherwise r goes through the
    // workspace and a row-dot kernel.
    bool fused = false;
    const int rc = read == 0 ? run_suffix_impl(&sd, x, x, upstream, nullptr, &ta, deta, -1.0f,
                                               &fused, ws, base, stream)
                             : run_suffix_impl(&sd, g_hat, g_out, upstream, nullptr, &ta, deta,
                                               -1.0f, &fused, ws, base, stream);
    if (rc == GRADLEV_OK && fused) return GRADLEV_OK;
    if (rc != GRADLEV_OK && rc != GRADLEV_ERR_UNSUPPORTED) return rc;
    const int rc2 = read == 0
                        ? run_suffix_impl(&sd, x, x, upstream, &rt, nullptr, nullptr, 0.f, nullptr,
                                          ws, base, stream)
                        : run_suffix_impl(&sd, g_hat, g_out, upstream, &rt, nullptr, nullptr, 0.f,
                                          nullptr, ws, base, stream);
    if (rc2 != GRADLEV_OK) return rc2;
    Tok trr;
    resolve(sd, &rt, sd.d_out, &trr, true);
    gl::TokStr as, rs;
    for (int i = 0; i < 4; ++i) {
        as.s[i] = ta.s[i];
        rs.s[i] = trr.s[i];
    }
    if (gl::launch_rowdot(ta.data, as, trr.data, rs, deta, d.L, d.B, d.T, d.H, sd.d_out, -1.0f,
                          d.dtype == GRADLEV_BF16, stream) != cudaSuccess)
        return GRADLEV_ERR_CUDA;
    return GRADLEV_OK;
}

// Gate derivatives of one map's read with per-token eta_t and retention alpha_t (Sec. 3,
// practical architecture and training), for 64 x 64 bf16 maps.  With D_t = W_t - W0
// and the read's upstream gradient u (read 0: y = W x, a = u, b = x; read 1:
// gin = W^T g_out, a = g_out, b = u):
//   dlog_alpha_j = alpha_j <D_j, R_j>,  deta_j = -ghat_j^T R_j x_j,
//   R_j = sum_{s>j} prod_{j<r<s} alpha_r a_s b_s^T.
// Three launches: per-chunk aggregates of the writes and of the pairs (a, b)
// (gate_agg_tc_kernel); D at every chunk start and R at every chunk end, carried over
// the chunks (gate_state_scan_kernel); the expansion inside each chunk of 128
// tokens (gate_chunk_tc_kernel).
size_t gate_grads_ws_bytes(const gradlev_desc& d, int /*sms*/) {
    const size_t units = (size_t)d.L * d.B * d.H;
    const size_t nch = ((size_t)d.T + 127) / 128;
    return 256 + 2 * round_up(units * nch * 64 * 64 * sizeof(float), 256) +
           round_up(units * nch * sizeof(float), 256);
}

int run_gate_grads(const gradlev_desc* desc, int read, const gradlev_tensor* x,
                   const gradlev_tensor* g_hat, const float* eta_t, const float* alpha_t,
                   const gradlev_tensor* g_out, const gradlev_tensor* upstream, float* dlog_alpha,
                   float* deta, void* ws, size_t ws_bytes, cudaStream_t stream) {
    if (!desc_ok(desc) || (read != 0 && read != 1)) return GRADLEV_ERR_INVALID_ARG;
    const gradlev_desc& d = *desc;
    if (d.T > 0 && (!eta_t || !dlog_alpha || !deta)) return GRADLEV_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(eta_t) | reinterpret_cast<uintptr_t>(alpha_t) |
         reinterpret_cast<uintptr_t>(dlog_alpha) | reinterpret_cast<uintptr_t>(deta)) & 3u)
        return GRADLEV_ERR_INVALID_ARG;
    if (d.dtype != GRADLEV_BF16 || d.d_in != 64 || d.d_out != 64) return GRADLEV_ERR_UNSUPPORTED;
    DevInfo dev;
    if (!device_info(&dev)) return GRADLEV_ERR_CUDA;
    if (!(dev.major == 10 && dev.minor == 3)) return GRADLEV_ERR_UNSUPPORTED;
    if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0 || ws_bytes < gate_grads_ws_bytes(d, dev.sms))
        return GRADLEV_ERR_WORKSPACE;
    Tok tx, tg, tu, tgo;
    if (!resolve(d, x, 64, &tx, true) || !resolve(d, g_hat, 64, &tg, true) ||
        !resolve(d, upstream, 64, &tu, true) || !resolve(d, g_out, 64, &tgo, read == 1))
        return GRADLEV_ERR_INVALID_ARG;
    if (d.T == 0) return GRADLEV_OK;
    const Tok* rows[4] = {&tx, &tg, &tu, &tgo};
    for (const Tok* t : rows)
        if (t->data && !tc_layout_ok(*t, 2)) return GRADLEV_ERR_UNSUPPORTED;
    const Tok& ta = read == 0 ? tu : tgo;
    const Tok& tb = read == 0 ? tx : tu;
    CUtensorMap mx, mg, ma, mb;
    if (!make_tmap(&mx, d, tx, 64) || !make_tmap(&mg, d, tg, 64) || !make_tmap(&ma, d, ta, 64) ||
        !make_tmap(&mb, d, tb, 64))
        return GRADLEV_ERR_UNSUPPORTED;
    const size_t units = (size_t)d.L * d.B * d.H;
    const int nch = (d.T + 127) / 128;
    const size_t st_bytes = units * (size_t)nch * 64 * 64 * sizeof(float);
    uint8_t* base = static_cast<uint8_t*>(ws);
    unsigned int* ctrl = reinterpret_cast<unsigned int*>(base);
    float* VS = reinterpret_cast<float*>(base + 256);
    float* UR = reinterpret_cast<float*>(base + 256 + round_up(st_bytes, 256));
    float* Ad = reinterpret_cast<float*>(base + 256 + 2 * round_up(st_bytes, 256));
    if (cudaMemsetAsync(ws, 0, 256, stream) != cudaSuccess) return GRADLEV_ERR_CUDA;
    if (gl::launch_gate_aggregates_tc(mx, mg, ma, mb, eta_t, alpha_t, VS, UR, Ad, d.L, d.B, d.T, d.H, ctrl + 1,
                                      stream) != cudaSuccess ||
        gl::launch_gate_state_scan(VS, UR, Ad, (long long)units, nch, stream) != cudaSuccess ||
        gl::launch_gate_chunks_tc(mx, mg, ma, mb, eta_t, alpha_t, VS, UR, dlog_alpha, deta, d.L, d.B, d.T, d.H,
                                  ctrl + 1, stream) != cudaSuccess)
        return GRADLEV_ERR_CUDA;
    return GRADLEV_OK;
}

// Deployment (decode) calls: one token per unit, Delta = W - W0 held by the caller.
constexpr long long kDecodeTileBytes = 64 << 10;  // bytes of Delta per CTA tile

struct DecodePlan {
    int lanes = 32, rows_read = 0, n_rt_read = 0, rows_write = 0, n_rt_write = 0, n_strips = 0;
    size_t off_cnt = 0, ws_bytes = 0;  // workspace of a write that returns g_in
};

// Tiles of about 64 KB of Delta: enough bytes in flight per CTA, and thousands of
// CTAs for the large maps.  Depends on the shape only, so the workspace size does too.
DecodePlan decode_plan(const gradlev_desc& d) {
    DecodePlan pl;
    const int cpr = d.d_in / 4;
    if (cpr < 32) {
        pl.lanes = 1;
        while (pl.lanes < cpr) pl.lanes <<= 1;
    }
    const int pass_rows = 8 * (32 / pl.lanes);  // rows the eight warps of a CTA cover at once
    const long long all_rows = (long long)(d.d_out + pass_rows - 1) / pass_rows * pass_rows;
    auto tile_rows = [&](long long row_bytes) {
        long long r = kDecodeTileBytes / row_bytes / pass_rows * pass_rows;
        if (r < pass_rows) r = pass_rows;
        return (int)(r < all_rows ? r : all_rows);
    };
    pl.rows_read = tile_rows(4ll * d.d_in);
    pl.n_rt_read = (d.d_out + pl.rows_read - 1) / pl.rows_read;
    pl.n_strips = (cpr + 31) / 32;
    pl.rows_write = tile_rows(cpr < 32 ? 4ll * d.d_in : 512ll);
    pl.n_rt_write = (d.d_out + pl.rows_write - 1) / pl.rows_write;
    if (pl.n_rt_write > 1) {
        const size_t units = (size_t)d.L * d.B * d.H;
        pl.off_cnt = round_up(units * pl.n_rt_write * (size_t)d.d_in * sizeof(float), 256);
        pl.ws_bytes = pl.off_cnt + round_up(units * pl.n_strips * sizeof(unsigned int), 256);
    }
    return pl;
}

// Checks shared by both decode calls.  The arguments the read or the write does
// not use are passed as NULL.
int decode_check(const gradlev_desc* desc, const float* delta, int act, DevInfo* dev) {
    if (!desc_ok(desc)) return GRADLEV_ERR_INVALID_ARG;
    const gradlev_desc& d = *desc;
    if (d.T != 1 || !delta) return GRADLEV_ERR_INVALID_ARG;
    if (act < GRADLEV_ACT_NONE || act > GRADLEV_ACT_TANH) return GRADLEV_ERR_INVALID_ARG;
    if (d.d_in % 4 != 0 || (long long)d.L * d.H > 65535 || !aligned16(delta))
        return GRADLEV_ERR_UNSUPPORTED;
    if (!device_info(dev)) return GRADLEV_ERR_CUDA;
    if (!(dev->major == 10 && dev->minor == 3)) return GRADLEV_ERR_UNSUPPORTED;
    return GRADLEV_OK;
}

void decode_common(gl::DecodeParams* p, const gradlev_desc& d, const DecodePlan& pl,
                   const float* W0, float* delta, const Tok& tx) {
    memset(p, 0, sizeof(*p));
    p->L = d.L;
    p->B = d.B;
    p->H = d.H;
    p->din = d.d_in;
    p->dout = d.d_out;
    p->cpr = d.d_in / 4;
    p->lanes = pl.lanes;
    p->n_strips = pl.n_strips;
    p->W0 = W0;
    p->delta = delta;
    p->x = tx.data;
    for (int i = 0; i < 4; ++i) p->x_s[i] = tx.s[i];
}

bool tok_elem_aligned(const Tok& t, int elem) {
    return !t.data || (reinterpret_cast<uintptr_t>(t.data) % elem) == 0;
}

int run_decode_read(const gradlev_desc* desc, const gradlev_tensor* x, const float* W0,
                    const float* delta, int act, const gradlev_tensor* y,
                    const gradlev_tensor* act_out, cudaStream_t stream) {
    DevInfo dev;
    const int rc = decode_check(desc, delta, act, &dev);
    if (rc != GRADLEV_OK) return rc;
    const gradlev_desc& d = *desc;
    if (!W0) return GRADLEV_ERR_INVALID_ARG;
    if (!aligned16(W0)) return GRADLEV_ERR_UNSUPPORTED;
    Tok tx, ty, ta, tz;
    if (!resolve(d, x, d.d_in, &tx, true) || !resolve(d, y, d.d_out, &ty, true) ||
        !resolve(d, act_out, d.d_out, &ta, false))
        return GRADLEV_ERR_INVALID_ARG;
    if (ta.data && act == GRADLEV_ACT_NONE) return GRADLEV_ERR_INVALID_ARG;
    const int elem = d.dtype == GRADLEV_BF16 ? 2 : 4;
    if (!tok_elem_aligned(tx, 4 * elem) || !tok_elem_aligned(ty, elem) ||
        !tok_elem_aligned(ta, elem))
        return GRADLEV_ERR_UNSUPPORTED;
    for (int i = 0; i < 4; ++i)  // x is read four elements at a time
        if (tx.s[i] % 4 != 0) return GRADLEV_ERR_UNSUPPORTED;
    const DecodePlan pl = decode_plan(d);
    gl::DecodeParams p;
    decode_common(&p, d, pl, W0, const_cast<float*>(delta), tx);
    p.rows = pl.rows_read;
    p.n_rt = pl.n_rt_read;
    fill_epi(&p.epi, ty, ta, tz, act);
    if (gl::launch_decode_read(p, d.dtype == GRADLEV_BF16, stream) != cudaSuccess)
        return GRADLEV_ERR_CUDA;
    return GRADLEV_OK;
}

int run_decode_write(const gradlev_desc* desc, const gradlev_tensor* x, const gradlev_tensor* g,
                     const float* W0, float* delta, const float* eta, const float* alpha, int act,
                     const gradlev_tensor* z, const gradlev_tensor* g_in, void* ws, size_t ws_bytes,
                     cudaStream_t stream) {
    DevInfo dev;
    const int rc = decode_check(desc, delta, act, &dev);
    if (rc != GRADLEV_OK) return rc;
    const gradlev_desc& d = *desc;
    if (!eta || (reinterpret_cast<uintptr_t>(eta) & 3u) ||
        (alpha && (reinterpret_cast<uintptr_t>(alpha) & 3u)))
        return GRADLEV_ERR_INVALID_ARG;
    Tok tx, tg, tgi, tz, none;
    if (!resolve(d, x, d.d_in, &tx, true) || !resolve(d, g, d.d_out, &tg, true) ||
        !resolve(d, g_in, d.d_in, &tgi, false) || !resolve(d, z, d.d_in, &tz, false))
        return GRADLEV_ERR_INVALID_ARG;
    const bool gin = tgi.data != nullptr;
    if (tz.data && (!gin || act == GRADLEV_ACT_NONE)) return GRADLEV_ERR_INVALID_ARG;
    if (gin && !W0) return GRADLEV_ERR_INVALID_ARG;
    if (gin && !aligned16(W0)) return GRADLEV_ERR_UNSUPPORTED;
    const int elem = d.dtype == GRADLEV_BF16 ? 2 : 4;
    if (!tok_elem_aligned(tx, elem) || !tok_elem_aligned(tg, elem) ||
        !tok_elem_aligned(tgi, elem) || !tok_elem_aligned(tz, elem))
        return GRADLEV_ERR_UNSUPPORTED;
    const DecodePlan pl = decode_plan(d);
    gl::DecodeParams p;
    decode_common(&p, d, pl, gin ? W0 : nullptr, delta, tx);
    p.rows = pl.rows_write;
    p.n_rt = pl.n_rt_write;
    p.g = tg.data;
    for (int i = 0; i < 4; ++i) p.g_s[i] = tg.s[i];
    p.eta = eta;
    p.alpha = alpha;
    fill_epi(&p.epi, tgi, none, tz, act);
    if (gin && pl.ws_bytes) {
        if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0 || ws_bytes < pl.ws_bytes)
            return GRADLEV_ERR_WORKSPACE;
        uint8_t* wsb = static_cast<uint8_t*>(ws);
        p.part = reinterpret_cast<float*>(wsb);
        p.cnt = reinterpret_cast<unsigned int*>(wsb + pl.off_cnt);
        if (cudaMemsetAsync(p.cnt, 0, pl.ws_bytes - pl.off_cnt, stream) != cudaSuccess)
            return GRADLEV_ERR_CUDA;
    }
    if (gl::launch_decode_write(p, d.dtype == GRADLEV_BF16, gin, stream) != cudaSuccess)
        return GRADLEV_ERR_CUDA;
    return GRADLEV_OK;
}

}  // namespace

namespace gl {
// Workspace bytes of the forward scan alone (gradlev_workspace_bytes covers both
// directions).  0 for an invalid descriptor.
size_t forward_workspace_bytes(const gradlev_desc* desc) {
    if (!desc_ok(desc)) return 0;
    DevInfo dev;
    const int sms = device_info(&dev) ? dev.sms : 160;
    return ws_bytes_for(*desc, desc->d_in, desc->d_out, sms);
}
}  // namespace gl

extern "C" {

int gradlev_forward_scan(const gradlev_desc* desc, const gradlev_tensor* x,
                         const gradlev_tensor* g_hat, const float* W0, float eta, int act,
                         const gradlev_tensor* y, const gradlev_tensor* act_out, void* workspace,
                         size_t workspace_bytes, gradlev_stream_t stream) {
    return run_scan(desc, false, x, g_hat, W0, eta, nullptr, act, y, act_out, nullptr, workspace,
                    workspace_bytes, reinterpret_cast<cudaStream_t>(stream));
}

int gradlev_costate_scan(const gradlev_desc* desc, const gradlev_tensor* x,
                         const gradlev_tensor* g_hat, const float* W0, float eta,
                         const gradlev_tensor* g_out, int act, const gradlev_tensor* z,
                         const gradlev_tensor* g_in, void* workspace, size_t workspace_bytes,
                         gradlev_stream_t stream) {
    return run_scan(desc, true, x, g_hat, W0, eta, g_out, act, g_in, nullptr, z, workspace,
                    workspace_bytes, reinterpret_cast<cudaStream_t>(stream));
}

int gradlev_fused_scan(const gradlev_desc* desc, const gradlev_tensor* x, const gradlev_tensor* g_hat,
                       const float* W0, float eta, const gradlev_tensor* g_out,
                       const gradlev_tensor* y, const gradlev_tensor* g_in,
                       const gradlev_tensor* cons_proposal, float* cons, void* workspace,
                       size_t workspace_bytes, gradlev_stream_t stream) {
    return run_fused(desc, x, g_hat, W0, eta, g_out, y, g_in, cons_proposal, cons, workspace,
                     workspace_bytes, reinterpret_cast<cudaStream_t>(stream));
}

int gradlev_forward_scan_gated(const gradlev_desc* desc, const gradlev_tensor* x,
                               const gradlev_tensor* g_hat, const float* W0, const float* eta_t,
                               const float* alpha_t, int act, const gradlev_tensor* y,
                               const gradlev_tensor* act_out, void* workspace,
                               size_t workspace_bytes, gradlev_stream_t stream) {
    return run_gated(desc, false, x, g_hat, W0, eta_t, alpha_t, nullptr, act, y, act_out, nullptr,
                     workspace, workspace_bytes, reinterpret_cast<cudaStream_t>(stream));
}

int gradlev_costate_scan_gated(const gradlev_desc* desc, const gradlev_tensor* x,
                               const gradlev_tensor* g_hat, const float* W0, const float* eta_t,
                               const float* alpha_t, const gradlev_tensor* g_out, int act,
                               const gradlev_tensor* z, const gradlev_tensor* g_in, void* workspace,
                               size_t workspace_bytes, gradlev_stream_t stream) {
    return run_gated(desc, true, x, g_hat, W0, eta_t, alpha_t, g_out, act, g_in, nullptr, z,
                     workspace, workspace_bytes, reinterpret_cast<cudaStream_t>(stream));
}

size_t gradlev_workspace_bytes_gated(const gradlev_desc* desc) {
    if (!desc_ok(desc)) return 0;
    DevInfo dev;
    int sms = device_info(&dev) ? dev.sms : 160;
    return gated_ws_bytes(*desc, sms);
}

int gradlev_suffix_scan(const gradlev_desc* desc, const gradlev_tensor* q,
                        const gradlev_tensor* k, const gradlev_tensor* v, const gradlev_tensor* r,
                        void* workspace, size_t workspace_bytes, gradlev_stream_t stream) {
    return run_suffix_impl(desc, q, k, v, r, nullptr, nullptr, 0.f, nullptr, workspace,
                           workspace_bytes, reinterpret_cast<cudaStream_t>(stream));
}

size_t gradlev_suffix_workspace_bytes(const gradlev_desc* desc) {
    if (!desc_ok(desc)) return 0;
    return suffix_ws_bytes(*desc, dev_sms_or_default());
}

int gradlev_eta_grad(const gradlev_desc* desc, int read, const gradlev_tensor* x,
                     const gradlev_tensor* g_hat, const gradlev_tensor* g_out,
                     const gradlev_tensor* upstream, float* deta, void* workspace,
                     size_t workspace_bytes, gradlev_stream_t stream) {
    return run_eta_grad(desc, read, x, g_hat, g_out, upstream, deta, workspace, workspace_bytes,
                        reinterpret_cast<cudaStream_t>(stream));
}

size_t gradlev_eta_grad_workspace_bytes(const gradlev_desc* desc, int read) {
    if (!desc_ok(desc) || (read != 0 && read != 1)) return 0;
    return eta_grad_ws_bytes(*desc, read, dev_sms_or_default());
}

int gradlev_gate_grads(const gradlev_desc* desc, int read, const gradlev_tensor* x,
                       const gradlev_tensor* g_hat, const float* eta_t, const float* alpha_t,
                       const gradlev_tensor* g_out, const gradlev_tensor* upstream, float* dlog_alpha,
                       float* deta, void* workspace, size_t workspace_bytes, gradlev_stream_t stream) {
    return run_gate_grads(desc, read, x, g_hat, eta_t, alpha_t, g_out, upstream, dlog_alpha, deta,
                          workspace, workspace_bytes, reinterpret_cast<cudaStream_t>(stream));
}

size_t gradlev_gate_grads_workspace_bytes(const gradlev_desc* desc, int read) {
    if (!desc_ok(desc) || (read != 0 && read != 1)) return 0;
    return gate_grads_ws_bytes(*desc, dev_sms_or_default());
}

int gradlev_decode_read(const gradlev_desc* desc, const gradlev_tensor* x, const float* W0,
                        const float* delta, int act, const gradlev_tensor* y,
                        const gradlev_tensor* act_out, gradlev_stream_t stream) {
    return run_decode_read(desc, x, W0, delta, act, y, act_out,
                           reinterpret_cast<cudaStream_t>(stream));
}

int gradlev_decode_write(const gradlev_desc* desc, const gradlev_tensor* x,
                         const gradlev_tensor* g, const float* W0, float* delta, const float* eta,
                         const float* alpha, int act, const gradlev_tensor* z,
                         const gradlev_tensor* g_in, void* workspace, size_t workspace_bytes,
                         gradlev_stream_t stream) {
    return run_decode_write(desc, x, g, W0, delta, eta, alpha, act, z, g_in, workspace,
                            workspace_bytes, reinterpret_cast<cudaStream_t>(stream));
}

size_t gradlev_decode_workspace_bytes(const gradlev_desc* desc) {
    if (!desc_ok(desc) || desc->T != 1 || desc->d_in % 4 != 0) return 0;
    return decode_plan(*desc).ws_bytes;
}

size_t gradlev_workspace_bytes(const gradlev_desc* desc) {
    if (!desc_ok(desc)) return 0;
    DevInfo dev;
    int sms = device_info(&dev) ? dev.sms : 160;
    size_t a = ws_bytes_for(*desc, desc->d_in, desc->d_out, sms);
    size_t b = ws_bytes_for(*desc, desc->d_out, desc->d_in, sms);
    return a > b ? a : b;
}

int gradlev_workspace_status(const void* workspace, gradlev_stream_t stream) {
    if (!workspace) return GRADLEV_ERR_INVALID_ARG;
    unsigned int word = 0;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (cudaStreamSynchronize(s) != cudaSuccess) return GRADLEV_ERR_CUDA;
    if (cudaMemcpy(&word, static_cast<const unsigned int*>(workspace) + 1, sizeof(word),
                   cudaMemcpyDeviceToHost) != cudaSuccess)
        return GRADLEV_ERR_CUDA;
    return word == 0 ? GRADLEV_OK : GRADLEV_ERR_TIMEOUT;
}

int gradlev_device_supported(void) {
    DevInfo dev;
    if (!device_info(&dev)) return 0;
    return (dev.major == 10 && dev.minor == 3) ? 1 : 0;
}

const char* gradlev_status_string(int code) {
    switch (code) {
    case GRADLEV_OK: return "ok";
    case GRADLEV_ERR_INVALID_ARG: return "invalid argument";
    case GRADLEV_ERR_UNSUPPORTED: return "unsupported shape, alignment, dtype or device";
    case GRADLEV_ERR_CUDA: return "CUDA runtime error";
    case GRADLEV_ERR_TIMEOUT: return "a bounded device-side wait expired";
    case GRADLEV_ERR_WORKSPACE: return "workspace missing, too small or misaligned";
    default: return "unknown status";
    }
}

int gradlev_abi_version(void) { return GRADLEV_ABI_VERSION; }

}  // extern "C"
