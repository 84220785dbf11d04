/*
 * gradlev.h -- C ABI of the GradLev token-scan library for GB300 (sm_103a).
 *
 * GradLev (Token-Parallel Test-Time Training via Costate Prediction) turns
 * token-by-token online gradient descent on a fast-weight matrix into two
 * associative scans once the per-token costates are supplied (Sec. 3, the
 * "Observation" paragraph).  With slow weights W0
 * (d_out x d_in), a step size eta and proposals ghat_t, the adapted weights
 * before token t are (Eq. 2 with unit retention, Eq. 3)
 *
 *     What_t = W0 + Deltahat_t,   Deltahat_t = -eta * sum_{s<t} ghat_s x_s^T,
 *
 * an EXCLUSIVE sum: every token reads the weights before its own write
 * (Sec. 3 step 2, "read before each write"; Deltahat_0 = 0).  The library
 * computes the two reads of those weights for every token in parallel:
 *
 *   forward scan  (Eq. 3):  y_t    = What_t x_t
 *                                   = W0 x_t - eta sum_{s<t} ghat_s (x_s . x_t)
 *   costate scan  (Eq. 4):  g_in_t = What_t^T g_out_t
 *                                   = W0^T g_out_t - eta sum_{s<t} x_s (ghat_s . g_out_t)
 *
 * (the transpose scan reuses the same historical writes (x_s, ghat_s),
 * queried by the incoming costate; Appendix C, eq. scan-reads).  An
 * elementwise activation can be fused on the outputs, for the two-layer
 * fast-weight MLP of Appendix A: the forward scan can also emit sigma(y_t),
 * and the costate scan can multiply its result by sigma'(z_t) (Sec. 3
 * step 3: g^z = sigma'(z) (.) g^x).
 *
 * Units.  A call covers L*B*H independent units (layer group l, batch row b,
 * head h).  Every unit starts with Deltahat = 0 at token 0 (a reset at the
 * start of each sequence) and has its own slow matrix W0[l][h]; batch rows
 * of one (l, h) share W0.
 *
 * Layouts.  Token tensors are 5-D [L][B][T][H][w] with w = d_in for x-like
 * tensors (x, g_in, z) and w = d_out for g-like tensors (ghat, g_out, y,
 * act_out).  The feature dimension is contiguous; the other four dimensions
 * use the element strides given in gradlev_tensor (all zero means the
 * contiguous default).  W0 is fp32 [L][H][d_out][d_in], contiguous.
 * All pointers are device pointers of the current CUDA device.
 *
 * Precision.  dtype GRADLEV_BF16: x, ghat, g_out and all outputs are bf16;
 * products run on the tensor cores with fp32 accumulation and an fp32 running
 * state; outputs are rounded to bf16 (round to nearest even).  dtype
 * GRADLEV_F32: everything is fp32 and computed with fp32 FMA.
 *
 * Ownership and concurrency.  The caller owns every buffer, including the
 * workspace.  Calls are asynchronous on the given stream, allocate nothing and
 * keep no state between calls.  A workspace must not be shared by calls that
 * may run concurrently.
 *
 * Errors.  Every entry point returns GRADLEV_OK (0) or a negative code; an
 * argument error is detected on the host before anything is launched, and
 * there is no CPU fallback.  A device-side wait that exceeds its time limit
 * (a defect, never expected) is reported through the workspace: see
 * gradlev_workspace_status.
 */
#ifndef GRADLEV_H
#define GRADLEV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define GRADLEV_ABI_VERSION 1

#define GRADLEV_OK 0
#define GRADLEV_ERR_INVALID_ARG (-1) /* null pointer, bad size or stride, non-finite eta */
#define GRADLEV_ERR_UNSUPPORTED (-2) /* shape, alignment, dtype or device not handled */
#define GRADLEV_ERR_CUDA (-3)        /* a CUDA runtime call or kernel launch failed */
#define GRADLEV_ERR_TIMEOUT (-4)     /* a bounded device-side wait expired */
#define GRADLEV_ERR_WORKSPACE (-5)   /* workspace missing, too small or misaligned */

typedef enum { GRADLEV_F32 = 0, GRADLEV_BF16 = 1 } gradlev_dtype;

/* Elementwise activations for the MLP fusion (App. A; App. E uses the tanh
 * approximation of GELU). */
typedef enum {
    GRADLEV_ACT_NONE = 0,
    GRADLEV_ACT_GELU_TANH = 1,
    GRADLEV_ACT_GELU_ERF = 2,
    GRADLEV_ACT_TANH = 3
} gradlev_act;

/* The same type as cudaStream_t; NULL is the legacy default stream. */
typedef struct CUstream_st* gradlev_stream_t;

/* Problem shape shared by both scans. */
typedef struct {
    int32_t L;      /* independent layer groups, each with its own W0 per head */
    int32_t B;      /* batch rows */
    int32_t T;      /* tokens per sequence (0 is allowed: nothing to do) */
    int32_t H;      /* heads */
    int32_t d_in;   /* width of x (input of the adapted map) */
    int32_t d_out;  /* width of y, ghat and g_out (output of the adapted map) */
    int32_t dtype;  /* gradlev_dtype of every token tensor */
    int32_t reserved; /* must be 0 */
} gradlev_desc;

/* A token tensor: device pointer plus element strides of (L, B, T, H).  The
 * feature dimension is contiguous.  stride all zero = contiguous default. */
typedef struct {
    void* data;
    int64_t stride[4];
} gradlev_tensor;

/*
 * gradlev_forward_scan -- forward exclusive prefix scan (Sec. 3 step 2, Eq. 3).
 *   x        [L][B][T][H][d_in]   layer inputs x_t (read)
 *   g_hat    [L][B][T][H][d_out]  costate proposals ghat_t: the writes (read)
 *   W0       [L][H][d_out][d_in]  fp32 slow weights (read)
 *   eta      step size of every write (finite; 0 gives y = W0 x).  On the tensor
 *            cores the running state is kept in units of -eta, so |eta| must lie
 *            in [2^-64, 2^64] there; any other finite eta runs on the CUDA-core
 *            kernel (exact fp32 FMA, slower), with the same results.
 *   act      activation applied for act_out (GRADLEV_ACT_NONE: act_out unused)
 *   y        [L][B][T][H][d_out]  out: y_t = What_t x_t (pre-activation)
 *   act_out  [L][B][T][H][d_out]  optional out (data NULL to skip): sigma(y_t)
 *   workspace/workspace_bytes  scratch of at least gradlev_workspace_bytes(desc)
 *            bytes, 256-byte aligned; its contents on entry are ignored.
 * Returns GRADLEV_OK or an error code; nothing is launched on error.
 */
int gradlev_forward_scan(const gradlev_desc* desc, const gradlev_tensor* x,
                         const gradlev_tensor* g_hat, const float* W0, float eta, int act,
                         const gradlev_tensor* y, const gradlev_tensor* act_out, void* workspace,
                         size_t workspace_bytes, gradlev_stream_t stream);

/*
 * gradlev_costate_scan -- costate (transpose) scan (Sec. 3 step 3, Eq. 4).
 *   x, g_hat, W0, eta  the same writes and slow weights as the forward scan
 *   g_out    [L][B][T][H][d_out]  incoming costates gtilde_t = dl_t/dy_t (read)
 *   act, z   optional fusion: with z.data non-NULL and act != NONE the output is
 *            sigma'(z_t) (.) (What_t^T g_out_t), z of shape [L][B][T][H][d_in]
 *            (the preactivation whose activation fed this map's input)
 *   g_in     [L][B][T][H][d_in]   out: What_t^T g_out_t (times sigma'(z_t) if fused)
 *   workspace/workspace_bytes  as for the forward scan.
 */
int gradlev_costate_scan(const gradlev_desc* desc, const gradlev_tensor* x,
                         const gradlev_tensor* g_hat, const float* W0, float eta,
                         const gradlev_tensor* g_out, int act, const gradlev_tensor* z,
                         const gradlev_tensor* g_in, void* workspace, size_t workspace_bytes,
                         gradlev_stream_t stream);

/*
 * gradlev_fused_scan -- the forward scan and the costate scan of one map in a single
 * call (Sec. 3, steps 2 and 3: both reads use the same historical writes), with the
 * optional per-token consistency term of the training objective (Eq. 5; Appendix A,
 * eq. consistency).
 *   x, g_hat, W0, eta  the writes and slow weights, as in gradlev_forward_scan
 *   g_out    [L][B][T][H][d_out]  incoming costates (read)
 *   y        [L][B][T][H][d_out]  out: What_t x_t          (as gradlev_forward_scan)
 *   g_in     [L][B][T][H][d_in]   out: What_t^T g_out_t    (as gradlev_costate_scan)
 *   cons_proposal  [L][B][T][H][d_in], optional (NULL or data NULL): proposals to
 *            compare with g_in, e.g. the proposals of the map below this one
 *   cons     fp32 [L][B][T][H] contiguous, 4-byte aligned; out when cons_proposal is
 *            given (and must then be non-NULL, else NULL):
 *            cons_t = ||cons_proposal_t - g_in_t||^2 / d_in, with g_in_t taken in fp32
 *            before its rounding to the output dtype
 *   workspace/workspace_bytes  at least gradlev_workspace_bytes(desc), 256-byte aligned.
 * bf16 maps with d_in = d_out = 64 and 16-byte aligned token rows (eta as for the
 * tensor-core forward scan) run one tensor-core kernel that reads x, g_hat and g_out
 * once and keeps one running state for both reads.  Every other shape runs the forward
 * and the costate scan one after the other, then (with cons) one row-reduction kernel;
 * the results are the same.  All arguments of both passes are checked before anything
 * is launched.  A timed-out device wait is reported by gradlev_workspace_status.
 * Returns GRADLEV_OK or an error code; nothing is launched on error.
 */
int gradlev_fused_scan(const gradlev_desc* desc, const gradlev_tensor* x,
                       const gradlev_tensor* g_hat, const float* W0, float eta,
                       const gradlev_tensor* g_out, const gradlev_tensor* y,
                       const gradlev_tensor* g_in, const gradlev_tensor* cons_proposal, float* cons,
                       void* workspace, size_t workspace_bytes, gradlev_stream_t stream);

/*
 * gradlev_forward_scan_gated / gradlev_costate_scan_gated -- the scans with the
 * general gates of Sec. 3 ("Observation", Eq. 2): a step size eta_t >= 0 per token
 * and, optionally, a retention alpha_t in [0, 1] with decay centred at W0,
 *     W_{t+1} = W0 + alpha_t (W_t - W0) - eta_t ghat_t x_t^T,   read before write.
 * alpha_t = 0 resets the fast weights to W0 (a document boundary).
 *   eta_t    fp32 [L][B][T][H], contiguous device array (read)
 *   alpha_t  fp32 [L][B][T][H], contiguous, or NULL for alpha = 1 (read)
 *   other arguments as in gradlev_forward_scan / gradlev_costate_scan (the scalar
 *   eta is replaced by eta_t).
 * Without alpha_t the proposals are scaled by eta_t into the workspace (one
 * elementwise pass, rounded to the input dtype) and the chunked scan runs with
 * eta = 1.  With alpha_t:
 *   - bf16 64 x 64 maps whose tensors a TMA map can describe (16-byte aligned
 *     rows and strides) run in chunks of 128 tokens on the tensor cores, with the
 *     decays formed as products of the alphas (exact zeros at resets; any real
 *     alpha_t is accepted); fewer than two units per SM over more than 1024 tokens
 *     are cut into segments whose states are carried (an aggregate pass first);
 *   - every other shape runs the recurrence token by token, the state W - W0 in
 *     fp32.  The read width (d_in forward, d_out costate) must be at most 256,
 *     else GRADLEV_ERR_UNSUPPORTED.
 * Workspace: at least gradlev_workspace_bytes_gated(desc) bytes, 256-byte aligned.
 */
int gradlev_forward_scan_gated(const gradlev_desc* desc, const gradlev_tensor* x,
                               const gradlev_tensor* g_hat, const float* W0, const float* eta_t,
                               const float* alpha_t, int act, const gradlev_tensor* y,
                               const gradlev_tensor* act_out, void* workspace,
                               size_t workspace_bytes, gradlev_stream_t stream);
int gradlev_costate_scan_gated(const gradlev_desc* desc, const gradlev_tensor* x,
                               const gradlev_tensor* g_hat, const float* W0, const float* eta_t,
                               const float* alpha_t, const gradlev_tensor* g_out, int act,
                               const gradlev_tensor* z, const gradlev_tensor* g_in, void* workspace,
                               size_t workspace_bytes, gradlev_stream_t stream);

/*
 * gradlev_document_gates -- gate arrays for sequences packed from several
 * documents.  A read sees only the writes of its own document, those since the
 * latest document start (Appendix C, scan reads; Appendix E, packed rows).  In
 * the gates of Eq. 2 a document starting at token s > 0 is alpha = 0 and eta = 0
 * at token s - 1:
 * the fast weights return to W0 and the previous document's last write (seen by
 * none of its reads) is dropped, so the read at s sees W0.  The outputs feed
 * gradlev_forward_scan_gated / gradlev_costate_scan_gated.
 *   desc       only L, B, T, H (and reserved = 0) are read
 *   doc_start  uint8 [B][T], contiguous device array, nonzero where a document
 *              begins; entry t = 0 is ignored (every row begins one).  The same
 *              documents hold for every layer and head.
 *   eta        step size of every write where eta_t is NULL (finite)
 *   eta_t      fp32 [L][B][T][H] contiguous per-token step sizes, or NULL
 *   alpha_t    fp32 [L][B][T][H] contiguous retention, or NULL for alpha = 1
 *   eta_out, alpha_out  fp32 [L][B][T][H] contiguous device outputs (written);
 *              eta_out may be eta_t and alpha_out may be alpha_t (in place)
 * Returns GRADLEV_OK (nothing to do when L*B*T*H = 0), GRADLEV_ERR_INVALID_ARG
 * for a null pointer, a non-finite eta or an fp32 array not 4-byte aligned, and
 * GRADLEV_ERR_CUDA if the launch fails.  Asynchronous on `stream`.
 */
int gradlev_document_gates(const gradlev_desc* desc, const uint8_t* doc_start, float eta,
                           const float* eta_t, const float* alpha_t, float* eta_out,
                           float* alpha_out, gradlev_stream_t stream);

/* Bytes of workspace the gated scans need for this shape (0 for an invalid
 * descriptor). */
size_t gradlev_workspace_bytes_gated(const gradlev_desc* desc);

/*
 * Deployment (decode) -- Sec. 3, training-objective paragraph, and Appendix A:
 * once deployed, the proposal network is gone and each adapted map updates from
 * its own costates after the target has been scored, one token at a time.  The
 * caller keeps each unit's fast weights as Delta = W - W0 (fp32
 * [L][B][H][d_out][d_in], contiguous, 16-byte aligned; all zero at the start of a
 * sequence) and calls, per token,
 *   gradlev_decode_read   y     = (W0 + Delta) x             (the read before the write)
 *   ... the model scores the target and back-propagates its true costate g ...
 *   gradlev_decode_write  g_in  = (W0 + Delta)^T g           (optional, pre-write weights)
 *                         Delta <- alpha Delta - eta g x^T   (Eq. 2, decay centred at W0)
 * The descriptor has T = 1: token tensors are [L][B][1][H][w] with the usual
 * strides.  d_in must be a multiple of 4 (GRADLEV_ERR_UNSUPPORTED otherwise), and
 * L*H at most 65535.  dtype as for the scans; Delta, W0 and every sum stay fp32.
 * Reads and writes of one Delta must be issued in order on one stream; both
 * calls are asynchronous and keep no state of their own.
 */

/*
 * gradlev_decode_read -- y = (W0 + Delta) x for one token per unit.
 *   x        [L][B][1][H][d_in]   (read)
 *   W0       fp32 [L][H][d_out][d_in], 16-byte aligned (read)
 *   delta    fp32 [L][B][H][d_out][d_in] (read)
 *   act, act_out  optional sigma(y) (act_out.data NULL to skip), as for the forward scan
 *   y        [L][B][1][H][d_out]  (out)
 * x is read four elements at a time: its base must be aligned to four elements
 * and its strides multiples of four (GRADLEV_ERR_UNSUPPORTED otherwise).
 */
int gradlev_decode_read(const gradlev_desc* desc, const gradlev_tensor* x, const float* W0,
                        const float* delta, int act, const gradlev_tensor* y,
                        const gradlev_tensor* act_out, gradlev_stream_t stream);

/*
 * gradlev_decode_write -- the write of one token per unit, with its costate read.
 *   x        [L][B][1][H][d_in]   the token's input (read)
 *   g        [L][B][1][H][d_out]  the true costate dl/dy of the scored token (read)
 *   W0       fp32 slow weights; needed only when g_in is requested (else may be NULL)
 *   delta    fp32 [L][B][H][d_out][d_in] (read and updated in place)
 *   eta      fp32 [L][B][H] step size per unit (read)
 *   alpha    fp32 [L][B][H] retention per unit, or NULL for 1; 0 resets Delta to zero
 *   g_in     optional [L][B][1][H][d_in] (data NULL to skip): (W0 + Delta)^T g with the
 *            weights BEFORE this write (Sec. 3 step 3 holds them fixed), times
 *            sigma'(z) when z is given with act != NONE (z of shape [L][B][1][H][d_in])
 *   workspace/workspace_bytes  at least gradlev_decode_workspace_bytes(desc) bytes,
 *            256-byte aligned, when g_in is requested (NULL if that is 0)
 * The column sums of g_in are combined in a fixed order: results are reproducible.
 */
int gradlev_decode_write(const gradlev_desc* desc, const gradlev_tensor* x,
                         const gradlev_tensor* g, const float* W0, float* delta, const float* eta,
                         const float* alpha, int act, const gradlev_tensor* z,
                         const gradlev_tensor* g_in, void* workspace, size_t workspace_bytes,
                         gradlev_stream_t stream);

/* Workspace bytes of a gradlev_decode_write that returns g_in (0: none needed, or
 * an invalid descriptor). */
size_t gradlev_decode_workspace_bytes(const gradlev_desc* desc);

/*
 * Outer gradients through the reads -- Sec. 3, practical architecture and
 * training: the gates are learned and their derivatives kept, while the writes
 * are detached.  The reads are then linear in every step size, and the derivative
 * with respect to eta_s is a read of the same writes in the other direction of time.
 *
 * gradlev_suffix_scan -- the anti-causal read
 *     r_s = sum_{t>s} (k_t . q_s) v_t          (r_{T-1} = 0)
 *   desc     d_in = width of q and k, d_out = width of v and r; T, strides and dtype
 *            as for the scans
 *   q, k     [L][B][T][H][d_in] (read);  v [L][B][T][H][d_out] (read)
 *   r        [L][B][T][H][d_out] (out)
 *   workspace/workspace_bytes  at least gradlev_suffix_workspace_bytes(desc) bytes
 *            (NULL if that is 0)
 * d_in at most 256 (GRADLEV_ERR_UNSUPPORTED otherwise).
 */
int gradlev_suffix_scan(const gradlev_desc* desc, const gradlev_tensor* q,
                        const gradlev_tensor* k, const gradlev_tensor* v, const gradlev_tensor* r,
                        void* workspace, size_t workspace_bytes, gradlev_stream_t stream);
size_t gradlev_suffix_workspace_bytes(const gradlev_desc* desc);

/*
 * gradlev_eta_grad -- dL/deta_s of one adapted map's read, for per-token step sizes
 * (unit retention):
 *   read 0 (forward, y_t = W_t x_t):        deta_s = -ghat_s . sum_{t>s} (x_t . x_s) u_t,
 *            u = dL/dy [L][B][T][H][d_out]
 *   read 1 (costate, gin_t = W_t^T g_out_t): deta_s = -x_s . sum_{t>s} (g_out_t . ghat_s) u_t,
 *            u = dL/dgin [L][B][T][H][d_in]; g_out required
 *   x, g_hat, g_out  the map's tensors as for the scans (read)
 *   deta     fp32 [L][B][T][H], contiguous (out)
 *   workspace/workspace_bytes  at least gradlev_eta_grad_workspace_bytes(desc, read)
 *            bytes, 256-byte aligned (it holds the suffix read)
 * The same value for every eta_t: the reads are linear in the step sizes.
 * With bf16 tensors and 64-wide q and k (d_in for read 0, d_out for read 1) the dot
 * is formed inside the tensor-core kernel; when the dotted width exceeds 128, its
 * 64-wide tiles add their dots atomically and the last bit may differ between runs.
 * Other shapes and fp32 go through the workspace and a row-dot kernel.
 */
int gradlev_eta_grad(const gradlev_desc* desc, int read, const gradlev_tensor* x,
                     const gradlev_tensor* g_hat, const gradlev_tensor* g_out,
                     const gradlev_tensor* upstream, float* deta, void* workspace,
                     size_t workspace_bytes, gradlev_stream_t stream);
size_t gradlev_eta_grad_workspace_bytes(const gradlev_desc* desc, int read);

/*
 * gradlev_gate_grads -- derivatives of one adapted map's read with respect to its
 * per-token gates, eta_t and retention alpha_t (Sec. 3, practical architecture and
 * training: the gates are learned and their derivatives kept, the writes detached;
 * Eq. 2 with decay centred at W0).  With D_t = W_t - W0 and u the read's upstream
 * gradient, a write i and a later read s > i contribute
 *     c_is = -eta_i (prod_{i<r<s} alpha_r) (u_s . ghat_i)(x_i . x_s)         (read 0)
 *     c_is = -eta_i (prod_{i<r<s} alpha_r) (g_out_s . ghat_i)(u_s . x_i)     (read 1)
 * and the outputs are
 *     deta_i       = dL/deta_i = sum_{s>i} c_is / eta_i
 *     dlog_alpha_j = alpha_j dL/dalpha_j = sum_{i<j<s} c_is = <D_j, R_j> alpha_j,
 * the derivative in log alpha_j (for alpha_t = sigmoid(a_t), dL/da_t =
 * (1 - alpha_t) dlog_alpha_t; no division, so a reset alpha_t = 0 is allowed).
 *   read 0 (forward, y = W x): u = dL/dy [L][B][T][H][d_out]; read 1 (costate,
 *            gin = W^T g_out): u = dL/dgin [L][B][T][H][d_in], g_out required
 *   x, g_hat, g_out  the map's tensors as for the scans (read); token rows 16-byte
 *            aligned with 16-byte strides, else GRADLEV_ERR_UNSUPPORTED
 *   eta_t    fp32 [L][B][T][H] contiguous (read); alpha_t the same or NULL (= 1)
 *   dlog_alpha, deta  fp32 [L][B][T][H], contiguous (written)
 *   workspace/workspace_bytes  at least gradlev_gate_grads_workspace_bytes(desc, read),
 *            256-byte aligned
 * W0 does not enter.  Only bf16 maps of 64 x 64 (else GRADLEV_ERR_UNSUPPORTED).
 * Per chunk of 128 tokens: aggregates of the writes and of the pairs (a, b) on the
 * tensor cores; D at every chunk start and R at every chunk end carried over the
 * chunks in fp32; then the exact expansion of alpha_j <D_j, R_j> and
 * -ghat_j^T R_j x_j inside each chunk (four local terms, no cancellation).  A
 * timed-out device wait is reported by gradlev_workspace_status(workspace).
 * Asynchronous on `stream`.
 */
int gradlev_gate_grads(const gradlev_desc* desc, int read, const gradlev_tensor* x,
                       const gradlev_tensor* g_hat, const float* eta_t, const float* alpha_t,
                       const gradlev_tensor* g_out, const gradlev_tensor* upstream, float* dlog_alpha,
                       float* deta, void* workspace, size_t workspace_bytes, gradlev_stream_t stream);
size_t gradlev_gate_grads_workspace_bytes(const gradlev_desc* desc, int read);

/* Size of the fixed device array used by gradlev_forward_scan_noalloc (4 MiB). */
#define GRADLEV_NOALLOC_SCRATCH_BYTES (4u << 20)

/*
 * gradlev_forward_scan_noalloc -- the forward scan without a caller workspace.
 * (The paper has no counterpart: this is a calling convention of this library.)
 *
 * For callers that cannot allocate device memory when they call and have no
 * workspace to pass, such as a plugin behind a fixed "inputs, outputs, stream"
 * signature, or a serving loop whose device memory is budgeted once at start-up.
 * Arguments and results are those of gradlev_forward_scan; the scratch
 * the kernel needs lives in a GRADLEV_NOALLOC_SCRATCH_BYTES array inside the
 * library, which every GPU that loads the library holds until the process
 * exits.  The call allocates nothing.
 *   - A shape whose scratch would exceed that array returns
 *     GRADLEV_ERR_WORKSPACE (gradlev_workspace_bytes(desc) tells the need);
 *     nothing is launched.  Long sequences over few units need the most.
 *   - The first call on each device looks up the array's device address with
 *     that device current; make that first call before any stream capture.
 *   - All calls on a device share the array and it keeps the last call's
 *     contents; each call clears what must start at zero on its own stream.
 *     Calls that may overlap on the GPU race on it and must not be issued.
 *   - The size check is against the forward scan's own scratch need.
 *   - A timed-out device wait is reported by
 *     gradlev_forward_scan_noalloc_status, not gradlev_workspace_status (there
 *     is no caller workspace).
 *   - The looked-up address is cached per device for the life of the process;
 *     do not use this entry point on a device after cudaDeviceReset.
 */
int gradlev_forward_scan_noalloc(const gradlev_desc* desc, const gradlev_tensor* x,
                                 const gradlev_tensor* g_hat, const float* W0, float eta, int act,
                                 const gradlev_tensor* y, const gradlev_tensor* act_out,
                                 gradlev_stream_t stream);

/* Waits for `stream`, then reads the status word that the last
 * gradlev_forward_scan_noalloc on the current device left in the library's
 * array: GRADLEV_OK, GRADLEV_ERR_TIMEOUT if a bounded device wait expired (that
 * call's outputs are then undefined), or GRADLEV_ERR_CUDA.  Allocates nothing. */
int gradlev_forward_scan_noalloc_status(gradlev_stream_t stream);

/* Bytes of workspace either scan needs for this shape (the same bound serves
 * both).  Returns 0 for an invalid descriptor. */
size_t gradlev_workspace_bytes(const gradlev_desc* desc);

/* Waits for `stream`, then reads the device-side status word a scan left in
 * `workspace`: GRADLEV_OK, or GRADLEV_ERR_TIMEOUT if a bounded device wait
 * expired (the outputs of that call are then undefined), or GRADLEV_ERR_CUDA. */
int gradlev_workspace_status(const void* workspace, gradlev_stream_t stream);

/* 1 if the current device can run this library (compute capability 10.3), else 0. */
int gradlev_device_supported(void);

/* Human-readable text for a status code (static storage). */
const char* gradlev_status_string(int code);

/* GRADLEV_ABI_VERSION of the loaded library. */
int gradlev_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* GRADLEV_H */
