/*
 * mone.h -- C ABI of the MoNe test-time-learning library (libmone.so).
 *
 * MoNe ("Modular Neural Memory") attaches a fast-weight memory network to every
 * layer of a frozen Transformer.  A context of N tokens is consumed in segments
 * of T tokens (Sec. 3.1); on each segment every layer's memory takes one
 * gradient step on a layer-local loss (Eq. 7-8, Sec. 3.4), so the state chains
 * W_0 -> W_1 -> ... -> W_S (Eq. 9) independently per layer (Eq. 11) and per
 * context.  At inference the final state turns query hidden states into memory
 * keys and values (Eq. 4-5).
 *
 * This library implements that hot path on one GPU.  The backbone is not part
 * of it: the caller hands in per-layer activations X and target keys/values K, V
 * (Eq. 6 outputs), already in the backbone's dtype.
 *
 * Memory network (the two-matrix form of Eq. 3):
 *     M(u; W1, W2) = SiLU(u W1^T) W2,   W1: [d_hid x d_in], W2: [d_hid x d_out]
 * rows of W1 and W2 are hidden units ("channels"); d_out = 2*n_kv_heads*head_dim
 * and the output is [K || V] (K heads first, then V heads).
 *
 * Conventions
 *   - A "chain" is one (context, layer) pair: chain = ctx * n_layers + layer.
 *     Multi-chain arrays are laid out [n_ctx][n_layers][...] row-major.
 *   - Every data pointer is a DEVICE pointer owned by the caller unless stated;
 *     the library owns only the state it allocates in mone_mem_init.
 *   - Calls are asynchronous and ordered on the CUDA stream passed in
 *     (a cudaStream_t cast to void*; NULL = legacy default stream).
 *   - Argument errors are returned synchronously and nothing is launched.
 *     Errors found on the device (a bounded wait that gave up, a non-finite
 *     weight, a failed index check of a MONE_DEBUG build) are latched in a device
 *     status word; mone_mem_sync returns them.
 *   - There is no CPU fallback: without a usable sm_103a GPU, init fails with
 *     MONE_ERR_CUDA.
 */
#ifndef MONE_H_
#define MONE_H_

#ifdef __cplusplus
extern "C" {
#endif

#define MONE_ABI_VERSION 7

typedef struct mone_mem mone_mem; /* opaque; created by mone_mem_init */

typedef enum {
    MONE_OK = 0,
    MONE_ERR_INVALID_ARG = 1,       /* null/misaligned pointer, bad index or count, freed handle */
    MONE_ERR_UNSUPPORTED_SHAPE = 2, /* widths or segment size outside what the kernels tile */
    MONE_ERR_OOM = 3,               /* device allocation failed */
    MONE_ERR_CUDA = 4,              /* a CUDA call failed (no device, launch failure, ...) */
    MONE_ERR_TIMEOUT = 5,           /* a bounded device-side wait gave up (latched) */
    MONE_ERR_NONFINITE = 6,         /* an updated fast weight was NaN/Inf (latched) */
    MONE_ERR_UNSUPPORTED = 7,       /* valid request this build does not implement */
    MONE_ERR_CHECK = 8              /* a device-side index check failed (MONE_DEBUG builds; latched) */
} mone_status;

enum { MONE_FP32 = 0, MONE_BF16 = 1 };  /* dtype of X, K, V, Xq and generated K/V */
enum { MONE_PLAIN = 0, MONE_PAPER = 1 };
enum { MONE_LOSS_DOT = 0, MONE_LOSS_MSE = 1 };  /* per-token loss of a segment step */
enum { MONE_MEM_MLP = 0, MONE_MEM_SWIGLU = 1 };  /* form of the memory network M */
enum { MONE_RENORM_ROWS = 0, MONE_RENORM_OUT = 1 };  /* channels of the App. A renormalisation */
enum { MONE_GATE_LINEAR = 0, MONE_GATE_SILU = 1 };   /* how the read's per-head gate scales a head */

/*
 * Configuration, fixed for the life of a handle.
 *
 * mode MONE_PLAIN: u_j = x_j, constant learning rate lr (or per-token rates the
 *     caller passes to mone_ttl_segment), no momentum, no renormalisation.
 * mode MONE_PAPER (App. A): u_j = SiLU(alpha*x_j + gamma) / |.|  (affine
 *     rescale, SiLU, per-token L2 norm); per-token rate
 *     eta_j = softplus(w_eta . x_j + b_eta); momentum
 *     mu_s = beta_s mu_{s-1} + g_s with beta_s = sigmoid(w_beta . mean_j x_j + b_beta);
 *     W_s = W_{s-1} - mu_s (Eq. 8); then every row of W1 and of W2 is rescaled to
 *     its L2 norm in W_0 ("channel-wise L2 renormalisation").
 * The gradient step on a segment of T' tokens is g = sum_j (eta_j / T') grad l_j
 * with l_j = -y_j . M(u_j) (loss MONE_LOSS_DOT: Eq. 7, Eq. 10).  loss MONE_LOSS_MSE
 * replaces l_j by 1/2 |M(u_j) - y_j|^2 (the squared-error, delta-rule form of the
 * same step; its gradient needs M(u_j) at the segment's starting weights, computed
 * by two more kernels per segment, tcgen05 on BF16, CUDA cores on FP32).  MONE_LOSS_MSE
 * is supported for the MLP memory on both paths.
 *
 * memory MONE_MEM_MLP: M(u) = SiLU(u W1^T) W2, W1 [d_hid][d_in], W2 [d_hid][d_out] per chain.
 * memory MONE_MEM_SWIGLU (Eq. 3 itself): u splits into mem_heads heads of width dh = d_in / mem_heads;
 *     head h: O_h = (SiLU(u_h Win^T) * (u_h Wg^T)) Wout with Win, Wg, Wout [d_hid][dh] (d_hid = hidden
 *     units per head), O = [O_0 || ... ]; d_out == d_in.  Per chain W1 = [Win; Wg] for each head
 *     ([mem_heads][2 d_hid][dh]) and W2 = Wout ([mem_heads][d_hid][dh]).  BF16 only, loss DOT only;
 *     dh and d_hid multiples of 32 and <= 256, (d_out / 2) a multiple of dh, seg_T a multiple of 128.
 *
 * renorm_axis (paper mode; App. A's "channel-wise" renormalisation): MONE_RENORM_ROWS rescales
 *     every row (hidden unit) of W1 and of W2 to its norm in W_0; MONE_RENORM_OUT takes the
 *     channels to be each matrix's output channels: rows of W1 and columns of W2 (every column
 *     of W2 rescaled to its norm in W_0, by a column pass after each segment's update).  MLP
 *     memory only (SwiGLU: MONE_ERR_UNSUPPORTED).  Ignored in MONE_PLAIN mode.
 * gate_act (the read, App. A's "SiLU-gated" output): MONE_GATE_LINEAR scales head h by its
 *     learned scalar gate g_h; MONE_GATE_SILU by SiLU(g_h).
 *
 * Supported shapes: FP32: d_in, d_hid, d_out multiples of 64, seg_T multiple of 64.
 *   BF16 (MLP): d_in, d_out/2, seg_T multiples of 128; d_hid a multiple of 256.  Both: head_dim in {64,128},
 *   d_out == 2*n_kv_heads*head_dim, seg_T <= 4096.
 */
typedef struct {
    int n_ctx, n_layers;
    int d_in, d_hid, d_out;
    int n_kv_heads, head_dim;
    int seg_T;
    int dtype;     /* MONE_FP32 | MONE_BF16; fast-weight masters are always fp32 */
    int mode;      /* MONE_PLAIN | MONE_PAPER */
    float lr;      /* plain-mode learning rate */
    float rms_eps; /* epsilon of the read-side RMSNorm (Sec. 3.2 after Eq. 4); e.g. 1e-6 */
    int loss;      /* MONE_LOSS_DOT (Eq. 7) | MONE_LOSS_MSE */
    int memory;    /* MONE_MEM_MLP | MONE_MEM_SWIGLU */
    int mem_heads; /* SwiGLU heads (ignored for the MLP; 0 reads as 1) */
    int renorm_axis; /* MONE_RENORM_ROWS | MONE_RENORM_OUT */
    int gate_act;    /* MONE_GATE_LINEAR | MONE_GATE_SILU */
} mone_config;

/*
 * Per-chain meta-parameters (Sec. 3.3: trained offline, frozen at test time).
 * Device fp32 arrays: alpha, gamma, w_eta, w_beta are [chains][d_in]; b_eta,
 * b_beta are [chains]; gate is [chains][2*n_kv_heads] (one scalar gate per
 * output head, K heads then V heads).  Copied at init; the caller may free them
 * afterwards.  In MONE_PLAIN mode only gate is read (NULL = all gates 1).
 */
typedef struct {
    const float *alpha, *gamma, *w_eta, *b_eta, *w_beta, *b_beta, *gate;
} mone_meta;

/*
 * Allocate the fast-weight state of every chain and set it to W_0.
 * W1_0: [chains][d_hid][d_in] fp32, W2_0: [chains][d_hid][d_out] fp32 (device;
 * copied); for MONE_MEM_SWIGLU W1_0 is [chains][mem_heads][2 d_hid][dh] ([Win; Wg]
 * per head) and W2_0 [chains][mem_heads][d_hid][dh] (Wout); mone_mem_read_state /
 * mone_mem_write_state use the same layouts.  Momentum starts at 0; renormalisation targets are the row norms of
 * W_0.  meta may be NULL in MONE_PLAIN mode.  On success *out owns the state.
 * Errors: INVALID_ARG, UNSUPPORTED_SHAPE, OOM, CUDA.
 */
mone_status mone_mem_init(const mone_config* cfg, const float* W1_0, const float* W2_0,
                          const mone_meta* meta, void* stream, mone_mem** out);

/*
 * One TTL step (Eq. 7-8) of ONE chain on one segment of n_tok <= seg_T tokens.
 * X: [n_tok][d_in], K, V: [n_tok][d_out/2], dtype cfg->dtype, rows contiguous,
 * 16-byte aligned.  eta: optional device fp32 [n_tok] per-token learning rates
 * that replace lr / the softplus rates.  loss_out: optional device fp32 scalar
 * that receives L_s = -(1/n_tok) sum_j y_j . M(u_j; W_{s-1}) (Eq. 7).
 * Errors: INVALID_ARG (bad ctx/layer/n_tok/pointer), CUDA.
 */
mone_status mone_ttl_segment(mone_mem* m, int ctx, int layer, const void* X, const void* K,
                             const void* V, int n_tok, const float* eta, float* loss_out,
                             void* stream);

/*
 * Test-time learning of a whole context on every chain (Eq. 9): consecutive
 * segments of seg_T tokens (the last may be shorter and is averaged over its own
 * length), continuing from the current state, so two calls on N1 (a multiple of
 * seg_T) and N2 tokens equal one call on N1+N2.
 * X: [n_ctx][n_layers][N][d_in]; K, V: [n_ctx][n_layers][N][d_out/2]; dtype
 * cfg->dtype, contiguous, 16-byte aligned.  N >= 1.
 * Errors: INVALID_ARG, CUDA.
 */
mone_status mone_ttl_context(mone_mem* m, const void* X, const void* K, const void* V,
                             long long N, void* stream);

/*
 * mone_ttl_context for a context held in HOST memory (the end-to-end form of Eq. 9's
 * chain: the inputs arrive from the host while the memory learns).  X, K, V have the
 * layouts of mone_ttl_context and live in host memory the device can read: page-locked
 * (cudaHostAlloc / cudaHostRegister) or, where the device reads host memory through the
 * host's page tables (Grace), any host memory.  The caller guarantees that each tensor's
 * whole range is allocated: the library checks its first and last bytes only.
 * The context is learned in chunks of chunk_tokens tokens (a multiple of seg_T; 0 lets
 * the library choose about 512 MB of X, K and V per chunk): the library gathers chunk
 * k+1 into one of two device windows (owned by the handle, grown on demand; growing
 * synchronises the stream) on its own staging stream while chunk k is learned on
 * `stream`, so the result equals mone_ttl_context on the same tokens.  Asynchronous:
 * the host buffers must stay valid and unchanged until `stream` has passed the call
 * (mone_mem_sync or a stream synchronisation).  Kernel kind 8 times the gathers.
 * Errors: INVALID_ARG (null or unaligned pointer, device or managed memory, a range
 * the device cannot read, N, chunk_tokens), UNSUPPORTED_SHAPE (a row of X, K or V not
 * a multiple of 16 bytes), OOM (windows), CUDA.
 */
mone_status mone_ttl_context_host(mone_mem* m, const void* X, const void* K, const void* V, long long N,
                                  long long chunk_tokens, void* stream);

/*
 * mone_ttl_context, with per-segment metrics of every chain written into caller
 * buffers, so the learning of a whole context can be followed segment by segment
 * (Sec. 3.4's chain W_0 -> ... -> W_S).  With S = ceil(N / seg_T) segments of this
 * call (numbered from the call's first token) and C = n_ctx * n_layers chains,
 * element [s * C + c] of
 *   seg_loss  is L_s of chain c: the segment mean of Eq. 7's loss (or of the
 *             squared-error variant) at the segment's starting weights;
 *   seg_step  is |mu_s|_F^2 of chain c: the squared Frobenius norm over all fast
 *             weights (W1 and W2; for the SwiGLU memory W_in, W_gate and W_out of
 *             every head) of the step of Eq. 8 (W_s = W_{s-1} - mu_s, before the row
 *             renormalisation; without momentum mu_s is the rate-weighted gradient).
 * Both are fp32 device buffers of S * C elements owned by the caller, 4-byte
 * aligned; either may be null.  The library zeroes them on the stream first, then
 * accumulates into them.  Same inputs, state update and ordering as mone_ttl_context.
 * Errors: INVALID_ARG, CUDA.
 */
mone_status mone_ttl_context_metrics(mone_mem* m, const void* X, const void* K, const void* V, long long N,
                                     float* seg_loss, float* seg_step, void* stream);

/*
 * Memory read (Eq. 4 and the normalisation after it): for every chain and query
 * token, o = M(phi(x_q); W_S) with phi the key/query transform of the mode, then
 * every output head h (width head_dim) becomes gate_h * o_h / sqrt(mean(o_h^2) + eps).
 * K heads are written to K_out, V heads to V_out, dtype cfg->dtype.
 * Xq: [n_ctx][n_layers][Q][d_in] contiguous.  strides[4] are ELEMENT strides of the
 * output for (ctx, layer, kv_head, q); head_dim is contiguous, so memory tokens can
 * be written straight into an attention cache (e.g. after the query's own K/V,
 * as in Eq. 5's concatenation).  1 <= Q <= 4096.  gate_h is SiLU(g_h) under
 * MONE_GATE_SILU.  The second and later consecutive calls with the same Xq, K_out,
 * V_out, Q and strides replay the launches of that read as one captured CUDA graph
 * (same kernels, same results; the weights and inputs are read when it runs).
 * Errors: INVALID_ARG, OOM (first call with a larger Q allocates scratch), CUDA.
 */
mone_status mone_mem_generate_kv(mone_mem* m, const void* Xq, int Q, void* K_out, void* V_out,
                                 const long long strides[4], void* stream);

/*
 * Memory read that allocates nothing.  The paper has no counterpart: this is a
 * service entry point for callers that must not allocate device memory while
 * serving, e.g. a framework whose caching allocator already owns the GPU's free
 * memory, or a latency-bound serving loop that cannot afford cudaMalloc (which
 * can synchronise the device and take a process-wide allocator lock).
 * mone_mem_generate_kv may allocate read scratch on its first call or when Q
 * grows; this variant instead uses one fixed 16 MiB device array compiled into
 * the library (every GPU that loads the library holds it until the process
 * exits).  Same arguments and outputs as mone_mem_generate_kv (bit for bit: the
 * same kernels on the same inputs), and its errors plus two of its own, both
 * returned before any GPU work with mone_last_error saying why:
 * MONE_ERR_UNSUPPORTED_SHAPE when chains * Q * (d_in + d_hid + d_out) exceeds
 * 4,194,304 floats, and MONE_ERR_UNSUPPORTED for a SwiGLU-memory handle
 * (MONE_MEM_SWIGLU), whose read has no fixed-scratch variant.
 * It calls no cudaMalloc, cudaFree or allocating library routine.
 * The first call on a device resolves the array's device address
 * (cudaGetSymbolAddress) with that device current; make that first call before
 * any stream capture.  All calls on a device share the array and every call
 * overwrites it completely before reading it, so nothing carries over between
 * calls, but calls whose GPU work overlaps (e.g. on two streams) race on it:
 * order them on one stream or with events.
 */
mone_status mone_mem_generate_kv_noalloc(mone_mem* m, const void* Xq, int Q, void* K_out, void* V_out,
                                         const long long strides[4], void* stream);

/* Release the state.  The handle is invalid afterwards; a second free returns
 * MONE_ERR_INVALID_ARG.  Synchronises the device. */
mone_status mone_mem_free(mone_mem* m);

/*
 * Copy the fp32 state out ([chains][d_hid][d_in] / [chains][d_hid][d_out]); any
 * argument may be NULL to skip it.  Device pointers; stream-ordered.
 */
mone_status mone_mem_read_state(const mone_mem* m, float* W1, float* W2, float* mu1, float* mu2,
                                void* stream);

/* Overwrite the fp32 state (NULL = keep); the renormalisation targets stay those
 * of W_0.  Device pointers; stream-ordered. */
mone_status mone_mem_write_state(mone_mem* m, const float* W1, const float* W2, const float* mu1,
                                 const float* mu2, void* stream);

/* Synchronise the stream and return (and clear) any latched device error.  A library
 * built with MONE_DEBUG also checks tile and row indices on the device: a failed check
 * skips the access, is latched, and is returned here as MONE_ERR_CHECK with the site in
 * mone_last_error. */
mone_status mone_mem_sync(mone_mem* m, void* stream);

/* Number of device kernels the library has launched on this handle so far. */
long long mone_mem_launch_count(const mone_mem* m);

/*
 * Consumer attention of the read (Eq. 5, with the attention of Eq. 2 per head).  For every
 * chain (context, layer), query head h and query token i:
 *     out[h][i] = sum_j softmax_j(q[h][i] . k[g][j] / sqrt(head_dim)) v[g][j],
 *     g = h / (n_q_heads / n_kv_heads)   (grouped heads),
 * over the keys j that token i sees: the n_mem memory tokens at cache positions
 * 0 .. n_mem-1 (for example written there by mone_mem_generate_kv) and the query
 * tokens' own keys at positions n_mem .. n_mem+i (causal among the query tokens).
 *   Q      [n_ctx][n_layers][n_q_heads][Lq][head_dim], dense, the handle's dtype
 *   K, V   caches of the handle's dtype with element strides kv_strides[4] =
 *          (context, layer, KV head, position), head_dim contiguous, holding at least
 *          n_mem + Lq positions
 *   out    [n_ctx][n_layers][n_q_heads][Lq][head_dim], dense, the handle's dtype
 * Reads the caches only; the memory state is not touched.  Constraints: n_q_heads a
 * multiple of n_kv_heads with n_q_heads / n_kv_heads <= 64; 1 <= Lq; 0 <= n_mem;
 * n_mem + Lq <= 2^20.  Errors: INVALID_ARG.  Asynchronous on stream.
 */
mone_status mone_attention(mone_mem* m, const void* Q, int n_q_heads, int Lq, const void* K, const void* V,
                           const long long kv_strides[4], int n_mem, void* out, void* stream);

/*
 * Per-kernel device timing for measurement.  While enabled, the library records
 * a pair of CUDA events on the caller's stream around every kernel it launches
 * (this adds host work per launch; leave it off outside measurement).
 * mone_mem_kernel_time waits for the recorded events and returns, for one kernel
 * kind, the summed device milliseconds and the launch count since timing was
 * last enabled.  Kinds: 0 input prepass, 1 phase A (forward + fused backward
 * epilogue), 2 phase B (gradient + fused update), 3 finalize (renorm apply /
 * operand refresh), 4 memory read, 5 squared-error pre-pass (M(u) and the residual
 * target, MONE_LOSS_MSE only), 6 consumer attention, 7 resident chains (the fp32 MLP
 * path when d_in + d_out <= 512: every segment of an input window in one launch,
 * forward, backward and update together), 8 host-input gathers (mone_ttl_context_host;
 * timed on the library's staging stream).  Errors: INVALID_ARG, CUDA.
 */
mone_status mone_mem_set_timing(mone_mem* m, int enable);
mone_status mone_mem_kernel_time(mone_mem* m, int kind, double* ms, long long* launches);

/*
 * Busy time of one kernel kind since timing was last enabled: the length (ms) of the union
 * of its launches' [start, end] event intervals, so launches that overlapped on different
 * streams (the two chain groups of a call) count once.  Same kinds and waiting as
 * mone_mem_kernel_time.  Errors: INVALID_ARG, CUDA.
 */
mone_status mone_mem_kernel_busy(mone_mem* m, int kind, double* busy_ms);

const char* mone_status_string(mone_status s);

/* Text of the last CUDA error this thread saw inside the library ("" if none);
 * valid until the thread's next library call. */
const char* mone_last_error(void);
int mone_abi_version(void);

#ifdef __cplusplus
}
#endif
#endif /* MONE_H_ */
