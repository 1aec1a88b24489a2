/*
 * sdm.h -- C ABI of the Sparse Delta Memory (SDM) hot path on one GB300 (sm_103a).
 *
 * Sparse Delta Memory (arXiv 2607.07386) replaces Gated DeltaNet's dense
 * d_qk x d_v state with an explicit per-head memory M in R^{N x d_v}.  For every
 * token t and head h:
 *   1. sparse key selection (Sec. 3.1 item 1, Sec. 2 "Product Key Memory"):
 *      s = P x in R^{2 sqrt(N)} is split into halves s1, s2; the N slot scores are
 *      the outer sum s1 (+) s2 (slot = i*sqrt(N) + j); the top-k slots are found as
 *      top_k(top_k(s1) (+) top_k(s2)) and their scores are softmax-normalised
 *      (Sec. 4, "SDM Configuration");
 *   2. gated delta write (Eqs. sdm-decay, sdm-write) on the k_write selected slots:
 *      M~[i] = alpha_t M[i];  M[i] = M~[i] + beta_t w_i (v_t - v~_t),
 *      v~_t = sum_i w_i M~[i];  unselected slots are unchanged;
 *   3. sparse read (Eq. sdm-read) of the post-write memory: y_t = sum_i r_i M_t[i].
 *   The memory of every sequence starts as a copy of the learned initial state M0
 *   (Sec. 3.1, "Learned Initial State").
 *
 * Conventions (all entry points):
 *   - Every buffer is caller-owned device memory (except where a host pointer is
 *     stated), contiguous row-major, 16-byte aligned.  The library never
 *     allocates device memory: scratch space is the caller's `workspace`.
 *   - One dtype (shape->dtype) for every floating-point tensor: memory, M0, P_q,
 *     P_k, q, k, v, alpha, beta and y.  Slot indices are int32, slot weights fp32.
 *     Arithmetic is fp32 (scores, prediction, delta, read), with storage rounding
 *     (round-to-nearest-even) of every written memory row and of y.
 *   - Asynchronous on `stream` (a cudaStream_t; NULL = legacy default stream);
 *     no hidden synchronisation.  Calls that overlap on the GPU must not share
 *     `mem` or `workspace`.
 *   - Errors: shape / pointer / workspace errors return SDM_ERR_INVALID_ARG (or
 *     SDM_ERR_UNSUPPORTED) before anything is launched; launch failures return
 *     SDM_ERR_CUDA.  sdm_last_error() gives a message (thread-local).  Kernels
 *     never trap: a slot index outside [0, N) is skipped and recorded in a device
 *     status word read by sdm_device_status().
 *   - Index lists are ascending by slot within each token and the weights of a
 *     token sum to 1.
 */
#ifndef SDM_H
#define SDM_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define SDM_ABI_VERSION 2

/* Same type as cudaStream_t. */
typedef struct CUstream_st* sdm_stream_t;

typedef enum {
    SDM_OK = 0,
    SDM_ERR_INVALID_ARG = 1,   /* bad shape, null pointer, misalignment, aliasing, small workspace */
    SDM_ERR_UNSUPPORTED = 2,   /* valid SDM shape this build has no kernel for (see sdm_last_error) */
    /* 3 is not used: the library never allocates device memory, so it has no out-of-memory code */
    SDM_ERR_CUDA = 4,          /* a CUDA runtime call or launch failed (message has cudaGetErrorString) */
    SDM_ERR_TIMEOUT = 5,       /* sdm_device_status: a bounded device wait gave up (status bit 2) */
    SDM_ERR_DEVICE = 6         /* sdm_device_status: any other device-side fault bit was set */
} sdm_status;

typedef enum { SDM_F32 = 0, SDM_BF16 = 1 } sdm_dtype;

/* PROJECTED: s = P x with P [H, 2 sqrt(N), d_k] (the paper's W_k / W_q factored through d_k).
 * DIRECT:    s = x itself; requires d_k == 2 sqrt(N) (the paper's k' in R^{2 sqrt(N)}); P unused. */
typedef enum { SDM_ADDR_PROJECTED = 0, SDM_ADDR_DIRECT = 1 } sdm_addr_mode;

typedef struct {
    int32_t B;        /* independent sequences */
    int32_t H;        /* SDM heads */
    int32_t T;        /* tokens per sequence in this call (1 for sdm_decode_step) */
    int32_t d_k;      /* key / query width */
    int32_t d_v;      /* value width = memory row width; d_v * elem_bytes must be a multiple of 16 */
    int64_t N;        /* memory slots per head; a perfect square S*S */
    int32_t k_write;  /* W: slots written per token, 1 <= W <= min(S, 64) for addressing */
    int32_t k_read;   /* R: slots read per token, 1 <= R <= min(S, 64) for addressing */
    int32_t dtype;    /* sdm_dtype */
    int32_t addr;     /* sdm_addr_mode */
} sdm_shape;

/* Returns SDM_ABI_VERSION of the loaded library. */
int sdm_abi_version(void);

/* Message of the last failing call on this host thread ("" if none). */
const char* sdm_last_error(void);

/* Bytes of workspace that sdm_forward / sdm_decode_step / sdm_address need for `shape`
 * (covers slot lists the caller does not request, PKM partial lists and row norms).
 * Returns 0 and sets sdm_last_error for an invalid shape. */
size_t sdm_workspace_bytes(const sdm_shape* shape);

/* Sec. 3.1 "Learned Initial State": mem[b, h] = M0[h] for every sequence b.
 * M0: [H, N, d_v] (read only);  mem: [B, H, N, d_v] (written).  Must not overlap. */
sdm_status sdm_init_memory(const sdm_shape* shape, const void* M0, void* mem, sdm_stream_t stream);

/* Sparse key selection only (Sec. 3.1 item 1; Sec. 2 PKM; Sec. 4 softmax), for every
 * (b, h, t): write slots from k with P_k, read slots from q with P_q.
 * P_q, P_k: [H, 2 sqrt(N), d_k] (NULL allowed in DIRECT mode);  q, k: [B, H, T, d_k].
 * idx_w/w_w: [B, H, T, k_write], idx_r/w_r: [B, H, T, k_read]; all four required here.
 * Selected slot sets equal the exact top-k of the float64 outer-sum scores under
 * (score desc, slot asc) order: fp32 scores are certified against an error bound and
 * near-ties are re-decided in float64. */
sdm_status sdm_address(const sdm_shape* shape, const void* P_q, const void* P_k,
                       const void* q, const void* k,
                       int32_t* idx_w, float* w_w, int32_t* idx_r, float* w_r,
                       void* workspace, size_t workspace_bytes, sdm_stream_t stream);

/* Whole hot path over T tokens: addressing (as sdm_address), then the fused
 * recurrence (Eqs. sdm-decay, sdm-write, sdm-read) in token order, per (b, h).
 * mem: [B, H, N, d_v] running memory, updated in place to M_T (must not alias inputs);
 * v: [B, H, T, d_v];  alpha, beta: [B, H, T] (gates in (0,1) and [0,1]);
 * y: [B, H, T, d_v] (written).  idx_w, w_w, idx_r, w_r may be NULL (kept in the
 * workspace) or caller buffers that receive the selection. */
sdm_status sdm_forward(const sdm_shape* shape, const void* P_q, const void* P_k,
                       const void* q, const void* k, const void* v,
                       const void* alpha, const void* beta, void* mem, void* y,
                       int32_t* idx_w, float* w_w, int32_t* idx_r, float* w_r,
                       void* workspace, size_t workspace_bytes, sdm_stream_t stream);

/* sdm_init_memory followed by sdm_forward in one call: every sequence's memory starts as
 * a copy of M0 [H, N, d_v] (Sec. 3.1 "Learned initial state"), then the whole hot path
 * runs over the T tokens.  Same results as the two calls.  The broadcast runs on a
 * library-owned side stream of the current device, ordered after the work already on
 * `stream` and joined back into `stream` before the recurrence, so it overlaps the
 * addressing.  M0 must not overlap mem.  Calls from several host threads on one device
 * are ordered by a lock while they enqueue. */
sdm_status sdm_forward_m0(const sdm_shape* shape, const void* M0, const void* P_q, const void* P_k,
                          const void* q, const void* k, const void* v,
                          const void* alpha, const void* beta, void* mem, void* y,
                          int32_t* idx_w, float* w_w, int32_t* idx_r, float* w_r,
                          void* workspace, size_t workspace_bytes, sdm_stream_t stream);

/* Bytes of workspace sdm_forward_lazy needs for `shape`: sdm_workspace_bytes plus a
 * first-writer table of B*H*N int32.  Returns 0 for an invalid shape. */
size_t sdm_lazy_workspace_bytes(const sdm_shape* shape);

/* sdm_forward on a copy-on-write memory seeded lazily from M0 (Sec. 3.1 "Learned initial
 * state"), in place of the B-fold broadcast of sdm_forward_m0.
 * touched: [B, H, ceil(N/32)] uint32 bitmaps, read and updated: bit (s % 32) of word
 * s / 32 of chain (b, h) is set once slot s has been written.  A clear bit means the
 * slot's value is M0[h, s] and mem[b, h, s] is neither read nor written; a set bit
 * means mem[b, h, s] holds the slot.  Start a sequence with all bits clear (mem may hold
 * anything); pass the same mem and touched to continue it.
 * After the call, the memory described by (M0, touched, mem) equals the memory of
 * sdm_forward_m0 (or of sdm_init_memory + sdm_forward calls), and y and the slot lists
 * are the same, bit for bit; sdm_materialize turns it into the dense memory.
 * M0: [H, N, d_v]; other arguments as in sdm_forward_m0; workspace: at least
 * sdm_lazy_workspace_bytes(shape), 256-byte aligned.  touched must not overlap any
 * other buffer; M0 must not overlap mem. */
sdm_status sdm_forward_lazy(const sdm_shape* shape, const void* M0, uint32_t* touched,
                            const void* P_q, const void* P_k, const void* q, const void* k,
                            const void* v, const void* alpha, const void* beta, void* mem, void* y,
                            int32_t* idx_w, float* w_w, int32_t* idx_r, float* w_r,
                            void* workspace, size_t workspace_bytes, sdm_stream_t stream);

/* Dense memory of a copy-on-write state: mem[b, h, s] = M0[h, s] for every slot whose
 * bit in touched ([B, H, ceil(N/32)] uint32, as sdm_forward_lazy leaves it) is clear;
 * other rows are left as they are.  M0: [H, N, d_v]; mem: [B, H, N, d_v]. */
sdm_status sdm_materialize(const sdm_shape* shape, const void* M0, const uint32_t* touched, void* mem,
                           sdm_stream_t stream);

/* Gates of every token and head from the layer input (Sec. 3.1, after Eq. sdm-write):
 *   alpha[b, h, t] = exp(-A[h] * softplus(W_a[h] . x[b, t] + b_dt[h])),
 *   beta[b, h, t]  = sigmoid(W_b[h] . x[b, t]).
 * x: [B, T, d_model], W_a, W_b: [H, d_model] (storage dtype, 16-byte aligned;
 * d_model * element size a multiple of 16 bytes); b_dt, A: [H] float32; alpha, beta:
 * [B, H, T] storage dtype (the layout sdm_forward takes).  H <= 32.  Uses shape B, H, T
 * and dtype only.  fp32 arithmetic; outputs rounded to nearest.  With bf16 storage, H = 16
 * or 32 and d_model % 8 == 0 the projections run on the tensor cores ([B*T, d_model] x
 * [d_model, 2H], bf16 products accumulated in fp32 blocks of 16, see sdm_gates_tensor_cores);
 * otherwise as fp32 fused multiply-adds. */
sdm_status sdm_gates(const sdm_shape* shape, int32_t d_model, const void* x, const void* W_a,
                     const void* W_b, const float* b_dt, const float* A, void* alpha, void* beta,
                     sdm_stream_t stream);

/* 1 if sdm_gates takes the tensor-core form for this shape and d_model, else 0 (its error
 * bound differs: bf16 products summed in fp32 blocks of 16, like the scores). */
int sdm_gates_tensor_cores(const sdm_shape* shape, int32_t d_model);

/* Head-mixing projection (Sec. 3.1, "Norm, Gating, and Head Mixing") on the tensor cores:
 *   out[m, n] = sum_k z[m, k] W_o[n, k],   m < B*T, n < d_model, k < H*d_v,
 * z: [B*T, H*d_v] (sdm_norm_gate's output), W_o: [d_model, H*d_v], out: [B*T, d_model], all
 * bf16, row-major, 16-byte aligned; fp32 accumulation, out rounded to nearest.  bf16 storage
 * only (SDM_ERR_UNSUPPORTED otherwise); d_model a multiple of 32, H*d_v a multiple of 8.  out
 * must not overlap z or W_o. */
sdm_status sdm_head_mix(const sdm_shape* shape, int32_t d_model, const void* z, const void* W_o,
                        void* out, sdm_stream_t stream);

/* Output gate of every head (Sec. 3.1, "Norm, Gating, and Head Mixing"):
 *   z[b, t, h, :] = g[b, h, t, :] * gamma * y[b, h, t, :] / sqrt(mean(y[b, h, t, :]^2) + eps).
 * y, g: [B, H, T, d_v] storage dtype; gamma: [d_v] float32 RMSNorm scale; eps >= 0;
 * z: [B, T, H, d_v] storage dtype, i.e. [B*T, H*d_v] row-major, the operand of the
 * head-mixing projection o = z W_o^T (a plain GEMM the caller runs).  d_v * element size
 * <= 1024 bytes.  16-byte aligned buffers; z must not overlap y, g or gamma. */
sdm_status sdm_norm_gate(const sdm_shape* shape, const void* y, const void* g, const float* gamma,
                         float eps, void* z, sdm_stream_t stream);

/* Bytes of workspace sdm_access_stats needs (two slot bitmaps per chain); 0 if invalid. */
size_t sdm_access_stats_workspace_bytes(const sdm_shape* shape);

/* Access diagnostics of a selection (App. "Memory Utilization and Access"), as float64
 * sums over all B*H*T tokens, written to the device array out (4 + k_write + k_read):
 *   out[0], out[1]: sum of u(p) = exp(H(p)) / k, H(p) = -sum p_i log p_i, over the write
 *                   weights w_w and over the read weights w_r (normalised effective keys);
 *   out[2], out[3]: distinct slots written (idx_w) and read (idx_r), summed over chains;
 *   out[4 + m - 1]            (m = 1..k_write): sum of C(m) of the write weights,
 *   out[4 + k_write + m - 1]  (m = 1..k_read):  sum of C(m) of the read weights,
 *                   C(m) = the sum of the m largest weights of the token.
 * Divide by B*H*T (or by N * B*H for the slot counts) for means and fractions.  Inputs as
 * sdm_address produces them ([B, H, T, k] each, k <= 64); indices outside [0, N) are not
 * counted.  workspace: >= sdm_access_stats_workspace_bytes(shape), 256-byte aligned. */
sdm_status sdm_access_stats(const sdm_shape* shape, const int32_t* idx_w, const float* w_w,
                            const int32_t* idx_r, const float* w_r, double* out,
                            void* workspace, size_t workspace_bytes, sdm_stream_t stream);

/* One decode step for B independent sequences: sdm_forward with shape->T == 1 and
 * the per-token tensors shaped [B, H, d] / [B, H]. */
sdm_status sdm_decode_step(const sdm_shape* shape, const void* P_q, const void* P_k,
                           const void* q, const void* k, const void* v,
                           const void* alpha, const void* beta, void* mem, void* y,
                           int32_t* idx_w, float* w_w, int32_t* idx_r, float* w_r,
                           void* workspace, size_t workspace_bytes, sdm_stream_t stream);

/* Bytes of workspace sdm_recur needs for `shape` (its hazard table); 0 if invalid. */
size_t sdm_recur_workspace_bytes(const sdm_shape* shape);

/* Recurrence with explicit addressing (Eqs. sdm-decay, sdm-write, sdm-read), no PKM:
 * idx_w [B,H,T,k_write] / w_w fp32, idx_r [B,H,T,k_read] / w_r fp32 (any weights,
 * e.g. dense key values for the GDN special case of Sec. 3.1; k_write, k_read <= 64).
 * Slot lists must be strictly ascending within each token, as sdm_address produces
 * them (App. A.2 sorts the selected indices); a violation is recorded in bit 1 of the
 * device status word and its results are undefined.  N need not be a square here.
 * v, alpha, beta, mem, y as in sdm_forward; shape->d_k and shape->addr are ignored.
 * workspace: >= sdm_recur_workspace_bytes(shape) bytes, 256-byte aligned. */
sdm_status sdm_recur(const sdm_shape* shape, const int32_t* idx_w, const float* w_w,
                     const int32_t* idx_r, const float* w_r, const void* v,
                     const void* alpha, const void* beta, void* mem, void* y,
                     void* workspace, size_t workspace_bytes, sdm_stream_t stream);

/* The recurrence of sdm_recur in chunkwise (WY) form (App. A.1-A.2): per chunk of `chunk`
 * tokens (1..32), segmented cumulative log-decays, gated sparse inner products by two-pointer
 * merge, a unit lower-triangular solve, then gather, correct, output and scatter against the
 * chunk-initial memory.  The memory is rounded to the storage dtype at chunk boundaries only
 * and reads inside a chunk see its unrounded writes, so results differ from sdm_recur's by
 * storage rounding alone (chunk = 1: reads of slots the same token writes).  Arguments and
 * layouts as in sdm_recur (no workspace); d_v <= 256, k_write, k_read <= 64.  Slot lists
 * must be strictly ascending (the two-pointer merges rely on it); a violation sets bit 1
 * of the device status word and leaves the results undefined.  A gate alpha of exactly 0
 * decays by e^-80 (below fp32 precision of any stored value) instead of 0. */
sdm_status sdm_recur_chunkwise(const sdm_shape* shape, const int32_t* idx_w, const float* w_w,
                               const int32_t* idx_r, const float* w_r, const void* v,
                               const void* alpha, const void* beta, void* mem, void* y,
                               int32_t chunk, sdm_stream_t stream);

/* Bytes of the undo log of sdm_recur_undo: B*H*T*k_write rows of d_v storage elements. */
size_t sdm_undo_log_bytes(const sdm_shape* shape);

/* sdm_recur that also writes the undo log of the backward (App. A.3): undo[b, h, t, n, :]
 * = the row M_{t-1}[idx_w[b, h, t, n]] the write of token t overwrote, in storage bits
 * ([B, H, T, k_write, d_v], sdm_undo_log_bytes(shape) bytes, 16-byte aligned, not
 * overlapping any other buffer).  Entries of out-of-range slots are not written.  y and
 * mem are those of sdm_recur, bit for bit. */
sdm_status sdm_recur_undo(const sdm_shape* shape, const int32_t* idx_w, const float* w_w,
                          const int32_t* idx_r, const float* w_r, const void* v,
                          const void* alpha, const void* beta, void* mem, void* y, void* undo,
                          void* workspace, size_t workspace_bytes, sdm_stream_t stream);

/* Backward of the recurrence with in-place undo (App. A.3): reverse-mode gradients of
 * L = sum_{b,h,t} <dy[b,h,t], y[b,h,t]> with the stored (rounded) rows treated as the
 * forward's values.  mem: M_T as sdm_recur_undo left it, restored in place to M_0 (the
 * state before that call) on return; undo: that call's log; dy: [B, H, T, d_v] storage
 * dtype.  Outputs (float32, written): dv [B, H, T, d_v], dalpha, dbeta [B, H, T], dw_w
 * [B, H, T, k_write], dw_r [B, H, T, k_read]; dM [B, H, N, d_v] float32 must be zero on
 * entry and receives dL/dM_0 per sequence (sum over b for a shared M0).  Other arguments as
 * in sdm_recur.  d_v must be a multiple of 32, at most 256; k_write and k_read at most 32
 * (SDM_ERR_UNSUPPORTED otherwise).  Outputs must not overlap each other or the inputs.  Slot
 * lists must be strictly ascending, as in sdm_recur; a violation sets bit 1 of the device
 * status word. */
sdm_status sdm_recur_backward(const sdm_shape* shape, const int32_t* idx_w, const float* w_w,
                              const int32_t* idx_r, const float* w_r, const void* v,
                              const void* alpha, const void* beta, void* mem, const void* undo,
                              const void* dy, float* dv, float* dalpha, float* dbeta, float* dw_w,
                              float* dw_r, float* dM, sdm_stream_t stream);

/* Quantised snapshots of the undo log (App. A.3: for long sequences the log can be kept as fp8
 * or int4, which the paper reports does not hurt training).  Row r of the log (r = ((b*H + h)*T
 * + t)*k_write + n, d_v elements) is kept as one float32 scale s_r = fl32(max|row| / top), 1 for
 * an all-zero row, and d_v codes q = round(fl32(row / s_r)), every step a correctly rounded
 * float32 operation: SDM_UNDO_FP8 codes are e4m3 values (top 448, round to nearest even, one
 * byte per element); SDM_UNDO_INT4 codes are the integers -7..7 (top 7, ties to even), two per
 * byte, element 2i in the low nibble, two's complement. */
enum { SDM_UNDO_FP8 = 1, SDM_UNDO_INT4 = 2 };

/* Bytes of the codes of a quantised log: B*H*T*k_write rows of d_v (fp8) or d_v / 2 (int4)
 * bytes; the scales take B*H*T*k_write floats more.  0 for an invalid shape or kind. */
size_t sdm_undo_code_bytes(const sdm_shape* shape, int kind);

/* Quantises the undo log of sdm_recur_undo (stored rows, [B, H, T, k_write, d_v]) into codes
 * and scales as above (caller-owned device buffers; codes 16-byte aligned, none of the three
 * overlapping).  Rows of write entries whose slot index is out of range were never written by
 * the forward; their codes are unspecified and the backward never reads them.  d_v must be a
 * multiple of 32, at most 256. */
sdm_status sdm_undo_quantize(const sdm_shape* shape, const void* undo, int kind, void* codes,
                             float* scales, sdm_stream_t stream);

/* sdm_recur_backward with the log read back from a quantised snapshot: each logged row is taken
 * as the stored value (storage dtype rounding) of q * s_r, both in the chain rule and in the
 * undo, so mem returns to M_0 only up to the snapshot's quantisation.  Arguments and outputs as
 * in sdm_recur_backward, with (kind, codes, scales) from sdm_undo_quantize in place of undo. */
sdm_status sdm_recur_backward_q(const sdm_shape* shape, const int32_t* idx_w, const float* w_w,
                                const int32_t* idx_r, const float* w_r, const void* v,
                                const void* alpha, const void* beta, void* mem, int kind,
                                const void* codes, const float* scales, const void* dy, float* dv,
                                float* dalpha, float* dbeta, float* dw_w, float* dw_r, float* dM,
                                sdm_stream_t stream);

/* Reads (host pointer `code`, synchronising on `stream`) and clears the device
 * status word of the current device: 0 = no fault; bit 0 = a slot index outside
 * [0, N) was skipped; bit 1 = a slot list given to the recurrence (forward, chunkwise
 * or backward) was not strictly ascending; bit 2 = a bounded device wait gave up (the
 * tensor-core score kernel's mbarrier waits, or the writer/reader hand-over of the
 * recurrence): the kernel returned early and its results are undefined; bit 3 = a
 * selection invariant failed (a candidate list not ordered by score; results
 * undefined).  Returns SDM_ERR_TIMEOUT when bit 2 was set, else SDM_ERR_DEVICE when the
 * word was non-zero, else SDM_OK; *code always receives the whole word. */
sdm_status sdm_device_status(int32_t* code, sdm_stream_t stream);

/* Size of the fixed device scratch behind sdm_recur_noalloc (its hazard table). */
#define SDM_RECUR_NOALLOC_SCRATCH_BYTES ((size_t)16 << 20)

/* sdm_recur without a workspace argument: the hazard table lives in a device array of
 * SDM_RECUR_NOALLOC_SCRATCH_BYTES reserved by the library (the paper has no counterpart;
 * this serves callers that cannot provide device memory, e.g. a runtime whose own pool
 * owns the device, or a serving loop that must not call an allocator).  Same arguments,
 * layouts and results as sdm_recur, bit for bit.  Needs B*H*T*max(k_write,k_read)*4 bytes
 * of that scratch; larger shapes return SDM_ERR_UNSUPPORTED before launching anything.
 * Allocates nothing.  The first call on a device looks the array's address up (host-side
 * set-up; make that first call before any stream capture); a device reset
 * (cudaDeviceReset) afterwards is not supported, since the cached address would be stale.
 * One array per device: calls that overlap on the GPU race on it and must be serialised
 * by the caller. */
sdm_status sdm_recur_noalloc(const sdm_shape* shape, const int32_t* idx_w, const float* w_w,
                             const int32_t* idx_r, const float* w_r, const void* v,
                             const void* alpha, const void* beta, void* mem, void* y,
                             sdm_stream_t stream);

/* Reads into host array `counts` (synchronising on `stream`) and clears the first n
 * (<= 15) event counters of the current device's selection diagnostics:
 *   [0] a per-half top-k boundary not certified by the fp32 scores (scores closer than
 *       their error bound): the band is re-ranked by compensated rescoring
 *   [1] ... whose band reached past the kept list (the whole half is rescanned)
 *   [2] an outer-sum boundary not certified by the fp32 scores
 *   [3] ... whose band reached past 64 candidates (serial float64 resolution)
 *   [4] a survivor-buffer overflow retried on the tensor-core score path
 *   [5] an outer-sum band that reached the last kept candidate (list extended to 64)
 *   [6] a band near-tie decided by float64 rescoring of its entries
 *   [7] the serial float64 fallback (heavy ties)
 *   [8] total entries of the half bands re-ranked ([0] bands)
 *   [9] total entries of the outer-sum bands re-ranked ([2] bands)
 * Counters wrap modulo 2^32. */
sdm_status sdm_device_stats(uint32_t* counts, int n, sdm_stream_t stream);

/* Launch plan of the recurrence kernels for `shape` (the paper has no counterpart; for
 * tests that must reach a given kernel variant, and for tuning).  Writes the first n
 * (<= 6) of, in order: the 16-byte chunks of a memory row each warp owns (its d-range),
 * the d-ranges per (b, h) chain, the slot positions each lane handles per token, the
 * hazard window in tokens (row prefetches in flight ahead of the processed token), the
 * token phases: warps that interleave the tokens of one (chain, d-range) (0 when T == 1:
 * one warp, no look-ahead), and each such warp's prefetch depth in its own tokens.  Host
 * only: launches nothing. */
sdm_status sdm_recur_plan(const sdm_shape* shape, int32_t* out, int n);

/* Test hook of the tensor-core score kernel (the paper has no counterpart): the raw fp32
 * scores s = P x (Sec. 3.1 item 1) the selection starts from, as the tcgen05 MMA accumulates
 * them, written to scores [2][H][B*T][2 sqrt(N)] float32 (side 0: q with P_q, side 1: k with
 * P_k; token index b*T + t; columns of both halves).  For testing the error bound the
 * selection certifies with.  Same arguments as sdm_address otherwise (workspace of
 * sdm_workspace_bytes).  Returns SDM_ERR_UNSUPPORTED for shapes that do not take the
 * tensor-core path (bf16, PROJECTED, d_k 64 or 128, k <= 32). */
sdm_status sdm_test_scores(const sdm_shape* shape, const void* P_q, const void* P_k, const void* q,
                           const void* k, float* scores, void* workspace, size_t workspace_bytes,
                           sdm_stream_t stream);

/* Test hook for the bounded device waits (the paper has no counterpart).  Runs sdm_recur
 * (same arguments and workspace) with every wait of the token-interleaved recurrence
 * kernel limited to wait_cycles SM clock cycles (1 .. 2^32), with the first warp of every
 * CTA withholding the progress word of token 0 and every later token waiting for it.  Those
 * waits run out; every CTA leaves its token loop and returns, and bit 2 of the device status
 * word is set (sdm_device_status then returns SDM_ERR_TIMEOUT).  y and mem are left undefined.
 * Returns SDM_ERR_UNSUPPORTED when that kernel does not serve `shape` (T == 1). */
sdm_status sdm_test_recur_wait_timeout(const sdm_shape* shape, const int32_t* idx_w, const float* w_w,
                                       const int32_t* idx_r, const float* w_r, const void* v,
                                       const void* alpha, const void* beta, void* mem, void* y,
                                       void* workspace, size_t workspace_bytes, int64_t wait_cycles,
                                       sdm_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* SDM_H */
