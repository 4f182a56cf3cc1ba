/*
 * blr.h — C ABI of the GB300 (sm_103a) BD-LRU scan library (libblr.so).
 *
 * The BD-LRU of RecBLR (arXiv 2406.12580, Sec. 3.2) is the diagonal, per-channel
 * linear recurrence
 *     h_t = alpha_t * h_{t-1} + beta_t * x_t                                (Sec. 3.2, Eq. linrnn)
 * whose coefficients depend only on the current input through two gates,
 *     r_t = sigmoid(rho_t),  i_t = sigmoid(iota_t)                          (Sec. 3.2, gate equations)
 *     alpha_t = exp(-c * softplus(Lambda) * r_t)                            (Sec. 3.2; c = 1 in the paper)
 *     beta_t  = sqrt(1 - alpha_t^2) * i_t                                   (Sec. 3.2)
 * where rho_t = W_r x_t + b_r and iota_t = W_i x_t + b_i are the gate logits.
 * The gate projections are NOT part of this library: callers pass their
 * pre-activation outputs ("gate_logits"). Lambda is the per-channel learnable
 * decay parameter; c generalises the paper's exponent (c = 1 reproduces it).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * Memory   All pointers except `desc` are DEVICE pointers of the calling
 *          thread's current CUDA device, owned by the caller. The library never
 *          allocates, frees or retains memory; inputs are never written.
 * Layout   Contiguous row-major. x, h, dh, dx: (B, L, D). gate_logits and
 *          dgate_logits: (B, L, 2D), row (b, t) holding rho in columns [0, D)
 *          and iota in columns [D, 2D) (the output layout of one Linear layer
 *          of width 2D). lambda, dlambda: (D). h0, h_last, dh_last, dh0: (B, D).
 * Dtypes   x, gate_logits, h, dh, dx, dgate_logits use the I/O dtype `io`
 *          (float32 or bfloat16). lambda, h0, h_last, dh_last, dh0, dlambda and
 *          the recurrent-step state are always float32. Internal state and all
 *          arithmetic are float32; bf16 outputs are rounded to nearest-even.
 * Streams  Every call is asynchronous on `stream` (NULL = the legacy default
 *          stream) and returns once the work is enqueued.
 * Checks   Arguments are validated on the host before anything is enqueued:
 *          a NULL required pointer, a negative size, c <= 0 or not finite, an
 *          unknown dtype, a too-small workspace or a tensor pointer that is not
 *          16-byte aligned (4-byte for h0, h_last, dh_last, dh0) returns
 *          BLR_ERR_INVALID_ARG; D not a multiple of 8, or a problem too large
 *          for the tiling, returns BLR_ERR_UNSUPPORTED. Nothing is enqueued on
 *          a validation error. A failed launch returns BLR_ERR_CUDA.
 * Empty    B == 0 or D == 0 is a no-op. L == 0 is a valid empty sequence:
 *          h_last = h0 (0 when h0 is NULL); the backward writes dh0 = dh_last
 *          (0 when NULL) and dlambda = 0.
 * Domain   Outputs are finite for finite inputs with r_t > 0 and
 *          softplus(Lambda) > 0 in float32 (|rho| below about 80). At
 *          alpha_t == 1 exactly the gradient through beta_t is infinite
 *          (the derivative of sqrt(1 - alpha^2)); such inputs give inf/nan.
 * Errors   The library never exits, traps or prints. Waits between thread
 *          blocks are bounded (about one second); an expired wait is recorded
 *          in the workspace and reported by blr_workspace_status().
 */
#ifndef BLR_H_
#define BLR_H_

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define BLR_API __attribute__((visibility("default")))
#else
#define BLR_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t. */
typedef struct CUstream_st* blr_stream_t;

typedef enum {
  BLR_F32 = 0,  /* IEEE binary32 */
  BLR_BF16 = 1  /* bfloat16 */
} blr_dtype;

typedef enum {
  BLR_OK = 0,
  BLR_ERR_INVALID_ARG = 1,  /* bad pointer, size, alignment, dtype, c or workspace size */
  BLR_ERR_UNSUPPORTED = 2,  /* valid but outside what the kernels handle (D % 8 != 0, too large) */
  BLR_ERR_CUDA = 3,         /* a CUDA runtime call or launch failed (see blr_last_error_string) */
  BLR_ERR_TIMEOUT = 4,      /* a bounded wait between thread blocks expired (outputs undefined) */
  BLR_ERR_WORKSPACE = 5     /* blr_scan_bwd was given a workspace without matching forward carries */
} blr_status;

/* Problem description of one scan call. */
typedef struct {
  int64_t B;    /* batch rows (independent sequences) */
  int64_t L;    /* sequence length (time steps) */
  int64_t D;    /* channels (the recurrence is independent per channel) */
  blr_dtype io; /* dtype of x, gate_logits, h, dh, dx, dgate_logits */
  float c;      /* decay exponent constant; 1.0 is the paper's alpha = exp(-softplus(Lambda) r) */
} blr_desc;

/*
 * Workspace size in bytes for blr_scan_fwd / blr_scan_bwd (and their _gated
 * and _varlen forms) on `desc`; 0 when the description is invalid or needs none
 * (B, L or D zero). The workspace holds what the forward keeps for the
 * backward, by kernel family (blr_scan_family):
 *   serial: the state every 16 float32 / 8 bfloat16 steps, 0.25-0.5 bytes per
 *           element;
 *   tiled: per-tile records (24 bytes per channel per 64-step tile, under 0.4
 *           bytes per element);
 *   segmented: the serial kernels' kept states, 8 bytes per channel per
 *           segment (of 128 steps or more) and the chained forward's records
 *           (12 bytes per channel per 128 steps), laid over the tiled forward
 *           records, plus the tiled backward records (for the _varlen forms),
 *           under 0.95 bytes per element;
 * plus the float64 partial sums of dlambda and a small header (about 72 bytes
 * per channel). It depends only on B, L, D and the I/O dtype.
 */
BLR_API size_t blr_workspace_bytes(const blr_desc* desc);

/*
 * Which kernels blr_scan_fwd / blr_scan_bwd (and their _gated forms; the
 * _varlen forms when with_lengths is nonzero) run on `desc` (diagnostic; the
 * choice depends only on B, L, D and the I/O dtype). A chain is 32 float32 or
 * 64 bfloat16 channels of one batch row.
 *   BLR_FAMILY_SERIAL     at least 256 chains: one warp walks each chain
 *                         through the whole sequence (one kernel per call).
 *   BLR_FAMILY_SEGMENTED  bfloat16 I/O, fewer chains, L >= 2048 and either
 *                         at least 8 Mi elements or L >= 16384, without
 *                         lengths. blr_scan_fwd and blr_scan_bwd run one
 *                         chained kernel each: 128-step tiles folded by 16
 *                         warps and chained along time by a decoupled
 *                         look-back (the operator of Sec. 3.3), after one
 *                         cudaMemsetAsync that empties the look-back records.
 *                         The _gated forms cut each chain into time segments
 *                         of 128 steps or more: a reduction kernel computes
 *                         every segment's affine map, then one warp walks each
 *                         segment from the carry the maps compose (two kernels
 *                         per call).
 *   BLR_FAMILY_TILED      otherwise: 64-step tiles chained by a decoupled
 *                         look-back (a preparation kernel, then the scan).
 *   BLR_FAMILY_NONE       an invalid or empty problem (nothing is launched).
 */
#define BLR_FAMILY_NONE 0
#define BLR_FAMILY_TILED 1
#define BLR_FAMILY_SERIAL 2
#define BLR_FAMILY_SEGMENTED 3
BLR_API int blr_scan_family(const blr_desc* desc, int with_lengths);

/*
 * Forward BD-LRU scan (Sec. 3.2, Eq. linrnn; the scan of Sec. 3.3):
 *   h[b,t,d] = alpha[b,t,d] * h[b,t-1,d] + beta[b,t,d] * x[b,t,d],
 *   h[b,-1,d] = h0[b,d]   (h0 == NULL: zero state, as in the paper)
 * x           (B, L, D)  io dtype, input of the recurrence
 * gate_logits (B, L, 2D) io dtype, [rho | iota] pre-activations
 * lambda      (D)        float32, Lambda
 * h0          (B, D)     float32 or NULL
 * h           (B, L, D)  io dtype, output; may be NULL to compute only the
 *                        carries the backward needs (and h_last)
 * h_last      (B, D)     float32 or NULL, the float32 state h[b, L-1, :]
 * ws, ws_bytes           device workspace of at least blr_workspace_bytes(desc)
 *                        bytes, 16-byte aligned. Its previous contents are
 *                        ignored; on return (in stream order) it holds the
 *                        kept states that blr_scan_bwd consumes.
 */
BLR_API blr_status blr_scan_fwd(const blr_desc* desc, const void* x, const void* gate_logits,
                        const float* lambda, const float* h0, void* h, float* h_last, void* ws,
                        size_t ws_bytes, blr_stream_t stream);

/*
 * Backward of blr_scan_fwd for the loss  sum_{b,t,d} dh * h + sum_{b,d} dh_last * h_last
 * (gradients derived from the definitions of Sec. 3.2; the paper prints none).
 * With g_t = dh_t + alpha_{t+1} g_{t+1} and g_{L-1} = dh_{L-1} + dh_last:
 *   dx    = g beta                        (direct term only: the gradient through
 *   drho  = dL/dalpha * dalpha/drho        the caller's gate projections is the
 *   diota = g sqrt(1-alpha^2) x i (1-i)    caller's, fed by drho and diota)
 *   dlambda[d] = sum over b, t of the Lambda-derivative (written, not accumulated)
 *   dh0   = alpha_0 g_0
 * dh          (B, L, D)  io dtype, upstream gradient of h
 * dh_last     (B, D)     float32 or NULL (zero)
 * x, gate_logits, lambda, h0: exactly the forward's inputs
 * dx          (B, L, D)  io dtype, output
 * dgate_logits(B, L, 2D) io dtype, output [drho | diota]
 * dlambda     (D)        float32, output
 * dh0         (B, D)     float32 or NULL
 * ws          the workspace a blr_scan_fwd with the same desc and inputs filled
 *             (h may have been NULL in that call). If ws does not hold
 *             carries of a completed forward of the same desc, no output is
 *             written and blr_workspace_status() reports BLR_ERR_WORKSPACE. The
 *             forward's carries survive the call, so the backward may be repeated.
 *             ws may be NULL (ws_bytes is then ignored): the call first
 *             recomputes the forward's carries (a forward without h) in the
 *             library's static scratch, the 128 MiB device array that
 *             blr_scan_fwd_noalloc uses, and runs the backward from them. It
 *             never allocates; problems whose workspace exceeds 128 MiB get
 *             BLR_ERR_UNSUPPORTED with nothing enqueued; calls that use the
 *             scratch must not overlap on the GPU; blr_workspace_status with
 *             ws == NULL reads the scratch's error word.
 * h_{t-1} is recomputed from the forward's kept states, not read from h.
 */
BLR_API blr_status blr_scan_bwd(const blr_desc* desc, const void* dh, const float* dh_last, const void* x,
                        const void* gate_logits, const float* lambda, const float* h0, void* dx,
                        void* dgate_logits, float* dlambda, float* dh0, void* ws, size_t ws_bytes,
                        blr_stream_t stream);

/*
 * Forward and backward scans of a batch whose rows carry their own lengths:
 * row b's sequence is its last lengths[b] steps, rows [L - lengths[b], L) (the
 * left-padded layout of Sec. 3.3's embedding padding). The rows before it are
 * padding: x, gate_logits and dh there are never read, and h, dx and
 * dgate_logits there are never written. The state before the sequence's
 * first step is h0[b] (0 when h0 is NULL); h_last[b] is the state after step
 * L - 1 (h0[b] for an empty row); dh0[b] is the gradient of the state before
 * the first step; dlambda sums over the sequences' steps only.
 * lengths     (B) int32 device array, 4-byte aligned; values outside [0, L]
 *             are clamped
 * Other arguments, the workspace (sized by blr_workspace_bytes for L) and the
 * errors as blr_scan_fwd / blr_scan_bwd; the backward's ws must come from a
 * blr_scan_fwd_varlen with the same lengths, or be NULL (the carries are then
 * recomputed with these lengths, as blr_scan_bwd does). Work and traffic scale with the
 * rows' lengths on problems served by the serial kernels (at least 256
 * chains); the tiled kernels still stream the padding and mask it.
 */
BLR_API blr_status blr_scan_fwd_varlen(const blr_desc* desc, const int32_t* lengths, const void* x,
                                       const void* gate_logits, const float* lambda, const float* h0,
                                       void* h, float* h_last, void* ws, size_t ws_bytes,
                                       blr_stream_t stream);
BLR_API blr_status blr_scan_bwd_varlen(const blr_desc* desc, const int32_t* lengths, const void* dh,
                                       const float* dh_last, const void* x, const void* gate_logits,
                                       const float* lambda, const float* h0, void* dx,
                                       void* dgate_logits, float* dlambda, float* dh0, void* ws,
                                       size_t ws_bytes, blr_stream_t stream);

/*
 * Forward scan fused with the merge of the gated recurrent layer (Alg. 1,
 * H'_y = H_y (x) SiLU(H_z), the line after the BD-LRU):
 *   y[b,t,d] = h[b,t,d] * SiLU(z[b,t,d]),   SiLU(z) = z * sigmoid(z),
 * with h the scan of blr_scan_fwd, which is not written. Saves the separate
 * merge's reading and writing of h.
 * z           (B, L, D)  io dtype, the second branch's input (H_z)
 * y           (B, L, D)  io dtype, output; may be NULL (then only h_last and
 *                        the carries, as blr_scan_fwd with h == NULL)
 * Other arguments, the workspace and the errors as blr_scan_fwd; z must be
 * 16-byte aligned and no output may overlap an input. The merge is fused into
 * the serial and segmented kernels; problems on the tiled kernels
 * (blr_scan_family) run the scan and then an elementwise merge kernel over y
 * in place.
 */
BLR_API blr_status blr_scan_fwd_gated(const blr_desc* desc, const void* x, const void* gate_logits,
                                      const float* lambda, const float* h0, const void* z, void* y,
                                      float* h_last, void* ws, size_t ws_bytes, blr_stream_t stream);

/*
 * Backward of blr_scan_fwd_gated for the loss
 *   sum_{b,t,d} dy * y + sum_{b,d} dh_last * h_last:
 * the scan's backward (outputs as blr_scan_bwd) for dh = dy * SiLU(z), and
 *   dz = dy * h * SiLU'(z),   SiLU'(z) = sigmoid(z) (1 + z (1 - sigmoid(z))),
 * with h recomputed, not read.
 * dy          (B, L, D)  io dtype, upstream gradient of y
 * z           (B, L, D)  io dtype, the forward's z
 * dz          (B, L, D)  io dtype, output
 * ws          the workspace of a blr_scan_fwd_gated (or blr_scan_fwd) of the same
 *             desc and inputs, or NULL, as for blr_scan_bwd.
 * Other arguments as blr_scan_bwd; no output may overlap an input. Problems on
 * the tiled kernels (blr_scan_family) recompute h into dz, form dh in dx and dz
 * in place with an elementwise kernel, then run the scan's backward from dx;
 * the serial and segmented kernels fuse the merge.
 */
BLR_API blr_status blr_scan_bwd_gated(const blr_desc* desc, const void* dy, const float* dh_last,
                                      const void* x, const void* gate_logits, const float* lambda,
                                      const float* h0, const void* z, void* dx, void* dgate_logits,
                                      void* dz, float* dlambda, float* dh0, void* ws, size_t ws_bytes,
                                      blr_stream_t stream);

/*
 * One recurrent-inference step for a batch of states (the low-cost recurrent
 * inference of Sec. 1 and Sec. 4.3): h_t = alpha_t * h_prev + beta_t * x_t.
 * h_prev (B, D) float32; x_t (B, D) io dtype; gate_logits_t (B, 2D) io dtype;
 * lambda (D) float32; h_t (B, D) float32 output (may alias h_prev exactly).
 * Needs no workspace.
 */
BLR_API blr_status blr_step(int64_t B, int64_t D, blr_dtype io, float c, const float* h_prev,
                    const void* x_t, const void* gate_logits_t, const float* lambda, float* h_t,
                    blr_stream_t stream);

/*
 * K consecutive recurrent-inference steps for a batch of states: serving K new
 * behaviors per user in one call (the low-cost recurrent inference of Sec. 1
 * and Sec. 4.3, K times):
 *   h_j = alpha_j * h_{j-1} + beta_j * x_j,  j = 1..K,  h_0 = h_prev.
 * io          dtype of x, gate_logits and h_seq
 * state       dtype of h_prev and h_out: BLR_F32, or BLR_BF16 to halve the state's
 *             memory (the K steps run in float32; h_out is rounded to
 *             nearest-even once)
 * h_prev      (B, D) state dtype
 * x           (B, K, D) io dtype, the K new inputs of every row, oldest first
 * gate_logits (B, K, 2D) io dtype, [rho | iota] of every step
 * lambda      (D) float32
 * h_out       (B, D) state dtype, the state after step K; may alias h_prev exactly
 * h_seq       (B, K, D) io dtype or NULL: the state after every step
 * K == 0 copies h_prev to h_out. Needs no workspace. Pointers 16-byte aligned;
 * no output may overlap an input except h_out == h_prev.
 */
BLR_API blr_status blr_steps(int64_t B, int64_t K, int64_t D, blr_dtype io, blr_dtype state, float c,
                             const void* h_prev, const void* x, const void* gate_logits,
                             const float* lambda, void* h_out, void* h_seq, blr_stream_t stream);

/*
 * Synchronises `stream`, then reads the error word that the kernels of
 * earlier calls on this workspace recorded: BLR_OK, BLR_ERR_TIMEOUT or
 * BLR_ERR_WORKSPACE (BLR_ERR_CUDA if the read itself fails). The word is
 * cleared by the next blr_scan_fwd on the workspace. ws == NULL reads the
 * library's static scratch (that of backward calls made without a workspace).
 */
BLR_API blr_status blr_workspace_status(const blr_desc* desc, const void* ws, size_t ws_bytes,
                                blr_stream_t stream);

/* Static text for a status code. */
BLR_API const char* blr_status_string(blr_status status);

/* Text of the last BLR_ERR_CUDA / validation failure on the calling host thread. */
BLR_API const char* blr_last_error_string(void);

/*
 * Forward scan for callers that cannot allocate device memory (the paper has
 * no counterpart; this is a deployment convenience). Code running inside CUDA
 * stream capture, plugins whose host framework owns every device allocation,
 * and serving loops that forbid allocator calls cannot provide the workspace
 * blr_scan_fwd needs. This entry point computes exactly what blr_scan_fwd
 * computes (same arguments except the workspace) on a scratch array that the
 * library holds in device memory: 128 MiB, allocated on every GPU that loads
 * the library and kept until the process exits. It never calls an allocator.
 *  - Problems whose workspace (blr_workspace_bytes) exceeds 128 MiB return
 *    BLR_ERR_UNSUPPORTED with nothing enqueued; use blr_scan_fwd for them.
 *  - The first call on each device (and the first after the device's CUDA
 *    context has been reset or re-created) looks up the scratch array's
 *    device address (cudaGetSymbolAddress); make that first call before any
 *    stream capture that includes it.
 *  - All calls on a device share the one scratch array, and each call reuses
 *    whatever the last one left there after clearing what must start empty.
 *    The backward entry points called with ws == NULL use the same array
 *    (they recompute the forward's carries in it). Calls of either kind that
 *    may overlap on the GPU (different streams without ordering between
 *    them) race on it: serialise them.
 *  - blr_workspace_status with ws == NULL reads the array's error word. The
 *    array is not a workspace a caller can name: a backward that should use
 *    this forward's carries cannot be given them (with ws == NULL it
 *    recomputes them), so this is in effect a forward-only (inference) path.
 */
BLR_API blr_status blr_scan_fwd_noalloc(const blr_desc* desc, const void* x, const void* gate_logits,
                                        const float* lambda, const float* h0, void* h,
                                        float* h_last, blr_stream_t stream);

/*
 * Diagnostic: runs one thread block that waits on a workspace flag nothing
 * sets, with the given bound in nanoseconds (at most 1e9), then records the
 * expired wait in the workspace. blr_workspace_status() then returns
 * BLR_ERR_TIMEOUT. This is how the bounded-wait path is tested without a
 * fault; it touches only the workspace.
 */
BLR_API blr_status blr_selftest_wait_timeout(const blr_desc* desc, void* ws, size_t ws_bytes,
                                     uint64_t timeout_ns, blr_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* BLR_H_ */
