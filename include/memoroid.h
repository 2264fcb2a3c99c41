/*
 * memoroid.h -- C ABI of the GB300 (sm_103a) resettable memoroid scans.
 *
 * The library evaluates memoroid memory models over one flat "tape" of
 * concatenated episodes ("Recurrent Reinforcement Learning with Memoroids",
 * arXiv 2402.09900): a begin flag b_t = 1 on the first step of each episode
 * (Section 2.1) drives the resettable monoid transform of Theorem 3.2, so
 * that no information crosses an episode boundary.  States are the inclusive
 * scan h_t = e_I . f(P_0) . ... . f(P_t) of Definition 3.1.
 *
 * Conventions shared by every entry point:
 *   - Every tensor argument is caller-owned DEVICE memory, row-major and
 *     contiguous.  The library never allocates or frees device memory; scratch
 *     space ("workspace") comes from the caller, sized by the *_workspace_bytes
 *     query, 256-byte aligned.
 *   - Complex tensors are interleaved (re, im) fp32 pairs (the memory layout
 *     of torch.complex64).  Complex arrays must be 16-byte aligned.
 *   - `stream` is a cudaStream_t (NULL = the legacy default stream).  Calls
 *     only enqueue work and return at once.  Argument errors are reported
 *     synchronously by the return value; launch failures map to
 *     MEMOROID_ERR_CUDA.  Kernels never trap: a bounded wait that runs out
 *     records MEMOROID_ERR_TIMEOUT in the workspace, read back by
 *     memoroid_get_device_error().
 *   - B independent tapes are scanned in one call.  start[b, 0] = 1, or a NULL
 *     initial state, means the tape starts from the monoid identity e_I.
 *   - Gradients of complex inputs follow PyTorch's convention
 *     (grad = dL/dRe + i dL/dIm).
 *   - Calls may be captured into a CUDA graph on a capturing stream (they
 *     allocate nothing and make no synchronous call): a captured call clears
 *     the part of its workspace it must read fresh on every replay, so
 *     replays with new data in the captured buffers are correct.  Calls that
 *     share a workspace must not overlap in time, captured or not.  (The
 *     workspace-free memoroid_scan_diag_fwd_static must make its first call
 *     on a device outside any capture.)
 */
#ifndef MEMOROID_H
#define MEMOROID_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    MEMOROID_OK = 0,
    MEMOROID_ERR_INVALID_ARG = 1, /* null, misaligned or out-of-range argument */
    MEMOROID_ERR_UNSUPPORTED = 2, /* a shape or mode this build does not implement */
    MEMOROID_ERR_WORKSPACE = 3,   /* workspace missing, misaligned or too small */
    MEMOROID_ERR_CUDA = 4,        /* a CUDA runtime call or launch failed */
    MEMOROID_ERR_TIMEOUT = 5,     /* a bounded device-side wait ran out */
    MEMOROID_ERR_BAD_DATA = 6     /* a device-side check of the data failed (see the call) */
} memoroid_status_t;

typedef enum { MEMOROID_F32 = 0, MEMOROID_BF16 = 1 } memoroid_dtype_t;

/* Human-readable name of a status code (static string). */
const char *memoroid_status_string(memoroid_status_t status);

/* Library version as major*10000 + minor*100 + patch. */
int memoroid_version(void);

/* ======================================================================== */
/* Diagonal complex scan (S5 / LRU memoroid, Appendix "Simplified State     */
/* Space Models" and "Linear Recurrent Unit", with diagonal X; reset per    */
/* Theorem 3.2):                                                            */
/*     h_t = u_t                          if b_t = 1                        */
/*     h_t = lambda_t * h_{t-1} + u_t     otherwise (h_{-1} = h0, or 0)     */
/* element-wise over D complex channels.                                    */
/* ======================================================================== */

/* Bytes of workspace needed by memoroid_scan_diag_fwd and _bwd for this
 * shape (one size serves both).  Returns 0 for an invalid shape. */
size_t memoroid_scan_diag_workspace_bytes(int64_t B, int64_t L, int64_t D);

/* Number of GPU kernels one memoroid_scan_diag_fwd (backward = 0) or
 * memoroid_scan_diag_bwd (backward = 1) call launches for this shape, not
 * counting the small workspace-header memset (-1 for an invalid shape). */
int memoroid_scan_diag_kernels_per_call(int64_t B, int64_t L, int64_t D, int lambda_per_step,
                                        int backward, int with_grad_lambda);

/*
 * Forward diagonal scan.
 *   lambda          complex [D] (lambda_per_step = 0) or [B,L,D] (= 1)
 *   u               complex [B,L,D]: the lifted inputs f(P_t)
 *   start           uint8 [B,L]: begin flags, 0 or 1 (any non-zero is 1)
 *   h0              complex [B,D] or NULL (identity): state before step 0,
 *                   used only where start[b,0] = 0
 *   h               complex [B,L,D] output; may alias u
 *   h_last          complex [B,D] output (h at step L-1) or NULL
 *   D must be even (two complex channels per 16-byte access).
 * Errors: INVALID_ARG (null/misaligned pointer, negative size, odd D),
 * WORKSPACE, CUDA.
 */
memoroid_status_t memoroid_scan_diag_fwd(const void *lambda, int lambda_per_step, const void *u,
                                         const uint8_t *start, const void *h0, void *h,
                                         void *h_last, int64_t B, int64_t L, int64_t D,
                                         void *workspace, size_t workspace_bytes, void *stream);

/*
 * Backward diagonal scan (reverse-mode of the forward; no truncation across
 * the tape, cf. the full-BPTT gradient of Section 3).  With delta_t = dL/dh_t
 * accumulated through the recurrence,
 *     delta_t = grad_h_t + [b_{t+1} = 0] conj(lambda_{t+1}) delta_{t+1},
 *     delta_{L-1} = grad_h_{L-1} + grad_h_last,
 * outputs grad_u_t = delta_t, grad_lambda = sum_{t: b_t=0} delta_t conj(h_{t-1})
 * (over B and L for a per-channel lambda -> [D]; per step -> [B,L,D]) and
 * grad_h0 = [b_0 = 0] conj(lambda_0) delta_0.
 *   h               complex [B,L,D]: the forward output (must not alias grad_u)
 *   grad_h          complex [B,L,D]
 *   grad_h_last     complex [B,D] or NULL
 *   grad_u          complex [B,L,D] output; may alias grad_h
 *   grad_lambda     complex [D] or [B,L,D] output, or NULL to skip
 *   grad_h0         complex [B,D] output or NULL
 * grad_lambda for a per-channel lambda is reduced in a fixed order, so
 * repeated calls are bit-identical.
 */
memoroid_status_t memoroid_scan_diag_bwd(const void *lambda, int lambda_per_step,
                                         const uint8_t *start, const void *h0, const void *h,
                                         const void *grad_h, const void *grad_h_last, void *grad_u,
                                         void *grad_lambda, void *grad_h0, int64_t B, int64_t L,
                                         int64_t D, void *workspace, size_t workspace_bytes,
                                         void *stream);

/* ------------------------------------------------------------------------ */
/* Forward scan without a workspace argument (the paper has no counterpart:  */
/* this is a deployment convenience).                                        */
/* ------------------------------------------------------------------------ */

/* Size of the library-owned scratch array used by memoroid_scan_diag_fwd_static. */
#define MEMOROID_STATIC_WORKSPACE_BYTES (16u << 20)

/*
 * Same inputs, outputs and result as memoroid_scan_diag_fwd, for callers that
 * cannot provide device scratch memory (code running where device allocation
 * is unavailable or not allowed, e.g. inside an allocator callback or under a
 * framework that owns the whole device memory budget).  The scratch space is a
 * MEMOROID_STATIC_WORKSPACE_BYTES array in the library's own device memory,
 * held on every device that loads the library until the process exits; this
 * call allocates nothing.
 *   - The first call on a device looks up the array's address with that
 *     device current; make it outside any stream capture.
 *   - All calls share the array: calls that overlap on the GPU (other streams,
 *     or other host threads without ordering) race and give wrong results.
 *   - Shapes needing more than MEMOROID_STATIC_WORKSPACE_BYTES of workspace
 *     (memoroid_scan_diag_workspace_bytes) return MEMOROID_ERR_WORKSPACE.
 *   - A device-side wait that runs out is reported by
 *     memoroid_get_static_device_error (the array is not the caller's to read).
 *   - The array's address is cached per device; after cudaDeviceReset do not
 *     call this entry point on that device again in the same process.
 */
memoroid_status_t memoroid_scan_diag_fwd_static(const void *lambda, int lambda_per_step,
                                                const void *u, const uint8_t *start, const void *h0,
                                                void *h, void *h_last, int64_t B, int64_t L,
                                                int64_t D, void *stream);

/* Synchronises `stream`, then reads the error word that the last
 * memoroid_scan_diag_fwd_static call on the current device left in the
 * library-owned scratch array: MEMOROID_OK or MEMOROID_ERR_TIMEOUT (the same
 * reading as memoroid_get_device_error gives for a caller's workspace). */
memoroid_status_t memoroid_get_static_device_error(void *stream);

/* ======================================================================== */
/* Decayed linear-attention memoroid: the Linear Transformer memoroid of    */
/* the appendix on rewriting sequence models as memoroids, with a decay and  */
/* reset by the begin flag through Theorem 3.2:                              */
/*   S_t = [b_t = 0] gamma_t S_{t-1} + k_t v_t^T,   y_t = S_t^T q_t          */
/* S_{-1} = S0 (NULL = 0).  No feature map and no normaliser: y is the raw   */
/* read-out of the state.                                                    */
/* ======================================================================== */

/* Workspace bytes for memoroid_scan_linattn_fwd and _bwd with this shape (0
 * for an unsupported shape).  dk == dv == D with D in {64, 128}; chunk in
 * {64, 128}.  The forward alone needs a few bytes per tile; the backward adds
 * a bf16 copy of grad_y and one bf16 D x D state per 128-step tile. */
size_t memoroid_scan_linattn_workspace_bytes(int64_t B, int64_t L, int64_t H, int64_t dk,
                                             int64_t dv, int64_t chunk);

/* Number of kernels one call launches for this shape (-1 if unsupported);
 * with_dgamma_per_head: a backward call with a per-head gamma and dgamma. */
int memoroid_scan_linattn_kernels_per_call(int64_t B, int64_t L, int64_t H, int64_t dk,
                                           int64_t dv, int backward, int with_dgamma_per_head);

/*
 * Forward pass.
 *   q, k        bf16 [B, L, H, dk]   (in_dtype must be MEMOROID_BF16)
 *   v           bf16 [B, L, H, dv]
 *   gamma       fp32 [H] (gamma_per_step = 0) or [B, L, H]; the decay applied
 *               to S_{t-1} at step t, ignored at start steps.  Values are
 *               used through log2(gamma), clamped to [-126, 0]: a decay
 *               above 1 acts as 1, one below 2^-126 (0 included) as 2^-126.
 *   start       uint8 [B, L], nonzero = b_t (first step of an episode)
 *   S0          fp32 [B, H, dk, dv] or NULL
 *   y           fp32 [B, L, H, dv] output
 *   S_last      fp32 [B, H, dk, dv] output (the state after step L-1) or NULL
 * All arrays are row-major, contiguous device memory owned by the caller;
 * q, k, v, S0, y and S_last must be 16-byte aligned, the workspace 256-byte
 * aligned and at least memoroid_scan_linattn_workspace_bytes.  `chunk` is the
 * block size of the chunked evaluation; 64 and 128 compute the same function
 * (the kernels tile the tape by 128 steps, the tensor-core M, for both).
 * Asynchronous on `stream`; argument errors return at once, device-side wait
 * timeouts are read with memoroid_get_device_error(workspace).
 */
memoroid_status_t memoroid_scan_linattn_fwd(const void *q, const void *k, const void *v,
                                            int in_dtype, const float *gamma, int gamma_per_step,
                                            const uint8_t *start, const float *S0, float *y,
                                            float *S_last, int64_t B, int64_t L, int64_t H,
                                            int64_t dk, int64_t dv, int64_t chunk, void *workspace,
                                            size_t workspace_bytes, void *stream);

/*
 * Backward pass of memoroid_scan_linattn_fwd (same inputs).  With
 * dS_t = dL/dS_t accumulated backwards,
 *   dS_t = q_t dy_t^T + [b_{t+1} = 0] gamma_{t+1} dS_{t+1},  dS_{L-1} += grad_S_last
 *   dq_t = S_t dy_t,  dk_t = dS_t v_t,  dv_t = dS_t^T k_t,
 *   dgamma_t = [b_t = 0] <dS_t, S_{t-1}>_F,  dS0 = [b_0 = 0] gamma_0 dS_0.
 *   grad_y       fp32 [B, L, H, dv]
 *   grad_S_last  fp32 [B, H, dk, dv] or NULL (= 0)
 *   dq, dk, dv   fp32 [B, L, H, dk|dv] outputs (all three required)
 *   dgamma       fp32 [H] (per-head gamma: summed over B and L) or [B, L, H]
 *                (per-step gamma; 0 at start steps), or NULL to skip
 *   dS0          fp32 [B, H, dk, dv] output or NULL
 * q, k, v are consumed as bf16 and grad_y is rounded to bf16 for the tensor
 * cores; all accumulation is fp32.  Every reduction has a fixed order, so
 * repeated calls are bit-identical.  Workspace: at least
 * memoroid_scan_linattn_workspace_bytes.
 */
memoroid_status_t memoroid_scan_linattn_bwd(const void *q, const void *k, const void *v,
                                            int in_dtype, const float *gamma, int gamma_per_step,
                                            const uint8_t *start, const float *S0,
                                            const float *grad_y, const float *grad_S_last,
                                            float *dq, float *dk_out, float *dv_out, float *dgamma,
                                            float *dS0, int64_t B, int64_t L, int64_t H, int64_t dk,
                                            int64_t dv, int64_t chunk, void *workspace,
                                            size_t workspace_bytes, void *stream);

/* ======================================================================== */
/* The Linear Transformer memoroid with its feature map and normalizer      */
/* (appendix "Linear Transformer"): (X, x) . (X', x') = (X + X', x + x'),   */
/* f(o) = (phi(k) v^T, phi(k)), y = X^T phi(q) / (x^T phi(q)),              */
/* phi(z) = 1 + ELU(z); the pair is decayed by gamma_t like the decayed     */
/* memoroid above (gamma = 1 is the paper's model) and reset at begin       */
/* flags.  Heads of width d in {8, 16, ..., 120}; q, k, v bf16.            */
/* ======================================================================== */

/* Workspace bytes for memoroid_linattn_norm_fwd/_bwd (0 for a bad shape). */
size_t memoroid_linattn_norm_workspace_bytes(int64_t B, int64_t L, int64_t H, int64_t d);

/* Kernel launches of one call (with_states: all optional state arguments given). */
int memoroid_linattn_norm_kernels_per_call(int64_t B, int64_t L, int64_t H, int64_t d, int backward,
                                           int with_dgamma_per_head, int with_states);

/*
 *   q, k, v  bf16 [B, L, H, d] (16-byte aligned); gamma fp32 [H] or
 *            [B, L, H] (gamma_per_step); start uint8 [B, L]
 *   S0, z0   fp32 [B, H, d, d] and [B, H, d]: the pair (X, x) before step 0
 *            of rows with start[b][0] = 0, or NULL (= 0)
 *   y        fp32 [B, L, H, d] output; den fp32 [B, L, H] output x^T phi(q)
 *            (needed by the backward), or NULL
 *   S_last, z_last  the pair after the last step, or NULL
 * An empty call (B, L or H = 0) copies S0 / z0 to S_last / z_last (the
 * backward: grad_S_last / grad_z_last to dS0 / dz0, dgamma = 0).  Workspace
 * 256-byte aligned, at least memoroid_linattn_norm_workspace_bytes; its
 * header reports device-side waits through memoroid_get_device_error.
 */
memoroid_status_t memoroid_linattn_norm_fwd(const void *q, const void *k, const void *v,
                                            const float *gamma, int gamma_per_step,
                                            const uint8_t *start, const float *S0, const float *z0,
                                            float *y, float *den, float *S_last, float *z_last,
                                            int64_t B, int64_t L, int64_t H, int64_t d,
                                            void *workspace, size_t workspace_bytes, void *stream);

/*
 * Backward: y and den are the forward's outputs; grad_y fp32 [B, L, H, d];
 * grad_S_last / grad_z_last or NULL; outputs dq, dk, dv fp32 [B, L, H, d]
 * (16-byte aligned; B * L * H * d < 2^32),
 * dgamma ([H] summed, or [B, L, H]; NULL to skip), dS0 / dz0 or NULL.
 */
memoroid_status_t memoroid_linattn_norm_bwd(const void *q, const void *k, const void *v,
                                            const float *gamma, int gamma_per_step,
                                            const uint8_t *start, const float *S0, const float *z0,
                                            const float *y, const float *den, const float *grad_y,
                                            const float *grad_S_last, const float *grad_z_last,
                                            float *dq, float *dk, float *dv, float *dgamma,
                                            float *dS0, float *dz0, int64_t B, int64_t L, int64_t H,
                                            int64_t d, void *workspace, size_t workspace_bytes,
                                            void *stream);

/* ======================================================================== */
/* Fast and Forgetful Memory memoroid (appendix "Fast and Forgetful         */
/* Memory"): (X, t) . (X', t') = (X (.) exp(t'(-|alpha| (+) i omega)) + X', */
/* t + t') with f(o, b) = (x~ repeated over the c columns, 1), made         */
/* resettable by Theorem 3.2.  With t' = 1 per step this is, per state      */
/* entry (i, j),                                                            */
/*   X_t[i,j] = [b_t = 0] lambda_ij X_{t-1}[i,j] + x~_t[i],                  */
/*   lambda_ij = exp(-|alpha_i| + i omega_j),                               */
/* the diagonal scan over D = m*c complex channels (channel i*c + j).  The  */
/* output is the cell's readout input Re(X_t) || Im(X_t), each flattened.   */
/* Shapes: m % 4 == 0, c in {1, 2, 4, 8, 16}.                               */
/* ======================================================================== */

/* Workspace bytes for memoroid_ffm_fwd and memoroid_ffm_bwd (0 for an
 * unsupported shape). */
size_t memoroid_ffm_workspace_bytes(int64_t B, int64_t L, int64_t m, int64_t c);

/* Kernel launches of one call (-1 for an unsupported shape). */
int memoroid_ffm_kernels_per_call(int64_t B, int64_t L, int64_t m, int64_t c, int backward,
                                  int with_param_grads);

/*
 *   x      fp32 [B, L, m]: the cell's gated input x~_t (16-byte aligned)
 *   alpha  fp32 [m] decay parameters (|alpha| is used), omega fp32 [c]
 *   start  uint8 [B, L], nonzero = first step of an episode
 *   S0     complex64 [B, m, c]: state before step 0 of rows with start[b][0]
 *          = 0, or NULL (= 0)
 *   z      fp32 [B, L, 2*m*c] output: Re(X_t) then Im(X_t), row-major (i, j)
 *   S_last complex64 [B, m, c] output, or NULL
 * Device memory owned by the caller; workspace 256-byte aligned, at least
 * memoroid_ffm_workspace_bytes; asynchronous on `stream`.  Errors:
 * INVALID_ARG (shape, NULL or misaligned pointer), WORKSPACE, CUDA; a
 * look-back wait that runs out is reported by memoroid_get_device_error.
 */
memoroid_status_t memoroid_ffm_fwd(const float *x, const float *alpha, const float *omega,
                                   const uint8_t *start, const void *S0, float *z, void *S_last,
                                   int64_t B, int64_t L, int64_t m, int64_t c, void *workspace,
                                   size_t workspace_bytes, void *stream);

/*
 * Backward of memoroid_ffm_fwd (PyTorch's complex-gradient convention for
 * S0 / S_last: grad = dL/dRe + i dL/dIm).
 *   z           the forward's output; grad_z fp32 [B, L, 2*m*c] = dL/dz
 *   grad_S_last complex64 [B, m, c] or NULL
 *   grad_x      fp32 [B, L, m] output: sum over j of Re(delta_t[i, j])
 *   grad_alpha  fp32 [m], grad_omega fp32 [c]: sums over B and L (either may
 *               be NULL); the order of every reduction is fixed
 *   grad_S0     complex64 [B, m, c] or NULL
 */
memoroid_status_t memoroid_ffm_bwd(const float *alpha, const float *omega, const uint8_t *start,
                                   const void *S0, const float *z, const float *grad_z,
                                   const void *grad_S_last, float *grad_x, float *grad_alpha,
                                   float *grad_omega, void *grad_S0, int64_t B, int64_t L,
                                   int64_t m, int64_t c, void *workspace, size_t workspace_bytes,
                                   void *stream);

/* ======================================================================== */
/* Tape-based batching, sampling (Algorithm 2 "Sampling transitions using   */
/* TBB"): starting from an empty batch, append the episode                 */
/* D[I[i] : I[i+1]] of a drawn index i while the batch is shorter than B,   */
/* then cut it to B transitions.  The draws are an input (the caller's      */
/* generator), so the batch is a pure function of (I, N, draws, B).  The    */
/* episode of the last index runs to the end of the buffer (I[E] = N).      */
/* ======================================================================== */

/* Workspace bytes for memoroid_tbb_sample with up to K draws (also enough
 * for memoroid_gather_rows, which needs the 256-byte header only). */
size_t memoroid_tbb_workspace_bytes(int64_t K);

/*
 *   begin   int64 [E]: the index list I, increasing, into a buffer of N
 *           transitions (episode i is [begin[i], begin[i+1]), the last one
 *           [begin[E-1], N))
 *   draws   int64 [K]: the drawn episode indices, in draw order
 *   start   uint8 [B] output: 1 where an appended episode begins in the batch
 *   src     int64 [B] output: buffer index of the transition at each step
 *   n_used  int64 [1] output (device), or NULL: the draws used (the fewest
 *           that fill B steps)
 * All device memory owned by the caller; asynchronous on `stream`.  Bad data
 * (an index outside [0, E), an empty episode, draws that do not fill B
 * steps; the uncovered steps get src = -1) is reported as
 * MEMOROID_ERR_BAD_DATA by memoroid_get_device_error(workspace).
 */
memoroid_status_t memoroid_tbb_sample(const int64_t *begin, int64_t E, int64_t N, const int64_t *draws,
                                      int64_t K, int64_t B, uint8_t *start, int64_t *src,
                                      int64_t *n_used, void *workspace, size_t workspace_bytes,
                                      void *stream);

/*
 * out[t] = rows[src[t]] for t in [0, B): rows is [N, row_bytes] (any row
 * size; 16-byte copies when row_bytes % 16 == 0 and both arrays are 16-byte
 * aligned), out is [B, row_bytes] and may not overlap rows.  A source index
 * outside [0, N) gives a zero row and MEMOROID_ERR_BAD_DATA from
 * memoroid_get_device_error(workspace).  Workspace: at least 256 bytes.
 */
memoroid_status_t memoroid_gather_rows(const void *rows, int64_t N, int64_t row_bytes,
                                       const int64_t *src, int64_t B, void *out, void *workspace,
                                       size_t workspace_bytes, void *stream);

/* ======================================================================== */
/* Discounted return and GAE memoroids (appendices "The Discounted Return   */
/* as a Memoroid" and "The Generalized Advantage Estimate as a Memoroid"):  */
/* (a, r) . (a', r') = (a a', a r' + r), evaluated for every step of every  */
/* episode of the tape, i.e. the reverse recurrences                        */
/*   G_t = r_t + gamma [b_{t+1} = 0] G_{t+1}                                */
/*   A_t = delta_t + gamma lambda [b_{t+1} = 0] A_{t+1},                    */
/*   delta_t = r_t + gamma V_{t+1} - V_t,                                   */
/* where V_{t+1} is 0 after an episode's last step and the tape's last step */
/* continues into boot / v_boot when given (a cut episode).                 */
/* ======================================================================== */

/* Workspace bytes for memoroid_discounted_return and memoroid_gae (a small
 * block: a header and one affine map per range of a tape, about 152 KB; a
 * call clears the header and launches one kernel, and keeps nothing in it
 * afterwards). */
size_t memoroid_returns_workspace_bytes(int64_t B, int64_t L);

/*
 *   r      fp32 [B, L] rewards
 *   start  uint8 [B, L], nonzero = first step of an episode
 *   boot   fp32 [B]: the return after each tape's last step, or NULL (= 0)
 *   G      fp32 [B, L] output (may not alias r)
 * Device memory owned by the caller; workspace 256-byte aligned, at least
 * memoroid_returns_workspace_bytes.  Asynchronous on `stream`.
 */
memoroid_status_t memoroid_discounted_return(const float *r, const uint8_t *start, float gamma,
                                             const float *boot, float *G, int64_t B, int64_t L,
                                             void *workspace, size_t workspace_bytes, void *stream);

/*
 *   r, v   fp32 [B, L] rewards and values V(s_t)
 *   v_boot fp32 [B]: V of the state after each tape's last step, or NULL (= 0)
 *   A      fp32 [B, L] output (may not alias r or v)
 */
memoroid_status_t memoroid_gae(const float *r, const float *v, const uint8_t *start, float gamma,
                               float lambda, const float *v_boot, float *A, int64_t B, int64_t L,
                               void *workspace, size_t workspace_bytes, void *stream);

/* ------------------------------------------------------------------------ */
/* Measurement only (the paper has no counterpart): throughput of the        */
/* intra-tile tensor-core contraction of memoroid_scan_linattn_fwd alone.    */
/* ------------------------------------------------------------------------ */

/* Scratch bytes for memoroid_bench_linattn_intra (0 if d is unsupported). */
size_t memoroid_bench_linattn_intra_scratch_bytes(int64_t d);

/*
 * Launches `ctas` CTAs; each stages one set of operand tiles taken from the
 * scratch bytes (their values are irrelevant) in shared memory and then
 * issues `reps` times the forward pass's two intra-tile contractions,
 * P = Q K^T (128 x 128 x d) and Y = Pm V (128 x d x 128), with the same
 * instruction shapes and operand layouts.  Executed flops: 4 * 128^2 * d per
 * rep and CTA.  Time it with events on `stream`.  scratch: device memory,
 * 256-byte aligned, at least memoroid_bench_linattn_intra_scratch_bytes(d).
 */
memoroid_status_t memoroid_bench_linattn_intra(int64_t d, int64_t reps, int64_t ctas, void *scratch,
                                               size_t scratch_bytes, void *stream);

/* ======================================================================== */
/* Episode index list <-> begin flags (Algorithm 1 keeps I = where(b)).     */
/* ======================================================================== */

/* start[t] = 1 for t in offsets[0..E), 0 elsewhere, t in [0, L).  Offsets
 * outside [0, L) are ignored.  offsets: int64 device array; start: uint8 [L]. */
memoroid_status_t memoroid_starts_from_offsets(const int64_t *offsets, int64_t E, int64_t L,
                                               uint8_t *start, void *stream);

/* Workspace bytes for memoroid_offsets_from_starts. */
size_t memoroid_offsets_workspace_bytes(int64_t L);

/* offsets[0..n) = increasing indices t with start[t] != 0; *count = n (int64,
 * device memory).  offsets must hold L entries. */
memoroid_status_t memoroid_offsets_from_starts(const uint8_t *start, int64_t L, int64_t *offsets,
                                               int64_t *count, void *workspace,
                                               size_t workspace_bytes, void *stream);

/* ======================================================================== */
/* Device-side error reporting and debug knobs.                             */
/* ======================================================================== */

/* Synchronises `stream`, then reads the error word that the last call using
 * `workspace` left there: MEMOROID_OK or MEMOROID_ERR_TIMEOUT. */
memoroid_status_t memoroid_get_device_error(const void *workspace, void *stream);

/* Process-wide limit for every bounded device-side wait, in nanoseconds
 * (0 restores the default of 1 s).  Applies to later calls. */
void memoroid_debug_set_wait_limit_ns(uint64_t ns);

/* Fault injection for tests (-1 = off, the default; applies to later calls):
 * in the diagonal scan the tile with this scheduling ticket skips publishing
 * its look-back status, so its successor's wait runs out; in the linear-
 * attention kernels the CTA with this index treats its first tensor-core wait
 * as timed out (it drains its in-flight work, records MEMOROID_ERR_TIMEOUT in
 * the workspace and stops). */
void memoroid_debug_withhold_tile(int64_t ticket);

/* Test knob (0 = off, the default; applies to later calls): the Linear
 * Transformer calls (memoroid_linattn_norm_*) always build padded operands in
 * separate kernels, instead of the in-kernel construction they use for
 * 64-channel heads; both compute the same bits. */
void memoroid_debug_lnorm_padded(int on);

#ifdef __cplusplus
}
#endif

#endif /* MEMOROID_H */
