/*
 * hla.h -- C ABI of the GB300 (sm_103a) implementation of Higher-order Linear
 * Attention (Zhang, Qin, Wang, Gu, "Higher-order Linear Attention").
 *
 * All entry points take plain pointers and sizes.  Device pointers refer to
 * memory of the current CUDA device; the caller owns every buffer (inputs,
 * outputs, states and the scratch workspace) and the library allocates no
 * device memory.  Work is enqueued asynchronously on `stream`; host-side
 * argument errors are returned synchronously before anything is launched.
 *
 * Common conventions
 * ------------------
 * Tokens are row vectors.  q, k are [B, H, n, d] and v, out are [B, H, n, dv],
 * contiguous, in the element type `dt` (out has the same type as the inputs).
 * Base pointers must be 16-byte aligned.
 *
 * Second-order state of one head (fp32, row-major), the tuple of Fig. 1(A):
 *   [ S (d*d) | C (d*dv) | m (d) | G (d*dv) | h (d) ]
 * with S = sum k k^T, C = sum q v^T, m = sum q, G = sum_i k_i k_i^T C_{i-1},
 * h = sum_i k_i k_i^T m_{i-1} (Sec. 3 and Sec. 3.2).  States of B*H heads are
 * stored back to back in [B, H] order.  With masked = 0 the operator does not
 * use G and h: they are ignored on input and written as zeros on output.
 *
 * Supported shapes: d, dv in {16, 32, 64, 128}; 1 <= chunk <= 128 (chunk is
 * the scan granularity of Theorem 2; the result does not depend on it up to
 * rounding); n >= 0 with any remainder n % chunk (a ragged last chunk).
 * Other values return HLA_ERR_UNSUPPORTED.
 */
#ifndef HLA_H_
#define HLA_H_

#include <stddef.h>

#ifdef __cplusplus
extern "C" {
#endif

struct CUstream_st;
/* A CUDA stream (the same object as cudaStream_t); NULL is the legacy default stream. */
typedef struct CUstream_st *hla_stream_t;

typedef enum {
    HLA_OK = 0,
    HLA_ERR_INVALID_ARGUMENT = 1, /* null pointer, negative size, misaligned pointer, bad flag */
    HLA_ERR_UNSUPPORTED = 2,      /* valid request outside the supported shapes/types        */
    HLA_ERR_CUDA = 3,             /* a CUDA runtime call or kernel launch failed              */
    HLA_ERR_TIMEOUT = 4,          /* a device-side wait ran past its budget (hla_poll_error)  */
    HLA_ERR_WORKSPACE = 5         /* workspace missing or smaller than the required size      */
} hla_status;

typedef enum {
    HLA_F32 = 0,  /* IEEE float32 tokens */
    HLA_BF16 = 1  /* bfloat16 tokens (fp32 accumulation everywhere) */
} hla_dtype;

/* Human-readable name of a status code (static storage). */
const char *hla_status_string(hla_status status);

/* Detail of the last error returned on the calling host thread (static,
 * thread-local storage; empty string if none). */
const char *hla_last_error(void);

/* Number of floats of one head's second-order state tuple: d*d + 2*d*dv + 2*d. */
size_t hla2_state_floats(int d, int dv);

/* Bytes of scratch workspace hla2_forward needs for these sizes (any flags).
 * Returns 0 for unsupported sizes. */
size_t hla2_workspace_bytes(int B, int H, int n, int d, int dv, int chunk, hla_dtype dt);

/*
 * hla2_forward -- chunk-parallel forward of second-order HLA over n tokens.
 *
 * Operator (per head, t = 1..n):
 *   masked = 1 (strictly causal, Theorem 1, Eq. masked-unnorm / Eq. masked):
 *     num_t = q_t^T (S_t C_t - G_t),   den_t = q_t^T (S_t m_t - h_t)
 *     = sum_{j<=t} sum_{i<=j} (q_t.k_i)(q_j.k_i) v_j   (and v_j -> 1 for den)
 *   masked = 0 (Eq. hla-unnorm / Eq. hla-row):
 *     num_t = q_t^T S_t C_t,           den_t = q_t^T S_t m_t
 *   out_t = num_t                       if normalized == 0 (the default operator)
 *   out_t = num_t / (den_t + eps)       if normalized == 1 (no clamp, no abs)
 * where the states include token t (inclusive) and start from state_in.  The
 * result equals the serial recurrence (online updates after Theorem 1) by
 * Theorem 2; chunking only changes rounding.
 *
 * q, k, v : device, [B, H, n, d] / [B, H, n, d] / [B, H, n, dv] of type dt (read only)
 * out     : device, [B, H, n, dv] of type dt (written)
 * state_in  : device fp32 [B*H * hla2_state_floats(d,dv)] or NULL (= zero state)
 * state_out : device fp32, same size, or NULL (= not written); receives the
 *             state after token n (Eq. semidirect applied to the whole
 *             sequence).  May equal state_in (read before written).
 * eps     : the stability constant of the normalised output (finite)
 * workspace / workspace_bytes : device scratch of at least
 *             hla2_workspace_bytes(B,H,n,d,dv,chunk,dt) bytes, 256-byte
 *             aligned; its contents on entry are ignored.  Calls that share a
 *             workspace must be ordered on one stream.
 * Errors: HLA_ERR_INVALID_ARGUMENT / UNSUPPORTED / WORKSPACE before launch;
 * HLA_ERR_CUDA if a launch fails.  A device-side wait that exceeds its budget
 * sets a flag in the workspace that hla_poll_error reports as HLA_ERR_TIMEOUT.
 */
hla_status hla2_forward(const void *q, const void *k, const void *v, void *out, hla_dtype dt,
                        int B, int H, int n, int d, int dv, int masked, int normalized, float eps,
                        int chunk, const float *state_in, float *state_out,
                        void *workspace, size_t workspace_bytes, hla_stream_t stream);

/*
 * hla2_step -- one streaming decode step of second-order HLA for B*H heads.
 *
 * For each head, with the state tuple (S, C, m, G, h) before the token
 * (online updates after Theorem 1; outputs of Theorem 1 / Eq. hla-row):
 *   masked:  G += k (k^T C),  h += k (k^T m)          (previous C and m)
 *   S += k k^T,  C += q v^T,  m += q
 *   masked:   num = (q^T S) C - q^T G,  den = (q^T S) m - q^T h
 *   unmasked: num = (q^T S) C,          den = (q^T S) m   (G, h untouched)
 *   out = num, or num / (den + eps) if normalized.
 *
 * q, k : device [B, H, d] of type dt; v : device [B, H, dv] of type dt
 * out  : device [B, H, dv] of type dt
 * state: device fp32 [B*H * hla2_state_floats(d,dv)], updated in place
 * Errors as for hla2_forward (no workspace, no device-side waits).
 */
hla_status hla2_step(const void *q, const void *k, const void *v, void *out, hla_dtype dt,
                     int B, int H, int d, int dv, int masked, int normalized, float eps,
                     float *state, hla_stream_t stream);

/* Bytes of scratch workspace hla2_backward needs (0 if unsupported). */
size_t hla2_backward_workspace_bytes(int B, int H, int n, int d, int dv, int chunk, hla_dtype dt);

/*
 * hla2_backward -- gradients of the masked second-order forward (from a zero
 * state) for L = sum_t dout_t . out_t: dq, dk, dv.  The paper's training
 * route (Sec. "Chunk-parallel training via associative scans"): the forward
 * prefixes are checkpointed at chunk boundaries and recomputed within a
 * chunk, and the gradient suffixes are carried by a reverse scan with the
 * adjoint of the semidirect product (Eq. semidirect); the result equals the
 * gradients of the serial recurrence (Theorem 2 and the chain rule) up to
 * rounding.  normalized selects out = num / (den + eps) (Eq. masked).
 * q, k, v : device [B, H, n, d] / [B, H, n, d] / [B, H, n, dv] of type dt
 * dout    : device [B, H, n, dv] of type dt (the gradient of the output)
 * dq, dk  : device [B, H, n, d] of type dt (written); dv : [B, H, n, dv] (written)
 * workspace : at least hla2_backward_workspace_bytes(...) bytes, 256-byte aligned.
 * Errors as for hla2_forward.
 */
hla_status hla2_backward(const void *q, const void *k, const void *v, const void *dout, void *dq, void *dk,
                         void *dv, hla_dtype dt, int B, int H, int n, int d, int dv_size, int normalized,
                         float eps, int chunk, void *workspace, size_t workspace_bytes, hla_stream_t stream);

/*
 * The (S, D, e) decode state of the masked operator (no counterpart printed in
 * the paper; it follows from Theorem 1 and Eq. semidirect).  With
 * D = S C - G (d x dv) and e = S m - h (d), Theorem 1's outputs read
 * num_t = q_t^T D_t and den_t = q_t^T e_t, and the online updates after
 * Theorem 1 collapse to
 *   S' = S + k k^T,   x = S' q,   D' = D + x v^T,   e' = e + x.
 * Per head (fp32, row-major): [ S (d*d) | D (d*dv) | e (d) ], heads in [B, H]
 * order.  It carries exactly what the masked outputs need with d*d + d*dv + d
 * floats instead of the tuple's d*d + 2*d*dv + 2*d (a third fewer bytes per
 * decode step at d = dv); the tuple cannot be recovered from it (C, m, G, h
 * are folded together).  This is one of the state-format options of the
 * paper's implementation considerations (Sec. "Implementation details and
 * complexity").
 */
size_t hla2_sde_state_floats(int d, int dv);

/*
 * hla2_state_to_sde -- convert B*H masked second-order tuples (S, C, m, G, h)
 * (hla2_state_floats each, e.g. a state_out of hla2_forward) into (S, D, e)
 * states: D = S C - G, e = S m - h, fp32 on the device.
 * state : device fp32 [B*H * hla2_state_floats(d,dv)] (read only)
 * sde   : device fp32 [B*H * hla2_sde_state_floats(d,dv)] (written); must not
 *         overlap state.  Both 16-byte aligned.
 * Errors: HLA_ERR_INVALID_ARGUMENT (null, misaligned, overlapping),
 * HLA_ERR_UNSUPPORTED (d, dv outside {16, 32, 64, 128}), HLA_ERR_CUDA.
 */
hla_status hla2_state_to_sde(const float *state, float *sde, int B, int H, int d, int dv, hla_stream_t stream);

/*
 * hla2_step_sde -- hla2_step of the masked operator on (S, D, e) states:
 *   S += k k^T;  x = S q;  D += x v^T;  e += x;
 *   num = q^T D,  den = q^T e,  out = num or num / (den + eps).
 * q, k : device [B, H, d] of type dt; v, out : device [B, H, dv] of type dt
 * sde  : device fp32 [B*H * hla2_sde_state_floats(d,dv)], updated in place
 * Errors as for hla2_step.
 */
hla_status hla2_step_sde(const void *q, const void *k, const void *v, void *out, hla_dtype dt,
                         int B, int H, int d, int dv, int normalized, float eps,
                         float *sde, hla_stream_t stream);

/*
 * hla2_forward_path -- which CUDA path hla2_forward takes for these arguments
 * on the current device, without launching anything:
 *   0  generic path: fp32 CUDA-core kernels (every supported shape);
 *   1  fused path: one persistent tcgen05/TMA kernel (bf16 tokens, d and dv
 *      in {64, 128}; masked: state_in only with d = dv = 128; unmasked: the
 *      plain output, no states, one SM per head) on sm_103, plus two small kernels for
 *      state_out (C = Q^T V and m = Q^T 1 on the tensor cores, then
 *      G = S C - D, h = S m - e from the forward's prefixes).  It works in
 *      128-token tiles whatever chunk is (chunk only changes the rounding,
 *      Theorem 2);
 *  -1  the arguments are not supported.
 * *launches (if not NULL) receives the number of kernels the call launches.
 */
int hla2_forward_path(int B, int H, int n, int d, int dv, int masked, int normalized, int chunk, hla_dtype dt,
                      int has_state_in, int has_state_out, int *launches);

/* Number of floats of one head's third-order state tuple (Theorem 3):
 * [ SK d*d | SQ d*d | P d*dv | mK d | G1 d*dv | G2 d*dv | G3 d*dv | h1 d | h2 d | h3 d ]. */
size_t hla3_state_floats(int d, int dv);

/* Bytes of scratch workspace hla3_forward needs (0 if unsupported). */
size_t hla3_workspace_bytes(int B, int H, int n, int d, int dv, int chunk, hla_dtype dt);

/*
 * hla3_forward -- forward of third-order HLA (Sec. 7).
 *
 *   masked = 1 (Theorem 3, Algorithm 3 at gamma = 1):
 *     num_t = q_t^T (S^K_t S^Q_t P^KV_t - G1_t - G2_t - G3_t)
 *     den_t = q_t^T (S^K_t S^Q_t m^K_t  - h1_t - h2_t - h3_t)
 *   masked = 0: num_t = q_t^T S^K_t S^Q_t P^KV_t, den_t = q_t^T S^K_t S^Q_t m^K_t
 *   out_t = num_t, or num_t / (den_t + eps) if normalized.
 * Arguments as for hla2_forward, with the third-order state layout.
 */
hla_status hla3_forward(const void *q, const void *k, const void *v, void *out, hla_dtype dt,
                        int B, int H, int n, int d, int dv, int masked, int normalized, float eps,
                        int chunk, const float *state_in, float *state_out,
                        void *workspace, size_t workspace_bytes, hla_stream_t stream);

/*
 * hla3_forward_path -- which CUDA path hla3_forward takes for these arguments on
 * the current device, without launching anything: 2 the tensor-core kernels
 * (fp32 tokens, d = dv = 32, masked = 1, normalized = 0, no states, an sm_103
 * device), 1 the chunk-parallel fp32 kernels, 0 the serial kernel, -1 the
 * arguments are not supported.  *launches (if not null) receives the number of
 * kernel launches of one call (0 when B*H = 0).
 */
int hla3_forward_path(int B, int H, int n, int d, int dv, int masked, int normalized, int chunk, hla_dtype dt,
                      int has_state_in, int has_state_out, int *launches);

/*
 * hla2_backward_path -- which CUDA path hla2_backward takes for these arguments
 * on the current device, without launching anything: 1 the tensor-core kernel
 * (bf16 tokens, d = dv = 64, normalized = 0, an sm_103 device; one launch),
 * 0 the fp32 CUDA-core kernels (five launches), -1 the arguments are not
 * supported.
 */
int hla2_backward_path(int B, int H, int n, int d, int dv, int normalized, int chunk, hla_dtype dt);

/*
 * hla2_forward_noalloc -- hla2_forward for callers that cannot allocate device
 * memory (no counterpart in the paper: it only changes where scratch lives).
 *
 * Some callers cannot call cudaMalloc or hand over a workspace: code that runs
 * under an allocator it does not own (a framework's caching pool, a memory
 * budget that forbids extra reservations), or host code that links this
 * library without any device-memory management of its own.  This entry point
 * computes exactly what hla2_forward computes (same arguments, minus the
 * workspace and state_out) and allocates nothing: its scratch is a 16 MiB
 * array in device memory that belongs to the library.  Every GPU on which the
 * library is used holds that array until the process exits.
 *
 * Scope: the arguments for which hla2_forward_path returns 1 without a final
 * state (the fused path: bf16 tokens, d and dv in {64, 128}, masked = 1,
 * state_in only with d = dv = 128, an sm_103 device); other arguments return
 * HLA_ERR_UNSUPPORTED.  Sizes whose scratch exceeds 16 MiB (it grows with
 * B*H, about 263 KiB per head, and with B*H*n*4 bytes when normalized) return
 * HLA_ERR_WORKSPACE before anything is launched.
 * Set-up: the first call on a device looks up the array's device address
 * (cudaGetSymbolAddress) with that device current; make that first call before
 * any stream capture.
 * Sharing: all calls use the same array and it keeps the last call's contents
 * (each call clears what must start at zero).  Calls whose kernels overlap on
 * the GPU (different streams, or several host threads) race on it: order them
 * on one stream.  A device-side wait that exceeds its budget sets the error
 * word at the start of the array; hla_poll_error_noalloc reads it.
 * An empty problem (B*H = 0 or n = 0) returns HLA_OK without launching.
 */
hla_status hla2_forward_noalloc(const void *q, const void *k, const void *v, void *out, hla_dtype dt,
                                int B, int H, int n, int d, int dv, int masked, int normalized, float eps,
                                int chunk, const float *state_in, hla_stream_t stream);

/*
 * Asymmetric second-order HLA (AHLA), Sec. "Asymmetric Higher-order Linear
 * Attention".  The operator is always causal:
 *   o_t = sum_{j<=t} sum_{i=j..t} (q_t.k_i)(q_i.k_j) v_j   (Eq. AHLA-explicit),
 * computed as q_t^T E_t with the streaming state of Theorem AHLA:
 *   P_t = P_{t-1} + k_t v_t^T,  m_t = m_{t-1} + k_t,
 *   E_t = E_{t-1} + k_t (q_t^T P_t),  n_t = n_{t-1} + k_t (q_t^T m_t),
 *   out_t = q_t^T E_t, or q_t^T E_t / (q_t^T n_t + eps) if normalized.
 * State of one head (fp32, row-major): [ P (d*dv) | m (d) | E (d*dv) | n (d) ].
 */
size_t ahla_state_floats(int d, int dv);

/* Bytes of scratch workspace ahla_forward needs (0 if unsupported). */
size_t ahla_workspace_bytes(int B, int H, int n, int d, int dv, int chunk, hla_dtype dt);

/*
 * ahla_forward -- chunk-parallel AHLA forward: chunk summaries composed with
 * the AHLA semidirect product (Eq. AHLA-semidirect, with the segment cross
 * moment R^KQ = sum k q^T of the later segment), which reproduces the serial
 * recurrence (scan equivalence); chunk is the scan granularity (results do not
 * depend on it up to rounding).  Arguments, layouts, shapes and errors as for
 * hla2_forward (no masked flag), with the AHLA state layout for state_in /
 * state_out (state_out may equal state_in).  bf16 tokens with d and dv in
 * {64, 128}, the plain output and no states run on the tensor cores (one
 * persistent tcgen05 kernel sweeping each head's 128-token tiles with the P
 * and E carries in tensor memory); every other call runs three fp32 kernels.
 * A device-side wait that exceeds its budget sets the flag hla_poll_error reads.
 */
hla_status ahla_forward(const void *q, const void *k, const void *v, void *out, hla_dtype dt,
                        int B, int H, int n, int d, int dv, int normalized, float eps, int chunk,
                        const float *state_in, float *state_out,
                        void *workspace, size_t workspace_bytes, hla_stream_t stream);

/*
 * ahla_forward_path -- which CUDA path ahla_forward takes for these arguments on
 * the current device, without launching anything: 1 the tensor-core kernel,
 * 0 the fp32 kernels, -1 the arguments are not supported.
 */
int ahla_forward_path(int B, int H, int n, int d, int dv, int normalized, int chunk, hla_dtype dt, int has_state_in,
                      int has_state_out);

/*
 * ahla_step -- one AHLA decode step for B*H heads (the online updates of
 * Theorem AHLA; Algorithm AHLA-stream at gamma = 1): q, k [B, H, d], v, out
 * [B, H, dv] of type dt; state fp32 [B*H * ahla_state_floats(d,dv)], updated
 * in place.  Errors as for hla2_step.
 */
hla_status ahla_step(const void *q, const void *k, const void *v, void *out, hla_dtype dt,
                     int B, int H, int d, int dv, int normalized, float eps,
                     float *state, hla_stream_t stream);

/*
 * hla_poll_error_noalloc -- hla_poll_error for hla2_forward_noalloc (no
 * counterpart in the paper): waits for `stream`, then reports and clears the
 * device-side error word of the library's scratch array on the current device:
 * HLA_OK, or HLA_ERR_TIMEOUT if a device-side wait of the last no-alloc call
 * gave up.  Returns HLA_ERR_CUDA if synchronisation or the read fails.
 */
hla_status hla_poll_error_noalloc(hla_stream_t stream);

/*
 * hla_poll_error -- wait for `stream`, then report the device-side error flag
 * kept in `workspace` by the last forward call that used it: HLA_OK, or
 * HLA_ERR_TIMEOUT if a device-side wait gave up.  Clears the flag.
 * Returns HLA_ERR_CUDA if synchronisation or the read fails.
 */
hla_status hla_poll_error(void *workspace, hla_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* HLA_H_ */
