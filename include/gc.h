/*
 * gc.h -- C ABI of the GB300 gradient-coding library (libgc.so).
 *
 * Implements the data-parallel hot path of the partial-straggler
 * gradient-coding protocol of "Leveraging partial stragglers within gradient
 * coding" (Ramamoorthy, Meng, Girimaji): chunk gradients (Sec. I), the
 * encoding coefficients of Algorithm 1, worker encoding (eq. 2), PS decoding
 * (Sec. II-B), batched over many straggler patterns, and the error measures
 * of Sec. II-A / Sec. IV.  Workers and the PS are simulated on one device.
 *
 * Notation: N chunks, m workers, delta chunks per worker (load), ell the
 * communication factor, d the parameter dimension, L = ceil(d / ell) the block
 * length, n_c points per chunk, N~ = N * n_c, npat straggler patterns.
 *
 * Conventions shared by every entry point
 *  - Return value: GC_OK (0) or a negative GC_ERR_* code.  On error,
 *    gc_last_error() returns a thread-local message.  No C++ exception
 *    crosses this boundary.
 *  - Ownership: every buffer belongs to the caller.  The library never
 *    allocates device or host memory and never frees caller memory.
 *    Pointers without the _h suffix are DEVICE pointers; *_h are host pointers.
 *  - Scratch: an entry point that needs scratch takes (ws, ws_bytes), a
 *    device buffer of at least the size its gc_*_workspace() function
 *    returns, 256-byte aligned.  The first 256 bytes are a status header
 *    that kernels set when they detect bad data on the device (a psi entry
 *    outside [0, delta], a rank-deficient least-squares system, a bounded
 *    wait that expired).  The header is sticky: it must be zeroed once
 *    before first use (gc_workspace_init) and is read and cleared by
 *    gc_status().
 *  - Streams: `stream` is a cudaStream_t (NULL = legacy default stream).
 *    All device entry points are asynchronous on it; gc_make_assignment is
 *    host-only and synchronous.
 *  - Layouts are row-major and dense unless stated.
 *  - Validation of sizes and pointers happens on the host before any
 *    launch; nothing is launched when a check fails.
 */
#ifndef GC_H_
#define GC_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes ---------------------------------------------------- */
#define GC_OK 0
#define GC_ERR_ARG (-1)         /* null pointer, out-of-range enum or scalar */
#define GC_ERR_SHAPE (-2)       /* inconsistent or out-of-range sizes        */
#define GC_ERR_UNSUPPORTED (-3) /* valid but not supported (ell > 8, delta > 32, ...) */
#define GC_ERR_CUDA (-4)        /* a CUDA runtime call failed                */
#define GC_ERR_TIMEOUT (-5)     /* a bounded device wait expired             */
#define GC_ERR_WORKSPACE (-6)   /* workspace missing, too small or misaligned */
#define GC_ERR_DATA (-7)        /* device-detected bad data (see gc_status)   */

/* ---- enums ----------------------------------------------------------- */
#define GC_CYCLIC 0   /* W_j holds chunks j, j+1, ..., j+delta-1 (mod N)   */
#define GC_EXPLICIT 1 /* orders given by the caller                        */

#define GC_F32 0  /* X element type: float32                              */
#define GC_BF16 1 /* X element type: bfloat16                             */

#define GC_LSQ 0      /* l = (x^T w - y)^2 / 2                             */
#define GC_LOGISTIC 1 /* l = log(1 + exp(-y x^T w)), y in {-1, +1}          */

/* Limits of this build. */
#define GC_MAX_ELL 8      /* communication factor ell                        */
#define GC_MAX_DELTA 32   /* chunks per worker                               */
#define GC_MAX_REPL 32    /* copies of one chunk in the cluster (gamma_i)    */

/* ---- library ---------------------------------------------------------- */
/* Thread-local text of the last error raised on this thread ("" if none). */
const char* gc_last_error(void);

/* Version as 10000*major + 100*minor + patch. */
int gc_version(void);

/* Number of CUDA kernels this library has launched since it was loaded
 * (launches recorded into a CUDA graph count once, at capture). */
uint64_t gc_kernel_launches(void);

/* Testing aid for the failure path: device waits (TMA and MMA mbarriers,
 * cluster exchanges) give up after `cycles` SM clock cycles in kernels
 * launched after this call (0 restores the defaults, about 1-2 s); a kernel
 * that gives up records GC_ERR_TIMEOUT in its workspace status, drains its
 * own copies and tensor-core work with separate fixed limits, and returns,
 * leaving the CUDA context usable.  Process-wide. */
int gc_set_wait_limit(int64_t cycles);

/* Testing aid for the failure path, together with gc_set_wait_limit: arms a
 * withheld copy in the NEXT launch of each kernel selected by `kernels` (an OR
 * of the bits below; 0 disarms).  That launch's loader issues no copy and
 * arrives on nothing, so its consumers wait on a barrier that nothing
 * completes; the wait expires after the wait limit, the kernel records
 * GC_ERR_TIMEOUT and returns, and the results of that call are undefined.  The
 * bit is consumed by the launch it affects.  Do not arm it while capturing a
 * CUDA graph (the capture would keep the withheld copy).  Process-wide. */
#define GC_STALL_CHUNK_GRADS 1 /* the chunk-gradient kernel (gc_chunk_grads)  */
#define GC_STALL_COMBINE 2     /* the tensor-core combine (decode apply, MSE;
                                  it waits only on tiles it computes, see
                                  gc_set_decode_policy) */
#define GC_STALL_BATCHED 4     /* the batched chunk-gradient GEMMs (first one) */
int gc_inject_stall(int kernels);

/* Path of the batched decode (gc_decode_batch, gc_decode_apply,
 * gc_decode_combine, gc_mse).  Every decode block Pi_i = R_{S_i} X^+ is the
 * identity I_ell when Delta_i >= ell (Sec. II-A), so the decoded gradient is
 *   ghat_b = sum_i g_{D_i} + sum_{i : Pi_{b,i} != I} (Pi_{b,i} - I) g_{D_i}   (blockwise),
 * which costs the write of ghat_b plus one chunk-gradient read per
 * non-identity block.  Each 128-row tile of the decode (128 / ell patterns)
 * is computed either that way (the residual path) or by the bf16x3
 * tensor-core GEMM Ghat = C . G; the choice is made on the device from the
 * decode matrix:
 *   GC_DECODE_AUTO      a tile takes the residual path when its patterns
 *                       average at most ceil(N*ell/64) non-identity blocks
 *                       (what the GEMM spends per pattern, in chunk-gradient
 *                       reads) and none has more than the list capacity
 *                       (16 blocks for ell <= 2, 8 for ell <= 4, else 4).
 *   GC_DECODE_DENSE     every tile on the GEMM.
 *   GC_DECODE_RESIDUAL  every tile whose patterns fit the list capacity on
 *                       the residual path.
 * Both paths give the same values up to fp32 rounding (the tests compare them
 * with each other and with the fp64 oracle); a pattern whose blocks are all
 * I_ell has grad_mse exactly 0 on the residual path.
 * Errors only (Ghat = NULL) under GC_DECODE_AUTO, when npat*ell >= 2*N*ell
 * and N*ell <= 256, take a third path: ghat_b - s = sum_a v_{b,k}[a] G_a with
 * v = C - (1_N (x) I_ell) row by row, so ||ghat_b - s||^2 = sum_k v H v^T with
 * H the (N*ell)^2 Gram matrix of the chunk blocks, formed once per call; each
 * pattern then costs its non-zero entries squared instead of N*ell*L (exact
 * patterns give 0 exactly).  Process-wide setting (default GC_DECODE_AUTO)
 * read at each launch; meant for tests and measurements. */
#define GC_DECODE_AUTO 0
#define GC_DECODE_DENSE 1
#define GC_DECODE_RESIDUAL 2
int gc_set_decode_policy(int policy);

/* Zero the status header of a workspace (asynchronous on `stream`). */
int gc_workspace_init(void* ws, size_t ws_bytes, void* stream);

/* Synchronise `stream`, read and clear the workspace status header.
 * Returns GC_OK, GC_ERR_DATA (bad psi / singular system) or GC_ERR_TIMEOUT;
 * the message names what was found. */
int gc_status(void* ws, void* stream);

/* ---- assignment (Sec. I assignment matrix A; Sec. III ordering matrix O) --
 * Host only.  kind = GC_CYCLIC: requires N == m; W_j processes chunks
 * (j + p) mod N for p = 0..delta-1 top to bottom (the cyclic assignment that
 * Sec. III shows optimal for the Q_max metric).  kind = GC_EXPLICIT: the
 * m x delta int32 array explicit_order_h lists, per worker, its chunks in
 * processing order, -1 marking an empty slot (empty slots only at the end
 * of a row); a chunk may appear at most once per worker and at most
 * GC_MAX_REPL times overall.
 * Outputs (host, caller-owned, any may be NULL):
 *   A_h      N x m uint8, A[i][j] = 1 iff D_i is assigned to W_j.
 *   order_h  m x delta int32, the processing order (copy of the input for
 *            GC_EXPLICIT).
 *   O_h      N x m uint8, O[i][j] = position (1-based) of D_i in W_j, 0 if
 *            not assigned.
 */
int gc_make_assignment(int N, int m, int delta, int kind, const int32_t* explicit_order_h,
                       uint8_t* A_h, int32_t* order_h, uint8_t* O_h);

/* ---- chunk ordering (Sec. III, Algorithm 2) ------------------------------
 * Host only.  Given an assignment matrix with N == m in which every row and
 * every column holds exactly delta non-zeros (e.g. the adjacency matrix of a
 * delta-regular graph), find an ordering that minimises
 * Q_max(O) = max_i sum_j O[i][j] + (m - delta - 1) * delta: the bipartite
 * graph of A is split into delta disjoint perfect matchings P_1..P_delta
 * (Claim 1 guarantees each exists) and O = sum_p p * P_p, so that every row
 * sum equals the lower bound delta (delta + 1) / 2.  Each matching is found
 * by augmenting paths with rows taken in increasing order and each row's
 * columns in increasing order, so the result is deterministic.
 *   A_h      N x m uint8 (non-zero = assigned), N == m.
 * Outputs (host, caller-owned, any may be NULL): order_h (m x delta int32,
 * W_j's chunks top to bottom) and O_h (N x m uint8) as in gc_make_assignment;
 * the order is accepted by gc_make_assignment(GC_EXPLICIT).
 * Errors: GC_ERR_SHAPE (N != m, or a row or column sum differs from delta),
 * GC_ERR_UNSUPPORTED (delta > GC_MAX_DELTA), GC_ERR_DATA (no perfect matching;
 * impossible for a valid input).
 */
int gc_chunk_ordering(const uint8_t* A_h, int N, int m, int delta, int32_t* order_h, uint8_t* O_h);

/* ---- chunk gradients for several parameter vectors (tensor cores) -------
 * For n_w parameter vectors at once (replicas, a learning-rate sweep):
 *   G[w][i] = X_i^T (f(X_i w_w) - y01_i)       (Sec. I, one per w_w)
 * computed as two tcgen05 GEMMs, Z = X W^T (K = d) with the residual
 * R = f(Z) - y01 formed in the epilogue, then G_i = X_i^T R_i (K = n_c).
 * W and R enter the MMAs as bf16 hi + lo parts (fp32 accumulation), X as
 * bf16 (exact).  f and y01 as in gc_chunk_grads.
 *   X    device N~ x d bf16, row-major, 16-byte aligned.
 *   y    device N~ fp32.   W  device n_w x d fp32 (row w = w_w).
 *   G    device output n_w x N x d fp32 (G[w] is the N x d chunk-gradient
 *        matrix of w_w, the layout the decode entry points take).
 *   Limits: 32 <= n_w <= 256, n_w % 32 == 0; d % 128 == 0; n_c % 64 == 0;
 *   N * n_c % 128 == 0.  No loss output.
 * Workspace: gc_chunk_grads_batched_workspace(N, n_c, d, n_w) bytes.
 */
size_t gc_chunk_grads_batched_workspace(int N, int n_c, int d, int n_w);
int gc_chunk_grads_batched(const void* X, const float* y, const float* W, int N, int n_c, int d,
                           int n_w, int loss, float* G, void* ws, size_t ws_bytes, void* stream);

/* ---- completion times and the encode-and-transmit trigger (Sec. IV) ----
 * Batched simulation of the cluster: realization r gives every worker a
 * time per chunk tau[r][j] (> 0, +inf for a failed worker); W_j finishes
 * the chunk in its slot p (1-based) at p * tau_j.  With n_i(T) the number of
 * processed copies of D_i at time T, the PS's error estimate is
 * est(T) = sum_i max(0, ell - n_i(T)) (eq. (7) and the sentence after it).
 * For each realization:
 *   T[r]       the first time with est(T) <= theta: the (N ell - theta)-th
 *              smallest of the N ell values t_i^(k) (k-th smallest completion
 *              time of D_i, k <= ell; +inf when too few copies can finish).
 *              theta = 0: every chunk processed ell times (exact recovery).
 *   psi[r][j]  chunks W_j has processed by T[r]: #{p <= delta_j : p tau_j <= T}
 *              (0 for a failed worker) -- the state the PS decodes from.
 *   T_full[r]  the same time when a copy counts only once its worker has
 *              finished all delta_j of its chunks (at delta_j tau_j), i.e.
 *              the original protocol's completion time (Sec. IV).
 * Times are formed with one double multiply each, exactly as defined, so
 * results are reproducible bit for bit.
 *   order   device m x delta int32 (as gc_make_assignment / gc_chunk_ordering).
 *   tau     device nsim x m fp64.
 *   T, psi, T_full  device outputs (nsim fp64, nsim x m int32, nsim fp64),
 *           each nullable.
 *   Limits: 1 <= ell <= GC_MAX_ELL, 0 <= theta, N * ell <= 2048, m <= 32767.
 * Workspace: gc_trigger_workspace(N) bytes.
 */
size_t gc_trigger_workspace(int N);
int gc_trigger_times(const int32_t* order, int N, int m, int delta, const double* tau, int64_t nsim,
                     int ell, int theta, double* T, int32_t* psi, double* T_full, void* ws,
                     size_t ws_bytes, void* stream);

/* ---- chunk gradients (Sec. I: g_{D_j} = sum_{i in D_j} grad l) --------
 * X        N~ x d, element type x_dtype, row-major, 16-byte aligned; chunk i
 *          is rows [i*n_c, (i+1)*n_c).
 * y        N~ float32 labels (+-1 for GC_LOGISTIC).
 * w        d float32 parameter vector.
 * G        N x d float32 output: G[i] = X_i^T (f(X_i w) - y01_i), f = identity
 *          (GC_LSQ, y01 = y) or the logistic sigmoid (GC_LOGISTIC,
 *          y01 = (y + 1) / 2).  Un-normalised sums, as in Sec. I.
 * loss_out NULL or one device double: L = (1/N~) sum_i l(x_i, y_i, w).
 * Requires d >= 1, n_c >= 1, N >= 1.  One pass over X.
 */
size_t gc_chunk_grads_workspace(int N, int n_c, int d, int x_dtype);
int gc_chunk_grads(const void* X, int x_dtype, const float* y, const float* w, int N, int n_c,
                   int d, int loss, float* G, double* loss_out, void* ws, size_t ws_bytes,
                   void* stream);

/* ---- Algorithm 1, Find-Encoding-Coeff, batched over patterns ----------
 * R      ell x m float64, the PS's Gaussian matrix (Sec. II).
 * order  m x delta int32 device copy of the processing order (-1 = empty).
 * psi    npat x m int32 state vectors: psi[b][j] = chunks W_j processed in
 *        pattern b, 0 <= psi <= delta (checked on the device: bad entries
 *        are treated as 0 and raise GC_ERR_DATA in the status header).
 * For every pattern b and chunk i, S_i = workers that processed D_i and
 * Delta_i = |S_i|; the block column B^(i) restricted to rows S_i is the
 * minimum-norm least-squares solution X^+ of eq. (6), X = R[:, S_i]
 * (computed in float64).  Outputs (each may be NULL):
 *   E         npat x m x delta x ell float64: E[b][j][p][k] = the coefficient
 *             W_j applies to g_{D_{order[j][p]}}[k] (eps_j of Algorithm 1 in
 *             processing order), 0 for p >= psi[b][j].
 *   C         npat x ell x (N*ell) float32: the decode matrix R B, i.e.
 *             C[b][k][i*ell + k'] = (R_{S_i} X^+)[k][k'] (a projector; the
 *             identity when Delta_i >= ell, Sec. II-A).
 *   delta_out npat x N uint8: Delta_i.
 *   support   npat x N x m uint8: 1 iff W_j processed D_i (supports of
 *             eqs. 3 and 8).
 *   coef_err  npat float64: || (1_N (x) I_ell)^T - R B ||_F^2.
 *   est       npat float64: sum_i max(0, ell - Delta_i) (eq. 7).
 */
size_t gc_coeff_workspace(int N, int m, int delta, int ell, int npat);
int gc_find_encoding_coeff(const double* R, int ell, const int32_t* order, int N, int m, int delta,
                           const int32_t* psi, int npat, double* E, float* C, uint8_t* delta_out,
                           uint8_t* support, double* coef_err, double* est, void* ws,
                           size_t ws_bytes, void* stream);

/* ---- Algorithm 1 without any allocation -------------------------------
 * The paper has no counterpart: this is a service for callers that cannot
 * allocate device memory at all (a runtime that reserves its memory once at
 * start-up and forbids later cudaMalloc, an embedding without a CUDA
 * allocator, a thread that must not take the allocator's locks), so cannot
 * pass the workspace gc_find_encoding_coeff needs.
 * Same arguments and outputs as gc_find_encoding_coeff, minus (ws, ws_bytes):
 * the scratch is a file-scope __device__ array of GC_NOALLOC_SCRATCH_BYTES
 * inside libgc.so, held by every GPU that loads the library until the process
 * exits.  Nothing is allocated or freed.
 *  - Sizes whose scratch (holder table, plus the memo table when it fits)
 *    exceeds GC_NOALLOC_SCRATCH_BYTES are rejected with GC_ERR_WORKSPACE.
 *  - The first call on each device looks up the array's device address
 *    (cudaGetSymbolAddress) with that device current and caches it with the
 *    current CUDA context; make that first call before any stream capture.
 *    A device reset (cudaDeviceReset) destroys the context and the array's
 *    memory: the next call, in the new context, looks the address up again
 *    (that call, too, must come before any capture).
 *  - All calls share the array: two calls whose executions overlap on the
 *    GPU (other streams, other host threads) race and give wrong results.
 *  - Device-detected data errors (psi out of range, a singular R_S) are
 *    handled as in gc_find_encoding_coeff but are not reported; run the
 *    workspace variant with gc_status to check inputs.
 */
#define GC_NOALLOC_SCRATCH_BYTES (8u << 20)
int gc_find_encoding_coeff_noalloc(const double* R, int ell, const int32_t* order, int N, int m,
                                   int delta, const int32_t* psi, int npat, double* E, float* C,
                                   uint8_t* delta_out, uint8_t* support, double* coef_err,
                                   double* est, void* stream);

/* ---- worker encoding (eq. 2) ------------------------------------------
 * Runs Algorithm 1 for every pattern, then each worker's transmission
 *   T[b][j] = sum_{p < psi[b][j]} sum_k E[b][j][p][k] g_{D_order[j][p]}[k],
 * where g[k] = g[k*L : (k+1)*L] zero-padded to length L.
 * G  N x d float32 chunk gradients; T npat x m x L float32 output.
 */
size_t gc_encode_workspace(int N, int m, int delta, int ell, int npat, int d);
int gc_encode(const double* R, int ell, const int32_t* order, int N, int m, int delta,
              const int32_t* psi, int npat, const float* G, int d, float* T, void* ws,
              size_t ws_bytes, void* stream);

/* ---- worker encoding from given coefficients (eq. 2 alone) -----------
 * T[b][j] = sum_{p < psi[b][j]} sum_k E[b][j][p][k] g_{D_order[j][p]}[k], with
 * E the npat x m x delta x ell coefficients gc_find_encoding_coeff returns
 * (Algorithm 1).  Lets a caller run Algorithm 1 while the chunk gradients
 * are still being computed.  No workspace.
 */
int gc_encode_with_coeffs(const double* E, int ell, const int32_t* order, int N, int m, int delta,
                          const int32_t* psi, int npat, const float* G, int d, float* T,
                          void* stream);

/* ---- PS decoding of received transmissions (Sec. II-B) ----------------
 * ghat[b][k*L + c] = sum_j R[k][j] T[b][j][c] for k*L + c < d.
 * T npat x m x L float32; ghat npat x d float32.  No workspace.
 */
int gc_decode_tx(const double* R, int ell, int m, const float* T, int npat, int d, float* ghat,
                 void* stream);

/* ---- batched decode-combine (Sec. II-B decode of the eq. (2) transmissions) --
 * The PS decode of Sec. II-B, sum_j R[k][j] T[b][j], applied to the
 * transmissions of eq. (2) for many patterns at once, through the identity
 * sum_j R[k][j] T[b][j] = sum_i sum_k' (R B_b)[k][i*ell+k'] g_{D_i}[k']:
 *   Ghat (npat*ell x L) = C (npat*ell x N*ell) . G (N*ell x L),
 * with C from Algorithm 1 (above) and G viewed as N*ell blocks of length L;
 * each 128-row tile is computed by the residual path or the tensor-core
 * GEMM (gc_set_decode_policy).  The supports (masks), Delta_i, the worker
 * coefficients E and C itself are outputs of gc_find_encoding_coeff on the
 * same psi; this call returns only the decoded gradients and errors.
 * G     N x d float32 chunk gradients.
 * Ghat  NULL or npat x d float32 decoded gradients.
 * coef_err, est   NULL or npat float64 (as gc_find_encoding_coeff).
 * grad_mse        NULL or npat float64: ||ghat_b - sum_i g_{D_i}||^2 / d,
 *                 reduced in a fixed order (deterministic).
 * At least one of Ghat / grad_mse must be non-NULL.
 */
size_t gc_decode_batch_workspace(int N, int m, int delta, int ell, int npat, int d);
int gc_decode_batch(const double* R, int ell, const int32_t* order, int N, int m, int delta,
                    const int32_t* psi, int npat, const float* G, int d, float* Ghat,
                    double* coef_err, double* est, double* grad_mse, void* ws, size_t ws_bytes,
                    void* stream);

/* ---- decoding in two halves: coefficients, then data --------------------
 * The decode coefficients depend only on psi and R, not on the gradients,
 * so a PS can solve them while the chunk gradients are still being computed.
 * gc_decode_plan runs Algorithm 1 for every pattern (as gc_find_encoding_coeff)
 * and writes the decode matrix R B into `plan`, an opaque caller-owned device
 * buffer of gc_decode_plan_bytes(N, ell, npat) bytes (256-byte aligned) laid
 * out for the tensor-core combine; coef_err and est as in
 * gc_find_encoding_coeff (each may be NULL).  gc_decode_apply then computes
 * Ghat and/or grad_mse from the plan and G exactly as gc_decode_batch does;
 * it must be given the same (N, ell, npat) as the plan.
 */
size_t gc_decode_plan_bytes(int N, int ell, int npat);
size_t gc_decode_plan_workspace(int N, int m, int delta, int ell, int npat);
int gc_decode_plan(const double* R, int ell, const int32_t* order, int N, int m, int delta,
                   const int32_t* psi, int npat, void* plan, size_t plan_bytes, double* coef_err,
                   double* est, void* ws, size_t ws_bytes, void* stream);
/* ---- prepared decode: the parts of Algorithm 1 that depend only on R and
 * the assignment, computed once -----------------------------------------
 * Every block problem of Algorithm 1 is X = R[:, S] for S a subset of the
 * holders of one chunk (Sec. II), so for an assignment with delta <= 14
 * chunks per worker all of them -- one per (chunk, subset of its holders) --
 * can be solved once and looked up for every pattern.  gc_decode_prepare
 * writes the holder table and, when delta <= 14, that memo table (the block
 * R_S X^+ and its error ||I - R_S X^+||_F^2 per subset) into a caller-owned
 * device buffer `prep` of gc_decode_prepare_bytes(N, m, delta, ell) bytes
 * (256-byte aligned; its first 256 bytes are a status header, read with
 * gc_status).  gc_decode_plan_prepared then does the psi side of the decode
 * for a batch as gc_decode_plan does, without recomputing them: the same
 * plan, coefficient error and estimate bit for bit whenever gc_decode_plan
 * itself uses its memo table (npat >= 2^delta), equal to rounding otherwise;
 * with delta > 14 it solves every block directly.  `prep` must come from the same R, ell,
 * order, N, m and delta; it is read-only afterwards and may serve any number
 * of calls.  ws needs gc_decode_plan_prepared_workspace() bytes (a status
 * header only). */
size_t gc_decode_prepare_bytes(int N, int m, int delta, int ell);
int gc_decode_prepare(const double* R, int ell, const int32_t* order, int N, int m, int delta,
                      void* prep, size_t prep_bytes, void* stream);
size_t gc_decode_plan_prepared_workspace(void);
int gc_decode_plan_prepared(const void* prep, const double* R, int ell, int N, int m, int delta,
                            const int32_t* psi, int npat, void* plan, size_t plan_bytes,
                            double* coef_err, double* est, void* ws, size_t ws_bytes,
                            void* stream);

size_t gc_decode_apply_workspace(int N, int ell, int npat, int d);
int gc_decode_apply(const void* plan, int ell, int N, int npat, const float* G, int d,
                    float* Ghat, double* grad_mse, void* ws, size_t ws_bytes, void* stream);

/* ---- decode-combine alone ----------------------------------------------
 * The GEMM step of gc_decode_batch for a decode matrix the caller already
 * has (e.g. from gc_find_encoding_coeff):
 *   Ghat (npat*ell x L) = C (npat*ell x N*ell) . G (N*ell x L).
 * C     npat x ell x (N*ell) float32 (layout of gc_find_encoding_coeff's C).
 * G     N x d float32; Ghat NULL or npat x d float32; grad_mse NULL or npat
 *       float64 (||ghat_b - sum_i g_{D_i}||^2 / d).  One of the two non-NULL.
 */
size_t gc_decode_combine_workspace(int N, int ell, int npat, int d);
int gc_decode_combine(const float* C, int ell, int N, int npat, const float* G, int d,
                      float* Ghat, double* grad_mse, void* ws, size_t ws_bytes, void* stream);

/* ---- error measures only (Sec. II-A eq. 7, Sec. IV) -------------------
 * gc_decode_batch with Ghat = NULL: coef_err, est and grad_mse per pattern;
 * the decoded gradients are never written (with enough patterns, grad_mse
 * comes from the Gram matrix of the chunk blocks: see GC_DECODE_AUTO).
 */
size_t gc_mse_workspace(int N, int m, int delta, int ell, int npat, int d);
int gc_mse(const double* R, int ell, const int32_t* order, int N, int m, int delta,
           const int32_t* psi, int npat, const float* G, int d, double* coef_err, double* est,
           double* grad_mse, void* ws, size_t ws_bytes, void* stream);

/* ---- parameter update (Sec. I: w_{t+1} from grad L = (1/N~) sum g) ----
 * w[c] -= lr * ghat[c] / Ntil for c < d.  w, ghat float32 device vectors.
 */
int gc_sgd_step(float* w, const float* ghat, int d, float lr, int64_t Ntil, void* stream);

/* ---- one live realization: eq. (2) encode, Sec. II-B decode, Sec. I update --
 * For one straggler pattern psi (m int32, device) with its coefficients E
 * (m x delta x ell fp64, gc_find_encoding_coeff), in one kernel:
 *   T[j][c]       = sum_{p < psi[j]} sum_k E[j][p][k] g_{D_order[j][p]}[k*L + c]   (eq. 2)
 *   ghat[k*L + c] = sum_j R[k][j] T[j][c]                                         (Sec. II-B)
 *   w[k*L + c]   -= lr * ghat[k*L + c] / Ntil                                     (Sec. I)
 * for k*L + c < d, with the same float32 operations in the same order as
 * gc_encode_with_coeffs, gc_decode_tx and gc_sgd_step, so T, ghat and w
 * equal theirs bit for bit.  One launch instead of three: the update that
 * the next step's chunk gradients wait for.
 *   R      device ell x m fp64.  order device m x delta int32.
 *   G      device N x d float32 chunk gradients.
 *   w      device d float32, updated in place.
 *   T      NULL or device m x L float32 output (the transmissions).
 *   ghat   NULL or device d float32 output (the decoded gradient).
 * E, R, the order, psi and the transmissions of 32 columns are staged in
 * shared memory: (m*delta*ell + ell*m + 32*m + m*delta + m) * 4 bytes must
 * not exceed 96 KB (GC_ERR_UNSUPPORTED otherwise).  No workspace.
 */
int gc_live_step(const double* E, const double* R, int ell, const int32_t* order, int N, int m,
                 int delta, const int32_t* psi, const float* G, int d, float lr, int64_t Ntil,
                 float* w, float* T, float* ghat, void* stream);

#ifdef __cplusplus
}
#endif
#endif /* GC_H_ */
