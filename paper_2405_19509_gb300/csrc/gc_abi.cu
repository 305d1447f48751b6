// extern "C" entry points of libgc.so: validation, workspace layout, launches.
// Every entry point validates on the host before launching anything and
// returns a GC_* status; the text of the last error is thread-local.
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <nvtx3/nvToolsExt.h>

#include <algorithm>
#include <atomic>
#include <vector>

#include "gc_internal.cuh"

namespace gc {

NvtxRange::NvtxRange(const char* name) { nvtxRangePushA(name); }
NvtxRange::~NvtxRange() { nvtxRangePop(); }

static thread_local char g_err[512] = "";

int fail(int code, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
  return code;
}

int cuda_check(cudaError_t e, const char* what) {
  if (e == cudaSuccess) return GC_OK;
  return fail(GC_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

static std::atomic<uint64_t> g_launches{0};
void count_launches(int n) { g_launches.fetch_add((uint64_t)n, std::memory_order_relaxed); }

static std::atomic<long long> g_wait_limit{0};
long long wait_limit(long long dflt) {
  const long long v = g_wait_limit.load(std::memory_order_relaxed);
  return v > 0 ? v : dflt;
}
static std::atomic<int> g_stall{0};
bool take_stall(int bit) { return (g_stall.fetch_and(~bit) & bit) != 0; }
static std::atomic<int> g_policy{GC_DECODE_AUTO};
int decode_policy() { return g_policy.load(std::memory_order_relaxed); }

int device_sm_count() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 152;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
    return 152;
  return n;
}

namespace {

cudaStream_t as_stream(void* s) { return static_cast<cudaStream_t>(s); }

int check_ws(void* ws, size_t ws_bytes, size_t need) {
  if (!ws) return fail(GC_ERR_WORKSPACE, "workspace is NULL (need %zu bytes)", need);
  if (reinterpret_cast<uintptr_t>(ws) % 256 != 0)
    return fail(GC_ERR_WORKSPACE, "workspace must be 256-byte aligned");
  if (ws_bytes < need)
    return fail(GC_ERR_WORKSPACE, "workspace too small: %zu < %zu bytes", ws_bytes, need);
  return GC_OK;
}

int check_dims(int N, int m, int delta, int ell, int npat) {
  if (N < 1 || m < 1) return fail(GC_ERR_SHAPE, "N=%d and m=%d must be >= 1", N, m);
  if (m > 32767) return fail(GC_ERR_UNSUPPORTED, "m=%d exceeds 32767", m);
  if (delta < 1) return fail(GC_ERR_SHAPE, "delta=%d must be >= 1", delta);
  if (delta > GC_MAX_DELTA) return fail(GC_ERR_UNSUPPORTED, "delta=%d exceeds %d", delta, GC_MAX_DELTA);
  if (ell < 1) return fail(GC_ERR_SHAPE, "ell=%d must be >= 1", ell);
  if (ell > GC_MAX_ELL) return fail(GC_ERR_UNSUPPORTED, "ell=%d exceeds %d", ell, GC_MAX_ELL);
  if (npat < 0) return fail(GC_ERR_SHAPE, "npat=%d must be >= 0", npat);
  if ((long long)N * ell > (1LL << 30)) return fail(GC_ERR_UNSUPPORTED, "N*ell too large");
  return GC_OK;
}

// Workspace layout of the pattern solve: holders, then the memo table.
struct SolveWs {
  Holders h;
  void* table;
  int bits;
};
SolveWs carve_solve(Carve& c, int N, int m, int delta, int ell, int npat) {
  SolveWs s;
  s.h = carve_holders(c, N);
  s.bits = solve_table_bits(N, m, delta, npat);
  const size_t tb = solve_table_bytes(N, ell, s.bits);
  s.table = tb ? c.take<char>(tb) : nullptr;
  return s;
}

uint32_t* status_of(void* ws) { return static_cast<uint32_t*>(ws); }


}  // namespace
}  // namespace gc

using namespace gc;

extern "C" {

const char* gc_last_error(void) { return g_err; }

int gc_version(void) { return 200; }

uint64_t gc_kernel_launches(void) { return g_launches.load(); }

int gc_inject_stall(int kernels) {
  if (kernels & ~(GC_STALL_CHUNK_GRADS | GC_STALL_COMBINE | GC_STALL_BATCHED))
    return fail(GC_ERR_ARG, "kernels=0x%x has unknown bits", kernels);
  g_stall.store(kernels);
  return GC_OK;
}

size_t gc_chunk_grads_batched_workspace(int N, int n_c, int d, int n_w) {
  if (N < 1 || n_c < 1 || d < 1 || n_w < 1) return 0;
  return kHeaderBytes + gemmw_ws_bytes(N, n_c, d, n_w);
}

int gc_chunk_grads_batched(const void* X, const float* y, const float* W, int N, int n_c, int d,
                           int n_w, int loss, float* G, void* ws, size_t ws_bytes, void* stream) {
  NvtxRange nvtx_("gc_chunk_grads_batched");
  if (N < 1 || n_c < 1 || d < 1 || n_w < 1) return fail(GC_ERR_SHAPE, "N, n_c, d, n_w must be >= 1");
  if (n_w % 32 != 0 || n_w > 256)
    return fail(GC_ERR_UNSUPPORTED, "n_w=%d must be a multiple of 32 in [32, 256]", n_w);
  if (d % 128 != 0) return fail(GC_ERR_UNSUPPORTED, "d=%d must be a multiple of 128", d);
  if (n_c % 64 != 0) return fail(GC_ERR_UNSUPPORTED, "n_c=%d must be a multiple of 64", n_c);
  if (((long long)N * n_c) % 128 != 0) return fail(GC_ERR_UNSUPPORTED, "N*n_c must be a multiple of 128");
  if ((long long)N * n_c > (1LL << 31) - 1) return fail(GC_ERR_UNSUPPORTED, "N*n_c too large");
  if (loss != GC_LSQ && loss != GC_LOGISTIC) return fail(GC_ERR_ARG, "unknown loss %d", loss);
  if (!X || !y || !W || !G) return fail(GC_ERR_ARG, "X, y, W and G must be non-NULL");
  if (reinterpret_cast<uintptr_t>(X) % 16 != 0) return fail(GC_ERR_ARG, "X must be 16-byte aligned");
  if (!ws || ws_bytes < gc_chunk_grads_batched_workspace(N, n_c, d, n_w))
    return fail(GC_ERR_WORKSPACE, "workspace too small");
  Carve c(ws);
  return launch_chunkgrad_batched(X, y, W, N, n_c, d, n_w, loss, G, c, status_of(ws),
                                  as_stream(stream));
}

size_t gc_trigger_workspace(int N) {
  if (N < 1) return 0;
  Carve c(nullptr);
  carve_holders(c, N);
  return c.bytes();
}

int gc_trigger_times(const int32_t* order, int N, int m, int delta, const double* tau, int64_t nsim,
                     int ell, int theta, double* T, int32_t* psi, double* T_full, void* ws,
                     size_t ws_bytes, void* stream) {
  NvtxRange nvtx_("gc_trigger_times");
  if (N < 1 || m < 1 || delta < 1 || nsim < 0) return fail(GC_ERR_SHAPE, "N, m, delta >= 1, nsim >= 0");
  if (ell < 1 || ell > GC_MAX_ELL) return fail(GC_ERR_UNSUPPORTED, "ell=%d outside [1, %d]", ell, GC_MAX_ELL);
  if (delta > GC_MAX_DELTA) return fail(GC_ERR_UNSUPPORTED, "delta=%d exceeds %d", delta, GC_MAX_DELTA);
  if (theta < 0) return fail(GC_ERR_ARG, "theta=%d must be >= 0", theta);
  if ((long long)N * ell > kTriggerMaxKeys)
    return fail(GC_ERR_UNSUPPORTED, "N*ell=%lld exceeds %d", (long long)N * ell, kTriggerMaxKeys);
  if (m > 32767) return fail(GC_ERR_UNSUPPORTED, "m=%d exceeds 32767", m);
  if (nsim == 0) return GC_OK;
  if (!order || !tau) return fail(GC_ERR_ARG, "order and tau must be non-NULL");
  if (!ws || ws_bytes < gc_trigger_workspace(N)) return fail(GC_ERR_WORKSPACE, "workspace too small");
  cudaStream_t s = as_stream(stream);
  Carve c(ws);
  Holders h = carve_holders(c, N);
  launch_holders(order, N, m, delta, h, status_of(ws), s);
  return launch_trigger(order, h, N, m, delta, tau, nsim, ell, theta, T, psi, T_full, s);
}

int gc_set_decode_policy(int policy) {
  if (policy != GC_DECODE_AUTO && policy != GC_DECODE_DENSE && policy != GC_DECODE_RESIDUAL)
    return fail(GC_ERR_ARG, "unknown decode policy %d", policy);
  g_policy.store(policy, std::memory_order_relaxed);
  return GC_OK;
}

int gc_set_wait_limit(int64_t cycles) {
  if (cycles < 0) return fail(GC_ERR_ARG, "cycles=%lld must be >= 0", (long long)cycles);
  g_wait_limit.store(cycles, std::memory_order_relaxed);
  return GC_OK;
}

int gc_workspace_init(void* ws, size_t ws_bytes, void* stream) {
  if (!ws || ws_bytes < kHeaderBytes) return fail(GC_ERR_WORKSPACE, "workspace missing or < 256 bytes");
  GC_CUDA(cudaMemsetAsync(ws, 0, kHeaderBytes, as_stream(stream)));
  return GC_OK;
}

int gc_status(void* ws, void* stream) {
  if (!ws) return fail(GC_ERR_WORKSPACE, "workspace is NULL");
  WsHeader h{};
  GC_CUDA(cudaStreamSynchronize(as_stream(stream)));
  GC_CUDA(cudaMemcpy(&h, ws, sizeof(h), cudaMemcpyDeviceToHost));
  GC_CUDA(cudaMemset(ws, 0, sizeof(h)));
  if (h.status & ST_TIMEOUT)
    return fail(GC_ERR_TIMEOUT, "a bounded device wait expired (status 0x%x)", h.status);
  if (h.status & (ST_BAD_PSI | ST_SINGULAR | ST_BAD_ORDER)) {
    return fail(GC_ERR_DATA, "device reported:%s%s%s", (h.status & ST_BAD_PSI) ? " psi outside [0, delta];" : "",
                (h.status & ST_SINGULAR) ? " rank-deficient least-squares system;" : "",
                (h.status & ST_BAD_ORDER) ? " invalid order entry or too many copies of a chunk;" : "");
  }
  return GC_OK;
}

int gc_make_assignment(int N, int m, int delta, int kind, const int32_t* explicit_order_h,
                       uint8_t* A_h, int32_t* order_h, uint8_t* O_h) {
  if (N < 1 || m < 1 || delta < 1) return fail(GC_ERR_SHAPE, "N, m, delta must be >= 1");
  if (delta > GC_MAX_DELTA) return fail(GC_ERR_UNSUPPORTED, "delta=%d exceeds %d", delta, GC_MAX_DELTA);
  if (delta > N) return fail(GC_ERR_SHAPE, "delta=%d exceeds N=%d", delta, N);
  std::vector<int32_t> order((size_t)m * delta, -1);
  if (kind == GC_CYCLIC) {
    if (N != m) return fail(GC_ERR_SHAPE, "cyclic assignment needs N == m (N=%d, m=%d)", N, m);
    for (int j = 0; j < m; ++j)
      for (int p = 0; p < delta; ++p) order[(size_t)j * delta + p] = (j + p) % N;
  } else if (kind == GC_EXPLICIT) {
    if (!explicit_order_h) return fail(GC_ERR_ARG, "explicit_order_h is NULL");
    std::vector<int> copies(N, 0);
    std::vector<char> seen(N, 0);
    for (int j = 0; j < m; ++j) {
      std::fill(seen.begin(), seen.end(), 0);
      bool ended = false;
      for (int p = 0; p < delta; ++p) {
        const int v = explicit_order_h[(size_t)j * delta + p];
        if (v == -1) {
          ended = true;
          continue;
        }
        if (v < -1 || v >= N) return fail(GC_ERR_ARG, "order[%d][%d]=%d outside [-1, N)", j, p, v);
        if (ended) return fail(GC_ERR_ARG, "order[%d]: chunk after an empty slot", j);
        if (seen[v]) return fail(GC_ERR_ARG, "order[%d]: chunk %d twice", j, v);
        seen[v] = 1;
        if (++copies[v] > GC_MAX_REPL)
          return fail(GC_ERR_UNSUPPORTED, "chunk %d has more than %d copies", v, GC_MAX_REPL);
        order[(size_t)j * delta + p] = v;
      }
    }
  } else {
    return fail(GC_ERR_ARG, "unknown assignment kind %d", kind);
  }
  if (A_h) memset(A_h, 0, (size_t)N * m);
  if (O_h) memset(O_h, 0, (size_t)N * m);
  for (int j = 0; j < m; ++j)
    for (int p = 0; p < delta; ++p) {
      const int v = order[(size_t)j * delta + p];
      if (v < 0) continue;
      if (A_h) A_h[(size_t)v * m + j] = 1;
      if (O_h) O_h[(size_t)v * m + j] = (uint8_t)(p + 1);
    }
  if (order_h) memcpy(order_h, order.data(), order.size() * sizeof(int32_t));
  return GC_OK;
}

// ---------------------------------------------------------------- chunk grads
size_t gc_chunk_grads_workspace(int N, int n_c, int d, int x_dtype) {
  if (N < 1 || n_c < 1 || d < 1) return 0;
  return kHeaderBytes + chunkgrad_ws_bytes(N, n_c, d, x_dtype);
}

int gc_chunk_grads(const void* X, int x_dtype, const float* y, const float* w, int N, int n_c,
                   int d, int loss, float* G, double* loss_out, void* ws, size_t ws_bytes,
                   void* stream) {
  NvtxRange nvtx_("gc_chunk_grads");
  if (!X || !y || !w || !G) return fail(GC_ERR_ARG, "X, y, w and G must be non-NULL");
  if (x_dtype != GC_F32 && x_dtype != GC_BF16) return fail(GC_ERR_ARG, "x_dtype=%d", x_dtype);
  if (loss != GC_LSQ && loss != GC_LOGISTIC) return fail(GC_ERR_ARG, "loss=%d", loss);
  if (N < 1 || n_c < 1 || d < 1) return fail(GC_ERR_SHAPE, "N, n_c, d must be >= 1");
  if ((long long)N * n_c > (1LL << 40)) return fail(GC_ERR_SHAPE, "N*n_c too large");
  int rc = check_ws(ws, ws_bytes, gc_chunk_grads_workspace(N, n_c, d, x_dtype));
  if (rc) return rc;
  Carve c(ws);
  return launch_chunkgrad(X, x_dtype, y, w, N, n_c, d, loss, G, loss_out, c, status_of(ws),
                          as_stream(stream));
}

// ---------------------------------------------------------------- Algorithm 1
size_t gc_coeff_workspace(int N, int m, int delta, int ell, int npat) {
  if (check_dims(N, m, delta, ell, npat)) return 0;
  Carve c(nullptr);
  carve_solve(c, N, m, delta, ell, npat);
  return c.bytes();
}

int gc_find_encoding_coeff(const double* R, int ell, const int32_t* order, int N, int m, int delta,
                           const int32_t* psi, int npat, double* E, float* C, uint8_t* delta_out,
                           uint8_t* support, double* coef_err, double* est, void* ws,
                           size_t ws_bytes, void* stream) {
  NvtxRange nvtx_("gc_find_encoding_coeff");
  int rc = check_dims(N, m, delta, ell, npat);
  if (rc) return rc;
  if (!R || !order || (!psi && npat > 0)) return fail(GC_ERR_ARG, "R, order and psi must be non-NULL");
  rc = check_ws(ws, ws_bytes, gc_coeff_workspace(N, m, delta, ell, npat));
  if (rc) return rc;
  if (npat == 0) return GC_OK;
  cudaStream_t s = as_stream(stream);
  Carve c(ws);
  SolveWs sw = carve_solve(c, N, m, delta, ell, npat);
  launch_holders(order, N, m, delta, sw.h, status_of(ws), s);
  SolveOut out{E, C, delta_out, support, coef_err, est};
  return launch_solve_impl(R, ell, psi, sw.h, N, m, delta, npat, out, sw.table, sw.bits,
                           status_of(ws), s);
}

// ---------------------------------------------------------------- encode
size_t gc_encode_workspace(int N, int m, int delta, int ell, int npat, int d) {
  if (check_dims(N, m, delta, ell, npat) || d < 1) return 0;
  Carve c(nullptr);
  carve_solve(c, N, m, delta, ell, npat);
  c.take<double>((size_t)npat * m * delta * ell);
  return c.bytes();
}

int gc_encode(const double* R, int ell, const int32_t* order, int N, int m, int delta,
              const int32_t* psi, int npat, const float* G, int d, float* T, void* ws,
              size_t ws_bytes, void* stream) {
  NvtxRange nvtx_("gc_encode");
  int rc = check_dims(N, m, delta, ell, npat);
  if (rc) return rc;
  if (d < 1) return fail(GC_ERR_SHAPE, "d=%d must be >= 1", d);
  if (!R || !order || !G || !T || (!psi && npat > 0))
    return fail(GC_ERR_ARG, "R, order, psi, G and T must be non-NULL");
  rc = check_ws(ws, ws_bytes, gc_encode_workspace(N, m, delta, ell, npat, d));
  if (rc) return rc;
  if (npat == 0) return GC_OK;
  cudaStream_t s = as_stream(stream);
  Carve c(ws);
  SolveWs sw = carve_solve(c, N, m, delta, ell, npat);
  double* E = c.take<double>((size_t)npat * m * delta * ell);
  launch_holders(order, N, m, delta, sw.h, status_of(ws), s);
  SolveOut out{E, nullptr, nullptr, nullptr, nullptr, nullptr};
  rc = launch_solve_impl(R, ell, psi, sw.h, N, m, delta, npat, out, sw.table, sw.bits,
                         status_of(ws), s);
  if (rc) return rc;
  return launch_encode(E, order, psi, N, m, delta, ell, npat, G, d, T, s);
}

int gc_encode_with_coeffs(const double* E, int ell, const int32_t* order, int N, int m, int delta,
                          const int32_t* psi, int npat, const float* G, int d, float* T,
                          void* stream) {
  NvtxRange nvtx_("gc_encode_with_coeffs");
  int rc = check_dims(N, m, delta, ell, npat);
  if (rc) return rc;
  if (d < 1) return fail(GC_ERR_SHAPE, "d=%d must be >= 1", d);
  if (!E || !order || !G || !T || (!psi && npat > 0))
    return fail(GC_ERR_ARG, "E, order, psi, G and T must be non-NULL");
  if (npat == 0) return GC_OK;
  return launch_encode(E, order, psi, N, m, delta, ell, npat, G, d, T, as_stream(stream));
}

int gc_decode_tx(const double* R, int ell, int m, const float* T, int npat, int d, float* ghat,
                 void* stream) {
  NvtxRange nvtx_("gc_decode_tx");
  if (!R || !T || !ghat) return fail(GC_ERR_ARG, "R, T and ghat must be non-NULL");
  if (m < 1 || npat < 0 || d < 1) return fail(GC_ERR_SHAPE, "m, d >= 1 and npat >= 0 required");
  if (ell < 1) return fail(GC_ERR_SHAPE, "ell=%d must be >= 1", ell);
  if (ell > GC_MAX_ELL) return fail(GC_ERR_UNSUPPORTED, "ell=%d exceeds %d", ell, GC_MAX_ELL);
  return launch_decode_tx(R, ell, m, T, npat, d, ghat, as_stream(stream));
}

// ---------------------------------------------------------------- decode plan / apply / batch
size_t gc_decode_plan_bytes(int N, int ell, int npat) {
  if (N < 1 || ell < 1 || ell > GC_MAX_ELL || npat < 0) return 0;
  return plan_bytes(N, ell, npat);
}

size_t gc_decode_plan_workspace(int N, int m, int delta, int ell, int npat) {
  return gc_coeff_workspace(N, m, delta, ell, npat);
}

int gc_decode_plan(const double* R, int ell, const int32_t* order, int N, int m, int delta,
                   const int32_t* psi, int npat, void* plan, size_t plan_bytes_, double* coef_err,
                   double* est, void* ws, size_t ws_bytes, void* stream) {
  NvtxRange nvtx_("gc_decode_plan");
  int rc = check_dims(N, m, delta, ell, npat);
  if (rc) return rc;
  if (!R || !order || (!psi && npat > 0)) return fail(GC_ERR_ARG, "R, order and psi must be non-NULL");
  if (npat == 0) return GC_OK;
  if (!plan) return fail(GC_ERR_ARG, "plan is NULL");
  if (plan_bytes_ < plan_bytes(N, ell, npat))
    return fail(GC_ERR_WORKSPACE, "plan buffer too small: %zu < %zu bytes", plan_bytes_,
                plan_bytes(N, ell, npat));
  if (reinterpret_cast<uintptr_t>(plan) % 256 != 0)
    return fail(GC_ERR_WORKSPACE, "plan buffer must be 256-byte aligned");
  rc = check_ws(ws, ws_bytes, gc_decode_plan_workspace(N, m, delta, ell, npat));
  if (rc) return rc;
  cudaStream_t s = as_stream(stream);
  Carve c(ws);
  SolveWs sw = carve_solve(c, N, m, delta, ell, npat);
  launch_holders(order, N, m, delta, sw.h, status_of(ws), s);
  SolveOut out{nullptr, nullptr, nullptr, nullptr, coef_err, est,
               static_cast<__nv_bfloat16*>(plan), combine_kp(N, ell)};
  return launch_solve_impl(R, ell, psi, sw.h, N, m, delta, npat, out, sw.table, sw.bits,
                           status_of(ws), s);
}

// Layout of a prepared buffer: status header, holders, memo table (delta <= 14).
static int prep_bits(int delta) { return delta <= 14 ? delta : -1; }

size_t gc_decode_prepare_bytes(int N, int m, int delta, int ell) {
  if (N < 1 || m < 1 || delta < 1 || ell < 1 || ell > GC_MAX_ELL || delta > GC_MAX_DELTA) return 0;
  Carve c(nullptr);
  carve_holders(c, N);
  c.take<char>(solve_table_bytes(N, ell, prep_bits(delta)));
  return c.bytes();
}

int gc_decode_prepare(const double* R, int ell, const int32_t* order, int N, int m, int delta,
                      void* prep, size_t prep_bytes, void* stream) {
  NvtxRange nvtx_("gc_decode_prepare");
  int rc = check_dims(N, m, delta, ell, 0);
  if (rc) return rc;
  if (!R || !order) return fail(GC_ERR_ARG, "R and order must be non-NULL");
  if (!prep || reinterpret_cast<uintptr_t>(prep) % 256 != 0)
    return fail(GC_ERR_WORKSPACE, "prep must be a 256-byte aligned device buffer");
  if (prep_bytes < gc_decode_prepare_bytes(N, m, delta, ell))
    return fail(GC_ERR_WORKSPACE, "prep buffer too small: %zu < %zu bytes", prep_bytes,
                gc_decode_prepare_bytes(N, m, delta, ell));
  cudaStream_t s = as_stream(stream);
  GC_CUDA(cudaMemsetAsync(prep, 0, kHeaderBytes, s));
  Carve c(prep);
  Holders h = carve_holders(c, N);
  const int bits = prep_bits(delta);
  void* table = bits >= 0 ? c.take<char>(solve_table_bytes(N, ell, bits)) : nullptr;
  launch_holders(order, N, m, delta, h, status_of(prep), s);
  if (bits < 0) return cuda_check(cudaGetLastError(), "k_holders");
  SolveOut out{nullptr, nullptr, nullptr, nullptr, nullptr, nullptr, nullptr, combine_kp(N, ell)};
  return launch_solve_impl(R, ell, nullptr, h, N, m, delta, 0, out, table, bits, status_of(prep),
                           s, true);
}

size_t gc_decode_plan_prepared_workspace(void) { return kHeaderBytes; }

int gc_decode_plan_prepared(const void* prep, const double* R, int ell, int N, int m, int delta,
                            const int32_t* psi, int npat, void* plan, size_t plan_bytes_,
                            double* coef_err, double* est, void* ws, size_t ws_bytes,
                            void* stream) {
  NvtxRange nvtx_("gc_decode_plan_prepared");
  int rc = check_dims(N, m, delta, ell, npat);
  if (rc) return rc;
  if (!prep || !R || (!psi && npat > 0)) return fail(GC_ERR_ARG, "prep, R and psi must be non-NULL");
  if (npat == 0) return GC_OK;
  if (!plan) return fail(GC_ERR_ARG, "plan is NULL");
  if (plan_bytes_ < plan_bytes(N, ell, npat))
    return fail(GC_ERR_WORKSPACE, "plan buffer too small: %zu < %zu bytes", plan_bytes_,
                plan_bytes(N, ell, npat));
  if (reinterpret_cast<uintptr_t>(plan) % 256 != 0)
    return fail(GC_ERR_WORKSPACE, "plan buffer must be 256-byte aligned");
  rc = check_ws(ws, ws_bytes, kHeaderBytes);
  if (rc) return rc;
  Carve c(const_cast<void*>(prep));
  Holders h = carve_holders(c, N);
  const int bits = prep_bits(delta);
  void* table = bits >= 0 ? c.take<char>(solve_table_bytes(N, ell, bits)) : nullptr;
  SolveOut out{nullptr, nullptr, nullptr, nullptr, coef_err, est,
               static_cast<__nv_bfloat16*>(plan), combine_kp(N, ell)};
  return launch_solve_impl(R, ell, psi, h, N, m, delta, npat, out, table, bits, status_of(ws),
                           as_stream(stream), false);
}

size_t gc_decode_apply_workspace(int N, int ell, int npat, int d) {
  if (N < 1 || ell < 1 || ell > GC_MAX_ELL || npat < 0 || d < 1) return 0;
  return kHeaderBytes + apply_ws_bytes(N, ell, npat, d);
}

static int check_apply(int N, int ell, int npat, int d, const void* G, const float* Ghat,
                       const double* grad_mse) {
  if (N < 1 || npat < 0 || d < 1) return fail(GC_ERR_SHAPE, "N, d >= 1 and npat >= 0 required");
  if (ell < 1) return fail(GC_ERR_SHAPE, "ell=%d must be >= 1", ell);
  if (ell > GC_MAX_ELL) return fail(GC_ERR_UNSUPPORTED, "ell=%d exceeds %d", ell, GC_MAX_ELL);
  if ((long long)N * ell > (1LL << 30)) return fail(GC_ERR_UNSUPPORTED, "N*ell too large");
  if (!G) return fail(GC_ERR_ARG, "G must be non-NULL");
  if (npat > 0 && !Ghat && !grad_mse) return fail(GC_ERR_ARG, "Ghat and grad_mse are both NULL");
  return GC_OK;
}

int gc_decode_apply(const void* plan, int ell, int N, int npat, const float* G, int d, float* Ghat,
                    double* grad_mse, void* ws, size_t ws_bytes, void* stream) {
  NvtxRange nvtx_("gc_decode_apply");
  int rc = check_apply(N, ell, npat, d, G, Ghat, grad_mse);
  if (rc) return rc;
  if (npat == 0) return GC_OK;
  if (!plan) return fail(GC_ERR_ARG, "plan is NULL");
  rc = check_ws(ws, ws_bytes, gc_decode_apply_workspace(N, ell, npat, d));
  if (rc) return rc;
  Carve c(ws);
  return launch_apply(static_cast<const __nv_bfloat16*>(plan), G, N, ell, npat, d, Ghat, grad_mse,
                      c, status_of(ws), as_stream(stream));
}

size_t gc_decode_batch_workspace(int N, int m, int delta, int ell, int npat, int d) {
  if (check_dims(N, m, delta, ell, npat) || d < 1) return 0;
  Carve c(nullptr);
  carve_solve(c, N, m, delta, ell, npat);
  c.take<char>(plan_bytes(N, ell, npat));
  c.take<char>(apply_ws_bytes(N, ell, npat, d));
  return c.bytes();
}

int gc_decode_batch(const double* R, int ell, const int32_t* order, int N, int m, int delta,
                    const int32_t* psi, int npat, const float* G, int d, float* Ghat,
                    double* coef_err, double* est, double* grad_mse, void* ws, size_t ws_bytes,
                    void* stream) {
  NvtxRange nvtx_("gc_decode_batch");
  int rc = check_dims(N, m, delta, ell, npat);
  if (rc) return rc;
  if (d < 1) return fail(GC_ERR_SHAPE, "d=%d must be >= 1", d);
  if (!R || !order || !G || (!psi && npat > 0))
    return fail(GC_ERR_ARG, "R, order, psi and G must be non-NULL");
  if (npat == 0) return GC_OK;
  if (!Ghat && !grad_mse) return fail(GC_ERR_ARG, "Ghat and grad_mse are both NULL");
  rc = check_ws(ws, ws_bytes, gc_decode_batch_workspace(N, m, delta, ell, npat, d));
  if (rc) return rc;
  cudaStream_t s = as_stream(stream);
  Carve c(ws);
  SolveWs sw = carve_solve(c, N, m, delta, ell, npat);
  __nv_bfloat16* Cs = c.take<__nv_bfloat16>(plan_bytes(N, ell, npat) / sizeof(__nv_bfloat16));
  launch_holders(order, N, m, delta, sw.h, status_of(ws), s);
  SolveOut out{nullptr, nullptr, nullptr, nullptr, coef_err, est, Cs, combine_kp(N, ell)};
  rc = launch_solve_impl(R, ell, psi, sw.h, N, m, delta, npat, out, sw.table, sw.bits,
                         status_of(ws), s);
  if (rc) return rc;
  return launch_apply(Cs, G, N, ell, npat, d, Ghat, grad_mse, c, status_of(ws), s);
}

size_t gc_decode_combine_workspace(int N, int ell, int npat, int d) {
  if (N < 1 || ell < 1 || ell > GC_MAX_ELL || npat < 0 || d < 1) return 0;
  Carve c(nullptr);
  c.take<char>(plan_bytes(N, ell, npat));
  c.take<char>(apply_ws_bytes(N, ell, npat, d));
  return c.bytes();
}

int gc_decode_combine(const float* C, int ell, int N, int npat, const float* G, int d,
                      float* Ghat, double* grad_mse, void* ws, size_t ws_bytes, void* stream) {
  NvtxRange nvtx_("gc_decode_combine");
  int rc = check_apply(N, ell, npat, d, G, Ghat, grad_mse);
  if (rc) return rc;
  if (!C) return fail(GC_ERR_ARG, "C must be non-NULL");
  if (npat == 0) return GC_OK;
  rc = check_ws(ws, ws_bytes, gc_decode_combine_workspace(N, ell, npat, d));
  if (rc) return rc;
  cudaStream_t s = as_stream(stream);
  Carve c(ws);
  __nv_bfloat16* Cs = c.take<__nv_bfloat16>(plan_bytes(N, ell, npat) / sizeof(__nv_bfloat16));
  rc = launch_split_c(C, N, ell, npat, Cs, s);
  if (rc) return rc;
  return launch_apply(Cs, G, N, ell, npat, d, Ghat, grad_mse, c, status_of(ws), s);
}

size_t gc_mse_workspace(int N, int m, int delta, int ell, int npat, int d) {
  return gc_decode_batch_workspace(N, m, delta, ell, npat, d);
}

int gc_mse(const double* R, int ell, const int32_t* order, int N, int m, int delta,
           const int32_t* psi, int npat, const float* G, int d, double* coef_err, double* est,
           double* grad_mse, void* ws, size_t ws_bytes, void* stream) {
  NvtxRange nvtx_("gc_mse");
  if (!grad_mse && npat > 0) return fail(GC_ERR_ARG, "grad_mse must be non-NULL");
  return gc_decode_batch(R, ell, order, N, m, delta, psi, npat, G, d, nullptr, coef_err, est,
                         grad_mse, ws, ws_bytes, stream);
}

int gc_sgd_step(float* w, const float* ghat, int d, float lr, int64_t Ntil, void* stream) {
  NvtxRange nvtx_("gc_sgd_step");
  if (!w || !ghat) return fail(GC_ERR_ARG, "w and ghat must be non-NULL");
  if (d < 1 || Ntil < 1) return fail(GC_ERR_SHAPE, "d and Ntil must be >= 1");
  return launch_sgd(w, ghat, d, lr, Ntil, as_stream(stream));
}

int gc_live_step(const double* E, const double* R, int ell, const int32_t* order, int N, int m,
                 int delta, const int32_t* psi, const float* G, int d, float lr, int64_t Ntil,
                 float* w, float* T, float* ghat, void* stream) {
  NvtxRange nvtx_("gc_live_step");
  int rc = check_dims(N, m, delta, ell, 1);
  if (rc) return rc;
  if (d < 1 || Ntil < 1) return fail(GC_ERR_SHAPE, "d and Ntil must be >= 1");
  if (!E || !R || !order || !psi || !G || !w)
    return fail(GC_ERR_ARG, "E, R, order, psi, G and w must be non-NULL");
  return launch_live_step(E, R, ell, order, N, m, delta, psi, G, d, lr, Ntil, w, T, ghat,
                          as_stream(stream));
}

}  // extern "C"
