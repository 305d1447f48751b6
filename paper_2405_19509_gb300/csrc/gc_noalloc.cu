// Algorithm 1 for callers that cannot allocate device memory.
//
// gc_find_encoding_coeff needs a scratch workspace (the table of each chunk's
// holders and, for large batches, the memo table of solved holder subsets).
// Some callers cannot provide one: a runtime that reserves all of its device
// memory once at start-up and forbids any later cudaMalloc, an embedding that
// owns no CUDA allocator, or a thread that must never take the allocator's
// locks.  gc_find_encoding_coeff_noalloc takes that scratch from the
// fixed-size array below instead.  The array is part of the library's device
// image: every GPU that loads libgc.so holds it (GC_NOALLOC_SCRATCH_BYTES)
// until the process exits.
//
// Host code must not use the array's name as a device address (in host code
// it names a host-side stand-in).  The first call on each device therefore
// looks the device address up with cudaGetSymbolAddress while that device is
// current, checks the result, and caches it with the CUDA context that was
// current; later calls in the same context reuse the cached address.  A
// device reset destroys the context and the module's memory with it, so a
// call made in a new context looks the address up again instead of using a
// dead one.  Make the first call in each context before any stream capture.
//
// All calls share the array and leave their contents in it: each call clears
// the status header it uses, and every other byte it reads is written earlier
// in the same call.  Calls whose executions overlap on the GPU (different
// streams, or different host threads on one device) race on the array.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>

#include "gc_internal.cuh"

namespace gc {
namespace {

__device__ __align__(256) unsigned char g_noalloc_scratch[GC_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
struct Cached {
  CUcontext ctx;  // context current when the address was looked up
  void* addr;
};
Cached g_addr[kMaxDevices] = {};

// The driver's cuCtxGetCurrent, through the runtime (no link to libcuda).
PFN_cuCtxGetCurrent_v4000 ctx_current_fn() {
  static PFN_cuCtxGetCurrent_v4000 fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 4000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      return reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(p);
    return static_cast<PFN_cuCtxGetCurrent_v4000>(nullptr);
  }();
  return fn;
}

CUcontext current_context() {
  CUcontext c = nullptr;
  auto fn = ctx_current_fn();
  if (!fn || fn(&c) != CUDA_SUCCESS) return nullptr;
  return c;
}

// Device address of the static scratch on the current device (set-up on the
// first call per device and context).
int scratch_address(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_check(e, "cudaGetDevice");
  if (dev < 0 || dev >= kMaxDevices)
    return fail(GC_ERR_UNSUPPORTED, "device ordinal %d beyond %d", dev, kMaxDevices);
  CUcontext ctx = current_context();
  std::lock_guard<std::mutex> lock(g_mu);
  Cached& c = g_addr[dev];
  if (!c.addr || !ctx || c.ctx != ctx) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);  // makes the device's context current
    if (e != cudaSuccess) return cuda_check(e, "cudaGetSymbolAddress(static scratch)");
    if (!p) return fail(GC_ERR_CUDA, "cudaGetSymbolAddress returned NULL");
    if (!ctx) ctx = current_context();
    c.ctx = ctx;
    c.addr = p;
  }
  *out = c.addr;
  return GC_OK;
}

}  // namespace
}  // namespace gc

using namespace gc;

extern "C" int gc_find_encoding_coeff_noalloc(const double* R, int ell, const int32_t* order, int N,
                                              int m, int delta, const int32_t* psi, int npat,
                                              double* E, float* C, uint8_t* delta_out,
                                              uint8_t* support, double* coef_err, double* est,
                                              void* stream) {
  if (N < 1 || m < 1 || delta < 1 || ell < 1 || npat < 0)
    return fail(GC_ERR_SHAPE, "N, m, delta, ell >= 1 and npat >= 0 required");
  if (m > 32767) return fail(GC_ERR_UNSUPPORTED, "m=%d exceeds 32767", m);
  if (delta > GC_MAX_DELTA) return fail(GC_ERR_UNSUPPORTED, "delta=%d exceeds %d", delta, GC_MAX_DELTA);
  if (ell > GC_MAX_ELL) return fail(GC_ERR_UNSUPPORTED, "ell=%d exceeds %d", ell, GC_MAX_ELL);
  if (!R || !order || (!psi && npat > 0)) return fail(GC_ERR_ARG, "R, order and psi must be non-NULL");
  if (npat == 0) return GC_OK;

  // Layout: status header, holder table, then the memo table when it fits;
  // without it every (pattern, chunk) block is solved directly.
  Carve probe(nullptr);
  carve_holders(probe, N);
  const size_t base = probe.bytes();
  int bits = solve_table_bits(N, m, delta, npat);
  size_t need = base + solve_table_bytes(N, ell, bits);
  if (need > GC_NOALLOC_SCRATCH_BYTES) {
    bits = -1;
    need = base;
  }
  if (need > GC_NOALLOC_SCRATCH_BYTES)
    return fail(GC_ERR_WORKSPACE,
                "N=%d needs %zu bytes of scratch; the static scratch holds %zu (use "
                "gc_find_encoding_coeff with a caller workspace)",
                N, need, (size_t)GC_NOALLOC_SCRATCH_BYTES);

  void* ws = nullptr;
  int rc = scratch_address(&ws);
  if (rc) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e = cudaMemsetAsync(ws, 0, kHeaderBytes, s);  // status header starts clear
  if (e != cudaSuccess) return cuda_check(e, "cudaMemsetAsync(static scratch header)");
  Carve c(ws);
  Holders h = carve_holders(c, N);
  void* table = bits >= 0 ? c.take<char>(solve_table_bytes(N, ell, bits)) : nullptr;
  uint32_t* status = static_cast<uint32_t*>(ws);
  launch_holders(order, N, m, delta, h, status, s);
  SolveOut out{E, C, delta_out, support, coef_err, est};
  return launch_solve_impl(R, ell, psi, h, N, m, delta, npat, out, table, bits, status, s);
}
