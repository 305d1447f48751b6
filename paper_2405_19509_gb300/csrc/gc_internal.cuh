// Internal declarations shared by the translation units of libgc.so.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "gc.h"

namespace gc {

// ---- status header at the start of every workspace ----------------------
enum : uint32_t {
  ST_BAD_PSI = 1u,     // psi outside [0, delta]
  ST_SINGULAR = 2u,    // a least-squares system was numerically rank deficient
  ST_TIMEOUT = 4u,     // a bounded mbarrier wait expired
  ST_BAD_ORDER = 8u,   // order entry outside [-1, N) or a chunk with > GC_MAX_REPL copies
};
constexpr size_t kHeaderBytes = 256;

struct WsHeader {
  uint32_t status;
  uint32_t info;
};

// ---- NVTX range around a host entry point (a named range on the profiler's
// timeline; no cost without a profiler attached) --------------------------
struct NvtxRange {
  explicit NvtxRange(const char* name);
  ~NvtxRange();
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

// ---- error reporting (thread-local, host) --------------------------------
int fail(int code, const char* fmt, ...);
int cuda_check(cudaError_t e, const char* what);
#define GC_CUDA(call)                                   \
  do {                                                  \
    cudaError_t e_ = (call);                            \
    if (e_ != cudaSuccess) return ::gc::cuda_check(e_, #call); \
  } while (0)

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Linear carving of a caller workspace into 256-byte aligned pieces.
struct Carve {
  char* base;
  size_t off;
  explicit Carve(void* b) : base(static_cast<char*>(b)), off(kHeaderBytes) {}
  template <typename T>
  T* take(size_t count) {
    T* p = base ? reinterpret_cast<T*>(base + off) : nullptr;
    off = align_up(off + count * sizeof(T), 256);
    return p;
  }
  size_t bytes() const { return off; }
};

int device_sm_count();

// Launch accounting for gc_kernel_launches().
void count_launches(int n);
// Limit (clock cycles) of the bounded device waits of kernels launched now:
// `dflt` unless gc_set_wait_limit set one.
long long wait_limit(long long dflt);
// True (once) when gc_inject_stall armed `bit` for the next launch.
bool take_stall(int bit);

// ---- holder table: copies of every chunk, sorted by worker --------------
// hold_w[i*GC_MAX_REPL + h], hold_p[...]: worker and slot of the h-th holder of
// chunk i (workers ascending, then slot); hold_cnt[i] holders.
struct Holders {
  int32_t* cnt;
  int16_t* w;
  int8_t* p;
};
Holders carve_holders(Carve& c, int N);
void launch_holders(const int32_t* order, int N, int m, int delta, Holders h, uint32_t* status,
                    cudaStream_t s);

// ---- batched chunk gradients on the tensor cores (k_gemm_w.cu) -----------
size_t gemmw_ws_bytes(int N, int n_c, int d, int n_w);
int launch_chunkgrad_batched(const void* X, const float* y, const float* W, int N, int n_c, int d,
                             int n_w, int loss, float* G, Carve& ws, uint32_t* status,
                             cudaStream_t s);

// ---- completion times and trigger (k_trigger.cu) --------------------------
constexpr int kTriggerMaxKeys = 2048;  // N * ell per realization
int launch_trigger(const int32_t* order, Holders h, int N, int m, int delta, const double* tau,
                   long long nsim, int ell, int theta, double* T, int32_t* psi, double* TF,
                   cudaStream_t s);

// ---- Algorithm 1 batched (k_solve.cu) -----------------------------------
struct SolveOut {
  double* E;          // npat x m x delta x ell (nullable)
  float* C;           // npat x ell x N*ell (nullable)
  uint8_t* delta_out; // npat x N (nullable)
  uint8_t* support;   // npat x N x m (nullable)
  double* coef_err;   // npat (nullable)
  double* est;        // npat (nullable)
  __nv_bfloat16* Cs;  // decode matrix as bf16 hi/lo planes [2][npat*ell][Kp] (nullable)
  int Kp;             // row stride of Cs: N*ell rounded up to whole 64-element blocks
};
// Memo table of every holder subset (bits = masks per chunk in log2, -1 = none).
int solve_table_bits(int N, int m, int delta, int npat);
size_t solve_table_bytes(int N, int ell, int bits);
int launch_solve_impl(const double* R, int ell, const int32_t* psi, Holders h, int N, int m,
                      int delta, int npat, SolveOut out, void* table_mem, int bits,
                      uint32_t* status, cudaStream_t s, bool build_table = true);

// ---- chunk gradients (k_chunkgrad.cu) -----------------------------------
size_t chunkgrad_ws_bytes(int N, int n_c, int d, int x_dtype);
int launch_chunkgrad(const void* X, int x_dtype, const float* y, const float* w, int N, int n_c,
                     int d, int loss, float* G, double* loss_out, Carve& ws, uint32_t* status,
                     cudaStream_t s);

// ---- encode / decode / update (k_encode.cu) -----------------------------
int launch_encode(const double* E, const int32_t* order, const int32_t* psi, int N, int m,
                  int delta, int ell, int npat, const float* G, int d, float* T, cudaStream_t s);
int launch_decode_tx(const double* R, int ell, int m, const float* T, int npat, int d, float* ghat,
                     cudaStream_t s);
int launch_sgd(float* w, const float* ghat, int d, float lr, int64_t Ntil, cudaStream_t s);
int launch_live_step(const double* E, const double* R, int ell, const int32_t* order, int N, int m,
                     int delta, const int32_t* psi, const float* G, int d, float lr, int64_t Ntil,
                     float* w, float* T, float* ghat, cudaStream_t s);

// ---- batched decode in residual form (k_decode_resid.cu) -----------------
// Per pattern the ordered list of decode blocks that differ from I_ell (chunk
// index and D = Pi - I); per 128-row tile of the decode the path that
// produces its rows (tflag = 1: the tensor-core GEMM; 0: the residual kernel)
// and, for a residual tile, the ordered list of its rows that need
// corrections, each with a slot of squared-error partials.
constexpr int kResidThreads = 256;
constexpr int kResidW = kResidThreads * 4;  // columns of one block per CTA (4 KB rows)
constexpr int kResidRcap = 32;              // corrected rows a residual tile may hold
struct ResidLists {
  int32_t* nnz;        // [npat] non-identity blocks (may exceed ksp)
  int32_t* idx;        // [npat][ksp] their chunks, ascending
  float* D;            // [npat][ksp][ell][ell] Pi - I
  int32_t* tflag;      // [ntiles]
  int32_t* dlist;      // [ntiles] the GEMM's tiles, ascending
  int32_t* ndense;     // one word: entries of dlist
  int32_t* rslot;      // [npat*ell] slot of a corrected row of a residual tile, else -1
  int32_t* rowlist;    // [ntiles][kResidRcap] corrected rows of each tile, ascending
  int32_t* tcount;     // [ntiles] entries of rowlist
  float* msp;          // [ntiles*kResidRcap][parts] squared-error partials, or null
  int ksp;             // list capacity per pattern
  int parts;           // partials per corrected row (column ranges x warps)
};
int resid_ksp(int ell);
size_t resid_ws_bytes(int N, int ell, int npat, int d);
ResidLists carve_resid(Carve& c, int N, int ell, int npat, int d, bool want_mse);
int launch_plan_scan(const __nv_bfloat16* Cs, int Kp, int N, int ell, int npat, int budget,
                     int policy, const ResidLists& rl, unsigned int* done_counter, cudaStream_t s);
int launch_gsum(const float* G, int N, int d, float* gsum, cudaStream_t s);
int launch_decode_resid(const float* G, const float* gsum, const ResidLists& rl, int ell, int npat,
                        int d, float* Ghat, cudaStream_t s);
// Process-wide path policy of the batched decode (gc_set_decode_policy).
int decode_policy();

// ---- batched decode-combine on the tensor cores (k_combine_tc.cu) --------
// K = N*ell padded to whole 64-element blocks (the GEMM's K extent).
inline int combine_kp(int N, int ell) { return (N * ell + 63) / 64 * 64; }
// bytes of the bf16 hi/lo planes of the decode matrix ("decode plan")
inline size_t plan_bytes(int N, int ell, int npat) {
  return align_up((size_t)2 * npat * ell * combine_kp(N, ell) * 2, 256);
}
// scratch of the GEMM side given the planes (G planes, sum of G, MSE partials)
size_t apply_ws_bytes(int N, int ell, int npat, int d);
// ---- gradient MSE through the Gram matrix of the chunk blocks (k_mse_gram.cu)
bool mse_gram_applies(int N, int ell, int npat);
size_t mse_gram_ws_bytes(int N, int ell, int d);
int launch_mse_gram(const __nv_bfloat16* Cs, int Kp, const float* G, int N, int ell, int npat,
                    int d, double* grad_mse, Carve& ws, cudaStream_t s);
int launch_apply(const __nv_bfloat16* Cs, const float* G, int N, int ell, int npat, int d,
                 float* Ghat, double* grad_mse, Carve& ws, uint32_t* status, cudaStream_t s);
// fp32 C (npat x ell x N*ell) -> planes
int launch_split_c(const float* C, int N, int ell, int npat, __nv_bfloat16* Cs, cudaStream_t s);

}  // namespace gc
