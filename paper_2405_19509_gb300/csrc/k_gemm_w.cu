// Chunk gradients for n_w parameter vectors at once on the tensor cores:
//   G[w][i] = X_i^T (f(X_i w_w) - y01_i)        (Sec. I, one column per w_w)
// With several parameter vectors (replicas, a learning-rate sweep) the two
// matrix-vector products per chunk become two dense contractions:
//   GEMM 1:  Z = X W^T            (N~ x n_w, K = d), epilogue R = f(Z) - y01
//   GEMM 2:  G_i = X_i^T R_i      (d x n_w per chunk, K = n_c)
// X is bf16 (exact as an MMA operand); W and R are fp32 split into bf16
// hi + lo planes (relative error 2^-17), so each K step issues two kind::f16
// MMAs (X W_hi + X W_lo) with fp32 accumulation in TMEM.
//
// One persistent kernel shape serves both GEMMs (MODE 0, MODE 1).  A tile is
// 256 x n_w: two 128-row halves that share every B load (the B operand is
// what each CTA would otherwise re-read from L2 per 128 rows).  Warp 0
// issues TMA loads into a ring of stages (two A halves 128 x 64 bf16, B
// n_w x 64 in two planes), warp 1 allocates 512 TMEM columns and one lane
// issues four MMAs per K step (two halves x W or R hi/lo), warps 2..9 drain
// the accumulators (tcgen05.ld; one warp per TMEM lane quarter and half).
// With n_w <= 128 the accumulators are double-buffered so that the
// epilogue of a tile overlaps the next tile's MMAs.
//   MODE 0: A = X rows (K-major, 128-byte swizzle); B = W planes (K-major).
//           The epilogue forms r = f(z) - y01 per (row, w) and writes R^T as
//           bf16 hi/lo planes [2][n_w][N~] -- GEMM 2's K-major B operand.
//   MODE 1: A = X_i^T, read MN-major straight from row-major X (two 64-column
//           boxes per K block: LBO = 8 KB between the 64-element MN atoms,
//           SBO = 1 KB between 8-row K groups); B = R^T planes of chunk i.
//           The epilogue writes G[w][i][col] (coalesced along col per w).
// Tiles are visited so that concurrently running CTAs share the B operand
// through L2 (all of W in MODE 0; R_i of one chunk in MODE 1).  Every wait
// is bounded (GC_ERR_TIMEOUT, drain, return).
#include <cudaTypedefs.h>
#include <string.h>

#include <algorithm>

#include "tc_ptx.cuh"

namespace gc {
namespace {

using namespace tcw;

constexpr int BM = 128, BK = 64;       // one MMA half: 128 rows (MODE 0) or columns (MODE 1)
constexpr int TM = 2 * BM;             // rows (columns) of a tile
constexpr int A_BYTES = BM * BK * 2;   // 16 KB per half
constexpr int kMaxStagesW = 4;
constexpr int kEpiW = 8;               // epilogue warps: 4 lane quarters x 2 halves
constexpr int kThreadsW = 64 + 32 * kEpiW;
constexpr long long kSpinW = 1LL << 32;

struct WParams {
  int n_w, d, n_c, N;
  long long Ntil;
  long long num_tiles;
  int num_m_tiles;   // MODE 0: ceil(N~ / 256); MODE 1: ceil(d / 256) (per chunk)
  int nkb;           // 64-wide K blocks per tile
  int stages;
  int stage_bytes;   // 2 * A_BYTES + 256 * n_w
  int nbuf;          // accumulator buffers (2 when 2 * n_w <= 256)
  int loss;
  const float* y;
  __nv_bfloat16* Rt;  // MODE 0 output: planes [2][n_w][N~]
  float* G;           // MODE 1 output: [n_w][N][d]
  long long spin_limit;
  int stall;  // failure-path test: the TMA producer issues nothing
  uint32_t* status;
};

template <int MODE>
__global__ void __launch_bounds__(kThreadsW, 1)
    k_gemm_w(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
             WParams p) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const int S = p.stages;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + (size_t)S * p.stage_bytes);
  uint64_t* empty = full + kMaxStagesW;
  uint64_t* tfull = empty + kMaxStagesW;  // [2]
  uint64_t* tempty = tfull + 2;           // [2]
  uint64_t* done = tempty + 2;
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(done + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], kEpiW);
    }
    mbar_init(done, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tmem_holder)),
                 "r"(512)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem_base = *tmem_holder;
  const int n_w = p.n_w;
  const uint32_t b_plane = (uint32_t)n_w * 128u;  // bytes of one B plane in a stage

  if (warp == 0) {
    // ------------------------------------------------------------- producer
    if (lane == 0) {
      uint32_t it = 0;
      bool ok = !p.stall;
      for (long long t = blockIdx.x; t < p.num_tiles && ok; t += gridDim.x) {
        int a_x, a_y;  // MODE 0: (k, row0); MODE 1: (col0, row0)
        if (MODE == 0) {
          a_x = 0;
          a_y = (int)(t * TM);
        } else {
          const int i = (int)(t / p.num_m_tiles), mt = (int)(t % p.num_m_tiles);
          a_x = mt * TM;
          a_y = i * p.n_c;
        }
        for (int kb = 0; kb < p.nkb; ++kb, ++it) {
          const int s = it % S;
          const uint32_t ph = (it / S) & 1;
          if (!mbar_wait(&empty[s], ph ^ 1, abort_flag, p.status, p.spin_limit)) {
            ok = false;
            break;
          }
          uint8_t* st = smem + (size_t)s * p.stage_bytes;
          mbar_expect_tx(&full[s], (uint32_t)p.stage_bytes);
          if (MODE == 0) {
            tma_load_2d(st, &tmA, kb * BK, a_y, &full[s]);
            tma_load_2d(st + A_BYTES, &tmA, kb * BK, a_y + BM, &full[s]);
            tma_load_3d(st + 2 * A_BYTES, &tmB, kb * BK, 0, 0, &full[s]);
          } else {
            for (int q = 0; q < 4; ++q)  // half q/2, 64-column atom q%2
              tma_load_2d(st + q * (A_BYTES / 2), &tmA, a_x + 64 * q, a_y + kb * BK, &full[s]);
            tma_load_3d(st + 2 * A_BYTES, &tmB, a_y + kb * BK, 0, 0, &full[s]);
          }
        }
      }
      // drain: every issued stage has landed before the CTA may exit
      const uint32_t issued = it;
      for (uint32_t k = (issued > (uint32_t)S ? issued - S : 0); k < issued; ++k) {
        volatile int no_abort = 0;
        mbar_wait(&full[k % S], (k / S) & 1, &no_abort, p.status, 1LL << 28);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(n_w, MODE == 1);
      uint32_t it = 0, tile_it = 0;
      bool ok = true;
      for (long long t = blockIdx.x; t < p.num_tiles && ok; t += gridDim.x, ++tile_it) {
        const int ab = p.nbuf == 2 ? (int)(tile_it & 1) : 0;
        const uint32_t use = p.nbuf == 2 ? (tile_it >> 1) : tile_it;  // uses of buffer ab so far
        if (!mbar_wait(&tempty[ab], (use & 1) ^ 1, abort_flag, p.status, p.spin_limit)) break;
        fence_after();
        // half h accumulates at column ab * 2 n_w + h n_w (nbuf 2) or h * 256 (nbuf 1)
        const uint32_t d0 = tmem_base + (uint32_t)(p.nbuf == 2 ? ab * 2 * n_w : 0);
        const uint32_t d1 = d0 + (uint32_t)(p.nbuf == 2 ? n_w : 256);
        for (int kb = 0; kb < p.nkb; ++kb, ++it) {
          const int s = it % S;
          if (!mbar_wait(&full[s], (it / S) & 1, abort_flag, p.status, p.spin_limit)) {
            ok = false;
            break;
          }
          fence_after();
          const uint32_t a0 = smem_u32(smem + (size_t)s * p.stage_bytes);
          const uint32_t a1 = a0 + A_BYTES;
          const uint32_t b0 = a0 + 2 * A_BYTES;
#pragma unroll
          for (int ks = 0; ks < BK / 16; ++ks) {
            const uint64_t x0 = MODE == 0 ? sdesc(a0 + ks * 32, 16, 1024)
                                          : sdesc(a0 + ks * 2048, A_BYTES / 2, 1024);
            const uint64_t x1 = MODE == 0 ? sdesc(a1 + ks * 32, 16, 1024)
                                          : sdesc(a1 + ks * 2048, A_BYTES / 2, 1024);
            const uint64_t bh = sdesc(b0 + ks * 32, 16, 1024);
            const uint64_t bl = sdesc(b0 + b_plane + ks * 32, 16, 1024);
            const uint32_t acc = (kb > 0 || ks > 0) ? 1u : 0u;
            mma_bf16(d0, x0, bh, idesc, acc);
            mma_bf16(d0, x0, bl, idesc, 1u);
            mma_bf16(d1, x1, bh, idesc, acc);
            mma_bf16(d1, x1, bl, idesc, 1u);
          }
          mma_commit(&empty[s]);
        }
        if (!ok) break;
        mma_commit(&tfull[ab]);
      }
      mma_commit(done);
      volatile int no_abort = 0;
      mbar_wait(done, 0, &no_abort, p.status, 1LL << 28);
    }
  } else {
    // ------------------------------------------------------------- epilogue
    const int quarter = warp & 3;   // TMEM lanes 32*quarter .. +31
    const int half = (warp - 2) >> 2;  // which 128-row (column) half of the tile
    uint32_t tile_it = 0;
    for (long long t = blockIdx.x; t < p.num_tiles; t += gridDim.x, ++tile_it) {
      const int ab = p.nbuf == 2 ? (int)(tile_it & 1) : 0;
      const uint32_t use = p.nbuf == 2 ? (tile_it >> 1) : tile_it;
      // warp-uniform: the TMEM loads below are warp-collective
      const bool ready = mbar_wait(&tfull[ab], use & 1, abort_flag, p.status, p.spin_limit);
      if (!__all_sync(0xffffffffu, ready)) break;
      fence_after();
      const uint32_t col_base = (uint32_t)(p.nbuf == 2 ? ab * 2 * n_w + half * n_w : half * 256);
      const uint32_t taddr = tmem_base + ((uint32_t)(quarter * 32) << 16) + col_base;
      if (MODE == 0) {
        const long long row = t * TM + half * BM + quarter * 32 + lane;
        const bool rv = row < p.Ntil;
        const float yv = rv ? __ldg(p.y + row) : 0.f;
        const float y01 = p.loss == GC_LSQ ? yv : 0.5f * (yv + 1.f);
        for (int c = 0; c < n_w / 32; ++c) {
          float v[32];
          __syncwarp();
          tmem_ld32(taddr + (uint32_t)(c * 32), v);
          if (rv) {
#pragma unroll
            for (int j = 0; j < 32; ++j) {
              const float z = v[j];
              const float f = p.loss == GC_LSQ ? z : 1.f / (1.f + __expf(-z));
              const float r = f - y01;
              const __nv_bfloat16 hi = __float2bfloat16_rn(r);
              const __nv_bfloat16 lo = __float2bfloat16_rn(r - __bfloat162float(hi));
              const size_t w = (size_t)(c * 32 + j);
              p.Rt[w * p.Ntil + row] = hi;
              p.Rt[((size_t)n_w + w) * p.Ntil + row] = lo;
            }
          }
        }
      } else {
        const int i = (int)(t / p.num_m_tiles), mt = (int)(t % p.num_m_tiles);
        const int col = mt * TM + half * BM + quarter * 32 + lane;
        for (int c = 0; c < n_w / 32; ++c) {
          float v[32];
          __syncwarp();
          tmem_ld32(taddr + (uint32_t)(c * 32), v);
          if (col < p.d) {
#pragma unroll
            for (int j = 0; j < 32; ++j)
              p.G[((size_t)(c * 32 + j) * p.N + i) * p.d + col] = v[j];
          }
        }
      }
      fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[ab]);
    }
  }
  fence_before();
  __syncthreads();
  if (warp == 1) {
    fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(512)
                 : "memory");
  }
}

// W (n_w x d fp32) -> planes [2][n_w][d] bf16: hi = bf16(w), lo = bf16(w - hi).
__global__ void k_split_w(const float* __restrict__ W, long long n, __nv_bfloat16* __restrict__ out) {
  const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= n) return;
  const float v = W[idx];
  const __nv_bfloat16 hi = __float2bfloat16_rn(v);
  out[idx] = hi;
  out[n + idx] = __float2bfloat16_rn(v - __bfloat162float(hi));
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn_w() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  }
  return fn;
}

// 2-D bf16 map over a row-major (rows x cols) matrix, box {64, box_rows}, 128-byte swizzle.
int map_2d(CUtensorMap* map, const void* base, long long rows, long long cols, int box_rows) {
  auto fn = encode_fn_w();
  if (!fn) return fail(GC_ERR_CUDA, "cuTensorMapEncodeTiled entry point unavailable");
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
  cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(GC_ERR_CUDA, "cuTensorMapEncodeTiled(2d) failed (%d)", (int)r);
  return GC_OK;
}

// 3-D bf16 map over planes [2][rows][cols], box {64, rows, 2}, 128-byte swizzle.
int map_planes(CUtensorMap* map, const void* base, int rows, long long cols) {
  auto fn = encode_fn_w();
  if (!fn) return fail(GC_ERR_CUDA, "cuTensorMapEncodeTiled entry point unavailable");
  cuuint64_t dims[3] = {(cuuint64_t)cols, (cuuint64_t)rows, 2};
  cuuint64_t strides[2] = {(cuuint64_t)cols * 2, (cuuint64_t)rows * cols * 2};
  cuuint32_t box[3] = {64, (cuuint32_t)rows, 2};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(GC_ERR_CUDA, "cuTensorMapEncodeTiled(planes) failed (%d)", (int)r);
  return GC_OK;
}

template <int MODE>
int launch_w(const CUtensorMap& mA, const CUtensorMap& mB, const WParams& p, cudaStream_t s) {
  const size_t smem = (size_t)p.stages * p.stage_bytes + 1024 + 256;
  static size_t smem_set = 0;
  if (smem > smem_set) {
    cudaError_t e = cudaFuncSetAttribute(k_gemm_w<MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return cuda_check(e, "cudaFuncSetAttribute(k_gemm_w)");
    smem_set = smem;
  }
  const int grid = (int)std::min<long long>(p.num_tiles, device_sm_count());
  k_gemm_w<MODE><<<grid, kThreadsW, smem, s>>>(mA, mB, p);
  count_launches(1);
  return cuda_check(cudaGetLastError(), "k_gemm_w");
}

}  // namespace

size_t gemmw_ws_bytes(int N, int n_c, int d, int n_w) {
  const size_t Ntil = (size_t)N * n_c;
  return align_up((size_t)2 * n_w * d * 2, 256) + align_up((size_t)2 * n_w * Ntil * 2, 256);
}

int launch_chunkgrad_batched(const void* X, const float* y, const float* W, int N, int n_c, int d,
                             int n_w, int loss, float* G, Carve& ws, uint32_t* status,
                             cudaStream_t s) {
  const long long Ntil = (long long)N * n_c;
  __nv_bfloat16* Wp = ws.take<__nv_bfloat16>((size_t)2 * n_w * d);
  __nv_bfloat16* Rt = ws.take<__nv_bfloat16>((size_t)2 * n_w * Ntil);
  {
    const long long n = (long long)n_w * d;
    k_split_w<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(W, n, Wp);
    count_launches(1);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_check(e, "k_split_w");
  }
  WParams p{};
  p.n_w = n_w;
  p.d = d;
  p.n_c = n_c;
  p.N = N;
  p.Ntil = Ntil;
  p.stage_bytes = 2 * A_BYTES + 256 * n_w;
  p.stages = std::min(kMaxStagesW, (200 * 1024) / p.stage_bytes);
  p.nbuf = 2 * n_w <= 256 ? 2 : 1;
  p.loss = loss;
  p.y = y;
  p.Rt = Rt;
  p.G = G;
  p.spin_limit = wait_limit(kSpinW);
  p.stall = take_stall(GC_STALL_BATCHED) ? 1 : 0;
  p.status = status;
  CUtensorMap mA, mB;
  // GEMM 1: Z = X W^T, residual epilogue -> R^T planes
  int rc = map_2d(&mA, X, Ntil, d, BM);
  if (rc) return rc;
  rc = map_planes(&mB, Wp, n_w, d);
  if (rc) return rc;
  p.num_m_tiles = (int)((Ntil + TM - 1) / TM);
  p.num_tiles = p.num_m_tiles;
  p.nkb = d / BK;
  rc = launch_w<0>(mA, mB, p, s);
  if (rc) return rc;
  // GEMM 2: G_i = X_i^T R_i
  rc = map_2d(&mA, X, Ntil, d, 64);
  if (rc) return rc;
  rc = map_planes(&mB, Rt, n_w, Ntil);
  if (rc) return rc;
  p.stall = 0;
  p.num_m_tiles = (d + TM - 1) / TM;
  p.num_tiles = (long long)N * p.num_m_tiles;
  p.nkb = n_c / BK;
  return launch_w<1>(mA, mB, p, s);
}

}  // namespace gc
