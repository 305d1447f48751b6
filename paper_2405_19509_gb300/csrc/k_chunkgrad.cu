// Chunk gradients (Sec. I): g_{D_i} = sum_{rows r of chunk i} grad l(x_r, y_r, w)
//                                    = X_i^T (f(X_i w) - y01_i),
// f = identity (least squares) or the logistic sigmoid, un-normalised as in
// Sec. I; the loss L = (1/N~) sum_r l(x_r, y_r, w) is fused in.
//
// GB300 design: the path is HBM bound (2 flops per element read), so X is read
// exactly once.  A cluster of CL CTAs owns a contiguous range of rows (a flat
// partition of all N~ rows, so every SM gets the same amount of X); CTA rank q
// of the cluster owns the column slice [q*Wc, (q+1)*Wc).  Rows arrive through
// a ring of S shared-memory stages filled by TMA bulk copies
// (cp.async.bulk, one per row slice, completion on an mbarrier).  For each
// stage of RB rows:
//   pass 1: every thread forms partial dot products of its columns with w;
//           they are reduced across the CTA (warp shuffles + shared memory)
//           and, when CL > 1, across the cluster through distributed shared
//           memory (st.shared::cluster + barrier.cluster);
//   then:   residual r = f(z) - y01 per row (and the loss term);
//   pass 2: acc[col] += r * x[row, col] from the same shared-memory stage.
// acc lives in registers; when the row range crosses into a new chunk the
// cluster writes its partial chunk gradient to a scratch slot, and a small
// second kernel adds the (at most a few) partials of every chunk in a fixed
// order, so results are deterministic.
//
// Rows that are not 16-byte multiples, or unaligned X, take the same kernel
// with plain cooperative loads instead of TMA (use_tma = 0).
#include <math.h>

#include <algorithm>
#include <mutex>

#include "gc_internal.cuh"

namespace gc {

namespace {

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
               : "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes,
                                         uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
          "r"(smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t mapa(uint32_t addr, uint32_t rank) {
  uint32_t out;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(out) : "r"(addr), "r"(rank));
  return out;
}
__device__ __forceinline__ void st_cluster_f32(uint32_t addr, float v) {
  asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(addr), "f"(v) : "memory");
}
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::
                   : "memory");
}

// Load V elements (16 bytes) of a row slice from shared memory as floats.
template <typename T>
struct Vec;
template <>
struct Vec<float> {
  static constexpr int V = 4;
  __device__ static __forceinline__ void load(const float* p, float (&o)[4]) {
    const float4 v = *reinterpret_cast<const float4*>(p);
    o[0] = v.x; o[1] = v.y; o[2] = v.z; o[3] = v.w;
  }
  __device__ static __forceinline__ float scalar(const float* p) { return *p; }
};
template <>
struct Vec<__nv_bfloat16> {
  static constexpr int V = 8;
  __device__ static __forceinline__ void load(const __nv_bfloat16* p, float (&o)[8]) {
    const uint4 u = *reinterpret_cast<const uint4*>(p);
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      o[2 * k] = __uint_as_float(w[k] << 16);
      o[2 * k + 1] = __uint_as_float(w[k] & 0xffff0000u);
    }
  }
  __device__ static __forceinline__ float scalar(const __nv_bfloat16* p) {
    return __bfloat162float(*p);
  }
};

constexpr int kMaxStages = 4;
constexpr long long kSpinLimit = 1LL << 31;  // clock cycles (~1 s) per wait

struct CGArgs {
  const void* X;
  const float* y;
  const float* w;
  int d;          // row length (elements)
  int Wc;         // columns per CTA slice (multiple of V)
  int ld_s;       // shared-memory row stride of a stage (elements, multiple of V)
  int n_c;        // rows per chunk
  long long Ntil; // rows
  long long rpc;  // rows per cluster (multiple of RB)
  int RB;         // rows per stage
  int S;          // stages
  int maxt;       // chunk slots per cluster in `parts`
  int loss;
  int want_loss;
  int use_tma;
  float* parts;        // [clusters][maxt][d]
  double* loss_parts;  // [clusters]
  uint32_t* status;
};

template <typename T, int CL, int NT, int NVT, int RBM>
__global__ void __launch_bounds__(NT, 1) k_chunkgrad(CGArgs a) {
  constexpr int V = Vec<T>::V;
  constexpr int NW = NT / 32;
  extern __shared__ __align__(128) unsigned char smem[];
  T* stages = reinterpret_cast<T*>(smem);
  const size_t stage_elems = (size_t)RBM * a.ld_s;
  float* red = reinterpret_cast<float*>(smem + a.S * stage_elems * sizeof(T));  // [2][NW][RBM]
  float* zcl = red + 2 * NW * RBM;                                               // [2][CL][RBM]
  uint64_t* full = reinterpret_cast<uint64_t*>(zcl + 2 * CL * RBM + 2);          // [S] (8B aligned)
  volatile int& s_abort = *reinterpret_cast<int*>(full + kMaxStages);

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int rank = CL > 1 ? (int)cluster_rank() : 0;
  const long long q = blockIdx.x / CL;
  const long long r0 = q * a.rpc;
  const long long r1 = min(r0 + a.rpc, a.Ntil);
  const int nb = r0 < r1 ? (int)((r1 - r0) / a.RB) : 0;
  const int c0 = rank * a.Wc;
  const int nvs = a.Wc / V;  // vectors in this CTA's slice
  const T* X = static_cast<const T*>(a.X);

  // w slice in registers (zeros past d)
  float wv[NVT][V];
#pragma unroll
  for (int u = 0; u < NVT; ++u) {
    const int v = tid + u * NT;
#pragma unroll
    for (int e = 0; e < V; ++e) {
      const int col = c0 + v * V + e;
      wv[u][e] = (v < nvs && col < a.d) ? a.w[col] : 0.f;
    }
  }
  float acc[NVT][V];
#pragma unroll
  for (int u = 0; u < NVT; ++u)
#pragma unroll
    for (int e = 0; e < V; ++e) acc[u][e] = 0.f;

  if (tid == 0) {
    s_abort = 0;
    for (int s = 0; s < a.S; ++s) mbar_init(&full[s], 1);
    fence_mbar_init();
  }
  __syncthreads();
  if (CL > 1) cluster_sync_all();  // every peer has started before any DSMEM store

  const uint32_t row_bytes = (uint32_t)(a.Wc * sizeof(T));
  auto issue = [&](int n) {  // TMA loads of batch n into stage n % S (thread 0 only)
    const int s = n % a.S;
    mbar_expect_tx(&full[s], row_bytes * a.RB);
    const long long row = r0 + (long long)n * a.RB;
    for (int r = 0; r < a.RB; ++r)
      bulk_g2s(stages + s * stage_elems + (size_t)r * a.ld_s, X + (row + r) * a.d + c0, row_bytes,
               &full[s]);
  };
  if (a.use_tma && tid == 0)
    for (int n = 0; n < min(a.S, nb); ++n) issue(n);

  const long long first_chunk = r0 / a.n_c;
  long long cur = -1;
  double loss_acc = 0.0;

  auto flush = [&](long long chunk) {
    float* dst = a.parts + ((size_t)q * a.maxt + (size_t)(chunk - first_chunk)) * a.d;
#pragma unroll
    for (int u = 0; u < NVT; ++u) {
      const int v = tid + u * NT;
      if (v < nvs) {
#pragma unroll
        for (int e = 0; e < V; ++e) {
          const int col = c0 + v * V + e;
          if (col < a.d) dst[col] = acc[u][e];
        }
      }
    }
  };

  for (int n = 0; n < nb; ++n) {
    const int s = n % a.S;
    const long long row0 = r0 + (long long)n * a.RB;
    const long long chunk = row0 / a.n_c;
    if (chunk != cur) {
      if (cur >= 0) flush(cur);
#pragma unroll
      for (int u = 0; u < NVT; ++u)
#pragma unroll
        for (int e = 0; e < V; ++e) acc[u][e] = 0.f;
      cur = chunk;
    }
    T* st = stages + s * stage_elems;
    if (a.use_tma) {
      if (!s_abort) {
        const uint32_t parity = (uint32_t)((n / a.S) & 1);
        if (!mbar_try_wait(&full[s], parity)) {
          const long long t0 = clock64();
          while (!mbar_try_wait(&full[s], parity)) {
            if (clock64() - t0 > kSpinLimit) {
              atomicOr(a.status, ST_TIMEOUT);
              s_abort = 1;
              break;
            }
          }
        }
      }
    } else {
      // cooperative load with bounds (zero fill past d)
      for (int r = 0; r < a.RB; ++r) {
        const T* src = X + (row0 + r) * a.d;
        for (int c = tid; c < a.ld_s; c += NT) {
          const int col = c0 + c;
          st[(size_t)r * a.ld_s + c] = (c < a.Wc && col < a.d) ? src[col] : T(0.f);
        }
      }
      __syncthreads();
    }
    // ---- pass 1: partial dot products
    float pd[RBM];
#pragma unroll
    for (int r = 0; r < RBM; ++r) {
      pd[r] = 0.f;
      if (r < a.RB) {
#pragma unroll
        for (int u = 0; u < NVT; ++u) {
          const int v = tid + u * NT;
          if (v < nvs) {
            float x[V];
            Vec<T>::load(st + (size_t)r * a.ld_s + v * V, x);
#pragma unroll
            for (int e = 0; e < V; ++e) pd[r] = fmaf(x[e], wv[u][e], pd[r]);
          }
        }
      }
    }
#pragma unroll
    for (int r = 0; r < RBM; ++r)
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) pd[r] += __shfl_xor_sync(0xffffffffu, pd[r], o);
    float* redn = red + (n & 1) * NW * RBM;
    if (lane == 0)
#pragma unroll
      for (int r = 0; r < RBM; ++r) redn[warp * RBM + r] = pd[r];
    __syncthreads();
    // the previous stage is free now: refill it with batch n - 1 + S
    if (a.use_tma && tid == 0 && n >= 1 && n - 1 + a.S < nb && !s_abort) issue(n - 1 + a.S);
    float z[RBM];
#pragma unroll
    for (int r = 0; r < RBM; ++r) {
      float t = 0.f;
      for (int w = 0; w < NW; ++w) t += redn[w * RBM + r];
      z[r] = t;
    }
    if (CL > 1) {
      float* zc = zcl + (n & 1) * CL * RBM;
      if (tid < CL * RBM) {
        const int peer = tid / RBM, r = tid % RBM;
        st_cluster_f32(mapa(smem_u32(zc + rank * RBM + r), peer), z[r]);
      }
      cluster_sync_all();
#pragma unroll
      for (int r = 0; r < RBM; ++r) {
        float t = 0.f;
        for (int p = 0; p < CL; ++p) t += zc[p * RBM + r];
        z[r] = t;
      }
    }
    // ---- residuals
    float res[RBM];
#pragma unroll
    for (int r = 0; r < RBM; ++r) {
      res[r] = 0.f;
      if (r < a.RB) {
        const float yv = __ldg(a.y + row0 + r);
        if (a.loss == GC_LSQ) {
          res[r] = z[r] - yv;
        } else {
          const float sg = 1.f / (1.f + __expf(-z[r]));
          res[r] = sg - 0.5f * (yv + 1.f);
        }
      }
    }
    // ---- the loss: lane r of warp 0 takes row r (fp32), one fp64 add per batch
    if (a.want_loss && rank == 0 && warp == 0) {
      float lr = 0.f;
#pragma unroll
      for (int r = 0; r < RBM; ++r) {
        if (r < a.RB && lane == r) {
          const float yv = __ldg(a.y + row0 + r);
          if (a.loss == GC_LSQ) {
            const float e = z[r] - yv;
            lr = 0.5f * e * e;
          } else {
            const float t = -yv * z[r];  // log(1 + e^t), stable
            lr = fmaxf(t, 0.f) + log1pf(expf(-fabsf(t)));
          }
        }
      }
#pragma unroll
      for (int o = 2; o > 0; o >>= 1) lr += __shfl_xor_sync(0xffffffffu, lr, o);
      if (lane == 0) loss_acc += (double)lr;
    }
    // ---- pass 2: acc += r * x
#pragma unroll
    for (int r = 0; r < RBM; ++r) {
      if (r < a.RB) {
#pragma unroll
        for (int u = 0; u < NVT; ++u) {
          const int v = tid + u * NT;
          if (v < nvs) {
            float x[V];
            Vec<T>::load(st + (size_t)r * a.ld_s + v * V, x);
#pragma unroll
            for (int e = 0; e < V; ++e) acc[u][e] = fmaf(res[r], x[e], acc[u][e]);
          }
        }
      }
    }
    if (!a.use_tma) __syncthreads();
  }
  if (cur >= 0) flush(cur);
  if (tid == 0 && rank == 0) a.loss_parts[q] = loss_acc;
  if (CL > 1) cluster_sync_all();  // keep shared memory alive until peers are done
}

// G[i][col] = sum of the partials of chunk i, clusters in increasing order.
__global__ void k_chunkgrad_reduce(const float* __restrict__ parts,
                                   const double* __restrict__ loss_parts, float* __restrict__ G,
                                   double* loss_out, int N, int n_c, int d, long long rpc,
                                   int maxt, int nclusters, long long Ntil) {
  const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx < (long long)N * d) {
    const int i = (int)(idx / d);
    const int col = (int)(idx - (long long)i * d);
    const long long qlo = ((long long)i * n_c) / rpc;
    const long long qhi = ((long long)(i + 1) * n_c - 1) / rpc;
    float s = 0.f;
    for (long long q = qlo; q <= qhi; ++q) {
      const long long first = (q * rpc) / n_c;
      s += parts[((size_t)q * maxt + (size_t)(i - first)) * d + col];
    }
    G[idx] = s;
  }
  if (loss_out && idx == 0) {
    double t = 0.0;
    for (int q = 0; q < nclusters; ++q) t += loss_parts[q];
    *loss_out = t / (double)Ntil;
  }
}

// ---------------------------------------------------------------------------
// Host-side plan
// ---------------------------------------------------------------------------
struct Plan {
  int CL, NT, NVT, RBM, RB, S, Wc, ld_s, V, use_tma;
  long long rpc;
  int nclusters, maxt;
  size_t smem;
};

Plan make_plan(int N, int n_c, int d, int x_dtype, bool tma_ok) {
  Plan p{};
  const int esz = x_dtype == GC_BF16 ? 2 : 4;
  p.V = 16 / esz;
  // cluster size: row slice per CTA at most 32 KB
  const long long row_bytes = (long long)d * esz;
  p.CL = 1;
  while (p.CL < 8 && row_bytes / p.CL > 32768) p.CL *= 2;
  p.use_tma = tma_ok && (row_bytes % 16 == 0) && (d % (p.CL * p.V) == 0);
  p.Wc = p.use_tma ? d / p.CL : (int)align_up((size_t)((d + p.CL - 1) / p.CL), (size_t)p.V);
  p.ld_s = p.Wc;  // stage row stride (elements)
  const int nv = p.Wc / p.V;
  p.NT = nv >= 1024 ? 512 : (nv >= 256 ? 256 : 128);
  p.NVT = (nv + p.NT - 1) / p.NT;
  if (p.NVT > 4) p.NVT = 4;  // nv <= 4 * 512 because Wc * esz <= 32 KB
  p.NVT = p.NVT <= 1 ? 1 : (p.NVT <= 2 ? 2 : 4);
  p.RBM = p.NVT >= 4 ? 2 : 4;
  p.RB = p.RBM;
  while (p.RB > 1 && n_c % p.RB != 0) p.RB /= 2;
  const size_t stage_bytes = (size_t)p.RBM * p.ld_s * esz;
  p.S = (int)std::min<size_t>(kMaxStages, std::max<size_t>(2, (192 * 1024) / stage_bytes));
  const int NW = p.NT / 32;
  p.smem = p.S * stage_bytes + (2 * NW * p.RBM + 2 * p.CL * p.RBM + 2) * sizeof(float) +
           kMaxStages * sizeof(uint64_t) + 16;
  // flat row partition over one wave of clusters
  const int sms = device_sm_count();
  const long long Ntil = (long long)N * n_c;
  long long waves_cl = std::max(1, sms / p.CL);
  long long rpc = (Ntil + waves_cl - 1) / waves_cl;
  rpc = ((rpc + p.RB - 1) / p.RB) * p.RB;
  if (rpc < p.RB) rpc = p.RB;
  p.rpc = rpc;
  p.nclusters = (int)((Ntil + rpc - 1) / rpc);
  p.maxt = (int)((rpc + n_c - 1) / n_c) + 1;
  return p;
}

template <typename T, int CL, int NT, int NVT, int RBM>
int launch_one(const Plan& p, const CGArgs& a, cudaStream_t s) {
  auto kern = k_chunkgrad<T, CL, NT, NVT, RBM>;
  static int smem_set = 0;  // largest opt-in so far (per instantiation)
  cudaError_t e;
  if ((int)p.smem > smem_set) {
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)p.smem);
    if (e != cudaSuccess) return cuda_check(e, "cudaFuncSetAttribute(chunkgrad smem)");
    smem_set = (int)p.smem;
  }
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(p.nclusters * CL);
  cfg.blockDim = dim3(NT);
  cfg.dynamicSmemBytes = p.smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = CL;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, kern, a);
  if (e != cudaSuccess) return cuda_check(e, "cudaLaunchKernelEx(chunkgrad)");
  count_launches(1);
  return GC_OK;
}

template <typename T, int CL>
int dispatch_nt(const Plan& p, const CGArgs& a, cudaStream_t s) {
  if (p.NT == 512) {
    if (p.NVT == 4) return launch_one<T, CL, 512, 4, 2>(p, a, s);
    if (p.NVT == 2) return launch_one<T, CL, 512, 2, 4>(p, a, s);
    return launch_one<T, CL, 512, 1, 4>(p, a, s);
  }
  if (p.NT == 256) {
    if (p.NVT == 4) return launch_one<T, CL, 256, 4, 2>(p, a, s);
    return launch_one<T, CL, 256, 1, 4>(p, a, s);
  }
  return launch_one<T, CL, 128, 1, 4>(p, a, s);
}

template <typename T>
int dispatch_cl(const Plan& p, const CGArgs& a, cudaStream_t s) {
  switch (p.CL) {
    case 1: return dispatch_nt<T, 1>(p, a, s);
    case 2: return dispatch_nt<T, 2>(p, a, s);
    case 4: return dispatch_nt<T, 4>(p, a, s);
    default: return dispatch_nt<T, 8>(p, a, s);
  }
}

}  // namespace

size_t chunkgrad_ws_bytes(int N, int n_c, int d, int x_dtype) {
  const Plan p = make_plan(N, n_c, d, x_dtype, true);
  const Plan p2 = make_plan(N, n_c, d, x_dtype, false);
  const size_t parts = std::max((size_t)p.nclusters * p.maxt, (size_t)p2.nclusters * p2.maxt) *
                       (size_t)d * sizeof(float);
  const size_t lp = (size_t)std::max(p.nclusters, p2.nclusters) * sizeof(double);
  return align_up(parts, 256) + align_up(lp, 256);
}

int launch_chunkgrad(const void* X, int x_dtype, const float* y, const float* w, int N, int n_c,
                     int d, int loss, float* G, double* loss_out, Carve& ws, uint32_t* status,
                     cudaStream_t s) {
  const bool aligned = (reinterpret_cast<uintptr_t>(X) % 16) == 0;
  const Plan p = make_plan(N, n_c, d, x_dtype, aligned);
  CGArgs a{};
  a.X = X;
  a.y = y;
  a.w = w;
  a.d = d;
  a.Wc = p.Wc;
  a.ld_s = p.ld_s;
  a.n_c = n_c;
  a.Ntil = (long long)N * n_c;
  a.rpc = p.rpc;
  a.RB = p.RB;
  a.S = p.S;
  a.maxt = p.maxt;
  a.loss = loss;
  a.want_loss = loss_out != nullptr;
  a.use_tma = p.use_tma;
  a.parts = ws.take<float>((size_t)p.nclusters * p.maxt * d);
  a.loss_parts = ws.take<double>(p.nclusters);
  a.status = status;
  int rc = x_dtype == GC_BF16 ? dispatch_cl<__nv_bfloat16>(p, a, s) : dispatch_cl<float>(p, a, s);
  if (rc != GC_OK) return rc;
  const long long tot = (long long)N * d;
  const int threads = 256;
  const long long blocks = std::max<long long>(1, (tot + threads - 1) / threads);
  k_chunkgrad_reduce<<<(unsigned)blocks, threads, 0, s>>>(a.parts, a.loss_parts, G, loss_out, N,
                                                          n_c, d, p.rpc, p.maxt, p.nclusters,
                                                          a.Ntil);
  count_launches(1);
  return cuda_check(cudaGetLastError(), "k_chunkgrad_reduce");
}

}  // namespace gc
