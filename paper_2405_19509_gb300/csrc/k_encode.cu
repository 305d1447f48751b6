// Worker encoding (eq. 2), PS decoding of transmissions (Sec. II-B) and the
// parameter update (Sec. I).
//
// All three are HBM-bound streaming kernels with coalesced accesses along the
// block coordinate c (consecutive threads, consecutive columns).
#include <algorithm>

#include "gc_internal.cuh"

namespace gc {

// T[b][j][c] = sum_{p < psi[b][j]} sum_k E[b][j][p][k] * g_{order[j][p]}[k*L + c]
// (g zero past d).  Block = (column stripe, worker j, group of up to
// kEncPats patterns).  The patterns share worker j's chunk list, so each
// thread loads g_{order[j][p]}[k*L + c] once per slot p and feeds it to
// every pattern of the group that processed slot p (kEncPats accumulators)
// instead of once per pattern; threads take V consecutive columns (16-byte
// loads when rows are 16-byte aligned) and stride over the block's columns,
// so the staging of the group's coefficients (fp32) and processed counts in
// shared memory -- kEncPats * (delta * ell + 1) + delta words, small enough to
// fit beside a resident kernel that holds nearly all of an SM's -- is paid
// once per block, not once per 256 columns.
constexpr int kEncPats = 8;
constexpr int kEncThreads = 256;
template <int V>
__global__ void __launch_bounds__(kEncThreads)
    k_encode(const double* __restrict__ E, const int32_t* __restrict__ order,
             const int32_t* __restrict__ psi, int N, int m, int delta, int ell, int npat,
             const float* __restrict__ G, int d, int L, float* __restrict__ T) {
  extern __shared__ float s_dyn[];
  // worker j varies fastest across the grid, so the blocks resident at one
  // time cover all workers on a few column stripes: the chunk-gradient
  // columns they read (each used by every holder of the chunk) stay in L2,
  // where worker-major order swept whole rows of many chunks and re-read them
  const int j = blockIdx.x, b0 = blockIdx.z * kEncPats;
  const int nb = min(kEncPats, npat - b0);
  const int de = delta * ell;
  float* s_e = s_dyn;                                                // [nb][delta * ell]
  int* s_np = reinterpret_cast<int*>(s_dyn + kEncPats * de);         // [kEncPats]
  int* s_chunk = s_np + kEncPats;                                    // [delta]
  if (threadIdx.x < kEncPats) {
    int np = 0;
    if ((int)threadIdx.x < nb) {
      np = psi[(size_t)(b0 + threadIdx.x) * m + j];
      np = np < 0 ? 0 : (np > delta ? delta : np);  // bad values are flagged by the solve
    }
    s_np[threadIdx.x] = np;
  }
  for (int t = threadIdx.x; t < nb * de; t += blockDim.x) {
    const int bb = t / de, r = t - bb * de;
    s_e[t] = (float)E[((size_t)(b0 + bb) * m + j) * de + r];
  }
  for (int t = threadIdx.x; t < delta; t += blockDim.x) s_chunk[t] = order[(size_t)j * delta + t];
  __syncthreads();
  int pmax = 0;
#pragma unroll
  for (int bb = 0; bb < kEncPats; ++bb) pmax = max(pmax, s_np[bb]);
  for (int c = (blockIdx.y * kEncThreads + threadIdx.x) * V; c < L; c += gridDim.y * kEncThreads * V) {
    float acc[kEncPats][V];
#pragma unroll
    for (int bb = 0; bb < kEncPats; ++bb)
#pragma unroll
      for (int v = 0; v < V; ++v) acc[bb][v] = 0.f;
    for (int p = 0; p < pmax; ++p) {
      const int i = s_chunk[p];
      if (i < 0 || i >= N) continue;
      const float* gi = G + (size_t)i * d;
      for (int k = 0; k < ell; ++k) {
        const int col = k * L + c;
        float g[V];
        if (V == 4 && col + 3 < d) {
          const float4 q = __ldg(reinterpret_cast<const float4*>(gi + col));
          g[0] = q.x; g[V > 1 ? 1 : 0] = q.y; g[V > 2 ? 2 : 0] = q.z; g[V > 3 ? 3 : 0] = q.w;
        } else {
#pragma unroll
          for (int v = 0; v < V; ++v) g[v] = (c + v < L && col + v < d) ? __ldg(gi + col + v) : 0.f;
        }
#pragma unroll
        for (int bb = 0; bb < kEncPats; ++bb)
          if (p < s_np[bb]) {
            const float e = s_e[bb * de + p * ell + k];
#pragma unroll
            for (int v = 0; v < V; ++v) acc[bb][v] = fmaf(e, g[v], acc[bb][v]);
          }
      }
    }
#pragma unroll
    for (int bb = 0; bb < kEncPats; ++bb) {
      if (bb >= nb) break;
      float* Tr = T + ((size_t)(b0 + bb) * m + j) * L + c;
      if (V == 4 && c + 3 < L) {
        *reinterpret_cast<float4*>(Tr) = make_float4(acc[bb][0], acc[bb][V > 1 ? 1 : 0],
                                                     acc[bb][V > 2 ? 2 : 0], acc[bb][V > 3 ? 3 : 0]);
      } else {
#pragma unroll
        for (int v = 0; v < V; ++v)
          if (c + v < L) Tr[v] = acc[bb][v];
      }
    }
  }
}

int launch_encode(const double* E, const int32_t* order, const int32_t* psi, int N, int m,
                  int delta, int ell, int npat, const float* G, int d, float* T, cudaStream_t s) {
  const int L = (d + ell - 1) / ell;
  if ((long long)npat * m * L == 0) return GC_OK;
  const int groups = (npat + kEncPats - 1) / kEncPats;
  if (groups > 65535 || m > 65535) return fail(GC_ERR_UNSUPPORTED, "encode grid: npat / 8 and m <= 65535");
  // 16-byte column vectors when every row start is 16-byte aligned
  const bool vec = d % 4 == 0 && L % 4 == 0 && reinterpret_cast<uintptr_t>(G) % 16 == 0 &&
                   reinterpret_cast<uintptr_t>(T) % 16 == 0;
  const int V = vec ? 4 : 1;
  const long long stripes = ((long long)L + (long long)kEncThreads * V - 1) / ((long long)kEncThreads * V);
  // enough blocks for a few waves; each block strides over the rest of its row
  const long long want = std::max<long long>(1, (long long)device_sm_count() * 32 / ((long long)m * groups));
  const int gx = (int)std::max<long long>(1, std::min<long long>(stripes, want));
  dim3 grid(m, gx, groups);
  const size_t smem = ((size_t)kEncPats * delta * ell + kEncPats + delta) * sizeof(float);
  if (vec)
    k_encode<4><<<grid, kEncThreads, smem, s>>>(E, order, psi, N, m, delta, ell, npat, G, d, L, T);
  else
    k_encode<1><<<grid, kEncThreads, smem, s>>>(E, order, psi, N, m, delta, ell, npat, G, d, L, T);
  count_launches(1);
  return cuda_check(cudaGetLastError(), "k_encode");
}

// ghat[b][k*L + c] = sum_j R[k][j] * T[b][j][c].  One thread per (b, c); R is
// staged in dynamic shared memory as fp32 (ELL * m words, m <= kDecodeSmemM)
// or read as fp64.  The transmissions are loaded eight workers at a time, so
// that eight independent loads are in flight per thread (the kernel is
// latency-bound at the sizes of one live realization).
constexpr int kDecodeSmemM = 1024;
template <int ELL, bool STAGED>
__global__ void k_decode_tx(const double* __restrict__ R, int m, const float* __restrict__ T,
                            int npat, int d, int L, float* __restrict__ ghat) {
  extern __shared__ float s_r[];
  if (STAGED) {
    for (int t = threadIdx.x; t < ELL * m; t += blockDim.x) s_r[t] = (float)R[t];
    __syncthreads();
  }
  const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (long long)npat * L) return;
  const int c = (int)(idx % L);
  const int b = (int)(idx / L);
  float acc[ELL];
#pragma unroll
  for (int k = 0; k < ELL; ++k) acc[k] = 0.f;
  const float* Tb = T + (size_t)b * m * L + c;
  for (int j0 = 0; j0 < m; j0 += 8) {
    float t[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) t[u] = j0 + u < m ? __ldg(Tb + (size_t)(j0 + u) * L) : 0.f;
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      if (j0 + u < m) {
#pragma unroll
        for (int k = 0; k < ELL; ++k) {
          const float r = STAGED ? s_r[k * m + j0 + u] : (float)__ldg(R + (size_t)k * m + j0 + u);
          acc[k] = fmaf(r, t[u], acc[k]);
        }
      }
    }
  }
#pragma unroll
  for (int k = 0; k < ELL; ++k) {
    const int col = k * L + c;
    if (col < d) ghat[(size_t)b * d + col] = acc[k];
  }
}

int launch_decode_tx(const double* R, int ell, int m, const float* T, int npat, int d, float* ghat,
                     cudaStream_t s) {
  const int L = (d + ell - 1) / ell;
  const long long tot = (long long)npat * L;
  if (tot == 0) return GC_OK;
  const int threads = 128;
  const unsigned blocks = (unsigned)((tot + threads - 1) / threads);
  const bool staged = m <= kDecodeSmemM;
  const size_t sm = staged ? (size_t)ell * m * sizeof(float) : 0;
#define GC_DTX(E)                                                                              \
  case E:                                                                                      \
    if (staged)                                                                                \
      k_decode_tx<E, true><<<blocks, threads, sm, s>>>(R, m, T, npat, d, L, ghat);             \
    else                                                                                       \
      k_decode_tx<E, false><<<blocks, threads, 0, s>>>(R, m, T, npat, d, L, ghat);             \
    break;
  switch (ell) {
    GC_DTX(1)
    GC_DTX(2)
    GC_DTX(3)
    GC_DTX(4)
    GC_DTX(5)
    GC_DTX(6)
    GC_DTX(7)
    GC_DTX(8)
    default: return fail(GC_ERR_UNSUPPORTED, "ell=%d exceeds GC_MAX_ELL", ell);
  }
#undef GC_DTX
  count_launches(1);
  return cuda_check(cudaGetLastError(), "k_decode_tx");
}

// w[c] -= lr * ghat[c] / N~
__global__ void k_sgd(float* __restrict__ w, const float* __restrict__ ghat, int d, float scale) {
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c < d) w[c] = fmaf(-scale, ghat[c], w[c]);
}

int launch_sgd(float* w, const float* ghat, int d, float lr, int64_t Ntil, cudaStream_t s) {
  const float scale = (float)((double)lr / (double)Ntil);
  k_sgd<<<(d + 255) / 256, 256, 0, s>>>(w, ghat, d, scale);
  count_launches(1);
  return cuda_check(cudaGetLastError(), "k_sgd");
}

}  // namespace gc
