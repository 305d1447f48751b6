// Worker encoding (eq. 2), PS decoding of transmissions (Sec. II-B) and the
// parameter update (Sec. I).
//
// All three are HBM-bound streaming kernels with coalesced accesses along the
// block coordinate c (consecutive threads, consecutive columns).
#include "gc_internal.cuh"

namespace gc {

// T[b][j][c] = sum_{p < psi[b][j]} sum_k E[b][j][p][k] * g_{order[j][p]}[k*L + c]
// (g zero past d).  Block = (column tile, worker j, pattern b); worker j's
// coefficients and chunk list are staged in shared memory (fp32) once per
// block -- delta * (ell + 1) words of dynamic shared memory, so the kernel
// still fits beside a resident kernel that holds nearly all of an SM's.
__global__ void k_encode(const double* __restrict__ E, const int32_t* __restrict__ order,
                         const int32_t* __restrict__ psi, int N, int m, int delta, int ell,
                         int npat, const float* __restrict__ G, int d, int L,
                         float* __restrict__ T) {
  extern __shared__ float s_dyn[];
  float* s_e = s_dyn;                                          // [delta * ell]
  int* s_chunk = reinterpret_cast<int*>(s_dyn + delta * ell);  // [delta]
  const int j = blockIdx.y, b = blockIdx.z;
  int np = psi[(size_t)b * m + j];
  np = np < 0 ? 0 : (np > delta ? delta : np);  // bad values are flagged by the solve
  const double* Ej = E + ((size_t)b * m + j) * delta * ell;
  for (int t = threadIdx.x; t < np * ell; t += blockDim.x) s_e[t] = (float)Ej[t];
  for (int t = threadIdx.x; t < np; t += blockDim.x) s_chunk[t] = order[(size_t)j * delta + t];
  __syncthreads();
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= L) return;
  float acc = 0.f;
#pragma unroll 4
  for (int p = 0; p < np; ++p) {
    const int i = s_chunk[p];
    if (i < 0 || i >= N) continue;
    const float* gi = G + (size_t)i * d;
    for (int k = 0; k < ell; ++k) {
      const int col = k * L + c;
      if (col < d) acc = fmaf(s_e[p * ell + k], __ldg(gi + col), acc);
    }
  }
  T[((size_t)b * m + j) * L + c] = acc;
}

int launch_encode(const double* E, const int32_t* order, const int32_t* psi, int N, int m,
                  int delta, int ell, int npat, const float* G, int d, float* T, cudaStream_t s) {
  const int L = (d + ell - 1) / ell;
  if ((long long)npat * m * L == 0) return GC_OK;
  if (npat > 65535 || m > 65535) return fail(GC_ERR_UNSUPPORTED, "encode grid: npat and m <= 65535");
  const int threads = 256;
  dim3 grid((L + threads - 1) / threads, m, npat);
  const size_t smem = (size_t)delta * (ell + 1) * sizeof(float);
  k_encode<<<grid, threads, smem, s>>>(E, order, psi, N, m, delta, ell, npat, G, d, L, T);
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
