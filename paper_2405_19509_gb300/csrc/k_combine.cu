// Batched decode-combine: the PS decode of Sec. II-B applied to the
// transmissions of eq. (2), for many straggler patterns at once.
//
// sum_j R[k][j] T_b[j] = sum_i sum_k' (R B_b)[k][i*ell+k'] g_{D_i}[k'], so with
// C (npat*ell x N*ell) from Algorithm 1 and G viewed as N*ell blocks of length
// L (row i*ell + k' = g_{D_i}[k'*L : (k'+1)*L], zero past d):
//     Ghat (npat*ell x L) = C . G.
// Row (b, k) of Ghat is block k of pattern b's decoded gradient.  Optionally
// the squared distance to sum_i g_{D_i} is reduced per pattern in the
// epilogue (partials per row and column slice, then a fixed-order sum).
//
// This file holds the portable SIMT fp32 kernel (register-tiled, 64 x 128
// tiles, K staged through shared memory).
#include <algorithm>

#include "gc_internal.cuh"

namespace gc {

namespace {
constexpr int BM = 64, BN = 128, BK = 16;

__device__ __forceinline__ void kahan_add(float& s, float& comp, float v) {
  const float y = v - comp;
  const float t = s + y;
  comp = (t - s) - y;
  s = t;
}

__global__ void __launch_bounds__(256) k_combine_simt(const float* __restrict__ C,
                                                      const float* __restrict__ G,
                                                      const float* __restrict__ gsum, int M,
                                                      int K, int L, int ell, int d, int nslices,
                                                      float* __restrict__ Ghat,
                                                      double* __restrict__ mse_part) {
  __shared__ float As[BK][BM + 4];
  __shared__ __align__(16) float Bs[BK][BN];
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  const int rbase = blockIdx.x * BM;
  const int slice = blockIdx.y;
  const int ntiles = (L + BN - 1) / BN;
  float sq[4], sqc[4];
#pragma unroll
  for (int r = 0; r < 4; ++r) sq[r] = sqc[r] = 0.f;

  for (int ct = slice; ct < ntiles; ct += nslices) {
    const int cbase = ct * BN;
    float acc[4][8];
#pragma unroll
    for (int r = 0; r < 4; ++r)
#pragma unroll
      for (int e = 0; e < 8; ++e) acc[r][e] = 0.f;
    for (int k0 = 0; k0 < K; k0 += BK) {
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        const int idx = tid + t * 256;
        const int r = idx / BK, kk = idx % BK;
        const int gr = rbase + r, gk = k0 + kk;
        As[kk][r] = (gr < M && gk < K) ? __ldg(C + (size_t)gr * K + gk) : 0.f;
      }
#pragma unroll
      for (int t = 0; t < 8; ++t) {
        const int idx = tid + t * 256;
        const int kk = idx / BN, c = idx % BN;
        const int gk = k0 + kk, gc = cbase + c;
        float v = 0.f;
        if (gk < K && gc < L) {
          const int i = gk / ell, kp = gk - i * ell;
          const int col = kp * L + gc;
          if (col < d) v = __ldg(G + (size_t)i * d + col);
        }
        Bs[kk][c] = v;
      }
      __syncthreads();
#pragma unroll
      for (int kk = 0; kk < BK; ++kk) {
        float a[4], b[8];
#pragma unroll
        for (int r = 0; r < 4; ++r) a[r] = As[kk][ty * 4 + r];
        const float4 b0 = *reinterpret_cast<const float4*>(&Bs[kk][tx * 4]);
        const float4 b1 = *reinterpret_cast<const float4*>(&Bs[kk][64 + tx * 4]);
        b[0] = b0.x; b[1] = b0.y; b[2] = b0.z; b[3] = b0.w;
        b[4] = b1.x; b[5] = b1.y; b[6] = b1.z; b[7] = b1.w;
#pragma unroll
        for (int r = 0; r < 4; ++r)
#pragma unroll
          for (int e = 0; e < 8; ++e) acc[r][e] = fmaf(a[r], b[e], acc[r][e]);
      }
      __syncthreads();
    }
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const int gr = rbase + ty * 4 + r;
      if (gr >= M) continue;
      const int b = gr / ell, k = gr - b * ell;
      float t = 0.f;
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        const int c = cbase + (e < 4 ? tx * 4 + e : 64 + tx * 4 + (e - 4));
        const int col = k * L + c;
        if (c < L && col < d) {
          if (Ghat) Ghat[(size_t)b * d + col] = acc[r][e];
          if (mse_part) {
            const float df = acc[r][e] - __ldg(gsum + col);
            t = fmaf(df, df, t);
          }
        }
      }
      if (mse_part) kahan_add(sq[r], sqc[r], t);
    }
  }
  if (mse_part) {
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      double v = (double)sq[r] - (double)sqc[r];
#pragma unroll
      for (int o = 8; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
      const int gr = rbase + ty * 4 + r;
      if (tx == 0 && gr < M) mse_part[(size_t)gr * nslices + slice] = v;
    }
  }
}

__global__ void k_mse_reduce(const double* __restrict__ mse_part, int npat, int ell, int nslices,
                             int d, double* __restrict__ grad_mse) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= npat) return;
  double s = 0.0;
  for (int k = 0; k < ell; ++k)
    for (int t = 0; t < nslices; ++t) s += mse_part[((size_t)b * ell + k) * nslices + t];
  grad_mse[b] = s / (double)d;
}

int combine_slices(long long M, int L) {
  const long long row_tiles = (M + BM - 1) / BM;
  const int col_tiles = (L + BN - 1) / BN;
  const long long target = 4LL * device_sm_count();
  long long s = (target + row_tiles - 1) / row_tiles;
  s = std::max(1LL, std::min<long long>(s, col_tiles));
  return (int)s;
}
}  // namespace

size_t combine_ws_bytes(int N, int ell, int npat, int d) {
  (void)N;
  const int L = (d + ell - 1) / ell;
  const long long M = (long long)npat * ell;
  const int ns = combine_slices(M, L);
  return align_up((size_t)M * ns * sizeof(double), 256) + align_up((size_t)d * sizeof(float), 256);
}

int launch_combine(const float* C, const float* G, const float* gsum, int N, int ell, int npat,
                   int d, float* Ghat, double* grad_mse, Carve& ws, uint32_t* status,
                   cudaStream_t s) {
  (void)status;
  const int L = (d + ell - 1) / ell;
  const long long M = (long long)npat * ell;
  const int K = N * ell;
  const int ns = combine_slices(M, L);
  double* mse_part = grad_mse ? ws.take<double>((size_t)M * ns) : nullptr;
  dim3 grid((unsigned)((M + BM - 1) / BM), (unsigned)ns);
  k_combine_simt<<<grid, 256, 0, s>>>(C, G, gsum, (int)M, K, L, ell, d, ns, Ghat, mse_part);
  count_launches(1);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_check(e, "k_combine_simt");
  if (grad_mse) {
    k_mse_reduce<<<(npat + 255) / 256, 256, 0, s>>>(mse_part, npat, ell, ns, d, grad_mse);
    count_launches(1);
    e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_check(e, "k_mse_reduce");
  }
  return GC_OK;
}

}  // namespace gc
