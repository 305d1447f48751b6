// Completion times and the encode-and-transmit trigger (Sec. II-A and
// Sec. IV), batched over simulated realizations of the cluster.
//
// Realization r gives every worker a time per chunk tau[r][j] (+inf for a
// failed worker).  W_j finishes the chunk in its slot p (1-based) at p *
// tau_j, so chunk D_i has been processed n_i(T) = #{holders j : O_ij tau_j
// <= T} times by time T, and the PS's error estimate (eq. (7) and the
// sentence after it) is est(T) = sum_i max(0, ell - n_i(T)).  With t_i^(k)
// the k-th smallest completion time of D_i, est(T) = #{(i, k <= ell) :
// t_i^(k) > T}; the first time the estimate reaches theta or less is
// therefore the (N ell - theta)-th smallest of the N ell values t_i^(k).
// theta = 0 gives the time at which every chunk has been processed ell
// times, i.e. exact recovery becomes possible.  The same time counting a
// copy only when its worker has finished all of its chunks (at delta_j
// tau_j) is the completion time of the original protocol (Sec. IV).
//
// GB300 design: one warp per realization.  Lanes take chunks, gather their
// holders' completion times from the holder table and keep the ell
// smallest in registers; the N ell values go to shared memory as 64-bit
// keys (the bit patterns of non-negative doubles order like the values),
// and a most-significant-digit radix select (4-bit digits, per-lane packed
// counters summed with warp reductions) finds the order statistic without
// sorting; for theta = 0 the statistic is the largest value, a warp max
// (and no keys are stored).  All arithmetic is the same double multiply the
// definition uses, so times and psi are bit-exact.
#include <math.h>

#include <algorithm>

#include "gc_internal.cuh"

namespace gc {
namespace {

constexpr int kWarpsPerBlock = 4;
// Resident blocks per SM the kernel is compiled for and the grid is sized
// to: 12 (at most 40 registers a thread) while the 2 x ELL running minima
// fit, else 8 (64 registers).  Many warps per SM keep the fp64 products and
// the tau loads of many realizations in flight.
constexpr int blocks_per_sm(int ell) { return ell <= 3 ? 12 : 8; }

// k-th smallest (1-based, 1 <= k <= n) of n keys in shared memory, by warp.
__device__ unsigned long long warp_select(const unsigned long long* keys, int n, int k, int lane) {
  unsigned long long prefix = 0, mask = 0;
  for (int shift = 60; shift >= 0; shift -= 4) {
    unsigned long long lo = 0, hi = 0;  // 8-bit counters for digits 0..7 and 8..15
    for (int t = lane; t < n; t += 32) {
      const unsigned long long key = keys[t];
      if ((key & mask) == prefix) {
        const int dg = (int)((key >> shift) & 15u);
        if (dg < 8) lo += 1ull << (8 * dg);
        else hi += 1ull << (8 * (dg - 8));
      }
    }
    int cum = 0, digit = 15;
    for (int dg = 0; dg < 16; ++dg) {
      const unsigned c = (unsigned)(((dg < 8 ? lo : hi) >> (8 * (dg & 7))) & 255u);
      const int tot = (int)__reduce_add_sync(0xffffffffu, c);
      if (cum + tot >= k) {
        digit = dg;
        break;
      }
      cum += tot;
    }
    k -= cum;
    prefix |= (unsigned long long)digit << shift;
    mask |= 15ull << shift;
  }
  return prefix;
}

// Keep the ELL smallest keys seen so far (ascending).  Keys are the bit
// patterns of non-negative doubles, which order like the values, so the
// comparisons are integer ones (GB300's fp64 pipe is 1/64 of fp32; only the
// multiplies that define the times stay in fp64).  Branch-free with static
// indices, so the array stays in registers: position k of the result is
// b[k-1] when v goes before it, else min(v, b[k]).
template <int ELL>
__device__ __forceinline__ void insert_smallest(unsigned long long (&b)[ELL], unsigned long long v) {
#pragma unroll
  for (int k = ELL - 1; k > 0; --k) b[k] = v < b[k - 1] ? b[k - 1] : (v < b[k] ? v : b[k]);
  b[0] = v < b[0] ? v : b[0];
}
__device__ __forceinline__ unsigned long long dbits(double x) {
  return (unsigned long long)__double_as_longlong(x);
}
// isfinite on the bit pattern (integer ops; a double compare would use the fp64 pipe)
__device__ __forceinline__ bool finite_bits(double x) {
  return (dbits(x) & 0x7ff0000000000000ull) != 0x7ff0000000000000ull;
}
// A float near a finite non-negative double, from its bits (integer ops; the
// mantissa is truncated, magnitudes outside the float range are clamped).
// Only a starting point for an exact search, so its accuracy is not critical.
__device__ __forceinline__ float approx_float(double x) {
  const unsigned long long b = dbits(x);
  const int e = (int)((b >> 52) & 0x7ff) - 1023 + 127;
  if (e <= 0) return 0.f;
  if (e >= 255) return 3.0e38f;
  return __uint_as_float(((unsigned)e << 23) | (unsigned)((b >> 29) & 0x7fffffu));
}

template <int ELL>
__global__ void __launch_bounds__(32 * kWarpsPerBlock, blocks_per_sm(ELL))
    k_trigger(const int32_t* __restrict__ order, Holders h, int N, int m, int delta,
              const double* __restrict__ tau, long long nsim, int theta, double* __restrict__ T_out,
              int32_t* __restrict__ psi_out, double* __restrict__ Tfull_out) {
  extern __shared__ unsigned long long s_dyn[];
  // the integers 0..GC_MAX_REPL as doubles: the slot factors (p + 1) of the
  // completion times are read here rather than converted per product (an
  // int -> double conversion runs on the fp64 pipe, 1/64 of fp32 on GB300)
  __shared__ double s_kd[GC_MAX_REPL + 1];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // per block: delta_j of every worker; per warp: the finishing time of every
  // worker (m keys) and, for theta > 0, 2 N ELL completion keys
  int8_t* s_dj = reinterpret_cast<int8_t*>(s_dyn);
  const size_t dj_words = ((size_t)m + 7) / 8;
  unsigned long long* fin = s_dyn + dj_words + (size_t)warp * m;
  unsigned long long* keys = s_dyn + dj_words + (size_t)kWarpsPerBlock * m +
                             (size_t)warp * 2 * N * ELL;
  unsigned long long* keysF = keys + (size_t)N * ELL;
  for (int j = threadIdx.x; j < m; j += blockDim.x) {
    int c = 0;
    for (int p = 0; p < delta; ++p) c += order[(size_t)j * delta + p] >= 0;
    s_dj[j] = (int8_t)c;
  }
  for (int c = threadIdx.x; c <= GC_MAX_REPL; c += blockDim.x) s_kd[c] = (double)c;
  __syncthreads();
  const int n = N * ELL;
  const int kth = n - theta;
  for (long long r = (long long)blockIdx.x * kWarpsPerBlock + warp; r < nsim;
       r += (long long)gridDim.x * kWarpsPerBlock) {
    const double* tr = tau + r * m;
    const unsigned long long kInf = dbits(INFINITY);
    // each worker's finishing time delta_j tau_j (+inf for a failed worker)
    for (int j = lane; j < m; j += 32) {
      const double tj = tr[j];
      fin[j] = finite_bits(tj) ? dbits(s_kd[s_dj[j]] * tj) : kInf;
    }
    __syncwarp();
    // theta = 0: the order statistic is the largest of the N ell values, i.e.
    // the largest ell-th completion time -- a max, no selection needed
    unsigned long long lmax = 0, lmaxF = 0;
    for (int i = lane; i < N; i += 32) {
      unsigned long long b[ELL], bf[ELL];
#pragma unroll
      for (int k = 0; k < ELL; ++k) b[k] = bf[k] = kInf;
      const int cnt = h.cnt[i];
      for (int q = 0; q < cnt; ++q) {
        const int j = h.w[(size_t)i * GC_MAX_REPL + q];
        const int p = h.p[(size_t)i * GC_MAX_REPL + q];
        const double tj = tr[j];
        if (finite_bits(tj)) {
          insert_smallest<ELL>(b, dbits(s_kd[p + 1] * tj));
          insert_smallest<ELL>(bf, fin[j]);
        }
      }
      if (theta == 0) {
        lmax = max(lmax, b[ELL - 1]);
        lmaxF = max(lmaxF, bf[ELL - 1]);
      } else {
#pragma unroll
        for (int k = 0; k < ELL; ++k) {
          keys[(size_t)i * ELL + k] = b[k];
          keysF[(size_t)i * ELL + k] = bf[k];
        }
      }
    }
    __syncwarp();
    unsigned long long Tb = 0, TFb = 0;
    if (theta == 0) {
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        lmax = max(lmax, (unsigned long long)__shfl_xor_sync(0xffffffffu, lmax, o));
        lmaxF = max(lmaxF, (unsigned long long)__shfl_xor_sync(0xffffffffu, lmaxF, o));
      }
      Tb = lmax;
      TFb = lmaxF;
    } else if (kth >= 1) {
      Tb = warp_select(keys, n, kth, lane);
      TFb = warp_select(keysF, n, kth, lane);
    }
    const double T = __longlong_as_double((long long)Tb);
    const double TF = __longlong_as_double((long long)TFb);
    if (lane == 0) {
      if (T_out) T_out[r] = T;
      if (Tfull_out) Tfull_out[r] = TF;
    }
    if (psi_out)
      for (int j = lane; j < m; j += 32) {
        // slots finish in order: psi_j is the largest c <= delta_j with
        // c tau_j <= T (the products are monotone in c).  An fp32 estimate of
        // T / tau_j is corrected with the exact double products, so that
        // typically two of them are formed instead of one per slot.
        const double tj = tr[j];
        const int dj = s_dj[j];
        int c = 0;
        if (finite_bits(tj) && dj > 0) {
          const float q = __fdividef(approx_float(T), approx_float(tj));
          c = q >= (float)dj ? dj : (q > 0.f ? (int)q : 0);
          while (c > 0 && dbits(s_kd[c] * tj) > Tb) --c;
          while (c < dj && dbits(s_kd[c + 1] * tj) <= Tb) ++c;
        }
        psi_out[r * m + j] = c;
      }
    __syncwarp();
  }
}

template <int ELL>
int launch_one(const int32_t* order, Holders h, int N, int m, int delta, const double* tau,
               long long nsim, int theta, double* T, int32_t* psi, double* TF, cudaStream_t s) {
  const size_t keys = theta == 0 ? 0 : (size_t)kWarpsPerBlock * 2 * N * ELL;
  const size_t smem = (((size_t)m + 7) / 8 + (size_t)kWarpsPerBlock * m + keys) * 8;
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(k_trigger<ELL>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return cuda_check(e, "cudaFuncSetAttribute(k_trigger)");
  }
  const long long blocks_needed = (nsim + kWarpsPerBlock - 1) / kWarpsPerBlock;
  const int blocks =
      (int)std::min<long long>(blocks_needed, (long long)device_sm_count() * blocks_per_sm(ELL));
  k_trigger<ELL><<<blocks, 32 * kWarpsPerBlock, smem, s>>>(order, h, N, m, delta, tau, nsim, theta,
                                                           T, psi, TF);
  count_launches(1);
  return cuda_check(cudaGetLastError(), "k_trigger");
}

}  // namespace

int launch_trigger(const int32_t* order, Holders h, int N, int m, int delta, const double* tau,
                   long long nsim, int ell, int theta, double* T, int32_t* psi, double* TF,
                   cudaStream_t s) {
  switch (ell) {
    case 1: return launch_one<1>(order, h, N, m, delta, tau, nsim, theta, T, psi, TF, s);
    case 2: return launch_one<2>(order, h, N, m, delta, tau, nsim, theta, T, psi, TF, s);
    case 3: return launch_one<3>(order, h, N, m, delta, tau, nsim, theta, T, psi, TF, s);
    case 4: return launch_one<4>(order, h, N, m, delta, tau, nsim, theta, T, psi, TF, s);
    case 5: return launch_one<5>(order, h, N, m, delta, tau, nsim, theta, T, psi, TF, s);
    case 6: return launch_one<6>(order, h, N, m, delta, tau, nsim, theta, T, psi, TF, s);
    case 7: return launch_one<7>(order, h, N, m, delta, tau, nsim, theta, T, psi, TF, s);
    case 8: return launch_one<8>(order, h, N, m, delta, tau, nsim, theta, T, psi, TF, s);
    default: return fail(GC_ERR_UNSUPPORTED, "ell=%d exceeds GC_MAX_ELL", ell);
  }
}

}  // namespace gc
