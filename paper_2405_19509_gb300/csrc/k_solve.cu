// Algorithm 1 (Find-Encoding-Coeff), batched over straggler patterns.
//
// For a pattern psi and chunk D_i, S_i is the set of workers that processed
// D_i and X = R[:, S_i] (ell x Delta_i).  The block column B^(i) restricted to
// the rows S_i is the minimum-norm least-squares solution X^+ of eq. (6); it
// separates column by column (Frobenius norm), and every holder of D_i
// computes the same block (Sec. II).  The decode matrix block is
// Pi_i = R_{S_i} X^+ = X X^+, the orthogonal projector onto range(X): the
// identity when Delta_i >= ell (exact recovery, Sec. II-A), rank Delta_i
// otherwise (approximate GC, eq. 7).
//
// Numerics (fp64 throughout):
//  * Delta >= ell (X has full row rank): X^+ = X^T Lambda with
//    Lambda = (X X^T)^{-1} from a Cholesky factorisation, followed by one step
//    of iterative refinement driven by the true residual e_k - X b_k, so the
//    error is O(eps * kappa(X)) instead of O(eps * kappa^2).
//  * 0 < Delta < ell (X has full column rank): QR of X by classical
//    Gram-Schmidt with re-orthogonalisation (CGS2); X^+ = R^{-1} Q^T.
//  * Delta = 0: X^+ is empty and Pi = 0.
//
// GB300 has a low fp64 rate, and Algorithm 1's result for chunk i depends
// only on (R, S_i), i.e. on which of the chunk's holders finished.  When the
// number of holder subsets is small compared with the number of (pattern,
// chunk) problems, every subset is solved once into a table (in the caller's
// workspace) and each pattern gathers from it; the values are bit-identical
// to solving the pattern directly, since the same function runs on the same
// inputs.
#include <math.h>

#include <algorithm>

#include "gc_internal.cuh"

namespace gc {

// ---------------------------------------------------------------------------
// Holder table
// ---------------------------------------------------------------------------
Holders carve_holders(Carve& c, int N) {
  Holders h;
  h.cnt = c.take<int32_t>(N);
  h.w = c.take<int16_t>((size_t)N * GC_MAX_REPL);
  h.p = c.take<int8_t>((size_t)N * GC_MAX_REPL);
  return h;
}

// One CTA per chunk: scan order[] in (worker, slot) order and compact the
// matches, which keeps holders sorted by worker then slot.
__global__ void k_holders(const int32_t* __restrict__ order, int N, int m, int delta, Holders h,
                          uint32_t* status) {
  const int i = blockIdx.x;
  __shared__ int s_warp[32];
  __shared__ int s_base;
  if (threadIdx.x == 0) s_base = 0;
  __syncthreads();
  const int total = m * delta;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarp = blockDim.x >> 5;
  for (int t0 = 0; t0 < total; t0 += blockDim.x) {
    const int t = t0 + threadIdx.x;
    int v = -1;
    if (t < total) {
      v = order[t];
      if ((v < -1 || v >= N) && i == 0) atomicOr(status, ST_BAD_ORDER);
    }
    const bool hit = (t < total) && v == i;
    const unsigned bal = __ballot_sync(0xffffffffu, hit);
    if (lane == 0) s_warp[warp] = __popc(bal);
    __syncthreads();
    int off = s_base;
    for (int w = 0; w < warp; ++w) off += s_warp[w];
    off += __popc(bal & ((1u << lane) - 1u));
    if (hit) {
      if (off < GC_MAX_REPL) {
        h.w[(size_t)i * GC_MAX_REPL + off] = (int16_t)(t / delta);
        h.p[(size_t)i * GC_MAX_REPL + off] = (int8_t)(t % delta);
      } else {
        atomicOr(status, ST_BAD_ORDER);
      }
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      int s = 0;
      for (int w = 0; w < nwarp; ++w) s += s_warp[w];
      s_base += s;
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) h.cnt[i] = s_base < GC_MAX_REPL ? s_base : GC_MAX_REPL;
}

void launch_holders(const int32_t* order, int N, int m, int delta, Holders h, uint32_t* status,
                    cudaStream_t s) {
  k_holders<<<N, 256, 0, s>>>(order, N, m, delta, h, status);
  count_launches(1);
}

// ---------------------------------------------------------------------------
// One least-squares block: chunk i, completion mask over its holders.
// emit(h, k, v) receives X^+ row of holder h (0 for holders not in S_i).
// Returns Delta; Pi (ell x ell) and err = ||I - Pi||_F^2 by reference.
// ---------------------------------------------------------------------------
template <int ELL, typename Emit>
__device__ __forceinline__ int solve_block(const double* __restrict__ R, int m, int cnt,
                                           const int16_t* __restrict__ hw, uint32_t mask,
                                           double (&Pi)[ELL][ELL], double& err, uint32_t* status,
                                           Emit emit) {
  const int D = __popc(mask);
#pragma unroll
  for (int a = 0; a < ELL; ++a)
#pragma unroll
    for (int k = 0; k < ELL; ++k) Pi[a][k] = 0.0;

  if (D >= ELL) {
    // Gram matrix M = X X^T (lower triangle) and its Cholesky factor.
    double Lc[ELL][ELL];
#pragma unroll
    for (int a = 0; a < ELL; ++a)
#pragma unroll
      for (int c = 0; c < ELL; ++c) Lc[a][c] = 0.0;
    for (int h = 0; h < cnt; ++h) {
      if (!((mask >> h) & 1u)) continue;
      const int j = hw[h];
      double x[ELL];
#pragma unroll
      for (int a = 0; a < ELL; ++a) x[a] = __ldg(R + (size_t)a * m + j);
#pragma unroll
      for (int a = 0; a < ELL; ++a)
#pragma unroll
        for (int c = 0; c <= a; ++c) Lc[a][c] = fma(x[a], x[c], Lc[a][c]);
    }
    // The diagonal is kept as reciprocals (one rsqrt per pivot): GB300's
    // fp64 divisions and square roots are long instruction sequences.
    bool bad = false;
    double rdiag[ELL];
#pragma unroll
    for (int a = 0; a < ELL; ++a) {
      double s = Lc[a][a];
#pragma unroll
      for (int c = 0; c < a; ++c) s -= Lc[a][c] * Lc[a][c];
      const double ref = Lc[a][a];
      // pivot^2 / M_aa below 1e-14 (kappa(X) of order 1e7 or more): numerically
      // rank deficient in fp64; flagged, and clamped so the result stays finite
      if (!(s > 1e-14 * ref) || !isfinite(s)) {
        bad = true;
        s = ref > 0.0 ? 1e-14 * ref : 1e-300;
      }
      const double rp = rsqrt(s);
      rdiag[a] = rp;
#pragma unroll
      for (int r = a + 1; r < ELL; ++r) {
        double t = Lc[r][a];
#pragma unroll
        for (int c = 0; c < a; ++c) t -= Lc[r][c] * Lc[a][c];
        Lc[r][a] = t * rp;
      }
    }
    if (bad) atomicOr(status, ST_SINGULAR);
    // Cholesky solve of M Y = Bm in place (column by column).
    auto chol_solve = [&](double (&Bm)[ELL][ELL]) {
#pragma unroll
      for (int k = 0; k < ELL; ++k) {
        double yv[ELL];
#pragma unroll
        for (int a = 0; a < ELL; ++a) {
          double t = Bm[a][k];
#pragma unroll
          for (int c = 0; c < a; ++c) t -= Lc[a][c] * yv[c];
          yv[a] = t * rdiag[a];
        }
#pragma unroll
        for (int a = ELL - 1; a >= 0; --a) {
          double t = yv[a];
#pragma unroll
          for (int c = a + 1; c < ELL; ++c) t -= Lc[c][a] * Bm[c][k];
          Bm[a][k] = t * rdiag[a];
        }
      }
    };
    double Lam[ELL][ELL];
#pragma unroll
    for (int a = 0; a < ELL; ++a)
#pragma unroll
      for (int k = 0; k < ELL; ++k) Lam[a][k] = (a == k) ? 1.0 : 0.0;
    chol_solve(Lam);
    // One refinement step on the residual of X b_k = e_k, b_k = X^T Lambda e_k.
    double Res[ELL][ELL];
#pragma unroll
    for (int a = 0; a < ELL; ++a)
#pragma unroll
      for (int k = 0; k < ELL; ++k) Res[a][k] = (a == k) ? 1.0 : 0.0;
    for (int h = 0; h < cnt; ++h) {
      if (!((mask >> h) & 1u)) continue;
      const int j = hw[h];
      double x[ELL];
#pragma unroll
      for (int a = 0; a < ELL; ++a) x[a] = __ldg(R + (size_t)a * m + j);
#pragma unroll
      for (int k = 0; k < ELL; ++k) {
        double bk = 0.0;
#pragma unroll
        for (int c = 0; c < ELL; ++c) bk = fma(x[c], Lam[c][k], bk);
#pragma unroll
        for (int a = 0; a < ELL; ++a) Res[a][k] = fma(-x[a], bk, Res[a][k]);
      }
    }
    chol_solve(Res);
#pragma unroll
    for (int a = 0; a < ELL; ++a)
#pragma unroll
      for (int k = 0; k < ELL; ++k) Lam[a][k] += Res[a][k];
    // Coefficients and the projector Pi = X X^+.
    for (int h = 0; h < cnt; ++h) {
      if (!((mask >> h) & 1u)) {
#pragma unroll
        for (int k = 0; k < ELL; ++k) emit(h, k, 0.0);
        continue;
      }
      const int j = hw[h];
      double x[ELL];
#pragma unroll
      for (int a = 0; a < ELL; ++a) x[a] = __ldg(R + (size_t)a * m + j);
#pragma unroll
      for (int k = 0; k < ELL; ++k) {
        double bk = 0.0;
#pragma unroll
        for (int c = 0; c < ELL; ++c) bk = fma(x[c], Lam[c][k], bk);
        emit(h, k, bk);
#pragma unroll
        for (int a = 0; a < ELL; ++a) Pi[a][k] = fma(x[a], bk, Pi[a][k]);
      }
    }
  } else if (D > 0) {
    constexpr int MQ = ELL > 1 ? ELL - 1 : 1;
    int jq[MQ];
    {
      int q = 0;
      for (int h = 0; h < cnt; ++h) {
        if (!((mask >> h) & 1u)) continue;
#pragma unroll
        for (int qq = 0; qq < MQ; ++qq)
          if (qq == q) jq[qq] = hw[h];
        ++q;
      }
    }
    double Xc[MQ][ELL], Q[MQ][ELL], Rr[MQ][MQ], Xp[MQ][ELL], rr[MQ];
#pragma unroll
    for (int qq = 0; qq < MQ; ++qq) {
#pragma unroll
      for (int r = 0; r < MQ; ++r) Rr[r][qq] = 0.0;
#pragma unroll
      for (int a = 0; a < ELL; ++a) {
        Xc[qq][a] = (qq < D) ? __ldg(R + (size_t)a * m + jq[qq]) : 0.0;
        Q[qq][a] = 0.0;
        Xp[qq][a] = 0.0;
      }
    }
    bool bad = false;
#pragma unroll
    for (int qq = 0; qq < MQ; ++qq) {
      if (qq < D) {
        double v[ELL];
        double n0 = 0.0;
#pragma unroll
        for (int a = 0; a < ELL; ++a) {
          v[a] = Xc[qq][a];
          n0 = fma(v[a], v[a], n0);
        }
#pragma unroll
        for (int pass = 0; pass < 2; ++pass) {
#pragma unroll
          for (int r = 0; r < MQ; ++r) {
            if (r < qq) {
              double dot = 0.0;
#pragma unroll
              for (int a = 0; a < ELL; ++a) dot = fma(Q[r][a], v[a], dot);
#pragma unroll
              for (int a = 0; a < ELL; ++a) v[a] = fma(-dot, Q[r][a], v[a]);
              Rr[r][qq] += dot;
            }
          }
        }
        double nn = 0.0;
#pragma unroll
        for (int a = 0; a < ELL; ++a) nn = fma(v[a], v[a], nn);
        if (!(nn > 1e-14 * n0) || !isfinite(nn)) {  // same criterion as the Cholesky pivot
          bad = true;
          nn = n0 > 0.0 ? 1e-14 * n0 : 1e-300;
        }
        const double rn = rsqrt(nn);
        Rr[qq][qq] = nn * rn;
        rr[qq] = rn;
#pragma unroll
        for (int a = 0; a < ELL; ++a) Q[qq][a] = v[a] * rn;
      }
    }
    if (bad) atomicOr(status, ST_SINGULAR);
    // X^+ = Rr^{-1} Q^T by back substitution.
#pragma unroll
    for (int qq = MQ - 1; qq >= 0; --qq) {
      if (qq < D) {
#pragma unroll
        for (int k = 0; k < ELL; ++k) {
          double t = Q[qq][k];
#pragma unroll
          for (int r = qq + 1; r < MQ; ++r)
            if (r < D) t -= Rr[qq][r] * Xp[r][k];
          Xp[qq][k] = t * rr[qq];
        }
      }
    }
    // Pi = X X^+
#pragma unroll
    for (int qq = 0; qq < MQ; ++qq)
      if (qq < D) {
#pragma unroll
        for (int a = 0; a < ELL; ++a)
#pragma unroll
          for (int k = 0; k < ELL; ++k) Pi[a][k] = fma(Xc[qq][a], Xp[qq][k], Pi[a][k]);
      }
    int q = 0;
    for (int h = 0; h < cnt; ++h) {
      const bool in = (mask >> h) & 1u;
#pragma unroll
      for (int k = 0; k < ELL; ++k) {
        double v = 0.0;
        if (in) {
#pragma unroll
          for (int qq = 0; qq < MQ; ++qq)
            if (qq == q) v = Xp[qq][k];
        }
        emit(h, k, v);
      }
      if (in) ++q;
    }
  } else {
    for (int h = 0; h < cnt; ++h)
#pragma unroll
      for (int k = 0; k < ELL; ++k) emit(h, k, 0.0);
  }
  double e = 0.0;
#pragma unroll
  for (int a = 0; a < ELL; ++a)
#pragma unroll
    for (int k = 0; k < ELL; ++k) {
      const double t = ((a == k) ? 1.0 : 0.0) - Pi[a][k];
      e = fma(t, t, e);
    }
  err = e;
  return D;
}

// ---------------------------------------------------------------------------
// Table of every holder subset: entry (i, mask) holds X^+ (cnt x ell), Pi and err.
// ---------------------------------------------------------------------------
struct Table {
  int bits;     // masks per chunk = 1 << bits
  double* xp;   // [N][1<<bits][bits][ell]
  float* pi;    // [N][1<<bits][ell][ell] (fp32: the decode matrix is emitted in fp32)
  double* err;  // [N][1<<bits]
};

template <int ELL>
__global__ void __launch_bounds__(32) k_table(const double* __restrict__ R, Holders hd, int N,
                                              int m, Table tb, int need_xp, uint32_t* status) {
  const long long e = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  const long long nent = (long long)N << tb.bits;
  if (e >= nent) return;
  const int i = (int)(e >> tb.bits);
  const uint32_t mask = (uint32_t)(e & ((1LL << tb.bits) - 1));
  const int cnt = hd.cnt[i];
  if (cnt > tb.bits) return;  // such chunks are solved directly per pattern
  if (mask >> cnt) return;    // masks beyond this chunk's holders never occur
  if (!need_xp && __popc(mask) >= ELL) {
    // full row rank: R_S X^+ = I exactly (Sec. II-A); nothing to solve when the
    // caller does not want the coefficients themselves
    float* pi = tb.pi + (size_t)e * ELL * ELL;
#pragma unroll
    for (int a = 0; a < ELL; ++a)
#pragma unroll
      for (int k = 0; k < ELL; ++k) pi[a * ELL + k] = a == k ? 1.f : 0.f;
    tb.err[e] = 0.0;
    return;
  }
  double Pi[ELL][ELL];
  double err;
  double* xp = tb.xp + (size_t)e * tb.bits * ELL;
  solve_block<ELL>(R, m, cnt, hd.w + (size_t)i * GC_MAX_REPL, mask, Pi, err, status,
                   [&](int h, int k, double v) { xp[h * ELL + k] = v; });
  float* pi = tb.pi + (size_t)e * ELL * ELL;
#pragma unroll
  for (int a = 0; a < ELL; ++a)
#pragma unroll
    for (int k = 0; k < ELL; ++k) pi[a * ELL + k] = (float)Pi[a][k];
  tb.err[e] = err;
}

// ---------------------------------------------------------------------------
// Per (pattern, chunk): completion mask, Delta, then table lookup or direct
// solve; per-pattern error sums reduced in a fixed order.
// ---------------------------------------------------------------------------
// Decode matrix block (pattern b, chunk i) as bf16 hi/lo planes, the layout
// the tensor-core combine reads: plane h, row b*ell + a, column i*ell + k.
template <int ELL>
__device__ __forceinline__ void write_planes(__nv_bfloat16* Cs, int Kp, int npat, int b, int i,
                                             const float (&Pf)[ELL][ELL]) {
  const size_t plane = (size_t)npat * ELL * Kp;
  if constexpr (ELL % 2 == 0) {
    // pairs of adjacent columns as one 4-byte store per plane (Kp and i*ELL
    // even; plan buffers are 256-byte aligned)
#pragma unroll
    for (int a = 0; a < ELL; ++a)
#pragma unroll
      for (int k = 0; k < ELL; k += 2) {
        const float v0 = Pf[a][k], v1 = Pf[a][k + 1 < ELL ? k + 1 : k];
        const __nv_bfloat16 h0 = __float2bfloat16_rn(v0), h1 = __float2bfloat16_rn(v1);
        const __nv_bfloat16 l0 = __float2bfloat16_rn(v0 - __bfloat162float(h0));
        const __nv_bfloat16 l1 = __float2bfloat16_rn(v1 - __bfloat162float(h1));
        const size_t idx = ((size_t)b * ELL + a) * Kp + (size_t)i * ELL + k;
        *reinterpret_cast<__nv_bfloat162*>(Cs + idx) = __halves2bfloat162(h0, h1);
        *reinterpret_cast<__nv_bfloat162*>(Cs + plane + idx) = __halves2bfloat162(l0, l1);
      }
  } else {
#pragma unroll
    for (int a = 0; a < ELL; ++a)
#pragma unroll
      for (int k = 0; k < ELL; ++k) {
        const float v = Pf[a][k];
        const __nv_bfloat16 hi = __float2bfloat16_rn(v);
        const __nv_bfloat16 lo = __float2bfloat16_rn(v - __bfloat162float(hi));
        const size_t idx = ((size_t)b * ELL + a) * Kp + (size_t)i * ELL + k;
        Cs[idx] = hi;
        Cs[plane + idx] = lo;
      }
  }
}
// Zero the padding columns [N*ell, Kp) of pattern b's rows (both planes);
// thread t of the `run` threads owning the pattern takes entries t, t+run, ...
template <int ELL>
__device__ __forceinline__ void zero_pad(__nv_bfloat16* Cs, int Kp, int N, int npat, int b, int t,
                                         int run) {
  const int K = N * ELL, pad = Kp - K;
  if (pad <= 0) return;
  const size_t plane = (size_t)npat * ELL * Kp;
  const __nv_bfloat16 z = __float2bfloat16_rn(0.f);
  for (int e = t; e < ELL * pad; e += run) {
    const size_t idx = ((size_t)b * ELL + e / pad) * Kp + K + e % pad;
    Cs[idx] = z;
    Cs[plane + idx] = z;
  }
}

// 128-thread blocks (64 registers each) so that the solve fits beside the
// chunk-gradient kernel's register file when both run concurrently.
constexpr int kPatThreads = 128;

template <int ELL, bool TABLE>
__global__ void __launch_bounds__(kPatThreads) k_patterns(const double* __restrict__ R,
                                                 const int32_t* __restrict__ psi, Holders hd,
                                                 int N, int m, int delta, int npat, int ppb,
                                                 Table tb, SolveOut out, uint32_t* status) {
  __shared__ double s_err[kPatThreads];
  __shared__ int s_def[kPatThreads];
  const int tid = threadIdx.x;
  int b, i, istep;
  bool active;
  if (ppb > 0) {  // N <= kPatThreads: ppb patterns per block, one chunk per thread
    const int lp = tid / N;
    b = blockIdx.x * ppb + lp;
    i = tid - lp * N;
    istep = N;  // single iteration
    active = (lp < ppb) && (b < npat);
  } else {  // one pattern per block, threads stride over chunks
    b = blockIdx.x;
    i = tid;
    istep = kPatThreads;
    active = b < npat;
  }
  double my_err = 0.0;
  int my_def = 0;
  if (active) {
    const int32_t* ps = psi + (size_t)b * m;
    for (; i < N; i += istep) {
      const int cnt = hd.cnt[i];
      const int16_t* hw = hd.w + (size_t)i * GC_MAX_REPL;
      const int8_t* hp = hd.p + (size_t)i * GC_MAX_REPL;
      // holders eight at a time with one 16-byte (workers) and one 8-byte
      // (slots) load: lanes take consecutive chunks whose rows lie 64 and 32
      // bytes apart, so per-entry loads cost a cache wavefront each
      uint32_t mask = 0;
      for (int h0 = 0; h0 < cnt; h0 += 8) {
        const uint4 w8 = *reinterpret_cast<const uint4*>(hw + h0);
        const uint2 p8 = *reinterpret_cast<const uint2*>(hp + h0);
        const uint32_t ww[4] = {w8.x, w8.y, w8.z, w8.w};
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          if (h0 + q < cnt) {
            const int wq = (int)(int16_t)(ww[q >> 1] >> (16 * (q & 1)));
            const int pq = (int)(int8_t)(((q < 4 ? p8.x : p8.y) >> (8 * (q & 3))) & 0xffu);
            int v = ps[wq];
            if (v < 0 || v > delta) {
              atomicOr(status, ST_BAD_PSI);
              v = 0;
            }
            if (pq < v) mask |= 1u << (h0 + q);
          }
        }
      }
      float Pf[ELL][ELL];
      double err;
      int D;
      double* E = out.E;
      auto emit = [&](int h, int k, double v) {
        if (E) E[(((size_t)b * m + hw[h]) * delta + hp[h]) * ELL + k] = v;
      };
      if (!E && __popc(mask) >= ELL) {
        // full row rank: the decode block is I exactly (Sec. II-A); no table
        // read (the table holds the same I and 0 for these masks)
        D = __popc(mask);
#pragma unroll
        for (int a = 0; a < ELL; ++a)
#pragma unroll
          for (int k = 0; k < ELL; ++k) Pf[a][k] = a == k ? 1.f : 0.f;
        err = 0.0;
      } else if (TABLE && cnt <= tb.bits) {
        const size_t e = ((size_t)i << tb.bits) | mask;
        const float* pi = tb.pi + e * ELL * ELL;
        if (ELL == 2) {  // one 16-byte load for the 2 x 2 block
          const float4 q = *reinterpret_cast<const float4*>(pi);
          Pf[0][0] = q.x;
          Pf[0][ELL - 1] = q.y;
          Pf[ELL - 1][0] = q.z;
          Pf[ELL - 1][ELL - 1] = q.w;
        } else {
#pragma unroll
          for (int a = 0; a < ELL; ++a)
#pragma unroll
            for (int k = 0; k < ELL; ++k) Pf[a][k] = pi[a * ELL + k];
        }
        err = tb.err[e];
        D = __popc(mask);
        if (E) {
          const double* xp = tb.xp + e * tb.bits * ELL;
          for (int h = 0; h < cnt; ++h)
#pragma unroll
            for (int k = 0; k < ELL; ++k) emit(h, k, xp[h * ELL + k]);
        }
      } else {
        double Pi[ELL][ELL];
        D = solve_block<ELL>(R, m, cnt, hw, mask, Pi, err, status, emit);
#pragma unroll
        for (int a = 0; a < ELL; ++a)
#pragma unroll
          for (int k = 0; k < ELL; ++k) Pf[a][k] = (float)Pi[a][k];
      }
      if (out.C) {
        float* Cb = out.C + (size_t)b * ELL * N * ELL + (size_t)i * ELL;
#pragma unroll
        for (int a = 0; a < ELL; ++a)
#pragma unroll
          for (int k = 0; k < ELL; ++k) Cb[(size_t)a * N * ELL + k] = Pf[a][k];
      }
      if (out.Cs) write_planes<ELL>(out.Cs, out.Kp, npat, b, i, Pf);
      if (out.delta_out) out.delta_out[(size_t)b * N + i] = (uint8_t)D;
      if (out.support) {
        uint8_t* row = out.support + ((size_t)b * N + i) * m;
        for (int j = 0; j < m; ++j) row[j] = 0;
        for (int h = 0; h < cnt; ++h)
          if ((mask >> h) & 1u) row[hw[h]] = 1;
      }
      my_err += err;
      my_def += D < ELL ? ELL - D : 0;
    }
    if (out.Cs) {
      const int t0 = ppb > 0 ? tid - (tid / N) * N : tid;
      zero_pad<ELL>(out.Cs, out.Kp, N, npat, b, t0, ppb > 0 ? N : kPatThreads);
    }
  }
  s_err[tid] = my_err;
  s_def[tid] = my_def;
  __syncthreads();
  if (!(out.coef_err || out.est)) return;
  // per pattern: lane l adds entries l, l + 32, ... of the pattern's run of
  // threads, then a fixed xor tree (deterministic); warp w takes patterns
  // w, w + 8, ...
  const int lane = tid & 31, warp = tid >> 5;
  const int npb = ppb > 0 ? ppb : 1;       // patterns in this block
  const int run = ppb > 0 ? N : kPatThreads;  // threads holding one pattern's sums
  for (int q = warp; q < npb; q += kPatThreads / 32) {
    const int bq = ppb > 0 ? blockIdx.x * ppb + q : blockIdx.x;
    if (bq >= npat) break;
    double se = 0.0;
    int sd = 0;
    for (int t = lane; t < run; t += 32) {
      se += s_err[q * run + t];
      sd += s_def[q * run + t];
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      se += __shfl_xor_sync(0xffffffffu, se, o);
      sd += __shfl_xor_sync(0xffffffffu, sd, o);
    }
    if (lane == 0) {
      if (out.coef_err) out.coef_err[bq] = se;
      if (out.est) out.est[bq] = (double)sd;
    }
  }
}

// Table width: masks over the first `bits` holders, bits = delta (the holder
// count of every chunk under N == m uniform loads).  Chunks with more holders
// than `bits` (possible with explicit orders) are solved directly.  The table
// is used when it has no more entries than there are (pattern, chunk)
// problems and at most 2^14 masks per chunk.
int solve_table_bits(int N, int m, int delta, int npat) {
  (void)m;
  const int bits = delta;
  if (bits > 14) return -1;
  if (((long long)N << bits) > (long long)npat * N) return -1;
  return bits;
}

size_t solve_table_bytes(int N, int ell, int bits) {
  if (bits < 0) return 0;
  const size_t ent = (size_t)N << bits;
  return align_up(ent * bits * ell * sizeof(double), 256) +
         align_up(ent * ell * ell * sizeof(float), 256) + align_up(ent * sizeof(double), 256);
}

// Lean variant without coefficient output for N <= 32 * CPL: one warp per
// pattern, lane l takes chunks l, l + 32, ... (at most CPL of them), and
// the warps stride over the patterns.  A lane's first eight holders of each
// of its chunks (worker and slot) are read once, before the pattern loop, and
// stay in registers; there is no shared memory and no block barrier, so the
// kernel also runs well beside other kernels.  Per pattern the completion
// masks of the lane's chunks are formed first (every psi load in flight),
// then the blocks are produced one chunk at a time.  Each lane adds its
// chunks' errors in chunk order starting from 0 and the lanes are summed by
// a fixed xor tree: the same sums, in the same order, as k_patterns.
template <int ELL, bool TABLE, int CPL>
__global__ void __launch_bounds__(128) k_patterns_warp(const double* __restrict__ R,
                                                       const int32_t* __restrict__ psi,
                                                       Holders hd, int N, int m, int delta,
                                                       int npat, Table tb, SolveOut out,
                                                       uint32_t* status) {
  const int lane = threadIdx.x & 31;
  const int gw = (int)((blockIdx.x * blockDim.x + threadIdx.x) >> 5);
  const int nw = (int)((gridDim.x * blockDim.x) >> 5);
  int cnt[CPL];
  uint4 hw8[CPL];
  uint2 hp8[CPL];
#pragma unroll
  for (int c = 0; c < CPL; ++c) {
    const int i = lane + 32 * c;
    cnt[c] = 0;
    hw8[c] = make_uint4(0u, 0u, 0u, 0u);
    hp8[c] = make_uint2(0u, 0u);
    if (i < N) {
      cnt[c] = hd.cnt[i];
      hw8[c] = *reinterpret_cast<const uint4*>(hd.w + (size_t)i * GC_MAX_REPL);
      hp8[c] = *reinterpret_cast<const uint2*>(hd.p + (size_t)i * GC_MAX_REPL);
    }
  }
  const uint32_t udelta = (uint32_t)delta;
  for (int b = gw; b < npat; b += nw) {
    const int32_t* ps = psi + (size_t)b * m;
    // completion masks of the lane's chunks; psi outside [0, delta] counts as 0
    uint32_t mask[CPL];
    bool bad = false;
#pragma unroll
    for (int c = 0; c < CPL; ++c) {
      uint32_t mk = 0;
      const uint32_t ww[4] = {hw8[c].x, hw8[c].y, hw8[c].z, hw8[c].w};
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        if (q < cnt[c]) {
          const int wq = (int)(int16_t)(ww[q >> 1] >> (16 * (q & 1)));
          const int pq = (int)(int8_t)(((q < 4 ? hp8[c].x : hp8[c].y) >> (8 * (q & 3))) & 0xffu);
          uint32_t v = (uint32_t)__ldg(ps + wq);
          if (v > udelta) {
            bad = true;
            v = 0;
          }
          if (pq < (int)v) mk |= 1u << q;
        }
      }
      // holders past the eighth (chunks with more than eight copies), eight a load
      for (int h0 = 8; h0 < cnt[c]; h0 += 8) {
        const size_t row = (size_t)(lane + 32 * c) * GC_MAX_REPL + h0;
        const uint4 w8 = *reinterpret_cast<const uint4*>(hd.w + row);
        const uint2 p8 = *reinterpret_cast<const uint2*>(hd.p + row);
        const uint32_t wx[4] = {w8.x, w8.y, w8.z, w8.w};
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          if (h0 + q < cnt[c]) {
            const int wq = (int)(int16_t)(wx[q >> 1] >> (16 * (q & 1)));
            const int pq = (int)(int8_t)(((q < 4 ? p8.x : p8.y) >> (8 * (q & 3))) & 0xffu);
            uint32_t v = (uint32_t)__ldg(ps + wq);
            if (v > udelta) {
              bad = true;
              v = 0;
            }
            if (pq < (int)v) mk |= 1u << (h0 + q);
          }
        }
      }
      mask[c] = mk;
    }
    if (__any_sync(0xffffffffu, bad) && lane == 0) atomicOr(status, ST_BAD_PSI);
    double err = 0.0;
    int def = 0;
#pragma unroll 1
    for (int c = 0; c < CPL; ++c) {
      const int i = lane + 32 * c;
      if (i >= N) break;
      // this chunk's mask and holder count, selected without indexing the arrays
      uint32_t mk = mask[0];
      int cn = cnt[0];
#pragma unroll
      for (int q = 1; q < CPL; ++q)
        if (c == q) {
          mk = mask[q];
          cn = cnt[q];
        }
      const int D = __popc(mk);
      float Pf[ELL][ELL];
      double e_i = 0.0;
      if (D >= ELL) {  // full row rank: the decode block is I exactly (Sec. II-A)
#pragma unroll
        for (int a = 0; a < ELL; ++a)
#pragma unroll
          for (int k = 0; k < ELL; ++k) Pf[a][k] = a == k ? 1.f : 0.f;
      } else if (TABLE && cn <= tb.bits) {
        const size_t e = ((size_t)i << tb.bits) | mk;
        const float* pi = tb.pi + e * ELL * ELL;
        if (ELL == 2) {  // one 16-byte load for the 2 x 2 block
          const float4 q = *reinterpret_cast<const float4*>(pi);
          Pf[0][0] = q.x;
          Pf[0][ELL - 1] = q.y;
          Pf[ELL - 1][0] = q.z;
          Pf[ELL - 1][ELL - 1] = q.w;
        } else {
#pragma unroll
          for (int a = 0; a < ELL; ++a)
#pragma unroll
            for (int k = 0; k < ELL; ++k) Pf[a][k] = pi[a * ELL + k];
        }
        e_i = tb.err[e];
      } else {
        double Pi[ELL][ELL];
        solve_block<ELL>(R, m, cn, hd.w + (size_t)i * GC_MAX_REPL, mk, Pi, e_i, status,
                         [](int, int, double) {});
#pragma unroll
        for (int a = 0; a < ELL; ++a)
#pragma unroll
          for (int k = 0; k < ELL; ++k) Pf[a][k] = (float)Pi[a][k];
      }
      if (out.C) {
        float* Cb = out.C + (size_t)b * ELL * N * ELL + (size_t)i * ELL;
#pragma unroll
        for (int a = 0; a < ELL; ++a)
#pragma unroll
          for (int k = 0; k < ELL; ++k) Cb[(size_t)a * N * ELL + k] = Pf[a][k];
      }
      if (out.Cs) write_planes<ELL>(out.Cs, out.Kp, npat, b, i, Pf);
      if (out.delta_out) out.delta_out[(size_t)b * N + i] = (uint8_t)D;
      if (out.support) {
        const int16_t* hw = hd.w + (size_t)i * GC_MAX_REPL;
        uint8_t* row = out.support + ((size_t)b * N + i) * m;
        for (int j = 0; j < m; ++j) row[j] = 0;
        for (int h = 0; h < cn; ++h)
          if ((mk >> h) & 1u) row[hw[h]] = 1;
      }
      // GB300's fp64 pipe retires 2 operations a clock per SM, so the
      // additions of +0 (every block with Delta >= ell) are skipped: adding
      // +0 to a sum that starts at +0 leaves its bits unchanged
      if (__double_as_longlong(e_i) != 0) err += e_i;
      def += D < ELL ? ELL - D : 0;
    }
    if (out.Cs) zero_pad<ELL>(out.Cs, out.Kp, N, npat, b, lane, 32);
    // fixed xor tree over the 32 lanes (deterministic); when every lane's
    // sum is +0 (an exactly decodable pattern) so is the total
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) def += __shfl_xor_sync(0xffffffffu, def, o);
    if (__any_sync(0xffffffffu, __double_as_longlong(err) != 0)) {
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) err += __shfl_xor_sync(0xffffffffu, err, o);
    }
    if (lane == 0) {
      if (out.coef_err) out.coef_err[b] = err;
      if (out.est) out.est[b] = (double)def;
    }
  }
}

template <int ELL>
static void run_solve(const double* R, const int32_t* psi, Holders h, int N, int m, int delta,
                      int npat, SolveOut out, Table tb, bool use_table, bool build_table,
                      uint32_t* status, cudaStream_t s) {
  if (use_table && build_table) {
    // one warp per block: the fp64 pipe is narrow, so spread the solves over SMs
    const long long nent = (long long)N << tb.bits;
    const int blocks = (int)((nent + 31) / 32);
    k_table<ELL><<<blocks, 32, 0, s>>>(R, h, N, m, tb, out.E != nullptr, status);
    count_launches(1);
  }
  if (npat == 0) return;
  // chunks a lane of the lean kernel takes: up to 4 for ell <= 4 (larger ell
  // keep one, their solves fill the register file), else k_patterns below
  const int cpl = N <= 32 ? 1 : (ELL <= 4 && N <= 64 ? 2 : (ELL <= 4 && N <= 128 ? 4 : 0));
  if (!out.E && cpl > 0) {
    // as many 128-thread blocks as are resident at once (all warps stride
    // over the patterns, so a second partial wave would only add a tail)
    auto go = [&](auto kern) {
      int per_sm = 0;
      if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, 128, 0) != cudaSuccess ||
          per_sm < 1) {
        cudaGetLastError();
        per_sm = 1;
      }
      const int warps = 4;  // per 128-thread block
      const int blocks =
          std::max(1, std::min((npat + warps - 1) / warps, per_sm * device_sm_count()));
      kern<<<blocks, 128, 0, s>>>(R, psi, h, N, m, delta, npat, tb, out, status);
      count_launches(1);
    };
    if (cpl == 1) {
      use_table ? go(k_patterns_warp<ELL, true, 1>) : go(k_patterns_warp<ELL, false, 1>);
    } else if constexpr (ELL <= 4) {
      if (cpl == 2)
        use_table ? go(k_patterns_warp<ELL, true, 2>) : go(k_patterns_warp<ELL, false, 2>);
      else
        use_table ? go(k_patterns_warp<ELL, true, 4>) : go(k_patterns_warp<ELL, false, 4>);
    }
    return;
  }
  int ppb = N <= kPatThreads ? kPatThreads / N : 0;
  const int grid = ppb > 0 ? (npat + ppb - 1) / ppb : npat;
  count_launches(1);
  if (use_table)
    k_patterns<ELL, true><<<grid, kPatThreads, 0, s>>>(R, psi, h, N, m, delta, npat, ppb, tb, out,
                                                      status);
  else
    k_patterns<ELL, false><<<grid, kPatThreads, 0, s>>>(R, psi, h, N, m, delta, npat, ppb, tb, out,
                                                       status);
}

// The table region is carved by the caller right after the holders.  With
// build_table = false the table already holds every entry (gc_decode_prepare)
// and npat may be 0 with build_table = true to build it alone.
int launch_solve_impl(const double* R, int ell, const int32_t* psi, Holders h, int N, int m,
                      int delta, int npat, SolveOut out, void* table_mem, int bits,
                      uint32_t* status, cudaStream_t s, bool build_table) {
  Table tb{bits < 0 ? 0 : bits, nullptr, nullptr, nullptr};
  const bool use_table = bits >= 0 && table_mem != nullptr;
  if (use_table) {
    const size_t ent = (size_t)N << bits;
    char* p = static_cast<char*>(table_mem);
    tb.xp = reinterpret_cast<double*>(p);
    p += align_up(ent * bits * ell * sizeof(double), 256);
    tb.pi = reinterpret_cast<float*>(p);
    p += align_up(ent * ell * ell * sizeof(float), 256);
    tb.err = reinterpret_cast<double*>(p);
  }
  if (out.E) {
    cudaError_t e = cudaMemsetAsync(out.E, 0, (size_t)npat * m * delta * ell * sizeof(double), s);
    if (e != cudaSuccess) return cuda_check(e, "cudaMemsetAsync(E)");
  }
  switch (ell) {
    case 1: run_solve<1>(R, psi, h, N, m, delta, npat, out, tb, use_table, build_table, status, s); break;
    case 2: run_solve<2>(R, psi, h, N, m, delta, npat, out, tb, use_table, build_table, status, s); break;
    case 3: run_solve<3>(R, psi, h, N, m, delta, npat, out, tb, use_table, build_table, status, s); break;
    case 4: run_solve<4>(R, psi, h, N, m, delta, npat, out, tb, use_table, build_table, status, s); break;
    case 5: run_solve<5>(R, psi, h, N, m, delta, npat, out, tb, use_table, build_table, status, s); break;
    case 6: run_solve<6>(R, psi, h, N, m, delta, npat, out, tb, use_table, build_table, status, s); break;
    case 7: run_solve<7>(R, psi, h, N, m, delta, npat, out, tb, use_table, build_table, status, s); break;
    case 8: run_solve<8>(R, psi, h, N, m, delta, npat, out, tb, use_table, build_table, status, s); break;
    default: return fail(GC_ERR_UNSUPPORTED, "ell=%d exceeds GC_MAX_ELL", ell);
  }
  return cuda_check(cudaGetLastError(), "solve kernels");
}

}  // namespace gc
