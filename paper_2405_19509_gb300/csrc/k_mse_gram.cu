// The gradient MSE of a batch of patterns without forming the decoded
// gradients (Sec. II-B decode, errors of Sec. IV).
//
// Pattern b's decoded gradient differs from s = sum_i g_{D_i} by, in block k,
//   ghat_b[k] - s[k] = sum_a v_{b,k}[a] G_a,   v_{b,k}[a] = C[b*ell + k][a] - [a mod ell == k],
// where a = i*ell + k' runs over the N*ell chunk blocks G_a = g_{D_i}[k'] (length
// L, zero past d) and C is the decode matrix of the plan.  Hence
//   ||ghat_b - s||^2 = sum_k v_{b,k} H v_{b,k}^T,   H[a][a'] = <G_a, G_a'>,
// so one Gram matrix of the chunk blocks (N*ell x N*ell, formed once per call)
// replaces the batch's (npat*ell) x (N*ell) x L product: each row costs at
// most (N*ell)^2 multiply-adds, only over its non-zero entries.  When ell does
// not divide d the last output block has only L_last = d - (ell-1) L columns,
// so its rows take H_last, the same sums over the first L_last columns (the
// other rows the full H); the slices are cut at L_last so that both come
// from one pass.
//
// k_gram_partial: H over column slices, 64 x 64 tiles of the upper triangle,
//   fp32 sums within a slice; k_gram_reduce adds the slices in order in fp64.
// k_mse_gram: one warp per pattern; the row vector's non-zero entries are
//   compacted in shared memory and q = v H v^T is summed lane-parallel over
//   the second index, then across the lanes and the ell rows in a fixed order.
#include <algorithm>
#include <type_traits>

#include "gc_internal.cuh"

namespace gc {

namespace {

constexpr int kGramTile = 64;    // H tile edge
constexpr int kGramCols = 32;    // columns staged per step
constexpr int kGramMaxSplits = 128;
constexpr int kGramMaxK = 256;   // N*ell beyond which the Gram path is not taken
constexpr int kMseWarps = 32;    // warps of a k_mse_gram block (H in shared memory)
constexpr int kHSmemMaxK = 128;  // H staged in shared memory up to this N*ell

// Upper-triangle tile t -> (ta, tb), ta <= tb, row-major over the triangle.
__device__ __forceinline__ void tri_tile(int t, int nt, int& ta, int& tb) {
  int a = 0, rem = t;
  while (rem >= nt - a) {
    rem -= nt - a;
    ++a;
  }
  ta = a;
  tb = a + rem;
}

// Block (tile t, slice z): partial[t][z][64 x 64] = sum over the slice's
// columns c of G_a[c] G_b[c] for the tile's rows a and columns b.  A step
// stages 64 rows x 32 columns of each side: thread (r, q) holds the 8
// columns 8q .. 8q + 7 of row r on both sides in registers, loaded one step
// ahead of the multiply-adds (16-byte loads when rows are 16-byte aligned);
// each thread sums a 4 x 4 block of the tile.
__device__ __forceinline__ void gram_load8(const float* __restrict__ G, int N, int ell, int d,
                                           int L, int c_hi, int a, int c, bool vec, float (&v)[8]) {
  const int K = N * ell;
#pragma unroll
  for (int e = 0; e < 8; ++e) v[e] = 0.f;
  if (a >= K) return;
  const int i = a / ell, k = a - i * ell;
  const float* p = G + (size_t)i * d + (size_t)k * L;
  const long long lim = min((long long)c_hi, (long long)d - (long long)k * L);  // columns < lim exist
  if (vec && (c & 3) == 0 && c + 8 <= lim) {
    const float4 x = __ldg(reinterpret_cast<const float4*>(p + c));
    const float4 y = __ldg(reinterpret_cast<const float4*>(p + c + 4));
    v[0] = x.x; v[1] = x.y; v[2] = x.z; v[3] = x.w;
    v[4] = y.x; v[5] = y.y; v[6] = y.z; v[7] = y.w;
  } else {
#pragma unroll
    for (int e = 0; e < 8; ++e)
      if (c + e < lim) v[e] = __ldg(p + c + e);
  }
}

__global__ void __launch_bounds__(256) k_gram_partial(const float* __restrict__ G, int N, int ell,
                                                      int d, int L, int slice, int nsa, int l_last,
                                                      int vec, float* __restrict__ partial) {
  // staged column-major, sa[c][r], so that a thread reads 4 rows as one 16-byte load
  __shared__ __align__(16) float sa[kGramCols][kGramTile];
  __shared__ __align__(16) float sb[kGramCols][kGramTile];
  const int K = N * ell, nt = (K + kGramTile - 1) / kGramTile;
  int ta, tb;
  tri_tile(blockIdx.x, nt, ta, tb);
  const int z = blockIdx.y;
  // slices z < nsa cover [0, l_last); slice nsa (when l_last < L) covers [l_last, L)
  const int c_lo = z < nsa ? z * slice : l_last;
  const int c_hi = z < nsa ? min(l_last, c_lo + slice) : L;
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;  // 4 x 4 outputs: rows 4 ty.., cols 4 tx..
  const int sr = threadIdx.x >> 2, sq = threadIdx.x & 3;    // staging: row sr, columns 8 sq .. 8 sq + 7
  float acc[4][4];
#pragma unroll
  for (int u = 0; u < 4; ++u)
#pragma unroll
    for (int v = 0; v < 4; ++v) acc[u][v] = 0.f;
  float xa[8], xb[8];
  if (c_lo < c_hi) {
    gram_load8(G, N, ell, d, L, c_hi, ta * kGramTile + sr, c_lo + 8 * sq, vec != 0, xa);
    gram_load8(G, N, ell, d, L, c_hi, tb * kGramTile + sr, c_lo + 8 * sq, vec != 0, xb);
  }
  for (int c0 = c_lo; c0 < c_hi; c0 += kGramCols) {
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      sa[8 * sq + e][sr] = xa[e];
      sb[8 * sq + e][sr] = xb[e];
    }
    __syncthreads();
    if (c0 + kGramCols < c_hi) {  // the next step's columns, in flight during this one
      gram_load8(G, N, ell, d, L, c_hi, ta * kGramTile + sr, c0 + kGramCols + 8 * sq, vec != 0, xa);
      gram_load8(G, N, ell, d, L, c_hi, tb * kGramTile + sr, c0 + kGramCols + 8 * sq, vec != 0, xb);
    }
#pragma unroll 8
    for (int cc = 0; cc < kGramCols; ++cc) {
      const float4 a4 = *reinterpret_cast<const float4*>(&sa[cc][4 * ty]);
      const float4 b4 = *reinterpret_cast<const float4*>(&sb[cc][4 * tx]);
      const float av[4] = {a4.x, a4.y, a4.z, a4.w}, bv[4] = {b4.x, b4.y, b4.z, b4.w};
#pragma unroll
      for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int v = 0; v < 4; ++v) acc[u][v] = fmaf(av[u], bv[v], acc[u][v]);
    }
    __syncthreads();
  }
  float* out = partial + ((size_t)blockIdx.x * gridDim.y + z) * (kGramTile * kGramTile);
#pragma unroll
  for (int u = 0; u < 4; ++u)
    *reinterpret_cast<float4*>(out + (4 * ty + u) * kGramTile + 4 * tx) =
        make_float4(acc[u][0], acc[u][1], acc[u][2], acc[u][3]);
}

// H_last[a][b] = H_last[b][a] = sum over the slices z < nsa of the partials,
// in fp64, and H = H_last + slice nsa when there is one: block (tile t, part y)
// takes 32 of the tile's entries; thread (entry j, group g) adds the slices
// z = g, g + 8, ... (< nsa) and the eight group sums are added in order
// g = 0 .. 7.
__global__ void __launch_bounds__(256) k_gram_reduce(const float* __restrict__ partial, int K,
                                                     int nsa, int nsplit, float* __restrict__ H,
                                                     float* __restrict__ H_last) {
  __shared__ double s_part[8][32];
  const int nt = (K + kGramTile - 1) / kGramTile;
  int ta, tb;
  tri_tile(blockIdx.x, nt, ta, tb);
  const int j = threadIdx.x & 31, g = threadIdx.x >> 5;
  const int e = blockIdx.y * 32 + j;
  const float* src = partial + (size_t)blockIdx.x * nsplit * (kGramTile * kGramTile) + e;
  double sum = 0.0;
  int z = g;
  for (; z + 56 < nsa; z += 64) {  // eight slices of this group at a time
    float v[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) v[u] = src[(size_t)(z + 8 * u) * (kGramTile * kGramTile)];
#pragma unroll
    for (int u = 0; u < 8; ++u) sum += (double)v[u];
  }
  for (; z < nsa; z += 8) sum += (double)src[(size_t)z * (kGramTile * kGramTile)];
  s_part[g][j] = sum;
  __syncthreads();
  if (g != 0) return;
  double tot = 0.0;
#pragma unroll
  for (int u = 0; u < 8; ++u) tot += s_part[u][j];
  const int r = e / kGramTile, c = e % kGramTile;
  const int a = ta * kGramTile + r, b = tb * kGramTile + c;
  if (a >= K || b >= K) return;
  if (nsplit > nsa) {  // a padded last block: H_last, then the full sums
    H_last[(size_t)a * K + b] = (float)tot;
    H_last[(size_t)b * K + a] = (float)tot;
    tot += (double)src[(size_t)nsa * (kGramTile * kGramTile)];
  }
  H[(size_t)a * K + b] = (float)tot;
  H[(size_t)b * K + a] = (float)tot;
}

// One warp per pattern b: grad_mse[b] = (1/d) sum_k q_k, q_k = v H v^T for the
// row vector v = C[b*ell + k] - [a mod ell == k] (C = hi + lo of the plan).
// Lane l holds entries a = 32 u + l (u < KW) of a row; the warp's rows are
// walked in order with the loads of the row two ahead issued before the
// current row is summed, so the load latency hides behind two rows' work.
template <bool HS, int KW, int W, bool PAD>
__global__ void __launch_bounds__(W * 32) k_mse_gram(const __nv_bfloat16* __restrict__ Cs,
                                                             int Kp, int N, int ell, int npat,
                                                             const float* __restrict__ H,
                                                             const float* __restrict__ H_last,
                                                             double inv_d,
                                                             double* __restrict__ grad_mse) {
  extern __shared__ float s_dyn[];
  const int K = N * ell;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float* s_h = s_dyn;                                       // [K][K] when HS
  float* s_val = s_dyn + (HS ? K * K : 0) + warp * 2 * K;   // [K] non-zero values of this warp's row
  int* s_idx = reinterpret_cast<int*>(s_val + K);           // [K] their indices
  if (HS) {
#pragma unroll 8
    for (int t = threadIdx.x; t < K * K; t += blockDim.x) s_h[t] = __ldg(H + t);
    __syncthreads();
  }
  const float* Hm = HS ? s_h : H;
  int am[KW];  // (32 u + lane) mod ell: the block of the row's entries
#pragma unroll
  for (int u = 0; u < KW; ++u) am[u] = (32 * u + lane) % ell;
  const size_t plane = (size_t)npat * ell * Kp;
  const long long stride = (long long)gridDim.x * W;
  // row j of this warp: pattern b0 + (j / ell) * stride, block j % ell
  const long long b0 = (long long)blockIdx.x * W + warp;
  auto load_row = [&](long long b, int k, float (&v)[KW]) {
    const size_t row = ((size_t)b * ell + k) * Kp;
#pragma unroll
    for (int u = 0; u < KW; ++u) {
      const int a = 32 * u + lane;
      v[u] = 0.f;
      if (b < npat && a < K)
        v[u] = __bfloat162float(Cs[row + a]) + __bfloat162float(Cs[plane + row + a]) -
               (am[u] == k ? 1.f : 0.f);
    }
  };
  double tot = 0.0;
  // Sum row (b, k) from its entries v (lane-held).
  auto process = [&](const float (&v)[KW], long long b, int k) {
    bool any = false;
#pragma unroll
    for (int u = 0; u < KW; ++u) any |= v[u] != 0.f;
    if (!__any_sync(0xffffffffu, any)) {  // the row's blocks are all I: q = 0
      if (lane == 0 && k == ell - 1) {
        grad_mse[b] = tot * inv_d;
        tot = 0.0;
      }
      return;
    }
    // compact the row's non-zero entries (ascending a)
    int nz = 0;
#pragma unroll
    for (int u = 0; u < KW; ++u) {
      const unsigned bal = __ballot_sync(0xffffffffu, v[u] != 0.f);
      if (v[u] != 0.f) {
        const int pos = nz + __popc(bal & ((1u << lane) - 1u));
        s_val[pos] = v[u];
        s_idx[pos] = 32 * u + lane;
      }
      nz += __popc(bal);
    }
    __syncwarp();
    // q = sum_{e'} v_{e'} sum_e v_e H[a_e][a_{e'}]: lane l takes e' = l + 32 t
    // (t < KW), u_t accumulates over e ascending, then q over t ascending
    float uu[KW], v2[KW];
    int a2[KW];
#pragma unroll
    for (int t = 0; t < KW; ++t) {
      const int e2 = lane + 32 * t;
      uu[t] = 0.f;
      v2[t] = e2 < nz ? s_val[e2] : 0.f;
      a2[t] = e2 < nz ? s_idx[e2] : 0;
    }
    // the last output block of a padded d has its own Gram matrix (read
    // through the cache)
    const float* Hk = (PAD && k == ell - 1) ? H_last : Hm;
    // only the t with some lane in range take part (no predicated-off work)
    auto sweep = [&](auto tn) {
      constexpr int TN = decltype(tn)::value;
#pragma unroll 4
      for (int e = 0; e < nz; ++e) {
        const float ve = s_val[e];
        const float* hr = Hk + (size_t)s_idx[e] * K;
#pragma unroll
        for (int t = 0; t < TN; ++t) uu[t] = fmaf(ve, hr[a2[t]], uu[t]);
      }
    };
    const int tmax = (nz + 31) / 32;
    if (tmax <= 1)
      sweep(std::integral_constant<int, 1>{});
    else
      sweep(std::integral_constant<int, KW>{});
    float q = 0.f;
#pragma unroll
    for (int t = 0; t < KW; ++t) q = fmaf(v2[t], uu[t], q);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) q += __shfl_xor_sync(0xffffffffu, q, o);
    if (lane == 0) {  // fp64 work on one lane only
      tot += (double)q;
      if (k == ell - 1) {
        grad_mse[b] = tot * inv_d;
        tot = 0.0;
      }
    }
    __syncwarp();  // the lists are rewritten by the next row
  };
  // Rows in order through three register buffers used in rotation, so that a
  // row's loads go out two rows before it is summed and no buffer is copied
  // (a copy would wait for the loads).
  auto advance = [&](long long& bb, int& kk) {
    if (++kk == ell) {
      kk = 0;
      bb += stride;
    }
  };
  float A[KW], B[KW], C[KW];
  long long rb0 = b0, rb1, rb2;
  int rk0 = 0, rk1, rk2;
  load_row(rb0, rk0, A);
  rb1 = rb0;
  rk1 = rk0;
  advance(rb1, rk1);
  load_row(rb1, rk1, B);
  for (;;) {
    rb2 = rb1;
    rk2 = rk1;
    advance(rb2, rk2);
    load_row(rb2, rk2, C);
    if (rb0 >= npat) break;
    process(A, rb0, rk0);
    rb0 = rb2;
    rk0 = rk2;
    advance(rb0, rk0);
    load_row(rb0, rk0, A);
    if (rb1 >= npat) break;
    process(B, rb1, rk1);
    rb1 = rb0;
    rk1 = rk0;
    advance(rb1, rk1);
    load_row(rb1, rk1, B);
    if (rb2 >= npat) break;
    process(C, rb2, rk2);
  }
}

template <bool HS, int KW, int W, bool PAD>
cudaError_t launch_mse_gram_t(int blocks, size_t smem, const __nv_bfloat16* Cs, int Kp, int N,
                              int ell, int npat, const float* H, const float* H_last, double inv_d,
                              double* grad_mse, cudaStream_t s) {
  if (HS) {
    static bool attr = false;
    if (!attr) {
      const cudaError_t e = cudaFuncSetAttribute(
          k_mse_gram<HS, KW, W, PAD>, cudaFuncAttributeMaxDynamicSharedMemorySize,
          (int)(((size_t)kHSmemMaxK * kHSmemMaxK + W * 2 * kHSmemMaxK) * sizeof(float)));
      if (e != cudaSuccess) return e;
      attr = true;
    }
  }
  k_mse_gram<HS, KW, W, PAD><<<blocks, W * 32, smem, s>>>(Cs, Kp, N, ell, npat, H, H_last,
                                                           inv_d, grad_mse);
  return cudaSuccess;
}

int gram_splits(int L) {
  // slices of at least 256 columns, at most kGramMaxSplits of them
  const int by_min = (L + 255) / 256;
  return std::max(1, std::min(kGramMaxSplits, by_min));
}

}  // namespace

bool mse_gram_applies(int N, int ell, int npat) {
  const int K = N * ell;
  return K <= kGramMaxK && (long long)npat * ell >= 2LL * K;
}

size_t mse_gram_ws_bytes(int N, int ell, int d) {
  const int K = N * ell;
  if (K > kGramMaxK) return 0;
  const int L = (d + ell - 1) / ell;
  const int nt = (K + kGramTile - 1) / kGramTile;
  const size_t ntri = (size_t)nt * (nt + 1) / 2;
  return align_up(ntri * (gram_splits(L) + 1) * kGramTile * kGramTile * sizeof(float), 256) +
         2 * align_up((size_t)K * K * sizeof(float), 256);
}

int launch_mse_gram(const __nv_bfloat16* Cs, int Kp, const float* G, int N, int ell, int npat,
                    int d, double* grad_mse, Carve& ws, cudaStream_t s) {
  const int K = N * ell;
  const int L = (d + ell - 1) / ell;
  const int l_last = d - (ell - 1) * L;  // real columns of the last block, 0 < l_last <= L
  const int nt = (K + kGramTile - 1) / kGramTile;
  const int ntri = nt * (nt + 1) / 2;
  const int nsa = gram_splits(l_last);                  // slices of [0, l_last)
  const int nsplit = nsa + (l_last < L ? 1 : 0);        // + the last block's padding range
  const int slice = ((l_last + nsa - 1) / nsa + kGramCols - 1) / kGramCols * kGramCols;
  float* partial = ws.take<float>((size_t)ntri * nsplit * kGramTile * kGramTile);
  float* H = ws.take<float>((size_t)K * K);
  float* H_last = ws.take<float>((size_t)K * K);
  if (npat == 0) return GC_OK;
  const bool vec = d % 4 == 0 && L % 4 == 0 && reinterpret_cast<uintptr_t>(G) % 16 == 0;
  k_gram_partial<<<dim3((unsigned)ntri, (unsigned)nsplit), 256, 0, s>>>(
      G, N, ell, d, L, slice, nsa, l_last, vec ? 1 : 0, partial);
  k_gram_reduce<<<dim3((unsigned)ntri, (kGramTile * kGramTile) / 32), 256, 0, s>>>(
      partial, K, nsa, nsplit, H, H_last);
  const float* hl = l_last < L ? H_last : nullptr;
  const bool hs = K <= kHSmemMaxK;
  // H from shared memory and no padded last block: blocks of 32 warps (96 KB,
  // 64 registers a thread); otherwise blocks of 16 warps (up to 128 registers)
  const int W = hs && !hl ? kMseWarps : kMseWarps / 2;
  const size_t smem = ((hs ? (size_t)K * K : 0) + (size_t)W * 2 * K) * sizeof(float);
  const int blocks = (int)std::min<long long>(((long long)npat + W - 1) / W,
                                              2LL * device_sm_count());
  const int kw = (K + 31) / 32;  // <= kGramMaxK / 32 = 8
  cudaError_t e = cudaSuccess;
#define GC_MSEG(HSV, KWV)                                                                         \
  e = hl ? launch_mse_gram_t<HSV, KWV, kMseWarps / 2, true>(                                      \
               blocks, smem, Cs, Kp, N, ell, npat, H, hl, 1.0 / (double)d, grad_mse, s)          \
         : launch_mse_gram_t<HSV, KWV, HSV ? kMseWarps : kMseWarps / 2, false>(                  \
               blocks, smem, Cs, Kp, N, ell, npat, H, hl, 1.0 / (double)d, grad_mse, s)
  if (hs) {
    if (kw <= 1) GC_MSEG(true, 1);
    else if (kw <= 2) GC_MSEG(true, 2);
    else GC_MSEG(true, 4);
  } else {
    GC_MSEG(false, 8);  // 128 < N*ell <= 256
  }
#undef GC_MSEG
  if (e != cudaSuccess) return cuda_check(e, "cudaFuncSetAttribute(k_mse_gram)");
  count_launches(3);
  return cuda_check(cudaGetLastError(), "k_mse_gram");
}

}  // namespace gc
