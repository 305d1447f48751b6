// Batched decode in residual form.
//
// The decode block of chunk i in pattern b is Pi_{b,i} = R_{S_i} X^+, which is
// exactly I_ell whenever Delta_i >= ell (Sec. II-A: X = R[:, S_i] then has full
// row rank).  Writing D_{b,i} = Pi_{b,i} - I_ell, the decoded gradient is
//
//   ghat_b[k*L + c] = s[k*L + c] + sum_{i : D_{b,i} != 0} sum_k' D_{b,i}[k][k'] g_{D_i}[k'*L + c],
//   s = sum_i g_{D_i}  (the full gradient; Sec. I),
//
// the same linear map as the combine GEMM (Ghat = C . G, C = [Pi_{b,1} ... Pi_{b,N}]),
// evaluated with the identity blocks summed once per batch.  Where few
// blocks of a pattern differ from I_ell the work is the write of ghat_b, so
// the rows of such patterns are produced here at HBM speed; row tiles whose
// patterns have many non-identity blocks stay with the tensor-core GEMM
// (k_combine_tc.cu).  The choice is made per 128-row tile on the device,
// from the decode plan itself:
//
//   k_plan_scan     one CTA per 128-row tile of the plan: per pattern the
//                   ordered list of non-identity blocks (chunk, D) and its
//                   length; per tile the ordered list of its rows that need
//                   corrections (each gets a slot for its squared-error
//                   partials) and the tile's path; the last CTA lists the
//                   GEMM's tiles in order (the GEMM and its operand split
//                   walk only those).
//   k_gsum          s = sum_i g_{D_i} over all of d (one pass over G).
//   k_decode_resid  one CTA per (residual tile, 1024-column range of each
//                   block): every row of the tile gets one contiguous 4 KB
//                   store -- s for exact patterns, s + corrections for the
//                   listed rows, whose chunk gradients come through L2 (the
//                   tiles of one column range run side by side, so each
//                   range of g_{D_i} is read from HBM about once); the
//                   squared error ||ghat_b - s||^2 = ||corrections||^2 is
//                   left as one partial per (corrected row, range, warp).
//                   CTAs of GEMM tiles return at once.
#include <algorithm>

#include "gc_internal.cuh"

namespace gc {

int resid_ksp(int ell) { return ell <= 2 ? 32 : (ell <= 4 ? 16 : 8); }

size_t resid_ws_bytes(int N, int ell, int npat, int d) {
  const int L = (d + ell - 1) / ell;
  const long long M = (long long)npat * ell;
  const long long nmt = (M + 127) / 128;
  const int ksp = std::min(resid_ksp(ell), N);
  const long long parts = (long long)((L + kResidW - 1) / kResidW) * (kResidThreads / 32);
  return align_up((size_t)npat * sizeof(int32_t), 256) +
         align_up((size_t)npat * ksp * sizeof(int32_t), 256) +
         align_up((size_t)npat * ksp * ell * ell * sizeof(float), 256) +
         align_up((size_t)nmt * sizeof(int32_t), 256) + align_up((size_t)nmt * sizeof(int32_t), 256) +
         align_up(sizeof(int32_t), 256) + align_up((size_t)M * sizeof(int32_t), 256) +
         align_up((size_t)nmt * kResidRcap * sizeof(int32_t), 256) +
         align_up((size_t)nmt * sizeof(int32_t), 256) +
         align_up((size_t)nmt * kResidRcap * parts * sizeof(float), 256);
}

ResidLists carve_resid(Carve& c, int N, int ell, int npat, int d, bool want_mse) {
  const int L = (d + ell - 1) / ell;
  const long long M = (long long)npat * ell;
  const long long nmt = (M + 127) / 128;
  ResidLists r{};
  r.ksp = std::min(resid_ksp(ell), N);
  r.parts = ((L + kResidW - 1) / kResidW) * (kResidThreads / 32);
  r.nnz = c.take<int32_t>(npat);
  r.idx = c.take<int32_t>((size_t)npat * r.ksp);
  r.D = c.take<float>((size_t)npat * r.ksp * ell * ell);
  r.tflag = c.take<int32_t>(nmt);
  r.dlist = c.take<int32_t>(nmt);
  r.ndense = c.take<int32_t>(1);
  r.rslot = c.take<int32_t>(M);
  r.rowlist = c.take<int32_t>((size_t)nmt * kResidRcap);
  r.tcount = c.take<int32_t>(nmt);
  float* msp = c.take<float>((size_t)nmt * kResidRcap * r.parts);
  r.msp = want_mse ? msp : nullptr;
  return r;
}

// ---------------------------------------------------------------------------
// Plan scan: non-identity blocks per pattern, corrected rows and path per tile.
// ---------------------------------------------------------------------------
constexpr int kScanMaxPat = 130;  // patterns overlapping one 128-row tile
constexpr int kScanThreads = 512;  // one warp per pattern at a time
constexpr int kScanWarps = kScanThreads / 32;

template <int ELL>
__global__ void __launch_bounds__(kScanThreads) k_plan_scan(const __nv_bfloat16* __restrict__ Cs, int Kp,
                                                   int N, int npat, int budget, int policy,
                                                   ResidLists rl, unsigned int* done_counter) {
  // the sum of the chunk gradients (next in the stream) does not read the
  // lists: let it start now
  if (threadIdx.x == 0) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int mt = blockIdx.x;
  const long long M = (long long)npat * ELL;
  const long long row0 = (long long)mt * 128;
  const long long row_last = min(row0 + 127, M - 1);
  const int b_lo = (int)(row0 / ELL), b_hi = (int)(row_last / ELL);
  const size_t plane = (size_t)M * Kp;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __shared__ int s_cnt[kScanMaxPat];
  __shared__ int s_or[kScanWarps], s_sum[kScanWarps], s_rows[kScanWarps];
  __shared__ int s_last;
  int w_over = 0, w_sum = 0;
  for (int b = b_lo + warp; b <= b_hi; b += kScanWarps) {
    // the tile holding the pattern's first row writes its list
    const bool owner = (long long)b * ELL >= row0;
    int count = 0;
    for (int i0 = 0; i0 < N; i0 += 32) {
      const int i = i0 + lane;
      float Dv[ELL][ELL];
      bool nz = false;
#pragma unroll
      for (int a = 0; a < ELL; ++a)
#pragma unroll
        for (int k = 0; k < ELL; ++k) {
          float v = 0.f;
          if (i < N) {
            const size_t e = ((size_t)b * ELL + a) * Kp + (size_t)i * ELL + k;
            v = __bfloat162float(Cs[e]) + __bfloat162float(Cs[plane + e]) - (a == k ? 1.f : 0.f);
          }
          Dv[a][k] = v;
          nz |= v != 0.f;
        }
      const unsigned bal = __ballot_sync(0xffffffffu, nz);
      const int pos = count + __popc(bal & ((1u << lane) - 1u));
      if (nz && owner && pos < rl.ksp) {
        rl.idx[(size_t)b * rl.ksp + pos] = i;
        float* dst = rl.D + ((size_t)b * rl.ksp + pos) * ELL * ELL;
#pragma unroll
        for (int a = 0; a < ELL; ++a)
#pragma unroll
          for (int k = 0; k < ELL; ++k) dst[a * ELL + k] = Dv[a][k];
      }
      count += __popc(bal);
    }
    if (owner && lane == 0) rl.nnz[b] = count;
    if (lane == 0) s_cnt[b - b_lo] = count;
    w_over |= count > rl.ksp ? 1 : 0;
    w_sum += count;
  }
  if (lane == 0) {
    s_or[warp] = w_over;
    s_sum[warp] = w_sum;
  }
  __syncthreads();
  // rows of this tile that need corrections, in row order: slot mt*RCAP + rank
  // (thread t < 128 takes row row0 + t)
  const long long row = row0 + threadIdx.x;
  const bool valid = threadIdx.x < 128 && row < M;
  const bool ne = valid && s_cnt[(int)(row / ELL) - b_lo] > 0;
  const unsigned bal = __ballot_sync(0xffffffffu, ne);
  if (lane == 0) s_rows[warp] = __popc(bal);
  __syncthreads();
  int rank = __popc(bal & ((1u << lane) - 1u));
  for (int w = 0; w < warp; ++w) rank += s_rows[w];
  int nrows = 0;
  for (int w = 0; w < kScanWarps; ++w) nrows += s_rows[w];
  if (valid) {
    const bool slotted = ne && rank < kResidRcap;
    rl.rslot[row] = slotted ? mt * kResidRcap + rank : -1;
    if (slotted) rl.rowlist[(size_t)mt * kResidRcap + rank] = (int)row;
  }
  if (threadIdx.x == 0) {
    int over = 0;
    long long sum = 0;
    for (int w = 0; w < kScanWarps; ++w) {
      over |= s_or[w];
      sum += s_sum[w];
    }
    // a list or a slot table that overflowed can only be decoded by the GEMM
    over |= nrows > kResidRcap ? 1 : 0;
    const long long nb = b_hi - b_lo + 1;
    int dense;
    if (policy == GC_DECODE_DENSE)
      dense = 1;
    else if (policy == GC_DECODE_RESIDUAL)
      dense = over;
    else
      dense = over || sum > (long long)budget * nb;
    rl.tflag[mt] = dense;
    rl.tcount[mt] = min(nrows, kResidRcap);
    __threadfence();
    // the counter wraps to 0 on the last CTA, ready for the next launch
    const unsigned prev = atomicInc(done_counter, gridDim.x - 1);
    s_last = prev == gridDim.x - 1;
  }
  __syncthreads();  // also: every read of s_rows above is done
  if (s_last) {
    // every tile's flag is written: list the GEMM's tiles in ascending order
    __threadfence();
    int base = 0;
    for (int t0 = 0; t0 < (int)gridDim.x; t0 += kScanThreads) {
      const int t = t0 + threadIdx.x;
      const bool f = t < (int)gridDim.x && *reinterpret_cast<volatile int*>(rl.tflag + t) != 0;
      const unsigned bf = __ballot_sync(0xffffffffu, f);
      if (lane == 0) s_rows[warp] = __popc(bf);
      __syncthreads();
      int pos = base + __popc(bf & ((1u << lane) - 1u));
      for (int w = 0; w < warp; ++w) pos += s_rows[w];
      if (f) rl.dlist[pos] = t;
      for (int w = 0; w < kScanWarps; ++w) base += s_rows[w];
      __syncthreads();
    }
    if (threadIdx.x == 0) *rl.ndense = base;
  }
}

// ---------------------------------------------------------------------------
// s = sum_i g_{D_i} (chunks added in order 0..N-1).
// ---------------------------------------------------------------------------
__device__ __forceinline__ void gsum_cols(const float* __restrict__ G, int N, int d, int vec,
                                          float* __restrict__ gsum) {
  const long long c0 = ((long long)blockIdx.x * blockDim.x + threadIdx.x) * 4;
  if (c0 >= d) return;
  if (vec) {
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    const float* p = G + c0;
    int i = 0;
    for (; i + 8 <= N; i += 8) {
      float4 q[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) q[u] = __ldg(reinterpret_cast<const float4*>(p + (size_t)(i + u) * d));
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        acc.x += q[u].x;
        acc.y += q[u].y;
        acc.z += q[u].z;
        acc.w += q[u].w;
      }
    }
    for (; i < N; ++i) {
      const float4 q = __ldg(reinterpret_cast<const float4*>(p + (size_t)i * d));
      acc.x += q.x;
      acc.y += q.y;
      acc.z += q.z;
      acc.w += q.w;
    }
    *reinterpret_cast<float4*>(gsum + c0) = acc;
  } else {
    for (int v = 0; v < 4; ++v) {
      const long long c = c0 + v;
      if (c >= d) break;
      float acc = 0.f;
      for (int i = 0; i < N; ++i) acc += __ldg(G + (size_t)i * d + c);
      gsum[c] = acc;
    }
  }
}

// Launched as a programmatic dependent of the plan scan, which it does not
// read: the two run side by side.  It waits for the scan before it exits, so
// that work ordered after it (the residual decode, which reads both) finds
// the scan complete.
__global__ void __launch_bounds__(128) k_gsum(const float* __restrict__ G, int N, int d, int vec,
                                              float* __restrict__ gsum) {
  gsum_cols(G, N, d, vec, gsum);
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  asm volatile("griddepcontrol.wait;" ::: "memory");
}

// ---------------------------------------------------------------------------
// Residual decode.  Block (tile mt, range r): columns c = r*W + 4*t .. +3 of
// every block k (the same offsets in all ell blocks, so one load of
// g_{D_i}[k'] serves every output block) for the rows of tile mt.
// ---------------------------------------------------------------------------
__device__ __forceinline__ float4 ld4(const float* p, long long off, bool vec, int nvalid) {
  if (vec && nvalid == 4) return __ldg(reinterpret_cast<const float4*>(p + off));
  float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
  if (nvalid > 0) v.x = __ldg(p + off);
  if (nvalid > 1) v.y = __ldg(p + off + 1);
  if (nvalid > 2) v.z = __ldg(p + off + 2);
  if (nvalid > 3) v.w = __ldg(p + off + 3);
  return v;
}
__device__ __forceinline__ void st4(float* p, long long off, bool vec, int nvalid, float4 v) {
  if (vec && nvalid == 4) {
    __stcs(reinterpret_cast<float4*>(p + off), v);  // written once, never re-read here
    return;
  }
  if (nvalid > 0) __stcs(p + off, v.x);
  if (nvalid > 1) __stcs(p + off + 1, v.y);
  if (nvalid > 2) __stcs(p + off + 2, v.z);
  if (nvalid > 3) __stcs(p + off + 3, v.w);
}

// One corrected row (pattern b, block k) over this thread's 4 columns:
// ghat = s + sum_e sum_k' D_e[k][k'] g_{i_e}[k'L + c], and its squared-error
// partial (one per warp) into the row's slot.
template <int ELL>
__device__ __forceinline__ void resid_row(const float* __restrict__ G, const ResidLists& rl, int b,
                                          int k, long long row, int r, int c, int d, int L,
                                          bool vecw, const int (&nv)[ELL], const float4 (&sv)[ELL],
                                          float* __restrict__ Ghat) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nz = __ldg(rl.nnz + b);  // <= ksp: longer lists make the tile dense
  float4 cr = make_float4(0.f, 0.f, 0.f, 0.f);
  for (int e = 0; e < nz; ++e) {
    const int i = __ldg(rl.idx + (size_t)b * rl.ksp + e);
    const float* Dr = rl.D + ((size_t)b * rl.ksp + e) * ELL * ELL + k * ELL;
#pragma unroll
    for (int kp = 0; kp < ELL; ++kp) {
      const float w = __ldg(Dr + kp);
      if (nv[kp] == 0 || w == 0.f) continue;
      const float4 g = ld4(G, (size_t)i * d + (size_t)kp * L + c, vecw, nv[kp]);
      cr.x = fmaf(w, g.x, cr.x);
      cr.y = fmaf(w, g.y, cr.y);
      cr.z = fmaf(w, g.z, cr.z);
      cr.w = fmaf(w, g.w, cr.w);
    }
  }
  int nvk = 0;
  float4 svk = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
  for (int kk = 0; kk < ELL; ++kk)
    if (kk == k) {
      nvk = nv[kk];
      svk = sv[kk];
    }
  // corrections only on the output columns that exist
  float sq = nvk > 0 ? cr.x * cr.x : 0.f;
  if (nvk > 1) sq = fmaf(cr.y, cr.y, sq);
  if (nvk > 2) sq = fmaf(cr.z, cr.z, sq);
  if (nvk > 3) sq = fmaf(cr.w, cr.w, sq);
  if (Ghat && nvk > 0)
    st4(Ghat, (size_t)b * d + (size_t)k * L + c, vecw, nvk,
        make_float4(svk.x + cr.x, svk.y + cr.y, svk.z + cr.z, svk.w + cr.w));
  if (rl.msp) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
    if (lane == 0) {
      const int slot = __ldg(rl.rslot + row);
      rl.msp[(size_t)slot * rl.parts + (size_t)r * (kResidThreads / 32) + warp] = sq;
    }
  }
}

// Block (tile mt, range r, row slice z): rows [row0 + z*rps, row0 + (z+1)*rps)
// of the tile (rps = 128 / gridDim.z; slices give small batches more blocks).
template <int ELL>
__global__ void __launch_bounds__(kResidThreads, ELL <= 4 ? 4 : 2) k_decode_resid(const float* __restrict__ G,
                                                                const float* __restrict__ gsum,
                                                                ResidLists rl, int npat, int d,
                                                                int L, int vec,
                                                                float* __restrict__ Ghat) {
  // a programmatic dependent of the sum of the chunk gradients: s and the
  // scan's lists are complete once this wait returns
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int mt = blockIdx.x;
  if (__ldg(rl.tflag + mt)) return;  // the GEMM writes this tile
  const int cnt = __ldg(rl.tcount + mt);
  if (!Ghat && cnt == 0) return;     // errors only and every pattern exact: nothing to do
  const int r = blockIdx.y;
  const long long M = (long long)npat * ELL;
  const int rps = 128 / gridDim.z;
  const long long lo = (long long)mt * 128 + (long long)blockIdx.z * rps;
  const long long hi = min(lo + rps, M);
  if (lo >= hi) return;
  const int c = r * kResidW + threadIdx.x * 4;
  const bool vecw = vec != 0;
  // valid columns of this thread in block k (padding past L and past d), and s there
  int nv[ELL];
  float4 sv[ELL];
#pragma unroll
  for (int k = 0; k < ELL; ++k) {
    const long long col = (long long)k * L + c;
    int n = min(4, L - c);
    n = (int)min((long long)n, (long long)d - col);
    nv[k] = n < 0 ? 0 : n;
    sv[k] = (Ghat && nv[k] > 0) ? ld4(gsum, col, vecw, nv[k]) : make_float4(0.f, 0.f, 0.f, 0.f);
  }
  if (!Ghat) {
    // errors only: the tile's listed rows in this slice
    for (int q = 0; q < cnt; ++q) {
      const int row = __ldg(rl.rowlist + (size_t)mt * kResidRcap + q);
      if (row < lo || row >= hi) continue;
      resid_row<ELL>(G, rl, row / ELL, row % ELL, row, r, c, d, L, vecw, nv, sv, nullptr);
    }
    return;
  }
  const int b_lo = (int)(lo / ELL), b_hi = (int)((hi - 1) / ELL);
  for (int b = b_lo; b <= b_hi; ++b) {
    const int nz = __ldg(rl.nnz + b);
#pragma unroll
    for (int k = 0; k < ELL; ++k) {
      const long long row = (long long)b * ELL + k;
      if (row < lo || row >= hi) continue;  // another slice's or tile's row
      if (nz == 0) {  // exact pattern: ghat_b = s, zero error
        if (nv[k] > 0) st4(Ghat, (size_t)b * d + (size_t)k * L + c, vecw, nv[k], sv[k]);
      } else {
        resid_row<ELL>(G, rl, b, k, row, r, c, d, L, vecw, nv, sv, Ghat);
      }
    }
  }
}

// ---------------------------------------------------------------------------
// launches
// ---------------------------------------------------------------------------
int launch_plan_scan(const __nv_bfloat16* Cs, int Kp, int N, int ell, int npat, int budget,
                     int policy, const ResidLists& rl, unsigned int* done_counter, cudaStream_t s) {
  const long long M = (long long)npat * ell;
  const long long nmt = (M + 127) / 128;
  if (nmt == 0) return GC_OK;
  if (nmt > (1LL << 31) - 1) return fail(GC_ERR_UNSUPPORTED, "too many row tiles");
#define GC_SCAN(E) \
  case E: k_plan_scan<E><<<(unsigned)nmt, kScanThreads, 0, s>>>(Cs, Kp, N, npat, budget, policy, rl, done_counter); break;
  switch (ell) {
    GC_SCAN(1)
    GC_SCAN(2)
    GC_SCAN(3)
    GC_SCAN(4)
    GC_SCAN(5)
    GC_SCAN(6)
    GC_SCAN(7)
    GC_SCAN(8)
    default: return fail(GC_ERR_UNSUPPORTED, "ell=%d exceeds GC_MAX_ELL", ell);
  }
#undef GC_SCAN
  count_launches(1);
  return cuda_check(cudaGetLastError(), "k_plan_scan");
}

int launch_gsum(const float* G, int N, int d, float* gsum, cudaStream_t s) {
  const bool vec = d % 4 == 0 && reinterpret_cast<uintptr_t>(G) % 16 == 0 &&
                   reinterpret_cast<uintptr_t>(gsum) % 16 == 0;
  const long long quads = ((long long)d + 3) / 4;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3((unsigned)((quads + 127) / 128));
  cfg.blockDim = dim3(128);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t e = cudaLaunchKernelEx(&cfg, k_gsum, G, N, d, vec ? 1 : 0, gsum);
  if (e != cudaSuccess) return cuda_check(e, "cudaLaunchKernelEx(k_gsum)");
  count_launches(1);
  return GC_OK;
}

int launch_decode_resid(const float* G, const float* gsum, const ResidLists& rl, int ell, int npat,
                        int d, float* Ghat, cudaStream_t s) {
  if (npat == 0) return GC_OK;
  const int L = (d + ell - 1) / ell;
  const bool vec = d % 4 == 0 && L % 4 == 0 && reinterpret_cast<uintptr_t>(G) % 16 == 0 &&
                   reinterpret_cast<uintptr_t>(gsum) % 16 == 0 &&
                   (!Ghat || reinterpret_cast<uintptr_t>(Ghat) % 16 == 0);
  const long long nmt = ((long long)npat * ell + 127) / 128;
  const long long nranges = (L + kResidW - 1) / kResidW;
  if (nmt > (1LL << 31) - 1 || nranges > 65535) return fail(GC_ERR_UNSUPPORTED, "residual decode grid too large");
  // tiles fastest: the CTAs of one column range run side by side and share
  // its chunk-gradient lines in L2; small batches split each tile's rows
  // over up to 8 blocks so that every SM has a few
  int slices = 1;
  while (slices < 8 && nmt * nranges * slices < 16LL * device_sm_count()) slices *= 2;
  dim3 grid((unsigned)nmt, (unsigned)nranges, (unsigned)slices);
  // a programmatic dependent of k_gsum (the launch overlaps its tail)
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(kResidThreads);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t e = cudaSuccess;
#define GC_RESID(E) \
  case E: e = cudaLaunchKernelEx(&cfg, k_decode_resid<E>, G, gsum, rl, npat, d, L, vec ? 1 : 0, Ghat); break;
  switch (ell) {
    GC_RESID(1)
    GC_RESID(2)
    GC_RESID(3)
    GC_RESID(4)
    GC_RESID(5)
    GC_RESID(6)
    GC_RESID(7)
    GC_RESID(8)
    default: return fail(GC_ERR_UNSUPPORTED, "ell=%d exceeds GC_MAX_ELL", ell);
  }
#undef GC_RESID
  if (e != cudaSuccess) return cuda_check(e, "cudaLaunchKernelEx(k_decode_resid)");
  count_launches(1);
  return GC_OK;
}

}  // namespace gc
