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
//                   partials) and the tile's path; the last CTA ORs the tile
//                   flags into one "some tile is on the GEMM" word.
//   k_decode_resid  one CTA per 32-column stripe of every block (and pattern
//                   group): stages the stripe of all N*ell chunk-gradient
//                   blocks in shared memory (G is read from HBM once in
//                   all), forms s from it, writes s to the rows of exact
//                   patterns and s + corrections to the listed rows, with
//                   ||ghat_b - s||^2 = ||corrections||^2 per (row, stripe).
//   k_gsum          s alone, for batches too wide for the stripe (N*ell >
//                   kResidMaxRows), which go to the GEMM.
#include <algorithm>

#include "gc_internal.cuh"

namespace gc {

int resid_ksp(int ell) { return ell <= 2 ? 32 : (ell <= 4 ? 16 : 8); }

bool resid_fits(int N, int ell) { return (long long)N * ell <= kResidMaxRows; }

static size_t resid_smem(int N, int ell) {
  return ((size_t)N * ell + ell) * kResidW * sizeof(float);
}

size_t resid_ws_bytes(int N, int ell, int npat, int d) {
  const int L = (d + ell - 1) / ell;
  const long long M = (long long)npat * ell;
  const long long nmt = (M + 127) / 128;
  const int ksp = std::min(resid_ksp(ell), N);
  const long long parts = (L + kResidW - 1) / kResidW;
  return align_up((size_t)npat * sizeof(int32_t), 256) +
         align_up((size_t)npat * ksp * sizeof(int32_t), 256) +
         align_up((size_t)npat * ksp * ell * ell * sizeof(float), 256) +
         align_up((size_t)nmt * sizeof(int32_t), 256) + align_up(sizeof(int32_t), 256) +
         align_up((size_t)M * sizeof(int32_t), 256) +
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
  r.parts = (L + kResidW - 1) / kResidW;
  r.nnz = c.take<int32_t>(npat);
  r.idx = c.take<int32_t>((size_t)npat * r.ksp);
  r.D = c.take<float>((size_t)npat * r.ksp * ell * ell);
  r.tflag = c.take<int32_t>(nmt);
  r.any_dense = c.take<int32_t>(1);
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

template <int ELL>
__global__ void __launch_bounds__(128) k_plan_scan(const __nv_bfloat16* __restrict__ Cs, int Kp,
                                                   int N, int npat, int budget, int policy,
                                                   ResidLists rl, unsigned int* done_counter) {
  const int mt = blockIdx.x;
  const long long M = (long long)npat * ELL;
  const long long row0 = (long long)mt * 128;
  const long long row_last = min(row0 + 127, M - 1);
  const int b_lo = (int)(row0 / ELL), b_hi = (int)(row_last / ELL);
  const size_t plane = (size_t)M * Kp;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __shared__ int s_cnt[kScanMaxPat];
  __shared__ int s_or[4], s_sum[4], s_rows[4];
  __shared__ int s_last;
  int w_over = 0, w_sum = 0;
  for (int b = b_lo + warp; b <= b_hi; b += 4) {
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
  const long long row = row0 + threadIdx.x;
  const bool valid = row < M;
  const bool ne = valid && s_cnt[(int)(row / ELL) - b_lo] > 0;
  const unsigned bal = __ballot_sync(0xffffffffu, ne);
  if (lane == 0) s_rows[warp] = __popc(bal);
  __syncthreads();
  int rank = __popc(bal & ((1u << lane) - 1u));
  for (int w = 0; w < warp; ++w) rank += s_rows[w];
  const int nrows = s_rows[0] + s_rows[1] + s_rows[2] + s_rows[3];
  if (valid) {
    const bool slotted = ne && rank < kResidRcap;
    rl.rslot[row] = slotted ? mt * kResidRcap + rank : -1;
    if (slotted) rl.rowlist[(size_t)mt * kResidRcap + rank] = (int)row;
  }
  if (threadIdx.x == 0) {
    int over = 0;
    long long sum = 0;
    for (int w = 0; w < 4; ++w) {
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
  __syncthreads();
  if (s_last) {
    __threadfence();
    int any = 0;
    for (int t = threadIdx.x; t < (int)gridDim.x; t += blockDim.x)
      any |= *reinterpret_cast<volatile int*>(rl.tflag + t);
    any = __syncthreads_or(any);
    if (threadIdx.x == 0) *rl.any_dense = any;
  }
}

// ---------------------------------------------------------------------------
// s = sum_i g_{D_i} (chunks added in order 0..N-1).
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(128) k_gsum(const float* __restrict__ G, int N, int d, int vec,
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

// ---------------------------------------------------------------------------
// Residual decode.  Block (stripe, group): columns c0 .. c0+31 of every block
// k (c0 = 32 * stripe; the same offsets in all ell blocks, so one staged row
// of g_{D_i}[k'] serves every output block), patterns [b0, b1).
// ---------------------------------------------------------------------------
template <int ELL>
__global__ void __launch_bounds__(kResidThreads) k_decode_resid(const float* __restrict__ G,
                                                                ResidLists rl, int N, int npat,
                                                                int d, int L, int ppg, int vec,
                                                                float* __restrict__ gsum,
                                                                float* __restrict__ Ghat) {
  extern __shared__ float sm[];
  constexpr int W = kResidW;
  constexpr int NW = kResidThreads / 32;
  const int rows = N * ELL;
  float* sg = sm;               // [rows][W]: row i*ELL + k' = g_{D_i}[k'*L + c0 ..]
  float* ss = sm + rows * W;    // [ELL][W]: s
  const int stripe = blockIdx.x;
  const int c0 = stripe * W;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // ---- stage the stripe (zero past L and past d)
  {
    const int q = tid & 7;           // 16-byte quarter of a 128-byte row
    const int c = c0 + 4 * q;
    constexpr int RPP = kResidThreads / 8;
    for (int r0 = 0; r0 < rows; r0 += RPP * 4) {
      float4 v[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int r = r0 + u * RPP + (tid >> 3);
        v[u] = make_float4(0.f, 0.f, 0.f, 0.f);
        if (r < rows) {
          const int i = r / ELL, kp = r - i * ELL;
          const long long col = (long long)kp * L + c;
          const float* src = G + (size_t)i * d + col;
          if (vec && c + 3 < L && col + 3 < d) {
            v[u] = __ldg(reinterpret_cast<const float4*>(src));
          } else {
            float t[4] = {0.f, 0.f, 0.f, 0.f};
            for (int e = 0; e < 4; ++e)
              if (c + e < L && col + e < d) t[e] = __ldg(src + e);
            v[u] = make_float4(t[0], t[1], t[2], t[3]);
          }
        }
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int r = r0 + u * RPP + (tid >> 3);
        if (r < rows) *reinterpret_cast<float4*>(sg + r * W + 4 * q) = v[u];
      }
    }
  }
  __syncthreads();
  // ---- s for the stripe, chunks added in order (the order k_gsum uses)
  for (int t = tid; t < ELL * W; t += kResidThreads) {
    const int k = t / W, c = t - k * W;
    float acc = 0.f;
    for (int i = 0; i < N; ++i) acc += sg[(i * ELL + k) * W + c];
    ss[t] = acc;
    const long long col = (long long)k * L + c0 + c;
    if (gsum && blockIdx.y == 0 && c0 + c < L && col < d) gsum[col] = acc;
  }
  __syncthreads();
  const int b0 = blockIdx.y * ppg;
  const int b1 = min(npat, b0 + ppg);
  bool ok[ELL];
  float sr[ELL];
#pragma unroll
  for (int k = 0; k < ELL; ++k) {
    ok[k] = c0 + lane < L && (long long)k * L + c0 + lane < d;
    sr[k] = ss[k * W + lane];
  }
  // ---- exact patterns: ghat_b = s (zero error)
  if (Ghat) {
    for (int b = b0 + warp; b < b1; b += NW) {
      if (__ldg(rl.nnz + b) != 0) continue;
      float* o = Ghat + (size_t)b * d + c0 + lane;
#pragma unroll
      for (int k = 0; k < ELL; ++k) {
        const long long row = (long long)b * ELL + k;
        if (__ldg(rl.tflag + (row >> 7)) == 0 && ok[k]) __stcs(o + (size_t)k * L, sr[k]);
      }
    }
  }
  // ---- rows with corrections, tile by tile from the scan's lists
  const long long t_lo = ((long long)b0 * ELL) >> 7, t_hi = ((long long)b1 * ELL - 1) >> 7;
  for (long long mt = t_lo; mt <= t_hi && b0 < b1; ++mt) {
    if (__ldg(rl.tflag + mt)) continue;
    const int cnt = __ldg(rl.tcount + mt);
    for (int q = warp; q < cnt; q += NW) {
      const int row = __ldg(rl.rowlist + mt * kResidRcap + q);
      const int b = row / ELL, k = row - b * ELL;
      if (b < b0 || b >= b1) continue;
      const int nz = __ldg(rl.nnz + b);  // <= ksp: longer lists make the tile dense
      float corr = 0.f;
      for (int e = 0; e < nz; ++e) {
        const int i = __ldg(rl.idx + (size_t)b * rl.ksp + e);
        const float* Dr = rl.D + ((size_t)b * rl.ksp + e) * ELL * ELL + k * ELL;
#pragma unroll
        for (int kp = 0; kp < ELL; ++kp) corr = fmaf(__ldg(Dr + kp), sg[(i * ELL + kp) * W + lane], corr);
      }
      // output column k*L + c0 + lane exists (padding past L and past d does not)
      const bool col_ok = c0 + lane < L && (long long)k * L + c0 + lane < d;
      if (Ghat && col_ok) __stcs(Ghat + (size_t)b * d + (size_t)k * L + c0 + lane, ss[k * W + lane] + corr);
      if (rl.msp) {
        float sq = col_ok ? corr * corr : 0.f;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
        if (lane == 0) rl.msp[((size_t)mt * kResidRcap + q) * rl.parts + stripe] = sq;
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
  case E: k_plan_scan<E><<<(unsigned)nmt, 128, 0, s>>>(Cs, Kp, N, npat, budget, policy, rl, done_counter); break;
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
  k_gsum<<<(unsigned)((quads + 127) / 128), 128, 0, s>>>(G, N, d, vec ? 1 : 0, gsum);
  count_launches(1);
  return cuda_check(cudaGetLastError(), "k_gsum");
}

template <int ELL>
static int launch_resid_t(dim3 grid, size_t smem, const float* G, const ResidLists& rl, int N,
                          int npat, int d, int L, int ppg, int vec, float* gsum, float* Ghat,
                          cudaStream_t s) {
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(k_decode_resid<ELL>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)resid_smem(kResidMaxRows / ELL, ELL));
    if (e != cudaSuccess) return cuda_check(e, "cudaFuncSetAttribute(k_decode_resid)");
    attr = true;
  }
  k_decode_resid<ELL><<<grid, kResidThreads, smem, s>>>(G, rl, N, npat, d, L, ppg, vec, gsum, Ghat);
  return GC_OK;
}

int launch_decode_resid(const float* G, const ResidLists& rl, int N, int ell, int npat, int d,
                        float* gsum, float* Ghat, cudaStream_t s) {
  if (npat == 0) return GC_OK;
  if (!resid_fits(N, ell)) return fail(GC_ERR_UNSUPPORTED, "residual decode: N*ell > %d", kResidMaxRows);
  const int L = (d + ell - 1) / ell;
  const bool vec = d % 4 == 0 && L % 4 == 0 && reinterpret_cast<uintptr_t>(G) % 16 == 0;
  const long long nstripes = (L + kResidW - 1) / kResidW;
  const size_t smem = resid_smem(N, ell);
  // enough blocks for a few per SM: the pattern groups split what the column
  // stripes leave (each group stages its stripe again, from L2)
  const int per_sm = std::max(1, std::min(8, (int)((200u << 10) / smem)));
  const long long want = 2LL * per_sm * device_sm_count();
  long long groups = std::max<long long>(1, (want + nstripes - 1) / nstripes);
  groups = std::min<long long>(groups, std::min<long long>(npat, 65535));
  const int ppg = (int)((npat + groups - 1) / groups);
  groups = (npat + ppg - 1) / ppg;
  if (nstripes > (1LL << 31) - 1) return fail(GC_ERR_UNSUPPORTED, "d too large");
  dim3 grid((unsigned)nstripes, (unsigned)groups);
  int rc;
  switch (ell) {
    case 1: rc = launch_resid_t<1>(grid, smem, G, rl, N, npat, d, L, ppg, vec, gsum, Ghat, s); break;
    case 2: rc = launch_resid_t<2>(grid, smem, G, rl, N, npat, d, L, ppg, vec, gsum, Ghat, s); break;
    case 3: rc = launch_resid_t<3>(grid, smem, G, rl, N, npat, d, L, ppg, vec, gsum, Ghat, s); break;
    case 4: rc = launch_resid_t<4>(grid, smem, G, rl, N, npat, d, L, ppg, vec, gsum, Ghat, s); break;
    case 5: rc = launch_resid_t<5>(grid, smem, G, rl, N, npat, d, L, ppg, vec, gsum, Ghat, s); break;
    case 6: rc = launch_resid_t<6>(grid, smem, G, rl, N, npat, d, L, ppg, vec, gsum, Ghat, s); break;
    case 7: rc = launch_resid_t<7>(grid, smem, G, rl, N, npat, d, L, ppg, vec, gsum, Ghat, s); break;
    case 8: rc = launch_resid_t<8>(grid, smem, G, rl, N, npat, d, L, ppg, vec, gsum, Ghat, s); break;
    default: return fail(GC_ERR_UNSUPPORTED, "ell=%d exceeds GC_MAX_ELL", ell);
  }
  if (rc) return rc;
  count_launches(1);
  return cuda_check(cudaGetLastError(), "k_decode_resid");
}

}  // namespace gc
