// Worker encoding (eq. 2), PS decoding of transmissions (Sec. II-B) and the
// parameter update (Sec. I).
//
// All three are HBM-bound streaming kernels with coalesced accesses along the
// block coordinate c (consecutive threads, consecutive columns).
#include <algorithm>

#include "gc_internal.cuh"

namespace gc {

// T[b][j][c] = sum_{p < psi[b][j]} sum_k E[b][j][p][k] * g_{order[j][p]}[k*L + c]
// (g zero past d), eq. (2).
//
// Under the cyclic assignment (order[j][p] = (j + p) mod N, Sec. III) the
// holders of chunk i are the workers i, i-1, ..., i-delta+1, so a block that
// sweeps the chunks in order over one column stripe keeps a ring of
// per-worker accumulators in registers: each loaded stripe of g_{D_i} feeds
// every holder of D_i once, and a worker's transmission is stored when its
// window of chunks has passed.  The chunk gradients are read once per
// (pattern, worker group) instead of once per worker and slot.
// Block = (pattern b, column stripe, worker group [j0, j1)).  The ring has DR
// slots (DR = the power of two >= delta): worker j0 + jj accumulates in ring
// slot jj mod DR.  The coefficients are staged by ring slot,
// s_e[k][w][s] = E[b][j0 + jj][p][k] with p = (w - s) mod DR and jj = w - p
// (the worker in slot s takes the chunk at sweep position w as its p-th; zero
// past its psi, for p >= delta and outside the group), so every chunk step is
// DR/4 vector loads from shared memory and DR*V FMAs with no branches, and the
// accumulators pair up by slot: one packed two-wide FMA takes the
// coefficients of slots (2r, 2r+1) as they lie in shared memory and one
// column's value twice.  Positions past the group's range add zeros.
// Each thread keeps its next kEncStages - 1 chunk-stripe loads in flight:
// cp.async copies its own columns of a coming (position, block) step into its
// slots of a shared-memory ring (zero-filled past L and past d) and waits
// with cp.async.wait_group, so no thread reads another's data and no barrier
// or spin-wait is needed.
// A transmission is summed over slots p ascending, blocks k ascending within
// a slot -- the same order in the direct form, which a block whose workers'
// orders are not cyclic (an explicit order) uses instead.
constexpr int kEncThreads = 128;
constexpr int kEncSmemFloats = 12288;  // staged coefficients (48 KB)
constexpr int kEncStages = 8;          // ring of chunk-stripe steps per thread

__device__ __forceinline__ uint32_t enc_smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
// cp.async of `bytes` (4, 8 or 16) with zero fill past `valid` bytes
template <int BYTES>
__device__ __forceinline__ void cp_async_zfill(uint32_t dst, const float* src, int valid) {
  if (BYTES == 16)
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(valid) : "memory");
  else if (BYTES == 8)
    asm volatile("cp.async.ca.shared.global [%0], [%1], 8, %2;" ::"r"(dst), "l"(src), "r"(valid) : "memory");
  else
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"(dst), "l"(src), "r"(valid) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

__device__ __forceinline__ void enc_load(const float* __restrict__ gi, long long col, int c, int L,
                                         int d, bool vec, float* g, int V) {
  if (vec && V == 4 && c + 3 < L && col + 3 < d) {
    const float4 q = __ldg(reinterpret_cast<const float4*>(gi + col));
    g[0] = q.x; g[1] = q.y; g[2] = q.z; g[3] = q.w;
  } else if (vec && V == 2 && c + 1 < L && col + 1 < d) {
    const float2 q = __ldg(reinterpret_cast<const float2*>(gi + col));
    g[0] = q.x; g[1] = q.y;
  } else {
    for (int v = 0; v < V; ++v) g[v] = (c + v < L && col + v < d) ? __ldg(gi + col + v) : 0.f;
  }
}

template <int V>
__device__ __forceinline__ void enc_store(float* __restrict__ Tr, int c, int L, bool vec, const float* a) {
  if (vec && V == 4 && c + 3 < L) {
    *reinterpret_cast<float4*>(Tr) = make_float4(a[0], a[V > 1 ? 1 : 0], a[V > 2 ? 2 : 0], a[V > 3 ? 3 : 0]);
  } else if (vec && V == 2 && c + 1 < L) {
    *reinterpret_cast<float2*>(Tr) = make_float2(a[0], a[V > 1 ? 1 : 0]);
  } else {
#pragma unroll
    for (int v = 0; v < V; ++v)
      if (c + v < L) Tr[v] = a[v];
  }
}

// Move the accumulators of ring slot S (half S & 1 of pair S >> 1) to a and
// clear them.
template <int DR, int V, int S>
__device__ __forceinline__ void enc_take(float2 (&acc)[DR / 2][V], float* a) {
#pragma unroll
  for (int v = 0; v < V; ++v) {
    float2& pr = acc[S >> 1][v];
    if (S & 1) {
      a[v] = pr.y;
      pr.y = 0.f;
    } else {
      a[v] = pr.x;
      pr.x = 0.f;
    }
  }
}

// enc_take of slot sc in [LO, HI), by binary search on sc
template <int DR, int V, int LO, int HI>
__device__ __forceinline__ void enc_take_any(float2 (&acc)[DR / 2][V], int sc, float* a) {
  if constexpr (HI - LO == 1) {
    enc_take<DR, V, LO>(acc, a);
  } else {
    constexpr int MID = (LO + HI) / 2;
    if (sc < MID)
      enc_take_any<DR, V, LO, MID>(acc, sc, a);
    else
      enc_take_any<DR, V, MID, HI>(acc, sc, a);
  }
}

// Workers per group so that the diagonal staging fits (and at most 256).
__host__ __device__ inline int enc_group_max(int DR, int ell) {
  const int j = kEncSmemFloats / (ell * DR) - DR;
  return j < 1 ? 1 : (j > 256 ? 256 : j);
}

// Shared memory of a block: the staged coefficients (diagonal layout, or the
// direct layout of a non-cyclic group) and the ring.
inline size_t enc_smem_bytes(int DR, int V, int ell, int delta, int J) {
  const size_t diag = (size_t)ell * (J + DR - 1) * DR;
  const size_t direct = (size_t)J * delta * ell;
  return (std::max(diag, direct) + (size_t)kEncStages * kEncThreads * V) * sizeof(float);
}

// Four blocks per SM (three with a 32-slot ring): about 120 registers a thread.
// A step of the sweep is KB consecutive blocks k of one chunk (KB divides
// ell): one copy group, one wait and KB times DR*V FMAs.
template <int DR, int V, int KB>
__global__ void __launch_bounds__(kEncThreads, DR == 32 ? 3 : 4)
    k_encode(const double* __restrict__ E, const int32_t* __restrict__ order,
             const int32_t* __restrict__ psi, int N, int m, int delta, int ell, int npat,
             const float* __restrict__ G, int d, int L, int J, int vec, float* __restrict__ T) {
  extern __shared__ __align__(16) float s_dyn[];
  __shared__ int s_np[256];               // processed counts of the group's workers (J <= 256)
  const int b = blockIdx.x;               // pattern fastest: blocks on one stripe share G in L2
  const int j0 = blockIdx.z * J, j1 = min(m, j0 + J);
  const int nj = j1 - j0;
  const int de = delta * ell;
  const int W = nj + DR - 1;              // sweep positions of the cyclic form
  float* s_e = s_dyn;
  float* s_ring = s_dyn + ((ell * W * DR > nj * de ? ell * W * DR : nj * de) + 3) / 4 * 4;
  const int c = (blockIdx.y * kEncThreads + threadIdx.x) * V;
  for (int t = threadIdx.x; t < nj; t += kEncThreads) {
    int np = psi[(size_t)b * m + j0 + t];
    s_np[t] = np < 0 ? 0 : (np > delta ? delta : np);  // bad values are flagged by the solve
  }
  int cyc = delta <= DR ? 1 : 0;
  for (int t = threadIdx.x; t < nj * delta; t += kEncThreads) {
    const int jj = t / delta, p = t - jj * delta;
    if (order[(size_t)(j0 + jj) * delta + p] != (j0 + jj + p) % N) cyc = 0;
  }
  cyc = __syncthreads_and(cyc);
  const double* Eb = E + ((size_t)b * m + j0) * de;
  if (!cyc) {
    // direct form: s_e[jj][p][k]
    for (int t = threadIdx.x; t < nj * de; t += kEncThreads) s_e[t] = (float)Eb[t];
    __syncthreads();
    if (c >= L) return;
    for (int jj = 0; jj < nj; ++jj) {
      float acc[V];
#pragma unroll
      for (int v = 0; v < V; ++v) acc[v] = 0.f;
      const int j = j0 + jj;
      for (int p = 0; p < s_np[jj]; ++p) {
        const int i = order[(size_t)j * delta + p];
        if (i < 0 || i >= N) continue;
        const float* gi = G + (size_t)i * d;
        for (int k = 0; k < ell; ++k) {
          float g[V];
          enc_load(gi, (long long)k * L + c, c, L, d, vec != 0, g, V);
          const float e = s_e[jj * de + p * ell + k];
#pragma unroll
          for (int v = 0; v < V; ++v) acc[v] = fmaf(e, g[v], acc[v]);
        }
      }
      enc_store<V>(T + ((size_t)b * m + j) * L + c, c, L, vec != 0, acc);
    }
    return;
  }
  // staging by ring slot, s_e[(k * W + w) * DR + s]: zero everywhere, then
  // each coefficient E[b][j0 + jj][p][k] (p < psi) lands at w = jj + p,
  // s = jj mod DR.  A thread takes whole workers (its loads, the worker's
  // p * ell + k run, are independent and go out together); consecutive
  // threads take consecutive workers, so the scattered stores hit distinct
  // banks (stride DR + 1 words).
  {
    float4* z = reinterpret_cast<float4*>(s_e);
    const int nz = ell * W * DR / 4;
    for (int t = threadIdx.x; t < nz; t += kEncThreads) z[t] = make_float4(0.f, 0.f, 0.f, 0.f);
  }
  __syncthreads();
  {
    const int kstep = W * DR;                     // next block k
    const int pstep = DR - (ell - 1) * W * DR;    // last block -> next slot p
    for (int jj = threadIdx.x; jj < nj; jj += kEncThreads) {
      const double* ej = Eb + (size_t)jj * de;
      float* sj = s_e + jj * (DR + 1) - (jj & ~(DR - 1));  // (jj + p) * DR + jj mod DR at p = 0
      const int n = s_np[jj] * ell;
      int off = 0, k = 0;
#pragma unroll 8
      for (int t = 0; t < n; ++t) {
        sj[off] = (float)__ldg(ej + t);
        if (++k == ell) {
          k = 0;
          off += pstep;
        } else {
          off += kstep;
        }
      }
    }
  }
  __syncthreads();
  if (c >= L) return;  // no barrier below
  // ring of NST stages, each [kb][thread][V]: this thread's V floats of each block
  constexpr int NST = kEncStages / KB;
  const uint32_t ring = enc_smem_u32(s_ring) + threadIdx.x * (V * 4);
  constexpr uint32_t kBlk = kEncThreads * V * 4;
  constexpr uint32_t kStage = kBlk * KB;
  // every step copies V whole floats (vector rows, no padding in this thread's columns)
  const bool full = vec && c + V <= L && (long long)ell * L <= d;
  // issue cursor: step (iw, ik) = blocks ik .. ik + KB - 1 of the chunk at
  // sweep position iw, read from src = G + ich * d + ik * L + c
  int iw = 0, ik = 0, slot = 0;
  int ich = j0 % N;
  const float* src = G + (size_t)ich * d + c;
  const int to_next = d - (ell - KB) * L;  // last step of a chunk -> first of the next
  auto issue = [&]() {
    if (iw < W) {
#pragma unroll
      for (int kb = 0; kb < KB; ++kb) {
        const uint32_t dst = ring + slot * kStage + kb * kBlk;
        const float* sk = src + (size_t)kb * L;
        if (full) {
          cp_async_zfill<V * 4>(dst, sk, V * 4);
        } else {
          const long long col = (long long)(ik + kb) * L + c;
          int nv = min(V, L - c);
          nv = (int)min((long long)nv, (long long)d - col);
          if (vec) {
            cp_async_zfill<V * 4>(dst, nv == V ? sk : G, nv == V ? V * 4 : 0);
          } else {
#pragma unroll
            for (int u = 0; u < V; ++u) cp_async_zfill<4>(dst + 4 * u, u < nv ? sk + u : G, u < nv ? 4 : 0);
          }
        }
      }
    }
    cp_async_commit();  // one group per step (possibly empty)
    ik += KB;
    if (ik == ell) {
      ik = 0;
      ++iw;
      src += to_next;
      if (++ich == N) {
        ich = 0;
        src = G + c;
      }
    } else {
      src += (size_t)KB * L;
    }
    slot = (slot + 1) & (NST - 1);
  };
  for (int q = 0; q < NST - 1; ++q) issue();
  const float* rd = s_ring + threadIdx.x * V;  // this thread's block 0 of stage 0
  int rs = 0;  // ring stage of the step being consumed
  // accumulators paired by ring slot: acc[r][v] = (slot 2r, slot 2r + 1) of
  // column v; one packed two-wide FMA (__ffma2_rn, the same rounding as two
  // fmaf) per pair
  float2 acc[DR / 2][V];
#pragma unroll
  for (int r = 0; r < DR / 2; ++r)
#pragma unroll
    for (int v = 0; v < V; ++v) acc[r][v] = make_float2(0.f, 0.f);
  // sweep position w holds chunk (j0 + w) mod N; worker j0 + w - DR + 1, in
  // ring slot (w + 1) mod DR, is complete after it
  const float* ecol = s_e;  // coefficients of (k = 0, w)
  float* tout = T + ((size_t)b * m + j0) * L + c;  // transmission of the next worker to complete
  const int kstride = W * DR;  // <= kEncSmemFloats
  // one copy of the step's code for every w (the FMAs do not depend on w);
  // the completed slot is taken through a switch on its index
#pragma unroll 1
  for (int w = 0; w < W; ++w) {
    {
      const float* ek = ecol;
      for (int kk = 0; kk < ell; kk += KB) {
        issue();
        cp_async_wait<NST - 1>();  // this step's copies have landed
        const float* gs = rd + rs * (kEncThreads * V * KB);
        rs = (rs + 1) & (NST - 1);
#pragma unroll
        for (int kb = 0; kb < KB; ++kb, ek += kstride) {
          float g[V];
          const float* gp = gs + kb * (kEncThreads * V);
          if (V == 4) {
            const float4 q = *reinterpret_cast<const float4*>(gp);
            g[0] = q.x;
            g[1 % V] = q.y;
            g[2 % V] = q.z;
            g[3 % V] = q.w;
          } else {
            const float2 q = *reinterpret_cast<const float2*>(gp);
            g[0] = q.x;
            g[1 % V] = q.y;
          }
          const float4* e4 = reinterpret_cast<const float4*>(ek);
#pragma unroll
          for (int q = 0; q < DR / 4; ++q) {
            const float4 e = e4[q];
            const float2 lo = make_float2(e.x, e.y), hi = make_float2(e.z, e.w);
#pragma unroll
            for (int v = 0; v < V; ++v) {
              const float2 gg = make_float2(g[v], g[v]);
              acc[2 * q][v] = __ffma2_rn(lo, gg, acc[2 * q][v]);
              acc[2 * q + 1][v] = __ffma2_rn(hi, gg, acc[2 * q + 1][v]);
            }
          }
        }
      }
      ecol += DR;
      const int jj = w - DR + 1;
      if (jj >= 0) {  // jj < nj since w < nj + DR - 1
        float a[V];
        enc_take_any<DR, V, 0, DR>(acc, (w + 1) & (DR - 1), a);
        enc_store<V>(tout, c, L, vec != 0, a);
        tout += L;
      }
    }
  }
  cp_async_wait<0>();  // no copy outlives the block
}

template <int DR, int V, int KB>
static int launch_enc_t(dim3 grid, size_t smem, const double* E, const int32_t* order,
                        const int32_t* psi, int N, int m, int delta, int ell, int npat,
                        const float* G, int d, int L, int J, int vec, float* T, cudaStream_t s) {
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(k_encode<DR, V, KB>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)((kEncSmemFloats + kEncStages * kEncThreads * V) * sizeof(float)));
    if (e != cudaSuccess) return cuda_check(e, "cudaFuncSetAttribute(k_encode)");
    attr = true;
  }
  k_encode<DR, V, KB><<<grid, kEncThreads, smem, s>>>(E, order, psi, N, m, delta, ell, npat, G, d, L, J, vec, T);
  return GC_OK;
}

int launch_encode(const double* E, const int32_t* order, const int32_t* psi, int N, int m,
                  int delta, int ell, int npat, const float* G, int d, float* T, cudaStream_t s) {
  const int L = (d + ell - 1) / ell;
  if ((long long)npat * m * L == 0) return GC_OK;
  // ring of the smallest power of two >= delta; 2 columns per thread with 32 slots
  const int DR = delta <= 4 ? 4 : delta <= 8 ? 8 : delta <= 16 ? 16 : 32;
  const int V = DR == 32 ? 2 : 4;
  const bool vec = d % V == 0 && L % V == 0 && reinterpret_cast<uintptr_t>(G) % (4 * V) == 0 &&
                   reinterpret_cast<uintptr_t>(T) % (4 * V) == 0;
  const long long stripes = ((long long)L + (long long)kEncThreads * V - 1) / ((long long)kEncThreads * V);
  // worker groups: as few as the staging allows, more when the patterns and
  // stripes alone give under about four blocks per SM
  int J = std::min(m, enc_group_max(DR, ell));
  const long long want = 4LL * device_sm_count();
  const long long have = (long long)npat * stripes;
  if (have < want) {
    const long long groups = (want + have - 1) / have;
    J = (int)std::min<long long>(J, std::max<long long>(std::min(delta, m), (m + groups - 1) / groups));
  }
  const int ngroups = (m + J - 1) / J;
  if (npat > 2147483647 || stripes > 65535 || ngroups > 65535)
    return fail(GC_ERR_UNSUPPORTED, "encode grid too large");
  const size_t smem = enc_smem_bytes(DR, V, ell, delta, J);
  const dim3 grid((unsigned)npat, (unsigned)stripes, (unsigned)ngroups);
  int rc;
  // two blocks of a chunk per step when ell is even
#define GC_ENC(R, VV)                                                                               \
  rc = ell % 2 == 0                                                                                 \
           ? launch_enc_t<R, VV, 2>(grid, smem, E, order, psi, N, m, delta, ell, npat, G, d, L, J, vec, T, s) \
           : launch_enc_t<R, VV, 1>(grid, smem, E, order, psi, N, m, delta, ell, npat, G, d, L, J, vec, T, s)
  switch (DR) {
    case 4: GC_ENC(4, 4); break;
    case 8: GC_ENC(8, 4); break;
    case 16: GC_ENC(16, 4); break;
    default: GC_ENC(32, 2); break;
  }
#undef GC_ENC
  if (rc) return rc;
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

// One live realization in one pass (eq. 2, Sec. II-B, Sec. I).  A block
// takes kLiveCols columns c; its warp w forms T[j][c] for the workers
// j = w, w + kLiveWG, ... (slots p ascending, blocks k ascending, as
// k_encode; the slots past psi_j and the padding past d add zeros there and
// are skipped here, which leaves every sum unchanged) into shared memory;
// then warp 0 forms ghat[k*L + c] = sum_j R[k][j] T[j][c] (j ascending, as
// k_decode_tx) and w[k*L + c] -= scale * ghat[k*L + c] (as k_sgd): the same
// fp32 operations in the same order, so T, ghat and w equal those of the
// three separate calls.  E, R, the order and psi are staged in shared
// memory, and with SG the block's columns of every chunk block too (loaded
// with all the block's loads in flight).
constexpr int kLiveCols = 32, kLiveWG = 8, kLiveThreads = kLiveCols * kLiveWG;
template <int ELL, bool SG>
__global__ void __launch_bounds__(kLiveThreads) k_live_step(const double* __restrict__ E,
                                                  const double* __restrict__ R,
                                                  const int32_t* __restrict__ order,
                                                  const int32_t* __restrict__ psi, int N, int m,
                                                  int delta, const float* __restrict__ G, int d,
                                                  int L, float scale, float* __restrict__ w,
                                                  float* __restrict__ T, float* __restrict__ ghat) {
  extern __shared__ float s_live[];
  const int ne = m * delta * ELL;
  float* s_g = s_live;                                  // [N][ELL][kLiveCols] with SG
  float* s_t = s_g + (SG ? N * ELL * kLiveCols : 0);    // [m][kLiveCols]
  float* s_e = s_t + m * kLiveCols;                     // [m][delta][ELL]
  float* s_r = s_e + ne;                                // [ELL][m]
  int* s_ord = reinterpret_cast<int*>(s_r + ELL * m);   // [m][delta]
  int* s_np = s_ord + m * delta;                        // [m]
  const int cl = threadIdx.x % kLiveCols, wg = threadIdx.x / kLiveCols;
  const int c0 = blockIdx.x * kLiveCols;
  if (SG) {
#pragma unroll 4
    for (int t = threadIdx.x; t < N * ELL * kLiveCols; t += kLiveThreads) {
      const int row = t / kLiveCols, cc = c0 + t % kLiveCols;
      const int i = row / ELL, k = row - i * ELL;
      const long long col = (long long)k * L + cc;
      s_g[t] = (cc < L && col < d) ? __ldg(G + (size_t)i * d + col) : 0.f;
    }
  }
  for (int t = threadIdx.x; t < ne; t += kLiveThreads) s_e[t] = (float)E[t];
  for (int t = threadIdx.x; t < ELL * m; t += kLiveThreads) s_r[t] = (float)R[t];
  for (int t = threadIdx.x; t < m * delta; t += kLiveThreads) s_ord[t] = order[t];
  for (int t = threadIdx.x; t < m; t += kLiveThreads) {
    const int np = psi[t];
    s_np[t] = np < 0 ? 0 : (np > delta ? delta : np);  // as the encode: bad values are flagged by the solve
  }
  __syncthreads();
  const int c = c0 + cl;
  const bool live = c < L;
  for (int j = wg; j < m; j += kLiveWG) {
    float t = 0.f;
    const int np = s_np[j];
    for (int p = 0; p < np; ++p) {
      const int i = s_ord[j * delta + p];
      if (i < 0 || i >= N) continue;
      const float* ej = s_e + (j * delta + p) * ELL;
#pragma unroll
      for (int k = 0; k < ELL; ++k) {
        const long long col = (long long)k * L + c;
        if (live && col < d) {
          const float g = SG ? s_g[(i * ELL + k) * kLiveCols + cl] : __ldg(G + (size_t)i * d + col);
          t = fmaf(ej[k], g, t);
        }
      }
    }
    s_t[j * kLiveCols + cl] = t;
    if (T && live) T[(size_t)j * L + c] = t;
  }
  __syncthreads();
  if (wg != 0 || !live) return;
  float acc[ELL];
#pragma unroll
  for (int k = 0; k < ELL; ++k) acc[k] = 0.f;
  for (int j = 0; j < m; ++j) {
    const float t = s_t[j * kLiveCols + cl];
#pragma unroll
    for (int k = 0; k < ELL; ++k) acc[k] = fmaf(s_r[k * m + j], t, acc[k]);
  }
#pragma unroll
  for (int k = 0; k < ELL; ++k) {
    const long long col = (long long)k * L + c;
    if (col < d) {
      if (ghat) ghat[col] = acc[k];
      w[col] = fmaf(-scale, acc[k], w[col]);
    }
  }
}

constexpr size_t kLiveSmemMax = 96 * 1024;

template <int ELL, bool SG>
static cudaError_t launch_live_t(unsigned blocks, size_t smem, const double* E, const double* R,
                                 const int32_t* order, const int32_t* psi, int N, int m, int delta,
                                 const float* G, int d, int L, float scale, float* w, float* T,
                                 float* ghat, cudaStream_t s) {
  static bool attr = false;
  if (!attr) {
    const cudaError_t e = cudaFuncSetAttribute(k_live_step<ELL, SG>,
                                               cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               (int)kLiveSmemMax);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  k_live_step<ELL, SG><<<blocks, kLiveThreads, smem, s>>>(E, R, order, psi, N, m, delta, G, d, L,
                                                          scale, w, T, ghat);
  return cudaSuccess;
}

int launch_live_step(const double* E, const double* R, int ell, const int32_t* order, int N, int m,
                     int delta, const int32_t* psi, const float* G, int d, float lr, int64_t Ntil,
                     float* w, float* T, float* ghat, cudaStream_t s) {
  const int L = (d + ell - 1) / ell;
  const size_t base = ((size_t)m * delta * ell + (size_t)ell * m + (size_t)m * kLiveCols) * sizeof(float) +
                      ((size_t)m * delta + m) * sizeof(int);
  if (base > kLiveSmemMax)
    return fail(GC_ERR_UNSUPPORTED, "live step: m=%d, delta=%d, ell=%d too large to stage", m,
                delta, ell);
  const size_t gbytes = (size_t)N * ell * kLiveCols * sizeof(float);
  const bool sg = base + gbytes <= kLiveSmemMax;
  const size_t smem = base + (sg ? gbytes : 0);
  const float scale = (float)((double)lr / (double)Ntil);
  const unsigned blocks = (unsigned)((L + kLiveCols - 1) / kLiveCols);
  cudaError_t e = cudaSuccess;
#define GC_LIVE(E_)                                                                              \
  case E_:                                                                                       \
    e = sg ? launch_live_t<E_, true>(blocks, smem, E, R, order, psi, N, m, delta, G, d, L, scale, \
                                     w, T, ghat, s)                                              \
           : launch_live_t<E_, false>(blocks, smem, E, R, order, psi, N, m, delta, G, d, L,      \
                                      scale, w, T, ghat, s);                                     \
    break;
  switch (ell) {
    GC_LIVE(1)
    GC_LIVE(2)
    GC_LIVE(3)
    GC_LIVE(4)
    GC_LIVE(5)
    GC_LIVE(6)
    GC_LIVE(7)
    GC_LIVE(8)
    default: return fail(GC_ERR_UNSUPPORTED, "ell=%d exceeds GC_MAX_ELL", ell);
  }
#undef GC_LIVE
  if (e != cudaSuccess) return cuda_check(e, "cudaFuncSetAttribute(k_live_step)");
  count_launches(1);
  return cuda_check(cudaGetLastError(), "k_live_step");
}

}  // namespace gc
