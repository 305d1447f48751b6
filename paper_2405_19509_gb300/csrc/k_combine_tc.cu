// Batched decode-combine on the 5th-generation tensor cores (tcgen05).
//
//   Ghat (M x L) = C (M x K) . Gv (K x L),  M = npat*ell, K = N*ell, L = ceil(d/ell),
//
// where row (b, k) of C is the decode matrix R B_b restricted to block k
// (Algorithm 1) and row (i, k') of Gv is block k' of g_{D_i} (zero past d).
// This is the PS decode of Sec. II-B applied to the eq. (2) transmissions of
// every straggler pattern at once (R B = [Pi_1 ... Pi_N]).
//
// Precision: the operands are fp32 (C from fp64 projectors, chunk gradients
// in fp32); each is split into bf16 hi + lo parts (x ~= hi + lo with relative
// error 2^-17) and the product is accumulated in fp32 as
//   C_hi G_hi + C_hi G_lo + C_lo G_hi       (the C_lo G_lo term, ~2^-16
// relative, is dropped), i.e. three kind::f16 MMAs per K step.
//
// Kernel structure (persistent, one CTA per SM, 192 threads):
//   warp 0      TMA producer: per k-block one 3-D tensor load for A (hi and
//               lo planes, 128 x 64) and one for B (hi and lo, 256 x 64),
//               128-byte swizzle, into a 2-stage shared-memory ring.
//   warp 1      allocates 512 TMEM columns (two 128 x 256 fp32 accumulators)
//               and one lane issues the MMAs; tcgen05.commit frees smem
//               stages and signals a finished accumulator.
//   warps 2..5  epilogue: tcgen05.ld (32 lanes x 32 columns per load), store
//               to Ghat and/or reduce the squared error to sum_i g_{D_i}
//               per row; the accumulator is handed back as soon as it is
//               read, so the epilogue of tile t overlaps the MMAs of t + 1.
// Tiles are visited n-tile-major so that concurrently running CTAs share the
// same B tile through L2.  When one 64-wide block holds all of K the output
// write bounds the kernel and the B tile is what the copies would mostly
// move, so each CTA keeps its B tile resident over a contiguous range of
// tiles and streams only A (the BRES shape below).
// Every mbarrier wait is bounded; on expiry the
// kernel flags GC_ERR_TIMEOUT in the status word, drains its own copies and
// MMAs (with bounded waits) and frees TMEM.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <string.h>

#include <algorithm>

#include "tc_ptx.cuh"

namespace gc {
namespace tc {

constexpr int BM = 128, BN = 256, BK = 64;
constexpr int A_PLANE = BM * BK * 2;                 // bytes of one bf16 plane (16 KB)
constexpr int B_PLANE = BN * BK * 2;                 // 32 KB
constexpr int STAGE_BYTES = 2 * A_PLANE + 2 * B_PLANE;  // 96 KB
constexpr uint32_t TMEM_COLS = 512;
constexpr long long kSpin = 1LL << 32;  // clock cycles per wait (~2 s)
constexpr int OUT_BUF = 32 * 32 * 4;                 // one 32 x 32 fp32 store box (4 KB)
// Two shapes.  Several 64-wide K blocks (MMA-bound): STAGES = 2 ring stages
// holding A and B, 4 epilogue warps, tiles dealt round-robin.  One K block
// (the output write bounds the kernel; BRES): each CTA takes a contiguous
// n-tile-major range of tiles, keeps the B tile of its current n-tile resident
// (reloaded only when the n-tile changes), streams A through STAGES = 3 ring
// stages, and runs 8 epilogue warps (two per TMEM lane quarter).
constexpr int A_STAGE = 2 * A_PLANE;  // 32 KB
constexpr int kBresStages = 2;        // A ring stages of the BRES shape
constexpr int B_TILE = 2 * B_PLANE;   // 64 KB
// NKBR > 0: B resident (NKBR k-blocks of the current n-tile), A streamed.
// OUT: output staging boxes for TMA stores of Ghat (none in MSE-only shapes).
template <int STAGES, int EPI, int NKBR, bool OUT>
struct Shape {
  static constexpr bool BRES = NKBR > 0;
  static constexpr int THREADS = 64 + 32 * EPI;
  static constexpr int OUT_BYTES = OUT ? EPI * 2 * OUT_BUF : 0;  // 2 staging boxes per epilogue warp
  static constexpr int RING = BRES ? STAGES * A_STAGE + NKBR * B_TILE : STAGES * STAGE_BYTES;
  static constexpr size_t SMEM = (size_t)RING + OUT_BYTES + 1024 + 256;
  static_assert(SMEM <= 232448, "shared memory per CTA");
};

struct Params {
  int M, K, Kp, L, ell, d;
  int num_m_tiles, num_n_tiles, nkb;
  long long num_tiles;
  int vec_ok;           // d % 4 == 0 && L % 4 == 0: 16-byte row segments
  int tma_store;        // Ghat written by TMA tensor stores (needs d == ell * L, L % 4 == 0)
  int evict_first;      // Ghat stores marked evict-first in L2
  float* Ghat;          // npat x d or null
  const float* gsum;    // d, or null when no MSE is wanted
  float* msep;          // M x parts_per_row partial squared errors, or null
  int parts_per_row;    // num_n_tiles * (epilogue warps per TMEM lane quarter)
  long long spin_limit; // clock cycles a wait may take before the kernel gives up
  int stall;            // failure-path test: the TMA producer issues nothing
  // The m-tiles this kernel computes (the others come from the residual
  // decode): dlist[0 .. *ndense) in ascending order, written by the plan scan
  // before the launch; null = every m-tile.
  const int32_t* dlist;
  const int32_t* ndense;
  uint32_t* status;
};

using namespace tcw;

// Descriptor of a K-major operand tile (128-byte swizzle, 8-row groups 1 KB apart).
__device__ __forceinline__ uint64_t sdesc(uint32_t saddr) { return tcw::sdesc(saddr, 16, 1024); }
// Instruction descriptor, kind::f16: D fp32, A and B bf16, both K-major, M = BM, N = BN.
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(BN >> 3) << 17) |
                            ((uint32_t)(BM >> 4) << 24);
__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t accum) {
  tcw::mma_bf16(d_tmem, a, b, kIdesc, accum);
}

template <int STAGES, int EPI, int NKBR, bool OUT>
__global__ void __launch_bounds__(64 + 32 * EPI, 1)
    k_combine_tc(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                 const __grid_constant__ CUtensorMap tmC, Params p) {
  using Sh = Shape<STAGES, EPI, NKBR, OUT>;
  constexpr bool BRES = Sh::BRES;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* bres = smem + STAGES * A_STAGE;                       // BRES: resident B k-blocks
  float* outbuf = reinterpret_cast<float*>(smem + Sh::RING);     // 1024-aligned
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + Sh::RING + Sh::OUT_BYTES);
  uint64_t* empty = full + STAGES;
  uint64_t* tfull = empty + STAGES;   // [2]
  uint64_t* tempty = tfull + 2;       // [2]
  uint64_t* done = tempty + 2;        // MMA drain
  uint64_t* bfull = done + 1;         // BRES: B tile landed
  uint64_t* bempty = bfull + 1;       // BRES: MMAs on the B tile finished
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(bempty + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], EPI);
    }
    mbar_init(done, 1);
    mbar_init(bfull, 1);
    mbar_init(bempty, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tmem_holder)),
                 "r"(TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem_base = *tmem_holder;
  // launched as a programmatic dependent of the operand split: the prologue
  // above overlaps its tail, the operands are read only after this point
  asm volatile("griddepcontrol.wait;" ::: "memory");
  // the tile space: nd listed m-tiles x the n-tiles, n-tile-major;
  // this CTA's tiles are t = t_first, t_first + t_step, ... < t_last
  const int nd = p.ndense ? *reinterpret_cast<volatile const int*>(p.ndense) : p.num_m_tiles;
  const long long ntiles = (long long)nd * p.num_n_tiles;
  long long t_first, t_last, t_step;
  if (BRES) {
    t_first = (long long)blockIdx.x * ntiles / gridDim.x;
    t_last = (long long)(blockIdx.x + 1) * ntiles / gridDim.x;
    t_step = 1;
  } else {
    t_first = blockIdx.x;
    t_last = ntiles;
    t_step = gridDim.x;
  }
  auto tile_mt = [&](long long t) -> int {
    const int mi = (int)(t % nd);
    return p.dlist ? __ldg(p.dlist + mi) : mi;
  };

  if (warp == 0) {
    // ------------------------------------------------------------- producer
    if (lane == 0 && BRES) {
      uint32_t it = 0, nb_loads = 0;
      int cur_nt = -1;
      bool ok = !p.stall;
      for (long long t = t_first; t < t_last && ok; t += t_step) {
        const int nt = (int)(t / nd), mt = tile_mt(t);
        if (nt != cur_nt) {
          // the MMAs on the previous B tile have finished before it is replaced
          if (nb_loads > 0 &&
              !mbar_wait(bempty, (nb_loads - 1) & 1, abort_flag, p.status, p.spin_limit))
            break;
          mbar_expect_tx(bfull, NKBR * B_TILE);
          for (int kb = 0; kb < NKBR; ++kb)
            tma_load_3d(bres + kb * B_TILE, &tmB, kb * BK, nt * BN, 0, bfull);
          cur_nt = nt;
          ++nb_loads;
        }
        for (int kb = 0; kb < NKBR && ok; ++kb, ++it) {
          const int s = it % STAGES;
          const uint32_t ph = (it / STAGES) & 1;
          if (!mbar_wait(&empty[s], ph ^ 1, abort_flag, p.status, p.spin_limit)) {
            ok = false;
            break;
          }
          uint8_t* st = smem + s * A_STAGE;
          mbar_expect_tx(&full[s], A_STAGE);
          tma_load_3d(st, &tmA, kb * BK, mt * BM, 0, &full[s]);
        }
      }
      // drain: every issued copy has landed before the CTA may exit
      volatile int no_abort = 0;
      for (uint32_t k = (it > (uint32_t)STAGES ? it - STAGES : 0); k < it; ++k)
        mbar_wait(&full[k % STAGES], (k / STAGES) & 1, &no_abort, p.status, 1LL << 28);
      if (nb_loads > 0) mbar_wait(bfull, (nb_loads - 1) & 1, &no_abort, p.status, 1LL << 28);
    } else if (lane == 0) {
      uint32_t it = 0;
      bool ok = !p.stall;
      for (long long t = t_first; t < t_last && ok; t += t_step) {
        const int nt = (int)(t / nd), mt = tile_mt(t);
        for (int kb = 0; kb < p.nkb; ++kb, ++it) {
          const int s = it % STAGES;
          const uint32_t ph = (it / STAGES) & 1;
          if (!mbar_wait(&empty[s], ph ^ 1, abort_flag, p.status, p.spin_limit)) {
            ok = false;
            break;
          }
          uint8_t* st = smem + s * STAGE_BYTES;
          mbar_expect_tx(&full[s], STAGE_BYTES);
          tma_load_3d(st, &tmA, kb * BK, mt * BM, 0, &full[s]);
          tma_load_3d(st + 2 * A_PLANE, &tmB, kb * BK, nt * BN, 0, &full[s]);
        }
      }
      // drain: every issued stage has landed before the CTA may exit
      const uint32_t issued = it;
      for (uint32_t k = (issued > (uint32_t)STAGES ? issued - STAGES : 0); k < issued; ++k) {
        volatile int no_abort = 0;
        mbar_wait(&full[k % STAGES], (k / STAGES) & 1, &no_abort, p.status, 1LL << 28);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------- MMA issuer
    if (lane == 0 && BRES) {
      uint32_t it = 0, tile_it = 0, nb_used = 0;
      int cur_nt = -1;
      for (long long t = t_first; t < t_last; t += t_step, ++tile_it) {
        const int nt = (int)(t / nd);
        if (nt != cur_nt) {
          if (!mbar_wait(bfull, nb_used & 1, abort_flag, p.status, p.spin_limit)) break;
          ++nb_used;
          cur_nt = nt;
        }
        const int ab = tile_it & 1;
        if (!mbar_wait(&tempty[ab], ((tile_it >> 1) & 1) ^ 1, abort_flag, p.status, p.spin_limit))
          break;
        const uint32_t d_tmem = tmem_base + (uint32_t)(ab * BN);
        bool ok = true;
        for (int kb = 0; kb < NKBR; ++kb, ++it) {
          const int s = it % STAGES;
          if (!mbar_wait(&full[s], (it / STAGES) & 1, abort_flag, p.status, p.spin_limit)) {
            ok = false;
            break;
          }
          fence_after();
          const uint32_t a_hi = smem_u32(smem + s * A_STAGE), a_lo = a_hi + A_PLANE;
          const uint32_t b_hi = smem_u32(bres + kb * B_TILE), b_lo = b_hi + B_PLANE;
          const int rem = p.K - kb * BK;
          const int nks = rem >= BK ? BK / 16 : (rem + 15) / 16;
          for (int ks = 0; ks < nks; ++ks) {
            const uint32_t off = ks * 32;
            const uint32_t acc = (kb > 0 || ks > 0) ? 1u : 0u;
            mma_bf16(d_tmem, sdesc(a_hi + off), sdesc(b_hi + off), acc);
            mma_bf16(d_tmem, sdesc(a_hi + off), sdesc(b_lo + off), 1u);
            mma_bf16(d_tmem, sdesc(a_lo + off), sdesc(b_hi + off), 1u);
          }
          mma_commit(&empty[s]);
        }
        if (!ok) break;
        mma_commit(&tfull[ab]);
        // last tile on this B tile: hand it back once these MMAs complete
        const bool last_on_b = t + t_step >= t_last || (int)((t + t_step) / nd) != nt;
        if (last_on_b) mma_commit(bempty);
      }
      mma_commit(done);
      volatile int no_abort = 0;
      mbar_wait(done, 0, &no_abort, p.status, 1LL << 28);
    } else if (lane == 0) {
      uint32_t it = 0, tile_it = 0;
      bool ok = true;
      for (long long t = t_first; t < t_last && ok; t += t_step, ++tile_it) {
        const int ab = tile_it & 1;
        if (!mbar_wait(&tempty[ab], ((tile_it >> 1) & 1) ^ 1, abort_flag, p.status, p.spin_limit))
          break;
        fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(ab * BN);
        for (int kb = 0; kb < p.nkb; ++kb, ++it) {
          const int s = it % STAGES;
          const uint32_t ph = (it / STAGES) & 1;
          if (!mbar_wait(&full[s], ph, abort_flag, p.status, p.spin_limit)) {
            ok = false;
            break;
          }
          fence_after();
          const uint32_t a_hi = smem_u32(smem + s * STAGE_BYTES);
          const uint32_t a_lo = a_hi + A_PLANE;
          const uint32_t b_hi = a_hi + 2 * A_PLANE;
          const uint32_t b_lo = b_hi + B_PLANE;
          const int rem = p.K - kb * BK;
          const int nks = rem >= BK ? BK / 16 : (rem + 15) / 16;
          for (int ks = 0; ks < nks; ++ks) {
            const uint32_t off = ks * 32;  // 16 bf16 along K inside the swizzle atom
            const uint32_t acc = (kb > 0 || ks > 0) ? 1u : 0u;
            mma_bf16(d_tmem, sdesc(a_hi + off), sdesc(b_hi + off), acc);
            mma_bf16(d_tmem, sdesc(a_hi + off), sdesc(b_lo + off), 1u);
            mma_bf16(d_tmem, sdesc(a_lo + off), sdesc(b_hi + off), 1u);
          }
          mma_commit(&empty[s]);
        }
        if (!ok) break;
        mma_commit(&tfull[ab]);
      }
      // drain: all issued MMAs have completed
      mma_commit(done);
      volatile int no_abort = 0;
      mbar_wait(done, 0, &no_abort, p.status, 1LL << 28);
    }
  } else {
    // ------------------------------------------------------------- epilogue
    const int quarter = warp & 3;  // TMEM lanes 32*quarter .. +31
    const int e = warp - 2;        // epilogue warp index
    constexpr int SPAN = BN / (EPI / 4);  // columns per epilogue warp
    const int cbeg = (e / 4) * SPAN;
    float* wbuf = outbuf + e * 2 * (OUT_BUF / 4);
    uint32_t tile_it = 0, chunk_it = 0;
    for (long long t = t_first; t < t_last; t += t_step, ++tile_it) {
      const int ab = tile_it & 1;
      const int nt = (int)(t / nd), mt = tile_mt(t);
      // warp-uniform: the TMEM loads below are warp-collective
      const bool ready = mbar_wait(&tfull[ab], (tile_it >> 1) & 1, abort_flag, p.status, p.spin_limit);
      if (!__all_sync(0xffffffffu, ready)) break;
      fence_after();
      const int row = mt * BM + quarter * 32 + lane;
      const bool rv = row < p.M;
      const int b = rv ? row / p.ell : 0;
      const int k = rv ? row - b * p.ell : 0;
      const int n0 = nt * BN;
      float* out = p.Ghat ? p.Ghat + (size_t)b * p.d + (size_t)k * p.L : nullptr;
      const float* gs = p.gsum ? p.gsum + (size_t)k * p.L : nullptr;
      float sq4[4] = {0.f, 0.f, 0.f, 0.f};  // four independent FMA chains
      const uint32_t taddr = tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(ab * BN);
      // the fast path's reference values are loaded one chunk ahead
      const bool fast_gs = gs && p.vec_ok && rv;
      float4 gnext[8];
      if (fast_gs && n0 + cbeg + 32 <= p.L) {
#pragma unroll
        for (int j = 0; j < 8; ++j)
          gnext[j] = __ldg(reinterpret_cast<const float4*>(gs + n0 + cbeg) + j);
      }
#pragma unroll 1
      for (int cc = cbeg; cc < cbeg + SPAN; cc += 32) {
        float v[32];
        float4 gcur[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) gcur[j] = gnext[j];
        if (fast_gs && cc + 32 < cbeg + SPAN && n0 + cc + 64 <= p.L) {
#pragma unroll
          for (int j = 0; j < 8; ++j)
            gnext[j] = __ldg(reinterpret_cast<const float4*>(gs + n0 + cc + 32) + j);
        }
        __syncwarp();
        tmem_ld32(taddr + cc, v);  // warp-collective: every lane, every chunk
        const int c0 = n0 + cc;
        if (OUT && p.tma_store && c0 < p.L) {
          // stage the 32 x 32 box (row = lane) with the 128-byte swizzle, then one TMA store
          float* buf = wbuf + (chunk_it & 1) * (OUT_BUF / 4);
          if (lane == 0) bulk_wait_read1();  // the store that used this buffer has read it
          __syncwarp();
          char* rowp = reinterpret_cast<char*>(buf) + lane * 128;
#pragma unroll
          for (int j = 0; j < 8; ++j)
            *reinterpret_cast<float4*>(rowp + ((j ^ (lane & 7)) << 4)) =
                make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
          asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
          __syncwarp();
          if (lane == 0) {
            if (p.evict_first)
              tma_store_2d_hint(&tmC, buf, c0, mt * BM + quarter * 32, policy_evict_first());
            else
              tma_store_2d(&tmC, buf, c0, mt * BM + quarter * 32);
            bulk_commit();
          }
          ++chunk_it;
        }
        const int lim = (rv && c0 < p.L) ? min(32, min(p.L - c0, p.d - k * p.L - c0)) : 0;
        if (lim <= 0) {
        } else if (lim == 32 && p.vec_ok) {
          if (out && !p.tma_store) {
            float4* o4 = reinterpret_cast<float4*>(out + c0);
#pragma unroll
            for (int j = 0; j < 8; ++j)
              o4[j] = make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
          }
          if (gs) {
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              const float4 g = gcur[j];
              float df = v[4 * j] - g.x;
              sq4[0] = fmaf(df, df, sq4[0]);
              df = v[4 * j + 1] - g.y;
              sq4[1] = fmaf(df, df, sq4[1]);
              df = v[4 * j + 2] - g.z;
              sq4[2] = fmaf(df, df, sq4[2]);
              df = v[4 * j + 3] - g.w;
              sq4[3] = fmaf(df, df, sq4[3]);
            }
          }
        } else {
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            if (j < lim) {
              if (out && !p.tma_store) out[c0 + j] = v[j];
              if (gs) {
                const float df = v[j] - __ldg(gs + c0 + j);
                sq4[j & 3] = fmaf(df, df, sq4[j & 3]);
              }
            }
          }
        }
      }
      fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[ab]);
      if (p.msep && rv)
        p.msep[(size_t)row * p.parts_per_row + nt * (EPI / 4) + e / 4] = (sq4[0] + sq4[1]) + (sq4[2] + sq4[3]);
    }
    if (lane == 0) bulk_wait_all();  // every store of this warp has completed
  }
  fence_before();
  __syncthreads();
  // every role is done: the MSE reduction may be scheduled (it waits for
  // this grid to finish); earlier, its waiting blocks would hold SM room
  if (threadIdx.x == 0) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  if (warp == 1) {
    fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base),
                 "r"(TMEM_COLS)
                 : "memory");
  }
}

// C (M x K fp32) -> planes [2][M][Kp] bf16: hi = bf16(c), lo = bf16(c - hi); zero pad.
__global__ void k_split_c(const float* __restrict__ C, int M, int K, int Kp,
                          __nv_bfloat16* __restrict__ out) {
  const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  const long long tot = (long long)M * Kp;
  if (idx >= tot) return;
  const int row = (int)(idx / Kp), kk = (int)(idx - (long long)row * Kp);
  const float v = kk < K ? __ldg(C + (size_t)row * K + kk) : 0.f;
  const __nv_bfloat16 hi = __float2bfloat16_rn(v);
  const __nv_bfloat16 lo = __float2bfloat16_rn(v - __bfloat162float(hi));
  out[idx] = hi;
  out[tot + idx] = lo;
}

// G (N x d fp32) -> planes [2][L][Kp] bf16 of Gv^T: element (c, i*ell + k') =
// g_{D_i}[k'*L + c] (zero past d and for padding columns).  Block (x, y)
// transposes the tile of 32 K-rows (kk = 32 y ..) by COLS columns
// (c = COLS x ..) through shared memory: 16-byte loads along c, 16-byte
// stores along kk (COLS = 128 for long rows, 32 when L is short and more
// blocks are wanted).  Blocks stride over the (column tile, K tile) pairs;
// nothing is done when *ndense is zero: no row tile of the batch is on the
// GEMM.
template <int COLS>
__global__ void __launch_bounds__(256) k_split_gt(const float* __restrict__ G, int N, int d,
                                                  int ell, int L, int Kp,
                                                  __nv_bfloat16* __restrict__ out,
                                                  const int32_t* __restrict__ ndense) {
  constexpr int kSplitCols = COLS;
  constexpr int TPR = COLS / 4;            // threads per row of the load phase
  constexpr int RPP = 256 / TPR;           // rows per pass
  // the combine kernel may be scheduled now; it waits for this grid to finish
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  if (ndense && __ldg(ndense) == 0) return;
  __shared__ float tile[32][kSplitCols + 1];
  const int ncx = (L + kSplitCols - 1) / kSplitCols;
  const long long npair = (long long)ncx * (Kp / 32);
  for (long long pr = blockIdx.x; pr < npair; pr += gridDim.x) {
  __syncthreads();  // the previous pair's tile has been read
  const int c0 = (int)(pr % ncx) * kSplitCols, k0 = (int)(pr / ncx) * 32;
  const int t = threadIdx.x;
  const int K = N * ell;
  const bool vec = (L % 4 == 0) && (d % 4 == 0) && (reinterpret_cast<uintptr_t>(G) % 16 == 0);
  // load: thread t takes columns 4 (t % TPR) .. +3 of rows t / TPR + RPP r
#pragma unroll
  for (int r = 0; r < 32 / RPP; ++r) {
    const int kr = t / TPR + RPP * r, kk = k0 + kr;
    const int cc = 4 * (t % TPR), c = c0 + cc;
    float v[4] = {0.f, 0.f, 0.f, 0.f};
    if (kk < K) {
      const int i = kk / ell, kp = kk - i * ell;
      const float* src = G + (size_t)i * d + (size_t)kp * L + c;
      if (vec && c + 3 < L && kp * L + c + 3 < d) {
        const float4 q = __ldg(reinterpret_cast<const float4*>(src));
        v[0] = q.x; v[1] = q.y; v[2] = q.z; v[3] = q.w;
      } else {
#pragma unroll
        for (int e = 0; e < 4; ++e)
          if (c + e < L && kp * L + c + e < d) v[e] = __ldg(src + e);
      }
    }
#pragma unroll
    for (int e = 0; e < 4; ++e) tile[kr][cc + e] = v[e];
  }
  __syncthreads();
  // store: thread t takes column t % COLS and K-rows 16 (t / COLS) .. +15
  if (t < 2 * kSplitCols) {
    const int cc = t % kSplitCols, h = t / kSplitCols, c = c0 + cc;
    if (c < L) {
      uint32_t hw[8], lw[8];
#pragma unroll
      for (int e = 0; e < 16; e += 2) {
        const float a = tile[16 * h + e][cc], b = tile[16 * h + e + 1][cc];
        const __nv_bfloat16 ha = __float2bfloat16_rn(a), hb = __float2bfloat16_rn(b);
        const __nv_bfloat16 la = __float2bfloat16_rn(a - __bfloat162float(ha));
        const __nv_bfloat16 lb = __float2bfloat16_rn(b - __bfloat162float(hb));
        hw[e / 2] = (uint32_t)__bfloat16_as_ushort(ha) | ((uint32_t)__bfloat16_as_ushort(hb) << 16);
        lw[e / 2] = (uint32_t)__bfloat16_as_ushort(la) | ((uint32_t)__bfloat16_as_ushort(lb) << 16);
      }
      const int kk = k0 + 16 * h;
      if (kk < Kp) {  // Kp is a multiple of 64, so the 16 entries are all inside
        const size_t plane = (size_t)L * Kp;
        uint4* dh = reinterpret_cast<uint4*>(out + (size_t)c * Kp + kk);
        uint4* dl = reinterpret_cast<uint4*>(out + plane + (size_t)c * Kp + kk);
        dh[0] = make_uint4(hw[0], hw[1], hw[2], hw[3]);
        dh[1] = make_uint4(hw[4], hw[5], hw[6], hw[7]);
        dl[0] = make_uint4(lw[0], lw[1], lw[2], lw[3]);
        dl[1] = make_uint4(lw[4], lw[5], lw[6], lw[7]);
      }
    }
  }
  }
}

// grad_mse[b] = (sum over the rows b*ell .. b*ell+ell-1 of their partial
// squared errors) / d: one warp per pattern; a row of a GEMM tile sums the
// combine's partials, a row of a residual tile the residual kernel's (none
// for a pattern whose blocks are all I_ell: its error is exactly zero).
// Lanes stride over a row's partials, then a fixed xor tree; rows are added
// in order (fp32 partial sums, the result scaled in fp64).  Launched as a
// programmatic dependent of the combine kernel.
__global__ void k_mse_reduce_tiles(const float* __restrict__ msep, int parts,
                                   const float* __restrict__ msp, int parts_r,
                                   const int32_t* __restrict__ tflag, const int32_t* __restrict__ rslot,
                                   int npat, int ell, double inv_d, double* __restrict__ grad_mse) {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const long long b = ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (b >= npat) return;
  float tot = 0.f;
  for (int k = 0; k < ell; ++k) {
    const long long row = b * ell + k;
    const float* r = nullptr;
    int n = 0;
    if (__ldg(tflag + (row >> 7))) {
      r = msep + (size_t)row * parts;
      n = parts;
    } else {
      const int slot = __ldg(rslot + row);
      if (slot >= 0) {
        r = msp + (size_t)slot * parts_r;
        n = parts_r;
      }
    }
    float s = 0.f;
    if (n % 4 == 0 && (reinterpret_cast<uintptr_t>(r) & 15) == 0) {
      // 16-byte loads, four in flight a lane (a row has up to a few thousand partials)
      const float4* r4 = reinterpret_cast<const float4*>(r);
      const int n4 = n / 4;
      float4 a[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) a[u] = make_float4(0.f, 0.f, 0.f, 0.f);
      int t = lane;
      for (; t + 96 < n4; t += 128) {
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const float4 x = __ldg(r4 + t + 32 * u);
          a[u].x += x.x;
          a[u].y += x.y;
          a[u].z += x.z;
          a[u].w += x.w;
        }
      }
      for (; t < n4; t += 32) {
        const float4 x = __ldg(r4 + t);
        a[0].x += x.x;
        a[0].y += x.y;
        a[0].z += x.z;
        a[0].w += x.w;
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) s += (a[u].x + a[u].y) + (a[u].z + a[u].w);
    } else {
      for (int t = lane; t < n; t += 32) s += __ldg(r + t);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    tot += s;
  }
  if (lane == 0) grad_mse[b] = (double)tot * inv_d;
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  }
  return fn;
}

// 2-D fp32 map over Ghat viewed as (npat*ell) rows of L (requires d == ell*L),
// box 32 x 32, 128-byte swizzle (matches the epilogue's staging layout).
int make_out_map(CUtensorMap* map, float* base, long long rows, int L) {
  auto fn = encode_fn();
  if (!fn) return fail(GC_ERR_CUDA, "cuTensorMapEncodeTiled entry point unavailable");
  cuuint64_t dims[2] = {(cuuint64_t)L, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)L * 4};
  cuuint32_t box[2] = {32, 32};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, base, dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(GC_ERR_CUDA, "cuTensorMapEncodeTiled(out) failed (%d)", (int)r);
  return GC_OK;
}

// 3-D map over [2][rows][Kp] bf16 planes, box {64, box_rows, 2}, 128-byte swizzle.
int make_map(CUtensorMap* map, const void* base, int rows, int Kp, int box_rows) {
  auto fn = encode_fn();
  if (!fn) return fail(GC_ERR_CUDA, "cuTensorMapEncodeTiled entry point unavailable");
  cuuint64_t dims[3] = {(cuuint64_t)Kp, (cuuint64_t)rows, 2};
  cuuint64_t strides[2] = {(cuuint64_t)Kp * 2, (cuuint64_t)rows * Kp * 2};
  cuuint32_t box[3] = {(cuuint32_t)BK, (cuuint32_t)box_rows, 2};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(GC_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", (int)r);
  return GC_OK;
}

}  // namespace tc

template <int STAGES, int EPI, int NKBR, bool OUT>
int launch_tc(int grid, const CUtensorMap& mA, const CUtensorMap& mB, const CUtensorMap& mC,
              const tc::Params& p, cudaStream_t s) {
  using Sh = tc::Shape<STAGES, EPI, NKBR, OUT>;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(tc::k_combine_tc<STAGES, EPI, NKBR, OUT>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Sh::SMEM);
    if (e != cudaSuccess) return cuda_check(e, "cudaFuncSetAttribute(k_combine_tc)");
    attr_set = true;
  }
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(Sh::THREADS);
  cfg.dynamicSmemBytes = Sh::SMEM;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t e = cudaLaunchKernelEx(&cfg, tc::k_combine_tc<STAGES, EPI, NKBR, OUT>, mA, mB, mC, p);
  if (e != cudaSuccess) return cuda_check(e, "cudaLaunchKernelEx(k_combine_tc)");
  count_launches(1);
  return cuda_check(cudaGetLastError(), "k_combine_tc");
}

size_t apply_ws_bytes(int N, int ell, int npat, int d) {
  const int L = (d + ell - 1) / ell;
  const long long M = (long long)npat * ell;
  const int Kp = combine_kp(N, ell);
  const int nnt = (L + tc::BN - 1) / tc::BN;
  return std::max(align_up((size_t)2 * L * Kp * 2, 256) + align_up((size_t)d * sizeof(float), 256) +
                      align_up((size_t)M * nnt * 2 * sizeof(float), 256) +
                      resid_ws_bytes(N, ell, npat, d),
                  mse_gram_ws_bytes(N, ell, d));
}

int launch_split_c(const float* C, int N, int ell, int npat, __nv_bfloat16* Cs, cudaStream_t s) {
  const long long M = (long long)npat * ell;
  const int K = N * ell, Kp = combine_kp(N, ell);
  const long long tot = M * Kp;
  if (tot == 0) return GC_OK;
  tc::k_split_c<<<(unsigned)((tot + 255) / 256), 256, 0, s>>>(C, (int)M, K, Kp, Cs);
  count_launches(1);
  return cuda_check(cudaGetLastError(), "k_split_c");
}

// The decode of a batch: the plan scan picks the path of every 128-row tile
// (k_decode_resid.cu); residual tiles are written by the residual kernel, the
// others by the tensor-core GEMM (whose operand split runs only when some
// tile needs it), then the per-pattern errors are reduced.
int launch_apply(const __nv_bfloat16* Cs, const float* G, int N, int ell, int npat, int d,
                 float* Ghat, double* grad_mse, Carve& ws, uint32_t* status, cudaStream_t s) {
  using namespace tc;
  const int L = (d + ell - 1) / ell;
  const long long M = (long long)npat * ell;
  const int K = N * ell;
  const int Kp = combine_kp(N, ell);  // every TMA row is one aligned 128-byte line
  if (M > (1LL << 31) - 1) return fail(GC_ERR_UNSUPPORTED, "npat*ell too large");
  const int policy = decode_policy();
  // errors only, and enough patterns to amortise one Gram matrix of the
  // chunk blocks: each pattern's MSE is a quadratic form in it
  if (!Ghat && grad_mse && policy == GC_DECODE_AUTO && mse_gram_applies(N, ell, npat))
    return launch_mse_gram(Cs, Kp, G, N, ell, npat, d, grad_mse, ws, s);
  const int nmt = (int)((M + BM - 1) / BM), nnt = (L + BN - 1) / BN;
  __nv_bfloat16* Gs = ws.take<__nv_bfloat16>((size_t)2 * L * Kp);
  float* gsum = ws.take<float>((size_t)d);
  float* msep_mem = ws.take<float>((size_t)M * nnt * 2);
  float* msep = grad_mse ? msep_mem : nullptr;
  const ResidLists rl = carve_resid(ws, N, ell, npat, d, grad_mse != nullptr);
  // a residual tile may spend up to Kp / 64 corrections per pattern: about
  // what the three MMAs per 64-wide K block cost against reading the ell
  // blocks of one chunk gradient
  const int budget = std::max(1, Kp / 64);
  // header word 4: completion counter of the plan scan (zeroed with the header)
  unsigned int* counter = reinterpret_cast<unsigned int*>(status) + 4;
  int rc = launch_plan_scan(Cs, Kp, N, ell, npat, budget, policy, rl, counter, s);
  if (rc) return rc;
  // s = sum_i g_{D_i}: the residual rows start from it, the GEMM's MSE uses it
  rc = launch_gsum(G, N, d, gsum, s);
  if (rc) return rc;
  if (policy != GC_DECODE_DENSE) {
    rc = launch_decode_resid(G, gsum, rl, ell, npat, d, Ghat, s);
    if (rc) return rc;
  }
  {
    // a grid of a few blocks per SM striding over the tiles: it costs little
    // to launch when no row tile is on the GEMM
    const int cols = L >= 16384 ? 128 : 32;
    const long long pairs = (long long)((L + cols - 1) / cols) * (Kp / 32);
    const unsigned blocks = (unsigned)std::min<long long>(pairs, 8LL * device_sm_count());
    if (cols == 128)
      k_split_gt<128><<<blocks, 256, 0, s>>>(G, N, d, ell, L, Kp, Gs, rl.ndense);
    else
      k_split_gt<32><<<blocks, 256, 0, s>>>(G, N, d, ell, L, Kp, Gs, rl.ndense);
    count_launches(1);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_check(e, "k_split_gt");
  }
  CUtensorMap mA, mB, mC;
  rc = make_map(&mA, Cs, (int)M, Kp, BM);
  if (rc) return rc;
  rc = make_map(&mB, Gs, L, Kp, BN);
  if (rc) return rc;
  const bool tma_store = Ghat && (long long)ell * L == d && L % 4 == 0 &&
                         reinterpret_cast<uintptr_t>(Ghat) % 16 == 0;
  memset(&mC, 0, sizeof(mC));
  if (tma_store) {
    rc = make_out_map(&mC, Ghat, M, L);
    if (rc) return rc;
  }
  Params p{};
  p.M = (int)M;
  p.K = K;
  p.Kp = Kp;
  p.L = L;
  p.ell = ell;
  p.d = d;
  p.num_m_tiles = nmt;
  p.num_n_tiles = nnt;
  p.nkb = (Kp + BK - 1) / BK;
  p.num_tiles = (long long)nmt * nnt;
  p.vec_ok = (d % 4 == 0) && (L % 4 == 0);
  p.tma_store = tma_store ? 1 : 0;
  // Ghat is written once and not read back by this kernel: its lines go
  // first when L2 needs room (measured ~1% per logistic step)
  p.evict_first = 1;
  p.Ghat = Ghat;
  p.gsum = grad_mse ? gsum : nullptr;
  p.msep = msep;
  p.dlist = rl.dlist;
  p.ndense = rl.ndense;
  p.status = status;
  p.spin_limit = wait_limit(kSpin);
  p.stall = take_stall(GC_STALL_COMBINE) ? 1 : 0;
  // shapes: one K block -> B resident, A streamed, output staged (write-bound);
  // two K blocks and no output (the MSE sweep) -> B resident over a 3-stage
  // A ring, so the next A tiles load while the MMAs run; else the 2-stage
  // ring of A and B tiles
  const bool one_block = p.nkb == 1;
  const bool two_res = p.nkb == 2 && !Ghat;
  p.parts_per_row = nnt * ((one_block || two_res) ? 2 : 1);
  const int sms = device_sm_count();
  const int grid = (int)std::min<long long>(p.num_tiles, sms);
  rc = one_block ? launch_tc<kBresStages, 8, 1, true>(grid, mA, mB, mC, p, s)
       : two_res ? launch_tc<3, 8, 2, false>(grid, mA, mB, mC, p, s)
                 : launch_tc<2, 4, 0, true>(grid, mA, mB, mC, p, s);
  if (rc) return rc;
  if (grad_mse) {
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3((unsigned)(((long long)npat * 32 + 255) / 256));
    cfg.blockDim = dim3(256);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cudaError_t e = cudaLaunchKernelEx(&cfg, k_mse_reduce_tiles, (const float*)msep, p.parts_per_row,
                                       (const float*)rl.msp, rl.parts, (const int32_t*)rl.tflag,
                                       (const int32_t*)rl.rslot, npat, ell, 1.0 / (double)d, grad_mse);
    if (e != cudaSuccess) return cuda_check(e, "cudaLaunchKernelEx(k_mse_reduce_tiles)");
    count_launches(1);
  }
  return GC_OK;
}

}  // namespace gc
