// Sec. 4.3, last paragraph: every pruned visual token joins its cosine-nearest
// kept token. The pruned x kept Gram fused with the row argmax, on pairs of SMs
// (tcgen05 cta_group::2).
//
// The operands are contiguous rows of the per-sample copy of E_v permuted to
// [pruned | kept] (gather_perm_kernel). A unit of work is a tile (sample b,
// 512-row group q of its pruned positions, range t of its kept positions):
// the group's rows as two M = 256 halves (A0 = the first 256, A1 = the next
// 256) against the range's kept rows c0 .. c0+N-1 (N <= 256). The two CTAs of
// a cluster issue, from the even CTA, one M = 256 MMA per half and K step;
// CTA r (0 or 1) holds rows 128r .. 128r+127 of each half and kept rows
// c0 + r*N/2 .. c0 + r*N/2 + N/2 - 1 of B, and receives rows 128r .. 128r+127
// of both accumulators in its own tensor memory (columns 0 .. N-1 for A0,
// 256 .. 256+N-1 for A1). Each SM thus loads 48 KiB (its A rows and half of
// B) per 64-element K slice of a 256-column tile, against 64 KiB when one SM
// runs both M = 128 halves against all of B, and its MMAs read its half of B
// once for both SMs.
//
// A group splits its kept columns into n_lo or n_lo + 1 ranges (see
// pair_tile); the tiles are dealt to the clusters in snake order (see
// pair_deal_tile), so that the busiest pair of SMs gets as little work as the
// ranges allow, and the tiles of one group run side by side on different pairs
// and share its A rows through L2. Each CTA loads only the N/2 kept rows its
// half of the MMA reads (one tensor map per distinct N/2 of the plan).
//
// The epilogue (eight warps: two per TMEM lane quadrant, each taking half of
// the 32-column pieces, their tensor-memory loads double-buffered) scales
// column k by 1/|e_k| and keeps per row the running (max, first index) over
// its columns in ascending kept position; range t of a row writes slot t of
// the partials, which merge_assign_kernel combines (ties to the lower kept
// position).
//
// Every wait is bounded; a CTA that times out marks itself failed, and both
// CTAs drain to the closing cluster barrier, after which each frees its half
// of the pair's tensor memory. Before that barrier each producer waits for the
// MMAs' releases of its last stages and the MMA issuer for both epilogues'
// release of the last tile, so that no arrival lands in a CTA that has exited.
#include "common.cuh"
#include "kernels.h"
#include "merge_epi.cuh"
#include "tc_gemm.cuh"

#include <math.h>

#include <mutex>
#include <vector>

namespace provip {
namespace {

using namespace tcg;

constexpr int kPairQuadRows = 4 * kBM;             // pruned rows of a quad (two M = 256 halves)
constexpr int kPairMaxN = 256;                     // columns of a tile
constexpr int kPairStages = 4;
constexpr int kPairStageBytes = 3 * kABytes;       // A0 rows | A1 rows | B rows of this CTA: 48 KiB
constexpr uint32_t kPairTmemCols = 2 * kPairMaxN;  // one accumulator per half
constexpr int kPairEpiWarps = 8;                   // two per TMEM lane quadrant, splitting the columns
constexpr int kPairThreads = 64 + 32 * kPairEpiWarps;

struct PairArgs {
  const int* pruned;    // [B][n_pruned] original row of each pruned position
  int n_pruned;
  const int* keep_idx;  // [B][keep]
  int keep;
  int N_v, D, B;
  const float* inv_v;   // [B][N_v]
  MergePairPlan plan;   // tiles and their deal to the pairs
  float* ws_best;       // [plan.n_slots][B][N_v]
  int* ws_bidx;
  unsigned* err;
};

// tensor maps of the permuted copy: A boxes of 128 rows, B boxes of each
// distinct half-width of the plan's tiles (so that a CTA loads only the N/2
// kept rows its half of the MMA reads)
struct PairMaps {
  CUtensorMap a;
  CUtensorMap b[kMergePairHeights];
};

struct PairPipe {
  uint64_t full[kPairStages];   // even CTA: both CTAs' boxes of the stage have landed
  uint64_t empty[kPairStages];  // each CTA: the MMAs that read its stage are done
  uint64_t acc_full;            // each CTA: the tile's accumulators are complete
  uint64_t acc_empty;           // even CTA: both CTAs' epilogues have read them
  uint32_t tmem;
  volatile int fail;
};

__device__ __forceinline__ uint32_t pair_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// shared::cluster address of `local`'s counterpart in cluster CTA `rank`
__device__ __forceinline__ uint32_t cluster_addr(const void* local, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_u32(local)), "r"(rank));
  return r;
}
__device__ __forceinline__ void pair_cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\t"
               "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// tensor memory of the CTA pair: one warp of each CTA takes part
__device__ __forceinline__ void tmem_alloc_pair(uint32_t* smem_result, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(smem_result)),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish_pair() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
// D (+)= A * B^T over the CTA pair: M = 256 (128 rows of A and N/2 rows of B
// from each CTA's shared memory at the same offsets), bf16 in, fp32 out.
__device__ __forceinline__ void mma_pair_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                              uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// arrive on the mbarrier at `bar`'s offset in both CTAs of the pair once every
// MMA issued so far by this thread has completed
__device__ __forceinline__ void commit_pair(uint64_t* bar) {
  const uint16_t both = 0x3;
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 "
      "[%0], %1;" ::"r"(smem_u32(bar)),
      "h"(both)
      : "memory");
}
// 2-D tiled load into this CTA's shared memory whose completion is counted on
// an mbarrier of either CTA of the pair (bar: shared::cluster address)
__device__ __forceinline__ void tma_load_2d_pair(void* smem_dst, const CUtensorMap* map, int x, int y,
                                                 uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.tile.mbarrier::complete_tx::bytes "
      "[%0], [%1, {%2, %3}], [%4];" ::"r"(smem_u32(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t bar) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait_cluster(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// bounded wait on a barrier that the other CTA of the pair also signals
__device__ __forceinline__ bool mbar_wait_cluster(uint64_t* bar, uint32_t parity, unsigned* err) {
  if (mbar_try_wait_cluster(bar, parity)) return true;
  const unsigned long long t0 = global_timer_ns();
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait_cluster(bar, parity)) return true;
    if ((it & 63u) == 0 && global_timer_ns() - t0 > kWaitBudgetNs) {
      set_error(err, kErrTimeout);
      return false;
    }
  }
}

// every epilogue thread passes its predicate; all get the AND (a barrier of
// the epilogue warps)
__device__ __forceinline__ bool epilogue_all(bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred q, p;\n\t"
      "setp.ne.u32 q, %1, 0;\n\t"
      "bar.red.and.pred p, 1, %2, q;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(r)
      : "r"(v ? 1u : 0u), "n"(32 * kPairEpiWarps)
      : "memory");
  return r != 0;
}
__device__ __forceinline__ void epilogue_sync() {
  asm volatile("bar.sync 1, %0;" ::"n"(32 * kPairEpiWarps) : "memory");
}
// Tile k of the plan. Quads are numbered b * n_quads + q; quads x_hi .. Q-1
// split their kept columns into n_lo ranges and come first (tiles 0 ..
// (Q - x_hi) * n_lo - 1, the wider ones), quads 0 .. x_hi-1 into n_lo + 1.
// Range t of n starts at t * keep / n rounded down to a multiple of 32.
struct PairTile {
  int b, m0, t, n, c0, nv, N;
  bool has1;
};
__host__ __device__ __forceinline__ int pair_range_start(int t, int n, int keep) {
  return t == 0 ? 0 : (t >= n ? keep : (int)((long long)t * keep / n) & ~31);
}
__host__ __device__ __forceinline__ PairTile pair_tile(const MergePairPlan& p, int n_pruned, int keep, int k) {
  PairTile g;
  const int n_wide = (p.Q - p.x_hi) * p.n_lo;
  int quad;
  if (k < n_wide) {
    g.n = p.n_lo;
    quad = p.x_hi + k / p.n_lo;
    g.t = k % p.n_lo;
  } else {
    g.n = p.n_lo + 1;
    quad = (k - n_wide) / g.n;
    g.t = (k - n_wide) % g.n;
  }
  g.b = quad / p.n_quads;
  g.m0 = (quad % p.n_quads) * kPairQuadRows;
  g.has1 = g.m0 + 2 * kBM < n_pruned;  // the second half holds pruned rows
  g.c0 = pair_range_start(g.t, g.n, keep);
  g.nv = pair_range_start(g.t + 1, g.n, keep) - g.c0;
  g.N = (g.nv + 31) / 32 * 32;         // MMA width: N / 2 rows of B per CTA, a multiple of 16
  return g;
}
// Tile of pair p in deal r (snake order: pairs 0 .. P-1 take tiles r*P ..
// in deals 0, 2, ..., and in reverse order in deals 1, 3, ..., so that a
// pair given one of the first, wider tiles gets one of the last, narrower ones);
// -1 past the last tile.
__host__ __device__ __forceinline__ int pair_deal_tile(const MergePairPlan& p, int pair, int r) {
  const int k = (r & 1) ? (r + 1) * p.P - 1 - pair : r * p.P + pair;
  return k < p.T ? k : -1;
}

__global__ void __launch_bounds__(kPairThreads, 1)
    merge_argmax_pair_tc(const PairArgs a, const __grid_constant__ PairMaps maps) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ PairPipe pipe;
  __shared__ int sidx[2 * kBM];      // original rows of this CTA's A0 and A1 rows (-1: none)
  __shared__ float skinv[kPairMaxN];  // 1/|e_k| of the tile's kept columns
  __shared__ float xbest[2][kBM];     // the upper column half's (max, position) per row
  __shared__ int xidx[2][kBM];
  const uint32_t rank = pair_rank();  // 0: issues the MMAs; 1: its peer
  const int pair = (int)(blockIdx.x >> 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_k = (a.D + kBK - 1) / kBK;
  const MergePairPlan& pl = a.plan;

  const uint32_t sbase = smem_u32(smem_raw);
  uint8_t* stages = smem_raw + (((sbase + 1023u) & ~1023u) - sbase);

  if (threadIdx.x == 0) {
    prefetch_tmap(&maps.a);
    for (int j = 0; j < pl.n_heights; ++j) prefetch_tmap(&maps.b[j]);
    for (int s = 0; s < kPairStages; ++s) {
      mbar_init(&pipe.full[s], 1);
      mbar_init(&pipe.empty[s], 1);
    }
    mbar_init(&pipe.acc_full, 1);
    mbar_init(&pipe.acc_empty, 2 * kPairEpiWarps);  // one arrival per epilogue warp of each CTA
    pipe.fail = 0;
    fence_mbar_init();
  }
  if (warp == 0) {
    tmem_alloc_pair(&pipe.tmem, kPairTmemCols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  pair_cluster_sync();  // both CTAs' barriers initialised, the pair's tensor memory allocated
  tc_fence_after();
  // launched as a programmatic dependent of the gather: the set-up above ran
  // under its tail; the permuted copy and the index tables are read after this
  pdl_wait_prior();
  pdl_allow_next();

  if (warp == 0) {
    if (lane == 0) {
      // both CTAs load their rows of every stage; completion counts on the
      // even CTA's full barrier, which expects the bytes of both
      int it = 0;
      for (int rd = 0, k; (k = pair_deal_tile(pl, pair, rd)) >= 0 && !pipe.fail; ++rd) {
        const PairTile g = pair_tile(pl, a.n_pruned, a.keep, k);
        const int row_a = g.b * a.N_v + g.m0 + (int)rank * kBM;
        const int row_b = g.b * a.N_v + a.n_pruned + g.c0 + (int)rank * (g.N / 2);
        int hj = 0, hrows = pl.heights[0];  // the B map whose box height is N / 2
#pragma unroll
        for (int j = 1; j < kMergePairHeights; ++j)
          if (j < pl.n_heights && pl.heights[j] == g.N / 2) {
            hj = j;
            hrows = pl.heights[j];
          }
        const CUtensorMap* mapB = maps.b + hj;
        const uint32_t tx = 2u * (uint32_t)((g.has1 ? 2 : 1) * kABytes + hrows * kBK * 2);
        for (int kb = 0; kb < n_k; ++kb, ++it) {
          const int s = it % kPairStages;
          const uint32_t ph = (uint32_t)(it / kPairStages) & 1u;
          if (pipe.fail || !mbar_wait(&pipe.empty[s], ph ^ 1u, a.err)) {
            pipe.fail = 1;
            break;
          }
          uint8_t* sa = stages + (size_t)s * kPairStageBytes;
          const uint32_t fb = cluster_addr(&pipe.full[s], 0);
          const int x = kb * kBK;
          if (rank == 0) mbar_arrive_expect_tx(&pipe.full[s], tx);
          tma_load_2d_pair(sa, &maps.a, x, row_a, fb);
          if (g.has1) tma_load_2d_pair(sa + kABytes, &maps.a, x, row_a + 2 * kBM, fb);
          tma_load_2d_pair(sa + 2 * kABytes, mapB, x, row_b, fb);
        }
      }
      // the MMAs' releases of the last stages land in this CTA before it may exit
      for (int i = it; i < it + kPairStages && !pipe.fail; ++i)
        if (!mbar_wait(&pipe.empty[i % kPairStages], ((uint32_t)(i / kPairStages) & 1u) ^ 1u, a.err)) pipe.fail = 1;
    }
  } else if (warp == 1) {
    if (rank == 0 && lane == 0) {
      int it = 0, ti = 0;
      for (int rd = 0, k; (k = pair_deal_tile(pl, pair, rd)) >= 0; ++rd, ++ti) {
        const PairTile g = pair_tile(pl, a.n_pruned, a.keep, k);
        // both epilogues have read the previous tile's accumulators
        if (!pipe.fail && !mbar_wait_cluster(&pipe.acc_empty, ((uint32_t)ti & 1u) ^ 1u, a.err)) pipe.fail = 1;
        tc_fence_after();
        const uint32_t idesc = idesc_bf16_f32(2 * kBM, g.N);
        for (int kb = 0; kb < n_k; ++kb, ++it) {
          const int s = it % kPairStages;
          const uint32_t ph = (uint32_t)(it / kPairStages) & 1u;
          if (pipe.fail || !mbar_wait_cluster(&pipe.full[s], ph, a.err)) {
            pipe.fail = 1;
            break;
          }
          tc_fence_after();
          const uint32_t sa = smem_u32(stages + (size_t)s * kPairStageBytes);
          const uint32_t sb = sa + 2 * kABytes;
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k) {
            const uint32_t acc = (kb > 0 || k > 0) ? 1u : 0u;
            const uint64_t bd = smem_desc_sw128(sb + k * 32);
            mma_pair_bf16(pipe.tmem, smem_desc_sw128(sa + k * 32), bd, idesc, acc);
            if (g.has1) mma_pair_bf16(pipe.tmem + kPairMaxN, smem_desc_sw128(sa + kABytes + k * 32), bd, idesc, acc);
          }
          commit_pair(&pipe.empty[s]);  // frees stage s in both CTAs
        }
        commit_pair(&pipe.acc_full);  // arrives in both CTAs when every MMA above has completed
        if (pipe.fail) break;
      }
      // both epilogues' releases of the last tile land before this CTA may exit
      if (!pipe.fail && !mbar_wait_cluster(&pipe.acc_empty, ((uint32_t)ti & 1u) ^ 1u, a.err)) pipe.fail = 1;
    }
  } else {
    // epilogue: thread = TMEM lane = row of this CTA's half of A0 and of A1;
    // the two warps of a lane quadrant take the lower and the upper half of
    // the tile's 32-column chunks, and the lower merges the upper's result
    const int et = threadIdx.x - 64;
    const int quad = warp & 3;
    const int half = (warp - 2) / 4;
    const int r = quad * 32 + lane;
    const uint32_t acc_empty = cluster_addr(&pipe.acc_empty, 0);
    int ti = 0;
    for (int rd = 0, k; (k = pair_deal_tile(pl, pair, rd)) >= 0; ++rd, ++ti) {
      const PairTile g = pair_tile(pl, a.n_pruned, a.keep, k);
      const int* pr = a.pruned + (size_t)g.b * a.n_pruned;
      const int* kp = a.keep_idx + (size_t)g.b * a.keep;
      for (int i = et; i < 2 * kBM; i += 32 * kPairEpiWarps) {
        const int pos = g.m0 + (i < kBM ? 0 : 2 * kBM) + (int)rank * kBM + (i & (kBM - 1));
        sidx[i] = pos < a.n_pruned ? pr[pos] : -1;
      }
      for (int q = et; q < g.nv; q += 32 * kPairEpiWarps) {
        int j = kp[g.c0 + q];
        if (j < 0 || j >= a.N_v) {
          set_error(a.err, kErrBadDeviceArg);
          j = 0;
        }
        skinv[q] = a.inv_v[(size_t)g.b * a.N_v + j];
      }
      RowBest r0, r1;
      r0.init();
      r1.init();
      // the epilogue warps agree on the outcome, so that they leave the loop
      // together (the barrier also completes the tables)
      const bool ok = epilogue_all(warp_mbar_wait(&pipe.acc_full, (uint32_t)ti & 1u, a.err) && !pipe.fail);
      if (ok) {
        tc_fence_after();
        const uint32_t taddr = pipe.tmem + ((uint32_t)(quad * 32) << 16);
        const int ncb = g.N / 32, mid = (ncb + 1) / 2;
        const int cb0 = half ? mid : 0, cb1 = half ? ncb : mid;
        // 32-column pieces (chunk cb of A0, then of A1 when the group has a
        // second half), double-buffered: piece j + 1 loads while j is reduced
        const int sh = g.has1 ? 1 : 0;
        const int npc = (cb1 - cb0) << sh;
        auto piece = [&](int j, float* v) {
          tmem_ld32(taddr + (uint32_t)((j & sh) * kPairMaxN + (cb0 + (j >> sh)) * 32), v);
        };
        auto reduce = [&](int j, const float* v) {
          const int cb = cb0 + (j >> sh);
          if (j & sh)
            r1.add32(v, skinv + cb * 32, cb * 32, g.nv, g.c0);
          else
            r0.add32(v, skinv + cb * 32, cb * 32, g.nv, g.c0);
        };
        float va[32], vb[32];
        if (npc > 0) piece(0, va);
#pragma unroll 1
        for (int j = 0; j < npc; j += 2) {
          tc_wait_ld_into(va);
          if (j + 1 < npc) piece(j + 1, vb);
          reduce(j, va);
          if (j + 1 < npc) {
            tc_wait_ld_into(vb);
            if (j + 2 < npc) piece(j + 2, va);
            reduce(j + 1, vb);
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(acc_empty);  // this warp is done with the accumulators
      if (!ok) {
        pipe.fail = 1;
        break;
      }
      float best0, best1;
      int bidx0, bidx1;
      r0.result(best0, bidx0);
      r1.result(best1, bidx1);
      if (half) {
        xbest[0][r] = best0;
        xidx[0][r] = bidx0;
        xbest[1][r] = best1;
        xidx[1][r] = bidx1;
      }
      epilogue_sync();  // the upper halves' results are in shared memory
      if (!half) {
        // the upper half's positions are all larger: it wins only if larger
        if (xbest[0][r] > best0) {
          best0 = xbest[0][r];
          bidx0 = xidx[0][r];
        }
        if (xbest[1][r] > best1) {
          best1 = xbest[1][r];
          bidx1 = xidx[1][r];
        }
        const size_t slot = (size_t)a.B * a.N_v;
        const size_t o = ((size_t)g.t * a.B + g.b) * a.N_v;
        // the last range of a quad with fewer ranges than slots also fills the
        // spare slot with an entry that never wins
        const bool spare = g.t + 1 == g.n && g.n < pl.n_slots;
        const int j0 = sidx[r], j1 = sidx[kBM + r];
        if (j0 >= 0) {
          a.ws_best[o + j0] = best0;
          a.ws_bidx[o + j0] = bidx0;
          if (spare) {
            a.ws_best[o + slot + j0] = -INFINITY;
            a.ws_bidx[o + slot + j0] = 0x7fffffff;
          }
        }
        if (g.has1 && j1 >= 0) {
          a.ws_best[o + j1] = best1;
          a.ws_bidx[o + j1] = bidx1;
          if (spare) {
            a.ws_best[o + slot + j1] = -INFINITY;
            a.ws_bidx[o + slot + j1] = 0x7fffffff;
          }
        }
      }
      epilogue_sync();  // tables and exchange free for the next tile
    }
  }
  tc_fence_before();
  __syncwarp();
  pair_cluster_sync();  // every MMA of the pair has completed and been read
  if (warp == 0) tmem_dealloc_pair(pipe.tmem, kPairTmemCols);
}

size_t pair_smem() { return (size_t)kPairStages * kPairStageBytes + 1024; }

// per device: 0 = not checked, 1 = two-CTA clusters of this kernel fit, 2 = they do not
std::atomic<int> g_pair_ok[64];
std::atomic<int> g_pair_enabled{1};

}  // namespace

void merge_pair_enable(int on) { g_pair_enabled.store(on ? 1 : 0); }

// Tiles and their deal for B samples of n_pruned pruned and keep kept rows
// of width D on num_sms SMs: among splits that give 1 to 4 tiles per pair of
// SMs (and the even splits), the one whose busiest pair has the fewest clocks
// by a model of a tile of N columns: per 64-element K slice the larger of its
// MMA clocks (4N with both halves of the group, 2N with one) and 960 (the
// ring's pace: a stage's loads take about 2700 clocks from issue to landing,
// and four stages fit in shared memory), plus 9000 clocks of epilogue and
// refill per tile.
static bool merge_pair_search(int B, int n_pruned, int keep, int D, int num_sms, MergePairPlan* p) {
  if (B < 1 || n_pruned < 1 || keep < 1 || D < 1 || num_sms < 2) return false;
  const int n_quads = (n_pruned + kPairQuadRows - 1) / kPairQuadRows;
  const long long Q = (long long)B * n_quads;
  const int max_pairs = num_sms / 2;
  const long long n_k = (D + kBK - 1) / kBK;
  if (Q > (1 << 20)) return false;
  double best = -1.0;
  std::vector<double> load;
  auto consider = [&](int n_lo, long long x_hi) {
    const int n_hi = n_lo + (x_hi > 0 ? 1 : 0);
    if (n_lo < 1 || n_hi > kMergeMaxSplit || x_hi < 0 || x_hi >= Q) return;
    MergePairPlan c;
    c.n_quads = n_quads;
    c.Q = (int)Q;
    c.n_lo = n_lo;
    c.x_hi = (int)x_hi;
    const long long T = x_hi * (n_lo + 1) + (Q - x_hi) * n_lo;
    if (T > (1 << 24)) return;
    c.T = (int)T;
    c.P = (int)(T < max_pairs ? T : max_pairs);
    c.n_slots = n_hi;
    c.n_heights = 0;
    for (int n = n_lo; n <= n_hi; ++n)
      for (int t = 0; t < n; ++t) {
        const int nv = pair_range_start(t + 1, n, keep) - pair_range_start(t, n, keep);
        if (nv < 1 || nv > kPairMaxN) return;
        const int h = (nv + 31) / 32 * 16;  // B rows per CTA
        int j = 0;
        while (j < c.n_heights && c.heights[j] != h) ++j;
        if (j == c.n_heights) {
          if (j == kMergePairHeights) return;
          c.heights[c.n_heights++] = h;
        }
      }
    load.assign(c.P, 0.0);
    for (int pr = 0; pr < c.P; ++pr) {
      for (int r = 0, k; (k = pair_deal_tile(c, pr, r)) >= 0; ++r) {
        const PairTile g = pair_tile(c, n_pruned, keep, k);
        load[pr] += (double)n_k * fmax((g.has1 ? 4.0 : 2.0) * g.N, 960.0) + 9000.0;
      }
    }
    double worst = 0.0;
    for (double l : load) worst = fmax(worst, l);
    if (best < 0 || worst < best) {
      best = worst;
      *p = c;
    }
  };
  for (int n_lo = (keep + kPairMaxN - 1) / kPairMaxN; n_lo <= kMergeMaxSplit; ++n_lo) {
    consider(n_lo, 0);
    for (int m = 1; m <= 4; ++m) {
      const long long x_hi = (long long)m * max_pairs - Q * n_lo;
      if (x_hi > 0 && x_hi < Q) consider(n_lo, x_hi);
    }
  }
  return best >= 0;
}

// The search simulates every candidate's deal (tens to hundreds of
// microseconds of host time): its results are kept per shape, the last
// kPlanCache shapes, for the calls that follow.
namespace {
constexpr int kPlanCache = 16;
struct PlanEntry {
  int B, n_pruned, keep, D, num_sms;
  bool ok;
  MergePairPlan plan;
};
std::mutex g_plan_mu;
PlanEntry g_plans[kPlanCache];
int g_plan_n = 0, g_plan_next = 0;
}  // namespace

bool merge_pair_plan(int B, int n_pruned, int keep, int D, int num_sms, MergePairPlan* p) {
  {
    std::lock_guard<std::mutex> lock(g_plan_mu);
    for (int i = 0; i < g_plan_n; ++i) {
      const PlanEntry& e = g_plans[i];
      if (e.B == B && e.n_pruned == n_pruned && e.keep == keep && e.D == D && e.num_sms == num_sms) {
        if (e.ok) *p = e.plan;
        return e.ok;
      }
    }
  }
  MergePairPlan plan;
  const bool ok = merge_pair_search(B, n_pruned, keep, D, num_sms, &plan);
  std::lock_guard<std::mutex> lock(g_plan_mu);
  PlanEntry& e = g_plans[g_plan_next];
  e = PlanEntry{B, n_pruned, keep, D, num_sms, ok, plan};
  g_plan_next = (g_plan_next + 1) % kPlanCache;
  if (g_plan_n < kPlanCache) ++g_plan_n;
  if (ok) *p = plan;
  return ok;
}

bool merge_pair_usable(const SimArgs& a) {
  if (!g_pair_enabled.load() || a.dtype != 1 || a.D % 8) return false;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return false;
  int st = g_pair_ok[dev].load(std::memory_order_acquire);
  if (st == 0) {
    st = 2;
    const size_t smem = pair_smem();
    cudaError_t e = cudaFuncSetAttribute(merge_argmax_pair_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e == cudaSuccess) {
      cudaLaunchConfig_t cfg = {};
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeClusterDimension;
      attr[0].val.clusterDim.x = 2;
      attr[0].val.clusterDim.y = 1;
      attr[0].val.clusterDim.z = 1;
      cfg.gridDim = dim3(2, 1, 1);
      cfg.blockDim = dim3(kPairThreads, 1, 1);
      cfg.dynamicSmemBytes = smem;
      cfg.attrs = attr;
      cfg.numAttrs = 1;
      int n = 0;
      e = cudaOccupancyMaxActiveClusters(&n, merge_argmax_pair_tc, &cfg);
      if (e == cudaSuccess && n > 0) st = 1;
    }
    // a refused attribute or query falls back to the single-SM form: clear the
    // error it left (only then, so that no earlier error of the caller is lost)
    if (e != cudaSuccess) cudaGetLastError();
    g_pair_ok[dev].store(st, std::memory_order_release);
  }
  return st == 1;
}

cudaError_t merge_argmax_pair_launch(const SimArgs& a, const int* keep_idx, int keep, const float* inv_v,
                                     const int* pruned, const void* perm, const MergePairPlan& plan,
                                     float* ws_best, int* ws_bidx, cudaStream_t s) {
  PairMaps maps;
  const uint64_t rows = (uint64_t)a.B * a.N_v;
  if (make_tmap_bf16_2d(&maps.a, perm, rows, (uint64_t)a.D, (uint64_t)a.D * 2, kBM))
    return cudaErrorInvalidValue;
  for (int j = 0; j < plan.n_heights; ++j)
    if (make_tmap_bf16_2d(&maps.b[j], perm, rows, (uint64_t)a.D, (uint64_t)a.D * 2, (uint32_t)plan.heights[j]))
      return cudaErrorInvalidValue;
  PairArgs m;
  m.pruned = pruned;
  m.n_pruned = a.N_v - keep;
  m.keep_idx = keep_idx;
  m.keep = keep;
  m.N_v = a.N_v;
  m.D = a.D;
  m.B = a.B;
  m.inv_v = inv_v;
  m.plan = plan;
  m.ws_best = ws_best;
  m.ws_bidx = ws_bidx;
  m.err = a.err;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.gridDim = dim3((unsigned)(2 * plan.P), 1, 1);
  cfg.blockDim = dim3(kPairThreads, 1, 1);
  cfg.dynamicSmemBytes = pair_smem();
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, merge_argmax_pair_tc, m, maps);
}

}  // namespace provip
