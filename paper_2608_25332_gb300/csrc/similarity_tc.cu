// Pre-LLM pass (Sec. 4.3) on 5th-generation tensor cores (bf16).
//
// merge_argmax_tc: the pruned x kept cosine Gram fused with the row argmax, on
//   single SMs (the form on pairs of SMs is merge_pair_tc.cu, the default).
//   A = the pruned visual rows of two 128-row M tiles, B = the kept rows of a
//   range of 256-row N tiles shared by both, read as contiguous tiles of a
//   per-sample copy of E_v permuted to [pruned | kept] by one bandwidth-bound
//   gather pass. The epilogue scales a column by 1/|e_k| and keeps, per row,
//   the running (max, first index) over the kept positions in ascending order,
//   so ties go to the lower kept position. The (N_v - N1) x N1 matrix never
//   leaves the SM.
// relevance_fused_tc: the visual x [visual ; text] Gram of a 128-row visual
//   tile, one read of the visual rows giving |v_j|^2 (the diagonal of the
//   visual block), the cosines and the de-meaning sums (p_j itself is formed by
//   a small second kernel once every tile's sums are known).
// crit_gram_tc: the text Gram E_t E_t^T, split over K.
#include "common.cuh"
#include "kernels.h"
#include "merge_epi.cuh"
#include "tc_gemm.cuh"

namespace provip {
namespace {

using namespace tcg;

// perm[b] = rows of E_v[b] reordered as [pruned rows (ascending) | kept rows
// (keep order)], so that the Gram reads both operands as contiguous tiles.
// One warp per output row, 16-byte vectors.
__global__ void __launch_bounds__(256) gather_perm_kernel(const __nv_bfloat16* E, const int* pruned,
                                                          const int* keep_idx, int n_pruned, int keep,
                                                          int N_v, int D, __nv_bfloat16* perm,
                                                          unsigned* err) {
  pdl_wait_prior();  // pruned and keep_idx come from the kernels before
  pdl_allow_next();  // the Gram may set itself up meanwhile
  const int b = blockIdx.y;
  const int r = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (r >= N_v) return;
  int j = r < n_pruned ? pruned[(size_t)b * n_pruned + r] : keep_idx[(size_t)b * keep + (r - n_pruned)];
  if (j < 0 || j >= N_v) {
    if (lane == 0) set_error(err, kErrBadDeviceArg);
    j = 0;
  }
  const uint4* src = reinterpret_cast<const uint4*>(E + ((size_t)b * N_v + j) * D);
  uint4* dst = reinterpret_cast<uint4*>(perm + ((size_t)b * N_v + r) * D);
  const int nvec = D / 8;
  // four 16-byte loads in flight per lane before their stores
  int v = lane;
  for (; v + 96 < nvec; v += 128) {
    const uint4 x0 = __ldg(src + v), x1 = __ldg(src + v + 32), x2 = __ldg(src + v + 64), x3 = __ldg(src + v + 96);
    dst[v] = x0;
    dst[v + 32] = x1;
    dst[v + 64] = x2;
    dst[v + 96] = x3;
  }
  for (; v < nvec; v += 32) dst[v] = __ldg(src + v);
}

struct MergeTcArgs {
  const int* pruned;   // [B][n_pruned]
  int n_pruned;
  const int* keep_idx; // [B][keep]
  int keep;
  int N_v, D, B;
  const float* inv_v;  // [B][N_v]
  int n_split;
  float* ws_best;      // [n_split][B][N_v]
  int* ws_bidx;
  unsigned* err;
};

constexpr int kMergeBN = 256;
constexpr int kMergeMaxKeep = 2560;  // kept rows handled by one split (shared index table)
constexpr int kMergeStages = 3;
constexpr int kMergeBBytes = kMergeBN * kBK * 2;                 // 32 KiB
constexpr int kMergeStageBytes = 2 * kABytes + kMergeBBytes;     // A0 | A1 | B: 64 KiB
constexpr uint32_t kMergeTmemCols = 2 * kMergeBN;                // one accumulator per M tile
constexpr int kMergeEpiWarps = 8;  // two per TMEM lane quadrant, splitting each tile's columns
constexpr int kMergeThreads = 64 + 32 * kMergeEpiWarps;

struct MergePipe {
  uint64_t full[kMergeStages];
  uint64_t empty[kMergeStages];
  uint64_t acc_full;
  uint64_t acc_empty;
  uint32_t tmem;
  volatile int fail;
};

// One CTA owns two 128-row M tiles of pruned rows (A0, A1) and sweeps its range
// of 256-row N tiles of kept rows; each stage holds A0, A1 and one B tile, and
// two MMAs (M = 128, N <= 256) share that B tile, so a stage carries 64 KiB for
// 8.4 MFLOP instead of 48 KiB for 4.2 MFLOP with a single M tile. The two
// accumulators fill the 512 TMEM columns: the epilogue of an N tile runs
// between that tile's last MMA and the next tile's first (the producer keeps
// loading meanwhile), so it is kept short: eight warps, two per TMEM lane
// quadrant, each taking half of a tile's 32-column pieces with its loads
// double-buffered and four interleaved running maxima per row (RowBest). The
// last N tile's MMA is only as wide as its kept rows (rounded up to 16).
__global__ void __launch_bounds__(kMergeThreads, 1)
    merge_argmax_tc(const MergeTcArgs a, const __grid_constant__ CUtensorMap mapE) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ MergePipe pipe;
  __shared__ int sidx_a[2 * kBM];
  __shared__ float xbest[2][kBM];  // the upper column halves' (max, position) per row
  __shared__ int xidx[2][kBM];
  const int b = blockIdx.z, split = blockIdx.y;
  const int m0 = blockIdx.x * 2 * kBM;
  const bool has1 = m0 + kBM < a.n_pruned;  // the second M tile holds pruned rows
  const int n_tiles_all = (a.keep + kMergeBN - 1) / kMergeBN;
  const int t0 = (int)((long long)n_tiles_all * split / a.n_split);
  const int t1 = (int)((long long)n_tiles_all * (split + 1) / a.n_split);
  const int n_tiles = t1 - t0;
  const int a0 = t0 * kMergeBN;                       // first kept position of the range
  const int n_keep = min(a.keep, t1 * kMergeBN) - a0;  // kept rows in the range
  const int n_k = (a.D + kBK - 1) / kBK;

  const uint32_t sbase = smem_u32(smem_raw);
  uint8_t* stages = smem_raw + (((sbase + 1023u) & ~1023u) - sbase);
  float* skinv = reinterpret_cast<float*>(stages + (size_t)kMergeStages * kMergeStageBytes);

  if (threadIdx.x == 0) {
    prefetch_tmap(&mapE);
    for (int s = 0; s < kMergeStages; ++s) {
      mbar_init(&pipe.full[s], 1);
      mbar_init(&pipe.empty[s], 1);
    }
    mbar_init(&pipe.acc_full, 1);
    mbar_init(&pipe.acc_empty, kMergeEpiWarps);  // one arrival per epilogue warp
    pipe.fail = 0;
    fence_mbar_init();
  }
  if (threadIdx.x < 32) {
    tmem_alloc(&pipe.tmem, kMergeTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();

  // N columns of tile t: 256, or the kept rows of a ragged last tile rounded up to 16
  auto tile_cols = [&](int t) { return min(kMergeBN, (n_keep - t * kMergeBN + 15) / 16 * 16); };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (n_tiles > 0) {
    if (warp == 0) {
      if (lane == 0) {
        // operands are contiguous rows of the permuted copy [pruned | kept];
        // rows past a tile's valid rows are computed and never used
        const int row_a = b * a.N_v + m0;
        const int row_b = b * a.N_v + a.n_pruned + a0;
        int it = 0;
        for (int t = 0; t < n_tiles && !pipe.fail; ++t) {
          const bool b_hi = tile_cols(t) > kBM;  // the tile's second 128-row box is used
          const uint32_t tx = (uint32_t)((has1 ? 2 : 1) * kABytes + (b_hi ? 2 : 1) * kABytes);
          for (int kb = 0; kb < n_k; ++kb, ++it) {
            const int s = it % kMergeStages;
            const uint32_t ph = (uint32_t)(it / kMergeStages) & 1u;
            if (pipe.fail || !mbar_wait(&pipe.empty[s], ph ^ 1u, a.err)) {
              pipe.fail = 1;
              break;
            }
            uint8_t* sa = stages + (size_t)s * kMergeStageBytes;
            uint8_t* sb = sa + 2 * kABytes;
            const int x = kb * kBK;
            mbar_arrive_expect_tx(&pipe.full[s], tx);
            tma_load_2d(sa, &mapE, x, row_a, &pipe.full[s]);
            if (has1) tma_load_2d(sa + kABytes, &mapE, x, row_a + kBM, &pipe.full[s]);
            tma_load_2d(sb, &mapE, x, row_b + t * kMergeBN, &pipe.full[s]);
            if (b_hi) tma_load_2d(sb + kABytes, &mapE, x, row_b + t * kMergeBN + kBM, &pipe.full[s]);
          }
        }
      }
    } else if (warp == 1) {
      if (lane == 0) {
        int it = 0;
        for (int t = 0; t < n_tiles; ++t) {
          if (!pipe.fail && !mbar_wait(&pipe.acc_empty, ((uint32_t)t & 1u) ^ 1u, a.err)) pipe.fail = 1;
          const uint32_t idesc = idesc_bf16_f32(kBM, tile_cols(t));
          for (int kb = 0; kb < n_k; ++kb, ++it) {
            const int s = it % kMergeStages;
            const uint32_t ph = (uint32_t)(it / kMergeStages) & 1u;
            if (pipe.fail || !mbar_wait(&pipe.full[s], ph, a.err)) {
              pipe.fail = 1;
              break;
            }
            tc_fence_after();
            const uint32_t sa = smem_u32(stages + (size_t)s * kMergeStageBytes);
            const uint32_t sb = sa + 2 * kABytes;
#pragma unroll
            for (int k = 0; k < kBK / 16; ++k) {
              const uint32_t acc = (kb > 0 || k > 0) ? 1u : 0u;
              const uint64_t bd = smem_desc_sw128(sb + k * 32);
              tc_mma_bf16(pipe.tmem, smem_desc_sw128(sa + k * 32), bd, idesc, acc);
              if (has1) tc_mma_bf16(pipe.tmem + kMergeBN, smem_desc_sw128(sa + kABytes + k * 32), bd, idesc, acc);
            }
            tc_commit(&pipe.empty[s]);
          }
          tc_commit(&pipe.acc_full);  // arrives when every MMA above has completed
          if (pipe.fail) break;
        }
      }
    } else {
      // the epilogue warps fill the index tables while the first stages load
      const int* pr = a.pruned + (size_t)b * a.n_pruned;
      const int* kp = a.keep_idx + (size_t)b * a.keep;
      const int et = threadIdx.x - 64;
      constexpr int kEpi = 32 * kMergeEpiWarps;
      for (int r = et; r < 2 * kBM; r += kEpi) sidx_a[r] = m0 + r < a.n_pruned ? pr[m0 + r] : 0;
      for (int q = et; q < n_keep; q += kEpi) {
        int j = kp[a0 + q];
        if (j < 0 || j >= a.N_v) {
          set_error(a.err, kErrBadDeviceArg);
          j = 0;
        }
        skinv[q] = a.inv_v[(size_t)b * a.N_v + j];
      }
      asm volatile("bar.sync 1, %0;" ::"n"(kEpi) : "memory");  // tables complete (epilogue warps)
      // epilogue: row r of each M tile; the two warps of a lane quadrant take
      // the lower and the upper half of each tile's 32-column pieces (their
      // tensor-memory loads double-buffered), each keeping a running (max,
      // first position) over the range, merged at the end
      const int quad = warp & 3;
      const int half = (warp - 2) / 4;
      const int r = quad * 32 + lane;
      RowBest r0, r1;
      r0.init();
      r1.init();
      bool ok = true;
      for (int t = 0; t < n_tiles; ++t) {
        ok = warp_mbar_wait(&pipe.acc_full, (uint32_t)t & 1u, a.err) && !pipe.fail;
        if (!ok) break;
        tc_fence_after();
        const uint32_t taddr = pipe.tmem + ((uint32_t)(quad * 32) << 16);
        const int ncb = (tile_cols(t) + 31) / 32, mid = (ncb + 1) / 2;
        const int cb0 = half ? mid : 0, cb1 = half ? ncb : mid;
        const int sh = has1 ? 1 : 0;
        const int npc = (cb1 - cb0) << sh;
        auto piece = [&](int j, float* v) {
          tmem_ld32(taddr + (uint32_t)((j & sh) * kMergeBN + (cb0 + (j >> sh)) * 32), v);
        };
        auto reduce = [&](int j, const float* v) {
          const int q0 = t * kMergeBN + (cb0 + (j >> sh)) * 32;  // position within the range
          if (j & sh)
            r1.add32(v, skinv + q0, q0, n_keep, a0);
          else
            r0.add32(v, skinv + q0, q0, n_keep, a0);
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
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&pipe.acc_empty);
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
      asm volatile("bar.sync 1, %0;" ::"n"(kEpi) : "memory");  // the upper halves' results
      if (!half) {
        if (merge_better(xbest[0][r], xidx[0][r], best0, bidx0)) {
          best0 = xbest[0][r];
          bidx0 = xidx[0][r];
        }
        if (merge_better(xbest[1][r], xidx[1][r], best1, bidx1)) {
          best1 = xbest[1][r];
          bidx1 = xidx[1][r];
        }
      }
      if (!half && ok && !pipe.fail) {
        const size_t o = ((size_t)split * a.B + b) * a.N_v;
        if (m0 + r < a.n_pruned) {
          a.ws_best[o + sidx_a[r]] = best0;
          a.ws_bidx[o + sidx_a[r]] = bidx0;
        }
        if (m0 + kBM + r < a.n_pruned) {
          a.ws_best[o + sidx_a[kBM + r]] = best1;
          a.ws_bidx[o + sidx_a[kBM + r]] = bidx1;
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x < 32) tmem_dealloc(pipe.tmem, kMergeTmemCols);
}

// relevance_fused_tc: one read of the visual rows gives, per tile of R visual
// rows of sample b (R = 128, 96 or 64, chosen so that the tiles spread evenly
// over the SMs; A = the tile's rows, B = [the same R visual rows ; the text
// rows], both already adjacent in the stage, so one MMA of N = R + NT; the
// MMA's 128 A rows run past the R visual rows and their results are unused),
//   * |v_j|^2 from the diagonal of the visual x visual block (thread = TMEM
//     lane = visual row j reads its own column),
//   * the cosines Y[b][j][i] = <v_j, t_i> |t_i|^-1 |v_j|^-1 (|t_i|^-1 from a
//     separate pass over the text rows),
//   * the tile's column sums part[b][tile][i] = sum_j Y[b][j][i] (warp
//     butterfly, then the four lane quadrants in order).
// relevance_finish_kernel then forms mu_i = (sum of the tile sums in tile
// order) / N_v and p_j = max_{i in T} (Y[b][j][i] - mu_i) (Sec. 4.3).
struct RelFusedArgs {
  int B, N_v, D, N_t_max;
  int NT;        // text rows in the MMA (N_t_max rounded up to 16)
  int R;         // visual rows per tile (128, 96 or 64)
  int n_vt;      // visual tiles per sample
  int n_stages;  // shared-memory ring depth
  const float* inv_t;  // [B][N_t_max]
  float* inv_v;  // [B][N_v]
  float* Y;      // [B][N_v][NT]
  float* part;   // [B][n_vt][NT]
  unsigned* err;
};

constexpr int kRelMaxStages = 8;
constexpr int kRelFinishRows = 8;  // rows per warp of relevance_finish_kernel
constexpr uint32_t kRelTmemCols = 256;  // 128 visual + <= 128 text columns

struct RelPipe {
  uint64_t full[kRelMaxStages];
  uint64_t empty[kRelMaxStages];
  uint64_t acc_full;
  uint32_t tmem;
  volatile int fail;
};

__global__ void __launch_bounds__(kThreads, 2)
    relevance_fused_tc(const RelFusedArgs a, const __grid_constant__ CUtensorMap mapV,
                       const __grid_constant__ CUtensorMap mapT) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ RelPipe pipe;
  __shared__ float s_invt[kBM];
  __shared__ float red[4][kBM];
  const int b = blockIdx.y, tile = blockIdx.x;
  const int R = a.R;
  const int n0 = tile * R;
  const int n_k = (a.D + kBK - 1) / kBK;
  const int NS = a.n_stages;
  const uint32_t st_bytes = (uint32_t)(R + a.NT) * 128u;
  const uint32_t sbase = smem_u32(smem_raw);
  uint8_t* stages = smem_raw + (((sbase + 1023u) & ~1023u) - sbase);
  if (threadIdx.x == 0) {
    prefetch_tmap(&mapV);
    prefetch_tmap(&mapT);
    for (int s = 0; s < NS; ++s) {
      mbar_init(&pipe.full[s], 1);
      mbar_init(&pipe.empty[s], 1);
    }
    mbar_init(&pipe.acc_full, 1);
    pipe.fail = 0;
    fence_mbar_init();
  }
  if (threadIdx.x < 32) {
    tmem_alloc(&pipe.tmem, kRelTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (warp == 0) {
    if (lane == 0) {
      for (int kb = 0; kb < n_k; ++kb) {
        const int s = kb % NS;
        const uint32_t ph = (uint32_t)(kb / NS) & 1u;
        if (pipe.fail || !mbar_wait(&pipe.empty[s], ph ^ 1u, a.err)) {
          pipe.fail = 1;
          break;
        }
        uint8_t* sa = stages + (size_t)s * st_bytes;
        mbar_arrive_expect_tx(&pipe.full[s], st_bytes);
        // rows past the sample's last visual row belong to the next sample (or
        // lie past the tensor and read as zeros): computed, never stored
        tma_load_2d(sa, &mapV, kb * kBK, b * a.N_v + n0, &pipe.full[s]);
        tma_load_2d(sa + R * 128, &mapT, kb * kBK, b * a.N_t_max, &pipe.full[s]);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16_f32(kBM, R + a.NT);
      for (int kb = 0; kb < n_k; ++kb) {
        const int s = kb % NS;
        const uint32_t ph = (uint32_t)(kb / NS) & 1u;
        if (pipe.fail || !mbar_wait(&pipe.full[s], ph, a.err)) {
          pipe.fail = 1;
          break;
        }
        tc_fence_after();
        const uint32_t sa = smem_u32(stages + (size_t)s * st_bytes);
#pragma unroll
        for (int k = 0; k < kBK / 16; ++k)
          tc_mma_bf16(pipe.tmem, smem_desc_sw128(sa + k * 32), smem_desc_sw128(sa + k * 32), idesc,
                      (kb > 0 || k > 0) ? 1u : 0u);
        tc_commit(&pipe.empty[s]);
      }
      tc_commit(&pipe.acc_full);  // arrives once every MMA above has completed
    }
  } else {
    const int quad = warp & 3;
    const int r = quad * 32 + lane;
    const int j = n0 + r;
    const bool rv = r < R && j < a.N_v;
    // launched as a programmatic dependent of the text-row norms: the loads and
    // MMAs ran under that kernel; its output (and every write below) waits here
    pdl_wait_prior();
    s_invt[r] = r < a.N_t_max ? a.inv_t[(size_t)b * a.N_t_max + r] : 0.f;
    asm volatile("bar.sync 1, 128;" ::: "memory");  // s_invt complete (epilogue warps)
    const bool ok = warp_mbar_wait(&pipe.acc_full, 0, a.err) && !pipe.fail;
    tc_fence_after();
    const uint32_t taddr = pipe.tmem + ((uint32_t)(quad * 32) << 16);
    float v[32];
    // |v_j|^2: column j of the visual block, i.e. element `lane` of the warp's 32 columns
    tmem_ld32(taddr + (uint32_t)(quad * 32), v);
    tc_wait_ld();
    float sqv = 0.f;
#pragma unroll
    for (int i = 0; i < 32; ++i) sqv = i == lane ? v[i] : sqv;
    const float iv = sqv > 0.f ? 1.f / sqrtf(sqv) : 0.f;
    if (rv && ok) a.inv_v[(size_t)b * a.N_v + j] = iv;
    float* yrow = a.Y + ((size_t)b * a.N_v + (rv ? j : 0)) * a.NT;
#pragma unroll 1
    for (int cb = 0; cb * 32 < a.NT; ++cb) {
      tmem_ld32(taddr + (uint32_t)(R + cb * 32), v);
      tc_wait_ld();
#pragma unroll
      for (int i = 0; i < 32; ++i) v[i] = v[i] * s_invt[cb * 32 + i] * iv;
      if (rv && ok) {
#pragma unroll
        for (int q = 0; q < 8; ++q)
          if (cb * 32 + q * 4 < a.NT)
            *reinterpret_cast<float4*>(yrow + cb * 32 + q * 4) =
                make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
      }
#pragma unroll
      for (int i = 0; i < 32; ++i) v[i] = rv ? v[i] : 0.f;
      // butterfly sum over the 32 rows of the warp: lane ends with column `lane`
#pragma unroll
      for (int sh = 16; sh >= 1; sh >>= 1) {
        const bool upper = (lane & sh) != 0;
#pragma unroll
        for (int i = 0; i < sh; ++i) {
          const float keep = upper ? v[i + sh] : v[i];
          const float send = upper ? v[i] : v[i + sh];
          v[i] = keep + __shfl_xor_sync(0xffffffffu, send, sh);
        }
      }
      red[quad][cb * 32 + lane] = v[0];
    }
    tc_fence_before();
    asm volatile("bar.sync 1, 128;" ::: "memory");
    const int c = threadIdx.x - 64;
    if (c < a.NT && ok)
      a.part[((size_t)b * a.n_vt + tile) * a.NT + c] = (red[0][c] + red[1][c]) + (red[2][c] + red[3][c]);
  }
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x < 32) tmem_dealloc(pipe.tmem, kRelTmemCols);
}

// mu_i from the tile sums (tile order; every CTA forms all of mu), then p_j =
// max over the critical rows of Y[b][j][i] - mu_i; an empty T gives -inf.
__global__ void __launch_bounds__(256) relevance_finish_kernel(const RelFusedArgs a, const int* text_len,
                                                               const uint8_t* mask, float* p) {
  pdl_allow_next();  // the top-k reads p only after this grid completes
  __shared__ float mu[kBM];
  __shared__ int valid[kBM];
  const int b = blockIdx.y;
  const int tl = min(max(text_len[b], 0), a.N_t_max);
  for (int c = threadIdx.x; c < a.NT; c += blockDim.x) {
    const bool v = c < tl && mask[(size_t)b * a.N_t_max + c] != 0;
    float s = 0.f;
    if (v) {
      const float* col = a.part + (size_t)b * a.n_vt * a.NT + c;
      for (int t0 = 0; t0 < a.n_vt; t0 += 32) {
        float x[32];
#pragma unroll
        for (int u = 0; u < 32; ++u) x[u] = t0 + u < a.n_vt ? col[(size_t)(t0 + u) * a.NT] : 0.f;
#pragma unroll
        for (int u = 0; u < 32; ++u)
          if (t0 + u < a.n_vt) s += x[u];
      }
    }
    mu[c] = s / (float)a.N_v;
    valid[c] = v;
  }
  __syncthreads();
  // a warp per kRelFinishRows rows: lane q reads the 16-byte piece q of each row
  // (NT <= 128: at most 32 pieces), every row's load in flight, then a warp max
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nq = a.NT / 4;
  const int j0 = (blockIdx.x * (blockDim.x >> 5) + warp) * kRelFinishRows;
  const bool has = lane < nq;
  const int c = lane * 4;
  const float m0 = has ? mu[c] : 0.f, m1 = has ? mu[c + 1] : 0.f, m2 = has ? mu[c + 2] : 0.f,
              m3 = has ? mu[c + 3] : 0.f;
  const bool v0 = has && valid[c], v1 = has && valid[c + 1], v2 = has && valid[c + 2], v3 = has && valid[c + 3];
  const float4* y = reinterpret_cast<const float4*>(a.Y + (size_t)b * a.N_v * a.NT);
  float4 f[kRelFinishRows];
#pragma unroll
  for (int r = 0; r < kRelFinishRows; ++r)
    f[r] = (has && j0 + r < a.N_v) ? y[(size_t)(j0 + r) * nq + lane] : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
  for (int r = 0; r < kRelFinishRows; ++r) {
    float best = -INFINITY;
    if (v0) best = fmaxf(best, f[r].x - m0);
    if (v1) best = fmaxf(best, f[r].y - m1);
    if (v2) best = fmaxf(best, f[r].z - m2);
    if (v3) best = fmaxf(best, f[r].w - m3);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) best = fmaxf(best, __shfl_xor_sync(0xffffffffu, best, o));
    if (lane == 0 && j0 + r < a.N_v) p[(size_t)b * a.N_v + j0 + r] = best;
  }
}

// G = E_t E_t^T for one sample (<= 128 text rows), split over K: CTA x of
// sample b sums the K slices [x * ks_per, (x + 1) * ks_per) and writes its part
// to G[x][b] as fp32; the softmax/column-mean step of Sec. 4.2 adds the parts
// in split order.
constexpr int kCritBN = 128;

__global__ void __launch_bounds__(kThreads, 1)
    crit_gram_tc(const __grid_constant__ CUtensorMap mapT, const int* text_len, int N_t_max, int D,
                 int B, int ks_per, float* G, unsigned* err) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ Pipe pipe;
  const int b = blockIdx.z;
  const int k0 = blockIdx.x * ks_per;
  const int n_k = min(ks_per, (D + kBK - 1) / kBK - k0);
  const uint32_t sbase = smem_u32(smem_raw);
  uint8_t* stages = smem_raw + (((sbase + 1023u) & ~1023u) - sbase);
  if (threadIdx.x == 0) {
    prefetch_tmap(&mapT);
    pipe_init(pipe);
  }
  if (threadIdx.x < 32) {
    tmem_alloc(&pipe.tmem, Cfg<kCritBN>::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (warp == 0) {
    if (lane == 0) {
      RowSrc ra{b * N_t_max, kBM};
      RowSrc rb{b * N_t_max, kCritBN};
      // both operands are the same text rows: one load per K slice
      producer<kCritBN>(pipe, stages, &mapT, &mapT, ra, rb, 1, n_k, err, k0, true);
    }
  } else if (warp == 1) {
    if (lane == 0) mma_issuer<kCritBN>(pipe, stages, 1, n_k, err, true);
  } else {
    const int quad = warp & 3;
    const int r = quad * 32 + lane;
    mbar_wait(&pipe.acc_full[0], 0, err);
    tc_fence_after();
    const uint32_t taddr = pipe.tmem + ((uint32_t)(quad * 32) << 16);
    float* g = G + (((size_t)blockIdx.x * B + b) * N_t_max + r) * N_t_max;
#pragma unroll 1
    for (int cb = 0; cb < kCritBN / 32; ++cb) {
      float v[32];
      tmem_ld32(taddr + cb * 32, v);
      tc_wait_ld();
      if (r < N_t_max && !pipe.fail) {
#pragma unroll
        for (int i = 0; i < 32; ++i)
          if (cb * 32 + i < N_t_max) g[cb * 32 + i] = v[i];
      }
    }
    tc_fence_before();
  }
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x < 32) tmem_dealloc(pipe.tmem, Cfg<kCritBN>::kTmemCols);
}

template <typename K>
cudaError_t set_smem(K kernel, size_t bytes, std::atomic<bool>* done) {
  if (done->load()) return cudaSuccess;
  cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
  if (e == cudaSuccess) done->store(true);  // idempotent: concurrent first calls may both set it
  return e;
}

}  // namespace

size_t merge_tc_smem() {
  return (size_t)kMergeStages * kMergeStageBytes + 1024 + (size_t)kMergeMaxKeep * sizeof(float);
}

int merge_tc_split(int B, int N_v, int keep, int num_sms) {
  const int m_tiles = B * ((N_v - keep + 2 * kBM - 1) / (2 * kBM));  // CTAs: pairs of M tiles
  const int n_tiles = (keep + kMergeBN - 1) / kMergeBN;
  int best = 1;
  long long best_cost = -1;
  for (int sp = 1; sp <= n_tiles && sp <= kMergeMaxSplit; ++sp) {
    const int per = (n_tiles + sp - 1) / sp;
    if (per * kMergeBN > kMergeMaxKeep) continue;
    const long long waves = ((long long)m_tiles * sp + num_sms - 1) / num_sms;
    const long long cost = waves * per;
    if (best_cost < 0 || cost < best_cost) {
      best_cost = cost;
      best = sp;
    }
  }
  return best;
}

bool merge_tc_supported(const SimArgs& a, int keep, int n_split) {
  if (a.dtype != 1 || a.D % 8) return false;
  const int n_tiles = (keep + kMergeBN - 1) / kMergeBN;
  const int per_split = (n_tiles + n_split - 1) / n_split;
  return per_split * kMergeBN <= kMergeMaxKeep && keep < a.N_v;
}

cudaError_t merge_argmax_tc_launch(const SimArgs& a, const int* keep_idx, int keep, const float* inv_v,
                                   const int* pruned, void* perm, int n_split,
                                   float* ws_best, int* ws_bidx, int num_sms, int* n_split_out,
                                   cudaStream_t s) {
  const int n_pruned = a.N_v - keep;  // pruned: the rows not kept, ascending (merge_index_kernel)
  MergePairPlan plan;
  const bool pairs = merge_pair_usable(a) && merge_pair_plan(a.B, n_pruned, keep, a.D, num_sms, &plan);
  cudaError_t e = cudaSuccess;
  if (!pairs) {
    static std::atomic<bool> smem_set[64];  // per device, zero-initialised
    int dev = 0;
    cudaGetDevice(&dev);
    e = set_smem(merge_argmax_tc, merge_tc_smem(), &smem_set[dev < 64 ? dev : 0]);
    if (e != cudaSuccess) return e;
  }
  dim3 gg((a.N_v + 7) / 8, a.B);
  e = launch_pdl(gather_perm_kernel, gg, dim3(256), 0, s, static_cast<const __nv_bfloat16*>(a.emb_v), pruned,
                 keep_idx, n_pruned, keep, a.N_v, a.D, static_cast<__nv_bfloat16*>(perm), a.err);
  if (e != cudaSuccess) return e;
  if (pairs) {
    *n_split_out = plan.n_slots;
    return merge_argmax_pair_launch(a, keep_idx, keep, inv_v, pruned, perm, plan, ws_best, ws_bidx, s);
  }
  *n_split_out = n_split;
  const size_t smem = merge_tc_smem();
  CUtensorMap mapE;
  if (make_tmap_bf16_2d(&mapE, perm, (uint64_t)a.B * a.N_v, (uint64_t)a.D, (uint64_t)a.D * 2, 128))
    return cudaErrorInvalidValue;
  MergeTcArgs m;
  m.pruned = pruned;
  m.n_pruned = n_pruned;
  m.keep_idx = keep_idx;
  m.keep = keep;
  m.N_v = a.N_v;
  m.D = a.D;
  m.B = a.B;
  m.inv_v = inv_v;
  m.n_split = n_split;
  m.ws_best = ws_best;
  m.ws_bidx = ws_bidx;
  m.err = a.err;
  dim3 grid((n_pruned + 2 * kBM - 1) / (2 * kBM), n_split, a.B);
  merge_argmax_tc<<<grid, kMergeThreads, smem, s>>>(m, mapE);
  return cudaGetLastError();
}

bool relevance_tc_supported(const SimArgs& a) { return a.dtype == 1 && a.N_t_max <= kBM && a.D % 8 == 0; }

static int rel_nt(int N_t_max) { return (N_t_max + 15) / 16 * 16; }

size_t relevance_fused_floats(int B, int N_v, int N_t_max) {
  const int NT = rel_nt(N_t_max), n_vt = (N_v + 63) / 64;  // tiles of the smallest R
  return (size_t)B * N_v * NT + (size_t)B * n_vt * NT;
}

// Visual rows per relevance tile: the R of 128, 96 and 64 whose tiles give the
// busiest SM the fewest rows to take in (its tiles' visual and text rows,
// ceil(tiles / SMs) tiles), the larger R on a tie.
static int rel_tile_rows(int B, int N_v, int NT, int num_sms) {
  int best = kBM;
  long long best_cost = -1;
  for (int R = kBM; R >= 64; R -= 32) {
    const long long tiles = (long long)B * ((N_v + R - 1) / R);
    const long long cost = ((tiles + num_sms - 1) / num_sms) * (R + NT);
    if (best_cost < 0 || cost < best_cost) {
      best_cost = cost;
      best = R;
    }
  }
  return best;
}

cudaError_t relevance_tc_launch(const SimArgs& a, const uint8_t* mask, const float* inv_t, float* inv_v,
                                float* p, float* ws, int num_sms, cudaStream_t s, cudaEvent_t mask_ready) {
  static std::atomic<bool> smem_set[64];  // per device, zero-initialised
  int dev = 0;
  cudaGetDevice(&dev);
  constexpr size_t kSmemMax = 200 * 1024;
  cudaError_t e = set_smem(relevance_fused_tc, kSmemMax, &smem_set[dev < 64 ? dev : 0]);
  if (e != cudaSuccess) return e;
  RelFusedArgs r;
  r.B = a.B;
  r.N_v = a.N_v;
  r.D = a.D;
  r.N_t_max = a.N_t_max;
  r.NT = rel_nt(a.N_t_max);
  r.R = rel_tile_rows(a.B, a.N_v, r.NT, num_sms);
  r.n_vt = (a.N_v + r.R - 1) / r.R;
  r.inv_t = inv_t;
  r.inv_v = inv_v;
  r.Y = ws;
  r.part = ws + (size_t)a.B * a.N_v * r.NT;
  r.err = a.err;
  // one CTA per SM when the tiles do not fill the GPU (deeper ring), else two
  // the MMA reads 128 A rows (16 KiB) from the start of a stage: the last
  // stage keeps that much room even when R + NT rows are fewer
  const size_t st_bytes = (size_t)(r.R + r.NT) * 128;
  const size_t tail = st_bytes > (size_t)kABytes ? 0 : (size_t)kABytes - st_bytes;
  const size_t budget = ((long long)a.B * r.n_vt <= num_sms ? kSmemMax - 1024 : 110 * 1024 - 1024) - tail;
  int ns = (int)(budget / st_bytes);
  r.n_stages = ns > kRelMaxStages ? kRelMaxStages : (ns < 2 ? 2 : ns);
  const size_t smem = (size_t)r.n_stages * st_bytes + tail + 1024;
  CUtensorMap mapV, mapT;
  if (make_tmap_bf16_2d(&mapV, a.emb_v, (uint64_t)a.B * a.N_v, (uint64_t)a.D, (uint64_t)a.D * 2, (uint32_t)r.R) ||
      make_tmap_bf16_2d(&mapT, a.emb_t, (uint64_t)a.B * a.N_t_max, (uint64_t)a.D, (uint64_t)a.D * 2,
                        (uint32_t)r.NT))
    return cudaErrorInvalidValue;
  e = launch_pdl(relevance_fused_tc, dim3(r.n_vt, a.B), dim3(kThreads), smem, s, r, mapV, mapT);
  if (e != cudaSuccess) return e;
  if (mask_ready != nullptr) {
    e = cudaStreamWaitEvent(s, mask_ready, 0);  // the first kernel that reads the mask
    if (e != cudaSuccess) return e;
  }
  relevance_finish_kernel<<<dim3((a.N_v + 8 * kRelFinishRows - 1) / (8 * kRelFinishRows), a.B), 256, 0, s>>>(
      r, a.text_len, mask, p);
  return cudaGetLastError();
}

}  // namespace provip

namespace provip {

bool crit_gram_tc_supported(const SimArgs& a) { return crit_splits(a.N_t_max, a.D, a.dtype) > 0; }

// K parts of the text Gram: 0 when the tcgen05 form does not apply; every part
// owns ceil(n_k / parts) slices of 64 (the last one possibly fewer)
int crit_splits(int N_t_max, int D, int dtype) {
  if (dtype != 1 || N_t_max > kBM || D % 8) return 0;
  const int n_k = (D + kBK - 1) / kBK;
  const int ns = n_k < kCritMaxSplits ? n_k : kCritMaxSplits;
  const int per = (n_k + ns - 1) / ns;
  return (n_k + per - 1) / per;
}

cudaError_t crit_gram_tc_launch(const SimArgs& a, float* G, cudaStream_t s) {
  static std::atomic<bool> smem_set[64];  // per device, zero-initialised
  int dev = 0;
  cudaGetDevice(&dev);
  const size_t smem = Cfg<kCritBN>::kStagesBytes + 1024;
  cudaError_t e = set_smem(crit_gram_tc, smem, &smem_set[dev < 64 ? dev : 0]);
  if (e != cudaSuccess) return e;
  CUtensorMap mapT;
  if (make_tmap_bf16_2d(&mapT, a.emb_t, (uint64_t)a.B * a.N_t_max, (uint64_t)a.D, (uint64_t)a.D * 2, 128))
    return cudaErrorInvalidValue;
  const int parts = crit_splits(a.N_t_max, a.D, a.dtype);
  const int n_k = (a.D + kBK - 1) / kBK, per = (n_k + parts - 1) / parts;
  crit_gram_tc<<<dim3(parts, 1, a.B), kThreads, smem, s>>>(mapT, a.text_len, a.N_t_max, a.D, a.B, per, G,
                                                          a.err);
  return cudaGetLastError();
}

}  // namespace provip
