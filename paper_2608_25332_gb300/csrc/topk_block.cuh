// Block-wide top-k of one sample held in shared memory (Sec. 4.3 top N1, Sec.
// 4.4 top N2): ties broken toward the lower index, indices in ascending order.
// Used by the top-k kernel. Any block size that is a multiple of 32 (<= 1024) works.
//
// keys[0..N) are order-preserving uint32 keys (float_key). An 8-bit MSD radix
// select (4 passes of a 256-bin shared histogram, one increment per group of
// lanes with the same digit) finds the exact key T of the k-th largest and how
// many keys equal to T are taken (need_eq); one block scan of packed
// (greater, equal) counts in index order then gives every selected element its
// slot #(greater before i) + min(#(equal before i), need_eq).
#pragma once

#include "common.cuh"

namespace provip {

struct TopkShared {
  int hist[256];
  uint32_t warp_tot[32];
  uint32_t prefix;
  int rem;
};

// exclusive block scan of one uint32 per thread
__device__ __forceinline__ uint32_t topk_block_exclusive_scan(uint32_t v, uint32_t* warp_tot) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  uint32_t incl = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += y;
  }
  if (lane == 31) warp_tot[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    const uint32_t t = lane < nw ? warp_tot[lane] : 0u;
    uint32_t ti = t;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, ti, o);
      if (lane >= o) ti += y;
    }
    warp_tot[lane] = ti - t;
  }
  __syncthreads();
  const uint32_t r = warp_tot[warp] + incl - v;
  __syncthreads();  // warp_tot may be reused by the caller
  return r;
}

// one shared-histogram increment per group of lanes holding the same digit
// (scores share their leading bytes, so plain per-lane atomics would serialise)
__device__ __forceinline__ void topk_hist_add(int* hist, uint32_t digit, bool active) {
  const unsigned act = __ballot_sync(0xffffffffu, active);
  if (!active) return;
  const unsigned peers = __match_any_sync(act, digit);
  if ((threadIdx.x & 31) == __ffs(peers) - 1) atomicAdd(&hist[digit], __popc(peers));
}

// Selects the k largest of keys[0..N) (shared memory) into out[0..k).
// Must be called by every thread of the block; keys must be visible (synced).
__device__ __forceinline__ void topk_block_select(const uint32_t* keys, int N, int k, int* out,
                                                  TopkShared& sh) {
  const int tid = threadIdx.x, nth = blockDim.x;
  uint32_t prefix = 0, pmask = 0;
  int rem = k;
  const int iters = (N + nth - 1) / nth;
  for (int shift = 24; shift >= 0; shift -= 8) {
    for (int q = tid; q < 256; q += nth) sh.hist[q] = 0;
    __syncthreads();
    for (int it = 0; it < iters; ++it) {
      const int i = it * nth + tid;
      const uint32_t u = i < N ? keys[i] : 0u;
      topk_hist_add(sh.hist, (u >> shift) & 255u, i < N && (u & pmask) == prefix);
    }
    __syncthreads();
    if (tid < 32) {
      const int lane = tid;
      int c[8], tot = 0;
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        c[q] = sh.hist[255 - 8 * lane - q];
        tot += c[q];
      }
      int incl = tot;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
      }
      const int excl = incl - tot;
      if (excl < rem && rem <= incl) {
        int cum = excl;
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          if (cum + c[q] >= rem) {
            sh.prefix = prefix | ((uint32_t)(255 - 8 * lane - q) << shift);
            sh.rem = rem - cum;
            break;
          }
          cum += c[q];
        }
      }
    }
    __syncthreads();
    prefix = sh.prefix;
    rem = sh.rem;
    pmask |= 255u << shift;
    __syncthreads();
  }
  const uint32_t T = prefix;
  const int need_eq = rem;
  const int ipt = (N + nth - 1) / nth;
  const int beg = min(N, tid * ipt), end = min(N, beg + ipt);
  uint32_t gt = 0, eq = 0;
  for (int i = beg; i < end; ++i) {
    const uint32_t u = keys[i];
    gt += u > T;
    eq += u == T;
  }
  const uint32_t base = topk_block_exclusive_scan((gt << 16) | eq, sh.warp_tot);
  uint32_t gtb = base >> 16, eqb = base & 0xffffu;
  for (int i = beg; i < end; ++i) {
    const uint32_t u = keys[i];
    if (u > T) {
      out[gtb + min(eqb, (uint32_t)need_eq)] = i;
      ++gtb;
    } else if (u == T) {
      if (eqb < (uint32_t)need_eq) out[gtb + eqb] = i;
      ++eqb;
    }
  }
}

// v_i = (sum over u of partial[row(u)][i], in order) / div: the head-score
// reduction shared by every path, so all of them give identical bits. Without
// a head subset, row(u) = u for u < n_part; with one (sel, n_sel positions in a
// head list of H_sel, in shared memory), row(u) = (u / n_sel) * H_sel +
// sel[u % n_sel] for u < (n_part / H_sel) * n_sel: the same rows, in the same
// order, as a head list made of the subset alone.
// Loads keys[i] and optionally writes the scores. cg: read through L2 only
// (the partials were written by other CTAs of a still-running grid).
template <bool CG>
__device__ __forceinline__ void topk_load_partials(const float* P0, int n_part, int N, float div,
                                                   bool zero, float* scores_out, uint32_t* keys,
                                                   const int* sel = nullptr, int n_sel = 0,
                                                   int H_sel = 1) {
  const int tid = threadIdx.x, nth = blockDim.x;
  const int n_sum = sel ? (n_part / H_sel) * n_sel : n_part;
  auto row = [&](int u) -> int { return sel ? (u / n_sel) * H_sel + sel[u % n_sel] : u; };
  auto ld = [&](size_t off) -> float { return CG ? __ldcg(P0 + off) : __ldg(P0 + off); };
  if (n_sum <= 8) {
    // up to 8 partial rows: 4 columns per thread, every load issued first
    int ro[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) ro[u] = u < n_sum ? row(u) * N : 0;
    for (int i0 = 0; i0 < N; i0 += 4 * nth) {
      float t[4][8];
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const int i = i0 + c * nth + tid;
#pragma unroll
        for (int u = 0; u < 8; ++u)
          if (u < n_sum && i < N) t[c][u] = ld((size_t)ro[u] + i);
      }
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const int i = i0 + c * nth + tid;
        if (i >= N) continue;
        float s = 0.f;
#pragma unroll
        for (int u = 0; u < 8; ++u)
          if (u < n_sum) s += t[c][u];
        const float v = zero ? 0.f : s / div;
        if (scores_out) scores_out[i] = v;
        keys[i] = float_key(v);
      }
    }
  } else {
    // more rows: 4 columns per thread, groups of 8 rows with the 32 loads of a
    // group issued first, each column's sum taken in row order
    for (int i0 = 0; i0 < N; i0 += 4 * nth) {
      float s[4] = {0.f, 0.f, 0.f, 0.f};
      for (int u0 = 0; u0 < n_sum; u0 += 8) {
        int ro[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) ro[u] = u0 + u < n_sum ? row(u0 + u) * N : 0;
        float t[4][8];
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          const int i = i0 + c * nth + tid;
#pragma unroll
          for (int u = 0; u < 8; ++u) t[c][u] = (u0 + u < n_sum && i < N) ? ld((size_t)ro[u] + i) : 0.f;
        }
#pragma unroll
        for (int c = 0; c < 4; ++c)
#pragma unroll
          for (int u = 0; u < 8; ++u)
            if (u0 + u < n_sum) s[c] += t[c][u];
      }
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const int i = i0 + c * nth + tid;
        if (i >= N) continue;
        const float v = zero ? 0.f : s[c] / div;
        if (scores_out) scores_out[i] = v;
        keys[i] = float_key(v);
      }
    }
  }
}

}  // namespace provip
