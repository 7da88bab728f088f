// Block-wide top-k of one sample held in shared memory (Sec. 4.3 top N1, Sec.
// 4.4 top N2): ties broken toward the lower index, indices in ascending order.
// Used by the top-k kernel. Any block size that is a multiple of 32 (<= 1024) works.
//
// keys[0..N) are order-preserving uint32 keys (float_key). The select narrows
// an inclusive key range [lo, hi] that holds the k-th largest key, starting
// from the block's min and max. Each pass takes the 11 bits of the keys below
// the leading bits that lo and hi share (a digit: every key of the range maps
// to one of at most 2048 bins, and at least half of the bins span the range),
// builds a shared histogram of the digits, and one warp finds the bin that
// holds the k-th largest key; the range becomes that bin's keys. A range of
// one key value ends the search, and so does a bin of at most kSmallCand keys:
// they are gathered and ranked exactly by (key, lower index first), a warp per
// 32 of them. Spread-out keys take one pass; a 32-bit range needs at most three.
// The threshold key T and how many keys equal to T are taken (need_eq) then
// give every selected element its output slot, #(greater before i) +
// min(#(equal before i), need_eq), from counts of (greater, equal) in index
// order scanned within warps and then across them. The same count gives, when
// asked for, the merge's index (Sec. 4.3): kpos[i] = the slot of a selected i,
// else -1, and the unselected elements in ascending order, pruned[i - slot].
#pragma once

#include "common.cuh"
#include "kernels.h"

namespace provip {

constexpr int kSelectBins = 2048;  // one 11-bit digit
constexpr int kSmallCand = 128;  // at most a warp per 32 candidates: blocks of >= 128 threads

struct TopkShared {
  __align__(16) int hist[2][kSelectBins];  // double-buffered: the next pass's is cleared during this one
  uint32_t wmin[32], wmax[32];
  uint32_t wcnt[32];         // packed (greater << 16 | equal) counts per warp
  int sel, above, cnt;       // chosen bin, keys above it in the range, keys in it
  int ncand;
  uint32_t rkey;             // the candidates' threshold key and the equal keys taken
  int rneed;
  __align__(16) uint32_t ckey[kSmallCand];
  __align__(16) int cidx[kSmallCand];
};

// Min and max of the block's keys. Every thread passes its own partial min and
// max; the result is valid in every thread after the call (one barrier).
__device__ __forceinline__ void topk_block_range(uint32_t mn, uint32_t mx, TopkShared& sh,
                                                 uint32_t& lo, uint32_t& hi) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    mn = min(mn, __shfl_xor_sync(0xffffffffu, mn, o));
    mx = max(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  }
  if (lane == 0) {
    sh.wmin[warp] = mn;
    sh.wmax[warp] = mx;
  }
  __syncthreads();
  mn = lane < nw ? sh.wmin[lane] : 0xffffffffu;
  mx = lane < nw ? sh.wmax[lane] : 0u;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    mn = min(mn, __shfl_xor_sync(0xffffffffu, mn, o));
    mx = max(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  }
  lo = mn;
  hi = mx;
}

// In descending bin order over hist[0..kSelectBins) (bins past the digit's
// range are zero), the bin where the count from the top first reaches rem:
// writes sh.sel, sh.above (keys in higher bins) and sh.cnt (keys in the bin).
// Every thread sums a segment of BPT consecutive bins (16-byte loads), a block
// scan of the segment counts finds the segment that holds the bin, and its
// thread walks it. Called by every thread; two barriers.
__device__ __forceinline__ void topk_block_find_bin(const int* hist, int rem, TopkShared& sh) {
  const int tid = threadIdx.x, nth = blockDim.x, lane = tid & 31, warp = tid >> 5;
  // bins per thread: 4, 8 or 16 (blocks of at least 128 threads)
  const int bpt = nth >= kSelectBins / 4 ? 4 : (nth >= kSelectBins / 8 ? 8 : 16);
  const int top = kSelectBins - tid * bpt;  // this thread's bins are [top - bpt, top)
  int h[16];
  int tot = 0;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    if (q * 4 < bpt && top - q * 4 - 4 >= 0) {
      const int4 v = *reinterpret_cast<const int4*>(hist + top - q * 4 - 4);
      h[q * 4 + 0] = v.w;  // descending: the highest bin first
      h[q * 4 + 1] = v.z;
      h[q * 4 + 2] = v.y;
      h[q * 4 + 3] = v.x;
    } else {
      h[q * 4 + 0] = h[q * 4 + 1] = h[q * 4 + 2] = h[q * 4 + 3] = 0;
    }
    tot += (h[q * 4 + 0] + h[q * 4 + 1]) + (h[q * 4 + 2] + h[q * 4 + 3]);
  }
  int incl = tot;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += y;
  }
  if (lane == 31) sh.wcnt[warp] = (uint32_t)incl;
  __syncthreads();
  int before = lane < warp ? (int)sh.wcnt[lane] : 0;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) before += __shfl_xor_sync(0xffffffffu, before, o);
  const int excl = before + incl - tot;
  if (excl < rem && rem <= excl + tot) {
    int cum = excl;
#pragma unroll
    for (int q = 0; q < 16; ++q) {
      if (q < bpt && cum + h[q] >= rem) {
        sh.sel = top - 1 - q;
        sh.above = cum;
        sh.cnt = h[q];
        break;
      }
      cum += h[q];
    }
  }
  __syncthreads();
}

// Exact rank of the rem-th largest of the nc <= kSmallCand candidates (key,
// index) in shared memory: the threshold key T and how many keys equal to T
// are taken. Warp w ranks candidates 32w..32w+31 against all of them (16-byte
// broadcast loads); the warp holding the candidate of rank rem - 1 (exactly one
// has it, 1 <= rem <= nc) counts the candidates above its key and publishes
// both. Called by every thread of a block of at least kSmallCand threads; one
// barrier.
__device__ __forceinline__ void topk_block_rank(TopkShared& sh, int nc, int rem, uint32_t& T,
                                                int& need_eq) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (warp * 32 < nc) {  // warp-uniform
    const int c = warp * 32 + lane;
    const uint32_t ku = c < nc ? sh.ckey[c] : 0u;
    const int ki = c < nc ? sh.cidx[c] : 0x7fffffff;
    int rank = 0;
    const int nq = (nc + 3) >> 2;
    for (int q = 0; q < nq; ++q) {
      const uint4 kv = reinterpret_cast<const uint4*>(sh.ckey)[q];
      const int4 iv = reinterpret_cast<const int4*>(sh.cidx)[q];
      // branch-free: (j < nc) & (key_j > key or (key_j == key and idx_j < idx))
      rank += (int)((4 * q + 0 < nc) & ((kv.x > ku) | ((kv.x == ku) & (iv.x < ki))));
      rank += (int)((4 * q + 1 < nc) & ((kv.y > ku) | ((kv.y == ku) & (iv.y < ki))));
      rank += (int)((4 * q + 2 < nc) & ((kv.z > ku) | ((kv.z == ku) & (iv.z < ki))));
      rank += (int)((4 * q + 3 < nc) & ((kv.w > ku) | ((kv.w == ku) & (iv.w < ki))));
    }
    const unsigned hit = __ballot_sync(0xffffffffu, c < nc && rank == rem - 1);
    if (hit) {
      const uint32_t t = __shfl_sync(0xffffffffu, ku, __ffs(hit) - 1);
      int gt = 0;
      for (int j = lane; j < nc; j += 32) gt += sh.ckey[j] > t ? 1 : 0;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) gt += __shfl_xor_sync(0xffffffffu, gt, o);
      if (lane == 0) {
        sh.rkey = t;
        sh.rneed = rem - gt;
      }
    }
  }
  __syncthreads();
  T = sh.rkey;
  need_eq = sh.rneed;
}

// Selects the k largest of keys[0..N) (shared memory) into out[0..k), given the
// keys' min lo and max hi. Must be called by every thread of the block; keys
// and sh.hist[0] (cleared) must be visible (synced).
__device__ __forceinline__ void topk_block_select(const uint32_t* keys, int N, int k, uint32_t lo,
                                                  uint32_t hi, int* out, TopkShared& sh, int* kpos = nullptr,
                                                  int* pruned = nullptr) {
  const int tid = threadIdx.x, nth = blockDim.x, lane = tid & 31, warp = tid >> 5;
  int rem = k;  // keys still to take from [lo, hi]
  int buf = 0;
  uint32_t T = lo;
  int need_eq = rem;
  for (int pass = 0; pass < 4; ++pass) {  // three passes at most (see above)
    if (lo == hi) {  // one key value left: take rem of it
      T = lo;
      need_eq = rem;
      break;
    }
    const int hb = 31 - __clz(lo ^ hi);  // highest bit where lo and hi differ
    const int shift = hb > 10 ? hb - 10 : 0;
    const uint32_t base = lo >> shift;  // digits (key >> shift) - base < kSelectBins
    int* hist = sh.hist[buf];
    for (int q = tid; q < kSelectBins; q += nth) sh.hist[buf ^ 1][q] = 0;
    for (int i = tid; i < N; i += nth) {
      const uint32_t u = keys[i];
      if (u >= lo && u <= hi) atomicAdd(&hist[(u >> shift) - base], 1);
    }
    if (tid == 0) sh.ncand = 0;
    __syncthreads();
    topk_block_find_bin(hist, rem, sh);
    const uint32_t b0 = (base + (uint32_t)sh.sel) << shift;  // <= hi
    const int cnt = sh.cnt;
    rem -= sh.above;
    lo = max(lo, b0);
    hi = min(hi, b0 + ((1u << shift) - 1u));
    buf ^= 1;
    if (lo != hi && cnt <= kSmallCand) {
      // few candidates: gather them and rank them exactly in one warp
      for (int i = tid; i < N; i += nth) {
        const uint32_t u = keys[i];
        if (u >= lo && u <= hi) {
          const int p = atomicAdd(&sh.ncand, 1);
          if (p < kSmallCand) {
            sh.ckey[p] = u;
            sh.cidx[p] = i;
          }
        }
      }
      __syncthreads();
      topk_block_rank(sh, min(sh.ncand, kSmallCand), rem, T, need_eq);
      break;
    }
  }
  // output slots in index order: thread t owns the keys [t * ipt, t * ipt + ipt)
  const int ipt = (N + nth - 1) / nth;
  const int beg = min(N, tid * ipt), end = min(N, beg + ipt);
  uint32_t cnt = 0;  // greater << 16 | equal (N <= 65535)
  for (int i = beg; i < end; ++i) {
    const uint32_t u = keys[i];
    cnt += (u > T ? 0x10000u : 0u) + (u == T ? 1u : 0u);
  }
  uint32_t incl = cnt;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += y;
  }
  if (lane == 31) sh.wcnt[warp] = incl;
  __syncthreads();
  uint32_t before = lane < warp ? sh.wcnt[lane] : 0u;  // the lower warps' totals
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) before += __shfl_xor_sync(0xffffffffu, before, o);
  const uint32_t slot = before + incl - cnt;
  uint32_t gtb = slot >> 16, eqb = slot & 0xffffu;
  for (int i = beg; i < end; ++i) {
    const uint32_t u = keys[i];
    const uint32_t before_i = gtb + min(eqb, (uint32_t)need_eq);  // elements kept before i
    bool kept = false;
    if (u > T) {
      kept = true;
      ++gtb;
    } else if (u == T) {
      kept = eqb < (uint32_t)need_eq;
      ++eqb;
    }
    if (kept) out[before_i] = i;
    if (kpos != nullptr) {
      kpos[i] = kept ? (int)before_i : -1;
      if (!kept) pruned[i - (int)before_i] = i;
    }
  }
}

// The select of topk_block_select on keys held in registers: thread t owns the
// KPT keys of indices [t * KPT, t * KPT + KPT) (valid below N), so every
// per-key loop is unrolled and its loads and atomics are in flight together.
// sh.hist[0] must be cleared and visible; lo/hi are the keys' min and max.
template <int KPT, bool kIndex = false>
__device__ __forceinline__ void topk_block_select_reg(const uint32_t (&key)[KPT], int N, int k,
                                                      uint32_t lo, uint32_t hi, int* out,
                                                      TopkShared& sh, int* kpos = nullptr,
                                                      int* pruned = nullptr) {
  const int tid = threadIdx.x, nth = blockDim.x, lane = tid & 31, warp = tid >> 5;
  const int i0 = tid * KPT;
  int rem = k;
  int buf = 0;
  uint32_t T = lo;
  int need_eq = rem;
  for (int pass = 0; pass < 4; ++pass) {
    if (lo == hi) {
      T = lo;
      need_eq = rem;
      break;
    }
    const int hb = 31 - __clz(lo ^ hi);
    const int shift = hb > 10 ? hb - 10 : 0;
    const uint32_t base = lo >> shift;
    int* hist = sh.hist[buf];
    for (int q = tid; q < kSelectBins; q += nth) sh.hist[buf ^ 1][q] = 0;
#pragma unroll
    for (int c = 0; c < KPT; ++c)
      if (i0 + c < N && key[c] >= lo && key[c] <= hi) atomicAdd(&hist[(key[c] >> shift) - base], 1);
    if (tid == 0) sh.ncand = 0;
    __syncthreads();
    topk_block_find_bin(hist, rem, sh);
    const uint32_t b0 = (base + (uint32_t)sh.sel) << shift;
    const int cnt = sh.cnt;
    rem -= sh.above;
    lo = max(lo, b0);
    hi = min(hi, b0 + ((1u << shift) - 1u));
    buf ^= 1;
    if (lo != hi && cnt <= kSmallCand) {
#pragma unroll
      for (int c = 0; c < KPT; ++c)
        if (i0 + c < N && key[c] >= lo && key[c] <= hi) {
          const int p = atomicAdd(&sh.ncand, 1);
          if (p < kSmallCand) {
            sh.ckey[p] = key[c];
            sh.cidx[p] = i0 + c;
          }
        }
      __syncthreads();
      topk_block_rank(sh, min(sh.ncand, kSmallCand), rem, T, need_eq);
      break;
    }
  }
  uint32_t cnt = 0;  // greater << 16 | equal
#pragma unroll
  for (int c = 0; c < KPT; ++c)
    if (i0 + c < N) cnt += (key[c] > T ? 0x10000u : 0u) + (key[c] == T ? 1u : 0u);
  uint32_t incl = cnt;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += y;
  }
  if (lane == 31) sh.wcnt[warp] = incl;
  __syncthreads();
  uint32_t before = lane < warp ? sh.wcnt[lane] : 0u;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) before += __shfl_xor_sync(0xffffffffu, before, o);
  const uint32_t slot = before + incl - cnt;
  uint32_t gtb = slot >> 16, eqb = slot & 0xffffu;
  if constexpr (kIndex) {
#pragma unroll
    for (int c = 0; c < KPT; ++c) {
      if (i0 + c >= N) continue;
      const uint32_t before_i = gtb + min(eqb, (uint32_t)need_eq);  // elements kept before i0 + c
      bool kept = false;
      if (key[c] > T) {
        kept = true;
        ++gtb;
      } else if (key[c] == T) {
        kept = eqb < (uint32_t)need_eq;
        ++eqb;
      }
      if (kept) out[before_i] = i0 + c;
      kpos[i0 + c] = kept ? (int)before_i : -1;
      if (!kept) pruned[i0 + c - (int)before_i] = i0 + c;
    }
  } else {
#pragma unroll
    for (int c = 0; c < KPT; ++c) {
      if (i0 + c >= N) continue;
      if (key[c] > T) {
        out[gtb + min(eqb, (uint32_t)need_eq)] = i0 + c;
        ++gtb;
      } else if (key[c] == T) {
        if (eqb < (uint32_t)need_eq) out[gtb + eqb] = i0 + c;
        ++eqb;
      }
    }
  }
}

// v_i = (sum over u of partial[row(u)][i], in order) / div: the head-score
// reduction shared by every path, so all of them give identical bits. Without
// a head subset, row(u) = u for u < n_part; with one (sel, n_sel positions in a
// head list of H_sel, in shared memory), row(u) = (u / n_sel) * H_sel +
// sel[u % n_sel] for u < (n_part / H_sel) * n_sel: the same rows, in the same
// order, as a head list made of the subset alone.
// Writes keys[i] (and optionally the scores) and returns the thread's min and
// max key. Every load of a group of columns is issued before the first sum.
__device__ __forceinline__ void topk_load_partials(const float* P0, int n_part, int N, float div,
                                                   bool zero, float* scores_out, uint32_t* keys,
                                                   uint32_t& mn, uint32_t& mx,
                                                   const int* sel = nullptr, int n_sel = 0,
                                                   int H_sel = 1) {
  const int tid = threadIdx.x, nth = blockDim.x;
  const int n_sum = sel ? (n_part / H_sel) * n_sel : n_part;
  auto row = [&](int u) -> int { return sel ? (u / n_sel) * H_sel + sel[u % n_sel] : u; };
  auto finish = [&](int i, float s) {
    const float v = zero ? 0.f : s / div;
    if (scores_out) scores_out[i] = v;
    const uint32_t key = float_key(v);
    keys[i] = key;
    mn = min(mn, key);
    mx = max(mx, key);
  };
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
          if (u < n_sum && i < N) t[c][u] = __ldg(P0 + (size_t)ro[u] + i);
      }
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const int i = i0 + c * nth + tid;
        if (i >= N) continue;
        float s = 0.f;
#pragma unroll
        for (int u = 0; u < 8; ++u)
          if (u < n_sum) s += t[c][u];
        finish(i, s);
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
          for (int u = 0; u < 8; ++u)
            t[c][u] = (u0 + u < n_sum && i < N) ? __ldg(P0 + (size_t)ro[u] + i) : 0.f;
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
        if (i < N) finish(i, s[c]);
      }
    }
  }
}

// keys[i] = float_key(scores[i]) (and optionally a copy of the scores), eight
// loads per thread issued before their keys are written; returns the thread's
// min and max key
__device__ __forceinline__ void topk_load_scores(const float* src, int N, float* scores_out,
                                                 uint32_t* keys, uint32_t& mn, uint32_t& mx) {
  const int tid = threadIdx.x, nth = blockDim.x;
  for (int i0 = 0; i0 < N; i0 += 8 * nth) {
    float v[8];
#pragma unroll
    for (int c = 0; c < 8; ++c) {
      const int i = i0 + c * nth + tid;
      v[c] = i < N ? __ldg(src + i) : 0.f;
    }
#pragma unroll
    for (int c = 0; c < 8; ++c) {
      const int i = i0 + c * nth + tid;
      if (i < N) {
        if (scores_out) scores_out[i] = v[c];
        const uint32_t key = float_key(v[c]);
        keys[i] = key;
        mn = min(mn, key);
        mx = max(mx, key);
      }
    }
  }
}

// Row count of sample b for the score division: the valid text rows, counted
// by the whole block (a block barrier inside).
__device__ __forceinline__ int block_count_rows(const TopkArgs& a, int b) {
  __shared__ int cnt;
  if (threadIdx.x == 0) cnt = 0;
  __syncthreads();
  const int tl = a.text_len[b];
  int mine = 0;
  for (int j = threadIdx.x; j < a.N_t_max; j += blockDim.x)
    mine += (j < tl) && (a.row_mask == nullptr || a.row_mask[(size_t)b * a.N_t_max + j] != 0);
  if (mine) atomicAdd(&cnt, mine);
  __syncthreads();
  return cnt;
}

// Thread t's KPT keys (indices t * KPT + c, c < KPT; 0 past N) from the scores
// or the head partials (the same sums, in the same order, as
// load_sample_keys), with the thread's min and max key. Every load of a group
// of partial rows is issued before the first sum.
template <int KPT>
__device__ __forceinline__ void load_keys_reg(const TopkArgs& a, int b, uint32_t (&key)[KPT],
                                              uint32_t& mn, uint32_t& mx) {
  const int N = a.N, i0 = threadIdx.x * KPT;
  float v[KPT];
  if (a.partial != nullptr) {
    __shared__ int sel[kMaxHeads];
    int nrows;
    if (a.row_mask == nullptr && a.sel == nullptr) {
      nrows = min(max(a.text_len[b], 0), a.N_t_max);
    } else {
      if (a.sel != nullptr)
        for (int q = threadIdx.x; q < a.n_sel; q += blockDim.x) sel[q] = a.sel[(size_t)b * a.n_sel + q];
      nrows = block_count_rows(a, b);  // synchronises the block (sel is visible after it)
    }
    const int n_sum = a.sel != nullptr ? (a.n_part / a.H_sel) * a.n_sel : a.n_part;
    const float div = (float)(a.sel != nullptr ? a.n_sel : a.H_sel) * (float)nrows;
    const float* P0 = a.partial + (size_t)b * a.n_part * N;
    // N % 4 == 0 and an aligned base: every row and every thread's columns start
    // on 16 bytes, and a group of 4 columns lies wholly below N or wholly past it
    const bool vec = (N & 3) == 0 && (reinterpret_cast<uintptr_t>(P0) & 15u) == 0;
    constexpr int G = KPT >= 16 ? 2 : 32 / KPT;  // rows per group: 32 to 64 loads in flight
    float s[KPT];
#pragma unroll
    for (int c = 0; c < KPT; ++c) s[c] = 0.f;
    for (int u0 = 0; u0 < n_sum; u0 += G) {
      int ro[G];
#pragma unroll
      for (int u = 0; u < G; ++u) {
        const int uu = u0 + u;
        ro[u] = uu < n_sum ? (a.sel != nullptr ? (uu / a.n_sel) * a.H_sel + sel[uu % a.n_sel] : uu) * N : 0;
      }
      float t[KPT][G];
      if (vec) {
        // 16-byte loads of the thread's KPT consecutive columns
#pragma unroll
        for (int u = 0; u < G; ++u)
#pragma unroll
          for (int c4 = 0; c4 < KPT / 4; ++c4) {
            float4 f = make_float4(0.f, 0.f, 0.f, 0.f);
            if (u0 + u < n_sum && i0 + 4 * c4 < N)
              f = __ldg(reinterpret_cast<const float4*>(P0 + (size_t)ro[u] + i0) + c4);
            t[4 * c4 + 0][u] = f.x;
            t[4 * c4 + 1][u] = f.y;
            t[4 * c4 + 2][u] = f.z;
            t[4 * c4 + 3][u] = f.w;
          }
      } else {
#pragma unroll
        for (int c = 0; c < KPT; ++c)
#pragma unroll
          for (int u = 0; u < G; ++u)
            t[c][u] = (u0 + u < n_sum && i0 + c < N) ? __ldg(P0 + (size_t)ro[u] + i0 + c) : 0.f;
      }
#pragma unroll
      for (int c = 0; c < KPT; ++c)
#pragma unroll
        for (int u = 0; u < G; ++u)
          if (u0 + u < n_sum) s[c] += t[c][u];
    }
#pragma unroll
    for (int c = 0; c < KPT; ++c) v[c] = nrows <= 0 ? 0.f : s[c] / div;
  } else {
    const float* src = a.scores + (size_t)b * N;
    if ((N & 3) == 0 && (reinterpret_cast<uintptr_t>(src) & 15u) == 0) {
#pragma unroll
      for (int c4 = 0; c4 < KPT / 4; ++c4) {
        float4 f = make_float4(0.f, 0.f, 0.f, 0.f);
        if (i0 + 4 * c4 < N) f = __ldg(reinterpret_cast<const float4*>(src + i0) + c4);
        v[4 * c4 + 0] = f.x;
        v[4 * c4 + 1] = f.y;
        v[4 * c4 + 2] = f.z;
        v[4 * c4 + 3] = f.w;
      }
    } else {
#pragma unroll
      for (int c = 0; c < KPT; ++c) v[c] = i0 + c < N ? __ldg(src + i0 + c) : 0.f;
    }
  }
  float* so = a.scores_out ? a.scores_out + (size_t)b * N : nullptr;
  mn = 0xffffffffu;
  mx = 0u;
#pragma unroll
  for (int c = 0; c < KPT; ++c) {
    key[c] = 0u;
    if (i0 + c < N) {
      if (so) so[i0 + c] = v[c];
      key[c] = float_key(v[c]);
      mn = min(mn, key[c]);
      mx = max(mx, key[c]);
    }
  }
}

}  // namespace provip
