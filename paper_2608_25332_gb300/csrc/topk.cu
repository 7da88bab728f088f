// Per-sample top-k with ties broken toward the lower index, indices written in
// ascending order (Sec. 4.3 top N1 of p, Sec. 4.4 top N2 of v).
//
// One 1024-thread CTA per sample; the N scores live in shared memory as
// order-preserving uint32 keys. An 8-bit MSD radix select (4 passes of a
// 256-bin shared histogram) finds the exact key T of the k-th largest score
// and how many keys equal to T must be taken (need_eq). One block-wide scan of
// packed (greater-than, equal) counts in index order then gives every selected
// element its output slot: #(greater before i) + min(#(equal before i), need_eq),
// which keeps the lowest-index ties and emits indices in ascending order.
//
// When fed head partials (the fused path), the kernel first sums them per
// column in a fixed order and divides by (heads x valid text rows): the same
// arithmetic as the stand-alone score reduction, so both give identical bits.
#include "common.cuh"
#include "kernels.h"

namespace provip {
namespace {

constexpr int kTopkThreads = 1024;

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

// exclusive block scan of one uint32 per thread (1024 threads)
__device__ __forceinline__ uint32_t block_exclusive_scan(uint32_t v, uint32_t* warp_tot) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t incl = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += y;
  }
  if (lane == 31) warp_tot[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    const uint32_t t = warp_tot[lane];
    uint32_t ti = t;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, ti, o);
      if (lane >= o) ti += y;
    }
    warp_tot[lane] = ti - t;
  }
  __syncthreads();
  return warp_tot[warp] + incl - v;
}

__global__ void __launch_bounds__(kTopkThreads) topk_kernel(const TopkArgs a) {
  extern __shared__ uint32_t keys[];
  __shared__ int hist[256];
  __shared__ uint32_t s_prefix;
  __shared__ int s_rem;
  __shared__ uint32_t warp_tot[32];
  const int b = blockIdx.x;
  const int N = a.N, k = a.k;
  const int tid = threadIdx.x;

  int nrows = 0;
  if (a.partial != nullptr) nrows = block_count_rows(a, b);
  for (int i = tid; i < N; i += kTopkThreads) {
    float v;
    if (a.partial != nullptr) {
      const float* p = a.partial + (size_t)b * a.n_part * N + i;
      float s = 0.f;
      for (int u = 0; u < a.n_part; ++u) s += p[(size_t)u * N];
      v = nrows > 0 ? s / ((float)a.H_sel * (float)nrows) : 0.f;
    } else {
      v = a.scores[(size_t)b * N + i];
    }
    if (a.scores_out) a.scores_out[(size_t)b * N + i] = v;
    keys[i] = float_key(v);
  }
  __syncthreads();

  // radix select of the k-th largest key, most significant byte first
  uint32_t prefix = 0, pmask = 0;
  int rem = k;
  for (int shift = 24; shift >= 0; shift -= 8) {
    if (tid < 256) hist[tid] = 0;
    __syncthreads();
    for (int i = tid; i < N; i += kTopkThreads) {
      const uint32_t u = keys[i];
      if ((u & pmask) == prefix) atomicAdd(&hist[(u >> shift) & 255u], 1);
    }
    __syncthreads();
    if (tid < 32) {
      const int lane = tid;
      int c[8], tot = 0;
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        c[q] = hist[255 - 8 * lane - q];
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
            s_prefix = prefix | ((uint32_t)(255 - 8 * lane - q) << shift);
            s_rem = rem - cum;
            break;
          }
          cum += c[q];
        }
      }
    }
    __syncthreads();
    prefix = s_prefix;
    rem = s_rem;
    pmask |= 255u << shift;
    __syncthreads();
  }
  const uint32_t T = prefix;
  const int need_eq = rem;

  // ordered selection: contiguous segment per thread, one packed scan
  const int ipt = (N + kTopkThreads - 1) / kTopkThreads;
  const int beg = min(N, tid * ipt), end = min(N, beg + ipt);
  uint32_t gt = 0, eq = 0;
  for (int i = beg; i < end; ++i) {
    const uint32_t u = keys[i];
    gt += u > T;
    eq += u == T;
  }
  const uint32_t base = block_exclusive_scan((gt << 16) | eq, warp_tot);
  uint32_t gtb = base >> 16, eqb = base & 0xffffu;
  int* out = a.idx_out + (size_t)b * k;
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

}  // namespace

cudaError_t topk_launch(const TopkArgs& a, cudaStream_t s) {
  static bool configured[64] = {false};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64 && !configured[dev]) {
    cudaError_t e = cudaFuncSetAttribute(topk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         kTopkMaxN * (int)sizeof(uint32_t));
    if (e != cudaSuccess) return e;
    configured[dev] = true;
  }
  topk_kernel<<<a.B, kTopkThreads, (size_t)a.N * sizeof(uint32_t), s>>>(a);
  return cudaGetLastError();
}

}  // namespace provip
