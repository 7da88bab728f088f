// Per-sample top-k kernel (Sec. 4.3 top N1 of p, Sec. 4.4 top N2 of v): one CTA
// per sample (about 4 keys per thread, 128 to 1024 threads), the N scores held
// in shared memory as order-preserving keys, selected by topk_block_select
// (topk_block.cuh): ties to the lower index, ascending output.
//
// When fed head partials (the in-LLM path), the kernel first sums them per
// column in a fixed order and divides by (heads x valid text rows): the same
// arithmetic as the stand-alone score reduction, so both give identical bits.
// With a per-sample head subset (the visual heads picked by their confidence)
// only the subset's partials are summed, in head-list order.
#include "common.cuh"
#include "kernels.h"
#include "topk_block.cuh"

namespace provip {
namespace {

constexpr int kTopkMaxThreads = 1024;

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

__global__ void __launch_bounds__(kTopkMaxThreads) topk_kernel(const TopkArgs a) {
  extern __shared__ uint32_t keys[];
  __shared__ TopkShared sh;
  // launched as a programmatic dependent: wait until the kernel that writes the
  // scores has completed (which, for overlapped calls, implies the previous
  // compaction has completed too)
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int b = blockIdx.x;
  const int N = a.N;
  float* so = a.scores_out ? a.scores_out + (size_t)b * N : nullptr;
  if (a.partial != nullptr) {
    __shared__ int sel[kMaxHeads];
    if (a.sel != nullptr)
      for (int q = threadIdx.x; q < a.n_sel; q += blockDim.x) sel[q] = a.sel[(size_t)b * a.n_sel + q];
    const int nrows = block_count_rows(a, b);  // synchronises the block
    const float nh = (float)(a.sel != nullptr ? a.n_sel : a.H_sel);
    topk_load_partials<false>(a.partial + (size_t)b * a.n_part * N, a.n_part, N, nh * (float)nrows,
                              nrows <= 0, so, keys, a.sel != nullptr ? sel : nullptr, a.n_sel,
                              a.H_sel);
  } else {
    for (int i = threadIdx.x; i < N; i += blockDim.x) {
      const float v = a.scores[(size_t)b * N + i];
      if (so) so[i] = v;
      keys[i] = float_key(v);
    }
  }
  __syncthreads();
  // The scores are in shared memory now: the next kernel (the compaction, and
  // through it the next call's head scores, which rewrite the partials) may
  // start. idx is only read by the compaction after this grid completes.
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  topk_block_select(keys, N, a.k, a.idx_out + (size_t)b * a.k, sh);
}

}  // namespace

cudaError_t topk_launch(const TopkArgs& a, cudaStream_t s, bool pdl) {
  static bool configured[64] = {false};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64 && !configured[dev]) {
    cudaError_t e = cudaFuncSetAttribute(topk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         kTopkMaxN * (int)sizeof(uint32_t));
    if (e != cudaSuccess) return e;
    configured[dev] = true;
  }
  // about 4 keys per thread, at least 128 and at most 1024 threads
  int threads = ((a.N + 3) / 4 + 31) / 32 * 32;
  threads = threads < 128 ? 128 : (threads > kTopkMaxThreads ? kTopkMaxThreads : threads);
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  cfg.gridDim = dim3((unsigned)a.B);
  cfg.blockDim = dim3((unsigned)threads);
  cfg.dynamicSmemBytes = (size_t)a.N * sizeof(uint32_t);
  cfg.stream = s;
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, topk_kernel, a);
}

}  // namespace provip
