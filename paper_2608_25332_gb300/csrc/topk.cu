// Per-sample top-k kernels (Sec. 4.3 top N1 of p, Sec. 4.4 top N2 of v): ties
// to the lower index, ascending output. Up to 512 scores: exact ranks in a
// cluster of CTAs per sample (topk_rank_kernel, built for latency). Larger N:
// one CTA per sample selecting on order-preserving keys (topk_block.cuh: a
// digit histogram over the keys' actual range, usually one pass, then exact
// ranks of the few candidates left) - up to 16384 keys held in registers, 4 to
// 32 per thread (topk_reg_kernel), more in shared memory (topk_kernel).
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

// keys[0..N) of sample b (and, when so is set, the scores) from the scores or
// the head partials, with the thread's min and max key; every thread of the
// block takes part. The keys are visible to the block after its next barrier.
__device__ __forceinline__ void load_sample_keys(const TopkArgs& a, int b, uint32_t* keys, float* so,
                                                 uint32_t& mn, uint32_t& mx) {
  const int N = a.N;
  mn = 0xffffffffu;
  mx = 0u;
  if (a.partial != nullptr) {
    __shared__ int sel[kMaxHeads];
    int nrows;
    if (a.row_mask == nullptr && a.sel == nullptr) {
      // every text row counts: no block-wide count needed
      nrows = min(max(a.text_len[b], 0), a.N_t_max);
    } else {
      if (a.sel != nullptr)
        for (int q = threadIdx.x; q < a.n_sel; q += blockDim.x) sel[q] = a.sel[(size_t)b * a.n_sel + q];
      nrows = block_count_rows(a, b);  // synchronises the block (sel is visible after it)
    }
    const float nh = (float)(a.sel != nullptr ? a.n_sel : a.H_sel);
    topk_load_partials(a.partial + (size_t)b * a.n_part * N, a.n_part, N, nh * (float)nrows, nrows <= 0, so,
                       keys, mn, mx, a.sel != nullptr ? sel : nullptr, a.n_sel, a.H_sel);
  } else {
    topk_load_scores(a.scores + (size_t)b * N, N, so, keys, mn, mx);
  }
}

__global__ void __launch_bounds__(kTopkMaxThreads) topk_kernel(const TopkArgs a) {
  extern __shared__ uint32_t keys[];
  __shared__ TopkShared sh;
  for (int q = threadIdx.x; q < kSelectBins; q += blockDim.x) sh.hist[0][q] = 0;
  // launched as a programmatic dependent: wait until the kernel that writes the
  // scores has completed (which, for overlapped calls, implies the previous
  // compaction has completed too)
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int b = blockIdx.x;
  uint32_t mn, mx, lo, hi;
  load_sample_keys(a, b, keys, a.scores_out ? a.scores_out + (size_t)b * a.N : nullptr, mn, mx);
  topk_block_range(mn, mx, sh, lo, hi);  // its barrier also publishes the keys and the cleared histogram
  // The scores are in shared memory now: the next kernel (the compaction, and
  // through it the next call's head scores, which rewrite the partials) may
  // start. idx is only read by the compaction after this grid completes.
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  topk_block_select(keys, a.N, a.k, lo, hi, a.idx_out + (size_t)b * a.k, sh,
                    a.kpos_out ? a.kpos_out + (size_t)b * a.N : nullptr,
                    a.kpos_out ? a.pruned_out + (size_t)b * (a.N - a.k) : nullptr);
}

// Up to 16384 keys: they stay in registers, 4 to 32 per thread (at most 512
// threads, so a thread may hold 128 registers), thread t owning the contiguous
// indices [t * KPT, t * KPT + KPT).
constexpr int kRegMaxThreads = 512;
// kIndex: also write the merge's index (kpos_out, pruned_out), a separate
// instantiation so that the plain selection carries none of that code
template <int KPT, bool kIndex>
__global__ void __launch_bounds__(kRegMaxThreads) topk_reg_kernel(const TopkArgs a) {
  __shared__ TopkShared sh;
  // the histogram is cleared while the kernel that writes the scores finishes
  for (int q = threadIdx.x; q < kSelectBins; q += blockDim.x) sh.hist[0][q] = 0;
  // a programmatic dependent: wait for that kernel
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int b = blockIdx.x;
  uint32_t key[KPT], mn, mx, lo, hi;
  load_keys_reg<KPT>(a, b, key, mn, mx);
  topk_block_range(mn, mx, sh, lo, hi);  // its barrier also publishes the cleared histogram
  // the scores are consumed: the next kernel may start (it waits for this
  // grid's completion before reading idx)
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  topk_block_select_reg<KPT, kIndex>(key, a.N, a.k, lo, hi, a.idx_out + (size_t)b * a.k, sh,
                                     kIndex ? a.kpos_out + (size_t)b * a.N : nullptr,
                                     kIndex ? a.pruned_out + (size_t)b * (a.N - a.k) : nullptr);
}

// Small N (<= kRankUseMaxN): selection by exact ranks, for latency. A cluster of
// ceil(N / 128) CTAs per sample; each CTA builds all N keys (the same
// arithmetic in every CTA), and each thread ranks one element against all of
// them: rank(i) = #{j : key_j > key_i, or key_j == key_i and j < i}, counted on
// 64-bit composites (key << 32 | ~j), so the k elements of rank < k are the k
// largest with ties to the lower index. Output positions: ballots inside a
// warp, warp counts inside the CTA, and the counts of the lower-ranked CTAs of
// the cluster read through distributed shared memory.
constexpr int kRankThreads = 128;
#ifndef PROVIP_TOPK_RANK_MAX_N
#define PROVIP_TOPK_RANK_MAX_N 512
#endif
constexpr int kRankMaxN = 1024;  // clusters of at most 8 CTAs (portable)
constexpr int kRankUseMaxN = PROVIP_TOPK_RANK_MAX_N;  // largest N sent to the rank kernel

__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\t"
               "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ int ld_peer_i32(const int* local, uint32_t rank) {
  uint32_t raddr;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(raddr) : "r"(smem_u32(local)), "r"(rank));
  int v;
  asm volatile("ld.shared::cluster.s32 %0, [%1];" : "=r"(v) : "r"(raddr) : "memory");
  return v;
}

__global__ void __launch_bounds__(kRankThreads) topk_rank_kernel(const TopkArgs a) {
  __shared__ uint32_t keys[kRankMaxN];
  __shared__ __align__(16) unsigned long long ck[kRankMaxN];
  __shared__ int warp_cnt[kRankThreads / 32];
  __shared__ int cta_cnt;
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const uint32_t crank = cluster_ctarank();
  const int b = blockIdx.y, N = a.N;
  // one CTA of the cluster writes the scores
  uint32_t mn, mx;
  load_sample_keys(a, b, keys, (a.scores_out && crank == 0) ? a.scores_out + (size_t)b * N : nullptr, mn, mx);
  __syncthreads();
  for (int j = threadIdx.x; j < N; j += kRankThreads)
    ck[j] = ((unsigned long long)keys[j] << 32) | (unsigned long long)(~(uint32_t)j);
  __syncthreads();
  // the scores are consumed: the next kernel may start (it waits for this grid
  // to complete before reading idx)
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int i = (int)crank * kRankThreads + threadIdx.x;
  bool sel = false;
  if (i < N) {
    const unsigned long long mine = ck[i];
    int c0 = 0, c1 = 0, c2 = 0, c3 = 0;
    const ulonglong2* v = reinterpret_cast<const ulonglong2*>(ck);
    int q = 0;
    for (; q + 1 < N / 2; q += 2) {
      const ulonglong2 p0 = v[q], p1 = v[q + 1];
      c0 += p0.x > mine;
      c1 += p0.y > mine;
      c2 += p1.x > mine;
      c3 += p1.y > mine;
    }
    for (int j = 2 * q; j < N; ++j) c0 += ck[j] > mine;
    sel = (c0 + c1) + (c2 + c3) < a.k;
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const unsigned bal = __ballot_sync(0xffffffffu, sel);
  if (lane == 0) warp_cnt[warp] = __popc(bal);
  __syncthreads();
  int before = 0, total = 0;
#pragma unroll
  for (int w = 0; w < kRankThreads / 32; ++w) {
    before += w < warp ? warp_cnt[w] : 0;
    total += warp_cnt[w];
  }
  if (threadIdx.x == 0) cta_cnt = total;
  cluster_sync_all();  // every CTA's count is visible
  int offset = 0;
  for (uint32_t r = 0; r < crank; ++r) offset += ld_peer_i32(&cta_cnt, r);
  if (sel) a.idx_out[(size_t)b * a.k + offset + before + __popc(bal & ((1u << lane) - 1u))] = i;
  cluster_sync_all();  // no CTA leaves while a peer may still read its count
}
}  // namespace

bool topk_writes_index(int N) { return !(N <= kRankUseMaxN && N <= kRankMaxN); }

cudaError_t topk_launch(const TopkArgs& a, cudaStream_t s, bool pdl) {
  static std::atomic<bool> configured[64];  // per device, zero-initialised
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
  if (a.N <= kRankUseMaxN && a.N <= kRankMaxN) {
    const int C = (a.N + kRankThreads - 1) / kRankThreads;
    cudaLaunchAttribute rattr[2];
    cfg.gridDim = dim3((unsigned)C, (unsigned)a.B);
    cfg.blockDim = dim3(kRankThreads);
    cfg.dynamicSmemBytes = 0;
    rattr[0].id = cudaLaunchAttributeClusterDimension;
    rattr[0].val.clusterDim.x = (unsigned)C;
    rattr[0].val.clusterDim.y = 1;
    rattr[0].val.clusterDim.z = 1;
    rattr[1] = attr[0];
    cfg.attrs = rattr;
    cfg.numAttrs = pdl ? 2 : 1;
    return cudaLaunchKernelEx(&cfg, topk_rank_kernel, a);
  }
  if (a.N <= 32 * kRegMaxThreads) {
    // keys in registers: 4, 8, 16 or 32 per thread, 128 to 512 threads
    const int kpt = a.N <= 4 * kRegMaxThreads ? 4
                    : (a.N <= 8 * kRegMaxThreads ? 8 : (a.N <= 16 * kRegMaxThreads ? 16 : 32));
    int nt = ((a.N + kpt - 1) / kpt + 31) / 32 * 32;
    cfg.blockDim = dim3((unsigned)(nt < 128 ? 128 : nt));
    cfg.dynamicSmemBytes = 0;
    if (a.kpos_out != nullptr) {
      if (kpt == 4) return cudaLaunchKernelEx(&cfg, topk_reg_kernel<4, true>, a);
      if (kpt == 8) return cudaLaunchKernelEx(&cfg, topk_reg_kernel<8, true>, a);
      if (kpt == 16) return cudaLaunchKernelEx(&cfg, topk_reg_kernel<16, true>, a);
      return cudaLaunchKernelEx(&cfg, topk_reg_kernel<32, true>, a);
    }
    if (kpt == 4) return cudaLaunchKernelEx(&cfg, topk_reg_kernel<4, false>, a);
    if (kpt == 8) return cudaLaunchKernelEx(&cfg, topk_reg_kernel<8, false>, a);
    if (kpt == 16) return cudaLaunchKernelEx(&cfg, topk_reg_kernel<16, false>, a);
    return cudaLaunchKernelEx(&cfg, topk_reg_kernel<32, false>, a);
  }
  return cudaLaunchKernelEx(&cfg, topk_kernel, a);
}

}  // namespace provip
