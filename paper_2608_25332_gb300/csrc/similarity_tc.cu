// Pre-LLM pass (Sec. 4.3) on 5th-generation tensor cores (bf16).
//
// merge_argmax_tc: the pruned x kept cosine Gram fused with the row argmax.
//   A = the pruned visual rows of a 128-row M tile, B = the kept rows of a range
//   of 256-row N tiles, read as contiguous tiles of a per-sample copy of E_v
//   permuted to [pruned | kept] by one bandwidth-bound gather pass. The
//   epilogue scales a column by 1/|e_k| and keeps, per row, the running (max,
//   first index) over the kept positions in ascending order, so ties go to the
//   lower kept position. The (N_v - N1) x N1 matrix never leaves the SM.
// relevance_tc: the text x visual cosine Gram fused with the de-meaned column
//   max: p_j = max_{i in T} (<t_i, v_j> / |t_i| / |v_j| - mu_i) for a 128-column
//   block of visual rows (A = the <= 128 text rows of the sample, B = 128
//   consecutive visual rows), the max over rows taken with a warp butterfly and
//   a fixed-order combine of the four epilogue warps.
#include "common.cuh"
#include "kernels.h"
#include "tc_gemm.cuh"

namespace provip {
namespace {

using namespace tcg;

// pruned[b][0..N_v - keep): the visual rows not in keep, ascending (kpos < 0)
__global__ void __launch_bounds__(1024) pruned_list_kernel(const int* kpos, int N_v, int* pruned,
                                                            int n_pruned) {
  __shared__ int warp_tot[32];
  const int b = blockIdx.x;
  const int* kp = kpos + (size_t)b * N_v;
  int* out = pruned + (size_t)b * n_pruned;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  int base = 0;
  for (int j0 = 0; j0 < N_v; j0 += blockDim.x) {
    const int j = j0 + threadIdx.x;
    const bool pr = j < N_v && kp[j] < 0;
    const unsigned bal = __ballot_sync(0xffffffffu, pr);
    if (lane == 0) warp_tot[warp] = __popc(bal);
    __syncthreads();
    int off = 0, tot = 0;
    for (int w = 0; w < nw; ++w) {
      off += w < warp ? warp_tot[w] : 0;
      tot += warp_tot[w];
    }
    const int pos = base + off + __popc(bal & ((1u << lane) - 1u));
    if (pr && pos < n_pruned) out[pos] = j;
    base += tot;
    __syncthreads();
  }
}

// perm[b] = rows of E_v[b] reordered as [pruned rows (ascending) | kept rows
// (keep order)], so that the Gram reads both operands as contiguous tiles.
// One warp per output row, 16-byte vectors.
__global__ void __launch_bounds__(256) gather_perm_kernel(const __nv_bfloat16* E, const int* pruned,
                                                          const int* keep_idx, int n_pruned, int keep,
                                                          int N_v, int D, __nv_bfloat16* perm,
                                                          unsigned* err) {
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
  for (int v = lane; v < nvec; v += 32) dst[v] = __ldg(src + v);
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

__global__ void __launch_bounds__(kThreads, 1)
    merge_argmax_tc(const MergeTcArgs a, const __grid_constant__ CUtensorMap mapE) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ Pipe pipe;
  __shared__ int sidx_a[kBM];
  const int b = blockIdx.z, split = blockIdx.y;
  const int m0 = blockIdx.x * kBM;
  const int n_tiles_all = (a.keep + kMergeBN - 1) / kMergeBN;
  const int t0 = (int)((long long)n_tiles_all * split / a.n_split);
  const int t1 = (int)((long long)n_tiles_all * (split + 1) / a.n_split);
  const int n_tiles = t1 - t0;
  const int a0 = t0 * kMergeBN;                       // first kept position of the range
  const int n_keep = min(a.keep, t1 * kMergeBN) - a0;  // kept rows in the range
  const int n_k = (a.D + kBK - 1) / kBK;

  const uint32_t sbase = smem_u32(smem_raw);
  uint8_t* stages = smem_raw + (((sbase + 1023u) & ~1023u) - sbase);
  int* sidx_b = reinterpret_cast<int*>(stages + Cfg<kMergeBN>::kStagesBytes);
  float* skinv = reinterpret_cast<float*>(sidx_b + kMergeMaxKeep);

  const int* pr = a.pruned + (size_t)b * a.n_pruned;
  const int* kp = a.keep_idx + (size_t)b * a.keep;
  for (int r = threadIdx.x; r < kBM; r += blockDim.x) sidx_a[r] = m0 + r < a.n_pruned ? pr[m0 + r] : 0;
  for (int q = threadIdx.x; q < n_keep; q += blockDim.x) {
    int j = kp[a0 + q];
    if (j < 0 || j >= a.N_v) {
      set_error(a.err, kErrBadDeviceArg);
      j = 0;
    }
    sidx_b[q] = j;
    skinv[q] = a.inv_v[(size_t)b * a.N_v + j];
  }
  if (threadIdx.x == 0) {
    prefetch_tmap(&mapE);
    pipe_init(pipe);
  }
  if (threadIdx.x < 32) {
    tmem_alloc(&pipe.tmem, Cfg<kMergeBN>::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (n_tiles > 0) {
    if (warp == 0) {
      if (lane == 0) {
        // operands are contiguous rows of the permuted copy: [pruned | kept]
        RowSrc ra{nullptr, b * a.N_v + m0, kBM};
        RowSrc rb{nullptr, b * a.N_v + a.n_pruned + a0, n_tiles * kMergeBN};
        producer<kMergeBN>(pipe, stages, &mapE, &mapE, ra, false, rb, false, n_tiles, n_k, a.err);
      }
    } else if (warp == 1) {
      if (lane == 0) mma_issuer<kMergeBN>(pipe, stages, n_tiles, n_k, a.err);
    } else {
      // epilogue: row r of the M tile, running (max, first index) over the range
      const int quad = warp & 3;
      const int r = quad * 32 + lane;
      const bool rv = m0 + r < a.n_pruned;
      float best = -INFINITY;
      int bidx = 0x7fffffff;
      for (int t = 0; t < n_tiles; ++t) {
        const int buf = t & 1;
        mbar_wait(&pipe.acc_full[buf], (uint32_t)(t >> 1) & 1u, a.err);
        tc_fence_after();
        const uint32_t taddr = pipe.tmem + ((uint32_t)(quad * 32) << 16) + (uint32_t)(buf * kMergeBN);
#pragma unroll 1
        for (int cb = 0; cb < kMergeBN / 32; ++cb) {
          float v[32];
          tmem_ld32(taddr + cb * 32, v);
          tc_wait_ld();
          const int q0 = t * kMergeBN + cb * 32;  // position within the range
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const int q = q0 + i;
            if (q < n_keep) {
              const float x = v[i] * skinv[q];
              if (x > best) {
                best = x;
                bidx = a0 + q;
              }
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&pipe.acc_empty[buf]);
      }
      if (rv && !pipe.fail) {
        const size_t o = ((size_t)split * a.B + b) * a.N_v + sidx_a[r];
        a.ws_best[o] = best;
        a.ws_bidx[o] = bidx;
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x < 32) tmem_dealloc(pipe.tmem, Cfg<kMergeBN>::kTmemCols);
}

struct RelTcArgs {
  int B, N_v, D, N_t_max;
  const int* text_len;
  const uint8_t* mask;  // [B][N_t_max]
  const float* inv_v;   // [B][N_v]
  const float* mu;      // [B][N_t_max]
  const float* invt;    // [B][N_t_max]
  float* p;             // [B][N_v]
  unsigned* err;
};

constexpr int kRelBN = 128;

__global__ void __launch_bounds__(kThreads, 1)
    relevance_tc(const RelTcArgs a, const __grid_constant__ CUtensorMap mapT,
                 const __grid_constant__ CUtensorMap mapV) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ Pipe pipe;
  __shared__ float red[4][kRelBN];
  const int b = blockIdx.z;
  const int n0 = blockIdx.x * kRelBN;
  const int n_k = (a.D + kBK - 1) / kBK;
  const uint32_t sbase = smem_u32(smem_raw);
  uint8_t* stages = smem_raw + (((sbase + 1023u) & ~1023u) - sbase);
  if (threadIdx.x == 0) {
    prefetch_tmap(&mapT);
    prefetch_tmap(&mapV);
    pipe_init(pipe);
  }
  if (threadIdx.x < 32) {
    tmem_alloc(&pipe.tmem, Cfg<kRelBN>::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (warp == 0) {
    if (lane == 0) {
      RowSrc ra{nullptr, b * a.N_t_max, kBM};
      RowSrc rb{nullptr, b * a.N_v + n0, kRelBN};
      producer<kRelBN>(pipe, stages, &mapT, &mapV, ra, false, rb, false, 1, n_k, a.err);
    }
  } else if (warp == 1) {
    if (lane == 0) mma_issuer<kRelBN>(pipe, stages, 1, n_k, a.err);
  } else {
    const int quad = warp & 3;
    const int r = quad * 32 + lane;
    const int tl = min(max(a.text_len[b], 0), a.N_t_max);
    const bool rv = r < tl && a.mask[(size_t)b * a.N_t_max + r] != 0;
    const float it = rv ? a.invt[(size_t)b * a.N_t_max + r] : 0.f;
    const float m = rv ? a.mu[(size_t)b * a.N_t_max + r] : 0.f;
    mbar_wait(&pipe.acc_full[0], 0, a.err);
    tc_fence_after();
    const uint32_t taddr = pipe.tmem + ((uint32_t)(quad * 32) << 16);
#pragma unroll 1
    for (int cb = 0; cb < kRelBN / 32; ++cb) {
      float v[32];
      tmem_ld32(taddr + cb * 32, v);
      tc_wait_ld();
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        const int j = n0 + cb * 32 + i;
        const float iv = j < a.N_v ? a.inv_v[(size_t)b * a.N_v + j] : 0.f;
        v[i] = rv ? v[i] * it * iv - m : -INFINITY;
      }
      // butterfly max over the 32 rows of the warp: lane ends with column `lane`
#pragma unroll
      for (int sh = 16; sh >= 1; sh >>= 1) {
        const bool upper = (lane & sh) != 0;
#pragma unroll
        for (int i = 0; i < sh; ++i) {
          const float keep = upper ? v[i + sh] : v[i];
          const float send = upper ? v[i] : v[i + sh];
          v[i] = fmaxf(keep, __shfl_xor_sync(0xffffffffu, send, sh));
        }
      }
      red[quad][cb * 32 + lane] = v[0];
    }
    tc_fence_before();
    // combine the four lane quadrants (epilogue warps only: named barrier)
    asm volatile("bar.sync 1, 128;" ::: "memory");
    const int c = threadIdx.x - 64;
    const int j = n0 + c;
    if (j < a.N_v && !pipe.fail)
      a.p[(size_t)b * a.N_v + j] = fmaxf(fmaxf(red[0][c], red[1][c]), fmaxf(red[2][c], red[3][c]));
  }
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x < 32) tmem_dealloc(pipe.tmem, Cfg<kRelBN>::kTmemCols);
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
      RowSrc ra{nullptr, b * N_t_max, kBM};
      RowSrc rb{nullptr, b * N_t_max, kCritBN};
      producer<kCritBN>(pipe, stages, &mapT, &mapT, ra, false, rb, false, 1, n_k, err, k0);
    }
  } else if (warp == 1) {
    if (lane == 0) mma_issuer<kCritBN>(pipe, stages, 1, n_k, err);
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
cudaError_t set_smem(K kernel, size_t bytes, bool* done) {
  if (*done) return cudaSuccess;
  cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
  if (e == cudaSuccess) *done = true;
  return e;
}

}  // namespace

size_t merge_tc_smem() {
  return Cfg<kMergeBN>::kStagesBytes + 1024 + (size_t)kMergeMaxKeep * (sizeof(int) + sizeof(float));
}

int merge_tc_split(int B, int N_v, int keep, int num_sms) {
  const int m_tiles = B * ((N_v - keep + kBM - 1) / kBM);
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
                                   const int* kpos, int* pruned, void* perm, int n_split,
                                   float* ws_best, int* ws_bidx, cudaStream_t s) {
  static bool smem_set[64] = {false};
  int dev = 0;
  cudaGetDevice(&dev);
  const size_t smem = merge_tc_smem();
  cudaError_t e = set_smem(merge_argmax_tc, smem, &smem_set[dev < 64 ? dev : 0]);
  if (e != cudaSuccess) return e;
  const int n_pruned = a.N_v - keep;
  pruned_list_kernel<<<a.B, 1024, 0, s>>>(kpos, a.N_v, pruned, n_pruned);
  dim3 gg((a.N_v + 7) / 8, a.B);
  gather_perm_kernel<<<gg, 256, 0, s>>>(static_cast<const __nv_bfloat16*>(a.emb_v), pruned, keep_idx,
                                        n_pruned, keep, a.N_v, a.D, static_cast<__nv_bfloat16*>(perm),
                                        a.err);
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
  dim3 grid((n_pruned + kBM - 1) / kBM, n_split, a.B);
  merge_argmax_tc<<<grid, kThreads, smem, s>>>(m, mapE);
  return cudaGetLastError();
}

bool relevance_tc_supported(const SimArgs& a) { return a.dtype == 1 && a.N_t_max <= kBM && a.D % 8 == 0; }

cudaError_t relevance_tc_launch(const SimArgs& a, const uint8_t* mask, const float* inv_v,
                                const float* mu, const float* invt, float* p, cudaStream_t s) {
  static bool smem_set[64] = {false};
  int dev = 0;
  cudaGetDevice(&dev);
  const size_t smem = Cfg<kRelBN>::kStagesBytes + 1024;
  cudaError_t e = set_smem(relevance_tc, smem, &smem_set[dev < 64 ? dev : 0]);
  if (e != cudaSuccess) return e;
  CUtensorMap mapT, mapV;
  if (make_tmap_bf16_2d(&mapT, a.emb_t, (uint64_t)a.B * a.N_t_max, (uint64_t)a.D, (uint64_t)a.D * 2, 128) ||
      make_tmap_bf16_2d(&mapV, a.emb_v, (uint64_t)a.B * a.N_v, (uint64_t)a.D, (uint64_t)a.D * 2, 128))
    return cudaErrorInvalidValue;
  RelTcArgs r;
  r.B = a.B;
  r.N_v = a.N_v;
  r.D = a.D;
  r.N_t_max = a.N_t_max;
  r.text_len = a.text_len;
  r.mask = mask;
  r.inv_v = inv_v;
  r.mu = mu;
  r.invt = invt;
  r.p = p;
  r.err = a.err;
  dim3 grid((a.N_v + kRelBN - 1) / kRelBN, 1, a.B);
  relevance_tc<<<grid, kThreads, smem, s>>>(r, mapT, mapV);
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
  static bool smem_set[64] = {false};
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
