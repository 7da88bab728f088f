// Head-aware visual-token scores (Sec. 4.4) on 5th-generation tensor cores.
//
// Same two passes and workspace layout as the CUDA-core path (head_scores.cu),
// with 128-key chunks. One 128-thread CTA per (chunk, row block x head, sample):
//   - thread 0 loads the 128 x 128 bf16 text-query tile of the head and the
//     128 x 128 key tile of its key/value head with 2-D TMA (128-byte swizzle,
//     two 64-column boxes each; rows outside the tensor read as zero),
//   - then issues eight K = 16 tcgen05.mma (M = N = 128, bf16 -> fp32) that
//     write S = Q K^T into 128 TMEM columns, and commits to an mbarrier;
//   - each of the 128 threads owns one TMEM lane = one text row and reads its
//     128 logits with tcgen05.ld (32 columns at a time).
// Pass 1 keeps an online (max, sum of exp2) per row over the causal keys of the
// chunk. Pass 2 turns the visual logits into probabilities with the row's
// global (max, sum) and sums them over the 128 rows: a butterfly
// transpose-reduction inside each warp (31 shuffles per 32 columns) and a
// fixed-order sum over the 4 warps, so the result is deterministic. When asked,
// pass 2 also writes each row's mean and M2 over the chunk's visual
// probabilities (head confidence).
#include "common.cuh"
#include "kernels.h"

namespace provip {
namespace {

constexpr int kTcThreads = 128;
constexpr int kTile = 128;                  // rows of Q tile, keys of K tile
constexpr int kHalfBytes = kTile * 128;     // one 64-column box: 128 rows x 128 B
constexpr int kTileBytes = 2 * kHalfBytes;  // 32 KiB
constexpr size_t kTcSmem = 2 * kTileBytes + 1024;
constexpr uint32_t kIdesc = idesc_bf16_f32(128, 128);

struct TcSmemCtl {
  uint64_t tma_bar;
  uint64_t mma_bar;
  uint32_t tmem;
  int fail;
};

__device__ __forceinline__ bool row_valid(const HSArgs& a, int b, int j, int tl) {
  return j < tl && (a.row_mask == nullptr || a.row_mask[(size_t)b * a.N_t_max + j] != 0);
}

// Loads the Q tile (rows y_q..y_q+127, columns x_q..x_q+127) and the K tile
// (rows y_k.., columns x_k..), runs S = Q K^T into TMEM. Executed by thread 0.
// Returns false if a wait timed out.
__device__ __forceinline__ bool tc_qk(const CUtensorMap* tmQ, const CUtensorMap* tmK,
                                      uint8_t* qs, uint8_t* ks, TcSmemCtl* ctl, int x_q, int y_q,
                                      int x_k, int y_k, unsigned* err) {
  mbar_arrive_expect_tx(&ctl->tma_bar, 2 * kTileBytes);
  tma_load_2d(qs, tmQ, x_q, y_q, &ctl->tma_bar);
  tma_load_2d(qs + kHalfBytes, tmQ, x_q + 64, y_q, &ctl->tma_bar);
  tma_load_2d(ks, tmK, x_k, y_k, &ctl->tma_bar);
  tma_load_2d(ks + kHalfBytes, tmK, x_k + 64, y_k, &ctl->tma_bar);
  if (!mbar_wait(&ctl->tma_bar, 0, err)) {
    mbar_wait(&ctl->tma_bar, 0, err);  // give the copies in flight one more bounded chance
    return false;
  }
  tc_fence_after();
  const uint32_t qa = smem_u32(qs), ka = smem_u32(ks);
#pragma unroll
  for (int kstep = 0; kstep < 8; ++kstep) {
    const uint32_t off = (kstep >> 2) * kHalfBytes + (kstep & 3) * 32;
    tc_mma_bf16(ctl->tmem, smem_desc_sw128(qa + off), smem_desc_sw128(ka + off), kIdesc,
                kstep > 0 ? 1u : 0u);
  }
  tc_commit(&ctl->mma_bar);
  return true;
}

// common prologue: carve smem, init barriers, allocate 128 TMEM columns
__device__ __forceinline__ void tc_setup(uint8_t* raw, uint8_t*& qs, uint8_t*& ks, TcSmemCtl* ctl) {
  const uint32_t base = smem_u32(raw);
  const uint32_t pad = ((base + 1023u) & ~1023u) - base;
  qs = raw + pad;
  ks = qs + kTileBytes;
  if (threadIdx.x == 0) {
    mbar_init(&ctl->tma_bar, 1);
    mbar_init(&ctl->mma_bar, 1);
    ctl->fail = 0;
    fence_mbar_init();
  }
  __syncwarp();
  if (threadIdx.x < 32) {
    tmem_alloc(&ctl->tmem, kTile);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
}

__device__ __forceinline__ void tc_teardown(TcSmemCtl* ctl) {
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x < 32) tmem_dealloc(ctl->tmem, kTile);
}

// waits for the MMA (or the failure signal) and returns whether S is valid
__device__ __forceinline__ bool tc_wait_mma(TcSmemCtl* ctl, unsigned* err) {
  const bool ok = mbar_wait(&ctl->mma_bar, 0, err);
  tc_fence_after();
  return ok && ctl->fail == 0;
}

__global__ void __launch_bounds__(kTcThreads) hs_stats_tc(const HSArgs a,
                                                          const __grid_constant__ CUtensorMap tmQ,
                                                          const __grid_constant__ CUtensorMap tmK) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ TcSmemCtl ctl;
  uint8_t *qs, *ks;
  const int c = blockIdx.x;
  const int hi = blockIdx.y % a.H_sel, rb = blockIdx.y / a.H_sel;
  const int b = blockIdx.z;
  const int h = a.heads[hi], g = h / (a.H_q / a.H_kv);
  const int ts = a.text_start[b], sl = a.seq_len[b];
  int tl = a.text_len[b];
  const bool ok = ts >= 0 && tl >= 0 && tl <= a.N_t_max && sl <= a.L_max && ts + tl <= sl;
  if (!ok) tl = 0;
  if (threadIdx.x == 0) {
    prefetch_tmap(&tmQ);
    prefetch_tmap(&tmK);
  }
  tc_setup(smem_raw, qs, ks, &ctl);
  if (threadIdx.x == 0) {
    if (!ok && c == 0 && blockIdx.y == 0) set_error(a.err, kErrBadDeviceArg);
    const bool done = tc_qk(&tmQ, &tmK, qs, ks, &ctl, h * kHeadDim,
                            b * a.L_max + ts + rb * kTile, g * kHeadDim, b * a.L_max + c * kTile,
                            a.err);
    if (!done) {
      ctl.fail = 1;
      mbar_arrive(&ctl.mma_bar);
    }
  }
  __syncwarp();
  const bool good = tc_wait_mma(&ctl, a.err);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = warp * 32 + lane;
  const int j = rb * kTile + r;
  const bool rv = good && row_valid(a, b, j, tl);
  const int t = ts + j;
  const int k0 = c * kTile;
  float m = -INFINITY, l = 0.f;
#pragma unroll 1
  for (int cb = 0; cb < kTile / 32; ++cb) {
    float v[32];
    tmem_ld32(ctl.tmem + ((uint32_t)(warp * 32) << 16) + cb * 32, v);
    tc_wait_ld();
    float cm = -INFINITY;
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      const bool kv = rv && (k0 + cb * 32 + i) <= t;
      v[i] = kv ? v[i] * a.scale_log2 : -INFINITY;
      cm = fmaxf(cm, v[i]);
    }
    if (cm != -INFINITY) {
      const float mn = fmaxf(m, cm);
      float s = 0.f;
#pragma unroll
      for (int i = 0; i < 32; ++i) s += exp2f(v[i] - mn);  // exp2f(-inf) = 0
      l = l * exp2f(m - mn) + s;
      m = mn;
    }
  }
  a.stats[((((size_t)b * a.n_rb + rb) * a.H_sel + hi) * a.n_kc + c) * kTile + r] =
      rv ? make_float2(m, l) : make_float2(-INFINITY, 0.f);
  tc_teardown(&ctl);
}

__global__ void __launch_bounds__(kTcThreads) hs_probs_tc(const HSArgs a,
                                                          const __grid_constant__ CUtensorMap tmQ,
                                                          const __grid_constant__ CUtensorMap tmK) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ TcSmemCtl ctl;
  __shared__ float red[4][kTile];
  uint8_t *qs, *ks;
  const int vc = blockIdx.x;
  const int hi = blockIdx.y % a.H_sel, rb = blockIdx.y / a.H_sel;
  const int b = blockIdx.z;
  const int h = a.heads[hi], g = h / (a.H_q / a.H_kv);
  const int ts = a.text_start[b], sl = a.seq_len[b];
  int tl = a.text_len[b];
  const bool ok = ts >= 0 && tl >= 0 && tl <= a.N_t_max && sl <= a.L_max && ts + tl <= sl &&
                  a.vis_start + a.N_v <= sl;
  if (!ok) tl = 0;
  if (threadIdx.x == 0) {
    prefetch_tmap(&tmQ);
    prefetch_tmap(&tmK);
  }
  tc_setup(smem_raw, qs, ks, &ctl);
  if (threadIdx.x == 0) {
    const bool done = tc_qk(&tmQ, &tmK, qs, ks, &ctl, h * kHeadDim, b * a.L_max + ts + rb * kTile,
                            g * kHeadDim, b * a.L_max + a.vis_start + vc * kTile, a.err);
    if (!done) {
      ctl.fail = 1;
      mbar_arrive(&ctl.mma_bar);
    }
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = warp * 32 + lane;
  const int j = rb * kTile + r;
  bool rv = row_valid(a, b, j, tl);
  const int t = ts + j;
  // the row's global (max, 1/sum) from the chunk statistics of pass 1
  float m = -INFINITY, inv = 0.f;
  if (rv) {
    const float2* st = a.stats + (((size_t)b * a.n_rb + rb) * a.H_sel + hi) * a.n_kc * kTile + r;
    for (int c = 0; c < a.n_kc; ++c) m = fmaxf(m, st[(size_t)c * kTile].x);
    float l = 0.f;
    for (int c = 0; c < a.n_kc; ++c) {
      const float2 v = st[(size_t)c * kTile];
      if (v.x != -INFINITY) l += v.y * exp2f(v.x - m);
    }
    inv = l > 0.f ? 1.f / l : 0.f;
  }
  __syncwarp();
  const bool good = tc_wait_mma(&ctl, a.err);
  rv = rv && good;
  const int col0 = vc * kTile;
  // head confidence: the row's mean and M2 over this chunk's visual columns
  // (per 32-column block, merged pairwise: Chan, Golub and LeVeque's update)
  const bool conf = a.conf_part != nullptr;
  float cn = 0.f, cmean = 0.f, cm2 = 0.f;
#pragma unroll 1
  for (int cb = 0; cb < kTile / 32; ++cb) {
    float v[32];
    tmem_ld32(ctl.tmem + ((uint32_t)(warp * 32) << 16) + cb * 32, v);
    tc_wait_ld();
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      const int col = col0 + cb * 32 + i;
      const bool kv = rv && col < a.N_v && (a.vis_start + col) <= t;
      v[i] = kv ? exp2f(v[i] * a.scale_log2 - m) * inv : 0.f;
    }
    const int nbi = min(32, a.N_v - (col0 + cb * 32));
    if (conf && nbi > 0) {
      const float nb = (float)nbi;
      float s4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int i = 0; i < 32; ++i) s4[i & 3] += v[i];
      const float mb = ((s4[0] + s4[1]) + (s4[2] + s4[3])) / nb;
      float q4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        const float d = i < nbi ? v[i] - mb : 0.f;
        q4[i & 3] += d * d;
      }
      const float n = cn + nb, dl = mb - cmean;
      cmean += dl * (nb / n);
      cm2 += ((q4[0] + q4[1]) + (q4[2] + q4[3])) + dl * dl * (cn * nb / n);
      cn = n;
    }
    // butterfly transpose-reduction: lane ends with the column sum of column `lane`
#pragma unroll
    for (int w = 16; w >= 1; w >>= 1) {
      const bool upper = (lane & w) != 0;
#pragma unroll
      for (int i = 0; i < w; ++i) {
        const float keep = upper ? v[i + w] : v[i];
        const float send = upper ? v[i] : v[i + w];
        v[i] = keep + __shfl_xor_sync(0xffffffffu, send, w);
      }
    }
    red[warp][cb * 32 + lane] = v[0];
  }
  if (conf && rv && (a.conf_mask == nullptr || a.conf_mask[(size_t)b * a.N_t_max + j] != 0))
    a.conf_part[(((size_t)b * a.H_sel + hi) * a.N_t_max + j) * a.conf_stride + vc] =
        make_float2(cmean, cm2);
  __syncthreads();
  {
    const int col = col0 + threadIdx.x;
    const float s = red[0][threadIdx.x] + red[1][threadIdx.x] + red[2][threadIdx.x] + red[3][threadIdx.x];
    if (good && col < a.N_v)
      a.partial[((size_t)b * a.n_rb * a.H_sel + (size_t)rb * a.H_sel + hi) * a.N_v + col] = s;
  }
  tc_teardown(&ctl);
}

}  // namespace

cudaError_t hs_launch_tc(const HSArgs& a, const CUtensorMap* tmQ, const CUtensorMap* tmK,
                         cudaStream_t s, ConfGeom* geom) {
  if (geom) *geom = ConfGeom{a.vis_start, kTile, a.n_vc};
  static std::atomic<bool> configured[64];  // per device, zero-initialised
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64 && !configured[dev]) {
    cudaError_t e = cudaFuncSetAttribute(hs_stats_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kTcSmem);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(hs_probs_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kTcSmem);
    if (e != cudaSuccess) return e;
    configured[dev] = true;
  }
  dim3 g1(a.n_kc, a.H_sel * a.n_rb, a.B), g2(a.n_vc, a.H_sel * a.n_rb, a.B);
  hs_stats_tc<<<g1, kTcThreads, kTcSmem, s>>>(a, *tmQ, *tmK);
  hs_probs_tc<<<g2, kTcThreads, kTcSmem, s>>>(a, *tmQ, *tmK);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// tensor-map encoding through the driver entry point (no libcuda link needed)
// ---------------------------------------------------------------------------
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

int make_tmap_bf16_2d(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols,
                      uint64_t row_stride_bytes, uint32_t box_rows) {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess || !p)
      return -1;
    fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  const cuuint64_t gdim[2] = {cols, rows};
  const cuuint64_t gstride[1] = {row_stride_bytes};
  const cuuint32_t box[2] = {64, box_rows};
  const cuuint32_t estride[2] = {1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), gdim, gstride,
                  box, estride, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? 0 : -1;
}

}  // namespace provip
