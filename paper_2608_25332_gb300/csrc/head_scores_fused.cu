// Head-aware visual-token scores (Sec. 4.4) in one pass over K: a cluster of
// CTAs per (row block x head, sample) on 5th-generation tensor cores.
//
// The keys 0..L_max are cut into 128-key chunks; CTA r of a cluster owns CPC
// consecutive chunks (CPC = 1, 2 or 4). Each CTA
//   1. loads the 128 x 128 bf16 text-query tile of its head and its CPC key
//      tiles with 2-D TMA (128-byte swizzle), and thread 0 issues 8 x CPC
//      tcgen05.mma (M = N = 128, K = 16) writing S = Q K^T into CPC x 128 TMEM
//      columns;
//   2. (thread = TMEM lane = text row; two warps per lane quadrant, each
//      taking half of the columns) sweeps its logits once, 32-column blocks at
//      a time, keeping a running max m and sum l over its causal keys;
//      e = exp2(s - mb) goes back into TMEM with tcgen05.st, mb being the
//      running max after that block (kept per block); the two halves' (m, l)
//      are combined in shared memory;
//   3. pushes its (m, l) of each row into every cluster CTA's shared memory
//      (remote stores into the key-tile region, free once every CTA's MMAs
//      are done: a split cluster barrier around pass 1 guarantees it), and
//      after one cluster barrier forms the row's global max M and sum L from
//      its own shared memory;
//   4. turns its visual columns into probabilities p = e * exp2(mb - M) / L and
//      sums them over the 128 rows (warp butterfly transpose-reduction, then a
//      fixed-order sum over the 4 warps) into partial[b][rb * H_sel + h][col];
//      the CONF variant also keeps, per row, the mean and M2 of its visual
//      probabilities (head confidence) and writes them per cluster rank;
//   5. frees its TMEM (no CTA touches another's shared memory after the
//      barrier of step 3).
// Every key is read from HBM once and every logit is exponentiated once; the
// attention matrix never leaves the SM. The host sizes the dynamic shared
// memory so that the CTAs an SM can hold never ask for more than its 512 TMEM
// columns (a tcgen05.alloc that has to wait inside a cluster could deadlock).
#include <mutex>

#include "common.cuh"
#include "kernels.h"

namespace provip {
namespace {

constexpr int kThreads = 256;  // 8 warps: two per TMEM lane quadrant, splitting the columns
constexpr int kTile = 128;
constexpr int kHalfBytes = kTile * 128;     // 64-column box: 128 rows x 128 B
constexpr int kTileBytes = 2 * kHalfBytes;  // 32 KiB
constexpr uint32_t kIdesc = idesc_bf16_f32(128, 128);

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cluster_size() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\t"
               "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_arrive_relaxed() {
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() {
  asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// lets a kernel launched as this grid's programmatic dependent start now
__device__ __forceinline__ void pdl_trigger() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
// stores v at the address of `local` in the shared memory of cluster CTA `rank`
__device__ __forceinline__ void st_peer_f2(float2* local, uint32_t rank, float2 v) {
  uint32_t raddr;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(raddr) : "r"(smem_u32(local)), "r"(rank));
  asm volatile("st.shared::cluster.v2.f32 [%0], {%1, %2};" ::"r"(raddr), "f"(v.x), "f"(v.y) : "memory");
}
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const float* v) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
      "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
      "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])),
      "r"(__float_as_uint(v[3])), "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])),
      "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])), "r"(__float_as_uint(v[8])),
      "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
      "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
      "r"(__float_as_uint(v[15])), "r"(__float_as_uint(v[16])), "r"(__float_as_uint(v[17])),
      "r"(__float_as_uint(v[18])), "r"(__float_as_uint(v[19])), "r"(__float_as_uint(v[20])),
      "r"(__float_as_uint(v[21])), "r"(__float_as_uint(v[22])), "r"(__float_as_uint(v[23])),
      "r"(__float_as_uint(v[24])), "r"(__float_as_uint(v[25])), "r"(__float_as_uint(v[26])),
      "r"(__float_as_uint(v[27])), "r"(__float_as_uint(v[28])), "r"(__float_as_uint(v[29])),
      "r"(__float_as_uint(v[30])), "r"(__float_as_uint(v[31]))
      : "memory");
}
__device__ __forceinline__ void tc_wait_st() {
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

struct Ctl {
  uint64_t tma_bar;
  uint64_t mma_bar;
  uint32_t tmem;
  int fail;
};

template <int CPC>
constexpr size_t smem_bytes() {
  return (size_t)(1 + CPC) * kTileBytes + 1024;
}

// CONF: also the head-confidence statistics of the visual probabilities
template <int CPC, bool CONF>
__global__ void __launch_bounds__(kThreads, CPC == 1 ? 3 : (CPC == 2 ? 2 : 1))
    hs_fused_tc(const HSArgs a,
                                                        const __grid_constant__ CUtensorMap tmQ,
                                                        const __grid_constant__ CUtensorMap tmK) {
  constexpr uint32_t kCols = CPC * kTile;  // 128, 256 or 512: a power of two
  extern __shared__ uint8_t smem_raw[];
  __shared__ Ctl ctl;
  __shared__ float2 halfstat[2][kTile];
  __shared__ float red[4][kCols];
  const uint32_t rank = cluster_rank(), nrank = cluster_size();
  const int hi = blockIdx.y % a.H_sel, rb = blockIdx.y / a.H_sel;
  const int b = blockIdx.z;
  const int h = a.heads[hi], g = h / (a.H_q / a.H_kv);
  const int ts = a.text_start[b], sl = a.seq_len[b];
  int tl = a.text_len[b];
  const bool ok = ts >= 0 && tl >= 0 && tl <= a.N_t_max && sl <= a.L_max && ts + tl <= sl &&
                  a.vis_start + a.N_v <= sl;
  if (!ok) tl = 0;
  const int key0 = (int)rank * CPC * kTile;  // first key of this CTA

  // shared memory: Q tile then CPC key tiles, 1024-byte aligned
  const uint32_t base = smem_u32(smem_raw);
  uint8_t* qs = smem_raw + (((base + 1023u) & ~1023u) - base);
  uint8_t* ks = qs + kTileBytes;
  pdl_trigger();  // a programmatic dependent (the top-k) may be scheduled now
  if (threadIdx.x == 0) {
    prefetch_tmap(&tmQ);
    prefetch_tmap(&tmK);
    mbar_init(&ctl.tma_bar, 1);
    mbar_init(&ctl.mma_bar, 1);
    ctl.fail = 0;
    fence_mbar_init();
    // the loads need no TMEM: issue them before the allocation
    mbar_arrive_expect_tx(&ctl.tma_bar, (uint32_t)(1 + CPC) * kTileBytes);
    const int yq = b * a.L_max + ts + rb * kTile, xq = h * kHeadDim;
    tma_load_2d(qs, &tmQ, xq, yq, &ctl.tma_bar);
    tma_load_2d(qs + kHalfBytes, &tmQ, xq + 64, yq, &ctl.tma_bar);
#pragma unroll
    for (int c = 0; c < CPC; ++c) {
      const int yk = b * a.L_max + key0 + c * kTile, xk = g * kHeadDim;
      tma_load_2d(ks + c * kTileBytes, &tmK, xk, yk, &ctl.tma_bar);
      tma_load_2d(ks + c * kTileBytes + kHalfBytes, &tmK, xk + 64, yk, &ctl.tma_bar);
    }
  }
  // warp 1 allocates the tensor memory while thread 0 issues the loads
  if (threadIdx.x >= 32 && threadIdx.x < 64) {
    tmem_alloc(&ctl.tmem, kCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();

  if (threadIdx.x == 0) {
    if (!ok && rank == 0 && blockIdx.y == 0) set_error(a.err, kErrBadDeviceArg);
    if (mbar_wait(&ctl.tma_bar, 0, a.err)) {
      tc_fence_after();
      const uint32_t qa = smem_u32(qs);
#pragma unroll
      for (int c = 0; c < CPC; ++c) {
        const uint32_t ka = smem_u32(ks + c * kTileBytes);
#pragma unroll
        for (int kstep = 0; kstep < 8; ++kstep) {
          const uint32_t off = (kstep >> 2) * kHalfBytes + (kstep & 3) * 32;
          tc_mma_bf16(ctl.tmem + c * kTile, smem_desc_sw128(qa + off), smem_desc_sw128(ka + off),
                      kIdesc, kstep > 0 ? 1u : 0u);
        }
      }
      tc_commit(&ctl.mma_bar);
    } else {
      mbar_wait(&ctl.tma_bar, 0, a.err);  // one more bounded wait for copies in flight
      ctl.fail = 1;
      mbar_arrive(&ctl.mma_bar);
    }
  }
  __syncwarp();
  const bool good = mbar_wait(&ctl.mma_bar, 0, a.err) && ctl.fail == 0;
  tc_fence_after();
  // this CTA's MMAs have read its Q and K tiles: from the matching wait on,
  // peers may write their row statistics into the key-tile region
  cluster_arrive_relaxed();

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int quad = warp & 3, half = warp >> 2;  // TMEM lanes 32*quad.., columns of this half
  const int r = quad * 32 + lane;
  const int j = rb * kTile + r;
  const bool rv = good && j < tl && (a.row_mask == nullptr || a.row_mask[(size_t)b * a.N_t_max + j] != 0);
  const int t = ts + j;
  constexpr int kHalfCols = (int)kCols / 2;
  constexpr int kBlocks = kHalfCols / 32;  // 32-column blocks per warp
  const int col0 = half * kHalfCols;        // first TMEM column of this warp
  const uint32_t tbase = ctl.tmem + ((uint32_t)(quad * 32) << 16) + (uint32_t)col0;
  const bool warp_live = __any_sync(0xffffffffu, rv);

  // pass 1, one sweep over this warp's logits, a 32-column block per TMEM
  // round trip: running max m and sum l over the causal keys; e = exp2(s - mb)
  // is stored back in TMEM with mb the running max after its block.
  float mblk[kBlocks];
  float m = -INFINITY, l = 0.f;
  const float sc = a.scale_log2;
  const int t_first = ts + rb * kTile;  // every row of the block sits at or after it
  if (warp_live) {
#pragma unroll
    for (int cb = 0; cb < kBlocks; ++cb) {
      float v[32];
      tmem_ld32(tbase + cb * 32, v);
      tc_wait_ld();
      const int k0 = key0 + col0 + cb * 32;
      float mn = m;
      if (rv) {
        // keys before the block's first row are causal for every row
        float bm = -INFINITY;
        if (k0 + 31 <= t_first) {
#pragma unroll
          for (int i = 0; i < 32; ++i) bm = fmaxf(bm, v[i]);
        } else {
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            v[i] = k0 + i <= t ? v[i] : -INFINITY;
            bm = fmaxf(bm, v[i]);
          }
        }
        mn = fmaxf(m, bm * sc);  // sc > 0: the max commutes with the scale
      }
      if (mn != -INFINITY) {
        float s4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          v[i] = ex2_approx(fmaf(v[i], sc, -mn));  // 2^-inf = 0 for masked keys
          s4[i & 3] += v[i];
        }
        l = l * ex2_approx(m - mn) + ((s4[0] + s4[1]) + (s4[2] + s4[3]));
      } else {
#pragma unroll
        for (int i = 0; i < 32; ++i) v[i] = 0.f;
      }
      m = mn;
      mblk[cb] = mn;
      tmem_st32(tbase + cb * 32, v);
    }
    tc_wait_st();
  }
  halfstat[half][r] = make_float2(rv ? m : -INFINITY, rv ? l : 0.f);
  __syncthreads();
  // every CTA of the cluster has finished its MMAs (and so has started): its
  // key-tile region may receive the row statistics of the whole cluster,
  // recv[rank][row] = that CTA's (max, sum) of the row over its keys
  float2* recv = reinterpret_cast<float2*>(ks);
  cluster_wait();
  if (half == 0) {
    // the CTA's (max, sum) of the row from its two column halves, pushed to
    // every CTA of the cluster (remote stores, made visible by the barrier)
    const float2 h0 = halfstat[0][r], h1 = halfstat[1][r];
    const float mm = fmaxf(h0.x, h1.x);
    float ll = 0.f;
    if (h0.x != -INFINITY) ll += h0.y * ex2_approx(h0.x - mm);
    if (h1.x != -INFINITY) ll += h1.y * ex2_approx(h1.x - mm);
    const float2 st = make_float2(mm, ll);
    for (uint32_t q = 0; q < nrank; ++q) st_peer_f2(&recv[rank * kTile + r], q, st);
  }
  cluster_sync_all();

  // global (max, sum) of the row over the cluster, from local shared memory
  float M = -INFINITY, L = 0.f;
  if (rv) {
    float2 st[16];
#pragma unroll
    for (uint32_t q = 0; q < 16; ++q)
      if (q < nrank) st[q] = recv[q * kTile + r];
#pragma unroll
    for (uint32_t q = 0; q < 16; ++q)
      if (q < nrank) M = fmaxf(M, st[q].x);
#pragma unroll
    for (uint32_t q = 0; q < 16; ++q)
      if (q < nrank && st[q].x != -INFINITY) L += st[q].y * ex2_approx(st[q].x - M);
  }
  const float invL = (rv && L > 0.f) ? 1.f / L : 0.f;

  // pass 2: probabilities of the visual columns, summed over the rows; with
  // CONF, the row's mean and M2 over this warp's visual columns as well (the
  // statistics of each 32-column block merged pairwise: Chan, Golub and
  // LeVeque's update)
  float cn = 0.f, cmean = 0.f, cm2 = 0.f;
#pragma unroll
  for (int cb = 0; cb < kBlocks; ++cb) {
    const int k0 = key0 + col0 + cb * 32;
    if (k0 + 32 <= a.vis_start || k0 >= a.vis_start + a.N_v) continue;  // warp-uniform
    float v[32];
    if (warp_live) {
      const float w = (mblk[cb] != -INFINITY) ? ex2_approx(mblk[cb] - M) * invL : 0.f;
      tmem_ld32(tbase + cb * 32, v);
      tc_wait_ld();
      if (k0 >= a.vis_start && k0 + 32 <= a.vis_start + a.N_v) {
#pragma unroll
        for (int i = 0; i < 32; ++i) v[i] *= w;
      } else {
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const int k = k0 + i;
          const bool kv = k >= a.vis_start && k < a.vis_start + a.N_v;
          v[i] = kv ? v[i] * w : 0.f;
        }
      }
      if (CONF) {
        const int lo = max(k0, a.vis_start), hi = min(k0 + 32, a.vis_start + a.N_v);
        const float nb = (float)(hi - lo);
        float s4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int i = 0; i < 32; ++i) s4[i & 3] += v[i];  // zero outside the visual range
        const float mb = ((s4[0] + s4[1]) + (s4[2] + s4[3])) / nb;
        float q4[4] = {0.f, 0.f, 0.f, 0.f};
        if (lo == k0 && hi == k0 + 32) {  // every column of the block is visual
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const float d = v[i] - mb;
            q4[i & 3] = fmaf(d, d, q4[i & 3]);
          }
        } else {
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const float d = (k0 + i >= lo && k0 + i < hi) ? v[i] - mb : 0.f;
            q4[i & 3] = fmaf(d, d, q4[i & 3]);
          }
        }
        const float n = cn + nb, dl = mb - cmean;
        cmean += dl * (nb / n);
        cm2 += ((q4[0] + q4[1]) + (q4[2] + q4[3])) + dl * dl * (cn * nb / n);
        cn = n;
      }
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
    } else {
      v[0] = 0.f;
    }
    red[quad][col0 + cb * 32 + lane] = v[0];
  }
  if (CONF) halfstat[half][r] = make_float2(cmean, cm2);  // last read before the cluster barrier
  __syncthreads();
  if (CONF && half == 0 && rv &&
      (a.conf_mask == nullptr || a.conf_mask[(size_t)b * a.N_t_max + j] != 0)) {
    // merge the two column halves of the row; counts from the column ranges
    const int vlo = a.vis_start, vhi = a.vis_start + a.N_v;
    const float n0 = (float)max(0, min(key0 + kHalfCols, vhi) - max(key0, vlo));
    const float n1 = (float)max(0, min(key0 + (int)kCols, vhi) - max(key0 + kHalfCols, vlo));
    const float2 s0 = halfstat[0][r], s1 = halfstat[1][r];
    float2 o = s0;
    if (n1 > 0.f) {
      if (n0 > 0.f) {
        const float n = n0 + n1, dl = s1.x - s0.x;
        o = make_float2(s0.x + dl * (n1 / n), s0.y + s1.y + dl * dl * (n0 * n1 / n));
      } else {
        o = s1;
      }
    }
    a.conf_part[(((size_t)b * a.H_sel + hi) * a.N_t_max + j) * a.conf_stride + rank] = o;
  }
  if (good) {
    float* out = a.partial + ((size_t)b * a.n_rb * a.H_sel + (size_t)rb * a.H_sel + hi) * a.N_v;
    for (int c = threadIdx.x; c < (int)kCols; c += kThreads) {
      const int k = key0 + c;
      if (k >= a.vis_start && k < a.vis_start + a.N_v)
        out[k - a.vis_start] = red[0][c] + red[1][c] + red[2][c] + red[3][c];
    }
  }
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x >= 32 && threadIdx.x < 64) tmem_dealloc(ctl.tmem, kCols);  // the allocating warp
  // When this grid is a programmatic dependent of the previous call's
  // compaction (independent batches), one CTA waits for that kernel before
  // exiting, so that this grid - and therefore the top-k that follows it and
  // rewrites idx - completes only after the compaction has read idx. The
  // partials need no such wait: the previous top-k has loaded them before the
  // compaction could start. A no-op without a programmatic dependency.
  if (blockIdx.x == 0 && blockIdx.y == 0 && blockIdx.z == 0)
    asm volatile("griddepcontrol.wait;" ::: "memory");
}

// One-time launch facts per (device, CPC, CONF): whether the kernel can be
// configured at all (state: 0 not yet checked, 1 usable, -1 not) and, per
// cluster size, whether such a cluster can be placed (0 unknown, 1 yes, -1 no).
// Each is worked out under g_cfg_mu and published with a release store, so a
// host thread that reads a non-zero value also sees the kernel attributes set
// before it; threads racing on a first call wait for the one doing the setup.
struct FusedCfg {
  std::atomic<int> state;
  std::atomic<int> clusters_ok[17];
};
FusedCfg g_cfg[64][3][2];  // static storage: every field starts at zero
std::mutex g_cfg_mu;

template <int CPC, bool CONF>
cudaError_t launch_cpc(const HSArgs& a, const CUtensorMap* tmQ, const CUtensorMap* tmK, int C,
                       cudaStream_t s, bool* launched, bool pdl) {
  *launched = false;
  // dynamic shared memory large enough that (CTAs per SM) x (TMEM columns) <= 512
  constexpr int max_ctas = 512 / (CPC * kTile);
  constexpr size_t per_sm = 233472;  // 228 KiB of shared memory per SM
  size_t smem = smem_bytes<CPC>();
  const size_t floor_bytes = per_sm / (max_ctas + 1) + 1;  // one more CTA would not fit
  if (smem < floor_bytes) smem = floor_bytes;
  int dev = 0;
  cudaGetDevice(&dev);
  const int slot = CPC == 1 ? 0 : (CPC == 2 ? 1 : 2);
  FusedCfg& fc = g_cfg[dev >= 0 && dev < 64 ? dev : 0][slot][CONF ? 1 : 0];
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[3];
  cfg.gridDim = dim3((unsigned)C, (unsigned)(a.H_sel * a.n_rb), (unsigned)a.B);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  // let the hardware put several CTAs of a cluster on one SM (the default
  // policy spreads them one per SM, which caps the CTAs in flight at ~1 per SM)
  attr[1].id = cudaLaunchAttributeClusterSchedulingPolicyPreference;
  attr[1].val.clusterSchedulingPolicyPreference = cudaClusterSchedulingPolicyLoadBalancing;
  attr[2].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[2].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  int state = fc.state.load(std::memory_order_acquire);
  if (state == 0) {
    std::lock_guard<std::mutex> lock(g_cfg_mu);
    state = fc.state.load(std::memory_order_relaxed);
    if (state == 0) {
      bool usable = false;
      cudaError_t e = cudaFuncSetAttribute(hs_fused_tc<CPC, CONF>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      if (e == cudaSuccess) e = cudaFuncSetAttribute(hs_fused_tc<CPC, CONF>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
      if (e == cudaSuccess) {
        int per = 0;
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per, hs_fused_tc<CPC, CONF>, kThreads, smem);
        usable = e == cudaSuccess && per >= 1 && per * CPC * kTile <= 512;
      }
      if (e != cudaSuccess) cudaGetLastError();  // not usable: the caller takes the two-kernel path
      state = usable ? 1 : -1;
      fc.state.store(state, std::memory_order_release);
    }
  }
  if (state < 0) return cudaSuccess;
  // a cluster of C CTAs must be placeable on this GPU (checked once per size)
  if (C < 1 || C > 16) return cudaSuccess;
  int placeable = fc.clusters_ok[C].load(std::memory_order_acquire);
  if (placeable == 0) {
    std::lock_guard<std::mutex> lock(g_cfg_mu);
    placeable = fc.clusters_ok[C].load(std::memory_order_relaxed);
    if (placeable == 0) {
      int nclusters = 0;
      cudaError_t q = cudaOccupancyMaxActiveClusters(&nclusters, hs_fused_tc<CPC, CONF>, &cfg);
      if (q != cudaSuccess) cudaGetLastError();
      placeable = (q == cudaSuccess && nclusters >= 1) ? 1 : -1;
      fc.clusters_ok[C].store(placeable, std::memory_order_release);
    }
  }
  if (placeable < 0) return cudaSuccess;
  if (pdl) cfg.numAttrs = 3;
  cudaError_t e = cudaLaunchKernelEx(&cfg, hs_fused_tc<CPC, CONF>, a, *tmQ, *tmK);
  if (e == cudaSuccess) *launched = true;
  return e;
}

template <int CPC>
cudaError_t launch_conf(const HSArgs& a, const CUtensorMap* tmQ, const CUtensorMap* tmK, int C,
                        cudaStream_t s, bool* launched, bool pdl, ConfGeom* geom) {
  if (a.conf_part != nullptr && C > a.conf_stride) return cudaSuccess;  // no room: two-pass path
  cudaError_t e = a.conf_part != nullptr ? launch_cpc<CPC, true>(a, tmQ, tmK, C, s, launched, pdl)
                                         : launch_cpc<CPC, false>(a, tmQ, tmK, C, s, launched, pdl);
  if (*launched && geom) *geom = ConfGeom{0, CPC * kTile, C};
  return e;
}

}  // namespace

// One-pass head scores; *launched is false when no cluster shape fits (the
// caller then runs the two-kernel path).
cudaError_t hs_launch_fused(const HSArgs& a, const CUtensorMap* tmQ, const CUtensorMap* tmK,
                            cudaStream_t s, bool* launched, bool pdl, ConfGeom* geom) {
  *launched = false;
  const int chunks = (a.L_max + kTile - 1) / kTile;
  if (chunks <= 16) return launch_conf<1>(a, tmQ, tmK, chunks, s, launched, pdl, geom);
  if (chunks <= 32) return launch_conf<2>(a, tmQ, tmK, (chunks + 1) / 2, s, launched, pdl, geom);
  if (chunks <= 64) return launch_conf<4>(a, tmQ, tmK, (chunks + 3) / 4, s, launched, pdl, geom);
  return cudaSuccess;
}

}  // namespace provip
