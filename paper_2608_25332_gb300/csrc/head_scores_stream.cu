// Head-aware visual-token scores (Sec. 4.4) for many (sample, head) pairs:
// one CTA per (row block x head, sample) streams that head's keys through a
// pipeline, with no cluster.
//
// Each CTA holds its 128 x 128 bf16 text-query tile in shared memory and
// visits n_A + n_B key chunks of 128 keys:
//   pass A (chunks 0 .. n_A - 1, every key up to the block's last text row):
//     S = Q K^T of the chunk, then per row a running max m and sum l of
//     exp2(s - m) over its causal keys - the row's global (max, sum);
//   pass B (the n_B chunks of visual keys, vis_start + 128 c ...): the
//     logits again (those keys are read a second time, from L2: the chunk was
//     loaded in pass A moments before), p = 2^(s - M) / L = 2^(s - c) with
//     c = M + log2 L, summed over the 128 rows into
//     partial[b][rb * H_sel + h][col]. Pass B computes S^T = K Q^T (TMEM lane =
//     key), so a key's sum over the rows stays in its thread (two halves of 64
//     rows, added in a fixed order).
// With CONF, pass A also keeps, per row, the count, mean and M2 (Chan, Golub
// and LeVeque) of 2^(s - m) over its visual keys, rescaled whenever the
// running max m rises (mean by 2^(m_old - m_new), M2 by its square); at the
// switch to pass B the two column halves are brought to the row max M and
// merged, and mean / L, M2 / L^2 are those of the visual probabilities p.
// Rows of the query tile past the block's text rows are zeroed in shared
// memory before the first MMA, so every logit the workers read is finite.
// Roles: warp 8 (one lane) issues the TMA loads into a 2-stage ring of key
// tiles, warp 9 (one lane) issues 8 tcgen05.mma (M = N = 128, K = 16) per
// chunk into one of two 128-column TMEM accumulators and commits, warps 0-7
// (two per TMEM lane quadrant, 64 columns each) turn accumulators into
// statistics and release them. The loads, the MMAs and the softmax work of
// consecutive chunks overlap. Two CTAs per SM (their shared memory rules out a
// third), so the two accumulators of each never wait for tensor memory.
// Every wait is bounded; a timeout sets the device error word.
#include "common.cuh"
#include "kernels.h"

namespace provip {
namespace {

constexpr int kTile = 128;
constexpr int kHalfBytes = kTile * 128;     // one 64-column box: 128 rows x 128 B
constexpr int kTileBytes = 2 * kHalfBytes;  // 32 KiB
constexpr int kStages = 2;                  // key tiles in shared memory
constexpr int kWorkerThreads = 256;         // warps 0-7
constexpr int kThreads = kWorkerThreads + 64;  // + TMA warp + MMA warp
constexpr uint32_t kTmemCols = 2 * kTile;   // two accumulators
constexpr size_t kSmem = (size_t)(1 + kStages) * kTileBytes + 1024;
constexpr uint32_t kIdesc = idesc_bf16_f32(128, 128);

struct Ctl {
  uint64_t q_full;
  uint64_t q_ready;  // rows past the text block zeroed (finite logits)
  uint64_t k_full[kStages];
  uint64_t k_empty[kStages];
  uint64_t acc_full[2];
  uint64_t acc_empty[2];
  uint32_t tmem;
  volatile int fail;
};

__device__ __forceinline__ void workers_sync() {
  asm volatile("bar.sync 1, %0;" ::"n"(kWorkerThreads) : "memory");
}
__device__ __forceinline__ void pdl_trigger() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
// one CTA of the grid waits for the kernel this grid depends on before the
// grid may complete (the overlap protocol of provip_prune; a no-op otherwise)
__device__ __forceinline__ void pdl_hold_completion() {
  if (blockIdx.x == 0 && blockIdx.y == 0) asm volatile("griddepcontrol.wait;" ::: "memory");
}

// pairwise (Chan, Golub and LeVeque) update of (n, mean, M2) with a block's
__device__ __forceinline__ void chan_merge(float& n, float& mean, float& m2, float nb, float mb,
                                           float m2b) {
  const float nn = n + nb, dl = mb - mean;
  mean += dl * (nb / nn);
  m2 += m2b + dl * dl * (n * nb / nn);
  n = nn;
}

template <bool CONF>
__global__ void __launch_bounds__(kThreads, 2)
    hs_stream_tc(const HSArgs a, const __grid_constant__ CUtensorMap tmQ,
                 const __grid_constant__ CUtensorMap tmK) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ Ctl ctl;
  __shared__ float2 halfstat[2][kTile];
  __shared__ float4 halfconf[CONF ? 2 : 1][CONF ? kTile : 1];  // (count, mean, M2, max) per half
  __shared__ float red[2][4][kTile];
  __shared__ __align__(16) float crow[kTile];  // M + log2(L) per row; +inf: not scored
  const int hi = blockIdx.x % a.H_sel, rb = blockIdx.x / a.H_sel;
  const int b = blockIdx.y;
  const int h = a.heads[hi], g = h / (a.H_q / a.H_kv);
  const int ts = a.text_start[b], sl = a.seq_len[b];
  int tl = a.text_len[b];
  const bool ok = ts >= 0 && tl >= 0 && tl <= a.N_t_max && sl <= a.L_max && ts + tl <= sl &&
                  a.vis_start + a.N_v <= sl;
  if (!ok) tl = 0;
  float* out = a.partial + ((size_t)b * a.n_rb * a.H_sel + (size_t)rb * a.H_sel + hi) * a.N_v;
  const int rows = min(kTile, tl - rb * kTile);  // candidate text rows of the block
  if (rows <= 0) {
    // nothing to score: the block's partial is zero
    if (!ok && threadIdx.x == 0 && blockIdx.x == 0) set_error(a.err, kErrBadDeviceArg);
    pdl_trigger();
    for (int c = threadIdx.x; c < a.N_v; c += kThreads) out[c] = 0.f;
    pdl_hold_completion();
    return;
  }
  const int t_last = ts + rb * kTile + rows - 1;
  const int nA = t_last / kTile + 1;
  const int nB = (a.N_v + kTile - 1) / kTile;
  const int n_it = nA + nB;

  const uint32_t base = smem_u32(smem_raw);
  uint8_t* qs = smem_raw + (((base + 1023u) & ~1023u) - base);
  uint8_t* ks = qs + kTileBytes;
  pdl_trigger();  // a programmatic dependent may be scheduled now
  if (threadIdx.x == 0) {
    prefetch_tmap(&tmQ);
    prefetch_tmap(&tmK);
    mbar_init(&ctl.q_full, 1);
    mbar_init(&ctl.q_ready, kWorkerThreads / 32);
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&ctl.k_full[s], 1);
      mbar_init(&ctl.k_empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&ctl.acc_full[s], 1);
      mbar_init(&ctl.acc_empty[s], kWorkerThreads / 32);
    }
    ctl.fail = 0;
    fence_mbar_init();
  }
  if (threadIdx.x < 32) {
    tmem_alloc(&ctl.tmem, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (warp == 8) {
    // ---- TMA producer ----
    if (lane == 0) {
      mbar_arrive_expect_tx(&ctl.q_full, kTileBytes);
      const int yq = b * a.L_max + ts + rb * kTile, xq = h * kHeadDim;
      tma_load_2d(qs, &tmQ, xq, yq, &ctl.q_full);
      tma_load_2d(qs + kHalfBytes, &tmQ, xq + 64, yq, &ctl.q_full);
      for (int it = 0; it < n_it; ++it) {
        const int s = it % kStages;
        const uint32_t ph = (uint32_t)(it / kStages) & 1u;
        if (ctl.fail || !mbar_wait(&ctl.k_empty[s], ph ^ 1u, a.err)) {
          ctl.fail = 1;
          break;
        }
        const int yk = b * a.L_max + (it < nA ? it * kTile : a.vis_start + (it - nA) * kTile);
        uint8_t* dst = ks + (size_t)s * kTileBytes;
        mbar_arrive_expect_tx(&ctl.k_full[s], kTileBytes);
        tma_load_2d(dst, &tmK, g * kHeadDim, yk, &ctl.k_full[s]);
        tma_load_2d(dst + kHalfBytes, &tmK, g * kHeadDim + 64, yk, &ctl.k_full[s]);
      }
    }
  } else if (warp == 9) {
    // ---- MMA issuer ----
    if (lane == 0) {
      bool live = mbar_wait(&ctl.q_ready, 0, a.err);
      if (!live) ctl.fail = 1;
      const uint32_t qa = smem_u32(qs);
      for (int it = 0; it < n_it && live; ++it) {
        const int s = it % kStages, buf = it & 1;
        const uint32_t ph_k = (uint32_t)(it / kStages) & 1u, ph_a = (uint32_t)(it >> 1) & 1u;
        if (ctl.fail || !mbar_wait(&ctl.acc_empty[buf], ph_a ^ 1u, a.err) ||
            !mbar_wait(&ctl.k_full[s], ph_k, a.err)) {
          ctl.fail = 1;
          break;
        }
        tc_fence_after();
        const uint32_t ka = smem_u32(ks + (size_t)s * kTileBytes);
        const uint32_t acc = ctl.tmem + (uint32_t)(buf * kTile);
        // pass A: S = Q K^T (lane = text row); pass B: S^T = K Q^T (lane =
        // key), so a key's sum over the rows stays in its thread
        const bool tr = it >= nA;
        const uint32_t opa = tr ? ka : qa, opb = tr ? qa : ka;
#pragma unroll
        for (int kstep = 0; kstep < 8; ++kstep) {
          const uint32_t off = (kstep >> 2) * kHalfBytes + (kstep & 3) * 32;
          tc_mma_bf16(acc, smem_desc_sw128(opa + off), smem_desc_sw128(opb + off), kIdesc,
                      kstep > 0 ? 1u : 0u);
        }
        tc_commit(&ctl.k_empty[s]);
        tc_commit(&ctl.acc_full[buf]);
      }
    }
  } else {
    // ---- softmax workers: thread = TMEM lane = text row, 64 columns per warp ----
    const int quad = warp & 3, half = warp >> 2;
    const int r = quad * 32 + lane;
    const int j = rb * kTile + r;
    const bool rv = j < tl && (a.row_mask == nullptr || a.row_mask[(size_t)b * a.N_t_max + j] != 0);
    const int t = ts + j;
    const uint32_t tbase = ctl.tmem + ((uint32_t)(quad * 32) << 16) + (uint32_t)(half * 64);
    const float sc = a.scale_log2;
    const int t_first = ts + rb * kTile;  // every row of the block sits at or after it
    bool failed = !warp_mbar_wait(&ctl.q_full, 0, a.err);  // warp-uniform from here on
    {
      // rows of the query tile past the block's text rows may hold anything
      // (other samples, padding): zero them, so every logit is finite
      const int nz = (kTile - rows) * 16;  // 16-byte pieces: 8 per 128-byte row, two halves
      for (int q = threadIdx.x; q < nz; q += kWorkerThreads) {
        const int row = rows + q / 16, piece = q % 16;
        *reinterpret_cast<uint4*>(qs + (piece >> 3) * kHalfBytes + row * 128 + (piece & 7) * 16) =
            make_uint4(0u, 0u, 0u, 0u);
      }
      fence_proxy_async_smem();  // visible to the tensor cores
      __syncwarp();
      if (lane == 0) mbar_arrive(&ctl.q_ready);
    }
    // m: running max of the scaled logits, l: sum of 2^(s - m); c = M + log2(L)
    float m = -INFINITY, l = 0.f, c = 0.f;
    float cn = 0.f, cmean = 0.f, cm2 = 0.f;
    for (int it = 0; it < n_it; ++it) {
      const int buf = it & 1;
      if (!failed) failed = !warp_mbar_wait(&ctl.acc_full[buf], (uint32_t)(it >> 1) & 1u, a.err);
      tc_fence_after();
      if (it == nA) {
        // the row's global (max, sum) from the two column halves
        halfstat[half][r] = make_float2(rv ? m : -INFINITY, rv ? l : 0.f);
        workers_sync();
        const float2 h0 = halfstat[0][r], h1 = halfstat[1][r];
        const float M = fmaxf(h0.x, h1.x);
        float L = 0.f;
        if (h0.x != -INFINITY) L += h0.y * ex2_approx(h0.x - M);
        if (h1.x != -INFINITY) L += h1.y * ex2_approx(h1.x - M);
        // p = 2^(s - M) / L = 2^(s - c); L >= 1 (the max term) for a valid row
        c = (rv && L > 0.f) ? M + lg2_approx(L) : 0.f;
        if (CONF) {
          // each half's statistics at the row max M, merged in half order, then
          // those of p = x / L; written for the rows of T
          halfconf[half][r] = make_float4(cn, cmean, cm2, m);
          workers_sync();
          if (half == 0 && rv && L > 0.f &&
              (a.conf_mask == nullptr || a.conf_mask[(size_t)b * a.N_t_max + j] != 0)) {
            float n = 0.f, mean = 0.f, m2 = 0.f;
#pragma unroll
            for (int q = 0; q < 2; ++q) {
              const float4 hc = halfconf[q][r];
              if (hc.x > 0.f) {
                const float f = ex2_approx(hc.w - M);
                chan_merge(n, mean, m2, hc.x, hc.y * f, hc.z * f * f);
              }
            }
            a.conf_part[(((size_t)b * a.H_sel + hi) * a.N_t_max + j) * a.conf_stride] =
                make_float2(mean / L, m2 / (L * L));
          }
        }
        if (half == 0) crow[r] = (rv && L > 0.f) ? c : INFINITY;  // 2^-inf = 0
        workers_sync();
      }
      const uint32_t tacc = tbase + (uint32_t)(buf * kTile);
      if (it < nA) {
#pragma unroll
        for (int cb = 0; cb < 2; ++cb) {
          float v[32];
          tmem_ld32(tacc + cb * 32, v);
          tc_wait_ld();
          const int k0 = it * kTile + half * 64 + cb * 32;
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
            const float mn = fmaxf(m, bm * sc);  // sc > 0: the max commutes with the scale
            if (mn != -INFINITY) {
              float s4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
              for (int i = 0; i < 32; ++i) {
                v[i] = ex2_approx(fmaf(v[i], sc, -mn));
                s4[i & 3] += v[i];
              }
              const float rs = ex2_approx(m - mn);
              l = l * rs + ((s4[0] + s4[1]) + (s4[2] + s4[3]));
              if (CONF) {
                // the visual keys of this block: [vlo, vhi) relative to k0
                const int vlo = max(a.vis_start - k0, 0), vhi = min(a.vis_start + a.N_v - k0, 32);
                if (cn > 0.f) {
                  cmean *= rs;
                  cm2 *= rs * rs;
                }
                if (vlo == 0 && vhi == 32) {
                  // every key of the block is visual (the common case)
                  float q4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
                  for (int i = 0; i < 32; ++i) q4[i & 3] += v[i];
                  const float mb = ((q4[0] + q4[1]) + (q4[2] + q4[3])) * (1.f / 32.f);
                  float d4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
                  for (int i = 0; i < 32; ++i) {
                    const float d = v[i] - mb;
                    d4[i & 3] = fmaf(d, d, d4[i & 3]);
                  }
                  chan_merge(cn, cmean, cm2, 32.f, mb, (d4[0] + d4[1]) + (d4[2] + d4[3]));
                } else if (vlo < vhi) {
                  const float nb = (float)(vhi - vlo);
                  float q4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
                  for (int i = 0; i < 32; ++i) q4[i & 3] += (i >= vlo && i < vhi) ? v[i] : 0.f;
                  const float mb = ((q4[0] + q4[1]) + (q4[2] + q4[3])) / nb;
                  float d4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
                  for (int i = 0; i < 32; ++i) {
                    const float d = (i >= vlo && i < vhi) ? v[i] - mb : 0.f;
                    d4[i & 3] = fmaf(d, d, d4[i & 3]);
                  }
                  chan_merge(cn, cmean, cm2, nb, mb, (d4[0] + d4[1]) + (d4[2] + d4[3]));
                }
              }
            }
            m = mn;
          }
        }
      } else {
        // transposed: thread = key kk of the chunk, 64 text rows per warp
        const int par = (it - nA) & 1;
        const int kk = quad * 32 + lane, key = a.vis_start + (it - nA) * kTile + kk;
        const bool all_causal = a.vis_start + (it - nA) * kTile + kTile - 1 <= t_first;
        float csum = 0.f;
#pragma unroll
        for (int cb = 0; cb < 2; ++cb) {
          const int i0 = half * 64 + cb * 32;  // first row of the block
          float v[32];
          tmem_ld32(tacc + cb * 32, v);
          tc_wait_ld();
          float s4[4] = {0.f, 0.f, 0.f, 0.f};
          const float4* cr = reinterpret_cast<const float4*>(crow + i0);
          if (all_causal) {
#pragma unroll
            for (int i4 = 0; i4 < 8; ++i4) {
              const float4 cc = cr[i4];
              s4[0] += ex2_approx(fmaf(v[4 * i4 + 0], sc, -cc.x));
              s4[1] += ex2_approx(fmaf(v[4 * i4 + 1], sc, -cc.y));
              s4[2] += ex2_approx(fmaf(v[4 * i4 + 2], sc, -cc.z));
              s4[3] += ex2_approx(fmaf(v[4 * i4 + 3], sc, -cc.w));
            }
          } else {
#pragma unroll
            for (int i4 = 0; i4 < 8; ++i4) {
              const float4 cc = cr[i4];
              const float cv[4] = {cc.x, cc.y, cc.z, cc.w};
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                const int i = 4 * i4 + e;
                s4[e] += key <= t_first + i0 + i ? ex2_approx(fmaf(v[i], sc, -cv[e])) : 0.f;
              }
            }
          }
          csum += (s4[0] + s4[1]) + (s4[2] + s4[3]);
        }
        red[par][half][kk] = csum;
      }
      // the accumulator may be overwritten
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&ctl.acc_empty[buf]);
      if (it >= nA) {
        const int par = (it - nA) & 1;
        workers_sync();  // red[par] complete (red[par ^ 1] is free: read before this barrier)
        const int c = (it - nA) * kTile + threadIdx.x;
        if (threadIdx.x < kTile && c < a.N_v)
          out[c] = red[par][0][threadIdx.x] + red[par][1][threadIdx.x];
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(ctl.tmem, kTmemCols);
  pdl_hold_completion();
}

template <bool CONF>
cudaError_t launch(const HSArgs& a, const CUtensorMap* tmQ, const CUtensorMap* tmK, cudaStream_t s,
                   bool pdl) {
  static std::atomic<bool> configured[64];  // per device, zero-initialised
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64 && !configured[dev]) {
    cudaError_t e = cudaFuncSetAttribute(hs_stream_tc<CONF>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)kSmem);
    if (e != cudaSuccess) return e;
    configured[dev] = true;
  }
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  cfg.gridDim = dim3((unsigned)(a.H_sel * a.n_rb), (unsigned)a.B);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = kSmem;
  cfg.stream = s;
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, hs_stream_tc<CONF>, a, *tmQ, *tmK);
}

}  // namespace

cudaError_t hs_launch_stream(const HSArgs& a, const CUtensorMap* tmQ, const CUtensorMap* tmK,
                             cudaStream_t s, bool pdl, ConfGeom* geom) {
  if (geom) *geom = ConfGeom{a.vis_start, ((a.N_v + kTile - 1) / kTile) * kTile, 1};
  return a.conf_part != nullptr ? launch<true>(a, tmQ, tmK, s, pdl) : launch<false>(a, tmQ, tmK, s, pdl);
}

}  // namespace provip
