// Head-aware visual-token scores (Sec. 4.4), CUDA-core path (fp32 and bf16).
//
// v_i = 1/(|R| |V|) sum_{j in R} sum_{h in V} softmax_k( q_{j,h} . k_{k,g(h)} / sqrt(d_h) )
//       evaluated at k = vis_start + i, the softmax running over the full causal
//       key range 0..t_j of text row j (t_j its absolute position).
//
// Pass 1 (hs_stats_simt): grid (key chunk, row block x head, sample); per text
//   row, the chunk max and exp-sum over its causal keys -> stats.
// Pass 2 (hs_probs_simt): grid (visual chunk, row block x head, sample); recompute
//   the logits of the chunk's visual keys, normalise by the row's global
//   (max, sum) combined from all chunk stats, sum over the block's rows ->
//   partial[b][rb * H_sel + head][col]. Deterministic: fixed reduction orders,
//   no atomics.
// hs_reduce: scores = sum of partials over (row block, head) / (|V| |R|).
// conf_select: head confidence from the pass-2 row statistics and the top
//   n_vis heads per sample.
#include "common.cuh"
#include "kernels.h"
#include "simt_gemm.cuh"

namespace provip {

namespace {

struct HSRow {
  int ts, tl, sl;
  bool ok;
};

__device__ __forceinline__ HSRow hs_sample(const HSArgs& a, int b) {
  HSRow r;
  r.ts = a.text_start[b];
  r.tl = a.text_len[b];
  r.sl = a.seq_len[b];
  r.ok = r.ts >= 0 && r.tl >= 0 && r.tl <= a.N_t_max && r.sl <= a.L_max && r.ts + r.tl <= r.sl &&
         a.vis_start + a.N_v <= r.sl;
  return r;
}

__device__ __forceinline__ bool hs_row_valid(const HSArgs& a, const HSRow& s, int b, int j) {
  return s.ok && j < s.tl && (a.row_mask == nullptr || a.row_mask[(size_t)b * a.N_t_max + j] != 0);
}

template <typename T>
__global__ void __launch_bounds__(256) hs_stats_simt(const HSArgs a) {
  __shared__ __align__(16) SimtSmem sm;
  __shared__ const T* arow[kSimtBM];
  __shared__ const T* brow[kSimtBN];
  const int c = blockIdx.x;
  const int hi = blockIdx.y % a.H_sel, rb = blockIdx.y / a.H_sel;
  const int b = blockIdx.z;
  const int h = a.heads[hi], g = h / (a.H_q / a.H_kv);
  const HSRow smp = hs_sample(a, b);
  if (!smp.ok && threadIdx.x == 0 && c == 0 && blockIdx.y == 0) set_error(a.err, kErrBadDeviceArg);
  const T* Q = static_cast<const T*>(a.Q);
  const T* K = static_cast<const T*>(a.K);
  const int k0 = c * kSimtBN;
  if (threadIdx.x < kSimtBM) {
    const int j = rb * kSimtBM + threadIdx.x;
    arow[threadIdx.x] = hs_row_valid(a, smp, b, j)
                            ? Q + (((size_t)b * a.L_max + smp.ts + j) * a.H_q + h) * a.d_h
                            : nullptr;
  }
  if (threadIdx.x < kSimtBN) {
    const int k = k0 + threadIdx.x;
    brow[threadIdx.x] = (smp.ok && k < smp.sl)
                            ? K + (((size_t)b * a.L_max + k) * a.H_kv + g) * a.d_h
                            : nullptr;
  }
  __syncthreads();
  float acc[8][4];
  simt_gemm_nt<T>(arow, brow, a.d_h, sm, acc);
  const int rg = threadIdx.x >> 4, kg = threadIdx.x & 15;
  float2* st = a.stats + ((((size_t)b * a.n_rb + rb) * a.H_sel + hi) * a.n_kc + c) * kSimtBM;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int r = rg + 16 * i;
    const bool rv = arow[r] != nullptr;
    const int t = smp.ts + rb * kSimtBM + r;
    float s[4];
    bool kv[4];
    float m = -INFINITY;
#pragma unroll
    for (int jj = 0; jj < 4; ++jj) {
      const int k = k0 + kg + 16 * jj;
      kv[jj] = rv && k <= t;
      s[jj] = acc[i][jj] * a.scale_log2;
      if (kv[jj]) m = fmaxf(m, s[jj]);
    }
    m = rowgroup_max(m);
    float l = 0.f;
#pragma unroll
    for (int jj = 0; jj < 4; ++jj)
      if (kv[jj]) l += exp2f(s[jj] - m);
    l = rowgroup_sum(l);
    if (kg == 0) st[r] = make_float2(m, l);
  }
}

template <typename T>
__global__ void __launch_bounds__(256) hs_probs_simt(const HSArgs a) {
  __shared__ __align__(16) SimtSmem sm;
  __shared__ const T* arow[kSimtBM];
  __shared__ const T* brow[kSimtBN];
  __shared__ float rowm[kSimtBM], rowinv[kSimtBM];
  __shared__ float red[8][kSimtBN];
  const int vc = blockIdx.x;
  const int hi = blockIdx.y % a.H_sel, rb = blockIdx.y / a.H_sel;
  const int b = blockIdx.z;
  const int h = a.heads[hi], g = h / (a.H_q / a.H_kv);
  const HSRow smp = hs_sample(a, b);
  const T* Q = static_cast<const T*>(a.Q);
  const T* K = static_cast<const T*>(a.K);
  const int col0 = vc * kSimtBN;
  if (threadIdx.x < kSimtBM) {
    const int r = threadIdx.x;
    const int j = rb * kSimtBM + r;
    const bool rv = hs_row_valid(a, smp, b, j);
    arow[r] = rv ? Q + (((size_t)b * a.L_max + smp.ts + j) * a.H_q + h) * a.d_h : nullptr;
    // combine this row's chunk statistics into its global (max, 1 / sum)
    float m = -INFINITY, l = 0.f;
    if (rv) {
      const float2* st = a.stats + (((size_t)b * a.n_rb + rb) * a.H_sel + hi) * a.n_kc * kSimtBM + r;
      for (int c = 0; c < a.n_kc; ++c) m = fmaxf(m, st[(size_t)c * kSimtBM].x);
      for (int c = 0; c < a.n_kc; ++c) {
        const float2 v = st[(size_t)c * kSimtBM];
        if (v.x != -INFINITY) l += v.y * exp2f(v.x - m);
      }
    }
    rowm[r] = m;
    rowinv[r] = l > 0.f ? 1.f / l : 0.f;
  }
  if (threadIdx.x < kSimtBN) {
    const int col = col0 + threadIdx.x;
    brow[threadIdx.x] = (smp.ok && col < a.N_v)
                            ? K + (((size_t)b * a.L_max + a.vis_start + col) * a.H_kv + g) * a.d_h
                            : nullptr;
  }
  __syncthreads();
  float acc[8][4];
  simt_gemm_nt<T>(arow, brow, a.d_h, sm, acc);
  const int rg = threadIdx.x >> 4, kg = threadIdx.x & 15;
  const bool conf = a.conf_part != nullptr;  // block-uniform
  const int ncol = min(kSimtBN, a.N_v - col0);
  float cs[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int r = rg + 16 * i;
    const bool rv = arow[r] != nullptr;
    const int t = smp.ts + rb * kSimtBM + r;
    const float m = rowm[r], inv = rowinv[r];
    float pv[4];
#pragma unroll
    for (int jj = 0; jj < 4; ++jj) {
      const int col = col0 + kg + 16 * jj;
      pv[jj] = (rv && col < a.N_v && a.vis_start + col <= t) ? exp2f(acc[i][jj] * a.scale_log2 - m) * inv : 0.f;
      cs[jj] += pv[jj];
    }
    if (conf) {
      // head confidence: the row's mean and M2 over the chunk's visual columns
      // (two-pass over the values in registers; row groups of 16 lanes)
      const float mean = rowgroup_sum((pv[0] + pv[1]) + (pv[2] + pv[3])) / (float)ncol;
      float q = 0.f;
#pragma unroll
      for (int jj = 0; jj < 4; ++jj) {
        const float d = (kg + 16 * jj < ncol) ? pv[jj] - mean : 0.f;
        q += d * d;
      }
      q = rowgroup_sum(q);
      const int j = rb * kSimtBM + r;
      if (kg == 0 && rv && (a.conf_mask == nullptr || a.conf_mask[(size_t)b * a.N_t_max + j] != 0))
        a.conf_part[(((size_t)b * a.H_sel + hi) * a.N_t_max + j) * a.conf_stride + vc] = make_float2(mean, q);
    }
  }
  // rows rg and rg + 1 of a warp: fold lanes 16..31 onto 0..15, then across warps
#pragma unroll
  for (int jj = 0; jj < 4; ++jj) cs[jj] += __shfl_xor_sync(0xffffffffu, cs[jj], 16);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane < 16) {
#pragma unroll
    for (int jj = 0; jj < 4; ++jj) red[warp][lane + 16 * jj] = cs[jj];
  }
  __syncthreads();
  if (threadIdx.x < kSimtBN) {
    const int col = col0 + threadIdx.x;
    float s = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) s += red[w][threadIdx.x];
    if (col < a.N_v)
      a.partial[((size_t)b * a.n_rb * a.H_sel + (size_t)rb * a.H_sel + hi) * a.N_v + col] = s;
  }
}

// number of valid text rows of sample b (block-wide; all threads get it)
__device__ int hs_count_rows(const HSArgs& a, int b) {
  __shared__ int cnt;
  if (threadIdx.x == 0) cnt = 0;
  __syncthreads();
  const HSRow smp = hs_sample(a, b);
  int mine = 0;
  for (int j = threadIdx.x; j < a.N_t_max; j += blockDim.x) mine += hs_row_valid(a, smp, b, j);
  if (mine) atomicAdd(&cnt, mine);
  __syncthreads();
  return cnt;
}

__global__ void __launch_bounds__(256) hs_reduce_kernel(const HSArgs a, float* scores) {
  const int b = blockIdx.y;
  const int n = hs_count_rows(a, b);
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= a.N_v) return;
  const int U = a.n_rb * a.H_sel;
  const float* p = a.partial + (size_t)b * U * a.N_v + i;
  float s = 0.f;
  for (int u = 0; u < U; ++u) s += p[(size_t)u * a.N_v];
  scores[(size_t)b * a.N_v + i] = n > 0 ? s / ((float)a.H_sel * (float)n) : 0.f;
}

// Head confidence and visual-head selection (Sec. 4.4), one CTA per sample.
// C[i] = sum over the confidence rows of (merged M2) / N_v for head-list
// position i; each warp takes heads i = warp, warp + 32, ...; each lane the rows
// lane, lane + 32, ... in batches of 4 (their loads in flight together), folded
// by a fixed butterfly, so C is deterministic. The chunk statistics of a row
// are merged in chunk order with Chan, Golub and LeVeque's pairwise update;
// chunk c holds the visual columns of [g.lo0 + c * g.w, g.lo0 + (c + 1) * g.w).
constexpr int kConfThreads = 1024;
constexpr int kConfBatch = 4;
__global__ void __launch_bounds__(kConfThreads) conf_select_kernel(const HSArgs a, const ConfGeom g,
                                                                  const ConfArgs c) {
  __shared__ float C[kMaxHeads];
  __shared__ int chosen[kMaxHeads];
  // programmatic dependent of the head-score kernel: wait for its statistics
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int b = blockIdx.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const HSRow smp = hs_sample(a, b);
  const int vlo = a.vis_start, vhi = a.vis_start + a.N_v;
  for (int i = warp; i < a.H_sel; i += kConfThreads / 32) {
    float acc = 0.f;
    const float2* base = a.conf_part + ((size_t)b * a.H_sel + i) * a.N_t_max * a.conf_stride;
    for (int j0 = 0; j0 < a.N_t_max; j0 += 32 * kConfBatch) {
      bool use[kConfBatch];
      float n[kConfBatch], mean[kConfBatch], m2[kConfBatch];
#pragma unroll
      for (int r = 0; r < kConfBatch; ++r) {
        const int j = j0 + 32 * r + lane;
        use[r] = j < a.N_t_max && hs_row_valid(a, smp, b, j) &&
                 (a.conf_mask == nullptr || a.conf_mask[(size_t)b * a.N_t_max + j] != 0);
        n[r] = 0.f;
        mean[r] = 0.f;
        m2[r] = 0.f;
      }
      for (int q = 0; q < g.n; ++q) {
        const int lo = max(g.lo0 + q * g.w, vlo), hi = min(g.lo0 + (q + 1) * g.w, vhi);
        if (hi <= lo) continue;
        const float nb = (float)(hi - lo);
        float2 v[kConfBatch];
#pragma unroll
        for (int r = 0; r < kConfBatch; ++r)
          v[r] = use[r] ? base[(size_t)(j0 + 32 * r + lane) * a.conf_stride + q] : make_float2(0.f, 0.f);
#pragma unroll
        for (int r = 0; r < kConfBatch; ++r) {
          const float nn = n[r] + nb, dl = v[r].x - mean[r];
          mean[r] += dl * (nb / nn);
          m2[r] += v[r].y + dl * dl * (n[r] * nb / nn);
          n[r] = nn;
        }
      }
#pragma unroll
      for (int r = 0; r < kConfBatch; ++r)
        if (use[r]) acc += m2[r] / (float)a.N_v;
    }
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if (lane == 0) C[i] = acc;
  }
  __syncthreads();
  // the next kernel (the top-k) may be scheduled; it waits for this grid
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int i = threadIdx.x;
  if (i < a.H_sel) {
    const uint32_t ki = float_key(C[i]);
    int rank = 0;
    for (int q = 0; q < a.H_sel; ++q) {
      const uint32_t kq = float_key(C[q]);
      rank += (kq > ki) || (kq == ki && q < i);
    }
    chosen[i] = rank < c.n_vis;
    if (c.conf_out) c.conf_out[(size_t)b * a.H_q + a.heads[i]] = C[i];
  }
  __syncthreads();
  if (i < a.H_sel && chosen[i]) {
    int pos = 0;
    for (int q = 0; q < i; ++q) pos += chosen[q];
    c.sel_out[(size_t)b * c.n_vis + pos] = i;
    if (c.vis_heads_out) c.vis_heads_out[(size_t)b * c.n_vis + pos] = a.heads[i];
  }
}

}  // namespace

cudaError_t conf_select_launch(const HSArgs& a, const ConfGeom& g, const ConfArgs& c,
                               cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  cfg.gridDim = dim3((unsigned)a.B);
  cfg.blockDim = dim3(kConfThreads);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = s;
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, conf_select_kernel, a, g, c);
}

cudaError_t hs_launch_simt(const HSArgs& a, int dtype, cudaStream_t s, ConfGeom* geom) {
  if (geom) *geom = ConfGeom{a.vis_start, kSimtBN, a.n_vc};
  dim3 g1(a.n_kc, a.H_sel * a.n_rb, a.B), g2(a.n_vc, a.H_sel * a.n_rb, a.B);
  if (dtype == 0) {
    hs_stats_simt<float><<<g1, 256, 0, s>>>(a);
    hs_probs_simt<float><<<g2, 256, 0, s>>>(a);
  } else {
    hs_stats_simt<__nv_bfloat16><<<g1, 256, 0, s>>>(a);
    hs_probs_simt<__nv_bfloat16><<<g2, 256, 0, s>>>(a);
  }
  return cudaGetLastError();
}

cudaError_t hs_launch_reduce(const HSArgs& a, float* scores, cudaStream_t s) {
  dim3 g((a.N_v + 255) / 256, a.B);
  hs_reduce_kernel<<<g, 256, 0, s>>>(a, scores);
  return cudaGetLastError();
}

}  // namespace provip
