// Pre-LLM pass (Sec. 4.2-4.3), CUDA-core kernels.
//
//   crit_text:  G = E_t E_t^T (no scale), row softmax, r_j = mean_i R_ij,
//               T = { j : r_j > mean(r) } (all rows when none exceeds it).
//   relevance:  p_j = max_{i in T} ( cos(t_i, v_j) - mu_i ), where the row mean
//               mu_i = (1/N_v) sum_k cos(t_i, v_k) = <t_i / |t_i|, sum_k v_k / |v_k|> / N_v
//               is computed from the sum of the normalised visual rows, so the
//               |T| x N_v cosine matrix is never stored.
//   merge:      for each visual row j, the kept row of largest cosine
//               (= largest <v_j, v_k> / |v_k|, since |v_j| is common), ties to
//               the lower kept position; merged_a = mean of centroid a and its
//               members, summed in ascending row order.
#include "common.cuh"
#include "kernels.h"
#include "simt_gemm.cuh"

namespace provip {
namespace {

template <typename T>
__device__ __forceinline__ const T* row_ptr(const void* base, size_t row, int D) {
  return static_cast<const T*>(base) + row * (size_t)D;
}

// ---------------------------------------------------------------------------
// Sec. 4.2
// ---------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(256) crit_gram_kernel(const SimArgs a, float* G) {
  __shared__ __align__(16) SimtSmem sm;
  __shared__ const T* arow[kSimtBM];
  __shared__ const T* brow[kSimtBN];
  const int b = blockIdx.z;
  const int r0 = blockIdx.y * kSimtBM, c0 = blockIdx.x * kSimtBN;
  int tl = a.text_len[b];
  if (tl < 0 || tl > a.N_t_max) tl = 0;
  if (threadIdx.x < kSimtBM) {
    const int j = r0 + threadIdx.x;
    arow[threadIdx.x] = j < tl ? row_ptr<T>(a.emb_t, (size_t)b * a.N_t_max + j, a.D) : nullptr;
  }
  if (threadIdx.x < kSimtBN) {
    const int j = c0 + threadIdx.x;
    brow[threadIdx.x] = j < tl ? row_ptr<T>(a.emb_t, (size_t)b * a.N_t_max + j, a.D) : nullptr;
  }
  __syncthreads();
  float acc[8][4];
  simt_gemm_nt<T>(arow, brow, a.D, sm, acc);
  const int rg = threadIdx.x >> 4, kg = threadIdx.x & 15;
#pragma unroll
  for (int i = 0; i < 8; ++i)
#pragma unroll
    for (int jj = 0; jj < 4; ++jj) {
      const int r = r0 + rg + 16 * i, c = c0 + kg + 16 * jj;
      if (r < a.N_t_max && c < a.N_t_max) G[((size_t)b * a.N_t_max + r) * a.N_t_max + c] = acc[i][jj];
    }
}

// one CTA per sample: row softmax statistics, column means r, threshold
// Adds the K parts of the text Gram into part 0, in part order: one thread per
// element, every part's load issued first.
constexpr int kCritMaxParts = 16;
__global__ void __launch_bounds__(256) crit_parts_sum_kernel(float* G, size_t n, int n_parts) {
  const size_t e = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (e >= n) return;
  float v[kCritMaxParts];
#pragma unroll
  for (int q = 0; q < kCritMaxParts; ++q)
    if (q < n_parts) v[q] = G[q * n + e];
  float s = v[0];
#pragma unroll
  for (int q = 1; q < kCritMaxParts; ++q)
    if (q < n_parts) s += v[q];
  G[e] = s;
}

// G: the sample Grams [B][Ntm][Ntm]. Up to kFinishSmemNt text rows the sample's
// Gram is staged in shared memory. One CTA of 1024 threads per sample: a warp
// per row for the softmax statistics, then the column sums of the softmax in
// kFinishThreads / n row groups whose partial sums are added in group order.
constexpr int kFinishSmemNt = 128;
constexpr int kFinishThreads = 1024;
__global__ void __launch_bounds__(kFinishThreads) crit_finish_kernel(const SimArgs a, const float* G,
                                                                     uint8_t* mask, float* r_out) {
  // rowm[Ntm], rowinv[Ntm], r[Ntm], part[kFinishThreads] (+ G[Ntm][Ntm] when staged)
  extern __shared__ float sh[];
  float* rowm = sh;
  float* rowinv = sh + a.N_t_max;
  float* rr = sh + 2 * a.N_t_max;
  float* part = sh + 3 * a.N_t_max;
  __shared__ float wsum[kFinishThreads / 32];
  __shared__ int wcnt[kFinishThreads / 32];
  constexpr int kWarps = kFinishThreads / 32;
  const int b = blockIdx.x;
  int n = a.text_len[b];
  if (n < 0 || n > a.N_t_max) {
    if (threadIdx.x == 0) set_error(a.err, kErrBadDeviceArg);
    n = 0;
  }
  const float* Gb = G + (size_t)b * a.N_t_max * a.N_t_max;
  const bool staged = a.N_t_max <= kFinishSmemNt;
  float* Gs = part + kFinishThreads;
  int ld = a.N_t_max;
  if (staged) {
    // eight loads in flight per thread
    for (int e0 = 0; e0 < n * n; e0 += 8 * (int)blockDim.x) {
      float v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int e = e0 + u * (int)blockDim.x + (int)threadIdx.x;
        if (e < n * n) v[u] = Gb[(size_t)(e / n) * a.N_t_max + (e - (e / n) * n)];
      }
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int e = e0 + u * (int)blockDim.x + (int)threadIdx.x;
        if (e < n * n) Gs[e] = v[u];
      }
    }
    __syncthreads();
    Gb = Gs;
    ld = n;
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int i = warp; i < n; i += kWarps) {
    float m = -INFINITY;
    for (int j = lane; j < n; j += 32) m = fmaxf(m, Gb[(size_t)i * ld + j]);
    m = warp_max(m);
    float z = 0.f;
    for (int j = lane; j < n; j += 32) z += expf(Gb[(size_t)i * ld + j] - m);
    z = warp_sum(z);
    if (lane == 0) {
      rowm[i] = m;
      rowinv[i] = 1.f / z;
    }
  }
  __syncthreads();
  if (n > 0 && n <= kFinishThreads) {
    // column j of row group g: rows g, g + groups, ... (in order)
    const int groups = kFinishThreads / n;
    const int g = threadIdx.x / n, j = threadIdx.x - g * n;
    if (g < groups) {
      float s = 0.f;
      for (int i = g; i < n; i += groups) s += expf(Gb[(size_t)i * ld + j] - rowm[i]) * rowinv[i];
      part[g * n + j] = s;
    }
    __syncthreads();
    for (int jj = threadIdx.x; jj < n; jj += blockDim.x) {
      float s = 0.f;
      for (int g2 = 0; g2 < groups; ++g2) s += part[g2 * n + jj];
      rr[jj] = s / (float)n;
    }
  } else {
    for (int j = threadIdx.x; j < n; j += blockDim.x) {
      float s = 0.f;
      for (int i = 0; i < n; ++i) s += expf(Gb[(size_t)i * ld + j] - rowm[i]) * rowinv[i];
      rr[j] = s / (float)n;
    }
  }
  __syncthreads();
  // mean(r), fixed-order block sum
  float pt = 0.f;
  for (int j = threadIdx.x; j < n; j += blockDim.x) pt += rr[j];
  pt = warp_sum(pt);
  if (lane == 0) wsum[warp] = pt;
  __syncthreads();
  float tot = 0.f;
  for (int w = 0; w < kWarps; ++w) tot += wsum[w];
  const float mean = n > 0 ? tot / (float)n : 0.f;
  int c = 0;
  for (int j = threadIdx.x; j < n; j += blockDim.x) c += rr[j] > mean;
  for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
  if (lane == 0) wcnt[warp] = c;
  __syncthreads();
  int cnt = 0;
  for (int w = 0; w < kWarps; ++w) cnt += wcnt[w];
  for (int j = threadIdx.x; j < a.N_t_max; j += blockDim.x) {
    const bool in = j < n && (cnt == 0 || rr[j] > mean);
    mask[(size_t)b * a.N_t_max + j] = in ? 1 : 0;
    if (r_out) r_out[(size_t)b * a.N_t_max + j] = j < n ? rr[j] : 0.f;
  }
}

// ---------------------------------------------------------------------------
// inverse row norms: one warp per row
// ---------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(256) inv_norm_kernel(const void* X, size_t rows, int D,
                                                       float* inv) {
  pdl_allow_next();  // a dependent reads inv only after this grid completes
  const size_t row = (size_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= rows) return;
  const T* p = static_cast<const T*>(X) + row * (size_t)D;
  float s = 0.f;
  for (int e = lane * 8; e < D; e += 256) {
    float v[8];
    load8(p + e, v);
#pragma unroll
    for (int q = 0; q < 8; ++q) s = fmaf(v[q], v[q], s);
  }
  s = warp_sum(s);
  if (lane == 0) inv[row] = s > 0.f ? 1.f / sqrtf(s) : 0.f;
}

// ---------------------------------------------------------------------------
// Sec. 4.3 relevance
// ---------------------------------------------------------------------------
// partial sums of normalised visual rows: part[z][b][d] over rows z*chunk..
// (8 rows in flight per step; the adds stay in row order)
template <typename T>
__global__ void __launch_bounds__(256) vis_sum_kernel(const SimArgs a, const float* inv_v,
                                                      float* part, int chunk) {
  const int d = blockIdx.x * 256 + threadIdx.x;
  const int b = blockIdx.y, z = blockIdx.z;
  if (d >= a.D) return;
  const int j0 = z * chunk, j1 = min(a.N_v, j0 + chunk);
  const T* E = static_cast<const T*>(a.emb_v) + (size_t)b * a.N_v * a.D;
  const float* iv = inv_v + (size_t)b * a.N_v;
  float s = 0.f;
  int j = j0;
  for (; j + 8 <= j1; j += 8) {
    float x[8], w[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      x[u] = to_f32(E[(size_t)(j + u) * a.D + d]);
      w[u] = iv[j + u];
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) s = fmaf(x[u], w[u], s);
  }
  for (; j < j1; ++j) s = fmaf(to_f32(E[(size_t)j * a.D + d]), iv[j], s);
  part[((size_t)z * a.B + b) * a.D + d] = s;
}

// One read of the visual rows for both the inverse norms and the normalised
// sum: a CTA per (row chunk z, sample) fetches its rows kNormRows at a time
// with bulk copies (cp.async.bulk, one thread issuing) into shared memory;
// warp w takes row w's squared norm (lane-strided 16-byte pieces, then a warp
// sum) -> inv_v; then every thread adds its 16-byte pieces of the rows, in row
// order, scaled by their inverse norms -> part[z][b][d].
constexpr int kNormRows = 8;
constexpr int kNormThreads = 256;
constexpr int kNormMaxPieces = 4;  // 16-byte pieces per thread: D x esize <= 16 KiB
size_t norm_sum_smem(int D, int esize) { return (size_t)kNormRows * D * esize; }
bool norm_sum_supported(const SimArgs& a) {
  const int es = a.dtype == 0 ? 4 : 2;
  return (size_t)a.D * es <= (size_t)kNormMaxPieces * kNormThreads * 16 && (a.D * es) % 16 == 0;
}

// 8 bf16 of a shared-memory row as fp32 (plain shared load, not the read-only
// global path)
__device__ __forceinline__ void unpack8_shared(const uint8_t* p, float* o) {
  const uint4 u = *reinterpret_cast<const uint4*>(p);
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 f = __bfloat1622float2(h[i]);
    o[2 * i] = f.x;
    o[2 * i + 1] = f.y;
  }
}

template <typename T>
__global__ void __launch_bounds__(kNormThreads) vis_norm_sum_kernel(const SimArgs a, float* inv_v,
                                                                    float* part, int chunk) {
  extern __shared__ __align__(128) uint8_t rows[];
  __shared__ __align__(8) uint64_t bar;
  __shared__ float inv_s[kNormRows];
  constexpr int kVec = 16 / (int)sizeof(T);
  const int z = blockIdx.x, b = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int j0 = z * chunk, j1 = min(a.N_v, j0 + chunk);
  const T* E = static_cast<const T*>(a.emb_v) + (size_t)b * a.N_v * a.D;
  const uint32_t row_bytes = (uint32_t)a.D * (uint32_t)sizeof(T);
  const int n_pieces = (int)(row_bytes / 16);
  float acc[kNormMaxPieces][kVec];
#pragma unroll
  for (int k = 0; k < kNormMaxPieces; ++k)
#pragma unroll
    for (int e = 0; e < kVec; ++e) acc[k][e] = 0.f;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_mbar_init();
  }
  __syncthreads();
  uint32_t phase = 0;
  bool ok = true;
  for (int r0 = j0; r0 < j1; r0 += kNormRows) {
    const int nb = min(kNormRows, j1 - r0);
    if (threadIdx.x == 0) {
      const uint64_t pol = policy_evict_last();  // read again by the relevance Gram
      mbar_arrive_expect_tx(&bar, (uint32_t)nb * row_bytes);
      for (int q = 0; q < nb; ++q)
        bulk_g2s(rows + (size_t)q * row_bytes, E + (size_t)(r0 + q) * a.D, row_bytes, &bar, pol);
    }
    if (ok && !mbar_wait(&bar, phase, a.err)) ok = false;
    phase ^= 1u;
    if (warp < nb) {
      const uint8_t* row = rows + (size_t)warp * row_bytes;
      float sq = 0.f;
      for (int pc = lane; pc < n_pieces; pc += 32) {
        float v[8];
        if constexpr (sizeof(T) == 2) {
          unpack8_shared(row + (size_t)pc * 16, v);
#pragma unroll
          for (int q = 0; q < 8; ++q) sq = fmaf(v[q], v[q], sq);
        } else {
          const float4 f = *reinterpret_cast<const float4*>(row + (size_t)pc * 16);
          sq = fmaf(f.x, f.x, sq);
          sq = fmaf(f.y, f.y, sq);
          sq = fmaf(f.z, f.z, sq);
          sq = fmaf(f.w, f.w, sq);
        }
      }
      sq = warp_sum(sq);
      const float iv = sq > 0.f ? 1.f / sqrtf(sq) : 0.f;
      if (lane == 0) {
        inv_s[warp] = iv;
        inv_v[(size_t)b * a.N_v + r0 + warp] = iv;
      }
    }
    __syncthreads();
    for (int q = 0; q < nb; ++q) {
      const uint8_t* row = rows + (size_t)q * row_bytes;
      const float w = inv_s[q];
#pragma unroll
      for (int k = 0; k < kNormMaxPieces; ++k) {
        const int pc = k * kNormThreads + (int)threadIdx.x;
        if (pc >= n_pieces) continue;
        if constexpr (sizeof(T) == 2) {
          float v[8];
          unpack8_shared(row + (size_t)pc * 16, v);
#pragma unroll
          for (int e = 0; e < 8; ++e) acc[k][e] = fmaf(v[e], w, acc[k][e]);
        } else {
          const float4 f = *reinterpret_cast<const float4*>(row + (size_t)pc * 16);
          acc[k][0] = fmaf(f.x, w, acc[k][0]);
          acc[k][1] = fmaf(f.y, w, acc[k][1]);
          acc[k][2] = fmaf(f.z, w, acc[k][2]);
          acc[k][3] = fmaf(f.w, w, acc[k][3]);
        }
      }
    }
    __syncthreads();  // the rows may be refilled
  }
  float* out = part + ((size_t)z * a.B + b) * a.D;
#pragma unroll
  for (int k = 0; k < kNormMaxPieces; ++k) {
    const int pc = k * kNormThreads + (int)threadIdx.x;
    if (pc >= n_pieces) continue;
#pragma unroll
    for (int e = 0; e < kVec; ++e) out[pc * kVec + e] = acc[k][e];
  }
}

// sum[b][d] = sum over the row chunks z of part[z][b][d] (fixed order)
__global__ void __launch_bounds__(256) vis_sum_reduce_kernel(const SimArgs a, const float* part,
                                                             int nz, float* sum) {
  const int d = blockIdx.x * 256 + threadIdx.x;
  const int b = blockIdx.y;
  if (d >= a.D) return;
  float s = 0.f;
  for (int z = 0; z < nz; ++z) s += part[((size_t)z * a.B + b) * a.D + d];
  sum[(size_t)b * a.D + d] = s;
}

// mu_i and 1/|t_i| for the text rows (one warp per row, 8 elements per lane step)
template <typename T>
__global__ void __launch_bounds__(256) text_mu_kernel(const SimArgs a, const float* sum,
                                                      float* mu, float* invt) {
  const int b = blockIdx.y;
  const int i = blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (i >= a.N_t_max) return;
  const int tl = min(max(a.text_len[b], 0), a.N_t_max);
  if (i >= tl) {
    if (lane == 0) {
      mu[(size_t)b * a.N_t_max + i] = 0.f;
      invt[(size_t)b * a.N_t_max + i] = 0.f;
    }
    return;
  }
  const T* t = static_cast<const T*>(a.emb_t) + ((size_t)b * a.N_t_max + i) * a.D;
  const float* sv = sum + (size_t)b * a.D;
  float ss = 0.f, dt = 0.f;
  for (int d = lane * 8; d < a.D; d += 256) {
    float x[8];
    load8(t + d, x);
    const float4 s0 = *reinterpret_cast<const float4*>(sv + d);
    const float4 s1 = *reinterpret_cast<const float4*>(sv + d + 4);
    const float sw[8] = {s0.x, s0.y, s0.z, s0.w, s1.x, s1.y, s1.z, s1.w};
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      ss = fmaf(x[q], x[q], ss);
      dt = fmaf(x[q], sw[q], dt);
    }
  }
  ss = warp_sum(ss);
  dt = warp_sum(dt);
  if (lane == 0) {
    const float iv = ss > 0.f ? 1.f / sqrtf(ss) : 0.f;
    invt[(size_t)b * a.N_t_max + i] = iv;
    mu[(size_t)b * a.N_t_max + i] = dt * iv / (float)a.N_v;
  }
}

// p_j = max over critical rows of cos - mu; CTA = 64 visual rows x all text rows
template <typename T>
__global__ void __launch_bounds__(256) relevance_kernel(const SimArgs a, const uint8_t* mask,
                                                        const float* inv_v, const float* mu,
                                                        const float* invt, float* p) {
  __shared__ __align__(16) SimtSmem sm;
  __shared__ const T* arow[kSimtBM];
  __shared__ const T* brow[kSimtBN];
  __shared__ float red[8][kSimtBN];
  const int b = blockIdx.y, c0 = blockIdx.x * kSimtBN;
  const int tl = min(max(a.text_len[b], 0), a.N_t_max);
  const int rg = threadIdx.x >> 4, kg = threadIdx.x & 15;
  float best[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
  if (threadIdx.x < kSimtBN) {
    const int j = c0 + threadIdx.x;
    brow[threadIdx.x] = j < a.N_v ? row_ptr<T>(a.emb_v, (size_t)b * a.N_v + j, a.D) : nullptr;
  }
  for (int r0 = 0; r0 < tl; r0 += kSimtBM) {
    __syncthreads();
    if (threadIdx.x < kSimtBM) {
      const int i = r0 + threadIdx.x;
      const bool in = i < tl && mask[(size_t)b * a.N_t_max + i] != 0;
      arow[threadIdx.x] = in ? row_ptr<T>(a.emb_t, (size_t)b * a.N_t_max + i, a.D) : nullptr;
    }
    __syncthreads();
    float acc[8][4];
    simt_gemm_nt<T>(arow, brow, a.D, sm, acc);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int r = rg + 16 * i;
      if (arow[r] == nullptr) continue;
      const float it = invt[(size_t)b * a.N_t_max + r0 + r], m = mu[(size_t)b * a.N_t_max + r0 + r];
#pragma unroll
      for (int jj = 0; jj < 4; ++jj) {
        const int j = c0 + kg + 16 * jj;
        if (j < a.N_v) best[jj] = fmaxf(best[jj], acc[i][jj] * it * inv_v[(size_t)b * a.N_v + j] - m);
      }
    }
  }
  // max across the 16 row groups
#pragma unroll
  for (int jj = 0; jj < 4; ++jj) best[jj] = fmaxf(best[jj], __shfl_xor_sync(0xffffffffu, best[jj], 16));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane < 16)
#pragma unroll
    for (int jj = 0; jj < 4; ++jj) red[warp][lane + 16 * jj] = best[jj];
  __syncthreads();
  if (threadIdx.x < kSimtBN) {
    const int j = c0 + threadIdx.x;
    float m = -INFINITY;
    for (int w = 0; w < 8; ++w) m = fmaxf(m, red[w][threadIdx.x]);
    if (j < a.N_v) p[(size_t)b * a.N_v + j] = m;
  }
}

// ---------------------------------------------------------------------------
// Sec. 4.3 merge
// ---------------------------------------------------------------------------
// Per sample (one CTA of 1024 threads): the kept-position map kpos[b][j] =
// a if j == keep[b][a], else -1, and, when `pruned` is given, the rows not
// kept in ascending order, pruned[b][0 .. N_v - keep) (ballot compaction).
__global__ void __launch_bounds__(1024) merge_index_kernel(const int* keep_idx, int keep, int N_v, int* kpos,
                                                           int* pruned, unsigned* err) {
  __shared__ int warp_tot[32];
  const int b = blockIdx.x;
  int* kp = kpos + (size_t)b * N_v;
  const int* ki = keep_idx + (size_t)b * keep;
  for (int j = threadIdx.x; j < N_v; j += blockDim.x) kp[j] = -1;
  __syncthreads();
  for (int q = threadIdx.x; q < keep; q += blockDim.x) {
    const int j = ki[q];
    if (j < 0 || j >= N_v || (q > 0 && ki[q - 1] >= j)) {
      set_error(err, kErrBadDeviceArg);
      continue;
    }
    kp[j] = q;
  }
  if (pruned == nullptr) return;
  __syncthreads();  // the map is complete (global writes of this block)
  const int n_pruned = N_v - keep;
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
__device__ __forceinline__ bool better(float v, int i, float bv, int bi) {
  return v > bv || (v == bv && i < bi);
}

// argmax over one split of the kept columns for a tile of 128 visual rows
template <typename T>
__global__ void __launch_bounds__(256) merge_argmax_kernel(const SimArgs a, const int* keep_idx,
                                                           int keep, const float* inv_v,
                                                           const int* kpos, int n_split,
                                                           float* ws_best, int* ws_bidx) {
  __shared__ __align__(16) SimtSmem sm;
  __shared__ const T* arow[kSimtBM];
  __shared__ const T* brow[kSimtBN];
  __shared__ float kinv[kSimtBN];
  const int b = blockIdx.y, r0 = blockIdx.x * kSimtBM, split = blockIdx.z;
  const int ntile = (keep + kSimtBN - 1) / kSimtBN;
  const int t0 = (int)((long long)ntile * split / n_split), t1 = (int)((long long)ntile * (split + 1) / n_split);
  const int rg = threadIdx.x >> 4, kg = threadIdx.x & 15;
  if (threadIdx.x < kSimtBM) {
    const int j = r0 + threadIdx.x;
    const bool pruned = j < a.N_v && kpos[(size_t)b * a.N_v + j] < 0;
    arow[threadIdx.x] = pruned ? row_ptr<T>(a.emb_v, (size_t)b * a.N_v + j, a.D) : nullptr;
  }
  float bv[8];
  int bi[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    bv[i] = -INFINITY;
    bi[i] = 0x7fffffff;
  }
  for (int t = t0; t < t1; ++t) {
    const int a0 = t * kSimtBN;
    __syncthreads();
    if (threadIdx.x < kSimtBN) {
      const int ap = a0 + threadIdx.x;
      if (ap < keep) {
        const int j = keep_idx[(size_t)b * keep + ap];
        const bool ok = j >= 0 && j < a.N_v;
        brow[threadIdx.x] = ok ? row_ptr<T>(a.emb_v, (size_t)b * a.N_v + j, a.D) : nullptr;
        kinv[threadIdx.x] = ok ? inv_v[(size_t)b * a.N_v + j] : 0.f;
      } else {
        brow[threadIdx.x] = nullptr;
        kinv[threadIdx.x] = 0.f;
      }
    }
    __syncthreads();
    float acc[8][4];
    simt_gemm_nt<T>(arow, brow, a.D, sm, acc);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
#pragma unroll
      for (int jj = 0; jj < 4; ++jj) {
        const int ap = a0 + kg + 16 * jj;
        if (ap < keep) {
          const float v = acc[i][jj] * kinv[kg + 16 * jj];
          if (better(v, ap, bv[i], bi[i])) {
            bv[i] = v;
            bi[i] = ap;
          }
        }
      }
    }
  }
  // combine the 16 lanes of each row group
#pragma unroll
  for (int i = 0; i < 8; ++i) {
#pragma unroll
    for (int o = 8; o > 0; o >>= 1) {
      const float ov = __shfl_xor_sync(0xffffffffu, bv[i], o);
      const int oi = __shfl_xor_sync(0xffffffffu, bi[i], o);
      if (better(ov, oi, bv[i], bi[i])) {
        bv[i] = ov;
        bi[i] = oi;
      }
    }
    const int j = r0 + rg + 16 * i;
    if (kg == 0 && j < a.N_v) {
      ws_best[((size_t)split * a.B + b) * a.N_v + j] = bv[i];
      ws_bidx[((size_t)split * a.B + b) * a.N_v + j] = bi[i];
    }
  }
}

// assign[b][j]: own position for kept rows, best over splits for the others
__global__ void merge_assign_kernel(const SimArgs a, const int* kpos, int n_split,
                                    const float* ws_best, const int* ws_bidx, int* assign) {
  pdl_wait_prior();  // the partials come from the Gram before
  pdl_allow_next();
  const size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (size_t)a.B * a.N_v) return;
  const int kp = kpos[i];
  if (kp >= 0) {
    assign[i] = kp;
    return;
  }
  float bv = -INFINITY;
  int bi = 0x7fffffff;
  for (int s = 0; s < n_split; ++s) {
    const float v = ws_best[(size_t)s * a.B * a.N_v + i];
    const int ix = ws_bidx[(size_t)s * a.B * a.N_v + i];
    if (better(v, ix, bv, bi)) {
      bv = v;
      bi = ix;
    }
  }
  // a zero or non-finite row compares equal everywhere: lowest position
  assign[i] = bi == 0x7fffffff ? 0 : bi;
}

// merged[b][a] = (sum of rows j with assign[b][j] == a, ascending j) / count.
// The member lists come from a counting sort per sample: counts (atomics),
// exclusive offsets, unordered fill. One CTA per kept row orders its members
// by rank (ascending row index, so the sum order is fixed), fetches the member
// rows with bulk copies (cp.async.bulk, one thread issuing) into a ring of
// shared-memory row slots, SLOTS rows per batch, and sums them slot by slot in
// rank order, each thread over its 16-byte pieces of the row. A centroid with
// more members than the sort buffer takes them from a scan of assign in
// windows (ascending by construction). Each CTA is a short chain of dependent
// steps, so the configuration is chosen for CTAs resident per SM: rows of at
// most 8 KiB take 128 threads with 4 pieces each (8 CTAs per SM), longer rows
// 256 threads (up to 8192 elements).
template <int THR, int PIECES, int SLOTS, int SORT, int MINB>
struct MeanCfg {
  static constexpr int kThreads = THR, kWarps = THR / 32, kPieces = PIECES, kSlots = SLOTS, kSort = SORT,
                       kMinBlocks = MINB;
};
using MeanSmall = MeanCfg<128, 4, 3, 256, 8>;       // row bytes <= 128 * 4 * 16
using MeanBf16 = MeanCfg<256, 4, 4, 1024, 4>;       // bf16 rows <= 8192 elements
using MeanF32 = MeanCfg<256, 8, 4, 1024, 2>;        // fp32 rows <= 8192 elements
constexpr int kMeanSmallRowBytes = 128 * 4 * 16;
constexpr int kSortSmemKeep = 6144;  // centroids whose counters the sort keeps in shared memory (48 KiB)
template <typename C> size_t merge_mean_smem(int row_bytes) { return (size_t)C::kSlots * row_bytes; }

// Counting sort of one sample's rows by centroid (one CTA of 1024 threads):
// count[b][a] = rows assigned to a, offset[b][.] its exclusive scan, and
// members[b][offset[a] ..] the rows of a in no particular order (the means
// rank them). The block-wide barriers order the phases (global memory of this
// block only).
template <bool kSmem>
__global__ void __launch_bounds__(1024) merge_sort_kernel(const int* assign, int N_v, int keep, int* count,
                                                          int* offset, int* cursor, int* members) {
  extern __shared__ int sort_sm[];  // kSmem: counts [keep], then offsets / cursors [keep]
  __shared__ uint32_t warp_tot[32];
  __shared__ uint32_t carry;
  pdl_wait_prior();  // the assignment comes from the kernel before
  pdl_allow_next();
  const int b = blockIdx.x;
  const int* as = assign + (size_t)b * N_v;
  int* cnt_g = count + (size_t)b * keep;
  int* off_g = offset + (size_t)b * keep;
  // the counters: shared memory for at most kSortSmemKeep centroids, else the
  // global scratch (cursor)
  int* cnt = kSmem ? sort_sm : cnt_g;
  int* cur = kSmem ? sort_sm + keep : cursor + (size_t)b * keep;
  for (int q = threadIdx.x; q < keep; q += blockDim.x) {
    cnt[q] = 0;
    cur[q] = 0;
  }
  if (threadIdx.x == 0) carry = 0;
  __syncthreads();
  for (int j = threadIdx.x; j < N_v; j += blockDim.x) {
    const int ap = as[j];
    if (ap >= 0 && ap < keep) atomicAdd(&cnt[ap], 1);
  }
  __syncthreads();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int a0 = 0; a0 < keep; a0 += 1024) {
    const int ap = a0 + threadIdx.x;
    const uint32_t v = ap < keep ? (uint32_t)cnt[ap] : 0u;
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
    if (ap < keep) {
      const int o = (int)(carry + warp_tot[warp] + incl - v);
      off_g[ap] = o;
      if (kSmem) {
        cnt_g[ap] = (int)v;
        cur[ap] = o;  // the fill's running position
      }
    }
    __syncthreads();
    if (threadIdx.x == 1023) carry += warp_tot[31] + incl;
    __syncthreads();
  }
  for (int j = threadIdx.x; j < N_v; j += blockDim.x) {
    const int ap = as[j];
    if (ap >= 0 && ap < keep) {
      const int pos = kSmem ? atomicAdd(&cur[ap], 1) : off_g[ap] + atomicAdd(&cur[ap], 1);
      members[(size_t)b * N_v + pos] = j;
    }
  }
}

// the addition of 16 raw bytes of a row to Acc values (8 bf16 or 4 fp32)
__device__ __forceinline__ void add16(float* acc, const uint4& u, const __nv_bfloat16*) {
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 f = __bfloat1622float2(h[i]);
    acc[2 * i] += f.x;
    acc[2 * i + 1] += f.y;
  }
}
__device__ __forceinline__ void add16(double* acc, const uint4& u, const float*) {
  acc[0] += (double)__uint_as_float(u.x);
  acc[1] += (double)__uint_as_float(u.y);
  acc[2] += (double)__uint_as_float(u.z);
  acc[3] += (double)__uint_as_float(u.w);
}
// 16 bytes of a row from Acc values, rounded to nearest even
__device__ __forceinline__ void store16(__nv_bfloat16* p, const float* v) {
  uint4 u;
  __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&u);
#pragma unroll
  for (int i = 0; i < 4; ++i) h[i] = __floats2bfloat162_rn(v[2 * i], v[2 * i + 1]);
  *reinterpret_cast<uint4*>(p) = u;
}
__device__ __forceinline__ void store16(float* p, const double* v) {
  *reinterpret_cast<float4*>(p) = make_float4((float)v[0], (float)v[1], (float)v[2], (float)v[3]);
}

template <typename T, typename Acc, typename C>
__global__ void __launch_bounds__(C::kThreads, C::kMinBlocks)
    merge_mean_kernel(const SimArgs a, const int* assign, const int* count, const int* offset,
                      const int* members_all, int keep, void* merged) {
  constexpr int kMeanThreads = C::kThreads, kMeanWarps = C::kWarps, kMeanSort = C::kSort,
                kMeanSlots = C::kSlots;
  extern __shared__ __align__(128) uint8_t slots[];  // kMeanSlots rows
  __shared__ int members[kMeanSort];
  __shared__ int unsorted[kMeanSort];
  __shared__ __align__(8) uint64_t bar;
  __shared__ int wcount[kMeanWarps];
  constexpr int kVec = 16 / (int)sizeof(T);  // elements per 16-byte piece
  constexpr int kPieces = C::kPieces;
  const int ap = blockIdx.x, b = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  pdl_wait_prior();  // the member lists come from the sort before
  const T* E = static_cast<const T*>(a.emb_v) + (size_t)b * a.N_v * a.D;
  T* out = static_cast<T*>(merged) + ((size_t)b * keep + ap) * a.D;
  const uint32_t row_bytes = (uint32_t)a.D * (uint32_t)sizeof(T);
  const int n_pieces = a.D / kVec;
  Acc acc[kPieces][kVec];
#pragma unroll
  for (int k = 0; k < kPieces; ++k)
#pragma unroll
    for (int e = 0; e < kVec; ++e) acc[k][e] = Acc(0);
  // count and offset issued together: the member list depends on both
  const int n_all = count[(size_t)b * keep + ap];
  const int off0 = offset[(size_t)b * keep + ap];
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_mbar_init();
  }
  uint32_t phase = 0;
  bool ok = true;
  // adds rows members[0..n) in order: batches of kMeanSlots bulk copies
  auto add_rows = [&](int n) {
    for (int m0 = 0; m0 < n; m0 += kMeanSlots) {
      const int nb = min(kMeanSlots, n - m0);
      if (threadIdx.x == 0 && ok) {
        const uint64_t pol = policy_evict_first();
        mbar_arrive_expect_tx(&bar, (uint32_t)nb * row_bytes);
        for (int q = 0; q < nb; ++q)
          bulk_g2s(slots + (size_t)q * row_bytes, E + (size_t)members[m0 + q] * a.D, row_bytes, &bar, pol);
      }
      if (ok && !mbar_wait(&bar, phase, a.err)) ok = false;
      phase ^= 1u;
      if (ok) {
        for (int q = 0; q < nb; ++q) {
          const uint8_t* row = slots + (size_t)q * row_bytes;
#pragma unroll
          for (int k = 0; k < kPieces; ++k) {
            const int pc = k * kMeanThreads + (int)threadIdx.x;
            if (pc < n_pieces) add16(acc[k], *reinterpret_cast<const uint4*>(row + (size_t)pc * 16), E);
          }
        }
      }
      __syncthreads();  // the slots may be refilled
    }
  };
  if (n_all <= kMeanSort) {
    const int* src = members_all + (size_t)b * a.N_v + off0;
    for (int m = threadIdx.x; m < n_all; m += kMeanThreads) unsorted[m] = src[m];
    __syncthreads();
    // rank = number of smaller row indices (they are distinct)
    for (int m = threadIdx.x; m < n_all; m += kMeanThreads) {
      const int v = unsorted[m];
      int rank = 0;
      for (int q = 0; q < n_all; ++q) rank += unsorted[q] < v;
      members[rank] = v;
    }
    __syncthreads();
    add_rows(n_all);
  } else {
    // many members: scan assign in windows, members in ascending order
    const int* as = assign + (size_t)b * a.N_v;
    int base = 0;
    for (int j0 = 0; j0 < a.N_v; j0 += kMeanThreads) {
      const int j = j0 + threadIdx.x;
      const bool hit = j < a.N_v && as[j] == ap;
      const unsigned bal = __ballot_sync(0xffffffffu, hit);
      if (lane == 0) wcount[warp] = __popc(bal);
      __syncthreads();
      int off = 0, tot = 0;
      for (int w = 0; w < kMeanWarps; ++w) {
        off += w < warp ? wcount[w] : 0;
        tot += wcount[w];
      }
      if (hit) members[base + off + __popc(bal & ((1u << lane) - 1u))] = j;
      __syncthreads();
      base += tot;
      if (base > kMeanSort - kMeanThreads || j0 + kMeanThreads >= a.N_v) {
        add_rows(base);
        base = 0;
      }
    }
  }
#pragma unroll
  for (int k = 0; k < kPieces; ++k) {
    const int pc = k * kMeanThreads + (int)threadIdx.x;
    if (pc >= n_pieces) continue;
    Acc v[kVec];
#pragma unroll
    for (int e = 0; e < kVec; ++e) v[e] = n_all > 0 ? acc[k][e] / (Acc)n_all : Acc(0);
    store16(out + (size_t)pc * kVec, v);
  }
}

}  // namespace

cudaError_t crit_text_launch(const SimArgs& a, uint8_t* mask, float* r_out, float* G,
                             cudaStream_t s) {
  dim3 g((a.N_t_max + kSimtBN - 1) / kSimtBN, (a.N_t_max + kSimtBM - 1) / kSimtBM, a.B);
  int parts = 1;
  if (a.dtype == 0) {
    crit_gram_kernel<float><<<g, 256, 0, s>>>(a, G);
  } else if (crit_gram_tc_supported(a)) {
    cudaError_t e = crit_gram_tc_launch(a, G, s);
    if (e != cudaSuccess) return e;
    parts = crit_splits(a.N_t_max, a.D, a.dtype);
    static_assert(kCritMaxSplits <= kCritMaxParts, "text Gram parts");
    const size_t n = (size_t)a.B * a.N_t_max * a.N_t_max;
    if (parts > 1) crit_parts_sum_kernel<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(G, n, parts);
  } else {
    crit_gram_kernel<__nv_bfloat16><<<g, 256, 0, s>>>(a, G);
  }
  static std::atomic<bool> configured[64];  // per device, zero-initialised
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64 && !configured[dev]) {
    const int lim = (3 * kFinishSmemNt + kFinishThreads + kFinishSmemNt * kFinishSmemNt) * (int)sizeof(float);
    cudaError_t e = cudaFuncSetAttribute(crit_finish_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, lim);
    if (e != cudaSuccess) return e;
    configured[dev] = true;
  }
  size_t smem = (3 * (size_t)a.N_t_max + kFinishThreads) * sizeof(float);
  if (a.N_t_max <= kFinishSmemNt) smem += (size_t)a.N_t_max * a.N_t_max * sizeof(float);
  if (smem > (size_t)(3 * kFinishSmemNt + kFinishThreads + kFinishSmemNt * kFinishSmemNt) * sizeof(float))
    return cudaErrorInvalidValue;  // N_t_max beyond what the shared-memory layout holds
  (void)parts;
  crit_finish_kernel<<<a.B, kFinishThreads, smem, s>>>(a, G, mask, r_out);
  return cudaGetLastError();
}

// 1/|e_j| (0 for a zero row) of the kept rows j = keep_idx[b][q] only, into
// inv_v[b][j] (the merge reads no other): a warp per row; an index out of range
// is reported and skipped.
template <typename T>
__global__ void __launch_bounds__(256) kept_inv_norm_kernel(const void* X, const int* keep_idx, int keep,
                                                            int N_v, int D, size_t rows, float* inv_v,
                                                            unsigned* err) {
  const size_t row = (size_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= rows) return;
  const size_t b = row / (size_t)keep;
  const int j = keep_idx[row];
  if (j < 0 || j >= N_v) {
    if (lane == 0) set_error(err, kErrBadDeviceArg);
    return;
  }
  const T* p = static_cast<const T*>(X) + (b * (size_t)N_v + (size_t)j) * (size_t)D;
  float s = 0.f;
  for (int e = lane * 8; e < D; e += 256) {
    float v[8];
    load8(p + e, v);
#pragma unroll
    for (int q = 0; q < 8; ++q) s = fmaf(v[q], v[q], s);
  }
  s = warp_sum(s);
  if (lane == 0) inv_v[b * (size_t)N_v + (size_t)j] = s > 0.f ? 1.f / sqrtf(s) : 0.f;
}

cudaError_t kept_inv_norm_launch(const SimArgs& a, const int* keep_idx, int keep, float* inv_v,
                                 cudaStream_t s) {
  const size_t rows = (size_t)a.B * keep;
  const unsigned grid = (unsigned)((rows + 7) / 8);
  if (a.dtype == 0)
    kept_inv_norm_kernel<float><<<grid, 256, 0, s>>>(a.emb_v, keep_idx, keep, a.N_v, a.D, rows, inv_v, a.err);
  else
    kept_inv_norm_kernel<__nv_bfloat16><<<grid, 256, 0, s>>>(a.emb_v, keep_idx, keep, a.N_v, a.D, rows, inv_v,
                                                            a.err);
  return cudaGetLastError();
}

cudaError_t vis_inv_norm_launch(const SimArgs& a, float* inv_v, cudaStream_t s) {
  const size_t rows = (size_t)a.B * a.N_v;
  const unsigned grid = (unsigned)((rows + 7) / 8);
  if (a.dtype == 0)
    inv_norm_kernel<float><<<grid, 256, 0, s>>>(a.emb_v, rows, a.D, inv_v);
  else
    inv_norm_kernel<__nv_bfloat16><<<grid, 256, 0, s>>>(a.emb_v, rows, a.D, inv_v);
  return cudaGetLastError();
}

cudaError_t relevance_launch(const SimArgs& a, const uint8_t* mask, float* inv_v, float* p,
                             float* ws_sum, float* ws_mu, float* ws_invt, int n_split,
                             int num_sms, cudaStream_t s, cudaEvent_t mask_ready) {
  // bf16 with at most 128 text rows: the text rows' inverse norms, one
  // tensor-core read of the visual rows (norms, cosines and de-meaning sums)
  // and a small max kernel
  if (relevance_tc_supported(a)) {
    const size_t rows = (size_t)a.B * a.N_t_max;
    inv_norm_kernel<__nv_bfloat16><<<(unsigned)((rows + 7) / 8), 256, 0, s>>>(a.emb_t, rows, a.D, ws_invt);
    return relevance_tc_launch(a, mask, ws_invt, inv_v, p, ws_sum, num_sms, s, mask_ready);
  }
  const int chunk = (a.N_v + n_split - 1) / n_split;
  dim3 g1((a.D + 255) / 256, a.B, n_split);
  dim3 g2((a.N_t_max + 7) / 8, a.B);
  dim3 g3((a.N_v + kSimtBN - 1) / kSimtBN, a.B);
  // ws_sum holds n_split partial sums followed by their total
  float* total = ws_sum + (size_t)n_split * a.B * a.D;
  dim3 g4((a.D + 255) / 256, a.B);
  // the inverse norms of the visual rows and their normalised sum, in one read
  // where the rows fit the shared-memory batch, else in two passes
  const bool fused = norm_sum_supported(a);
  if (fused) {
    static std::atomic<bool> configured[64];  // per device, zero-initialised
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && !configured[dev]) {
      const int lim = kNormMaxPieces * kNormThreads * 16 * kNormRows;
      cudaError_t e = cudaFuncSetAttribute(vis_norm_sum_kernel<float>,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, lim);
      if (e == cudaSuccess)
        e = cudaFuncSetAttribute(vis_norm_sum_kernel<__nv_bfloat16>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, lim);
      if (e != cudaSuccess) return e;
      configured[dev] = true;
    }
    const size_t smem = norm_sum_smem(a.D, a.dtype == 0 ? 4 : 2);
    dim3 gn(n_split, a.B);
    if (a.dtype == 0)
      vis_norm_sum_kernel<float><<<gn, kNormThreads, smem, s>>>(a, inv_v, ws_sum, chunk);
    else
      vis_norm_sum_kernel<__nv_bfloat16><<<gn, kNormThreads, smem, s>>>(a, inv_v, ws_sum, chunk);
  } else {
    cudaError_t e = vis_inv_norm_launch(a, inv_v, s);
    if (e != cudaSuccess) return e;
  }
  if (a.dtype == 0) {
    if (!fused) vis_sum_kernel<float><<<g1, 256, 0, s>>>(a, inv_v, ws_sum, chunk);
    vis_sum_reduce_kernel<<<g4, 256, 0, s>>>(a, ws_sum, n_split, total);
    text_mu_kernel<float><<<g2, 256, 0, s>>>(a, total, ws_mu, ws_invt);
    if (mask_ready != nullptr) {
      const cudaError_t e = cudaStreamWaitEvent(s, mask_ready, 0);  // the first kernel that reads the mask
      if (e != cudaSuccess) return e;
    }
    relevance_kernel<float><<<g3, 256, 0, s>>>(a, mask, inv_v, ws_mu, ws_invt, p);
  } else {
    if (!fused) vis_sum_kernel<__nv_bfloat16><<<g1, 256, 0, s>>>(a, inv_v, ws_sum, chunk);
    vis_sum_reduce_kernel<<<g4, 256, 0, s>>>(a, ws_sum, n_split, total);
    text_mu_kernel<__nv_bfloat16><<<g2, 256, 0, s>>>(a, total, ws_mu, ws_invt);
    if (mask_ready != nullptr) {
      const cudaError_t e = cudaStreamWaitEvent(s, mask_ready, 0);
      if (e != cudaSuccess) return e;
    }
    relevance_kernel<__nv_bfloat16><<<g3, 256, 0, s>>>(a, mask, inv_v, ws_mu, ws_invt, p);
  }
  return cudaGetLastError();
}

cudaError_t merge_launch(const SimArgs& a, const int* keep_idx, int keep, const float* inv_v,
                         int* assign, void* merged, float* ws_best, int* ws_bidx, int n_split,
                         int* ws_pruned, void* ws_perm, int num_sms, cudaStream_t s, bool index_ready) {
  // kpos lives in `assign` until the final assignment overwrites it: it is
  // read by merge_argmax_kernel and merge_assign_kernel (same index only).
  int* kpos = assign;
  const size_t nb = (size_t)a.B * a.N_v;
  const int tc_split = merge_tc_split(a.B, a.N_v, keep, num_sms);
  const bool tc = ws_pruned != nullptr && ws_perm != nullptr && merge_tc_supported(a, keep, tc_split);
  // the kept-position map, and the pruned rows for the tensor-core Gram
  if (!index_ready)
    merge_index_kernel<<<a.B, 1024, 0, s>>>(keep_idx, keep, a.N_v, kpos, tc ? ws_pruned : nullptr, a.err);
  if (tc) {
    cudaError_t e = merge_argmax_tc_launch(a, keep_idx, keep, inv_v, ws_pruned, ws_perm, tc_split, ws_best,
                                           ws_bidx, num_sms, &n_split, s);
    if (e != cudaSuccess) return e;
  } else {
    dim3 g((a.N_v + kSimtBM - 1) / kSimtBM, a.B, n_split);
    if (a.dtype == 0)
      merge_argmax_kernel<float><<<g, 256, 0, s>>>(a, keep_idx, keep, inv_v, kpos, n_split, ws_best, ws_bidx);
    else
      merge_argmax_kernel<__nv_bfloat16><<<g, 256, 0, s>>>(a, keep_idx, keep, inv_v, kpos, n_split, ws_best,
                                                           ws_bidx);
  }
  cudaError_t el = launch_pdl(merge_assign_kernel, dim3((unsigned)((nb + 255) / 256)), dim3(256), 0, s, a,
                              (const int*)kpos, n_split, (const float*)ws_best, (const int*)ws_bidx, assign);
  if (el != cudaSuccess) return el;
  if (merged != nullptr) {
    // counting sort of the rows by centroid; the scratch reuses ws_best/ws_bidx
    // (the argmax partials are consumed by merge_assign_kernel above)
    int* cnt = ws_bidx;
    int* off = cnt + (size_t)a.B * keep;
    int* cur = off + (size_t)a.B * keep;
    int* mem = reinterpret_cast<int*>(ws_best);
    cudaError_t es = keep <= kSortSmemKeep
                         ? launch_pdl(merge_sort_kernel<true>, dim3(a.B), dim3(1024),
                                      (size_t)2 * keep * sizeof(int), s, (const int*)assign, a.N_v, keep, cnt,
                                      off, cur, mem)
                         : launch_pdl(merge_sort_kernel<false>, dim3(a.B), dim3(1024), 0, s, (const int*)assign,
                                      a.N_v, keep, cnt, off, cur, mem);
    if (es != cudaSuccess) return es;
    dim3 gm(keep, a.B);
    static std::atomic<bool> configured[64];  // per device, zero-initialised
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && !configured[dev]) {
      cudaError_t e = cudaFuncSetAttribute(merge_mean_kernel<float, double, MeanF32>,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)merge_mean_smem<MeanF32>(8192 * 4));
      if (e == cudaSuccess)
        e = cudaFuncSetAttribute(merge_mean_kernel<__nv_bfloat16, float, MeanBf16>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)merge_mean_smem<MeanBf16>(8192 * 2));
      if (e != cudaSuccess) return e;
      configured[dev] = true;
    }
    const int row_bytes = a.D * (a.dtype == 0 ? 4 : 2);
    cudaError_t em;
    if (row_bytes <= kMeanSmallRowBytes) {
      const size_t smem = merge_mean_smem<MeanSmall>(row_bytes);
      if (a.dtype == 0)
        em = launch_pdl(merge_mean_kernel<float, double, MeanSmall>, gm, dim3(MeanSmall::kThreads), smem, s, a,
                        (const int*)assign, (const int*)cnt, (const int*)off, (const int*)mem, keep, merged);
      else
        em = launch_pdl(merge_mean_kernel<__nv_bfloat16, float, MeanSmall>, gm, dim3(MeanSmall::kThreads), smem,
                        s, a, (const int*)assign, (const int*)cnt, (const int*)off, (const int*)mem, keep, merged);
    } else if (a.dtype == 0) {
      em = launch_pdl(merge_mean_kernel<float, double, MeanF32>, gm, dim3(MeanF32::kThreads),
                      merge_mean_smem<MeanF32>(row_bytes), s, a, (const int*)assign, (const int*)cnt,
                      (const int*)off, (const int*)mem, keep, merged);
    } else {
      em = launch_pdl(merge_mean_kernel<__nv_bfloat16, float, MeanBf16>, gm, dim3(MeanBf16::kThreads),
                      merge_mean_smem<MeanBf16>(row_bytes), s, a, (const int*)assign, (const int*)cnt,
                      (const int*)off, (const int*)mem, keep, merged);
    }
    if (em != cudaSuccess) return em;
  }
  return cudaGetLastError();
}

}  // namespace provip
