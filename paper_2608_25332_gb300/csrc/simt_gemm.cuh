// CUDA-core (FFMA) tile of an "NT" product C = A * B^T used by the fp32 path
// and by the small contractions that do not warrant tensor cores.
//
// One 256-thread CTA computes a 128 x 64 tile. Thread (rg = tid / 16,
// kg = tid % 16) owns rows rg + 16 i (i < 8) and columns kg + 16 j (j < 4), so
// a row's 64 columns live in 16 consecutive lanes (xor-shuffles over 1..8
// reduce across them) and the column reads of B are bank-conflict free.
// A and B rows are given as per-row pointers (a null pointer is a zero row), so
// strided heads, gathered rows and padded tails need no copies.
#pragma once

#include "common.cuh"

namespace provip {

constexpr int kSimtBM = 128;
constexpr int kSimtBN = 64;
constexpr int kSimtKT = 32;
constexpr int kSimtLD = kSimtKT + 4;  // padded smem row (floats)

struct SimtSmem {
  float A[kSimtBM][kSimtLD];
  float B[kSimtBN][kSimtLD];
};

// acc[i][j] = <arow[rg + 16 i], brow[kg + 16 j]> over kdim elements (kdim % 8 == 0).
template <typename T>
__device__ __forceinline__ void simt_gemm_nt(const T* const* arow, const T* const* brow, int kdim,
                                             SimtSmem& sm, float acc[8][4]) {
  const int tid = threadIdx.x, rg = tid >> 4, kg = tid & 15;
#pragma unroll
  for (int i = 0; i < 8; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
  for (int k0 = 0; k0 < kdim; k0 += kSimtKT) {
    for (int g = tid; g < kSimtBM * (kSimtKT / 8); g += 256) {
      const int r = g >> 2, c = (g & 3) * 8;
      float v[8];
      const T* p = arow[r];
      if (p != nullptr && k0 + c < kdim) {
        load8(p + k0 + c, v);
      } else {
#pragma unroll
        for (int e = 0; e < 8; ++e) v[e] = 0.f;
      }
      *reinterpret_cast<float4*>(&sm.A[r][c]) = make_float4(v[0], v[1], v[2], v[3]);
      *reinterpret_cast<float4*>(&sm.A[r][c + 4]) = make_float4(v[4], v[5], v[6], v[7]);
    }
    for (int g = tid; g < kSimtBN * (kSimtKT / 8); g += 256) {
      const int r = g >> 2, c = (g & 3) * 8;
      float v[8];
      const T* p = brow[r];
      if (p != nullptr && k0 + c < kdim) {
        load8(p + k0 + c, v);
      } else {
#pragma unroll
        for (int e = 0; e < 8; ++e) v[e] = 0.f;
      }
      *reinterpret_cast<float4*>(&sm.B[r][c]) = make_float4(v[0], v[1], v[2], v[3]);
      *reinterpret_cast<float4*>(&sm.B[r][c + 4]) = make_float4(v[4], v[5], v[6], v[7]);
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < kSimtKT; kk += 4) {
      float4 a[8], b[4];
#pragma unroll
      for (int i = 0; i < 8; ++i) a[i] = *reinterpret_cast<const float4*>(&sm.A[rg + 16 * i][kk]);
#pragma unroll
      for (int j = 0; j < 4; ++j) b[j] = *reinterpret_cast<const float4*>(&sm.B[kg + 16 * j][kk]);
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          acc[i][j] = fmaf(a[i].x, b[j].x, acc[i][j]);
          acc[i][j] = fmaf(a[i].y, b[j].y, acc[i][j]);
          acc[i][j] = fmaf(a[i].z, b[j].z, acc[i][j]);
          acc[i][j] = fmaf(a[i].w, b[j].w, acc[i][j]);
        }
    }
    __syncthreads();
  }
}

// reductions across the 16 lanes that share a row group
__device__ __forceinline__ float rowgroup_max(float v) {
#pragma unroll
  for (int o = 8; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float rowgroup_sum(float v) {
#pragma unroll
  for (int o = 8; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

}  // namespace provip
