// Epilogue helpers of the nearest-centroid Grams (Sec. 4.3, last paragraph):
// reading 32-column pieces of a tensor-memory accumulator and keeping each
// row's running (max, first position) over scaled columns.
#pragma once

#include "common.cuh"

namespace provip {

// waits for this thread's tensor-memory loads; v (the destination of the
// last one) is an operand, so that no use of it is scheduled before the wait
__device__ __forceinline__ void tc_wait_ld_into(float* v) {
  asm volatile(
      "tcgen05.wait::ld.sync.aligned;"
      : "+f"(v[0]), "+f"(v[1]), "+f"(v[2]), "+f"(v[3]), "+f"(v[4]), "+f"(v[5]), "+f"(v[6]), "+f"(v[7]),
        "+f"(v[8]), "+f"(v[9]), "+f"(v[10]), "+f"(v[11]), "+f"(v[12]), "+f"(v[13]), "+f"(v[14]),
        "+f"(v[15]), "+f"(v[16]), "+f"(v[17]), "+f"(v[18]), "+f"(v[19]), "+f"(v[20]), "+f"(v[21]),
        "+f"(v[22]), "+f"(v[23]), "+f"(v[24]), "+f"(v[25]), "+f"(v[26]), "+f"(v[27]), "+f"(v[28]),
        "+f"(v[29]), "+f"(v[30]), "+f"(v[31])
      :
      : "memory");
}

// (v, i) beats (bv, bi): larger, or equal at a lower kept position
__device__ __forceinline__ bool merge_better(float v, int i, float bv, int bi) {
  return v > bv || (v == bv && i < bi);
}
// Running (max, first position) of one accumulator row over 32 columns, as
// four interleaved running maxima (independent chains) merged at the end.
struct RowBest {
  float v[4];
  int i[4];
  __device__ __forceinline__ void init() {
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      v[j] = -INFINITY;
      i[j] = 0x7fffffff;
    }
  }
  __device__ __forceinline__ void add32(const float* acc, const float* sk, int q0, int nv, int pos0) {
#pragma unroll
    for (int c = 0; c < 32; c += 4) {
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int q = q0 + c + j;
        const float x = acc[c + j] * sk[c + j];
        if (q < nv && x > v[j]) {  // strict: the first of equal values stays
          v[j] = x;
          i[j] = pos0 + q;
        }
      }
    }
  }
  __device__ __forceinline__ void result(float& bv, int& bi) const {
    bv = v[0];
    bi = i[0];
#pragma unroll
    for (int j = 1; j < 4; ++j)
      if (merge_better(v[j], i[j], bv, bi)) {
        bv = v[j];
        bi = i[j];
      }
  }
};

}  // namespace provip
