// Warp-specialised tcgen05 "NT" Gram core for the pre-LLM pass (Sec. 4.3):
//   D[M x N] = A[M x K] * B[N x K]^T, bf16 operands, fp32 accumulation in TMEM,
// with A and B fetched by 2-D TMA (128-byte swizzle) as blocks of consecutive
// rows (boxes of 128 rows).
//
// One CTA owns one 128-row M tile and sweeps a range of BN-column N tiles
// (BN = 128 or 256):
//   warp 0 (one lane)  TMA producer: K slices of 64 elements, kStages-deep ring
//                      of shared-memory stages (A 16 KiB + B BN x 128 B each);
//   warp 1 (one lane)  MMA issuer: 4 x tcgen05.mma (M=128, N=BN, K=16) per
//                      stage, tcgen05.commit frees the stage, and a commit per
//                      N tile hands the accumulator to the epilogue;
//   warps 2-5          epilogue: thread = TMEM lane = row of the M tile; two
//                      BN-column accumulators alternate so that the epilogue
//                      of tile n overlaps the main loop of tile n + 1.
// Every mbarrier wait is bounded (mbar_wait); a timeout marks the CTA failed,
// and the roles drain and exit.
#pragma once

#include "common.cuh"

namespace provip {
namespace tcg {

constexpr int kBM = 128;
constexpr int kBK = 64;                      // bf16 elements per stage row (128 B)
constexpr int kStages = 4;
constexpr int kABytes = kBM * kBK * 2;       // 16 KiB
constexpr int kThreads = 192;                // 6 warps

// per N-tile width (128 or 256)
template <int BN>
struct Cfg {
  static constexpr int kBBytes = BN * kBK * 2;
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr uint32_t kIdesc = idesc_bf16_f32(kBM, BN);
  static constexpr size_t kStagesBytes = (size_t)kStages * kStageBytes;
  static constexpr uint32_t kTmemCols = 2 * BN;  // two accumulators
};

struct Pipe {
  uint64_t full[kStages];
  uint64_t empty[kStages];
  uint64_t acc_full[2];
  uint64_t acc_empty[2];
  uint32_t tmem;
  volatile int fail;
};

// Row source of an operand: rows base + r, r < count (rows >= count are loaded
// but their results are masked by the caller).
struct RowSrc {
  int base;   // first row
  int count;  // valid rows
};

// Loads rows [r0, r0 + nrows) of an operand for K slice x into a 128-B-row tile,
// in boxes of 128 rows (the tensor map's box height).
__device__ __forceinline__ void load_rows(uint8_t* dst, const CUtensorMap* map, const RowSrc& src,
                                          int r0, int nrows, int x, uint64_t* bar) {
  for (int r = 0; r < nrows; r += 128) tma_load_2d(dst + r * 128, map, x, src.base + r0 + r, bar);
}

// Producer: for each N tile t in [0, n_tiles), all K slices.
template <int BN>
// k0: first K slice (a split-K part starts past the others' slices); b_is_a:
// the B operand is the A tile itself (a Gram of one row block), loaded once
__device__ __forceinline__ void producer(Pipe& p, uint8_t* stages, const CUtensorMap* mapA,
                                         const CUtensorMap* mapB, const RowSrc& a, const RowSrc& b,
                                         int n_tiles, int n_k, unsigned* err, int k0 = 0,
                                         bool b_is_a = false) {
  int it = 0;
  for (int t = 0; t < n_tiles && !p.fail; ++t) {
    for (int kb = 0; kb < n_k; ++kb, ++it) {
      const int s = it % kStages;
      const uint32_t ph = (uint32_t)(it / kStages) & 1u;
      if (!mbar_wait(&p.empty[s], ph ^ 1u, err)) {
        p.fail = 1;
        return;
      }
      uint8_t* sa = stages + (size_t)s * Cfg<BN>::kStageBytes;
      uint8_t* sb = sa + kABytes;
      mbar_arrive_expect_tx(&p.full[s], b_is_a ? (uint32_t)kABytes : (uint32_t)Cfg<BN>::kStageBytes);
      load_rows(sa, mapA, a, 0, kBM, (k0 + kb) * kBK, &p.full[s]);
      if (!b_is_a) load_rows(sb, mapB, b, t * BN, BN, (k0 + kb) * kBK, &p.full[s]);
    }
  }
}

// MMA issuer.
template <int BN>
__device__ __forceinline__ void mma_issuer(Pipe& p, uint8_t* stages, int n_tiles, int n_k,
                                           unsigned* err, bool b_is_a = false) {
  int it = 0;
  for (int t = 0; t < n_tiles; ++t) {
    const int buf = t & 1;
    const uint32_t acc_addr = p.tmem + (uint32_t)(buf * BN);
    if (!mbar_wait(&p.acc_empty[buf], ((uint32_t)(t >> 1) & 1u) ^ 1u, err)) {
      p.fail = 1;
    }
    for (int kb = 0; kb < n_k; ++kb, ++it) {
      const int s = it % kStages;
      const uint32_t ph = (uint32_t)(it / kStages) & 1u;
      if (p.fail || !mbar_wait(&p.full[s], ph, err)) {
        p.fail = 1;
        break;
      }
      tc_fence_after();
      const uint32_t sa = smem_u32(stages + (size_t)s * Cfg<BN>::kStageBytes);
      const uint32_t sb = b_is_a ? sa : sa + kABytes;
#pragma unroll
      for (int k = 0; k < kBK / 16; ++k)
        tc_mma_bf16(acc_addr, smem_desc_sw128(sa + k * 32), smem_desc_sw128(sb + k * 32),
                    Cfg<BN>::kIdesc, (kb > 0 || k > 0) ? 1u : 0u);
      tc_commit(&p.empty[s]);
    }
    tc_commit(&p.acc_full[buf]);  // arrives when every MMA above has completed
    if (p.fail) {
      // let the epilogue drain: the commit above still arrives
      for (int t2 = t + 1; t2 < n_tiles; ++t2) tc_commit(&p.acc_full[t2 & 1]);
      return;
    }
  }
}

__device__ __forceinline__ void pipe_init(Pipe& p) {
  for (int s = 0; s < kStages; ++s) {
    mbar_init(&p.full[s], 1);
    mbar_init(&p.empty[s], 1);
  }
  for (int b = 0; b < 2; ++b) {
    mbar_init(&p.acc_full[b], 1);
    mbar_init(&p.acc_empty[b], 4);  // one arrival per epilogue warp
  }
  p.fail = 0;
  fence_mbar_init();
}

}  // namespace tcg
}  // namespace provip
