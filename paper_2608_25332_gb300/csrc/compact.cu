// Survivor compaction (Sec. 4.1: pruned tokens are excluded from every later
// computation): out-of-place gather of the rows
//   [0, vis_start) ++ (vis_start + idx[b][0..keep)) ++ [vis_start + N_v, seq_len[b])
// of hidden states, K and V (any row size that is a multiple of 16 bytes),
// plus the position-id rows (int32, P of them; carried, not renumbered).
//
// Bulk-TMA pipeline: the work is the list of (output row, tensor, <= 8 KiB
// piece) items, in two phases - first the rows that do not depend on the kept
// indices (prefix and text rows), then the kept visual rows - and every CTA
// owns a contiguous range of each phase. Launched as a programmatic dependent
// of the kernel that writes idx, the first phase overlaps that kernel; the
// threads that read idx wait for it (griddepcontrol.wait). A call on its own
// (no programmatic dependency) splits the two phases as one list over four
// CTAs per SM, and each CTA loads its kept indices at once, alongside the
// sequence lengths: its few rows are then one short chain of round trips. One thread per CTA
// streams its range through a ring of shared-memory slots: a cp.async.bulk load
// (global -> shared, completion on the slot's mbarrier) and, once it lands, a
// cp.async.bulk store (shared -> global, bulk group). A slot is refilled as soon
// as the store that drained it has finished reading, so up to kSlots - 1 loads
// and a store are in flight per CTA (kSlots = 5, or 6 when the rows fill every
// CTA slot of the GPU and the caller allows it). The other warps copy the position ids and,
// with 16-byte vector loads and stores (a warp per row), the rows of tensors
// whose rows are at most 2 KiB (the K/V rows of a GQA layer with few key/value
// heads), which per-row bulk copies would move inefficiently.
// Every wait is bounded; a timeout sets the device error word and the CTA
// drains what it issued before returning.
#include "common.cuh"
#include "kernels.h"

namespace provip {
namespace {

#ifndef PROVIP_COMPACT_SLOTS
#define PROVIP_COMPACT_SLOTS 5
#endif
#ifndef PROVIP_COMPACT_DEEP_SLOTS
#define PROVIP_COMPACT_DEEP_SLOTS 6
#endif
#ifndef PROVIP_COMPACT_CTAS_PER_SM
#define PROVIP_COMPACT_CTAS_PER_SM 2
#endif
#ifndef PROVIP_COMPACT_SLOT_BYTES
#define PROVIP_COMPACT_SLOT_BYTES 8192
#endif
constexpr int kSlotBytes = PROVIP_COMPACT_SLOT_BYTES;
// ring of shared-memory slots per CTA: the short ring when the compaction does
// not fill every CTA slot of the GPU (small batches, many of them running side
// by side) or when the caller's previous kernel needs room beside it; the deep
// one otherwise (more bytes in flight per CTA; two such CTAs and a streaming
// head-score CTA of the next step still fit an SM's shared memory)
constexpr int kSlotsShort = PROVIP_COMPACT_SLOTS;
constexpr int kSlotsDeep = PROVIP_COMPACT_DEEP_SLOTS;
constexpr int kCtasPerSm = PROVIP_COMPACT_CTAS_PER_SM;
// a producer warp and three helper warps; a fourth helper warp when the helpers
// copy rows of small tensors (one round of copies for four rows per CTA)
constexpr int kCompactThreads = 128;
constexpr int kCompactThreadsSmall = 160;
#ifndef PROVIP_COMPACT_MIN_CTA_KIB
#define PROVIP_COMPACT_MIN_CTA_KIB 160
#endif
constexpr long long kMinCtaBytes = (long long)PROVIP_COMPACT_MIN_CTA_KIB * 1024;
// tensors with rows of at most this many bytes are copied by the helper warps
// with vector loads and stores (per-row bulk copies would cost more than they
// move)
#ifndef PROVIP_COMPACT_SMALL_ROW
#define PROVIP_COMPACT_SMALL_ROW 2048
#endif
constexpr int kSmallRow = PROVIP_COMPACT_SMALL_ROW;
// 16-byte pieces a helper lane holds in flight (the K and V rows of 1 KiB of a
// GQA layer with four key/value heads in one round trip)
constexpr int kSmallPieces = 4;
// bytes of rows per CTA below which a compaction that runs alone uses fewer
// CTAs than two per SM
constexpr long long kMinCtaBytesAlone = 16 * 1024;
// kept rows of a CTA whose indices the producer stages in shared memory, and
// how many of those loads it keeps in flight at once
constexpr int kIdxStage = 256;
constexpr int kStageBatch = 16;
// rows whose (sample, output row, source row) the helper threads work out
// together before copying them
constexpr int kMetaRows = 96;

// barrier of the helper threads (warps 1..; the producer warp does not take part)
__device__ __forceinline__ void helpers_sync() {
  asm volatile("bar.sync 1, %0;" ::"r"(blockDim.x - 32) : "memory");
}

__device__ __forceinline__ int src_row(const CompactArgs& a, int b, int r, bool& ok) {
  if (r < a.vis_start) return r;
  if (r < a.vis_start + a.keep) {
    const int v = a.idx[(size_t)b * a.keep + (r - a.vis_start)];
    if (v < 0 || v >= a.N_v) {
      ok = false;
      return 0;
    }
    return a.vis_start + v;
  }
  return r - a.keep + a.N_v;
}

struct Item {
  const char* src;
  char* dst;
  uint32_t bytes;
};

__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// Output row of item-space row q: phase 0 enumerates, per sample, the
// L_out - keep rows outside the kept block; phase 1 the keep kept rows.
__device__ __forceinline__ void phase_row(const CompactArgs& a, int phase, long long row, int& b,
                                          int& r) {
  if (phase == 0) {
    const int per = a.L_out - a.keep;
    b = (int)(row / per);
    const int q = (int)(row - (long long)b * per);
    r = q < a.vis_start ? q : q + a.keep;
  } else {
    b = (int)(row / a.keep);
    r = a.vis_start + (int)(row - (long long)b * a.keep);
  }
}

// alone: launched with no programmatic dependency (nothing to overlap, idx is
// ready at the start): the two phases' items are split over the CTAs as one
// list, the producer stages its kept indices before its first load, and the
// helpers resolve and copy all their rows in one pass. Otherwise each phase is
// split over every CTA, and idx is read only after the wait.
template <int kSlots>
__global__ void __launch_bounds__(kCompactThreadsSmall) compact_kernel(const CompactArgs a, int np0,
                                                                   int np1, int np2, int small,
                                                                   int alone) {
  extern __shared__ __align__(128) uint8_t slots[];
  __shared__ __align__(8) uint64_t bars[kSlots];
  __shared__ char* ring_dst[kSlots];
  __shared__ uint32_t ring_bytes[kSlots];
  __shared__ int idx_s[kIdxStage];  // the producer's staged kept indices
  __shared__ int4 meta_s[kMetaRows];  // the helpers' rows: (sample, output row, source row)
  // items per output row: the pieces of the bulk-copied tensors (at least one,
  // so that rows are spread over CTAs even when every tensor is small)
  const int NB = np0 + np1 + np2;
  const int NP = NB > 0 ? NB : 1;
  const long long items[2] = {(long long)a.B * (a.L_out - a.keep) * NP, (long long)a.B * a.keep * NP};
  long long beg[2], fin[2];
  if (alone) {
    // [phase 0 | phase 1] as one list, in equal shares (they differ by at most one)
    const long long T = items[0] + items[1];
    const long long lo = T * blockIdx.x / gridDim.x, hi = T * (blockIdx.x + 1) / gridDim.x;
    beg[0] = min(lo, items[0]);
    fin[0] = min(hi, items[0]);
    beg[1] = max(lo, items[0]) - items[0];
    fin[1] = max(hi, items[0]) - items[0];
  } else {
    for (int ph = 0; ph < 2; ++ph) {
      const long long per = (items[ph] + gridDim.x - 1) / gridDim.x;
      beg[ph] = min(items[ph], (long long)blockIdx.x * per);
      fin[ph] = min(items[ph], beg[ph] + per);
    }
  }

  // a kernel launched as this grid's programmatic dependent may start now (it
  // waits for this grid's completion before touching anything written here)
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  if (blockIdx.x == 0 && a.seq_len_out != nullptr)
    for (int b = threadIdx.x; b < a.B; b += blockDim.x)
      a.seq_len_out[b] = a.seq_len[b] - a.N_v + a.keep;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kSlots; ++s) mbar_init(&bars[s], 1);
    fence_mbar_init();
  }
  __syncthreads();

  if (threadIdx.x == 0 && NB > 0) {
    const uint64_t pol = policy_evict_first();
    // The items of a phase are walked in order with running counters (piece
    // q of row w of sample b), so no item needs a division. The kept visual
    // indices of the CTA's phase-1 rows are loaded once, kStageBatch at a time
    // with every load of a batch in flight, right after the wait for the kernel
    // that writes them; longer ranges read the rest from global memory.
    int phase = 0;
    long long next = beg[0];
    int b = 0, w = 0, q = 0, per = 1;
    int ord = 0;  // rows of the phase started so far (the staged index of a phase-1 row)
    int sl = 0;
    // the kept indices of this CTA's phase-1 rows into idx_s
    auto stage_idx = [&]() {
      if (beg[1] >= fin[1]) return;
      const long long r1 = (fin[1] + NP - 1) / NP;
      const int n = (int)min((long long)kIdxStage, r1 - beg[1] / NP);
      const int* src = a.idx + beg[1] / NP;
      for (int j0 = 0; j0 < n; j0 += kStageBatch) {
        int v[kStageBatch];
#pragma unroll
        for (int j = 0; j < kStageBatch; ++j) v[j] = j0 + j < n ? src[j0 + j] : 0;
#pragma unroll
        for (int j = 0; j < kStageBatch; ++j)
          if (j0 + j < n) idx_s[j0 + j] = v[j];
      }
    };
    auto start_phase = [&](int ph) {
      if (beg[ph] >= fin[ph]) return;  // nothing of this phase here (per may be 0)
      per = ph == 0 ? a.L_out - a.keep : a.keep;
      const long long row = beg[ph] / NP;
      q = (int)(beg[ph] - row * NP);
      ord = 0;
      b = (int)(row / per);
      w = (int)(row - (long long)b * per);
      sl = a.seq_len[b];
      if (ph == 1 && !alone) {
        pdl_wait();  // idx is written by the previous kernel
        stage_idx();
      }
    };
    if (alone) stage_idx();  // in flight with the lengths start_phase loads
    start_phase(0);
    // next valid item; false when both phases are exhausted
    auto fetch = [&](Item& it) -> bool {
      for (;;) {
        if (next >= fin[phase]) {
          if (phase == 1) return false;
          phase = 1;
          next = beg[1];
          start_phase(1);
          continue;
        }
        ++next;
        const int cq = q, cw = w, cb = b, csl = sl, cord = ord;
        if (++q == NP) {  // advance the counters to item i + 1
          q = 0;
          ++ord;
          if (++w == per) {
            w = 0;
            ++b;
            if (next < fin[phase]) sl = a.seq_len[b];
          }
        }
        if (csl > a.L_max || csl < a.vis_start + a.N_v) {
          set_error(a.err, kErrBadDeviceArg);
          continue;
        }
        const int r = phase == 0 ? (cw < a.vis_start ? cw : cw + a.keep) : a.vis_start + cw;
        if (r >= csl - a.N_v + a.keep) continue;
        int sr = r;
        if (phase == 1) {
          const int v = cord < kIdxStage ? idx_s[cord] : a.idx[(size_t)cb * a.keep + cw];
          if (v < 0 || v >= a.N_v) {
            set_error(a.err, kErrBadDeviceArg);
            continue;
          }
          sr = a.vis_start + v;
        } else if (r >= a.vis_start) {
          sr = r - a.keep + a.N_v;
        }
        int t = 0, pq = cq;
        if (pq >= np0) {
          pq -= np0;
          t = 1;
          if (pq >= np1) {
            pq -= np1;
            t = 2;
          }
        }
        const long long rb = a.row_bytes[t];
        const long long off = (long long)pq * kSlotBytes;
        it.bytes = (uint32_t)min((long long)kSlotBytes, rb - off);
        it.src = a.src[t] + ((long long)cb * a.L_max + sr) * rb + off;
        it.dst = a.dst[t] + ((long long)cb * a.L_out + r) * rb + off;
        return true;
      }
    };
    auto issue = [&](int slot, const Item& it) {
      ring_dst[slot] = it.dst;
      ring_bytes[slot] = it.bytes;
      mbar_arrive_expect_tx(&bars[slot], it.bytes);
      bulk_g2s(slots + (size_t)slot * kSlotBytes, it.src, it.bytes, &bars[slot], pol);
    };
    int loaded = 0;
    Item it;
    while (loaded < kSlots && fetch(it)) issue(loaded++, it);
    bool failed = false;
    int i = 0;
    for (; i < loaded; ++i) {
      const int s = i % kSlots;
      if (!mbar_wait(&bars[s], (uint32_t)(i / kSlots) & 1u, a.err)) {
        failed = true;
        break;
      }
      bulk_s2g(ring_dst[s], slots + (size_t)s * kSlotBytes, ring_bytes[s]);
      bulk_commit();
      if (i >= 1) {
        bulk_wait_read<1>();  // the store of item i - 1 has read its slot
        if (fetch(it)) {
          issue(loaded % kSlots, it);
          ++loaded;
        }
      }
    }
    if (failed) {
      // drain the loads still in flight (bounded) before the CTA exits
      for (int j = i; j < loaded; ++j) mbar_wait(&bars[j % kSlots], (uint32_t)(j / kSlots) & 1u, a.err);
    }
    bulk_wait<0>();
  } else if (threadIdx.x >= 32 && (a.pos != nullptr || small != 0)) {
    // rows whose first item lies in this CTA's ranges: their position ids, and
    // the rows of the small tensors (16-byte vector copies, a warp per row)
    // a thread per row for the position ids alone, a warp per row with small tensors
    // Rows are taken kMetaRows at a time: first every helper thread works out
    // the (sample, output row, source row) of its own rows - their dependent
    // loads of lengths and kept indices all in flight at once - into shared
    // memory, then (after a barrier of the helper threads) the copies run.
    const int ht = (int)threadIdx.x - 32, n_ht = (int)blockDim.x - 32;
    const int lane = small ? (int)(threadIdx.x & 31) : 0;
    const int worker = small ? (int)(threadIdx.x >> 5) - 1 : ht;
    const int n_workers = small ? (int)blockDim.x / 32 - 1 : n_ht;
    // (sample, output row, source row) of row `row` of phase ph into meta_s[k]
    auto meta_row = [&](int ph, long long row, int k) {
      int b, r;
      phase_row(a, ph, row, b, r);
      const int sl = a.seq_len[b];
      bool ok = !(sl > a.L_max || sl < a.vis_start + a.N_v || r >= sl - a.N_v + a.keep);
      const int sr = ok ? src_row(a, b, r, ok) : 0;
      meta_s[k] = ok ? make_int4(b, r, sr, 0) : make_int4(-1, 0, 0, 0);
    };
    // the copies of the rows in meta_s[0..nrow)
    auto copy_rows = [&](int nrow) {
      for (int k = worker; k < nrow; k += n_workers) {
        const int4 mt = meta_s[k];
        if (mt.x < 0) continue;
        const int b = mt.x, r = mt.y, sr = mt.z;
        if (a.pos != nullptr)
          for (int p = lane; p < a.P; p += 32)
            a.pos_out[((size_t)p * a.B + b) * a.L_out + r] = a.pos[((size_t)p * a.B + b) * a.L_max + sr];
        // the row's pieces of every small tensor, as one list of 16-byte
        // pieces: all of a lane's loads are issued before its stores (one
        // memory round trip per row, not one per tensor)
        const uint4 *s0 = nullptr, *s1 = nullptr, *s2 = nullptr;
        uint4 *d0 = nullptr, *d1 = nullptr, *d2 = nullptr;
        int n0 = 0, n1 = 0, n2 = 0;
        if (small & 1) {
          const long long rb = a.row_bytes[0];
          s0 = reinterpret_cast<const uint4*>(a.src[0] + ((long long)b * a.L_max + sr) * rb);
          d0 = reinterpret_cast<uint4*>(a.dst[0] + ((long long)b * a.L_out + r) * rb);
          n0 = (int)(rb / 16);
        }
        if (small & 2) {
          const long long rb = a.row_bytes[1];
          s1 = reinterpret_cast<const uint4*>(a.src[1] + ((long long)b * a.L_max + sr) * rb);
          d1 = reinterpret_cast<uint4*>(a.dst[1] + ((long long)b * a.L_out + r) * rb);
          n1 = (int)(rb / 16);
        }
        if (small & 4) {
          const long long rb = a.row_bytes[2];
          s2 = reinterpret_cast<const uint4*>(a.src[2] + ((long long)b * a.L_max + sr) * rb);
          d2 = reinterpret_cast<uint4*>(a.dst[2] + ((long long)b * a.L_out + r) * rb);
          n2 = (int)(rb / 16);
        }
        const int tot = n0 + n1 + n2;
        for (int q0 = 0; q0 < tot; q0 += 32 * kSmallPieces) {
          uint4 v[kSmallPieces];
#pragma unroll
          for (int j = 0; j < kSmallPieces; ++j) {
            const int q = q0 + lane + 32 * j;
            if (q < tot)
              v[j] = __ldcs(q < n0 ? s0 + q : (q < n0 + n1 ? s1 + (q - n0) : s2 + (q - n0 - n1)));
          }
#pragma unroll
          for (int j = 0; j < kSmallPieces; ++j) {
            const int q = q0 + lane + 32 * j;
            if (q < tot) __stcs(q < n0 ? d0 + q : (q < n0 + n1 ? d1 + (q - n0) : d2 + (q - n0 - n1)), v[j]);
          }
        }
      }
    };
    const long long r0[2] = {(beg[0] + NP - 1) / NP, (beg[1] + NP - 1) / NP};
    const long long r1[2] = {(fin[0] + NP - 1) / NP, (fin[1] + NP - 1) / NP};
    const int n0 = (int)(r1[0] - r0[0]), n1 = (int)(r1[1] - r0[1]);
    if (alone && n0 + n1 <= kMetaRows) {
      // every row of both phases resolved, then copied, in one pass
      for (int k = ht; k < n0 + n1; k += n_ht) meta_row(k < n0 ? 0 : 1, k < n0 ? r0[0] + k : r0[1] + (k - n0), k);
      helpers_sync();
      copy_rows(n0 + n1);
    } else {
      for (int ph = 0; ph < 2; ++ph) {
        if (ph == 1) pdl_wait();
        for (long long c0 = r0[ph]; c0 < r1[ph]; c0 += kMetaRows) {
          const int nrow = (int)min((long long)kMetaRows, r1[ph] - c0);
          for (int k = ht; k < nrow; k += n_ht) meta_row(ph, c0 + k, k);
          helpers_sync();
          copy_rows(nrow);
          helpers_sync();  // meta_s is rewritten by the next chunk
        }
      }
    }
  }
}

// The compaction for rows in mapped host memory (or any mix of host and device
// memory): every row is copied by one warp with 16-byte loads and stores, all
// of a lane's loads of a round (kVecPieces pieces, 4 KiB per warp) issued
// before its stores, with no bulk (TMA) copies. Rows are dealt to the warps of
// the grid in turn, phase 0 (the rows that do not depend on idx) first; a
// warp's lanes resolve a row's (sample, output row, source row) together (the
// same loads, one transaction).
constexpr int kVecThreads = 128;
constexpr int kVecPieces = 8;
__global__ void __launch_bounds__(kVecThreads) compact_vec_kernel(const CompactArgs a) {
  const int lane = threadIdx.x & 31;
  const long long warp = (long long)blockIdx.x * (kVecThreads / 32) + (threadIdx.x >> 5);
  const long long n_warps = (long long)gridDim.x * (kVecThreads / 32);
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  if (blockIdx.x == 0 && a.seq_len_out != nullptr)
    for (int b = threadIdx.x; b < a.B; b += blockDim.x) a.seq_len_out[b] = a.seq_len[b] - a.N_v + a.keep;
  const int n16[3] = {a.n_tensors > 0 ? (int)(a.row_bytes[0] / 16) : 0,
                      a.n_tensors > 1 ? (int)(a.row_bytes[1] / 16) : 0,
                      a.n_tensors > 2 ? (int)(a.row_bytes[2] / 16) : 0};
  const int tot = n16[0] + n16[1] + n16[2];
  for (int ph = 0; ph < 2; ++ph) {
    if (ph == 1) pdl_wait();  // idx is written by the previous kernel
    const long long nrows = ph == 0 ? (long long)a.B * (a.L_out - a.keep) : (long long)a.B * a.keep;
    for (long long row = warp; row < nrows; row += n_warps) {
      int b, r;
      phase_row(a, ph, row, b, r);
      const int sl = a.seq_len[b];
      if (sl > a.L_max || sl < a.vis_start + a.N_v) {
        if (lane == 0) set_error(a.err, kErrBadDeviceArg);
        continue;
      }
      if (r >= sl - a.N_v + a.keep) continue;
      int sr = r;
      if (ph == 1) {
        const int v = a.idx[row];  // row = b * keep + position
        if (v < 0 || v >= a.N_v) {
          if (lane == 0) set_error(a.err, kErrBadDeviceArg);
          continue;
        }
        sr = a.vis_start + v;
      } else if (r >= a.vis_start) {
        sr = r - a.keep + a.N_v;
      }
      if (a.pos != nullptr)
        for (int p = lane; p < a.P; p += 32)
          a.pos_out[((size_t)p * a.B + b) * a.L_out + r] = a.pos[((size_t)p * a.B + b) * a.L_max + sr];
      const uint4* s0 = n16[0] ? reinterpret_cast<const uint4*>(a.src[0] + ((long long)b * a.L_max + sr) * a.row_bytes[0]) : nullptr;
      const uint4* s1 = n16[1] ? reinterpret_cast<const uint4*>(a.src[1] + ((long long)b * a.L_max + sr) * a.row_bytes[1]) : nullptr;
      const uint4* s2 = n16[2] ? reinterpret_cast<const uint4*>(a.src[2] + ((long long)b * a.L_max + sr) * a.row_bytes[2]) : nullptr;
      uint4* d0 = n16[0] ? reinterpret_cast<uint4*>(a.dst[0] + ((long long)b * a.L_out + r) * a.row_bytes[0]) : nullptr;
      uint4* d1 = n16[1] ? reinterpret_cast<uint4*>(a.dst[1] + ((long long)b * a.L_out + r) * a.row_bytes[1]) : nullptr;
      uint4* d2 = n16[2] ? reinterpret_cast<uint4*>(a.dst[2] + ((long long)b * a.L_out + r) * a.row_bytes[2]) : nullptr;
      const int n0 = n16[0], n1 = n16[1];
      for (int q0 = 0; q0 < tot; q0 += 32 * kVecPieces) {
        uint4 v[kVecPieces];
#pragma unroll
        for (int j = 0; j < kVecPieces; ++j) {
          const int q = q0 + lane + 32 * j;
          if (q < tot) v[j] = __ldcs(q < n0 ? s0 + q : (q < n0 + n1 ? s1 + (q - n0) : s2 + (q - n0 - n1)));
        }
#pragma unroll
        for (int j = 0; j < kVecPieces; ++j) {
          const int q = q0 + lane + 32 * j;
          if (q < tot) __stcs(q < n0 ? d0 + q : (q < n0 + n1 ? d1 + (q - n0) : d2 + (q - n0 - n1)), v[j]);
        }
      }
    }
  }
}

}  // namespace

cudaError_t compact_launch(const CompactArgs& a, int num_sms, cudaStream_t s, bool pdl, bool allow_deep,
                           bool concurrent, bool host_rows) {
  if (host_rows) {
    // rows in mapped host memory: plain vector copies over the whole GPU
    const long long rows = (long long)a.B * a.L_out;
    long long grid = (long long)kCtasPerSm * num_sms;
    const long long need = (rows + kVecThreads / 32 - 1) / (kVecThreads / 32);
    if (grid > need) grid = need > 0 ? need : 1;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3(kVecThreads);
    cfg.stream = s;
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, compact_vec_kernel, a);
  }
  static std::atomic<bool> configured[64];  // per device, zero-initialised
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64 && !configured[dev]) {
    cudaError_t e = cudaFuncSetAttribute(compact_kernel<kSlotsShort>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)((size_t)kSlotsShort * kSlotBytes));
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(compact_kernel<kSlotsDeep>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               (int)((size_t)kSlotsDeep * kSlotBytes));
    if (e != cudaSuccess) return e;
    configured[dev] = true;
  }
  int np[3] = {0, 0, 0};
  int small = 0;
  for (int t = 0; t < a.n_tensors; ++t) {
    if (a.row_bytes[t] <= kSmallRow)
      small |= 1 << t;
    else
      np[t] = (int)((a.row_bytes[t] + kSlotBytes - 1) / kSlotBytes);
  }
  const int nb = np[0] + np[1] + np[2];
  const long long total = (long long)a.B * a.L_out * (nb > 0 ? nb : 1);
  // Two CTAs per SM when the call follows a kernel it overlaps (room is left
  // for the next step's head-score CTAs), four when it runs on its own.
  long long grid = (long long)(pdl ? kCtasPerSm : 2 * kCtasPerSm) * num_sms;
  // Alone, the compaction spreads over every SM (a small problem is bound by
  // the latency of each CTA's few copies, so more CTAs finish it sooner). With
  // concurrent calls on other streams, a small problem takes at least
  // kMinCtaBytes of rows per CTA, so that every CTA's pipeline fills and the
  // kernels running beside it keep the SMs it does not need.
  const long long row_sum = a.row_bytes[0] + a.row_bytes[1] + a.row_bytes[2];
  const long long bytes = (long long)a.B * a.L_out * row_sum;
  const long long by_bytes = (bytes + kMinCtaBytes - 1) / kMinCtaBytes;
  const bool deep = allow_deep && by_bytes >= grid;  // the rows fill every CTA slot
  const long long cap = concurrent ? by_bytes : (bytes + kMinCtaBytesAlone - 1) / kMinCtaBytesAlone;
  if (grid > cap) grid = cap;
  if (grid > total) grid = total > 0 ? total : 1;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(small ? kCompactThreadsSmall : kCompactThreads);
  cfg.dynamicSmemBytes = (size_t)(deep ? kSlotsDeep : kSlotsShort) * kSlotBytes;
  cfg.stream = s;
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  const int alone = pdl ? 0 : 1;
  return deep ? cudaLaunchKernelEx(&cfg, compact_kernel<kSlotsDeep>, a, np[0], np[1], np[2], small, alone)
              : cudaLaunchKernelEx(&cfg, compact_kernel<kSlotsShort>, a, np[0], np[1], np[2], small, alone);
}

}  // namespace provip
