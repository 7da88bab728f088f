// C-ABI layer of the ProViP GB300 library: host-side argument validation,
// workspace carving and kernel launches. Declarations and the contract of each
// entry point are in include/provip.h.
#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <atomic>
#include <initializer_list>
#include <mutex>

#include <nvtx3/nvToolsExt.h>

#include "../../include/provip.h"
#include "common.cuh"
#include "kernels.h"

using namespace provip;

// device status word (one per device that loads the library)
__device__ unsigned int g_provip_status;

namespace {

thread_local char g_last_error[512] = {0};

// An NVTX range named after the entry point for the duration of the host call,
// so that a profiler timeline attributes the kernels each call enqueues to the
// call (header-only NVTX: a no-op unless a profiling tool is attached).
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

int fail(int code, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_last_error, sizeof(g_last_error), fmt, ap);
  va_end(ap);
  return code;
}

int cuda_fail(cudaError_t e, const char* where) {
  return fail(PROVIP_ERR_CUDA, "%s: %s", where, cudaGetErrorString(e));
}

struct DevInfo {
  std::atomic<bool> init{false};  // set (release) once sms and status are written
  int sms = 0;
  unsigned* status = nullptr;
};
DevInfo g_dev[64];
std::mutex g_dev_mu;  // serialises the first lookup of each device

// A second stream per host thread and device for the part of a call that can
// run beside the rest (forked from the caller's stream and joined back with
// the two events), so that calls from different threads never share one. They
// live until the process ends: destroying them at thread exit could run after
// the CUDA runtime has shut down.
struct SideStream {
  cudaStream_t s = nullptr;
  cudaEvent_t fork = nullptr, join = nullptr;
};
thread_local SideStream tl_side[64];
int side_stream(SideStream** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if (dev < 0 || dev >= 64) return fail(PROVIP_ERR_UNSUPPORTED, "device ordinal %d >= 64", dev);
  SideStream& x = tl_side[dev];
  if (x.s == nullptr) {
    e = cudaStreamCreateWithFlags(&x.s, cudaStreamNonBlocking);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&x.fork, cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&x.join, cudaEventDisableTiming);
    if (e != cudaSuccess) {
      x = SideStream();
      return cuda_fail(e, "side stream");
    }
  }
  *out = &x;
  return PROVIP_OK;
}

// per-device facts, looked up once with that device current (safe from several
// host threads: the first caller fills them under the lock, later ones read them
// after an acquire of `init`)
int dev_info(DevInfo** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if (dev < 0 || dev >= 64) return fail(PROVIP_ERR_UNSUPPORTED, "device ordinal %d >= 64", dev);
  DevInfo& d = g_dev[dev];
  if (!d.init.load(std::memory_order_acquire)) {
    std::lock_guard<std::mutex> lock(g_dev_mu);
    if (!d.init.load(std::memory_order_relaxed)) {
      int sms = 0;
      e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
      if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceGetAttribute");
      void* p = nullptr;
      e = cudaGetSymbolAddress(&p, g_provip_status);
      if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(status)");
      d.sms = sms;
      d.status = static_cast<unsigned*>(p);
      d.init.store(true, std::memory_order_release);
    }
  }
  *out = &d;
  return PROVIP_OK;
}

constexpr size_t kAlign = 256;
inline size_t align_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

// bump allocator over the caller's workspace (also used to size it)
struct Carve {
  char* base;
  size_t off = 0;
  explicit Carve(void* b) : base(static_cast<char*>(b)) {}
  template <typename T>
  T* take(size_t count) {
    T* p = base ? reinterpret_cast<T*>(base + off) : nullptr;
    off += align_up(count * sizeof(T));
    return p;
  }
};

inline int esize(int dtype) { return dtype == PROVIP_F32 ? 4 : 2; }
inline bool dtype_ok(int dtype) { return dtype == PROVIP_F32 || dtype == PROVIP_BF16; }
inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// ---------------------------------------------------------------------------
// head scores: shapes and workspace
// ---------------------------------------------------------------------------
int resolve_algo(int algo, int dtype) {
  if (algo == PROVIP_ALGO_AUTO) return dtype == PROVIP_BF16 ? PROVIP_ALGO_TCGEN05 : PROVIP_ALGO_SIMT;
  return algo;
}
bool is_tc(int algo) {
  return algo == PROVIP_ALGO_TCGEN05 || algo == PROVIP_ALGO_TCGEN05_TWOPASS ||
         algo == PROVIP_ALGO_TCGEN05_STREAM || algo == PROVIP_ALGO_TCGEN05_CLUSTER;
}
// PROVIP_ALGO_TCGEN05: the streaming form once the (sample, head, row block)
// units fill the SMs, else the cluster form (spreads one unit over its key chunks)
int tc_form(int algo, int B, int H_sel, int n_rb, int sms) {
  if (algo != PROVIP_ALGO_TCGEN05) return algo;
  return (long long)B * H_sel * n_rb >= sms ? PROVIP_ALGO_TCGEN05_STREAM : PROVIP_ALGO_TCGEN05_CLUSTER;
}
int key_chunk(int algo) { return is_tc(algo) ? 128 : 64; }
int vis_chunk(int algo) { return is_tc(algo) ? 128 : 64; }

struct HSShape {
  int n_rb, kc, n_kc, vc, n_vc;
};
HSShape hs_shape(int L_max, int N_t_max, int N_v, int algo) {
  HSShape s;
  s.n_rb = (N_t_max + kRowBlock - 1) / kRowBlock;
  s.kc = key_chunk(algo);
  s.n_kc = (L_max + s.kc - 1) / s.kc;
  s.vc = vis_chunk(algo);
  s.n_vc = (N_v + s.vc - 1) / s.vc;
  return s;
}
size_t hs_ws(Carve& c, int B, int H_sel, const HSShape& s, int N_v, float2** stats,
             float** partial) {
  *stats = c.take<float2>((size_t)B * s.n_rb * H_sel * s.n_kc * kRowBlock);
  *partial = c.take<float>((size_t)B * s.n_rb * H_sel * N_v);
  return c.off;
}

// head confidence: chunk capacity per row (every chunk layout the resolved
// path may take) and the workspace it needs
int conf_stride(const HSShape& sh, int algo) {
  return (algo == PROVIP_ALGO_TCGEN05 || algo == PROVIP_ALGO_TCGEN05_CLUSTER)
             ? (sh.n_vc > kFusedMaxChunks ? sh.n_vc : kFusedMaxChunks)
             : sh.n_vc;  // TWOPASS, SIMT: n_vc; STREAM uses 1
}
struct ConfWs {
  float2* part = nullptr;
  int* sel = nullptr;
};
size_t conf_ws(Carve& c, int B, int H_sel, int N_t_max, const HSShape& sh, int algo, int n_vis,
               ConfWs& w) {
  w.part = c.take<float2>((size_t)B * H_sel * N_t_max * conf_stride(sh, algo));
  w.sel = c.take<int>((size_t)B * (n_vis > 0 ? n_vis : 1));
  return c.off;
}

int hs_validate(const void* Q, const void* K, int B, int L_max, int H_q, int H_kv, int d_h,
                const int* head_list, int H_sel, const int* text_start, const int* text_len,
                int N_t_max, int vis_start, int N_v, const int* seq_len, int dtype, int algo) {
  if (!Q || !K || !text_start || !text_len || !seq_len)
    return fail(PROVIP_ERR_INVALID_ARG, "head_scores: null pointer argument");
  if (B < 1 || L_max < 1 || H_q < 1 || H_kv < 1 || N_t_max < 1 || N_v < 1 || vis_start < 0)
    return fail(PROVIP_ERR_INVALID_ARG, "head_scores: non-positive size");
  if (H_q % H_kv != 0) return fail(PROVIP_ERR_INVALID_ARG, "head_scores: H_q %% H_kv != 0");
  if (vis_start + N_v > L_max) return fail(PROVIP_ERR_INVALID_ARG, "head_scores: visual range exceeds L_max");
  if (N_t_max > L_max) return fail(PROVIP_ERR_INVALID_ARG, "head_scores: N_t_max > L_max");
  if (!dtype_ok(dtype)) return fail(PROVIP_ERR_UNSUPPORTED, "head_scores: dtype %d", dtype);
  if (d_h != kHeadDim) return fail(PROVIP_ERR_UNSUPPORTED, "head_scores: d_h must be 128");
  if (H_sel < 1 || H_sel > kMaxHeads) return fail(PROVIP_ERR_INVALID_ARG, "head_scores: H_sel %d", H_sel);
  if (!head_list && H_sel != H_q)
    return fail(PROVIP_ERR_INVALID_ARG, "head_scores: a null head_list (all heads) needs H_sel == H_q");
  for (int i = 0; head_list && i < H_sel; ++i) {
    if (head_list[i] < 0 || head_list[i] >= H_q)
      return fail(PROVIP_ERR_INVALID_ARG, "head_scores: head_list[%d] = %d out of range", i, head_list[i]);
    for (int j = 0; j < i; ++j)
      if (head_list[j] == head_list[i])
        return fail(PROVIP_ERR_INVALID_ARG, "head_scores: duplicate head %d", head_list[i]);
  }
  if (algo != PROVIP_ALGO_SIMT && !is_tc(algo))
    return fail(PROVIP_ERR_INVALID_ARG, "head_scores: algo %d", algo);
  if (is_tc(algo) && dtype != PROVIP_BF16)
    return fail(PROVIP_ERR_UNSUPPORTED, "head_scores: tcgen05 path needs bf16");
  if (!aligned16(Q) || !aligned16(K)) return fail(PROVIP_ERR_UNSUPPORTED, "head_scores: Q/K not 16-byte aligned");
  if ((size_t)B * L_max * H_q * d_h >= (1ull << 40))
    return fail(PROVIP_ERR_UNSUPPORTED, "head_scores: tensor too large");
  return PROVIP_OK;
}

HSArgs hs_args(const void* Q, const void* K, int B, int L_max, int H_q, int H_kv, int d_h,
               const int* head_list, int H_sel, const int* text_start, const int* text_len,
               const uint8_t* row_mask, int N_t_max, int vis_start, int N_v, const int* seq_len,
               const HSShape& sh, float2* stats, float* partial, unsigned* err) {
  HSArgs a;
  memset(&a, 0, sizeof(a));
  a.Q = Q;
  a.K = K;
  a.B = B;
  a.L_max = L_max;
  a.H_q = H_q;
  a.H_kv = H_kv;
  a.d_h = d_h;
  a.H_sel = H_sel;
  for (int i = 0; i < H_sel; ++i) a.heads[i] = head_list ? head_list[i] : i;
  a.text_start = text_start;
  a.text_len = text_len;
  a.row_mask = row_mask;
  a.N_t_max = N_t_max;
  a.vis_start = vis_start;
  a.N_v = N_v;
  a.seq_len = seq_len;
  a.n_rb = sh.n_rb;
  a.kc = sh.kc;
  a.n_kc = sh.n_kc;
  a.vc = sh.vc;
  a.n_vc = sh.n_vc;
  a.scale_log2 = (float)(1.4426950408889634 / sqrt((double)d_h));
  a.stats = stats;
  a.partial = partial;
  a.err = err;
  return a;
}

// both passes of the head scores (partials in the workspace); overlap: the
// one-pass kernel may start before the previous kernel on the stream finishes;
// geom: the chunks of the confidence statistics, when a.conf_part is set
int hs_run(const HSArgs& a, int dtype, int algo, cudaStream_t s, bool overlap = false,
           ConfGeom* geom = nullptr) {
  cudaError_t e;
  if (is_tc(algo)) {
    DevInfo* d;
    int rc = dev_info(&d);
    if (rc) return rc;
    algo = tc_form(algo, a.B, a.H_sel, a.n_rb, d->sms);
    CUtensorMap tq, tk;
    const uint64_t qstride = (uint64_t)a.H_q * a.d_h * 2, kstride = (uint64_t)a.H_kv * a.d_h * 2;
    if (make_tmap_bf16_2d(&tq, a.Q, (uint64_t)a.B * a.L_max, (uint64_t)a.H_q * a.d_h, qstride, 128) ||
        make_tmap_bf16_2d(&tk, a.K, (uint64_t)a.B * a.L_max, (uint64_t)a.H_kv * a.d_h, kstride, 128))
      return fail(PROVIP_ERR_CUDA, "head_scores: cuTensorMapEncodeTiled failed");
    bool launched = false;
    e = cudaSuccess;
    if (algo == PROVIP_ALGO_TCGEN05_STREAM) {
      e = hs_launch_stream(a, &tq, &tk, s, overlap, geom);
      launched = true;
    } else if (algo == PROVIP_ALGO_TCGEN05_CLUSTER) {
      e = hs_launch_fused(a, &tq, &tk, s, &launched, overlap, geom);
    }
    if (e == cudaSuccess && !launched) e = hs_launch_tc(a, &tq, &tk, s, geom);
  } else {
    e = hs_launch_simt(a, dtype, s, geom);
  }
  if (e != cudaSuccess) return cuda_fail(e, "head_scores launch");
  return PROVIP_OK;
}

int compact_validate(const int* idx, int B, int N_v, int keep, const void* hidden, int D,
                     const void* K, const void* V, int H_kv, int d_h, const int* pos, int P,
                     const int* seq_len, int L_max, int vis_start, int dtype, void* hidden_out,
                     void* K_out, void* V_out, int* pos_out) {
  if (!idx || !seq_len) return fail(PROVIP_ERR_INVALID_ARG, "compact: null idx/seq_len");
  if (!hidden || !hidden_out) return fail(PROVIP_ERR_INVALID_ARG, "compact: hidden is required");
  if (B < 1 || N_v < 1 || D < 1 || L_max < 1 || vis_start < 0 || vis_start + N_v > L_max)
    return fail(PROVIP_ERR_INVALID_ARG, "compact: bad sizes");
  if (keep < 1 || keep > N_v) return fail(PROVIP_ERR_INVALID_ARG, "compact: keep %d not in [1, N_v]", keep);
  if (!dtype_ok(dtype)) return fail(PROVIP_ERR_UNSUPPORTED, "compact: dtype %d", dtype);
  if ((K == nullptr) != (K_out == nullptr) || (V == nullptr) != (V_out == nullptr))
    return fail(PROVIP_ERR_INVALID_ARG, "compact: K/V given without output (or vice versa)");
  if ((K || V) && (H_kv < 1 || d_h < 1)) return fail(PROVIP_ERR_INVALID_ARG, "compact: bad H_kv/d_h");
  if (pos && (!pos_out || P < 1)) return fail(PROVIP_ERR_INVALID_ARG, "compact: pos without pos_out/P");
  const long long hb = (long long)D * esize(dtype), kb = (long long)H_kv * d_h * esize(dtype);
  if (hb % 16 || ((K || V) && kb % 16))
    return fail(PROVIP_ERR_UNSUPPORTED, "compact: row bytes must be multiples of 16");
  const void* ptrs[6] = {hidden, hidden_out, K, K_out, V, V_out};
  for (const void* p : ptrs)
    if (p && !aligned16(p)) return fail(PROVIP_ERR_UNSUPPORTED, "compact: tensor not 16-byte aligned");
  return PROVIP_OK;
}

CompactArgs compact_args(const int* idx, int B, int N_v, int keep, const void* hidden, int D,
                         const void* K, const void* V, int H_kv, int d_h, const int* pos, int P,
                         const int* seq_len, int L_max, int vis_start, int dtype,
                         void* hidden_out, void* K_out, void* V_out, int* pos_out,
                         int* seq_len_out, unsigned* err) {
  CompactArgs a;
  memset(&a, 0, sizeof(a));
  const long long hb = (long long)D * esize(dtype), kb = (long long)H_kv * d_h * esize(dtype);
  int t = 0;
  a.src[t] = static_cast<const char*>(hidden);
  a.dst[t] = static_cast<char*>(hidden_out);
  a.row_bytes[t++] = hb;
  if (K) {
    a.src[t] = static_cast<const char*>(K);
    a.dst[t] = static_cast<char*>(K_out);
    a.row_bytes[t++] = kb;
  }
  if (V) {
    a.src[t] = static_cast<const char*>(V);
    a.dst[t] = static_cast<char*>(V_out);
    a.row_bytes[t++] = kb;
  }
  a.n_tensors = t;
  a.pos = pos;
  a.pos_out = pos_out;
  a.P = pos ? P : 0;
  a.idx = idx;
  a.keep = keep;
  a.N_v = N_v;
  a.vis_start = vis_start;
  a.seq_len = seq_len;
  a.seq_len_out = seq_len_out;
  a.B = B;
  a.L_max = L_max;
  a.L_out = L_max - N_v + keep;
  a.err = err;
  return a;
}

// similarity pass: workspace partition
// row chunks of the visual-row norm/sum pass: about 400 CTAs over the batch,
// at least 8 rows each
int rel_splits(int B, int N_v) {
  int n = (400 + B - 1) / B;
  const int by_rows = (N_v + 7) / 8;
  if (n > by_rows) n = by_rows;
  return n < 1 ? 1 : n;
}
int merge_splits(int B, int N_v, int keep) {
  const int rows = ((N_v + 127) / 128) * B;
  const int cols = (keep + 63) / 64;
  int n = (512 + rows - 1) / rows;
  if (n > cols) n = cols;
  if (n > 16) n = 16;
  return n < 1 ? 1 : n;
}
// rows of the per-split argmax workspace: enough for either merge path
int merge_ws_splits(int B, int N_v, int keep) {
  const int a = merge_splits(B, N_v, keep);
  return a > kMergeMaxSplit ? a : kMergeMaxSplit;
}

struct SimWs {
  float* G = nullptr;
  uint8_t* mask = nullptr;
  float* inv_v = nullptr;
  float* sum = nullptr;
  float* mu = nullptr;
  float* invt = nullptr;
  float* p = nullptr;
  float* best = nullptr;
  int* bidx = nullptr;
  int* assign = nullptr;
  int* pruned = nullptr;
  void* perm = nullptr;
};

int sim_validate_common(const void* emb, int B, int N, int D, int dtype, const char* what) {
  if (!emb) return fail(PROVIP_ERR_INVALID_ARG, "%s: null embeddings", what);
  if (B < 1 || N < 1 || D < 1) return fail(PROVIP_ERR_INVALID_ARG, "%s: non-positive size", what);
  if (!dtype_ok(dtype)) return fail(PROVIP_ERR_UNSUPPORTED, "%s: dtype %d", what, dtype);
  if (D % 8) return fail(PROVIP_ERR_UNSUPPORTED, "%s: D must be a multiple of 8", what);
  if (!aligned16(emb)) return fail(PROVIP_ERR_UNSUPPORTED, "%s: embeddings not 16-byte aligned", what);
  return PROVIP_OK;
}

int check_ws(size_t need, void* ws, size_t ws_bytes, const char* what) {
  if (need == 0) return PROVIP_OK;
  if (!ws || ws_bytes < need)
    return fail(PROVIP_ERR_WORKSPACE, "%s: workspace %zu < %zu bytes", what, ws ? ws_bytes : (size_t)0, need);
  if (reinterpret_cast<uintptr_t>(ws) % kAlign)
    return fail(PROVIP_ERR_INVALID_ARG, "%s: workspace not 256-byte aligned", what);
  return PROVIP_OK;
}

SimArgs sim_args(const void* emb_v, const void* emb_t, const int* text_len, int B, int N_v, int D,
                 int N_t_max, int dtype, unsigned* err) {
  SimArgs a;
  a.emb_v = emb_v;
  a.emb_t = emb_t;
  a.text_len = text_len;
  a.B = B;
  a.N_v = N_v;
  a.D = D;
  a.N_t_max = N_t_max;
  a.dtype = dtype;
  a.err = err;
  return a;
}

}  // namespace

// ===========================================================================
// status
// ===========================================================================
extern "C" const char* provip_status_string(int status) {
  switch (status) {
    case PROVIP_OK: return "PROVIP_OK";
    case PROVIP_ERR_INVALID_ARG: return "PROVIP_ERR_INVALID_ARG";
    case PROVIP_ERR_UNSUPPORTED: return "PROVIP_ERR_UNSUPPORTED";
    case PROVIP_ERR_WORKSPACE: return "PROVIP_ERR_WORKSPACE";
    case PROVIP_ERR_CUDA: return "PROVIP_ERR_CUDA";
    case PROVIP_ERR_TIMEOUT: return "PROVIP_ERR_TIMEOUT";
    default: return "PROVIP_ERR_UNKNOWN";
  }
}

extern "C" const char* provip_last_error(void) { return g_last_error; }

extern "C" int provip_version(void) { return 10000; }

extern "C" int provip_set_option(int option, int value) {
  if (value != 0 && value != 1) return fail(PROVIP_ERR_INVALID_ARG, "set_option: value %d", value);
  if (option == PROVIP_OPT_MERGE_PAIRS) {
    merge_pair_enable(value);
    return PROVIP_OK;
  }
  return fail(PROVIP_ERR_INVALID_ARG, "set_option: unknown option %d", option);
}

extern "C" int provip_device_status(unsigned* bits, int clear) {
  DevInfo* d;
  int rc = dev_info(&d);
  if (rc) return rc;
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceSynchronize");
  unsigned v = 0;
  e = cudaMemcpy(&v, d->status, sizeof(v), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "read device status");
  if (clear) {
    e = cudaMemset(d->status, 0, sizeof(unsigned));
    if (e != cudaSuccess) return cuda_fail(e, "clear device status");
  }
  if (bits) *bits = v;
  if (v & PROVIP_DEVSTAT_TIMEOUT) return PROVIP_ERR_TIMEOUT;
  if (v & PROVIP_DEVSTAT_BAD_ARG) return PROVIP_ERR_INVALID_ARG;
  return PROVIP_OK;
}

namespace {
// one thread waits on an mbarrier whose single expected arrival never comes
__global__ void selftest_wait_kernel(unsigned* err) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_mbar_init();
    mbar_wait(&bar, 0, err);  // gives up after the wait budget and sets kErrTimeout
  }
}
}  // namespace

extern "C" int provip_selftest_wait_timeout(void* stream) {
  DevInfo* d;
  int rc = dev_info(&d);
  if (rc) return rc;
  selftest_wait_kernel<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(d->status);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "selftest_wait_kernel launch");
  return PROVIP_OK;
}

// ===========================================================================
// pre-LLM pass
// ===========================================================================
// the text Gram, in as many K parts as its tcgen05 form uses (bf16)
static size_t crit_gram_floats(int B, int N_t_max, int D, int dtype) {
  const int parts = crit_splits(N_t_max, D, dtype);
  return (size_t)(parts > 0 ? parts : 1) * B * N_t_max * N_t_max;
}

extern "C" size_t provip_crit_text_workspace_size(int B, int N_t_max, int D) {
  Carve c(nullptr);
  c.take<float>(crit_gram_floats(B, N_t_max, D, PROVIP_BF16));  // the larger of the two dtypes' needs
  return c.off;
}

extern "C" int provip_crit_text(const void* emb_t, int B, int N_t_max, int D, const int* text_len,
                                int dtype, uint8_t* mask_out, float* r_out, void* ws,
                                size_t ws_bytes, void* stream) {
  NvtxRange nvtx_range("provip_crit_text");
  int rc = sim_validate_common(emb_t, B, N_t_max, D, dtype, "crit_text");
  if (rc) return rc;
  if (!text_len || !mask_out) return fail(PROVIP_ERR_INVALID_ARG, "crit_text: null text_len/mask_out");
  if (N_t_max > 4096) return fail(PROVIP_ERR_UNSUPPORTED, "crit_text: N_t_max > 4096");
  if ((rc = check_ws(provip_crit_text_workspace_size(B, N_t_max, D), ws, ws_bytes, "crit_text"))) return rc;
  DevInfo* d;
  if ((rc = dev_info(&d))) return rc;
  Carve c(ws);
  float* G = c.take<float>(crit_gram_floats(B, N_t_max, D, PROVIP_BF16));
  SimArgs a = sim_args(nullptr, emb_t, text_len, B, 1, D, N_t_max, dtype, d->status);
  cudaError_t e = crit_text_launch(a, mask_out, r_out, G, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? PROVIP_OK : cuda_fail(e, "crit_text launch");
}

static size_t relevance_ws(Carve& c, int B, int N_v, int D, int N_t_max, SimWs& w) {
  const int ns = rel_splits(B, N_v);
  w.inv_v = c.take<float>((size_t)B * N_v);
  // the split column sums of the CUDA-core form, or the cosines and tile sums
  // of the tensor-core form
  const size_t sum_f = (size_t)(ns + 1) * B * D, fused_f = relevance_fused_floats(B, N_v, N_t_max);
  w.sum = c.take<float>(sum_f > fused_f ? sum_f : fused_f);
  w.mu = c.take<float>((size_t)B * N_t_max);
  w.invt = c.take<float>((size_t)B * N_t_max);
  return c.off;
}

extern "C" size_t provip_relevance_workspace_size(int B, int N_v, int D, int N_t_max) {
  Carve c(nullptr);
  SimWs w;
  return relevance_ws(c, B, N_v, D, N_t_max, w);
}

extern "C" int provip_relevance(const void* emb_v, int B, int N_v, int D, const void* emb_t,
                                const int* text_len, int N_t_max, const uint8_t* crit_mask,
                                int dtype, float* p_out, void* ws, size_t ws_bytes, void* stream) {
  NvtxRange nvtx_range("provip_relevance");
  int rc = sim_validate_common(emb_v, B, N_v, D, dtype, "relevance");
  if (rc) return rc;
  if ((rc = sim_validate_common(emb_t, B, N_t_max, D, dtype, "relevance"))) return rc;
  if (!text_len || !crit_mask || !p_out) return fail(PROVIP_ERR_INVALID_ARG, "relevance: null pointer");
  if ((rc = check_ws(provip_relevance_workspace_size(B, N_v, D, N_t_max), ws, ws_bytes, "relevance"))) return rc;
  DevInfo* d;
  if ((rc = dev_info(&d))) return rc;
  Carve c(ws);
  SimWs w;
  relevance_ws(c, B, N_v, D, N_t_max, w);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  SimArgs a = sim_args(emb_v, emb_t, text_len, B, N_v, D, N_t_max, dtype, d->status);
  cudaError_t e =
      relevance_launch(a, crit_mask, w.inv_v, p_out, w.sum, w.mu, w.invt, rel_splits(B, N_v), d->sms, s);
  return e == cudaSuccess ? PROVIP_OK : cuda_fail(e, "relevance launch");
}

extern "C" int provip_topk(const float* scores, int B, int N, int k, int* idx_out, void* stream) {
  NvtxRange nvtx_range("provip_topk");
  if (!scores || !idx_out) return fail(PROVIP_ERR_INVALID_ARG, "topk: null pointer");
  if (B < 1 || N < 1 || k < 1 || k > N) return fail(PROVIP_ERR_INVALID_ARG, "topk: need 1 <= k <= N");
  if (N > kTopkMaxN) return fail(PROVIP_ERR_UNSUPPORTED, "topk: N > %d", kTopkMaxN);
  DevInfo* d;
  int rc = dev_info(&d);
  if (rc) return rc;
  TopkArgs a;
  memset(&a, 0, sizeof(a));
  a.scores = scores;
  a.B = B;
  a.N = N;
  a.k = k;
  a.idx_out = idx_out;
  a.err = d->status;
  cudaError_t e = topk_launch(a, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? PROVIP_OK : cuda_fail(e, "topk launch");
}

static size_t merge_ws(Carve& c, int B, int N_v, int D, int keep, SimWs& w) {
  const int ns = merge_ws_splits(B, N_v, keep);
  w.inv_v = c.take<float>((size_t)B * N_v);
  w.best = c.take<float>((size_t)ns * B * N_v);
  w.bidx = c.take<int>((size_t)ns * B * N_v);
  w.pruned = c.take<int>((size_t)B * N_v);
  w.perm = c.take<uint16_t>((size_t)B * N_v * D);
  return c.off;
}

extern "C" size_t provip_merge_workspace_size(int B, int N_v, int D, int keep) {
  Carve c(nullptr);
  SimWs w;
  return merge_ws(c, B, N_v, D, keep, w);
}

static int merge_validate(const void* emb_v, int B, int N_v, int D, const int* keep_idx, int keep,
                          int dtype, int* assign_out) {
  int rc = sim_validate_common(emb_v, B, N_v, D, dtype, "merge");
  if (rc) return rc;
  if (!keep_idx || !assign_out) return fail(PROVIP_ERR_INVALID_ARG, "merge: null keep_idx/assign_out");
  if (keep < 1 || keep > N_v) return fail(PROVIP_ERR_INVALID_ARG, "merge: keep %d not in [1, N_v]", keep);
  if (D > 8192) return fail(PROVIP_ERR_UNSUPPORTED, "merge: D > 8192");
  return PROVIP_OK;
}

extern "C" int provip_merge(const void* emb_v, int B, int N_v, int D, const int* keep_idx, int keep,
                            int dtype, int* assign_out, void* merged_out, void* ws, size_t ws_bytes,
                            void* stream) {
  NvtxRange nvtx_range("provip_merge");
  int rc = merge_validate(emb_v, B, N_v, D, keep_idx, keep, dtype, assign_out);
  if (rc) return rc;
  if ((rc = check_ws(provip_merge_workspace_size(B, N_v, D, keep), ws, ws_bytes, "merge"))) return rc;
  DevInfo* d;
  if ((rc = dev_info(&d))) return rc;
  Carve c(ws);
  SimWs w;
  merge_ws(c, B, N_v, D, keep, w);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  SimArgs a = sim_args(emb_v, nullptr, nullptr, B, N_v, D, 1, dtype, d->status);
  // the cosine's kept-row factor 1/|e_k| is all the nearest-centroid argmax
  // needs (the pruned row's own norm is the same for every kept k)
  cudaError_t e = kept_inv_norm_launch(a, keep_idx, keep, w.inv_v, s);
  if (e == cudaSuccess)
    e = merge_launch(a, keep_idx, keep, w.inv_v, assign_out, merged_out, w.best, w.bidx,
                     merge_splits(B, N_v, keep), w.pruned, dtype == PROVIP_BF16 ? w.perm : nullptr,
                     d->sms, s);
  return e == cudaSuccess ? PROVIP_OK : cuda_fail(e, "merge launch");
}

static size_t simred_ws(Carve& c, int B, int N_v, int D, int N_t_max, int keep_pre, SimWs& w) {
  w.G = c.take<float>(crit_gram_floats(B, N_t_max, D, PROVIP_BF16));
  w.mask = c.take<uint8_t>((size_t)B * N_t_max);
  w.p = c.take<float>((size_t)B * N_v);
  w.assign = c.take<int>((size_t)B * N_v);
  SimWs r;
  relevance_ws(c, B, N_v, D, N_t_max, r);
  const int ns = merge_ws_splits(B, N_v, keep_pre);
  w.inv_v = r.inv_v;
  w.sum = r.sum;
  w.mu = r.mu;
  w.invt = r.invt;
  w.best = c.take<float>((size_t)ns * B * N_v);
  w.bidx = c.take<int>((size_t)ns * B * N_v);
  w.pruned = c.take<int>((size_t)B * N_v);
  w.perm = c.take<uint16_t>((size_t)B * N_v * D);
  return c.off;
}

extern "C" size_t provip_similarity_reduce_workspace_size(int B, int N_v, int D, int N_t_max,
                                                          int keep_pre) {
  Carve c(nullptr);
  SimWs w;
  return simred_ws(c, B, N_v, D, N_t_max, keep_pre, w);
}

extern "C" int provip_similarity_reduce(const void* emb_v, int B, int N_v, int D, const void* emb_t,
                                        const int* text_len, int N_t_max,
                                        const uint8_t* crit_mask_or_null, int keep_pre, int dtype,
                                        int* idx_out, void* merged_out_or_null,
                                        int* assign_out_or_null, float* p_out_or_null,
                                        uint8_t* mask_out_or_null, void* ws, size_t ws_bytes,
                                        void* stream) {
  NvtxRange nvtx_range("provip_similarity_reduce");
  int rc = sim_validate_common(emb_v, B, N_v, D, dtype, "similarity_reduce");
  if (rc) return rc;
  if ((rc = sim_validate_common(emb_t, B, N_t_max, D, dtype, "similarity_reduce"))) return rc;
  if (!text_len || !idx_out) return fail(PROVIP_ERR_INVALID_ARG, "similarity_reduce: null text_len/idx_out");
  if (keep_pre < 1 || keep_pre > N_v) return fail(PROVIP_ERR_INVALID_ARG, "similarity_reduce: keep_pre %d", keep_pre);
  if (N_v > kTopkMaxN) return fail(PROVIP_ERR_UNSUPPORTED, "similarity_reduce: N_v > %d", kTopkMaxN);
  if (N_t_max > 4096) return fail(PROVIP_ERR_UNSUPPORTED, "similarity_reduce: N_t_max > 4096");
  if (merged_out_or_null && D > 8192) return fail(PROVIP_ERR_UNSUPPORTED, "similarity_reduce: D > 8192");
  if ((rc = check_ws(provip_similarity_reduce_workspace_size(B, N_v, D, N_t_max, keep_pre), ws,
                     ws_bytes, "similarity_reduce")))
    return rc;
  DevInfo* d;
  if ((rc = dev_info(&d))) return rc;
  Carve c(ws);
  SimWs w;
  simred_ws(c, B, N_v, D, N_t_max, keep_pre, w);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  SimArgs a = sim_args(emb_v, emb_t, text_len, B, N_v, D, N_t_max, dtype, d->status);
  const uint8_t* mask = crit_mask_or_null;
  uint8_t* mask_dst = mask_out_or_null ? mask_out_or_null : w.mask;
  cudaError_t e = cudaSuccess;
  cudaEvent_t mask_ready = nullptr;
  if (!mask) {
    // the critical text rows (their Gram and threshold) run on a side stream
    // beside the relevance Gram, which reads no mask; the stream waits for
    // them before the kernel that takes the max over the critical rows
    SideStream* side;
    if ((rc = side_stream(&side))) return rc;
    e = cudaEventRecord(side->fork, s);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(side->s, side->fork, 0);
    if (e == cudaSuccess) e = crit_text_launch(a, mask_dst, nullptr, w.G, side->s);
    if (e == cudaSuccess) e = cudaEventRecord(side->join, side->s);
    if (e == cudaSuccess) mask_ready = side->join;
    mask = mask_dst;
  } else if (mask_out_or_null) {
    e = cudaMemcpyAsync(mask_out_or_null, mask, (size_t)B * N_t_max, cudaMemcpyDeviceToDevice, s);
  }
  float* p = p_out_or_null ? p_out_or_null : w.p;
  if (e == cudaSuccess) {
    e = relevance_launch(a, mask, w.inv_v, p, w.sum, w.mu, w.invt, rel_splits(B, N_v), d->sms, s, mask_ready);
    if (e != cudaSuccess && mask_ready != nullptr) cudaStreamWaitEvent(s, mask_ready, 0);  // join even so
  }
  if (e == cudaSuccess) {
    TopkArgs t;
    memset(&t, 0, sizeof(t));
    t.scores = p;
    t.B = B;
    t.N = N_v;
    t.k = keep_pre;
    t.idx_out = idx_out;
    t.err = d->status;
    if (merged_out_or_null && topk_writes_index(N_v)) {
      // the selection also writes the merge's kept-position map and pruned list
      t.kpos_out = assign_out_or_null ? assign_out_or_null : w.assign;
      t.pruned_out = w.pruned;
    }
    e = topk_launch(t, s, true);  // a programmatic dependent of the relevance's last kernel
  }
  if (e == cudaSuccess && merged_out_or_null)
    e = merge_launch(a, idx_out, keep_pre, w.inv_v, assign_out_or_null ? assign_out_or_null : w.assign,
                     merged_out_or_null, w.best, w.bidx,
                     merge_splits(B, N_v, keep_pre), w.pruned,
                     dtype == PROVIP_BF16 ? w.perm : nullptr, d->sms, s, topk_writes_index(N_v));
  return e == cudaSuccess ? PROVIP_OK : cuda_fail(e, "similarity_reduce launch");
}

// ===========================================================================
// in-LLM pass
// ===========================================================================
extern "C" size_t provip_head_scores_workspace_size(int B, int L_max, int H_sel, int N_t_max,
                                                    int N_v, int algo, int dtype) {
  algo = resolve_algo(algo, dtype);
  HSShape sh = hs_shape(L_max, N_t_max, N_v, algo);
  Carve c(nullptr);
  float2* st;
  float* pa;
  return hs_ws(c, B, H_sel, sh, N_v, &st, &pa);
}

extern "C" int provip_head_scores(const void* Q, const void* K, int B, int L_max, int H_q, int H_kv,
                                  int d_h, const int* head_list, int H_sel, const int* text_start,
                                  const int* text_len, const uint8_t* row_mask_or_null, int N_t_max,
                                  int vis_start, int N_v, const int* seq_len, int dtype, int algo,
                                  float* scores, void* ws, size_t ws_bytes, void* stream) {
  NvtxRange nvtx_range("provip_head_scores");
  algo = resolve_algo(algo, dtype);
  int rc = hs_validate(Q, K, B, L_max, H_q, H_kv, d_h, head_list, H_sel, text_start, text_len,
                       N_t_max, vis_start, N_v, seq_len, dtype, algo);
  if (rc) return rc;
  if (!scores) return fail(PROVIP_ERR_INVALID_ARG, "head_scores: null scores");
  if ((rc = check_ws(provip_head_scores_workspace_size(B, L_max, H_sel, N_t_max, N_v, algo, dtype),
                     ws, ws_bytes, "head_scores")))
    return rc;
  DevInfo* d;
  if ((rc = dev_info(&d))) return rc;
  HSShape sh = hs_shape(L_max, N_t_max, N_v, algo);
  Carve c(ws);
  float2* stats;
  float* partial;
  hs_ws(c, B, H_sel, sh, N_v, &stats, &partial);
  HSArgs a = hs_args(Q, K, B, L_max, H_q, H_kv, d_h, head_list, H_sel, text_start, text_len,
                     row_mask_or_null, N_t_max, vis_start, N_v, seq_len, sh, stats, partial,
                     d->status);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if ((rc = hs_run(a, dtype, algo, s))) return rc;
  cudaError_t e = hs_launch_reduce(a, scores, s);
  return e == cudaSuccess ? PROVIP_OK : cuda_fail(e, "head_scores reduce");
}

// true if any pointer is host memory (pinned and mapped, or memory the device
// reaches through the system's address translation): the rows are then copied
// with vector loads and stores, which work on any memory the device can
// dereference, instead of bulk copies
static bool any_host_memory(std::initializer_list<const void*> ptrs) {
  for (const void* p : ptrs) {
    if (p == nullptr) continue;
    cudaPointerAttributes at;
    if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
      cudaGetLastError();  // not known to the runtime: not device memory
      return true;
    }
    if (at.type != cudaMemoryTypeDevice && at.type != cudaMemoryTypeManaged) return true;
  }
  return false;
}

extern "C" int provip_compact(const int* idx, int B, int N_v, int keep, const void* hidden, int D,
                              const void* K, const void* V, int H_kv, int d_h, const int* pos,
                              int P, const int* seq_len, int L_max, int vis_start, int dtype,
                              void* hidden_out, void* K_out, void* V_out, int* pos_out,
                              int* seq_len_out, void* stream) {
  NvtxRange nvtx_range("provip_compact");
  int rc = compact_validate(idx, B, N_v, keep, hidden, D, K, V, H_kv, d_h, pos, P, seq_len, L_max,
                            vis_start, dtype, hidden_out, K_out, V_out, pos_out);
  if (rc) return rc;
  DevInfo* d;
  if ((rc = dev_info(&d))) return rc;
  CompactArgs a = compact_args(idx, B, N_v, keep, hidden, D, K, V, H_kv, d_h, pos, P, seq_len,
                               L_max, vis_start, dtype, hidden_out, K_out, V_out, pos_out,
                               seq_len_out, d->status);
  const bool host_rows = any_host_memory({hidden, K, V, pos, hidden_out, K_out, V_out, pos_out});
  cudaError_t e = compact_launch(a, d->sms, static_cast<cudaStream_t>(stream), false, true, false, host_rows);
  return e == cudaSuccess ? PROVIP_OK : cuda_fail(e, "compact launch");
}

extern "C" int provip_topk_compact(const float* scores, int B, int N_v, int keep, const void* hidden,
                                   int D, const void* K, const void* V, int H_kv, int d_h,
                                   const int* pos, int P, const int* seq_len, int L_max,
                                   int vis_start, int dtype, void* hidden_out, void* K_out,
                                   void* V_out, int* pos_out, int* idx_out, int* seq_len_out,
                                   void* stream) {
  NvtxRange nvtx_range("provip_topk_compact");
  if (!scores || !idx_out) return fail(PROVIP_ERR_INVALID_ARG, "topk_compact: null scores/idx_out");
  int rc = compact_validate(idx_out, B, N_v, keep, hidden, D, K, V, H_kv, d_h, pos, P, seq_len,
                            L_max, vis_start, dtype, hidden_out, K_out, V_out, pos_out);
  if (rc) return rc;
  if ((rc = provip_topk(scores, B, N_v, keep, idx_out, stream))) return rc;
  return provip_compact(idx_out, B, N_v, keep, hidden, D, K, V, H_kv, d_h, pos, P, seq_len, L_max,
                        vis_start, dtype, hidden_out, K_out, V_out, pos_out, seq_len_out, stream);
}

extern "C" size_t provip_prune_workspace_size(int B, int L_max, int H_sel, int N_t_max, int N_v,
                                              int algo, int dtype) {
  return provip_head_scores_workspace_size(B, L_max, H_sel, N_t_max, N_v, algo, dtype);
}

static int head_topk_impl(const void* Q, const void* K, int B, int L_max, int H_q, int H_kv,
                                int d_h, const int* head_list, int H_sel, const int* text_start,
                                const int* text_len, const uint8_t* row_mask_or_null, int N_t_max,
                                int vis_start, int N_v, const int* seq_len, int keep, int dtype,
                                int algo, int* idx_out, float* scores_out_or_null, void* ws,
                                size_t ws_bytes, void* stream, bool overlap) {
  algo = resolve_algo(algo, dtype);
  int rc = hs_validate(Q, K, B, L_max, H_q, H_kv, d_h, head_list, H_sel, text_start, text_len,
                       N_t_max, vis_start, N_v, seq_len, dtype, algo);
  if (rc) return rc;
  if (!idx_out) return fail(PROVIP_ERR_INVALID_ARG, "head_topk: null idx_out");
  if (keep < 1 || keep > N_v) return fail(PROVIP_ERR_INVALID_ARG, "head_topk: keep %d not in [1, N_v]", keep);
  if (N_v > kTopkMaxN) return fail(PROVIP_ERR_UNSUPPORTED, "head_topk: N_v > %d", kTopkMaxN);
  if ((long long)((N_t_max + kRowBlock - 1) / kRowBlock) * H_sel * N_v >= (1ll << 31))
    return fail(PROVIP_ERR_UNSUPPORTED, "head_topk: too many head partials");
  if ((rc = check_ws(provip_head_scores_workspace_size(B, L_max, H_sel, N_t_max, N_v, algo, dtype), ws,
                     ws_bytes, "head_topk")))
    return rc;
  DevInfo* d;
  if ((rc = dev_info(&d))) return rc;
  HSShape sh = hs_shape(L_max, N_t_max, N_v, algo);
  Carve c(ws);
  float2* stats;
  float* partial;
  hs_ws(c, B, H_sel, sh, N_v, &stats, &partial);
  HSArgs a = hs_args(Q, K, B, L_max, H_q, H_kv, d_h, head_list, H_sel, text_start, text_len,
                     row_mask_or_null, N_t_max, vis_start, N_v, seq_len, sh, stats, partial,
                     d->status);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if ((rc = hs_run(a, dtype, algo, s, overlap))) return rc;
  TopkArgs t;
  memset(&t, 0, sizeof(t));
  t.partial = partial;
  t.n_part = sh.n_rb * H_sel;
  t.text_len = text_len;
  t.row_mask = row_mask_or_null;
  t.N_t_max = N_t_max;
  t.H_sel = H_sel;
  t.scores_out = scores_out_or_null;
  t.B = B;
  t.N = N_v;
  t.k = keep;
  t.idx_out = idx_out;
  t.err = d->status;
  // a programmatic dependent of the head-score kernel: launched early, waits
  // for the partials on the device
  cudaError_t e = topk_launch(t, s, true);
  return e == cudaSuccess ? PROVIP_OK : cuda_fail(e, "head_topk topk");
}

extern "C" int provip_head_topk(const void* Q, const void* K, int B, int L_max, int H_q, int H_kv,
                                int d_h, const int* head_list, int H_sel, const int* text_start,
                                const int* text_len, const uint8_t* row_mask_or_null, int N_t_max,
                                int vis_start, int N_v, const int* seq_len, int keep, int dtype,
                                int algo, int* idx_out, float* scores_out_or_null, void* ws,
                                size_t ws_bytes, void* stream) {
  NvtxRange nvtx_range("provip_head_topk");
  return head_topk_impl(Q, K, B, L_max, H_q, H_kv, d_h, head_list, H_sel, text_start, text_len,
                        row_mask_or_null, N_t_max, vis_start, N_v, seq_len, keep, dtype, algo,
                        idx_out, scores_out_or_null, ws, ws_bytes, stream, false);
}

extern "C" int provip_prune(const void* Q, const void* K, const void* V, const void* hidden, int B,
                            int L_max, int H_q, int H_kv, int d_h, int D, const int* head_list,
                            int H_sel, const int* text_start, const int* text_len,
                            const uint8_t* row_mask_or_null, int N_t_max, int vis_start, int N_v,
                            const int* seq_len, const int* pos, int P, int keep, int dtype,
                            int algo, void* hidden_out, void* K_out, void* V_out, int* pos_out,
                            int* idx_out, int* seq_len_out, float* scores_out_or_null, void* ws,
                            size_t ws_bytes, unsigned flags, void* stream) {
  NvtxRange nvtx_range("provip_prune");
  // validate both halves before enqueueing anything
  if (flags & ~(unsigned)(PROVIP_PRUNE_OVERLAP_PREVIOUS | PROVIP_PRUNE_CONCURRENT | PROVIP_PRUNE_HOST_ROWS))
    return fail(PROVIP_ERR_INVALID_ARG, "prune: unknown flags 0x%x", flags);
  int rc = hs_validate(Q, K, B, L_max, H_q, H_kv, d_h, head_list, H_sel, text_start, text_len,
                       N_t_max, vis_start, N_v, seq_len, dtype, resolve_algo(algo, dtype));
  if (rc) return rc;
  if ((rc = compact_validate(idx_out ? idx_out : reinterpret_cast<int*>(16), B, N_v, keep, hidden, D,
                             K, V, H_kv, d_h, pos, P, seq_len, L_max, vis_start, dtype, hidden_out,
                             K_out, V_out, pos_out)))
    return rc;
  rc = head_topk_impl(Q, K, B, L_max, H_q, H_kv, d_h, head_list, H_sel, text_start, text_len,
                      row_mask_or_null, N_t_max, vis_start, N_v, seq_len, keep, dtype, algo,
                      idx_out, scores_out_or_null, ws, ws_bytes, stream,
                      (flags & PROVIP_PRUNE_OVERLAP_PREVIOUS) != 0);
  if (rc) return rc;
  // the compaction is a programmatic dependent of the selection: the rows that
  // do not depend on idx are copied while the selection finishes
  DevInfo* d;
  if ((rc = dev_info(&d))) return rc;
  CompactArgs ca = compact_args(idx_out, B, N_v, keep, hidden, D, K, V, H_kv, d_h, pos, P, seq_len,
                                L_max, vis_start, dtype, hidden_out, K_out, V_out, pos_out,
                                seq_len_out, d->status);
  // the next step's head scores overlap this compaction: the deeper ring only
  // beside the streaming form
  const int form = tc_form(resolve_algo(algo, dtype), B, H_sel, hs_shape(L_max, N_t_max, N_v, algo).n_rb,
                           d->sms);
  cudaError_t e = compact_launch(ca, d->sms, static_cast<cudaStream_t>(stream), true,
                                 form == PROVIP_ALGO_TCGEN05_STREAM, (flags & PROVIP_PRUNE_CONCURRENT) != 0,
                                 (flags & PROVIP_PRUNE_HOST_ROWS) != 0);
  return e == cudaSuccess ? PROVIP_OK : cuda_fail(e, "prune compact");
}

// ===========================================================================
// visual-head identification (Sec. 4.4): head confidence over every head on
// the critical text rows, the N_vis most confident heads per sample, and the
// token importance from those heads alone
// ===========================================================================
extern "C" size_t provip_visual_heads_workspace_size(int B, int L_max, int H_q, int N_t_max,
                                                     int N_v, int N_vis, int algo, int dtype) {
  algo = resolve_algo(algo, dtype);
  HSShape sh = hs_shape(L_max, N_t_max, N_v, algo);
  Carve c(nullptr);
  float2* st;
  float* pa;
  hs_ws(c, B, H_q, sh, N_v, &st, &pa);
  ConfWs w;
  return conf_ws(c, B, H_q, N_t_max, sh, algo, N_vis, w);
}

// keep == 0: confidence and selection only; keep >= 1: also the top-keep
// tokens by the selected heads' scores
static int visual_heads_impl(const void* Q, const void* K, int B, int L_max, int H_q, int H_kv,
                             int d_h, const int* text_start, const int* text_len,
                             const uint8_t* crit_mask_or_null, int N_t_max, int vis_start, int N_v,
                             const int* seq_len, int N_vis, int keep, int dtype, int algo,
                             float* conf_out_or_null, int* vis_heads_out, int* idx_out,
                             float* scores_out_or_null, void* ws, size_t ws_bytes, void* stream,
                             bool overlap, const char* what) {
  algo = resolve_algo(algo, dtype);
  if (H_q > kMaxHeads) return fail(PROVIP_ERR_UNSUPPORTED, "%s: H_q %d > %d", what, H_q, kMaxHeads);
  int rc = hs_validate(Q, K, B, L_max, H_q, H_kv, d_h, nullptr, H_q, text_start, text_len, N_t_max,
                       vis_start, N_v, seq_len, dtype, algo);
  if (rc) return rc;
  if (N_vis < 1 || N_vis > H_q) return fail(PROVIP_ERR_INVALID_ARG, "%s: N_vis %d not in [1, H_q]", what, N_vis);
  if (keep > 0) {
    if (!idx_out) return fail(PROVIP_ERR_INVALID_ARG, "%s: null idx_out", what);
    if (keep > N_v) return fail(PROVIP_ERR_INVALID_ARG, "%s: keep %d not in [1, N_v]", what, keep);
    if (N_v > kTopkMaxN) return fail(PROVIP_ERR_UNSUPPORTED, "%s: N_v > %d", what, kTopkMaxN);
  }
  const HSShape sh = hs_shape(L_max, N_t_max, N_v, algo);
  if ((long long)sh.n_rb * H_q * N_v >= (1ll << 31))
    return fail(PROVIP_ERR_UNSUPPORTED, "%s: too many head partials", what);
  if ((rc = check_ws(provip_visual_heads_workspace_size(B, L_max, H_q, N_t_max, N_v, N_vis, algo, dtype),
                     ws, ws_bytes, what)))
    return rc;
  DevInfo* d;
  if ((rc = dev_info(&d))) return rc;
  Carve c(ws);
  float2* stats;
  float* partial;
  hs_ws(c, B, H_q, sh, N_v, &stats, &partial);
  ConfWs cw;
  conf_ws(c, B, H_q, N_t_max, sh, algo, N_vis, cw);
  HSArgs a = hs_args(Q, K, B, L_max, H_q, H_kv, d_h, nullptr, H_q, text_start, text_len, nullptr,
                     N_t_max, vis_start, N_v, seq_len, sh, stats, partial, d->status);
  a.conf_mask = crit_mask_or_null;
  a.conf_part = cw.part;
  a.conf_stride = conf_stride(sh, algo);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  ConfGeom geom{0, 0, 0};
  if ((rc = hs_run(a, dtype, algo, s, overlap, &geom))) return rc;
  ConfArgs ca;
  ca.n_vis = N_vis;
  ca.sel_out = cw.sel;
  ca.vis_heads_out = vis_heads_out;
  ca.conf_out = conf_out_or_null;
  cudaError_t e = conf_select_launch(a, geom, ca, s, true);
  if (e != cudaSuccess) return cuda_fail(e, "visual heads: selection launch");
  if (keep <= 0) return PROVIP_OK;
  TopkArgs t;
  memset(&t, 0, sizeof(t));
  t.partial = partial;
  t.n_part = sh.n_rb * H_q;
  t.text_len = text_len;
  t.N_t_max = N_t_max;
  t.H_sel = H_q;
  t.sel = cw.sel;
  t.n_sel = N_vis;
  t.scores_out = scores_out_or_null;
  t.B = B;
  t.N = N_v;
  t.k = keep;
  t.idx_out = idx_out;
  t.err = d->status;
  e = topk_launch(t, s, true);
  return e == cudaSuccess ? PROVIP_OK : cuda_fail(e, "visual heads: top-k launch");
}

extern "C" int provip_head_confidence(const void* Q, const void* K, int B, int L_max, int H_q,
                                      int H_kv, int d_h, const int* text_start, const int* text_len,
                                      const uint8_t* crit_mask_or_null, int N_t_max, int vis_start,
                                      int N_v, const int* seq_len, int N_vis, int dtype, int algo,
                                      float* conf_out_or_null, int* vis_heads_out, void* ws,
                                      size_t ws_bytes, void* stream) {
  NvtxRange nvtx_range("provip_head_confidence");
  if (!vis_heads_out) return fail(PROVIP_ERR_INVALID_ARG, "head_confidence: null vis_heads_out");
  return visual_heads_impl(Q, K, B, L_max, H_q, H_kv, d_h, text_start, text_len, crit_mask_or_null,
                           N_t_max, vis_start, N_v, seq_len, N_vis, 0, dtype, algo,
                           conf_out_or_null, vis_heads_out, nullptr, nullptr, ws, ws_bytes, stream,
                           false, "head_confidence");
}

extern "C" int provip_prune_visual_heads(
    const void* Q, const void* K, const void* V, const void* hidden, int B, int L_max, int H_q,
    int H_kv, int d_h, int D, const int* text_start, const int* text_len,
    const uint8_t* crit_mask_or_null, int N_t_max, int vis_start, int N_v, const int* seq_len,
    const int* pos, int P, int N_vis, int keep, int dtype, int algo, void* hidden_out, void* K_out,
    void* V_out, int* pos_out, int* idx_out, int* seq_len_out, float* scores_out_or_null,
    int* vis_heads_out_or_null, float* conf_out_or_null, void* ws, size_t ws_bytes,
    unsigned flags, void* stream) {
  NvtxRange nvtx_range("provip_prune_visual_heads");
  if (flags & ~(unsigned)(PROVIP_PRUNE_OVERLAP_PREVIOUS | PROVIP_PRUNE_CONCURRENT | PROVIP_PRUNE_HOST_ROWS))
    return fail(PROVIP_ERR_INVALID_ARG, "prune_visual_heads: unknown flags 0x%x", flags);
  if (keep < 1) return fail(PROVIP_ERR_INVALID_ARG, "prune_visual_heads: keep %d < 1", keep);
  int rc = compact_validate(idx_out ? idx_out : reinterpret_cast<int*>(16), B, N_v, keep, hidden, D,
                            K, V, H_kv, d_h, pos, P, seq_len, L_max, vis_start, dtype, hidden_out,
                            K_out, V_out, pos_out);
  if (rc) return rc;
  rc = visual_heads_impl(Q, K, B, L_max, H_q, H_kv, d_h, text_start, text_len, crit_mask_or_null,
                         N_t_max, vis_start, N_v, seq_len, N_vis, keep, dtype, algo,
                         conf_out_or_null, vis_heads_out_or_null, idx_out, scores_out_or_null, ws,
                         ws_bytes, stream, (flags & PROVIP_PRUNE_OVERLAP_PREVIOUS) != 0,
                         "prune_visual_heads");
  if (rc) return rc;
  DevInfo* d;
  if ((rc = dev_info(&d))) return rc;
  CompactArgs ca = compact_args(idx_out, B, N_v, keep, hidden, D, K, V, H_kv, d_h, pos, P, seq_len,
                                L_max, vis_start, dtype, hidden_out, K_out, V_out, pos_out,
                                seq_len_out, d->status);
  // every head is scored: the streaming form unless the units are fewer than the SMs
  const int form = tc_form(resolve_algo(algo, dtype), B, H_q, hs_shape(L_max, N_t_max, N_v, algo).n_rb,
                           d->sms);
  cudaError_t e = compact_launch(ca, d->sms, static_cast<cudaStream_t>(stream), true,
                                 form == PROVIP_ALGO_TCGEN05_STREAM, (flags & PROVIP_PRUNE_CONCURRENT) != 0,
                                 (flags & PROVIP_PRUNE_HOST_ROWS) != 0);
  return e == cudaSuccess ? PROVIP_OK : cuda_fail(e, "prune_visual_heads compact");
}

// ===========================================================================
// head scores without a workspace
//
// Some callers cannot hand the library any device memory: a host framework
// that owns every allocation and passes a plugin only its input and output
// tensors, or a serving loop that forbids allocator calls once it is running.
// For them the scratch of the head scores (per-chunk row statistics and
// per-head partial sums) lives in this file-scope device array instead of a
// workspace. Every GPU that loads the library keeps the array until the
// process exits.
// ===========================================================================
static constexpr size_t kNoAllocScratchBytes = (size_t)PROVIP_NOALLOC_SCRATCH_BYTES;
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];
// Device address of the array on each device. In host code the symbol only
// names a host-side stand-in, so a kernel must be given this address, looked up
// with the device current. Published with a release store: host threads making
// their first call on a device at the same moment may both look it up (the
// same value), and a reader that sees it non-null sees a complete lookup.
static std::atomic<void*> g_noalloc_addr[64];

static int noalloc_scratch_addr(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "head_scores_noalloc: cudaGetDevice");
  if (dev < 0 || dev >= 64) return fail(PROVIP_ERR_UNSUPPORTED, "head_scores_noalloc: device %d >= 64", dev);
  void* p = g_noalloc_addr[dev].load(std::memory_order_acquire);
  if (p == nullptr) {
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess || p == nullptr)
      return cuda_fail(e != cudaSuccess ? e : cudaErrorInvalidSymbol,
                       "head_scores_noalloc: cudaGetSymbolAddress(scratch)");
    g_noalloc_addr[dev].store(p, std::memory_order_release);
  }
  *out = p;
  return PROVIP_OK;
}

extern "C" int provip_head_scores_noalloc(const void* Q, const void* K, int B, int L_max, int H_q,
                                          int H_kv, int d_h, const int* head_list, int H_sel,
                                          const int* text_start, const int* text_len,
                                          const uint8_t* row_mask_or_null, int N_t_max,
                                          int vis_start, int N_v, const int* seq_len, int dtype,
                                          int algo, float* scores, void* stream) {
  NvtxRange nvtx_range("provip_head_scores_noalloc");
  const int ralgo = resolve_algo(algo, dtype);
  int rc = hs_validate(Q, K, B, L_max, H_q, H_kv, d_h, head_list, H_sel, text_start, text_len,
                       N_t_max, vis_start, N_v, seq_len, dtype, ralgo);
  if (rc) return rc;
  if (!scores) return fail(PROVIP_ERR_INVALID_ARG, "head_scores_noalloc: null scores");
  const size_t need = provip_head_scores_workspace_size(B, L_max, H_sel, N_t_max, N_v, ralgo, dtype);
  if (need > kNoAllocScratchBytes)
    return fail(PROVIP_ERR_UNSUPPORTED,
                "head_scores_noalloc: this shape needs %zu bytes of scratch, more than the %zu-byte "
                "static array; use provip_head_scores with a workspace",
                need, kNoAllocScratchBytes);
  void* scratch = nullptr;
  if ((rc = noalloc_scratch_addr(&scratch))) return rc;
  // Nothing in the scratch has to start at zero: every statistic and partial
  // sum is written by the first pass of this call before anything reads it.
  return provip_head_scores(Q, K, B, L_max, H_q, H_kv, d_h, head_list, H_sel, text_start, text_len,
                            row_mask_or_null, N_t_max, vis_start, N_v, seq_len, dtype, ralgo,
                            scores, scratch, kNoAllocScratchBytes, stream);
}
