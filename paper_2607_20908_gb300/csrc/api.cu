// api.cu -- the C ABI declared in include/spo.h: argument validation on the
// host, workspace carving, and the launch sequence of each call.
#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <mutex>
#include <vector>

#include "../../include/spo.h"
#include "internal.h"

namespace {

thread_local char g_err_text[512] = "";
thread_local int g_err_status = SPO_OK;

// Device error word written by bounded waits that expire.
__device__ int g_dev_error = 0;

spo_status fail(spo_status st, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err_text, sizeof(g_err_text), fmt, ap);
  va_end(ap);
  g_err_status = st;
  return st;
}

spo_status ok() {
  g_err_status = SPO_OK;
  g_err_text[0] = '\0';
  return SPO_OK;
}

spo_status cuda_fail(cudaError_t e, const char* what) {
  return fail(SPO_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

#define SPO_CUDA(call, what)                       \
  do {                                             \
    cudaError_t e_ = (call);                       \
    if (e_ != cudaSuccess) return cuda_fail(e_, what); \
  } while (0)

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }
long long round_up(long long x, long long m) { return (x + m - 1) / m * m; }

struct DevInfo {
  int dev = -1;
  int sms = 0;
  int major = 0;
  int* err = nullptr;
};

spo_status device_info(DevInfo* info) {
  int dev = 0;
  SPO_CUDA(cudaGetDevice(&dev), "cudaGetDevice");
  static DevInfo cache[64];
  static std::mutex cache_mu;  // calls may come from several host threads
  if (dev < 0 || dev >= 64) return fail(SPO_ERR_UNSUPPORTED, "device ordinal %d out of range", dev);
  std::lock_guard<std::mutex> lock(cache_mu);
  DevInfo& c = cache[dev];
  if (c.dev != dev) {
    DevInfo n;
    n.dev = dev;
    SPO_CUDA(cudaDeviceGetAttribute(&n.sms, cudaDevAttrMultiProcessorCount, dev), "attribute");
    SPO_CUDA(cudaDeviceGetAttribute(&n.major, cudaDevAttrComputeCapabilityMajor, dev), "attribute");
    if (n.major != 10)
      return fail(SPO_ERR_UNSUPPORTED, "device %d has compute capability %d.x; libspo needs sm_103a",
                  dev, n.major);
    SPO_CUDA(cudaGetSymbolAddress(reinterpret_cast<void**>(&n.err), g_dev_error),
             "cudaGetSymbolAddress(error word)");
    c = n;
  }
  *info = c;
  return SPO_OK;
}

// Host-side shape checks shared by the forward and backward.
// Sizes and temperature shared by every call on the logits.
spo_status check_dims(int64_t T, int64_t d, int64_t V, float inv_temp) {
  if (T < 1 || T > (1ll << 24)) return fail(SPO_ERR_SHAPE, "T = %lld outside [1, 2^24]", (long long)T);
  if (d < 64 || d > 65536 || d % 64 != 0)
    return fail(SPO_ERR_SHAPE, "d = %lld must be a multiple of 64 in [64, 65536]", (long long)d);
  if (V < 256 || V > (1ll << 24) || V % 8 != 0)
    return fail(SPO_ERR_SHAPE, "V = %lld must be a multiple of 8 in [256, 2^24]", (long long)V);
  if (!(inv_temp > 0.f) || !isfinite(inv_temp))
    return fail(SPO_ERR_INVALID_ARG, "inv_temp must be finite and > 0");
  return SPO_OK;
}

spo_status check_hwv(const void* H, const void* W, const int32_t* tgt, int64_t T, int64_t d,
                     int64_t V, float inv_temp) {
  if (!H || !W || !tgt) return fail(SPO_ERR_INVALID_ARG, "H, W and tgt must be non-NULL");
  spo_status st = check_dims(T, d, V, inv_temp);
  if (st != SPO_OK) return st;
  if (!aligned16(H) || !aligned16(W)) return fail(SPO_ERR_ALIGNMENT, "H and W must be 16-byte aligned");
  return SPO_OK;
}

// ------------------------------------------------------------ workspaces
struct FwdWs {
  int* idx;
  int* count;
  int* counters;  // tile counters of the dynamic schedule (4), then the throttle's progress slots
  int* scratch;
  int* tgt_c;
  float* ztgt;
  __nv_bfloat16* Hc;
  float* partials;
  long long T_pad;
  int nsplit;
  size_t bytes;
};

FwdWs carve_fwd(void* base, long long T, long long d, long long V) {
  FwdWs w{};
  w.T_pad = round_up(T, spo::kRowPad);
  w.nsplit = static_cast<int>((V + spo::BN - 1) / spo::BN);
  const int nb = spo::compact_blocks(T);
  char* p = static_cast<char*>(base);
  size_t off = 0;
  auto take = [&](size_t n) {
    char* q = p ? p + off : nullptr;
    off += align256(n);
    return q;
  };
  w.idx = reinterpret_cast<int*>(take(sizeof(int) * w.T_pad));
  w.count = reinterpret_cast<int*>(take(sizeof(int)));
  w.counters = reinterpret_cast<int*>(take(sizeof(int) * (4 + spo::kKsyncSlots)));
  w.scratch = reinterpret_cast<int*>(take(sizeof(int) * 2 * nb));
  w.tgt_c = reinterpret_cast<int*>(take(sizeof(int) * w.T_pad));
  w.ztgt = reinterpret_cast<float*>(take(sizeof(float) * w.T_pad));
  w.Hc = reinterpret_cast<__nv_bfloat16*>(take(sizeof(__nv_bfloat16) * w.T_pad * d));
  w.partials = reinterpret_cast<float*>(
      take(sizeof(float) * spo::kPartialBlock / 32 * w.nsplit * w.T_pad));
  w.bytes = off;
  return w;
}

constexpr long long kBwdChunkRows = 32768;  // G scratch rows per chunk (multiple of kRowPad)

struct BwdWs {
  int* idx;
  int* count;
  int* counters;  // tile counters of the dynamic schedule (4), then the throttle's progress slots
  int* scratch;
  int* tgt_c;
  float* lse_c;
  float* g_c;
  __nv_bfloat16* Hc;
  __nv_bfloat16* G;
  long long T_pad;
  long long chunk;
  size_t bytes;
};

BwdWs carve_bwd(void* base, long long T, long long d, long long V) {
  BwdWs w{};
  w.T_pad = round_up(T, spo::kRowPad);
  w.chunk = w.T_pad < kBwdChunkRows ? w.T_pad : kBwdChunkRows;
  const int nb = spo::compact_blocks(T);
  char* p = static_cast<char*>(base);
  size_t off = 0;
  auto take = [&](size_t n) {
    char* q = p ? p + off : nullptr;
    off += align256(n);
    return q;
  };
  w.idx = reinterpret_cast<int*>(take(sizeof(int) * w.T_pad));
  w.count = reinterpret_cast<int*>(take(sizeof(int)));
  w.counters = reinterpret_cast<int*>(take(sizeof(int) * (4 + spo::kKsyncSlots)));
  w.scratch = reinterpret_cast<int*>(take(sizeof(int) * 2 * nb));
  w.tgt_c = reinterpret_cast<int*>(take(sizeof(int) * w.T_pad));
  w.lse_c = reinterpret_cast<float*>(take(sizeof(float) * w.T_pad));
  w.g_c = reinterpret_cast<float*>(take(sizeof(float) * w.T_pad));
  w.Hc = reinterpret_cast<__nv_bfloat16*>(take(sizeof(__nv_bfloat16) * w.T_pad * d));
  w.G = reinterpret_cast<__nv_bfloat16*>(take(sizeof(__nv_bfloat16) * w.chunk * V));
  w.bytes = off;
  return w;
}

// ------------------------------------------------------------ tuning
// Host-global launch choices (spo_set_tuning): CTA-pair MMA on/off and the
// number of tile rows walked together by the raster.
int g_tune_pair = 1;
using spo::kDefaultGroupM;
using spo::kDefaultRaster;
int g_tune_group_m[4] = {kDefaultGroupM[0], kDefaultGroupM[1], kDefaultGroupM[2], kDefaultGroupM[3]};
int g_tune_raster[4] = {kDefaultRaster[0], kDefaultRaster[1], kDefaultRaster[2], kDefaultRaster[3]};
// Bit k set: GEMM kind k takes its tiles from an atomic counter (dynamic
// schedule) instead of the static round robin, so the tiles in flight stay a
// contiguous window of the raster however the CTA pairs drift.  Default: all.
int g_tune_dynamic_mask = spo::kDefaultDynamicMask;
// dW = G^T H runs as passes over at most this many token rows (0: one pass
// per chunk): smaller operand slabs keep a wave's working set inside L2.
int g_tune_dw_split = spo::kDefaultDwSplitRows;
// k-progress throttle per GEMM kind: window in k-blocks (0 = off), and the
// k-blocks between two checks.
int g_tune_ksync[4] = {spo::kDefaultKsync[0], spo::kDefaultKsync[1], spo::kDefaultKsync[2],
                       spo::kDefaultKsync[3]};
int g_tune_ksync_epoch = spo::kDefaultKsyncEpoch;
// dH with 256 x 512 tiles per CTA pair (pair mode only): 0 never, 1 for
// reductions of at least spo::kDhWideMinK vocabulary rows, 2 always.
int g_tune_dh_wide = spo::kDefaultDhWide;
// The logits GEMMs with 256 x 512 tiles: bit 0 the forward in every call, bit 1
// the recompute, bit 2 the forward inside spo_grpo_step.
int g_tune_logits_wide = spo::kDefaultLogitsWide;

// ------------------------------------------------------------ tracing
// When enabled, a start/stop CUDA event pair is recorded on the launch stream
// around every tensor-core GEMM launch; spo_trace_read returns the durations.
struct TraceRec {
  int kind;
  int dev;
  cudaEvent_t start, stop;
};
std::mutex g_trace_mu;
bool g_trace_on = false;
std::vector<TraceRec> g_trace;
std::vector<TraceRec> g_trace_pool;  // event pairs ready for reuse

// Runs `launch` (which enqueues one or more kernels on s and returns the
// launch status), bracketed by a recorded event pair when tracing is on.
template <class F>
spo_status traced(int kind, cudaStream_t s, const char* what, F&& launch) {
  int dev = 0;
  TraceRec rec{kind, 0, nullptr, nullptr};
  bool tracing;
  {
    std::lock_guard<std::mutex> lk(g_trace_mu);
    tracing = g_trace_on;
  }
  if (tracing) {
    SPO_CUDA(cudaGetDevice(&dev), "cudaGetDevice");
    rec.dev = dev;
    std::lock_guard<std::mutex> lk(g_trace_mu);
    for (size_t i = 0; i < g_trace_pool.size(); ++i) {
      if (g_trace_pool[i].dev == dev) {
        rec.start = g_trace_pool[i].start;
        rec.stop = g_trace_pool[i].stop;
        g_trace_pool.erase(g_trace_pool.begin() + i);
        break;
      }
    }
  }
  if (tracing && !rec.start) {
    SPO_CUDA(cudaEventCreate(&rec.start), "cudaEventCreate");
    SPO_CUDA(cudaEventCreate(&rec.stop), "cudaEventCreate");
  }
  if (tracing) SPO_CUDA(cudaEventRecord(rec.start, s), "cudaEventRecord");
  SPO_CUDA(launch(), what);
  if (tracing) {
    SPO_CUDA(cudaEventRecord(rec.stop, s), "cudaEventRecord");
    std::lock_guard<std::mutex> lk(g_trace_mu);
    g_trace.push_back(rec);
  }
  return SPO_OK;
}

// Trace kinds (spo_trace_read): the four tensor-core GEMMs keep their EPI ids.
enum TraceKind : int {
  kTraceLseCombine = 4,
  kTraceSelectGatherFwd = 5,
  kTraceSelectGatherBwd = 6,
  kTracePolicyLoss = 7,
  kTraceAdvantages = 8,
  kTraceTokenSelect = 9,
  kTraceReward = 10,
  kTraceRanker = 11,
  kTraceMergeSlices = 12,
  kTraceFormG = 13,
};

// counters: the workspace's four tile counters (the one of this kind is
// zeroed on the stream and used when the kind's dynamic-schedule bit is set).
// Launches GEMM epilogue `epi`.  Its schedule, tile counter and trace kind are
// those of the product it computes (0 logits, 1 recompute, 2 dH, 3 dW): the
// kept-exponential forward is the logits product.
// in_step: the launch belongs to spo_grpo_step (the forward then takes wide
// tiles under bit 2 of the logits setting).
spo_status traced_gemm(int epi, bool a_mn, bool b_mn, const CUtensorMap& ta, const CUtensorMap& tb,
                       const CUtensorMap& tc, const spo::GemmArgs& args_in, int grid, cudaStream_t s,
                       int* counters, bool in_step = false) {
  const int kind = epi == spo::EPI_LSE_KEEP ? spo::EPI_LSE : epi;
  if (kind < 0 || kind > 3) return fail(SPO_ERR_INVALID_ARG, "GEMM kind %d", epi);
  spo::GemmArgs args = args_in;
  args.group_m = g_tune_group_m[kind];
  args.raster = g_tune_raster[kind];
  args.tile_counter = nullptr;
  if (counters && ((g_tune_dynamic_mask >> kind) & 1)) {
    args.tile_counter = counters + kind;
    SPO_CUDA(cudaMemsetAsync(args.tile_counter, 0, sizeof(int), s), "memset tile counter");
  }
  args.kprog = nullptr;
  if (counters && g_tune_ksync[kind] > 0) {
    args.kprog = counters + 4;
    args.ksync_window = g_tune_ksync[kind];
    args.ksync_epoch = g_tune_ksync_epoch;
    SPO_CUDA(cudaMemsetAsync(args.kprog, 0, sizeof(int) * spo::kKsyncSlots, s),
             "memset progress slots");
  }
  const bool wide = (kind == spo::EPI_DH &&
                     (g_tune_dh_wide == 2 || (g_tune_dh_wide == 1 && args.k_static >= spo::kDhWideMinK))) ||
                    (epi == spo::EPI_LSE && ((g_tune_logits_wide & 1) || (in_step && (g_tune_logits_wide & 4)))) ||
                    (epi == spo::EPI_GRAD && (g_tune_logits_wide & 2));
  return traced(kind, s, "gemm launch", [&] {
    return spo::launch_gemm(epi, a_mn, b_mn, g_tune_pair != 0, ta, tb, tc, args, grid, s, wide);
  });
}

spo::GemmArgs base_args(const DevInfo& di) {
  spo::GemmArgs a;
  memset(&a, 0, sizeof(a));
  a.group_m = 1;  // set per kind at launch
  a.scale = 1.f;
  a.err = di.err;
  return a;
}

// Persistent grid: one CTA per SM (pairs in pair mode), never more than tiles;
// `reserve` SMs are left free for kernels that run alongside (a collective).
int grid_for(const DevInfo& di, long long max_m, long long n, int reserve = 0) {
  const bool pair = g_tune_pair != 0;
  const long long tm = spo::gemm_tile_m(pair);
  const long long tiles = ((max_m + tm - 1) / tm) * ((n + spo::BN - 1) / spo::BN);
  const int sms = di.sms - reserve > 2 ? di.sms - reserve : 2;
  const long long units = pair ? sms / 2 : sms;
  long long g = tiles < units ? tiles : units;
  if (g < 1) g = 1;
  return static_cast<int>(pair ? 2 * g : g);
}

uint32_t b_box_rows() { return static_cast<uint32_t>(spo::gemm_b_box_rows(g_tune_pair != 0)); }

// a1 selection + gather, a2 and a3 over vocabulary rows [v_offset, v_offset + V)
// (W points at row v_offset).  rec == NULL: logp / entropy / lse; otherwise the
// slice records.  Arguments are validated by the caller.
spo_status logprobs_impl(const void* H, const void* W, const int32_t* tgt, const uint8_t* mask,
                         int64_t T, int64_t d, int64_t V, int64_t v_offset, float inv_temp,
                         float* logp, float* entropy, float* lse, float* rec, void* ws,
                         cudaStream_t s, void* keep = nullptr, bool in_step = false) {
  spo_status st;
  DevInfo di;
  if ((st = device_info(&di)) != SPO_OK) return st;
  const FwdWs w = carve_fwd(ws, T, d, V);

  // a1 (row selection) + gather of the kept rows into a dense bf16 block
  st = traced(kTraceSelectGatherFwd, s, "compact/gather", [&] {
    cudaError_t e = spo::launch_compact(0, mask, tgt, nullptr, T, w.scratch, w.idx, w.count, s);
    if (e != cudaSuccess) return e;
    return spo::launch_gather(static_cast<const __nv_bfloat16*>(H), static_cast<int>(d), w.idx,
                              w.count, static_cast<int>(w.T_pad), w.Hc, tgt, w.tgt_c, v_offset, V,
                              nullptr, nullptr, nullptr, nullptr, s);
  });
  if (st != SPO_OK) return st;
  // a2: logits tile by tile + online logsumexp partials
  CUtensorMap ta, tb;
  SPO_CUDA(spo::make_tmap_bf16(&ta, w.Hc, d, w.T_pad, d * 2, spo::BK, spo::BM), "tensor map H");
  SPO_CUDA(spo::make_tmap_bf16(&tb, W, d, V, d * 2, spo::BK, b_box_rows()), "tensor map W");
  spo::GemmArgs a = base_args(di);
  a.m_count = w.count;
  a.m_offset = 0;
  a.m_cap = static_cast<int>(w.T_pad);
  a.n = static_cast<int>(V);
  a.k_static = static_cast<int>(d);
  a.scale = inv_temp;
  a.tgt = w.tgt_c;
  a.partials = w.partials;
  a.nsplit = w.nsplit;
  a.ztgt = w.ztgt;
  if (keep) {  // also keep E = 2^(t - tile max) in bf16 for spo_policy_loss_bwd_kept
    CUtensorMap tk;
    SPO_CUDA(spo::make_tmap_bf16(&tk, keep, V, w.T_pad, V * 2, 64, spo::kStoreBoxRows),
             "tensor map E (store)");
    st = traced_gemm(spo::EPI_LSE_KEEP, false, false, ta, tb, tk, a, grid_for(di, w.T_pad, V), s,
                     w.counters);
  } else {
    st = traced_gemm(spo::EPI_LSE, false, false, ta, tb, ta, a, grid_for(di, w.T_pad, V), s,
                     w.counters, in_step);
  }
  if (st != SPO_OK) return st;
  // a3: split-vocab combine, scattered back to token positions (skipped tokens read 0)
  if (rec) {
    SPO_CUDA(cudaMemsetAsync(rec, 0, sizeof(float) * 4 * T, s), "memset rec");
  } else {
    SPO_CUDA(cudaMemsetAsync(logp, 0, sizeof(float) * T, s), "memset logp");
    if (entropy) SPO_CUDA(cudaMemsetAsync(entropy, 0, sizeof(float) * T, s), "memset entropy");
    if (lse) SPO_CUDA(cudaMemsetAsync(lse, 0, sizeof(float) * T, s), "memset lse");
  }
  st = traced(kTraceLseCombine, s, "combine launch", [&] {
    return spo::launch_lse_combine(w.partials, w.nsplit, w.ztgt, w.idx, w.count,
                                   static_cast<int>(w.T_pad), logp, entropy, lse, w.tgt_c,
                                   reinterpret_cast<float4*>(rec), s);
  });
  return st == SPO_OK ? ok() : st;
}

spo_status check_fwd_ws(int64_t T, int64_t d, int64_t V, const void* ws, size_t ws_bytes) {
  const FwdWs need = carve_fwd(nullptr, T, d, V);
  if (!ws || ws_bytes < need.bytes)
    return fail(SPO_ERR_WORKSPACE, "workspace needs %zu bytes, got %zu", need.bytes, ws_bytes);
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0)
    return fail(SPO_ERR_ALIGNMENT, "workspace must be 256-byte aligned");
  return SPO_OK;
}

// Hooks of a backward: dW computed in contiguous vocabulary blocks, with a
// caller's event recorded on the stream as soon as each block (and, before
// that, every dH row) is final, so a collective on another stream can start
// on it while the remaining GEMMs run.  reserve_sms: the GEMMs that follow the
// first event leave that many SMs free for such a collective.
struct BwdHooks {
  int n_dw_blocks = 1;
  int reserve_sms = 0;
  const cudaEvent_t* dw_events = nullptr;  // [n_dw_blocks] entries, each may be NULL
  cudaEvent_t dh_event = nullptr;
};

// First row of vocabulary block k of n (block starts are multiples of 256
// rows, one GEMM tile; the last block ends at V; blocks may be empty).
long long dw_block_start(long long V, int n, int k) {
  if (k >= n) return V;
  return (V * k / n) / 256 * 256;
}

spo_status record_hook_events(const BwdHooks* hooks, cudaStream_t s) {
  if (!hooks) return SPO_OK;
  if (hooks->dh_event) SPO_CUDA(cudaEventRecord(hooks->dh_event, s), "record dH event");
  if (hooks->dw_events)
    for (int k = 0; k < hooks->n_dw_blocks; ++k)
      if (hooks->dw_events[k]) SPO_CUDA(cudaEventRecord(hooks->dw_events[k], s), "record dW event");
  return SPO_OK;
}

// a7 + a8 over a block of compacted rows [r0, r0 + rows): G holds them from
// its first row (bf16, pitch ldG elements), Hc0 the same rows of the
// compacted H, idx their token positions.  dH rows are scattered to token
// rows (bf16, or fp32 with dH_f32); dW (+)= G^T Hc in passes of at most
// g_tune_dw_split rows, the first pass adding into dW only when
// accumulate_first.  With hooks, dW runs block by block over the vocabulary
// and the hook events are recorded as dH and each dW block become final
// (the per-element reduction order is the same as without them).
spo_status dh_dw_block(const DevInfo& di, const void* W, int64_t d, int64_t V,
                       const __nv_bfloat16* G, long long ldG, long long rows,
                       const __nv_bfloat16* Hc0, long long r0, const int* count, const int* idx,
                       void* dH, bool dH_f32, float* dW, bool accumulate_first, int* counters,
                       cudaStream_t s, const BwdHooks* hooks = nullptr) {
  spo_status st;
  CUtensorMap tG_k, tW_mn;
  SPO_CUDA(spo::make_tmap_bf16(&tG_k, G, V, rows, ldG * 2, spo::BK, spo::BM), "tensor map G");
  SPO_CUDA(spo::make_tmap_bf16(&tW_mn, W, d, V, d * 2, 64, spo::BK), "tensor map W (MN)");
  // a7: dH rows = G W, scattered to token rows
  if (dH) {
    spo::GemmArgs b = base_args(di);
    b.m_count = count;
    b.m_offset = static_cast<int>(r0);
    b.m_cap = static_cast<int>(rows);
    b.n = static_cast<int>(d);
    b.k_static = static_cast<int>(V);
    b.row_idx = idx + r0;
    if (dH_f32)
      b.out_f32 = static_cast<float*>(dH);
    else
      b.out_bf16 = static_cast<__nv_bfloat16*>(dH);
    b.ld_out = d;
    if ((st = traced_gemm(spo::EPI_DH, false, true, tG_k, tW_mn, tG_k, b, grid_for(di, rows, d), s,
                          counters)) != SPO_OK)
      return st;
  }
  if (hooks && hooks->dh_event) SPO_CUDA(cudaEventRecord(hooks->dh_event, s), "record dH event");
  // a8: dW (+)= G^T Hc over these rows, in passes of at most g_tune_dw_split
  // rows (later passes reduce-add into dW), vocabulary block by block
  const int nb = hooks && hooks->n_dw_blocks > 1 ? hooks->n_dw_blocks : 1;
  const int reserve = hooks ? hooks->reserve_sms : 0;
  for (int kb = 0; kb < nb; ++kb) {
    const long long v0 = dw_block_start(V, nb, kb), v1 = dw_block_start(V, nb, kb + 1);
    if (dW && v1 > v0) {
      CUtensorMap tdW;
      SPO_CUDA(spo::make_tmap_f32(&tdW, dW + v0 * d, d, v1 - v0, d * 4, 32, spo::kStoreBoxRows),
               "tensor map dW");
      const long long split = g_tune_dw_split > 0 ? g_tune_dw_split : rows;
      for (long long q0 = 0; q0 < rows; q0 += split) {
        const long long qrows = (rows - q0) < split ? (rows - q0) : split;
        CUtensorMap tGq, tHq;
        SPO_CUDA(spo::make_tmap_bf16(&tGq, G + q0 * ldG + v0, v1 - v0, qrows, ldG * 2, 64, spo::BK),
                 "tensor map G (MN)");
        SPO_CUDA(spo::make_tmap_bf16(&tHq, Hc0 + q0 * d, d, qrows, d * 2, 64, spo::BK),
                 "tensor map Hc (MN)");
        spo::GemmArgs b = base_args(di);
        b.m_static = static_cast<int>(v1 - v0);
        b.n = static_cast<int>(d);
        b.k_count = count;
        b.k_offset = static_cast<int>(r0 + q0);
        b.k_cap = static_cast<int>(qrows);
        b.out_f32 = dW + v0 * d;
        b.ld_out = d;
        b.accumulate = (q0 == 0 && !accumulate_first) ? 0 : 1;
        if ((st = traced_gemm(spo::EPI_DW, true, true, tGq, tHq, tdW, b,
                              grid_for(di, v1 - v0, d, reserve), s, counters)) != SPO_OK)
          return st;
      }
    }
    if (hooks && hooks->dw_events && kb < hooks->n_dw_blocks && hooks->dw_events[kb])
      SPO_CUDA(cudaEventRecord(hooks->dw_events[kb], s), "record dW event");
  }
  if (hooks && hooks->dw_events)  // blocks beyond the ones run (n_dw_blocks <= 1 uses one)
    for (int kb = nb; kb < hooks->n_dw_blocks; ++kb)
      if (hooks->dw_events[kb]) SPO_CUDA(cudaEventRecord(hooks->dw_events[kb], s), "record dW event");
  return SPO_OK;
}

// The rows a backward runs over: a compaction (Hc, idx, count, compacted
// targets) and the per-row lse and g, either compacted (lse[r], g[r]) or at
// token positions (lse[idx[r]], g[idx[r]]: by_token).
struct BwdRows {
  const __nv_bfloat16* Hc;
  const int* idx;
  const int* count;
  const int* tgt_c;
  const float* lse;
  const float* g;
  bool by_token;
  long long T_pad;
};

// a6-a8 over vocabulary rows [0, V) of W (a slice's rows when W points into a
// larger head) for the given rows, in chunks of at most `chunk` rows of G.
spo_status bwd_core(const DevInfo& di, const void* W, int64_t d, int64_t V, float inv_temp,
                    const BwdRows& r, __nv_bfloat16* G, long long chunk, void* dH, bool dH_f32,
                    float* dW, int accumulate_dW, int* counters, const BwdHooks* hooks,
                    cudaStream_t s) {
  spo_status st;
  CUtensorMap tW_k, tG_store;
  SPO_CUDA(spo::make_tmap_bf16(&tW_k, W, d, V, d * 2, spo::BK, b_box_rows()), "tensor map W");
  SPO_CUDA(spo::make_tmap_bf16(&tG_store, G, V, chunk, V * 2, 64, spo::kStoreBoxRows),
           "tensor map G (store)");
  const long long n_chunks = (r.T_pad + chunk - 1) / chunk;
  for (long long c = 0; c < n_chunks; ++c) {
    const long long r0 = c * chunk;
    const long long rows = (r.T_pad - r0) < chunk ? (r.T_pad - r0) : chunk;
    const __nv_bfloat16* Hc0 = r.Hc + r0 * d;
    CUtensorMap tH_k;
    SPO_CUDA(spo::make_tmap_bf16(&tH_k, Hc0, d, rows, d * 2, spo::BK, spo::BM), "tensor map Hc");

    // a6: G = inv_temp * g * (onehot - softmax), logits recomputed
    spo::GemmArgs a = base_args(di);
    a.m_count = r.count;
    a.m_offset = static_cast<int>(r0);
    a.m_cap = static_cast<int>(chunk);
    a.n = static_cast<int>(V);
    a.k_static = static_cast<int>(d);
    a.scale = inv_temp;
    a.tgt = r.tgt_c + r0;
    if (r.by_token) {
      a.lse = r.lse;
      a.gvec = r.g;
      a.vec_idx = r.idx + r0;
    } else {
      a.lse = r.lse + r0;
      a.gvec = r.g + r0;
    }
    a.G = G;
    a.ldG = V;
    if ((st = traced_gemm(spo::EPI_GRAD, false, false, tH_k, tW_k, tG_store, a,
                          grid_for(di, rows, V), s, counters)) != SPO_OK)
      return st;
    if ((st = dh_dw_block(di, W, d, V, G, V, rows, Hc0, r0, r.count, r.idx, dH, dH_f32, dW,
                          c > 0 || accumulate_dW, counters, s,
                          c == n_chunks - 1 ? hooks : nullptr)) != SPO_OK)
      return st;
  }
  return SPO_OK;
}

// a6-a8 over vocabulary rows [v_offset, v_offset + V) (W points at row
// v_offset); dH is bf16, or fp32 with dH_f32.  Arguments are validated by the caller.
spo_status bwd_impl(const void* H, const void* W, const int32_t* tgt, const float* lse,
                    const float* g, int64_t T, int64_t d, int64_t V, int64_t v_offset,
                    float inv_temp, void* dH, bool dH_f32, float* dW, int accumulate_dW, void* ws,
                    cudaStream_t s, const BwdHooks* hooks = nullptr) {
  spo_status st;
  DevInfo di;
  if ((st = device_info(&di)) != SPO_OK) return st;
  const BwdWs w = carve_bwd(ws, T, d, V);
  if (!dH && !dW) return (st = record_hook_events(hooks, s)) == SPO_OK ? ok() : st;

  // rows with g != 0 are the only ones with a non-zero gradient row
  st = traced(kTraceSelectGatherBwd, s, "compact/gather", [&] {
    cudaError_t e = spo::launch_compact(1, nullptr, nullptr, g, T, w.scratch, w.idx, w.count, s);
    if (e != cudaSuccess) return e;
    return spo::launch_gather(static_cast<const __nv_bfloat16*>(H), static_cast<int>(d), w.idx,
                              w.count, static_cast<int>(w.T_pad), w.Hc, tgt, w.tgt_c, v_offset, V,
                              lse, w.lse_c, g, w.g_c, s);
  });
  if (st != SPO_OK) return st;
  // rows the compaction skips get zero; the dH GEMM writes all the others
  if (dH)
    SPO_CUDA(spo::launch_zero_skipped_rows(g, T, static_cast<int>((dH_f32 ? 4 : 2) * d), dH, s),
             "zero skipped dH rows");
  const BwdRows rows{w.Hc, w.idx, w.count, w.tgt_c, w.lse_c, w.g_c, false, w.T_pad};
  st = bwd_core(di, W, d, V, inv_temp, rows, w.G, w.chunk, dH, dH_f32, dW, accumulate_dW,
                w.counters, hooks, s);
  return st == SPO_OK ? ok() : st;
}


spo_status check_bwd_args(const void* H, const void* W, const int32_t* tgt, const float* lse,
                          const float* g, int64_t T, int64_t d, int64_t V, float inv_temp,
                          const void* dH, const float* dW, const void* ws, size_t ws_bytes) {
  spo_status st = check_hwv(H, W, tgt, T, d, V, inv_temp);
  if (st != SPO_OK) return st;
  if (!lse || !g) return fail(SPO_ERR_INVALID_ARG, "lse and g must be non-NULL");
  if (dH && !aligned16(dH)) return fail(SPO_ERR_ALIGNMENT, "dH must be 16-byte aligned");
  if (dW && !aligned16(dW)) return fail(SPO_ERR_ALIGNMENT, "dW must be 16-byte aligned");
  const BwdWs need = carve_bwd(nullptr, T, d, V);
  if (!ws || ws_bytes < need.bytes)
    return fail(SPO_ERR_WORKSPACE, "workspace needs %zu bytes, got %zu", need.bytes, ws_bytes);
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0)
    return fail(SPO_ERR_ALIGNMENT, "workspace must be 256-byte aligned");
  return SPO_OK;
}

spo_status check_adv_args(const float* rewards, const int32_t* group_id, int32_t n_seq,
                          int32_t n_groups, int std_mode, float eps, const float* adv) {
  if (!rewards || !group_id || !adv)
    return fail(SPO_ERR_INVALID_ARG, "rewards, group_id and adv must be non-NULL");
  if (n_seq < 1 || n_groups < 1 || n_seq > (1 << 26) || n_groups > (1 << 26))
    return fail(SPO_ERR_SHAPE, "n_seq = %d, n_groups = %d out of range", n_seq, n_groups);
  if (std_mode != SPO_STD_UNBIASED && std_mode != SPO_STD_POPULATION)
    return fail(SPO_ERR_INVALID_ARG, "std_mode %d unknown", std_mode);
  if (!(eps >= 0.f) || !isfinite(eps)) return fail(SPO_ERR_INVALID_ARG, "eps must be finite and >= 0");
  return SPO_OK;
}

// Workspace of spo_grpo_step: the forward's region first (its compaction,
// gathered rows and targets serve the backward too), then the per-token and
// per-sequence vectors the caller did not ask for, the advantage and loss
// scratch, and one bf16 G chunk.
struct StepWs {
  uint8_t* loss_mask;
  int* n_tok;
  float* logp;
  float* lse;
  float* g;
  float* adv;
  void* adv_ws;
  void* loss_ws;
  __nv_bfloat16* G;
  long long chunk;
  size_t bytes;
};

StepWs carve_step(void* base, long long T, long long d, long long V, int n_seq, int n_groups) {
  StepWs w{};
  char* p = static_cast<char*>(base);
  size_t off = carve_fwd(nullptr, T, d, V).bytes;
  auto take = [&](size_t n) {
    char* q = p ? p + off : nullptr;
    off += align256(n);
    return q;
  };
  const long long T_pad = round_up(T, spo::kRowPad);
  w.loss_mask = reinterpret_cast<uint8_t*>(take(static_cast<size_t>(T)));
  w.n_tok = reinterpret_cast<int*>(take(sizeof(int) * static_cast<size_t>(n_seq)));
  w.logp = reinterpret_cast<float*>(take(sizeof(float) * T));
  w.lse = reinterpret_cast<float*>(take(sizeof(float) * T));
  w.g = reinterpret_cast<float*>(take(sizeof(float) * T));
  w.adv = reinterpret_cast<float*>(take(sizeof(float) * static_cast<size_t>(n_seq)));
  w.adv_ws = take(spo::adv_ws_bytes(n_groups));
  w.loss_ws = take(spo::loss_ws_bytes(n_seq, n_groups));
  w.chunk = T_pad < kBwdChunkRows ? T_pad : kBwdChunkRows;
  w.G = reinterpret_cast<__nv_bfloat16*>(take(sizeof(__nv_bfloat16) * w.chunk * V));
  w.bytes = off;
  return w;
}

// Public hooks -> internal form (events copied), checked against the device.
spo_status convert_hooks(const spo_bwd_hooks* h, const DevInfo& di, BwdHooks* out,
                         std::vector<cudaEvent_t>* events) {
  *out = BwdHooks{};
  if (!h) return SPO_OK;
  if (h->n_dw_blocks < 1 || h->n_dw_blocks > 4096)
    return fail(SPO_ERR_INVALID_ARG, "n_dw_blocks = %d outside [1, 4096]", h->n_dw_blocks);
  if (h->reserve_sms < 0 || h->reserve_sms > di.sms - 2)
    return fail(SPO_ERR_INVALID_ARG, "reserve_sms = %d outside [0, %d]", h->reserve_sms, di.sms - 2);
  out->n_dw_blocks = h->n_dw_blocks;
  out->reserve_sms = h->reserve_sms;
  out->dh_event = static_cast<cudaEvent_t>(h->dh_event);
  if (h->dw_block_events) {
    events->assign(static_cast<size_t>(h->n_dw_blocks), nullptr);
    for (int k = 0; k < h->n_dw_blocks; ++k)
      (*events)[k] = static_cast<cudaEvent_t>(h->dw_block_events[k]);
    out->dw_events = events->data();
  }
  return SPO_OK;
}

spo_status check_loss_scalars(int32_t n_seq, int32_t n_groups, int agg, float clip_eps,
                              float kl_beta) {
  if (n_seq < 1 || n_groups < 1 || n_seq > (1 << 24) || n_groups > (1 << 24))
    return fail(SPO_ERR_SHAPE, "n_seq = %d, n_groups = %d out of range", n_seq, n_groups);
  if (agg != SPO_AGG_SEQ_GROUP && agg != SPO_AGG_TOKEN)
    return fail(SPO_ERR_INVALID_ARG, "agg %d unknown", agg);
  if (!(clip_eps >= 0.f && clip_eps < 1.f)) return fail(SPO_ERR_INVALID_ARG, "clip_eps must be in [0, 1)");
  if (!isfinite(kl_beta)) return fail(SPO_ERR_INVALID_ARG, "kl_beta must be finite");
  return SPO_OK;
}

}  // namespace

extern "C" {

SPO_API int spo_version(void) { return (0 << 16) | 1; }

SPO_API const char* spo_status_string(int status) {
  switch (status) {
    case SPO_OK: return "SPO_OK";
    case SPO_ERR_INVALID_ARG: return "SPO_ERR_INVALID_ARG";
    case SPO_ERR_SHAPE: return "SPO_ERR_SHAPE";
    case SPO_ERR_ALIGNMENT: return "SPO_ERR_ALIGNMENT";
    case SPO_ERR_WORKSPACE: return "SPO_ERR_WORKSPACE";
    case SPO_ERR_UNSUPPORTED: return "SPO_ERR_UNSUPPORTED";
    case SPO_ERR_CUDA: return "SPO_ERR_CUDA";
    case SPO_ERR_TIMEOUT: return "SPO_ERR_TIMEOUT";
    default: return "SPO_ERR_UNKNOWN";
  }
}

SPO_API int spo_last_error(char* buf, size_t n) {
  if (buf && n) {
    strncpy(buf, g_err_text, n - 1);
    buf[n - 1] = '\0';
  }
  return g_err_status;
}

SPO_API spo_status spo_device_error(int* code, void* stream) {
  if (!code) return fail(SPO_ERR_INVALID_ARG, "code must be non-NULL");
  DevInfo di;
  spo_status st = device_info(&di);
  if (st != SPO_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int v = 0;
  SPO_CUDA(cudaMemcpyAsync(&v, di.err, sizeof(int), cudaMemcpyDeviceToHost, s), "read error word");
  SPO_CUDA(cudaMemsetAsync(di.err, 0, sizeof(int), s), "clear error word");
  SPO_CUDA(cudaStreamSynchronize(s), "cudaStreamSynchronize");
  *code = v;
  if (v != 0) return fail(SPO_ERR_TIMEOUT, "device wait expired (code 0x%x)", v);
  return ok();
}

SPO_API spo_status spo_selftest_bounded_wait(void* stream) {
  DevInfo di;
  spo_status st = device_info(&di);
  if (st != SPO_OK) return st;
  SPO_CUDA(spo::launch_bounded_wait_selftest(di.err, static_cast<cudaStream_t>(stream)),
           "self-test launch");
  return ok();
}

SPO_API spo_status spo_token_select(const int32_t* cu_seqlens, const uint8_t* mask,
                                    const int32_t* tgt, int32_t n_seq, int64_t T, int32_t window,
                                    uint8_t* loss_mask, int32_t* n_tok, void* stream) {
  if (!cu_seqlens || !tgt || !loss_mask || !n_tok)
    return fail(SPO_ERR_INVALID_ARG, "cu_seqlens, tgt, loss_mask and n_tok must be non-NULL");
  if (n_seq < 1 || n_seq > (1 << 24)) return fail(SPO_ERR_SHAPE, "n_seq = %d outside [1, 2^24]", n_seq);
  if (T < 1 || T > (1ll << 30)) return fail(SPO_ERR_SHAPE, "T = %lld outside [1, 2^30]", (long long)T);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  spo_status st = traced(kTraceTokenSelect, s, "token_select launch", [&] {
    return spo::launch_token_select(cu_seqlens, mask, tgt, n_seq, window, loss_mask, n_tok, s);
  });
  return st == SPO_OK ? ok() : st;
}

SPO_API spo_status spo_logprobs_workspace_size(int64_t T, int64_t d, int64_t V, size_t* bytes) {
  if (!bytes) return fail(SPO_ERR_INVALID_ARG, "bytes must be non-NULL");
  if (T < 1 || d < 1 || V < 1) return fail(SPO_ERR_SHAPE, "sizes must be positive");
  *bytes = carve_fwd(nullptr, T, d, V).bytes;
  return ok();
}

SPO_API spo_status spo_logprobs_fwd(const void* H, const void* W, const int32_t* tgt,
                                    const uint8_t* mask, int64_t T, int64_t d, int64_t V,
                                    float inv_temp, float* logp, float* entropy, float* lse,
                                    void* ws, size_t ws_bytes, void* stream) {
  spo_status st = check_hwv(H, W, tgt, T, d, V, inv_temp);
  if (st != SPO_OK) return st;
  if (!logp) return fail(SPO_ERR_INVALID_ARG, "logp must be non-NULL");
  if ((st = check_fwd_ws(T, d, V, ws, ws_bytes)) != SPO_OK) return st;
  return logprobs_impl(H, W, tgt, mask, T, d, V, 0, inv_temp, logp, entropy, lse, nullptr, ws,
                       static_cast<cudaStream_t>(stream));
}

SPO_API spo_status spo_logprobs_fwd_slice(const void* H, const void* W_slice, const int32_t* tgt,
                                          const uint8_t* mask, int64_t T, int64_t d,
                                          int64_t V_slice, int64_t v_offset, float inv_temp,
                                          float* rec, void* ws, size_t ws_bytes, void* stream) {
  spo_status st = check_hwv(H, W_slice, tgt, T, d, V_slice, inv_temp);
  if (st != SPO_OK) return st;
  if (v_offset < 0 || v_offset > (1ll << 31) - 1)
    return fail(SPO_ERR_SHAPE, "v_offset = %lld outside [0, 2^31)", (long long)v_offset);
  if (!rec) return fail(SPO_ERR_INVALID_ARG, "rec must be non-NULL");
  if (!aligned16(rec)) return fail(SPO_ERR_ALIGNMENT, "rec must be 16-byte aligned");
  if ((st = check_fwd_ws(T, d, V_slice, ws, ws_bytes)) != SPO_OK) return st;
  return logprobs_impl(H, W_slice, tgt, mask, T, d, V_slice, v_offset, inv_temp, nullptr, nullptr,
                       nullptr, rec, ws, static_cast<cudaStream_t>(stream));
}

SPO_API spo_status spo_logprobs_merge_slices(const float* rec, int32_t n_slices, int64_t T,
                                             float* logp, float* entropy, float* lse,
                                             void* stream) {
  if (!rec || !logp) return fail(SPO_ERR_INVALID_ARG, "rec and logp must be non-NULL");
  if (!aligned16(rec)) return fail(SPO_ERR_ALIGNMENT, "rec must be 16-byte aligned");
  if (n_slices < 1 || n_slices > 1024)
    return fail(SPO_ERR_SHAPE, "n_slices = %d outside [1, 1024]", n_slices);
  if (T < 1 || T > (1ll << 24)) return fail(SPO_ERR_SHAPE, "T = %lld outside [1, 2^24]", (long long)T);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  spo_status st = traced(kTraceMergeSlices, s, "merge launch", [&] {
    return spo::launch_merge_slices(reinterpret_cast<const float4*>(rec), n_slices, T, logp,
                                    entropy, lse, s);
  });
  return st == SPO_OK ? ok() : st;
}

SPO_API spo_status spo_reward_compose(const uint8_t* compiled, const float* pass_rate,
                                      const float* speedup, const float* cv, const float* r_struct,
                                      int32_t n, const spo_reward_params* params, float* rewards,
                                      void* stream) {
  if (!compiled || !pass_rate || !speedup || !cv || !rewards)
    return fail(SPO_ERR_INVALID_ARG, "compiled, pass_rate, speedup, cv and rewards must be non-NULL");
  if (n < 1 || n > (1 << 30)) return fail(SPO_ERR_SHAPE, "n = %d out of range", n);
  spo::RewardParams q{3.0f, 2.0f, 1.0f, 0.5f, -0.5f, 4.0f};  // the paper's constants
  if (params) {
    q = spo::RewardParams{params->alpha_comp, params->alpha_wrong, params->alpha_speed,
                          params->alpha_cv, params->s_min, params->s_max};
    const float v[6] = {q.alpha_comp, q.alpha_wrong, q.alpha_speed, q.alpha_cv, q.s_min, q.s_max};
    for (float x : v)
      if (!isfinite(x)) return fail(SPO_ERR_INVALID_ARG, "reward parameters must be finite");
    if (q.s_min > q.s_max) return fail(SPO_ERR_INVALID_ARG, "s_min must not exceed s_max");
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  spo_status st = traced(kTraceReward, s, "reward launch", [&] {
    return spo::launch_reward_compose(compiled, pass_rate, speedup, cv, r_struct, n, q, rewards, s);
  });
  return st == SPO_OK ? ok() : st;
}

SPO_API spo_status spo_ranker_scores(const float* phi, const float* mu, const float* sigma,
                                     int32_t n, const float* params, float* scores, void* stream) {
  if (!phi || !mu || !sigma || !params || !scores)
    return fail(SPO_ERR_INVALID_ARG, "phi, mu, sigma, params and scores must be non-NULL");
  if (n < 1 || n > (1 << 30)) return fail(SPO_ERR_SHAPE, "n = %d out of range", n);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  spo_status st = traced(kTraceRanker, s, "ranker launch", [&] {
    return spo::launch_ranker_scores(phi, mu, sigma, n, params, scores, s);
  });
  return st == SPO_OK ? ok() : st;
}

SPO_API spo_status spo_ranker_workspace_size(int32_t n_pairs, size_t* bytes) {
  if (!bytes) return fail(SPO_ERR_INVALID_ARG, "bytes must be non-NULL");
  if (n_pairs < 1) return fail(SPO_ERR_SHAPE, "n_pairs must be >= 1");
  *bytes = spo::ranker_ws_bytes(n_pairs);
  return ok();
}

SPO_API spo_status spo_ranker_pair_loss(const float* phi, const float* mu, const float* sigma,
                                        const int32_t* pos, const int32_t* neg, int32_t n_pairs,
                                        const float* params, const uint8_t* keep1,
                                        const uint8_t* keep2, float drop_p, float* loss,
                                        float* grad, void* ws, size_t ws_bytes, void* stream) {
  if (!phi || !mu || !sigma || !pos || !neg || !params || !loss)
    return fail(SPO_ERR_INVALID_ARG, "a required pointer is NULL");
  if (n_pairs < 1 || n_pairs > (1 << 28)) return fail(SPO_ERR_SHAPE, "n_pairs = %d out of range", n_pairs);
  if (!(drop_p >= 0.f && drop_p < 1.f)) return fail(SPO_ERR_INVALID_ARG, "drop_p must be in [0, 1)");
  const size_t need = spo::ranker_ws_bytes(n_pairs);
  if (!ws || ws_bytes < need)
    return fail(SPO_ERR_WORKSPACE, "workspace needs %zu bytes, got %zu", need, ws_bytes);
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0)
    return fail(SPO_ERR_ALIGNMENT, "workspace must be 256-byte aligned");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  spo_status st = traced(kTraceRanker, s, "ranker launch", [&] {
    return spo::launch_ranker_pair_loss(phi, mu, sigma, pos, neg, n_pairs, params, keep1, keep2,
                                        drop_p, loss, grad, static_cast<float*>(ws), s);
  });
  return st == SPO_OK ? ok() : st;
}

SPO_API spo_status spo_scale_f32(float* x, int64_t n, float alpha, const float* alpha_dev,
                                 void* stream) {
  if (n < 0 || n > (1ll << 40)) return fail(SPO_ERR_SHAPE, "n = %lld out of range", (long long)n);
  if (!alpha_dev && !isfinite(alpha)) return fail(SPO_ERR_INVALID_ARG, "alpha must be finite");
  if (n == 0) return ok();
  if (!x) return fail(SPO_ERR_INVALID_ARG, "x must be non-NULL");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  SPO_CUDA(spo::launch_scale(x, n, alpha, alpha_dev, s), "scale launch");
  return ok();
}

SPO_API spo_status spo_validate_inputs(const int32_t* tgt, int64_t T, int64_t V,
                                       const int32_t* cu_seqlens, int32_t n_seq,
                                       const int32_t* group_id, int32_t n_groups,
                                       const float* rewards, const float* old_logp,
                                       const float* ref_logp, const uint8_t* mask,
                                       int32_t* counts, void* stream) {
  if (!counts) return fail(SPO_ERR_INVALID_ARG, "counts must be non-NULL");
  if (T < 0 || V < 0 || n_seq < 0 || n_groups < 0) return fail(SPO_ERR_SHAPE, "sizes must be >= 0");
  if ((cu_seqlens || group_id || rewards) && n_seq < 1)
    return fail(SPO_ERR_SHAPE, "n_seq must be >= 1 when per-sequence arrays are given");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  SPO_CUDA(spo::launch_validate(tgt, T, V, cu_seqlens, n_seq, group_id, n_groups, rewards, old_logp,
                                ref_logp, mask, counts, s),
           "validate launch");
  return ok();
}

SPO_API spo_status spo_group_advantages(const float* rewards, const int32_t* group_id,
                                        int32_t n_seq, int32_t n_groups, int std_mode, float eps,
                                        float* adv, void* stream) {
  spo_status st = check_adv_args(rewards, group_id, n_seq, n_groups, std_mode, eps, adv);
  if (st != SPO_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  st = traced(kTraceAdvantages, s, "advantage launch", [&] {
    return spo::launch_group_advantages(rewards, group_id, n_seq, n_groups, std_mode, eps, adv, s);
  });
  return st == SPO_OK ? ok() : st;
}

SPO_API spo_status spo_group_advantages_workspace_size(int32_t n_seq, int32_t n_groups,
                                                       size_t* bytes) {
  if (!bytes) return fail(SPO_ERR_INVALID_ARG, "bytes must be non-NULL");
  if (n_seq < 1 || n_groups < 1 || n_seq > (1 << 26) || n_groups > (1 << 26))
    return fail(SPO_ERR_SHAPE, "n_seq = %d, n_groups = %d out of range", n_seq, n_groups);
  *bytes = spo::adv_ws_bytes(n_groups);
  return ok();
}

SPO_API spo_status spo_group_advantages_ws(const float* rewards, const int32_t* group_id,
                                           int32_t n_seq, int32_t n_groups, int std_mode,
                                           float eps, float* adv, void* ws, size_t ws_bytes,
                                           void* stream) {
  spo_status st = check_adv_args(rewards, group_id, n_seq, n_groups, std_mode, eps, adv);
  if (st != SPO_OK) return st;
  const size_t need = spo::adv_ws_bytes(n_groups);
  if (!ws || ws_bytes < need)
    return fail(SPO_ERR_WORKSPACE, "workspace needs %zu bytes, got %zu", need, ws_bytes);
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0)
    return fail(SPO_ERR_ALIGNMENT, "workspace must be 256-byte aligned");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  st = traced(kTraceAdvantages, s, "advantage launch", [&] {
    return spo::launch_group_advantages_runs(rewards, group_id, n_seq, n_groups, std_mode, eps,
                                             adv, ws, s);
  });
  return st == SPO_OK ? ok() : st;
}

SPO_API spo_status spo_logprobs_keep_size(int64_t T, int64_t V, size_t* bytes) {
  if (!bytes) return fail(SPO_ERR_INVALID_ARG, "bytes must be non-NULL");
  if (T < 1 || V < 1) return fail(SPO_ERR_SHAPE, "sizes must be positive");
  *bytes = static_cast<size_t>(round_up(T, spo::kRowPad)) * static_cast<size_t>(V) * 2;
  return ok();
}

SPO_API spo_status spo_logprobs_fwd_keep(const void* H, const void* W, const int32_t* tgt,
                                         const uint8_t* mask, int64_t T, int64_t d, int64_t V,
                                         float inv_temp, float* logp, float* entropy, float* lse,
                                         void* keep, size_t keep_bytes, void* ws, size_t ws_bytes,
                                         void* stream) {
  spo_status st = check_hwv(H, W, tgt, T, d, V, inv_temp);
  if (st != SPO_OK) return st;
  if (!logp || !lse) return fail(SPO_ERR_INVALID_ARG, "logp and lse must be non-NULL");
  const size_t need = static_cast<size_t>(round_up(T, spo::kRowPad)) * static_cast<size_t>(V) * 2;
  if (!keep || keep_bytes < need)
    return fail(SPO_ERR_WORKSPACE, "keep buffer needs %zu bytes, got %zu", need, keep_bytes);
  if (!aligned16(keep)) return fail(SPO_ERR_ALIGNMENT, "keep buffer must be 16-byte aligned");
  if ((st = check_fwd_ws(T, d, V, ws, ws_bytes)) != SPO_OK) return st;
  return logprobs_impl(H, W, tgt, mask, T, d, V, 0, inv_temp, logp, entropy, lse, nullptr, ws,
                       static_cast<cudaStream_t>(stream), keep);
}

SPO_API spo_status spo_policy_loss_bwd_kept(const void* W, const float* lse, const float* g,
                                            int64_t T, int64_t d, int64_t V, float inv_temp,
                                            void* keep, size_t keep_bytes, void* fwd_ws,
                                            size_t fwd_ws_bytes, void* dH, float* dW,
                                            int accumulate_dW, void* stream) {
  // H and the targets come from the forward's workspace (compacted rows)
  if (!W) return fail(SPO_ERR_INVALID_ARG, "W must be non-NULL");
  spo_status st = check_dims(T, d, V, inv_temp);
  if (st != SPO_OK) return st;
  if (!aligned16(W)) return fail(SPO_ERR_ALIGNMENT, "W must be 16-byte aligned");
  if (!lse || !g) return fail(SPO_ERR_INVALID_ARG, "lse and g must be non-NULL");
  if (dH && !aligned16(dH)) return fail(SPO_ERR_ALIGNMENT, "dH must be 16-byte aligned");
  if (dW && !aligned16(dW)) return fail(SPO_ERR_ALIGNMENT, "dW must be 16-byte aligned");
  const size_t need = static_cast<size_t>(round_up(T, spo::kRowPad)) * static_cast<size_t>(V) * 2;
  if (!keep || keep_bytes < need)
    return fail(SPO_ERR_WORKSPACE, "keep buffer needs %zu bytes, got %zu", need, keep_bytes);
  if (!aligned16(keep)) return fail(SPO_ERR_ALIGNMENT, "keep buffer must be 16-byte aligned");
  if ((st = check_fwd_ws(T, d, V, fwd_ws, fwd_ws_bytes)) != SPO_OK) return st;
  DevInfo di;
  if ((st = device_info(&di)) != SPO_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (!dH && !dW) return ok();
  const FwdWs w = carve_fwd(fwd_ws, T, d, V);
  __nv_bfloat16* G = static_cast<__nv_bfloat16*>(keep);
  // a6 without the recompute: G from E, in place
  st = traced(kTraceFormG, s, "form G", [&] {
    return spo::launch_form_g(G, V, static_cast<int>(V), static_cast<int>(w.T_pad), w.partials,
                              w.nsplit, w.idx, w.count, w.tgt_c, lse, g, inv_temp, s);
  });
  if (st != SPO_OK) return st;
  if (dH) SPO_CUDA(cudaMemsetAsync(dH, 0, sizeof(uint16_t) * T * d, s), "memset dH");
  st = dh_dw_block(di, W, d, V, G, V, w.T_pad, w.Hc, 0, w.count, w.idx, dH, false, dW,
                   accumulate_dW != 0, w.counters, s);
  return st == SPO_OK ? ok() : st;
}

SPO_API spo_status spo_policy_loss_workspace_size(int32_t n_seq, int32_t n_groups, size_t* bytes) {
  if (!bytes) return fail(SPO_ERR_INVALID_ARG, "bytes must be non-NULL");
  if (n_seq < 1 || n_groups < 1) return fail(SPO_ERR_SHAPE, "n_seq and n_groups must be >= 1");
  *bytes = spo::loss_ws_bytes(n_seq, n_groups);
  return ok();
}

SPO_API spo_status spo_policy_loss_fwd(const float* logp, const float* old_logp,
                                       const float* ref_logp, const float* adv,
                                       const int32_t* cu_seqlens, const int32_t* group_id,
                                       int32_t n_seq, int32_t n_groups, const uint8_t* loss_mask,
                                       int64_t T, float clip_eps, float kl_beta, int agg,
                                       float* loss, float* g, float* stats, void* ws,
                                       size_t ws_bytes, void* stream) {
  if (!logp || !old_logp || !adv || !cu_seqlens || !group_id || !loss_mask || !loss || !g)
    return fail(SPO_ERR_INVALID_ARG, "a required pointer is NULL");
  if (n_seq < 1 || n_groups < 1 || n_seq > (1 << 24) || n_groups > (1 << 24))
    return fail(SPO_ERR_SHAPE, "n_seq = %d, n_groups = %d out of range", n_seq, n_groups);
  if (T < 1 || T > (1ll << 30)) return fail(SPO_ERR_SHAPE, "T = %lld outside [1, 2^30]", (long long)T);
  if (agg != SPO_AGG_SEQ_GROUP && agg != SPO_AGG_TOKEN)
    return fail(SPO_ERR_INVALID_ARG, "agg %d unknown", agg);
  if (!(clip_eps >= 0.f && clip_eps < 1.f)) return fail(SPO_ERR_INVALID_ARG, "clip_eps must be in [0, 1)");
  if (!isfinite(kl_beta)) return fail(SPO_ERR_INVALID_ARG, "kl_beta must be finite");
  const size_t need = spo::loss_ws_bytes(n_seq, n_groups);
  if (!ws || ws_bytes < need)
    return fail(SPO_ERR_WORKSPACE, "workspace needs %zu bytes, got %zu", need, ws_bytes);
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0)
    return fail(SPO_ERR_ALIGNMENT, "workspace must be 256-byte aligned");
  DevInfo di;
  spo_status st = device_info(&di);
  if (st != SPO_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const spo::LossWs w = spo::carve_loss_ws(ws, n_seq, n_groups);
  st = traced(kTracePolicyLoss, s, "policy loss launch", [&] {
    return spo::launch_policy_loss(logp, old_logp, ref_logp, adv, cu_seqlens, group_id, n_seq,
                                   n_groups, loss_mask, T, clip_eps, kl_beta, agg, loss, g, stats,
                                   w, s, di.err);
  });
  return st == SPO_OK ? ok() : st;
}

SPO_API spo_status spo_policy_loss_bwd_workspace_size(int64_t T, int64_t d, int64_t V,
                                                      size_t* bytes) {
  if (!bytes) return fail(SPO_ERR_INVALID_ARG, "bytes must be non-NULL");
  if (T < 1 || d < 1 || V < 1) return fail(SPO_ERR_SHAPE, "sizes must be positive");
  *bytes = carve_bwd(nullptr, T, d, V).bytes;
  return ok();
}

SPO_API spo_status spo_policy_loss_bwd(const void* H, const void* W, const int32_t* tgt,
                                       const float* lse, const float* g, int64_t T, int64_t d,
                                       int64_t V, float inv_temp, void* dH, float* dW,
                                       int accumulate_dW, void* ws, size_t ws_bytes, void* stream) {
  spo_status st = check_bwd_args(H, W, tgt, lse, g, T, d, V, inv_temp, dH, dW, ws, ws_bytes);
  if (st != SPO_OK) return st;
  return bwd_impl(H, W, tgt, lse, g, T, d, V, 0, inv_temp, dH, false, dW, accumulate_dW, ws,
                  static_cast<cudaStream_t>(stream));
}

SPO_API spo_status spo_policy_loss_bwd_slice(const void* H, const void* W_slice,
                                             const int32_t* tgt, const float* lse, const float* g,
                                             int64_t T, int64_t d, int64_t V_slice,
                                             int64_t v_offset, float inv_temp, float* dH_part,
                                             float* dW_slice, int accumulate_dW, void* ws,
                                             size_t ws_bytes, void* stream) {
  spo_status st = check_bwd_args(H, W_slice, tgt, lse, g, T, d, V_slice, inv_temp, dH_part,
                                 dW_slice, ws, ws_bytes);
  if (st != SPO_OK) return st;
  if (v_offset < 0 || v_offset > (1ll << 31) - 1)
    return fail(SPO_ERR_SHAPE, "v_offset = %lld outside [0, 2^31)", (long long)v_offset);
  return bwd_impl(H, W_slice, tgt, lse, g, T, d, V_slice, v_offset, inv_temp, dH_part, true,
                  dW_slice, accumulate_dW, ws, static_cast<cudaStream_t>(stream));
}

SPO_API spo_status spo_last_error_detail(char* buf, size_t n) {
  return static_cast<spo_status>(spo_last_error(buf, n));
}

SPO_API spo_status spo_sync_check(void* stream) {
  SPO_CUDA(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)), "stream work");
  int code = 0;
  return spo_device_error(&code, stream);
}

SPO_API spo_status spo_scale_f32_ratio(float* x, int64_t n, const double* num, const double* den,
                                       void* stream) {
  if (n < 0 || n > (1ll << 40)) return fail(SPO_ERR_SHAPE, "n = %lld out of range", (long long)n);
  if (n == 0) return ok();
  if (!x || !num || !den) return fail(SPO_ERR_INVALID_ARG, "x, num and den must be non-NULL");
  SPO_CUDA(spo::launch_scale_ratio(x, n, num, den, static_cast<cudaStream_t>(stream)),
           "scale launch");
  return ok();
}

SPO_API spo_status spo_dw_block_starts(int64_t V, int32_t n_blocks, int64_t* starts) {
  if (!starts) return fail(SPO_ERR_INVALID_ARG, "starts must be non-NULL");
  if (V < 1) return fail(SPO_ERR_SHAPE, "V must be positive");
  if (n_blocks < 1 || n_blocks > 4096)
    return fail(SPO_ERR_INVALID_ARG, "n_blocks = %d outside [1, 4096]", n_blocks);
  for (int k = 0; k <= n_blocks; ++k) starts[k] = dw_block_start(V, n_blocks, k);
  return ok();
}

SPO_API spo_status spo_policy_loss_bwd_ex(const void* H, const void* W, const int32_t* tgt,
                                          const float* lse, const float* g, int64_t T, int64_t d,
                                          int64_t V, int64_t v_offset, float inv_temp, void* dH,
                                          int dH_fp32, float* dW, int accumulate_dW,
                                          const spo_bwd_hooks* hooks, void* ws, size_t ws_bytes,
                                          void* stream) {
  spo_status st = check_bwd_args(H, W, tgt, lse, g, T, d, V, inv_temp, dH, dW, ws, ws_bytes);
  if (st != SPO_OK) return st;
  if (v_offset < 0 || v_offset > (1ll << 31) - 1)
    return fail(SPO_ERR_SHAPE, "v_offset = %lld outside [0, 2^31)", (long long)v_offset);
  DevInfo di;
  if ((st = device_info(&di)) != SPO_OK) return st;
  BwdHooks hk;
  std::vector<cudaEvent_t> events;
  if ((st = convert_hooks(hooks, di, &hk, &events)) != SPO_OK) return st;
  return bwd_impl(H, W, tgt, lse, g, T, d, V, v_offset, inv_temp, dH, dH_fp32 != 0, dW,
                  accumulate_dW, ws, static_cast<cudaStream_t>(stream), hooks ? &hk : nullptr);
}

SPO_API spo_status spo_grpo_workspace_size(int64_t T, int64_t d, int64_t V, int32_t n_seq,
                                           int32_t n_groups, size_t* bytes) {
  if (!bytes) return fail(SPO_ERR_INVALID_ARG, "bytes must be non-NULL");
  if (T < 1 || d < 1 || V < 1 || n_seq < 1 || n_groups < 1)
    return fail(SPO_ERR_SHAPE, "sizes must be positive");
  *bytes = carve_step(nullptr, T, d, V, n_seq, n_groups).bytes;
  return ok();
}

SPO_API spo_status spo_workspace_size(int64_t T, int64_t d, int64_t V, int32_t n_seq,
                                      size_t* bytes) {
  if (!bytes) return fail(SPO_ERR_INVALID_ARG, "bytes must be non-NULL");
  if (T < 1 || d < 1 || V < 1 || n_seq < 1) return fail(SPO_ERR_SHAPE, "sizes must be positive");
  size_t b = carve_step(nullptr, T, d, V, n_seq, n_seq).bytes;
  const size_t others[4] = {carve_fwd(nullptr, T, d, V).bytes, carve_bwd(nullptr, T, d, V).bytes,
                            spo::loss_ws_bytes(n_seq, n_seq), spo::adv_ws_bytes(n_seq)};
  for (size_t x : others) b = x > b ? x : b;
  *bytes = b;
  return ok();
}

SPO_API spo_status spo_grpo_step(const spo_grpo_batch* b, const spo_grpo_params* q,
                                 const spo_grpo_outputs* o, const spo_bwd_hooks* hooks, void* ws,
                                 size_t ws_bytes, void* stream) {
  if (!b || !q || !o) return fail(SPO_ERR_INVALID_ARG, "batch, params and out must be non-NULL");
  spo_status st = check_hwv(b->H, b->W, b->tgt, b->T, b->d, b->V, q->inv_temp);
  if (st != SPO_OK) return st;
  if (!b->cu_seqlens || !b->group_id || !b->rewards || !b->old_logp)
    return fail(SPO_ERR_INVALID_ARG, "cu_seqlens, group_id, rewards and old_logp must be non-NULL");
  if (!o->loss) return fail(SPO_ERR_INVALID_ARG, "out->loss must be non-NULL");
  if ((st = check_loss_scalars(b->n_seq, b->n_groups, q->agg, q->clip_eps, q->kl_beta)) != SPO_OK)
    return st;
  if (q->std_mode != SPO_STD_UNBIASED && q->std_mode != SPO_STD_POPULATION)
    return fail(SPO_ERR_INVALID_ARG, "std_mode %d unknown", q->std_mode);
  if (!(q->adv_eps >= 0.f) || !isfinite(q->adv_eps))
    return fail(SPO_ERR_INVALID_ARG, "adv_eps must be finite and >= 0");
  if (o->dH && !aligned16(o->dH)) return fail(SPO_ERR_ALIGNMENT, "dH must be 16-byte aligned");
  if (o->dW && !aligned16(o->dW)) return fail(SPO_ERR_ALIGNMENT, "dW must be 16-byte aligned");
  const StepWs need = carve_step(nullptr, b->T, b->d, b->V, b->n_seq, b->n_groups);
  if (!ws || ws_bytes < need.bytes)
    return fail(SPO_ERR_WORKSPACE, "workspace needs %zu bytes, got %zu", need.bytes, ws_bytes);
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0)
    return fail(SPO_ERR_ALIGNMENT, "workspace must be 256-byte aligned");
  DevInfo di;
  if ((st = device_info(&di)) != SPO_OK) return st;
  BwdHooks hk;
  std::vector<cudaEvent_t> events;
  if ((st = convert_hooks(hooks, di, &hk, &events)) != SPO_OK) return st;

  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const StepWs w = carve_step(ws, b->T, b->d, b->V, b->n_seq, b->n_groups);
  uint8_t* lm = o->loss_mask ? o->loss_mask : w.loss_mask;
  float* logp = o->logp ? o->logp : w.logp;
  float* lse = o->lse ? o->lse : w.lse;
  float* g = o->g ? o->g : w.g;
  float* adv = o->adv ? o->adv : w.adv;
  // a1: loss tokens
  st = traced(kTraceTokenSelect, s, "token_select launch", [&] {
    return spo::launch_token_select(b->cu_seqlens, b->mask, b->tgt, b->n_seq, q->window, lm,
                                    w.n_tok, s);
  });
  if (st != SPO_OK) return st;
  // a2 + a3 over the loss tokens (the forward's region of the workspace)
  if ((st = logprobs_impl(b->H, b->W, b->tgt, lm, b->T, b->d, b->V, 0, q->inv_temp, logp,
                          o->entropy, lse, nullptr, ws, s, nullptr, true)) != SPO_OK)
    return st;
  // a4 + a5.  At a step's few hundred sequences the per-group scan of the
  // advantages runs inside the loss launch (its first phase, with the group
  // counts); otherwise the run path first (same bits), then the loss.
  // g = dL/dlogp, times the rank weight if any.
  const bool scan = static_cast<long long>(b->n_seq) * b->n_groups <= (1ll << 22);
  if (!scan) {
    st = traced(kTraceAdvantages, s, "advantage launch", [&] {
      return spo::launch_group_advantages_runs(b->rewards, b->group_id, b->n_seq, b->n_groups,
                                               q->std_mode, q->adv_eps, adv, w.adv_ws, s);
    });
    if (st != SPO_OK) return st;
  }
  const spo::LossWs lw = spo::carve_loss_ws(w.loss_ws, b->n_seq, b->n_groups);
  st = traced(kTracePolicyLoss, s, "policy loss launch", [&] {
    return spo::launch_policy_loss(logp, b->old_logp, b->ref_logp, adv, b->cu_seqlens,
                                   b->group_id, b->n_seq, b->n_groups, lm, b->T, q->clip_eps,
                                   q->kl_beta, q->agg, o->loss, g, o->stats, lw, s, di.err,
                                   q->loss_scale, scan ? b->rewards : nullptr, q->std_mode,
                                   q->adv_eps, scan ? adv : nullptr);
  });
  if (st != SPO_OK) return st;
  // a6 - a8 over the forward's compaction (loss tokens); lse and g read at token positions
  if (!o->dH && !o->dW) return (st = record_hook_events(hooks ? &hk : nullptr, s)) == SPO_OK ? ok() : st;
  const FwdWs f = carve_fwd(ws, b->T, b->d, b->V);
  if (o->dH)
    SPO_CUDA(spo::launch_zero_skipped_rows(g, b->T, static_cast<int>(2 * b->d), o->dH, s),
             "zero skipped dH rows");
  const BwdRows rows{f.Hc, f.idx, f.count, f.tgt_c, lse, g, true, f.T_pad};
  st = bwd_core(di, b->W, b->d, b->V, q->inv_temp, rows, w.G, w.chunk, o->dH, false, o->dW,
                o->accumulate_dW, f.counters, hooks ? &hk : nullptr, s);
  return st == SPO_OK ? ok() : st;
}

SPO_API spo_status spo_trace_enable(int on) {
  std::lock_guard<std::mutex> lk(g_trace_mu);
  g_trace_on = on != 0;
  return ok();
}

SPO_API spo_status spo_trace_read(int* kinds, float* ms, int max_records, int* n_records) {
  if (!n_records || max_records < 0 || (max_records > 0 && (!kinds || !ms)))
    return fail(SPO_ERR_INVALID_ARG, "kinds/ms/n_records invalid");
  std::vector<TraceRec> recs;
  {
    std::lock_guard<std::mutex> lk(g_trace_mu);
    recs.swap(g_trace);
  }
  int n = 0;
  spo_status st = SPO_OK;
  for (const TraceRec& r : recs) {
    float t = 0.f;
    cudaError_t e = cudaEventSynchronize(r.stop);
    if (e == cudaSuccess) e = cudaEventElapsedTime(&t, r.start, r.stop);
    if (e != cudaSuccess && st == SPO_OK) st = cuda_fail(e, "trace event");
    if (n < max_records) {
      kinds[n] = r.kind;
      ms[n] = t;
    }
    ++n;
  }
  {
    std::lock_guard<std::mutex> lk(g_trace_mu);
    for (const TraceRec& r : recs) g_trace_pool.push_back(r);
  }
  *n_records = n;
  return st == SPO_OK ? ok() : st;
}

SPO_API long long spo_launch_count(void) { return spo::launches(); }

SPO_API spo_status spo_set_tuning(int key, int64_t value) {
  switch (key) {
    case SPO_TUNE_PAIR_MMA:
      if (value != 0 && value != 1) return fail(SPO_ERR_INVALID_ARG, "pair must be 0 or 1");
      g_tune_pair = static_cast<int>(value);
      return ok();
    case SPO_TUNE_GROUP_M:
      if (value < 1 || value > 4096) return fail(SPO_ERR_INVALID_ARG, "group_m must be in [1, 4096]");
      for (int k = 0; k < 4; ++k) g_tune_group_m[k] = static_cast<int>(value);
      return ok();
    case SPO_TUNE_DYNAMIC_MASK:
      if (value < 0 || value > 15) return fail(SPO_ERR_INVALID_ARG, "dynamic mask must be in [0, 15]");
      g_tune_dynamic_mask = static_cast<int>(value);
      return ok();
    case SPO_TUNE_DW_SPLIT_ROWS:
      if (value < 0 || value > (1 << 24) || value % 256 != 0)
        return fail(SPO_ERR_INVALID_ARG, "dW split rows must be a multiple of 256 in [0, 2^24]");
      g_tune_dw_split = static_cast<int>(value);
      return ok();
    case SPO_TUNE_GROUP_M_FWD:
    case SPO_TUNE_GROUP_M_GRAD:
    case SPO_TUNE_GROUP_M_DH:
    case SPO_TUNE_GROUP_M_DW:
      if (value < 1 || value > 4096) return fail(SPO_ERR_INVALID_ARG, "group_m must be in [1, 4096]");
      g_tune_group_m[key - SPO_TUNE_GROUP_M_FWD] = static_cast<int>(value);
      return ok();
    case SPO_TUNE_RASTER_FWD:
    case SPO_TUNE_RASTER_GRAD:
    case SPO_TUNE_RASTER_DH:
    case SPO_TUNE_RASTER_DW:
      if (value != 0 && value != 1) return fail(SPO_ERR_INVALID_ARG, "raster must be 0 or 1");
      g_tune_raster[key - SPO_TUNE_RASTER_FWD] = static_cast<int>(value);
      return ok();
    case SPO_TUNE_KSYNC_FWD:
    case SPO_TUNE_KSYNC_GRAD:
    case SPO_TUNE_KSYNC_DH:
    case SPO_TUNE_KSYNC_DW:
      if (value < 0 || value > (1 << 20))
        return fail(SPO_ERR_INVALID_ARG, "throttle window must be in [0, 2^20] k-blocks");
      g_tune_ksync[key - SPO_TUNE_KSYNC_FWD] = static_cast<int>(value);
      return ok();
    case SPO_TUNE_KSYNC_EPOCH:
      if (value < 1 || value > 4096)
        return fail(SPO_ERR_INVALID_ARG, "throttle epoch must be in [1, 4096] k-blocks");
      g_tune_ksync_epoch = static_cast<int>(value);
      return ok();
    case SPO_TUNE_DH_WIDE:
      if (value < 0 || value > 2) return fail(SPO_ERR_INVALID_ARG, "dH wide must be 0, 1 or 2");
      g_tune_dh_wide = static_cast<int>(value);
      return ok();
    case SPO_TUNE_LOGITS_WIDE:
      if (value < 0 || value > 7) return fail(SPO_ERR_INVALID_ARG, "logits wide must be in [0, 7]");
      g_tune_logits_wide = static_cast<int>(value);
      return ok();
    case SPO_TUNE_DEFAULTS:
      g_tune_pair = 1;
      for (int k = 0; k < 4; ++k) {
        g_tune_group_m[k] = kDefaultGroupM[k];
        g_tune_raster[k] = kDefaultRaster[k];
        g_tune_ksync[k] = spo::kDefaultKsync[k];
      }
      g_tune_ksync_epoch = spo::kDefaultKsyncEpoch;
      g_tune_dynamic_mask = spo::kDefaultDynamicMask;
      g_tune_dw_split = spo::kDefaultDwSplitRows;
      g_tune_dh_wide = spo::kDefaultDhWide;
      g_tune_logits_wide = spo::kDefaultLogitsWide;
      return ok();
    case SPO_TUNE_RASTER:
      if (value != 0 && value != 1) return fail(SPO_ERR_INVALID_ARG, "raster must be 0 or 1");
      for (int k = 0; k < 4; ++k) g_tune_raster[k] = static_cast<int>(value);
      return ok();
    default:
      return fail(SPO_ERR_INVALID_ARG, "unknown tuning key %d", key);
  }
}

}  // extern "C"

// ------------------------------------------------------------ no-allocation loss forward
// Scratch of spo_policy_loss_fwd_noalloc.  It is part of the library's device
// image: every GPU that loads libspo holds these bytes until the process exits.
namespace {

constexpr size_t kNoAllocLossScratchBytes = static_cast<size_t>(1) << 20;  // 1 MiB

static __device__ __align__(256) unsigned char g_noalloc_loss_scratch[kNoAllocLossScratchBytes];

std::mutex g_noalloc_mu;
void* g_noalloc_scratch_ptr[64] = {};

// The array's name is only a host-side handle; its device address is looked
// up once per device (with that device current) and cached.
spo_status noalloc_scratch(int dev, void** out) {
  std::lock_guard<std::mutex> lk(g_noalloc_mu);
  if (!g_noalloc_scratch_ptr[dev]) {
    void* p = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_loss_scratch);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(no-alloc loss scratch)");
    g_noalloc_scratch_ptr[dev] = p;
  }
  *out = g_noalloc_scratch_ptr[dev];
  return SPO_OK;
}

}  // namespace

extern "C" {

SPO_API spo_status spo_policy_loss_fwd_noalloc(const float* logp, const float* old_logp,
                                               const float* ref_logp, const float* adv,
                                               const int32_t* cu_seqlens, const int32_t* group_id,
                                               int32_t n_seq, int32_t n_groups,
                                               const uint8_t* loss_mask, int64_t T, float clip_eps,
                                               float kl_beta, int agg, float* loss, float* g,
                                               float* stats, void* stream) {
  if (!logp || !old_logp || !adv || !cu_seqlens || !group_id || !loss_mask || !loss || !g)
    return fail(SPO_ERR_INVALID_ARG, "a required pointer is NULL");
  if (n_seq < 1 || n_groups < 1 || n_seq > (1 << 24) || n_groups > (1 << 24))
    return fail(SPO_ERR_SHAPE, "n_seq = %d, n_groups = %d out of range", n_seq, n_groups);
  if (T < 1 || T > (1ll << 30)) return fail(SPO_ERR_SHAPE, "T = %lld outside [1, 2^30]", (long long)T);
  if (agg != SPO_AGG_SEQ_GROUP && agg != SPO_AGG_TOKEN)
    return fail(SPO_ERR_INVALID_ARG, "agg %d unknown", agg);
  if (!(clip_eps >= 0.f && clip_eps < 1.f)) return fail(SPO_ERR_INVALID_ARG, "clip_eps must be in [0, 1)");
  if (!isfinite(kl_beta)) return fail(SPO_ERR_INVALID_ARG, "kl_beta must be finite");
  const size_t need = spo::loss_ws_bytes(n_seq, n_groups);
  if (need > kNoAllocLossScratchBytes)
    return fail(SPO_ERR_WORKSPACE,
                "n_seq = %d, n_groups = %d need %zu scratch bytes but the static scratch of "
                "spo_policy_loss_fwd_noalloc holds %zu; use spo_policy_loss_fwd with a workspace",
                n_seq, n_groups, need, kNoAllocLossScratchBytes);
  DevInfo di;
  spo_status st = device_info(&di);
  if (st != SPO_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // The scratch looked up below is the current device's copy of the array; a
  // stream of another device would run the kernels against it.
  int stream_dev = -1;
  SPO_CUDA(cudaStreamGetDevice(s, &stream_dev), "cudaStreamGetDevice");
  if (stream_dev != di.dev)
    return fail(SPO_ERR_INVALID_ARG,
                "stream belongs to device %d but device %d is current; make the stream's device "
                "current before calling spo_policy_loss_fwd_noalloc",
                stream_dev, di.dev);
  void* scratch = nullptr;
  if ((st = noalloc_scratch(di.dev, &scratch)) != SPO_OK) return st;
  // carve_loss_ws lays out the same buffers as the workspace entry point; the
  // group-size counters are cleared on the stream by launch_policy_loss.
  const spo::LossWs w = spo::carve_loss_ws(scratch, n_seq, n_groups);
  st = traced(kTracePolicyLoss, s, "policy loss launch", [&] {
    return spo::launch_policy_loss(logp, old_logp, ref_logp, adv, cu_seqlens, group_id, n_seq,
                                   n_groups, loss_mask, T, clip_eps, kl_beta, agg, loss, g, stats,
                                   w, s, di.err);
  });
  return st == SPO_OK ? ok() : st;
}

}  // extern "C"
