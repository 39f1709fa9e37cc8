// C ABI of libdblast: argument checks, prep/workspace layouts, launch order.
// Every entry point is asynchronous on the caller's stream and allocates no
// device memory.
#include <algorithm>
#include <atomic>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <vector>

#include <cuda.h>
#include <nvtx3/nvToolsExt.h>

#include "dblast_internal.cuh"

namespace dblast {

static uint32_t g_wait_limit = 0;  // 0 = default; read by the tensor-core launchers
uint32_t wait_limit() { return g_wait_limit; }

// Device-side index checks (dblast_set_checks; DBLAST_CHECK=1 turns them on
// from the start): data-dependent token indices are tested against [0, V)
// and a value outside it is recorded in the workspace status word.
static std::atomic<int> g_checks{-1};
static bool checks_on() {
  int v = g_checks.load(std::memory_order_relaxed);
  if (v < 0) {
    const char* e = getenv("DBLAST_CHECK");
    v = (e && e[0] == '1') ? 1 : 0;
    int expect = -1;
    g_checks.compare_exchange_strong(expect, v);
    v = g_checks.load(std::memory_order_relaxed);
  }
  return v == 1;
}

// An NVTX range around each entry point (a no-op unless a profiler is attached).
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

// ------------------------------------------------------------ measurement
static std::mutex g_stats_mu;
static std::atomic<uint64_t> g_launches{0}, g_calls{0}, g_tc_launches{0};
// Per-pass timing: CUDA events around every g_period-th draft pass and
// verify pass (0: off).  An event between two kernels keeps the later one
// from being scheduled while the earlier one finishes, so a period above 1
// leaves most passes undisturbed.
static int g_period = 0;
constexpr int kMaxTimed = 4096;
static std::vector<cudaEvent_t> g_ev[2];  // pairs (begin, end) per timed call
static int g_n_ev[2] = {0, 0};
static uint64_t g_seen[2] = {0, 0};       // passes seen since the reset
static bool g_open[2] = {false, false};   // a begin event awaits its end

void count_launches(int n) { g_launches.fetch_add((uint64_t)n, std::memory_order_relaxed); }
void count_tc_launch() { g_tc_launches.fetch_add(1, std::memory_order_relaxed); }

// DBLAST_DEBUG_SYNC=1: synchronise after every launcher and name the one that failed
static bool debug_sync() {
  static int v = -1;
  if (v < 0) {
    const char* e = getenv("DBLAST_DEBUG_SYNC");
    v = (e && e[0] == '1') ? 1 : 0;
  }
  return v == 1;
}
void debug_kernel(const char* name, cudaStream_t s) {
  if (!debug_sync()) return;
  cudaError_t e = cudaGetLastError();
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  fprintf(stderr, "dblast debug kernel: %-20s %s\n", name, cudaGetErrorString(e));
}

// DBLAST_FUSE_TSTATS=0: target statistics as a kernel of their own (the
// fused step's default computes them in the draft pass)
static bool fuse_tstats_enabled() {
  const char* e = getenv("DBLAST_FUSE_TSTATS");
  return !(e && e[0] == '0');
}

static cudaError_t dbg(cudaError_t e, const char* what, cudaStream_t s) {
  if (e != cudaSuccess || !debug_sync()) return e;
  e = cudaStreamSynchronize(s);
  if (e == cudaSuccess) e = cudaGetLastError();
  fprintf(stderr, "dblast debug: %-22s %s\n", what, cudaGetErrorString(e));
  return e;
}

static cudaEvent_t pool_event(int which, int idx) {
  auto& v = g_ev[which];
  while ((int)v.size() <= idx) {
    cudaEvent_t e;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    v.push_back(e);
  }
  return v[idx];
}

void pass_event_begin(int which, cudaStream_t s) {
  std::lock_guard<std::mutex> lk(g_stats_mu);
  g_open[which] = false;
  if (g_period <= 0 || g_n_ev[which] >= kMaxTimed) return;
  if (g_seen[which]++ % (uint64_t)g_period != 0) return;
  cudaEvent_t e = pool_event(which, 2 * g_n_ev[which]);
  g_open[which] = e && cudaEventRecord(e, s) == cudaSuccess;
}

void pass_event_end(int which, cudaStream_t s) {
  std::lock_guard<std::mutex> lk(g_stats_mu);
  if (!g_open[which]) return;
  g_open[which] = false;
  cudaEvent_t e = pool_event(which, 2 * g_n_ev[which] + 1);
  if (e && cudaEventRecord(e, s) == cudaSuccess) ++g_n_ev[which];
}

PrepLayout prep_layout(int V, int H, int K, int r, bool has_e) {
  PrepLayout p{};
  p.V = V;
  p.K = K;
  p.rr = r + (has_e ? 1 : 0);
  p.rp = ceil_div(p.rr, 16) * 16;
  p.KC = K * 2 * p.rp;
  size_t o = 0;
  p.off_wu = o;
  o = align_up(o + (size_t)V * K * p.rr * sizeof(float), 256);
  p.off_wuop = o;
  o = align_up(o + (size_t)V * p.KC * sizeof(__half), 256);
  p.off_sw = o;
  o = align_up(o + (size_t)K * sizeof(float), 256);
  p.off_ut = o;
  o = align_up(o + (size_t)ceil_div(K * p.rr, MTILE) * MTILE * H * 2, 256);
  p.off_vt = o;
  o = align_up(o + (size_t)ceil_div(K * p.rr, MTILE) * MTILE * H * 2, 256);
  p.off_status = o;
  o = align_up(o + sizeof(DevStatus), 256);
  p.total = o;
  return p;
}

WsLayout ws_layout(int V, int K, int r, bool has_e, int N, int B, int has_bonus) {
  WsLayout w{};
  w.N = N;
  w.B = B;
  w.M = N * B;
  w.Mpad = ceil_div(w.M, MTILE) * MTILE;
  w.K = K;
  w.rr = r + (has_e ? 1 : 0);
  w.rp = ceil_div(w.rr, 16) * 16;
  w.KC = K * 2 * w.rp;
  w.V = V;
  w.nt = ceil_div(V, TILE_V);
  (void)has_bonus;  // the layout is the same with or without a bonus row
  w.Rt = N * (B + 1);
  size_t o = 0;
  auto take = [&](size_t bytes) {
    size_t at = o;
    o = align_up(o + bytes, 256);
    return at;
  };
  w.off_status = take(256);
  w.off_codes = take((size_t)w.Mpad * K * w.rr * sizeof(float));
  w.off_cscale = take((size_t)w.Mpad * K * sizeof(float));
  w.off_cop = take((size_t)w.Mpad * w.KC * sizeof(__half));
  w.off_zhat = take((size_t)N * sizeof(int32_t));
  w.off_log2pi = take((size_t)N * K * sizeof(float));
  // the stash [M, V]; before the draft pass writes it, the same bytes hold
  // the split-K partials of the codes (up to CODES_MAX_SPLIT splits of
  // [M, K rr]), so it is never smaller than those
  w.off_stash = take((size_t)w.M * std::max<size_t>((size_t)V, (size_t)CODES_MAX_SPLIT * K * w.rr) *
                     sizeof(float));
  w.off_partd = take((size_t)w.nt * K * w.Mpad * sizeof(float2));
  w.off_lsep = take((size_t)LSE_SPLIT * w.M * K * sizeof(float4));
  w.off_lse2 = take((size_t)w.M * K * sizeof(float2));
  w.off_lq2 = take((size_t)w.M * K * sizeof(float2));
  w.off_w2 = take((size_t)w.M * K * sizeof(float2));
  w.off_qtok = take((size_t)w.M * sizeof(float));
  w.off_tok = take((size_t)w.M * sizeof(int32_t));
  w.off_vcz = take((size_t)w.M * K * sizeof(float2));
  w.off_vb0 = take((size_t)w.M * sizeof(float));
  w.off_partt = take((size_t)w.nt * w.Rt * sizeof(float2));
  w.off_lt2 = take((size_t)w.Rt * sizeof(float2));
  w.off_partv = take((size_t)w.nt * w.Mpad * sizeof(float2));
  w.off_ties = take((size_t)2 * N * sizeof(uint32_t));  // tie flags, then per-sequence counters
  w.off_xhat = take((size_t)w.M * K * sizeof(int32_t));
  w.off_cmask = take((size_t)w.M * sizeof(uint32_t));
  w.off_coll = take((size_t)w.Rt * sizeof(float));
  w.off_ftok = take((size_t)w.Rt * FILTER_MAX_K * sizeof(int32_t));
  w.off_fp = take((size_t)w.Rt * FILTER_MAX_K * sizeof(float));
  w.off_fcnt = take((size_t)w.Rt * sizeof(int32_t));
  w.off_ftie = take((size_t)w.Rt * sizeof(uint32_t));
  w.off_partg = take((size_t)w.nt * K * w.Mpad * sizeof(float));
  w.total = o;
  return w;
}

cudaError_t launch_draft_pass_tc(const StepCtx& c);
cudaError_t launch_verify_pass_tc(const StepCtx& c);

}  // namespace dblast

using namespace dblast;

static bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

namespace dblast {
typedef CUresult (*CtxGetCurrentFn)(CUcontext*);
typedef CUresult (*CtxGetIdFn)(CUcontext, unsigned long long*);

unsigned long long current_context_id() {
  static CtxGetCurrentFn get_cur = nullptr;
  static CtxGetIdFn get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      get_cur = reinterpret_cast<CtxGetCurrentFn>(p);
    p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<CtxGetIdFn>(p);
  });
  if (!get_cur || !get_id) return 0ull;
  CUcontext ctx = nullptr;
  unsigned long long id = 0ull;
  if (get_cur(&ctx) != CUDA_SUCCESS || !ctx || get_id(ctx, &id) != CUDA_SUCCESS) return 0ull;
  return id;
}
}  // namespace dblast

static dblast_status check_head(const dblast_head* h, bool need_prep) {
  if (!h) return DBLAST_ERR_INVALID_ARG;
  if (h->V < 1 || h->H < 8 || (h->H % 8) != 0 || h->K < 1 || h->K > 32 || h->r < 1 || h->r > 64)
    return DBLAST_ERR_INVALID_ARG;
  if (h->dtype != DBLAST_BF16 && h->dtype != DBLAST_F32) return DBLAST_ERR_INVALID_ARG;
  if (!h->W || !h->U || !h->Vf || !h->Wp) return DBLAST_ERR_INVALID_ARG;
  const void* ptrs[] = {h->W, h->U, h->Vf, h->e, h->Wp, h->bp, h->vbias};
  for (const void* p : ptrs)
    if (p && !aligned16(p)) return DBLAST_ERR_INVALID_ARG;
  if (need_prep) {
    if (!h->prep || !aligned16(h->prep)) return DBLAST_ERR_WORKSPACE;
    if (h->prep_bytes < dblast_prep_bytes(h)) return DBLAST_ERR_WORKSPACE;
  }
  return DBLAST_OK;
}

static dblast_status check_args(const dblast_head* h, const dblast_block_args* a) {
  if (!a) return DBLAST_ERR_INVALID_ARG;
  if (a->N < 1 || a->B < 1 || a->B > 32) return DBLAST_ERR_INVALID_ARG;
  if (!(a->temperature > 0.f) || !(a->z_temperature >= 0.f)) return DBLAST_ERR_INVALID_ARG;
  if (!a->hidden || !a->pos || !a->round) return DBLAST_ERR_INVALID_ARG;
  if (!aligned16(a->hidden) || (a->anchor && !aligned16(a->anchor))) return DBLAST_ERR_INVALID_ARG;
  if ((long long)a->N * a->B > (1LL << 24)) return DBLAST_ERR_INVALID_ARG;
  if (a->impl == DBLAST_IMPL_TCGEN05 && !tc_supported(h)) return DBLAST_ERR_UNSUPPORTED;
  if (a->impl != DBLAST_IMPL_AUTO && a->impl != DBLAST_IMPL_SIMT && a->impl != DBLAST_IMPL_TCGEN05)
    return DBLAST_ERR_INVALID_ARG;
  if (a->mode != DBLAST_MODE_SOFT && a->mode != DBLAST_MODE_GREEDY) return DBLAST_ERR_INVALID_ARG;
  return DBLAST_OK;
}

static bool use_tc(const dblast_head* h, const dblast_block_args* a) {
  if (a->impl == DBLAST_IMPL_SIMT) return false;
  if (a->impl == DBLAST_IMPL_TCGEN05) return true;
  return tc_supported(h);
}

static dblast_status make_ctx(const dblast_head* h, const dblast_block_args* a, void* ws,
                              size_t ws_bytes, int has_bonus, dblast_stream_t stream,
                              StepCtx* c) {
  if (!ws || !aligned16(ws)) return DBLAST_ERR_WORKSPACE;
  if (ws_bytes < dblast_workspace_bytes(h, a->N, a->B, has_bonus)) return DBLAST_ERR_WORKSPACE;
  c->head = h;
  c->args = a;
  c->has_e = h->e != nullptr;
  c->pl = prep_layout(h->V, h->H, h->K, h->r, c->has_e);
  c->wl = ws_layout(h->V, h->K, h->r, c->has_e, a->N, a->B, has_bonus);
  c->ws = static_cast<unsigned char*>(ws);
  c->prep = static_cast<const unsigned char*>(h->prep);
  c->stream = reinterpret_cast<cudaStream_t>(stream);
  c->k2 = LOG2E / a->temperature;
  c->tc = use_tc(h, a);
  c->greedy = a->mode == DBLAST_MODE_GREEDY;
  c->target = nullptr;
  c->Bt = a->B + (has_bonus ? 1 : 0);
  c->fuse_tstats = false;
  c->lse_target = nullptr;
  c->chk = checks_on() ? reinterpret_cast<DevStatus*>(c->ws + c->wl.off_status) : nullptr;
  return DBLAST_OK;
}

// top-k / top-p of a verify call: on, and the number of tokens it keeps at most
static bool filter_on(const dblast_head* h, const dblast_verify_out* o) {
  const bool k_on = o->top_k >= 1 && o->top_k < h->V;
  const bool p_on = o->top_p > 0.f && o->top_p < 1.f;
  return k_on || p_on;
}
static dblast_status check_filter(const dblast_head* h, const dblast_verify_out* o) {
  if (o->top_k < 0 || !(o->top_p >= 0.f)) return DBLAST_ERR_INVALID_ARG;
  if (!filter_on(h, o)) return DBLAST_OK;
  const int k_eff = (o->top_k >= 1 && o->top_k < h->V) ? o->top_k : h->V;
  if (k_eff > FILTER_MAX_K || ceil_div(h->V, TILE_V) > FILTER_MAX_TILES)
    return DBLAST_ERR_UNSUPPORTED;
  return DBLAST_OK;
}
// the dblast_verify_out the filter kernel reads: top_k clamped to what stays
static dblast_verify_out filter_args(const dblast_head* h, const dblast_verify_out* o) {
  dblast_verify_out f = *o;
  f.top_k = (o->top_k >= 1 && o->top_k < h->V) ? o->top_k : h->V;
  if (!(f.top_p > 0.f && f.top_p < 1.f)) f.top_p = 1.f;
  return f;
}

static dblast_status cuda_status(cudaError_t e) {
  if (e == cudaSuccess) return DBLAST_OK;
  fprintf(stderr, "dblast: CUDA error %s\n", cudaGetErrorString(e));
  return DBLAST_ERR_CUDA;
}

extern "C" {

size_t dblast_prep_bytes(const dblast_head* h) {
  if (!h || h->V < 1 || h->K < 1 || h->r < 1) return 0;
  return prep_layout(h->V, h->H, h->K, h->r, h->e != nullptr).total;
}

size_t dblast_workspace_bytes(const dblast_head* h, int N, int B, int has_bonus) {
  if (!h || N < 1 || B < 1 || h->V < 1 || h->K < 1 || h->r < 1) return 0;
  return ws_layout(h->V, h->K, h->r, h->e != nullptr, N, B, has_bonus).total;
}

dblast_status dblast_head_prepare(const dblast_head* h, dblast_stream_t stream) {
  NvtxRange nvtx("dblast_head_prepare");
  dblast_status st = check_head(h, true);
  if (st != DBLAST_OK) return st;
  PrepLayout pl = prep_layout(h->V, h->H, h->K, h->r, h->e != nullptr);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  return cuda_status(dbg(launch_prep(h, pl, s), "prep", s));
}

static dblast_status draft_impl(const StepCtx& c, dblast_draft_out* out) {
  g_calls.fetch_add(1, std::memory_order_relaxed);
  // the tie words and draft-token counters start in the launch that computes
  // the prior (no memset: it would end the chain of dependent launches)
  cudaError_t e = dbg(launch_codes(c), "codes", c.stream);
  if (e == cudaSuccess) {
    pass_event_begin(0, c.stream);
    e = c.tc ? launch_draft_pass_tc(c) : launch_draft_pass_simt(c);
    pass_event_end(0, c.stream);
    e = dbg(e, "draft_pass", c.stream);
  }
  if (e == cudaSuccess)
    e = dbg(c.greedy ? launch_greedy_draft_finalize(c, out) : launch_draft_finalize(c, out),
            "draft_finalize", c.stream);
  return cuda_status(e);
}

static cudaError_t verify_passes(const StepCtx& c, dblast_verify_out* out) {
  // with a target filter p' has at most k tokens: one kernel verifies against
  // it in either mode (the filter itself ran after the target statistics)
  if (filter_on(c.head, out)) {
    const dblast_verify_out f = filter_args(c.head, out);
    return dbg(launch_filtered_verify(c, &f), "filtered_verify", c.stream);
  }
  // greedy-branch mode has no vocabulary-wide verify pass: q_greedy has at
  // most K atoms, so one kernel reads p at them and draws the residual
  if (c.greedy) return dbg(launch_greedy_verify_finalize(c, out), "verify_finalize", c.stream);
  pass_event_begin(1, c.stream);
  cudaError_t e = c.tc ? launch_verify_pass_tc(c) : launch_verify_pass_simt(c);
  pass_event_end(1, c.stream);
  e = dbg(e, "verify_pass", c.stream);
  if (e == cudaSuccess) e = dbg(launch_verify_finalize(c, out), "verify_finalize", c.stream);
  return e;
}

static dblast_status verify_impl(StepCtx c, dblast_verify_out* out) {
  c.target = out->target;
  c.Bt = c.args->B + (out->has_bonus ? 1 : 0);
  g_calls.fetch_add(1, std::memory_order_relaxed);
  cudaError_t e = dbg(launch_target_stats(c, out), "target_stats", c.stream);
  if (e == cudaSuccess && filter_on(c.head, out)) {
    const dblast_verify_out f = filter_args(c.head, out);
    e = dbg(launch_target_filter(c, &f), "target_filter", c.stream);
  }
  if (e == cudaSuccess) e = verify_passes(c, out);
  return cuda_status(e);
}


// One internal stream and four events per device for the fork/join of
// kernels that do not depend on each other inside dblast_draft_and_verify
// (no device memory; created by the first such call on the device and held
// until the process exits, or made again after a device reset gave the
// device a new context).  The mutex keeps one call's fork/join pairs
// together when several host threads call in.
struct SideStream {
  cudaStream_t s = nullptr;
  cudaEvent_t ev[4] = {nullptr, nullptr, nullptr, nullptr};
  unsigned long long ctx = 0ull;  // context the handles belong to
};
static std::mutex g_side_mu;
static SideStream g_side[64];

static cudaError_t side_stream(SideStream** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  SideStream& ss = g_side[dev];
  const unsigned long long ctx = current_context_id();
  if (ss.s && ctx != ss.ctx) ss = SideStream{};  // handles of a context that was reset
  if (!ss.s) {
    ss.ctx = ctx;
    e = cudaStreamCreateWithFlags(&ss.s, cudaStreamNonBlocking);
    for (int i = 0; i < 4 && e == cudaSuccess; ++i)
      e = cudaEventCreateWithFlags(&ss.ev[i], cudaEventDisableTiming);
    if (e != cudaSuccess) return e;
  }
  *out = &ss;
  return cudaSuccess;
}

// draft and verify of one block.  The category prior runs in the launch that
// reduces the codes; the target statistics run inside the draft pass (bf16
// targets with 16-byte rows), else on the library's second stream beside the
// draft finalize kernels, where the target filter also runs.
static dblast_status step_impl(StepCtx c, dblast_draft_out* dout, dblast_verify_out* vout) {
  if (debug_sync()) {  // serial order, so a failing launcher is named
    dblast_status st = draft_impl(c, dout);
    return st != DBLAST_OK ? st : verify_impl(c, vout);
  }
  c.target = vout->target;
  c.Bt = c.args->B + (vout->has_bonus ? 1 : 0);
  // bf16 targets with 16-byte rows: the draft pass's idle warps compute the
  // target statistics while its tensor cores run.  The pass takes about 4%
  // longer, but the latency-bound draft finalize kernels after it then run
  // alone: beside a stand-alone statistics kernel, which fills HBM and the
  // SMs, they took twice as long as on their own.
  c.fuse_tstats = c.tc && c.head->dtype == DBLAST_BF16 && (c.head->V % 8) == 0 &&
                  aligned16(vout->target) && fuse_tstats_enabled();
  c.lse_target = vout->lse_target;
  g_calls.fetch_add(2, std::memory_order_relaxed);
  std::lock_guard<std::mutex> lk(g_side_mu);
  SideStream* ss = nullptr;
  cudaError_t e = side_stream(&ss);
  StepCtx side = c;
  if (e == cudaSuccess) side.stream = ss->s;
  // the codes GEMM, then the codes reduction and the category prior in one
  // launch (which also starts the tie words and the draft-token counters),
  // then the draft pass
  if (e == cudaSuccess) e = launch_codes(c);
  if (e == cudaSuccess) {
    pass_event_begin(0, c.stream);
    e = c.tc ? launch_draft_pass_tc(c) : launch_draft_pass_simt(c);
    pass_event_end(0, c.stream);
  }
  // fork: target statistics (unless the draft pass took them) and the target
  // filter | draft finalize
  const bool side_work = !c.fuse_tstats || filter_on(c.head, vout);
  if (side_work) {
    if (e == cudaSuccess) e = cudaEventRecord(ss->ev[2], c.stream);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(side.stream, ss->ev[2], 0);
    if (e == cudaSuccess && !c.fuse_tstats) e = launch_target_stats(side, vout);
    if (e == cudaSuccess && filter_on(c.head, vout)) {
      const dblast_verify_out f = filter_args(c.head, vout);
      e = launch_target_filter(side, &f);
    }
    if (e == cudaSuccess) e = cudaEventRecord(ss->ev[3], side.stream);
  }
  // greedy mode with the statistics in the draft pass and no filter: nothing
  // runs beside the draft finalize, so one kernel per sequence takes the
  // greedy draft and verifies it
  if (c.greedy && c.fuse_tstats && !side_work) {
    if (e == cudaSuccess) e = launch_greedy_step_finalize(c, dout, vout);
    return cuda_status(e);
  }
  if (e == cudaSuccess)
    e = c.greedy ? launch_greedy_draft_finalize(c, dout) : launch_draft_finalize(c, dout);
  // join
  if (e == cudaSuccess && side_work) e = cudaStreamWaitEvent(c.stream, ss->ev[3], 0);
  if (e == cudaSuccess) e = verify_passes(c, vout);
  return cuda_status(e);
}

dblast_status dblast_draft_block(const dblast_head* h, const dblast_block_args* a,
                                 dblast_draft_out* out, void* ws, size_t ws_bytes,
                                 dblast_stream_t stream) {
  NvtxRange nvtx("dblast_draft_block");
  dblast_status st = check_head(h, true);
  if (st == DBLAST_OK) st = check_args(h, a);
  if (st != DBLAST_OK) return st;
  StepCtx c;
  st = make_ctx(h, a, ws, ws_bytes, 1, stream, &c);
  if (st != DBLAST_OK) return st;
  return draft_impl(c, out);
}

dblast_status dblast_verify_block(const dblast_head* h, const dblast_block_args* a,
                                  dblast_verify_out* out, void* ws, size_t ws_bytes,
                                  dblast_stream_t stream) {
  NvtxRange nvtx("dblast_verify_block");
  dblast_status st = check_head(h, true);
  if (st == DBLAST_OK) st = check_args(h, a);
  if (st != DBLAST_OK) return st;
  if (!out || !out->target || !aligned16(out->target)) return DBLAST_ERR_INVALID_ARG;
  st = check_filter(h, out);
  if (st != DBLAST_OK) return st;
  StepCtx c;
  st = make_ctx(h, a, ws, ws_bytes, out->has_bonus ? 1 : 0, stream, &c);
  if (st != DBLAST_OK) return st;
  return verify_impl(c, out);
}

dblast_status dblast_draft_and_verify(const dblast_head* h, const dblast_block_args* a,
                                      dblast_draft_out* dout, dblast_verify_out* vout, void* ws,
                                      size_t ws_bytes, dblast_stream_t stream) {
  NvtxRange nvtx("dblast_draft_and_verify");
  dblast_status st = check_head(h, true);
  if (st == DBLAST_OK) st = check_args(h, a);
  if (st != DBLAST_OK) return st;
  if (!vout || !vout->target || !aligned16(vout->target)) return DBLAST_ERR_INVALID_ARG;
  st = check_filter(h, vout);
  if (st != DBLAST_OK) return st;
  StepCtx c;
  st = make_ctx(h, a, ws, ws_bytes, vout->has_bonus ? 1 : 0, stream, &c);
  if (st != DBLAST_OK) return st;
  return step_impl(c, dout, vout);
}

dblast_status dblast_device_status(void* ws, dblast_stream_t stream) {
  if (!ws) return DBLAST_ERR_INVALID_ARG;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  DevStatus hs{};
  cudaError_t e = cudaMemcpyAsync(&hs, ws, sizeof(hs), cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_status(e);
  if (hs.timeout || hs.bounds) {
    e = cudaMemsetAsync(ws, 0, sizeof(DevStatus), s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_status(e);
    return hs.timeout ? DBLAST_ERR_TIMEOUT : DBLAST_ERR_BOUNDS;
  }
  return DBLAST_OK;
}

void dblast_set_wait_limit(uint32_t spins) { g_wait_limit = spins; }

void dblast_set_checks(int enable) { g_checks.store(enable ? 1 : 0, std::memory_order_relaxed); }

void dblast_stats_reset(int enable_pass_timing) {
  std::lock_guard<std::mutex> lk(g_stats_mu);
  g_launches = 0;
  g_calls = 0;
  g_tc_launches = 0;
  g_n_ev[0] = g_n_ev[1] = 0;
  g_seen[0] = g_seen[1] = 0;
  g_open[0] = g_open[1] = false;
  g_period = enable_pass_timing > 0 ? enable_pass_timing : 0;
}

dblast_status dblast_stats_get(dblast_stats* out) {
  if (!out) return DBLAST_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> lk(g_stats_mu);
  out->calls = g_calls.load();
  out->kernel_launches = g_launches.load();
  out->tc_launches = g_tc_launches.load();
  double ms[2] = {0.0, 0.0};
  for (int w = 0; w < 2; ++w) {
    for (int i = 0; i < g_n_ev[w]; ++i) {
      cudaError_t e = cudaEventSynchronize(g_ev[w][2 * i + 1]);
      float t = 0.f;
      if (e == cudaSuccess) e = cudaEventElapsedTime(&t, g_ev[w][2 * i], g_ev[w][2 * i + 1]);
      if (e != cudaSuccess) return cuda_status(e);
      ms[w] += t;
    }
  }
  out->timed_draft = (uint64_t)g_n_ev[0];
  out->timed_verify = (uint64_t)g_n_ev[1];
  out->draft_pass_ms = ms[0];
  out->verify_pass_ms = ms[1];
  return DBLAST_OK;
}

dblast_status dblast_al_objective(const dblast_head* h, const dblast_block_args* a,
                                  const dblast_al_args* al, void* ws, size_t ws_bytes,
                                  dblast_stream_t stream) {
  NvtxRange nvtx("dblast_al_objective");
  dblast_status st = check_head(h, true);
  if (st == DBLAST_OK) st = check_args(h, a);
  if (st != DBLAST_OK) return st;
  if (!al || !al->tokens || !al->target || !aligned16(al->target)) return DBLAST_ERR_INVALID_ARG;
  if (a->mode != DBLAST_MODE_SOFT || !(al->tau >= 0.f) || al->tau == INFINITY)
    return DBLAST_ERR_INVALID_ARG;
  dblast_verify_out vo{};
  vo.target = al->target;
  vo.has_bonus = al->has_bonus ? 1 : 0;
  vo.top_k = al->top_k;
  vo.top_p = al->top_p;
  st = check_filter(h, &vo);
  if (st != DBLAST_OK) return st;
  StepCtx c;
  st = make_ctx(h, a, ws, ws_bytes, vo.has_bonus, stream, &c);
  if (st != DBLAST_OK) return st;
  c.target = al->target;
  c.Bt = a->B + vo.has_bonus;
  g_calls.fetch_add(1, std::memory_order_relaxed);
  // the tie words and draft-token counters start in the launch that computes
  // the prior (no memset: it would end the chain of dependent launches)
  cudaError_t e = dbg(launch_codes(c), "codes", c.stream);
  if (e == cudaSuccess)
    e = dbg(c.tc ? launch_draft_pass_tc(c) : launch_draft_pass_simt(c), "draft_pass", c.stream);
  if (e == cudaSuccess) e = dbg(launch_draft_finalize(c, nullptr, al->tokens), "draft_finalize", c.stream);
  if (e == cudaSuccess) e = dbg(launch_target_stats(c, &vo), "target_stats", c.stream);
  const bool filtered = filter_on(h, &vo);
  if (e == cudaSuccess && filtered) {
    const dblast_verify_out f = filter_args(h, &vo);
    e = dbg(launch_target_filter(c, &f), "target_filter", c.stream);
  }
  if (e == cudaSuccess) e = dbg(launch_al_objective(c, al, filtered), "al_objective", c.stream);
  return cuda_status(e);
}

// Workspace of dblast_target_determinism: the target statistics of the
// N x rows target rows (tile records, log-sum-exp, collision probability) and
// p_i(x_i^(m)) of every sample.
struct DetLayout {
  size_t off_partt, off_lt2, off_coll, off_pval, total;
  int nt, Rt;
};
static DetLayout det_layout(int N, int rows, int b, int V, int M) {
  DetLayout d{};
  d.nt = ceil_div(V, TILE_V);
  d.Rt = N * rows;
  size_t o = 0;
  auto take = [&](size_t bytes) {
    size_t at = o;
    o = align_up(o + bytes, 256);
    return at;
  };
  d.off_partt = take((size_t)d.nt * d.Rt * sizeof(float2));
  d.off_lt2 = take((size_t)d.Rt * sizeof(float2));
  d.off_coll = take((size_t)d.Rt * sizeof(float));
  d.off_pval = take((size_t)N * (M > 0 ? M : 1) * b * sizeof(float));
  d.total = o;
  return d;
}

size_t dblast_determinism_workspace_bytes(int N, int rows, int b, int V, int M) {
  if (N < 1 || rows < 1 || b < 1 || V < 1 || M < 0) return 0;
  return det_layout(N, rows, b, V, M).total;
}

dblast_status dblast_target_determinism(const void* target, dblast_dtype dtype, int N, int rows,
                                        int b, int V, float temperature, int M, uint64_t seed,
                                        float* collision, float* d_exact, float* d_hat,
                                        int32_t* samples, void* ws, size_t ws_bytes,
                                        dblast_stream_t stream) {
  NvtxRange nvtx("dblast_target_determinism");
  if (!target || !aligned16(target)) return DBLAST_ERR_INVALID_ARG;
  if (dtype != DBLAST_BF16 && dtype != DBLAST_F32) return DBLAST_ERR_INVALID_ARG;
  if (N < 1 || rows < 1 || V < 1 || b < 1 || b > 32 || b > rows || M < 0 || M > (1 << 24))
    return DBLAST_ERR_INVALID_ARG;
  if (!(temperature > 0.f)) return DBLAST_ERR_INVALID_ARG;
  if ((d_hat || samples) && M < 1) return DBLAST_ERR_INVALID_ARG;
  if ((long long)N * rows > (1LL << 24)) return DBLAST_ERR_INVALID_ARG;
  const DetLayout d = det_layout(N, rows, b, V, M);
  if (!ws || !aligned16(ws) || ws_bytes < d.total) return DBLAST_ERR_WORKSPACE;
  dblast_head h{};
  h.V = V;
  h.dtype = dtype;
  dblast_block_args a{};
  a.N = N;
  a.B = rows - 1;  // the target-statistics kernels index rows as n (B + 1) + i
  StepCtx c{};
  c.head = &h;
  c.args = &a;
  c.wl.N = N;
  c.wl.B = rows - 1;
  c.wl.V = V;
  c.wl.nt = d.nt;
  c.wl.Rt = d.Rt;
  c.wl.off_partt = d.off_partt;
  c.wl.off_lt2 = d.off_lt2;
  c.wl.off_coll = d.off_coll;
  c.ws = static_cast<unsigned char*>(ws);
  c.stream = reinterpret_cast<cudaStream_t>(stream);
  c.k2 = LOG2E / temperature;
  c.Bt = rows;
  dblast_verify_out o{};
  o.target = target;
  o.has_bonus = 1;
  g_calls.fetch_add(1, std::memory_order_relaxed);
  return cuda_status(dbg(launch_determinism(c, &o, rows, b, M, seed, collision, d_exact, d_hat,
                                            samples, d.off_pval),
                         "determinism", c.stream));
}

const char* dblast_status_string(dblast_status s) {
  switch (s) {
    case DBLAST_OK: return "ok";
    case DBLAST_ERR_INVALID_ARG: return "invalid argument";
    case DBLAST_ERR_UNSUPPORTED: return "unsupported shape or dtype for the requested implementation";
    case DBLAST_ERR_WORKSPACE: return "prep or workspace buffer too small or misaligned";
    case DBLAST_ERR_CUDA: return "CUDA runtime error";
    case DBLAST_ERR_TIMEOUT: return "device-side wait ran out";
    case DBLAST_ERR_NO_DEVICE: return "no usable device";
    case DBLAST_ERR_BOUNDS: return "a device-side index check failed";
  }
  return "unknown status";
}

const char* dblast_version(void) { return "dblast 0.1 (sm_103a)"; }

}  // extern "C"
