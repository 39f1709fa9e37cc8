// Internal declarations shared by the CUDA translation units of libdblast.
// Layouts of the prep buffer and the workspace, device helpers (Philox,
// reductions, the (max, sum) log-sum-exp pairs) and the kernel launchers.
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/dblast.h"

namespace dblast {

// vocabulary tile of every partial reduction (log-sum-exp pairs, overlap and
// residual masses): each tile of TILE_V consecutive tokens gets one record.
constexpr int TILE_V = 128;
constexpr int MTILE = 128;  // rows (positions) per tensor-core tile
constexpr float LOG2E = 1.4426950408889634f;
constexpr float LN2 = 0.6931471805599453f;
constexpr float TIE_TOL = 1e-6f;
// greedy-branch mode: an argmax whose top-two logit gap is below this is
// reported as a tie (the logits are formed in fp32, within about 1e-5 of the
// exact values at the Qwen3 shapes)
constexpr float GREEDY_TIE_TOL = 1e-4f;

enum TieBits : uint32_t {
  TIE_ZHAT = 1u, TIE_DRAFT = 2u, TIE_ACCEPT = 4u, TIE_RESID = 8u, TIE_RMASS = 16u, TIE_TOPP = 32u,
  TIE_TAU = 64u
};
// "Near" bits (the tie bit of the same kind, shifted): the decision is within
// TIE_TOL of its threshold once the kernels' own precision is allowed for.
// The vocabulary-head logits come from fp32 tensor-core accumulation of H
// bf16 products: at H = 4096 they are within 5.7e-6 (RMS, 3.8e-5 at most) of
// the exact values, which moves a draw's CDF by up to about 1e-5 of the total
// mass and an acceptance ratio p/q by up to about 1e-4 (relative).  A decision
// whose own margin is below TIE_TOL plus these allowances may be a tie.
constexpr uint32_t NEAR_SHIFT = 8u;
constexpr float NEAR_DRAW = 5e-5f;    // probability mass, for every inverse-CDF draw
constexpr float NEAR_ACCEPT = 1e-4f;  // relative to q(x_i|x_<i), for the acceptance test

// target filter (top-k / top-p): at most FILTER_MAX_K kept tokens per row,
// and vocabularies of at most FILTER_MAX_TILES tiles
constexpr int FILTER_MAX_K = 256;
constexpr int FILTER_MAX_TILES = 2048;
constexpr int FILTER_STAGE = 4096;  // candidate tokens staged in shared memory (else read twice)

__host__ __device__ inline int ceil_div(int a, int b) { return (a + b - 1) / b; }
__host__ __device__ inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// ---------------------------------------------------------------- layouts
struct PrepLayout {
  int V, K, rr, rp, KC;    // rr = r + (e != NULL); rp = rr rounded up to 16; KC = K*2*rp
  size_t off_wu, off_wuop, off_sw, off_ut, off_vt, off_status, total;
  // WU   fp32 [V, K, rr]: (W U_z)_v and, if e, (W e_z)_v in column r
  // WUop fp16 [V, KC]   : per z, [hi(rp) | lo(rp)] of WU_z * sw[z]
  // sw   fp32 [K]       : power-of-two scale of WUop's z block
  // ut   bf16 [rows_pad, H]: [U_z | e_z]^T, the A operand of the tensor-core prep
  // vt   bf16 [rows_pad, H]: [V_z | 0]^T, the A operand of the tensor-core codes GEMM
  // status DevStatus      : bounded-wait record of the tensor-core prep
};

// Workspace regions (each 256-byte aligned), with their element types (ff: a
// float pair hi + lo, see FF below):
//   status DevStatus | codes f32 [Mpad,K,rr] | cscale f32 [Mpad,K] | cop f16 [Mpad,KC]
//   zhat i32 [N] | log2pi f32 [N,K] | stash f32 [M,V] | partd float2 [nt,K,Mpad]
//   lsep float4 [LSE_SPLIT,M,K] | lse2, lq2, w2 ff [M,K] | qtok f32 [M] | tok i32 [M]
//   vcz float2 [M,K] | vb0 f32 [M] | partt float2 [nt,Rt] | lt2 ff [Rt]
//   partv float2 [nt,Mpad] | ties u32 [N] then done u32 [N] (rows of a sequence
//   with their draft token: the last one runs the posterior; zeroed per step)
//   xhat i32 [M,K] | cmask u32 [M]   (greedy-branch mode: every branch's greedy
//   token and the consistent-branch set C_i as a bit mask over z)
//   partg f32 [nt,K,Mpad]  (greedy-branch mode: the second-largest logit of
//   every draft record's tile, for the argmax tie report)
//   coll f32 [Rt]  (collision probability sum_v p(v)^2 of every target row)
//   ftok i32 [Rt, FILTER_MAX_K] | fp f32 [Rt, FILTER_MAX_K] | fcnt i32 [Rt] | ftie u32 [Rt]
//   (target filter: kept tokens by index, their filtered probabilities, count, top-p tie)
constexpr int LSE_SPLIT = 2;  // partial merges of the draft records per (m, z) (one wave of blocks)
struct WsLayout {
  int N, B, M, Mpad, K, rr, rp, KC, V, nt, Rt;
  size_t off_status, off_codes, off_cscale, off_cop, off_zhat, off_log2pi, off_stash,
      off_partd, off_lsep, off_lse2, off_lq2, off_w2, off_qtok, off_tok, off_vcz, off_vb0,
      off_partt, off_lt2, off_partv, off_ties, off_xhat, off_cmask, off_coll, off_ftok,
      off_fp, off_fcnt, off_ftie, off_partg, total;
};

PrepLayout prep_layout(int V, int H, int K, int r, bool has_e);
WsLayout ws_layout(int V, int K, int r, bool has_e, int N, int B, int has_bonus);

// device status word at the start of the workspace
// most split-K partials of the per-call codes GEMM (both kernel families)
constexpr int CODES_MAX_SPLIT = 16;

struct DevStatus {
  uint32_t timeout;      // set to 1 by a bounded wait that ran out
  uint32_t where;        // id of the wait that ran out
  uint32_t bounds;       // set to 1 by a failed index check (checks on)
  uint32_t bounds_where; // id of the check that failed
};

// A data-dependent token index, kept inside [0, V) as always; with checks
// on (chk != nullptr) a value outside it is also recorded in the status word
// (no trap: the access that follows uses the clamped index).
__device__ __forceinline__ int checked_token(int x, int V, DevStatus* chk, uint32_t where) {
  if (chk != nullptr && (x < 0 || x >= V)) {
    atomicExch(&chk->bounds, 1u);
    atomicExch(&chk->bounds_where, where);
  }
  return min(max(x, 0), V - 1);
}

// ------------------------------------------------------------- Philox
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int i = 0; i < 10; ++i) {
    const uint32_t hi0 = __umulhi(0xD2511F53u, c.x), lo0 = 0xD2511F53u * c.x;
    const uint32_t hi1 = __umulhi(0xCD9E8D57u, c.z), lo1 = 0xCD9E8D57u * c.z;
    c = make_uint4(hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0);
    k0 += 0x9E3779B9u;
    k1 += 0xBB67AE85u;
  }
  return c;
}

// One decision uniform in (0, 1), exactly representable in fp32.
__device__ __forceinline__ float decision_uniform(uint64_t seed, uint32_t stream, uint32_t round,
                                                  uint32_t seq, uint32_t pos_abs) {
  const uint4 c = make_uint4(0u, pos_abs, seq, (stream << 24) | (round & 0xFFFFFFu));
  const uint4 w = philox4x32_10(c, (uint32_t)seed, (uint32_t)(seed >> 32));
  return ((float)(w.x >> 9) + 0.5f) * 0x1p-23f;
}

// ------------------------------------------------------------- loads
template <typename T> __device__ __forceinline__ float ldf(const T* p);
template <> __device__ __forceinline__ float ldf<float>(const float* p) { return *p; }
template <> __device__ __forceinline__ float ldf<__nv_bfloat16>(const __nv_bfloat16* p) {
  return __bfloat162float(*p);
}

// 8 consecutive values of a row starting at v0 (v0 % 8 == 0), -inf past V.
// `vec` (16-byte aligned rows, V % 8 == 0): one unconditional load from an
// in-bounds offset, then a select, so loads of consecutive calls can overlap.
__device__ __forceinline__ void load8(const __nv_bfloat16* row, int v0, int V, bool vec,
                                      float (&x)[8]) {
  if (vec) {
    const bool in = v0 < V;
    const uint4 u = *reinterpret_cast<const uint4*>(row + (in ? v0 : 0));
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float2 f = __bfloat1622float2(h[j]);
      x[2 * j] = in ? f.x : -INFINITY;
      x[2 * j + 1] = in ? f.y : -INFINITY;
    }
  } else {
#pragma unroll
    for (int j = 0; j < 8; ++j) x[j] = (v0 + j < V) ? __bfloat162float(row[v0 + j]) : -INFINITY;
  }
}
__device__ __forceinline__ void load8(const float* row, int v0, int V, bool vec, float (&x)[8]) {
  if (vec) {
    const bool in = v0 < V;
    const float4 a = *reinterpret_cast<const float4*>(row + (in ? v0 : 0));
    const float4 b = *reinterpret_cast<const float4*>(row + (in ? v0 : 0) + 4);
    x[0] = in ? a.x : -INFINITY; x[1] = in ? a.y : -INFINITY;
    x[2] = in ? a.z : -INFINITY; x[3] = in ? a.w : -INFINITY;
    x[4] = in ? b.x : -INFINITY; x[5] = in ? b.y : -INFINITY;
    x[6] = in ? b.z : -INFINITY; x[7] = in ? b.w : -INFINITY;
  } else {
#pragma unroll
    for (int j = 0; j < 8; ++j) x[j] = (v0 + j < V) ? row[v0 + j] : -INFINITY;
  }
}

// ------------------------------------------------- (max, sum) pairs in base 2
// A pair (m, s) stands for s * 2^m; the empty pair is (-inf, 0).
__device__ __forceinline__ float2 lse_merge(float2 a, float2 b) {
  const float m = fmaxf(a.x, b.x);
  if (m == -INFINITY) return make_float2(-INFINITY, 0.f);
  return make_float2(m, a.y * exp2f(a.x - m) + b.y * exp2f(b.x - m));
}

__device__ __forceinline__ float2 warp_lse_merge(float2 p) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    float2 q;
    q.x = __shfl_xor_sync(0xffffffffu, p.x, o);
    q.y = __shfl_xor_sync(0xffffffffu, p.y, o);
    p = lse_merge(p, q);
  }
  return p;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ double warp_sum_d(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
// ------------------------------------------------------------ float-float
// This GPU issues double-precision arithmetic at a small fraction of the fp32
// rate and with long latency, so the device path carries extended precision
// as an unevaluated pair of floats (TwoSum / TwoProd, about 44 significant
// bits) and never uses doubles.
struct FF {
  float hi, lo;  // value hi + lo, |lo| <= ulp(hi) / 2
};
__device__ __forceinline__ FF ff_add(FF a, FF b) {
  const float s = a.hi + b.hi;
  const float bb = s - a.hi;
  const float e = ((a.hi - (s - bb)) + (b.hi - bb)) + (a.lo + b.lo);
  const float hi = s + e;
  return FF{hi, e - (hi - s)};
}
__device__ __forceinline__ FF ff_neg(FF a) { return FF{-a.hi, -a.lo}; }
__device__ __forceinline__ FF ff_sub(FF a, FF b) { return ff_add(a, ff_neg(b)); }
__device__ __forceinline__ FF ff_addf(FF a, float b) { return ff_add(a, FF{b, 0.f}); }
// exact product of two floats as a pair
__device__ __forceinline__ FF ff_prod(float a, float b) {
  const float p = a * b;
  return FF{p, fmaf(a, b, -p)};
}
__device__ __forceinline__ FF ff_mulf(FF a, float b) {
  const float p = a.hi * b;
  const float e = fmaf(a.hi, b, -p) + a.lo * b;
  const float hi = p + e;
  return FF{hi, e - (hi - p)};
}
__device__ __forceinline__ bool ff_gt(FF a, FF b) {
  return a.hi > b.hi || (a.hi == b.hi && a.lo > b.lo);
}
__device__ __forceinline__ float ff_f(FF a) { return a.hi + a.lo; }
__device__ __forceinline__ FF ff_ld(const float2* p) {
  const float2 v = *p;
  return FF{v.x, v.y};
}
__device__ __forceinline__ float2 ff_st(FF a) { return make_float2(a.hi, a.lo); }
// 2^a: exp2f of the high part times the first-order factor of the low part
__device__ __forceinline__ float ff_exp2(FF a) { return exp2f(a.hi) * fmaf(a.lo, LN2, 1.f); }
// log2 of a positive pair: exact binary exponent, log2f of the mantissa in
// [1, 2) (absolute error about 1e-7), and a first-order term for lo / hi
__device__ __forceinline__ FF ff_log2(FF a) {
  if (!(a.hi > 0.f)) return FF{-INFINITY, 0.f};
  if (a.hi == INFINITY) return FF{INFINITY, 0.f};
  float x = a.hi;
  int bias = 0;
  if (x < 0x1p-100f) {
    x *= 0x1p64f;
    bias = 64;
  }
  const unsigned b = __float_as_uint(x);
  const int e = (int)((b >> 23) & 0xffu) - 127 - bias;
  const float m = __uint_as_float((b & 0x7fffffu) | 0x3f800000u);
  return ff_add(FF{(float)e, 0.f}, FF{log2f(m) + (a.lo / a.hi) * LOG2E, 0.f});
}

// ------------------------------------------------------------ launchers
struct StepCtx {
  const dblast_head* head;
  const dblast_block_args* args;
  PrepLayout pl;
  WsLayout wl;
  unsigned char* ws;
  const unsigned char* prep;
  cudaStream_t stream;
  float k2;  // log2(e) / T
  bool has_e;
  bool tc;   // tensor-core passes
  bool greedy;  // greedy-branch mode (App. A) instead of sampled draft tokens
  const void* target;  // verify only: [N, Bt, V]
  int Bt;              // target rows per sequence (B + has_bonus)
  bool fuse_tstats;    // fused step: the draft pass computes the target statistics
  float* lse_target;   // its natural log-sum-exp output (or null)
  DevStatus* chk;      // index checks on: the workspace status word, else null
};

template <typename T> T* wsp(const StepCtx& c, size_t off) { return reinterpret_cast<T*>(c.ws + off); }
template <typename T> const T* prp(const StepCtx& c, size_t off) {
  return reinterpret_cast<const T*>(c.prep + off);
}

// measurement hooks (dblast_api.cu)
void count_launches(int n);
void count_tc_launch();
// Process-unique id of the calling thread's current CUDA context (0 when the
// driver cannot tell).  Per-device caches of device addresses, streams and
// kernel attributes compare it with the id they were made under: after a
// cudaDeviceReset the device gets a new context and they are made again.
unsigned long long current_context_id();
// with DBLAST_DEBUG_SYNC=1: synchronise and report the kernel just launched
void debug_kernel(const char* name, cudaStream_t s);

// Programmatic dependent launch: a kernel launched this way may be scheduled
// while the previous kernel of the stream is still finishing (its blocks
// fill the SMs that kernel's blocks leave), and must run griddep_wait()
// before it touches memory that kernel writes.  In a kernel launched the
// ordinary way griddep_wait() returns at once.
__device__ __forceinline__ void griddep_wait() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}
template <typename... KArgs, typename... Args>
inline cudaError_t launch_dep(void (*k)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t s, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, k, static_cast<KArgs>(args)...);
}
void pass_event_begin(int which, cudaStream_t s);  // which: 0 draft pass, 1 verify pass
void pass_event_end(int which, cudaStream_t s);

cudaError_t launch_prep(const dblast_head* head, const PrepLayout& pl, cudaStream_t s);
cudaError_t launch_prep_tc(const dblast_head* head, const PrepLayout& pl, cudaStream_t s);
cudaError_t launch_codes_tc(const StepCtx& c, float* part, int* nsplit);
bool tc_supported(const dblast_head* h);
cudaError_t launch_codes(const StepCtx& c);
cudaError_t launch_draft_pass_simt(const StepCtx& c);
cudaError_t launch_draft_finalize(const StepCtx& c, const dblast_draft_out* out,
                                  const int32_t* given = nullptr);
cudaError_t launch_al_objective(const StepCtx& c, const dblast_al_args* al, bool filtered);
cudaError_t launch_target_stats(const StepCtx& c, const dblast_verify_out* out);
cudaError_t launch_verify_pass_simt(const StepCtx& c);
cudaError_t launch_verify_finalize(const StepCtx& c, const dblast_verify_out* out);
cudaError_t launch_greedy_draft_finalize(const StepCtx& c, const dblast_draft_out* out);
cudaError_t launch_greedy_verify_finalize(const StepCtx& c, const dblast_verify_out* out);
cudaError_t launch_greedy_step_finalize(const StepCtx& c, const dblast_draft_out* dout,
                                        const dblast_verify_out* out);
cudaError_t launch_target_filter(const StepCtx& c, const dblast_verify_out* o);
cudaError_t launch_filtered_verify(const StepCtx& c, const dblast_verify_out* o);
cudaError_t launch_determinism(const StepCtx& c, const dblast_verify_out* o, int rows, int b,
                               int M, uint64_t seed, float* collision, float* d_exact,
                               float* d_hat, int32_t* samples, size_t off_pval);

}  // namespace dblast
