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

enum TieBits : uint32_t {
  TIE_ZHAT = 1u, TIE_DRAFT = 2u, TIE_ACCEPT = 4u, TIE_RESID = 8u, TIE_RMASS = 16u
};

__host__ __device__ inline int ceil_div(int a, int b) { return (a + b - 1) / b; }
__host__ __device__ inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// ---------------------------------------------------------------- layouts
struct PrepLayout {
  int V, K, rr, rp, KC;    // rr = r + (e != NULL); rp = rr rounded up to 16; KC = K*2*rp
  size_t off_wu, off_wuop, off_sw, off_ut, off_status, total;
  // WU   fp32 [V, K, rr]: (W U_z)_v and, if e, (W e_z)_v in column r
  // WUop fp16 [V, KC]   : per z, [hi(rp) | lo(rp)] of WU_z * sw[z]
  // sw   fp32 [K]       : power-of-two scale of WUop's z block
  // ut   bf16 [rows_pad, H]: [U_z | e_z]^T, the A operand of the tensor-core prep
  // status DevStatus      : bounded-wait record of the tensor-core prep
};

// Workspace regions (each 256-byte aligned), with their element types:
//   status DevStatus | codes f32 [Mpad,K,rr] | cscale f32 [Mpad,K] | cop f16 [Mpad,KC]
//   zhat i32 [N] | log2pi f32 [N,K] | stash f32 [M,V] | partd float2 [nt,K,Mpad]
//   lse2, lq2, w2 f64 [M,K] | tok i32 [M] | partt float2 [nt,Rt] | lse2t f64 [Rt]
//   partv float2 [nt,Mpad] | av double2 [M] | ties u32 [N]
struct WsLayout {
  int N, B, M, Mpad, K, rr, rp, KC, V, nt, Rt;
  size_t off_status, off_codes, off_cscale, off_cop, off_zhat, off_log2pi, off_stash,
      off_partd, off_lse2, off_lq2, off_w2, off_tok, off_partt, off_lse2t, off_partv,
      off_av, off_ties, total;
};

PrepLayout prep_layout(int V, int H, int K, int r, bool has_e);
WsLayout ws_layout(int V, int K, int r, bool has_e, int N, int B, int has_bonus);

// device status word at the start of the workspace
struct DevStatus {
  uint32_t timeout;      // set to 1 by a bounded wait that ran out
  uint32_t where;        // id of the wait that ran out
};

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
// inclusive prefix sum over lanes
__device__ __forceinline__ double warp_incl_scan_d(double v) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const double t = __shfl_up_sync(0xffffffffu, v, o);
    if (lane >= o) v += t;
  }
  return v;
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
  const void* target;  // verify only: [N, Bt, V]
  int Bt;              // target rows per sequence (B + has_bonus)
};

template <typename T> T* wsp(const StepCtx& c, size_t off) { return reinterpret_cast<T*>(c.ws + off); }
template <typename T> const T* prp(const StepCtx& c, size_t off) {
  return reinterpret_cast<const T*>(c.prep + off);
}

// measurement hooks (dblast_api.cu)
void count_launches(int n);
void count_tc_launch();
// with DBLAST_DEBUG_SYNC=1: synchronise and report the kernel just launched
void debug_kernel(const char* name, cudaStream_t s);
void pass_event_begin(int which, cudaStream_t s);  // which: 0 draft pass, 1 verify pass
void pass_event_end(int which, cudaStream_t s);

cudaError_t launch_prep(const dblast_head* head, const PrepLayout& pl, cudaStream_t s);
cudaError_t launch_prep_tc(const dblast_head* head, const PrepLayout& pl, cudaStream_t s);
bool tc_supported(const dblast_head* h);
cudaError_t launch_prior_codes(const StepCtx& c);
cudaError_t launch_draft_pass_simt(const StepCtx& c);
cudaError_t launch_draft_finalize(const StepCtx& c, const dblast_draft_out* out);
cudaError_t launch_target_stats(const StepCtx& c, const dblast_verify_out* out);
cudaError_t launch_verify_pass_simt(const StepCtx& c);
cudaError_t launch_verify_finalize(const StepCtx& c, const dblast_verify_out* out);

}  // namespace dblast
