// Vocabulary-wide passes on CUDA cores (any dtype / shape): the draft pass
// (stash = W h + b and per-tile (max, sum) records of every branch) and the
// verify pass (per-tile sum min(p, q) and residual mass).  They write the same
// records as the tensor-core passes; the finalize kernels merge them.
#include "dblast_internal.cuh"

namespace dblast {

constexpr int RB = 16;  // rows (positions) per CTA of the CUDA-core passes

// ---------------------------------------------------------------------------
// draft pass on CUDA cores: stash = W h + b; partd per (tile, z, row).
// Greedy-branch mode: no stash, and the records hold (max logit, its token)
// with ties to the lowest index (the token's bits stored in the float), plus
// the tile's second-largest logit in partg.
// (max, token) merge, ties to the lower token, carrying the second-largest
// values sa, sb of both sides
__device__ __forceinline__ void arg_merge2s(float2& a, float& sa, float2 b, float sb) {
  const int ia = __float_as_int(a.y), ib = __float_as_int(b.y);
  if (b.x > a.x || (b.x == a.x && ib < ia)) {
    sa = fmaxf(a.x, sb);
    a = b;
  } else {
    sa = fmaxf(sa, b.x);
  }
}
template <typename Tin>
__global__ void __launch_bounds__(TILE_V)
    k_draft_simt(const Tin* __restrict__ W, const Tin* __restrict__ hid,
                 const float* __restrict__ vbias, const float* __restrict__ wu,
                 const float* __restrict__ codes, int V, int H, int K, int rr, int M, int Mpad,
                 float k2, bool greedy, float* __restrict__ stash, float2* __restrict__ partd,
                 float* __restrict__ partg) {
  extern __shared__ float smem[];
  float* hs = smem;                    // [RB][64]
  float* cs = smem + RB * 64;          // [K*rr]
  float2* red = reinterpret_cast<float2*>(cs + 32 * 65);  // [RB*K][4] (8-byte aligned offset)
  float* redg = reinterpret_cast<float*>(red + RB * 32 * 4);  // [RB*K][4] greedy seconds
  const int t = blockIdx.x, m0 = blockIdx.y * RB, tid = threadIdx.x;
  const int lane = tid & 31, warp = tid >> 5;
  const int v = t * TILE_V + tid;
  const bool vok = v < V;
  float acc[RB];
#pragma unroll
  for (int r = 0; r < RB; ++r) acc[r] = 0.f;
  for (int h0 = 0; h0 < H; h0 += 64) {
    for (int idx = tid; idx < RB * 64; idx += TILE_V) {
      const int r = idx >> 6, c = idx & 63, m = m0 + r, hh = h0 + c;
      hs[idx] = (m < M && hh < H) ? ldf(hid + (size_t)m * H + hh) : 0.f;
    }
    __syncthreads();
    if (vok) {
      const int hend = min(64, H - h0);
      for (int c = 0; c < hend; ++c) {
        const float w = ldf(W + (size_t)v * H + h0 + c);
#pragma unroll
        for (int r = 0; r < RB; ++r) acc[r] = fmaf(w, hs[r * 64 + c], acc[r]);
      }
    }
    __syncthreads();
  }
  const float b = (vok && vbias) ? vbias[v] : 0.f;
  for (int r = 0; r < RB; ++r) {
    const int m = m0 + r;
    if (m >= M) break;  // uniform over the block
    const float base = acc[r] + b;
    if (vok && !greedy) stash[(size_t)m * V + v] = base;
    for (int idx = tid; idx < K * rr; idx += TILE_V) cs[idx] = codes[(size_t)m * K * rr + idx];
    __syncthreads();
    for (int z = 0; z < K; ++z) {
      float2 p = greedy ? make_float2(-INFINITY, __int_as_float(0x7fffffff))
                        : make_float2(-INFINITY, 0.f);
      float sg = -INFINITY;  // greedy: second-largest logit of the merged lanes
      if (vok) {
        float corr = 0.f;
        const float* wr = wu + ((size_t)v * K + z) * rr;
        for (int k = 0; k < rr; ++k) corr = fmaf(wr[k], cs[z * rr + k], corr);
        p = greedy ? make_float2(base + corr, __int_as_float(v)) : make_float2((base + corr) * k2, 1.f);
      }
      if (greedy) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
          const float2 q = make_float2(__shfl_xor_sync(0xffffffffu, p.x, o),
                                       __shfl_xor_sync(0xffffffffu, p.y, o));
          const float qs = __shfl_xor_sync(0xffffffffu, sg, o);
          arg_merge2s(p, sg, q, qs);
        }
      } else {
        p = warp_lse_merge(p);
      }
      if (lane == 0) {
        red[(r * K + z) * 4 + warp] = p;
        redg[(r * K + z) * 4 + warp] = sg;
      }
    }
    __syncthreads();
  }
  for (int idx = tid; idx < RB * K; idx += TILE_V) {
    const int r = idx / K, z = idx - r * K, m = m0 + r;
    if (m >= M) continue;
    float2 p = red[idx * 4];
    float sg = redg[idx * 4];
    for (int j = 1; j < 4; ++j) {
      if (greedy) arg_merge2s(p, sg, red[idx * 4 + j], redg[idx * 4 + j]);
      else p = lse_merge(p, red[idx * 4 + j]);
    }
    partd[((size_t)t * K + z) * Mpad + m] = p;
    if (greedy) partg[((size_t)t * K + z) * Mpad + m] = sg;
  }
}

template <typename Tin> static cudaError_t draft_simt_typed(const StepCtx& c) {
  const dblast_head* h = c.head;
  const WsLayout& w = c.wl;
  dim3 grid(w.nt, ceil_div(w.M, RB));
  const size_t smem = (RB * 64 + 32 * 65) * sizeof(float) + RB * 32 * 4 * sizeof(float2) +
                      RB * 32 * 4 * sizeof(float);
  k_draft_simt<Tin><<<grid, TILE_V, smem, c.stream>>>(
      static_cast<const Tin*>(h->W), static_cast<const Tin*>(c.args->hidden), h->vbias,
      prp<float>(c, c.pl.off_wu), wsp<float>(c, w.off_codes), h->V, h->H, h->K, w.rr, w.M,
      w.Mpad, c.k2, c.greedy, wsp<float>(c, w.off_stash), wsp<float2>(c, w.off_partd),
      wsp<float>(c, w.off_partg));
  debug_kernel("k_draft_simt", c.stream);
  count_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_draft_pass_simt(const StepCtx& c) {
  return c.head->dtype == DBLAST_F32 ? draft_simt_typed<float>(c)
                                     : draft_simt_typed<__nv_bfloat16>(c);
}

// ---------------------------------------------------------------------------
// verify pass on CUDA cores: partv[t][m] = (sum min(p, q), sum [p - q]_+)
template <typename Tin>
__global__ void __launch_bounds__(TILE_V)
    k_verify_simt(const Tin* __restrict__ target, const float* __restrict__ stash,
                  const float* __restrict__ wu, const float* __restrict__ codes,
                  const float2* __restrict__ lse2, const float2* __restrict__ w2,
                  const float2* __restrict__ lt2, int V, int K, int rr, int B, int Bt, int M,
                  int Mpad, float k2, float2* __restrict__ partv) {
  extern __shared__ float smem[];
  float* cs = smem;                       // [K*rr]
  float* off = cs + 32 * 65;              // [K]: w2 - lse2 (log2 domain)
  float2* red = reinterpret_cast<float2*>(off + 32 + 2);  // [RB][4] (8-byte aligned offset)
  const int t = blockIdx.x, m0 = blockIdx.y * RB, tid = threadIdx.x;
  const int lane = tid & 31, warp = tid >> 5;
  const int v = t * TILE_V + tid;
  const bool vok = v < V;
  for (int r = 0; r < RB; ++r) {
    const int m = m0 + r;
    if (m >= M) break;
    const int n = m / B, i = m - n * B;
    for (int idx = tid; idx < K * rr; idx += TILE_V) cs[idx] = codes[(size_t)m * K * rr + idx];
    if (tid < K) {
      const FF wz = ff_ld(w2 + (size_t)m * K + tid);
      off[tid] = wz.hi == -INFINITY ? -INFINITY : ff_f(ff_sub(wz, ff_ld(lse2 + (size_t)m * K + tid)));
    }
    __syncthreads();
    float2 acc = make_float2(0.f, 0.f);
    if (vok) {
      const float base = stash[(size_t)m * V + v];
      float q = 0.f;
      for (int z = 0; z < K; ++z) {
        const float o = off[z];
        if (o == -INFINITY) continue;
        float corr = 0.f;
        const float* wr = wu + ((size_t)v * K + z) * rr;
        for (int k = 0; k < rr; ++k) corr = fmaf(wr[k], cs[z * rr + k], corr);
        q += exp2f(fmaf(base + corr, k2, o));
      }
      const FF Lt = ff_ld(lt2 + (size_t)n * (B + 1) + i);
      const float p = exp2f(fmaf(ldf(target + ((size_t)n * Bt + i) * V + v), k2, -Lt.hi) - Lt.lo);
      const float mn = fminf(p, q);
      acc = make_float2(mn, p - mn);
    }
    acc.x = warp_sum(acc.x);
    acc.y = warp_sum(acc.y);
    if (lane == 0) red[r * 4 + warp] = acc;
    __syncthreads();
  }
  if (tid < RB && m0 + tid < M) {
    float2 s = red[tid * 4];
    for (int j = 1; j < 4; ++j) {
      s.x += red[tid * 4 + j].x;
      s.y += red[tid * 4 + j].y;
    }
    partv[(size_t)t * Mpad + m0 + tid] = s;
  }
}

template <typename Tin> static cudaError_t verify_simt_typed(const StepCtx& c) {
  const WsLayout& w = c.wl;
  dim3 grid(w.nt, ceil_div(w.M, RB));
  const size_t smem = (32 * 65 + 32 + 2) * sizeof(float) + RB * 4 * sizeof(float2) + 16;
  k_verify_simt<Tin><<<grid, TILE_V, smem, c.stream>>>(
      static_cast<const Tin*>(c.target), wsp<float>(c, w.off_stash), prp<float>(c, c.pl.off_wu),
      wsp<float>(c, w.off_codes), wsp<float2>(c, w.off_lse2), wsp<float2>(c, w.off_w2),
      wsp<float2>(c, w.off_lt2), w.V, c.head->K, w.rr, w.B, c.Bt, w.M, w.Mpad, c.k2,
      wsp<float2>(c, w.off_partv));
  debug_kernel("k_verify_simt", c.stream);
  count_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_verify_pass_simt(const StepCtx& c) {
  return c.head->dtype == DBLAST_F32 ? verify_simt_typed<float>(c)
                                     : verify_simt_typed<__nv_bfloat16>(c);
}

}  // namespace dblast
