// Once-per-weights preparation (dblast_head_prepare) and the per-call code
// vectors c_{i,z} = V_z^T h_i (Sec. 3.1, Architecture, rank-r expander
// g_z(h) = U_z V_z^T h + e_z), plus the category prior and latent draw.
//
// The factored branch logits are
//     l_{i,z,v} = (W h_i)_v + (W U_z)_v . c_{i,z} + (W e_z)_v + b_v,
// so the head is prepared once as WU = [W U_z | W e_z] (fp32, [V, K, rr]) and
// as split-fp16 operands for the tensor-core correction GEMM: for every z the
// operand row is [hi(rp) | lo(rp)] of WU_z * sw_z, sw_z a power of two that
// brings max|WU_z| near 2^14 (hi + lo carries 22 bits of mantissa).
#include <cstdlib>

#include "dblast_internal.cuh"

namespace dblast {

// C[m][o] = sum_h A[m][h] * Bf(h, o), A row-major [Ma, H]; split-K over gridDim.z
// writes out + z * split_stride.  64x64 tile per CTA, 256 threads, 4x4 per thread.
template <typename Tin, typename BF>
__global__ void __launch_bounds__(256) k_gemm_simt(const Tin* __restrict__ A, int Ma, int H, BF bf,
                                                   int Nb, int hchunk, float* __restrict__ out,
                                                   size_t split_stride) {
  __shared__ float As[64][33];
  __shared__ float Bs[32][65];
  const int m0 = blockIdx.x * 64, o0 = blockIdx.y * 64;
  const int hs = blockIdx.z * hchunk, he = min(H, hs + hchunk);
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  float acc[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
  for (int h0 = hs; h0 < he; h0 += 32) {
    for (int idx = threadIdx.x; idx < 64 * 32; idx += 256) {
      const int r = idx >> 5, c = idx & 31, m = m0 + r, h = h0 + c;
      As[r][c] = (m < Ma && h < he) ? ldf(A + (size_t)m * H + h) : 0.f;
    }
    for (int idx = threadIdx.x; idx < 32 * 64; idx += 256) {
      const int r = idx >> 6, c = idx & 63, h = h0 + r, o = o0 + c;
      Bs[r][c] = (o < Nb && h < he) ? bf(h, o) : 0.f;
    }
    __syncthreads();
#pragma unroll 8
    for (int k = 0; k < 32; ++k) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = As[ty * 4 + i][k];
#pragma unroll
      for (int j = 0; j < 4; ++j) b[j] = Bs[k][tx + 16 * j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
  float* o = out + (size_t)blockIdx.z * split_stride;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int m = m0 + ty * 4 + i;
    if (m >= Ma) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int oc = o0 + tx + 16 * j;
      if (oc < Nb) o[(size_t)m * Nb + oc] = acc[i][j];
    }
  }
}

// B operand of the prep GEMM: column o = z*rr + k holds U[z][h][k] (k < r) or e[z][h] (k == r).
template <typename Tin> struct ExpanderCols {
  const Tin* F;  // [K, H, r]
  const Tin* e;  // [K, H] or nullptr
  int H, r, rr;
  __device__ float operator()(int h, int o) const {
    const int z = o / rr, k = o - z * rr;
    if (k < r) return ldf(F + ((size_t)z * H + h) * r + k);
    return e ? ldf(e + (size_t)z * H + h) : 0.f;
  }
};

__device__ __forceinline__ float pow2_scale_for(float amax) {
  if (!(amax > 0.f)) return 1.f;
  int E;
  frexpf(amax, &E);  // amax = f 2^E, f in [0.5, 1)
  return ldexpf(1.f, 14 - E);
}

// per-z max |WU| (as ordered uint bits of non-negative floats)
__global__ void k_prep_amax(const float* __restrict__ wu, int V, int K, int rr,
                            unsigned* __restrict__ amax_bits) {
  __shared__ unsigned sm[32];
  if (threadIdx.x < 32) sm[threadIdx.x] = 0u;
  __syncthreads();
  const size_t n = (size_t)V * K * rr;
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n;
       i += (size_t)gridDim.x * blockDim.x) {
    const int z = (int)((i / rr) % K);
    atomicMax(&sm[z], __float_as_uint(fabsf(wu[i])));
  }
  __syncthreads();
  if (threadIdx.x < K) atomicMax(&amax_bits[threadIdx.x], sm[threadIdx.x]);
}

// split WU_z * sw_z into fp16 hi/lo planes: WUop[v][z*2rp + k] = hi, [.. + rp + k] = lo
__global__ void k_prep_split(const float* __restrict__ wu, int V, int K, int rr, int rp,
                             const unsigned* __restrict__ amax_bits, __half* __restrict__ wuop) {
  const size_t n = (size_t)V * K * rp;
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n;
       i += (size_t)gridDim.x * blockDim.x) {
    const int k = (int)(i % rp);
    const int z = (int)((i / rp) % K);
    const size_t v = i / ((size_t)rp * K);
    const float s = pow2_scale_for(__uint_as_float(amax_bits[z]));
    const float x = (k < rr) ? wu[(v * K + z) * rr + k] * s : 0.f;
    const __half hi = __float2half_rn(x);
    const __half lo = __float2half_rn(x - __half2float(hi));
    __half* row = wuop + v * (size_t)(K * 2 * rp) + (size_t)z * 2 * rp;
    row[k] = hi;
    row[rp + k] = lo;
  }
}

__global__ void k_prep_scale(float* __restrict__ sw, int K) {
  const int z = threadIdx.x;
  if (z < K) sw[z] = pow2_scale_for(__uint_as_float(__float_as_uint(sw[z])));
}

template <typename Tin>
static cudaError_t prep_typed(const dblast_head* h, const PrepLayout& pl, cudaStream_t s) {
  unsigned char* base = static_cast<unsigned char*>(h->prep);
  float* wu = reinterpret_cast<float*>(base + pl.off_wu);
  __half* wuop = reinterpret_cast<__half*>(base + pl.off_wuop);
  float* sw = reinterpret_cast<float*>(base + pl.off_sw);
  const int Nb = h->K * pl.rr;
  ExpanderCols<Tin> bf{static_cast<const Tin*>(h->U), static_cast<const Tin*>(h->e), h->H, h->r,
                       pl.rr};
  cudaError_t e = cudaSuccess;
  const char* force_simt = getenv("DBLAST_PREP_SIMT");  // test hook: compare the two prep GEMMs
  if (tc_supported(h) && !(force_simt && force_simt[0] == '1')) {
    e = launch_prep_tc(h, pl, s);
  } else {
    dim3 grid(ceil_div(h->V, 64), ceil_div(Nb, 64), 1);
    k_gemm_simt<Tin><<<grid, 256, 0, s>>>(static_cast<const Tin*>(h->W), h->V, h->H, bf, Nb,
                                          h->H, wu, 0);
    debug_kernel("k_gemm_simt", s);
    count_launches(1);
    e = cudaGetLastError();
  }
  if (e != cudaSuccess) return e;
  e = cudaMemsetAsync(sw, 0, h->K * sizeof(float), s);
  if (e != cudaSuccess) return e;
  k_prep_amax<<<1024, 256, 0, s>>>(wu, h->V, h->K, pl.rr, reinterpret_cast<unsigned*>(sw));
  debug_kernel("k_prep_amax", s);
  k_prep_split<<<2048, 256, 0, s>>>(wu, h->V, h->K, pl.rr, pl.rp,
                                    reinterpret_cast<const unsigned*>(sw), wuop);
  debug_kernel("k_prep_split", s);
  k_prep_scale<<<1, 32, 0, s>>>(sw, h->K);
  debug_kernel("k_prep_scale", s);
  count_launches(3);
  return cudaGetLastError();
}

cudaError_t launch_prep(const dblast_head* h, const PrepLayout& pl, cudaStream_t s) {
  return h->dtype == DBLAST_F32 ? prep_typed<float>(h, pl, s) : prep_typed<__nv_bfloat16>(h, pl, s);
}

// ------------------------------------------------------------- prior and codes
// Prior of sequence n, run by one block of 256 threads: l = Wp a + bp (a warp
// per category, 16-byte loads), then warp 0 with lane z: pi = softmax(l / Z_T)
// (Z_T = 0: one-hot argmax, lowest index on ties) and z-hat by an inverse-CDF
// draw (stream 0).
template <typename Tin>
__device__ __forceinline__ void prior_body(int n, const Tin* __restrict__ Wp,
                                           const float* __restrict__ bp,
                                           const Tin* __restrict__ anchor,
                                           const Tin* __restrict__ hidden, int H, int K, int B,
                                           float zt, uint64_t seed,
                                           const int64_t* __restrict__ pos,
                                           const uint32_t* __restrict__ rnd,
                                           int32_t* __restrict__ zhat_ws,
                                           float* __restrict__ log2pi_ws,
                                           uint32_t* __restrict__ ties, uint32_t* __restrict__ done,
                                           float* ell) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const Tin* a = anchor ? anchor + (size_t)n * H : hidden + (size_t)n * B * H;
  for (int z = warp; z < K; z += blockDim.x >> 5) {
    const Tin* w = Wp + (size_t)z * H;
    float acc = 0.f;
#pragma unroll 4
    for (int h0 = lane * 8; h0 < H; h0 += 256) {
      float w8[8], a8[8];
      load8(w, h0, H, true, w8);
      load8(a, h0, H, true, a8);
#pragma unroll
      for (int j = 0; j < 8; ++j) acc = fmaf(w8[j], a8[j], acc);
    }
    acc = warp_sum(acc);
    if (lane == 0) ell[z] = acc + (bp ? bp[z] : 0.f);
  }
  __syncthreads();
  if (warp != 0) return;
  const bool on = lane < K;
  const float lz = on ? ell[lane] : -INFINITY;
  float pz;
  if (zt == 0.f) {
    float best = lz;
    int bi = on ? lane : 32;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float ob = __shfl_xor_sync(0xffffffffu, best, o);
      const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
      if (ob > best || (ob == best && oi < bi)) {
        best = ob;
        bi = oi;
      }
    }
    pz = (lane == bi) ? 1.f : 0.f;
  } else {
    const float x = on ? lz / zt : -INFINITY;
    const float mx = warp_max(x);
    const float e = on ? exp2f((x - mx) * LOG2E) : 0.f;
    pz = e / warp_sum(e);
  }
  // inverse CDF over the categories in index order (float-pair prefix sums)
  const float u = decision_uniform(seed, 0u, rnd[n], (uint32_t)n, (uint32_t)pos[n]);
  FF cum{pz, 0.f};
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const FF t{__shfl_up_sync(0xffffffffu, cum.hi, o), __shfl_up_sync(0xffffffffu, cum.lo, o)};
    if (lane >= o) cum = ff_add(t, cum);
  }
  const FF tot{__shfl_sync(0xffffffffu, cum.hi, 31), __shfl_sync(0xffffffffu, cum.lo, 31)};
  const FF target = ff_mulf(tot, u);
  const unsigned hit = __ballot_sync(0xffffffffu, on && ff_gt(cum, target));
  const unsigned posm = __ballot_sync(0xffffffffu, on && pz > 0.f);
  int zh;
  float margin = 0.f;
  if (hit) {
    zh = __ffs(hit) - 1;
    const FF c{__shfl_sync(0xffffffffu, cum.hi, zh), __shfl_sync(0xffffffffu, cum.lo, zh)};
    const float p = __shfl_sync(0xffffffffu, pz, zh);
    margin = fminf(ff_f(ff_sub(target, ff_addf(c, -p))), ff_f(ff_sub(c, target))) / ff_f(tot);
  } else {
    zh = posm ? 31 - __clz(posm) : 0;
  }
  if (lane == 0) {
    // this call's tie word of the sequence starts here (the kernels after
    // this one add their bits), and so does the draft-token block counter
    uint32_t bits = 0u;
    if (zt != 0.f && margin < TIE_TOL) bits |= TIE_ZHAT;
    if (zt != 0.f && margin < TIE_TOL + NEAR_DRAW) bits |= TIE_ZHAT << NEAR_SHIFT;
    ties[n] = bits;
    done[n] = 0u;
    zhat_ws[n] = zh;
  }
  if (on) log2pi_ws[n * K + lane] = pz > 0.f ? log2f(pz) : -INFINITY;
}

// Deterministic split-K reduction of the codes of one (m, z) by one warp, the
// constant code for e, the per-(m, z) power-of-two scale and the split-fp16
// operand rows.
__device__ __forceinline__ void codes_finish_warp(int gw, int lane, const float* __restrict__ part,
                                                  int nsplit, int M, int Mpad, int K, int r,
                                                  int rr, int rp, bool has_e,
                                                  float* __restrict__ codes,
                                                  float* __restrict__ cscale,
                                                  __half* __restrict__ cop) {
  if (gw >= Mpad * K) return;
  const int m = gw / K, z = gw - m * K;
  const int Nb = K * rr;
  float c[3];
  float amax = 0.f;
#pragma unroll
  for (int j = 0; j < 3; ++j) {
    const int k = lane + 32 * j;
    float v = 0.f;
    if (k < rr && m < M) {
      if (k < r) {
        for (int s = 0; s < nsplit; ++s) v += part[((size_t)s * M + m) * Nb + z * rr + k];
      } else if (has_e) {
        v = 1.f;
      }
    }
    c[j] = v;
    amax = fmaxf(amax, fabsf(v));
    if (k < rr) codes[((size_t)m * K + z) * rr + k] = v;
  }
  amax = warp_max(amax);
  const float sc = pow2_scale_for(amax);
  if (lane == 0) cscale[(size_t)m * K + z] = sc;
  __half* row = cop + (size_t)m * K * 2 * rp + (size_t)z * 2 * rp;
#pragma unroll
  for (int j = 0; j < 3; ++j) {
    const int k = lane + 32 * j;
    if (k < rp) {
      const float x = c[j] * sc;
      const __half hi = __float2half_rn(x);
      row[k] = hi;
      row[rp + k] = __float2half_rn(x - __half2float(hi));
    }
  }
}

// One launch after the codes GEMM: blocks [0, nfin) reduce the codes (a warp
// per (m, z)), blocks nfin + n compute the prior of sequence n.  The prior
// reads the positions and round counters that the previous step's
// verify-final kernel wrote, so it too waits for the preceding grids.
struct PriorArgs {
  const void* Wp;
  const float* bp;
  const void* anchor;
  const void* hidden;
  int H, K, B;
  float zt;
  uint64_t seed;
  const int64_t* pos;
  const uint32_t* rnd;
  int32_t* zhat;
  float* log2pi;
  uint32_t* ties;
  uint32_t* done;  // draft-token block counters [N]
};
template <typename Tin>
__global__ void __launch_bounds__(256)
    k_codes_prior(const float* __restrict__ part, int nsplit, int M, int Mpad, int K, int r,
                  int rr, int rp, bool has_e, float* __restrict__ codes,
                  float* __restrict__ cscale, __half* __restrict__ cop, int nfin,
                  const PriorArgs pa) {
  griddep_wait();  // launched as a dependent of the codes GEMM
  __shared__ float ell[32];
  if ((int)blockIdx.x < nfin) {
    const int gw = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    codes_finish_warp(gw, threadIdx.x & 31, part, nsplit, M, Mpad, K, r, rr, rp, has_e, codes,
                      cscale, cop);
    return;
  }
  prior_body<Tin>((int)blockIdx.x - nfin, static_cast<const Tin*>(pa.Wp), pa.bp,
                  static_cast<const Tin*>(pa.anchor), static_cast<const Tin*>(pa.hidden), pa.H,
                  pa.K, pa.B, pa.zt, pa.seed, pa.pos, pa.rnd, pa.zhat, pa.log2pi, pa.ties, pa.done,
                  ell);
}

template <typename Tin> static cudaError_t codes_typed(const StepCtx& c) {
  const dblast_head* h = c.head;
  const dblast_block_args* a = c.args;
  const WsLayout& w = c.wl;
  cudaStream_t s = c.stream;
  // codes: split-K partials go to the stash region (not yet written by this call)
  const int Nb = h->K * w.rr;
  float* part = wsp<float>(c, w.off_stash);
  int nsplit = 1;
  if (c.tc) {
    cudaError_t e = launch_codes_tc(c, part, &nsplit);
    if (e != cudaSuccess) return e;
  } else {
    nsplit = max(1, min(CODES_MAX_SPLIT, h->H / 256));
    const int hchunk = ceil_div(ceil_div(h->H, nsplit), 32) * 32;
    ExpanderCols<Tin> bf{static_cast<const Tin*>(h->Vf), nullptr, h->H, h->r, w.rr};
    dim3 grid(ceil_div(w.M, 64), ceil_div(Nb, 64), ceil_div(h->H, hchunk));
    k_gemm_simt<Tin><<<grid, 256, 0, s>>>(static_cast<const Tin*>(a->hidden), w.M, h->H, bf, Nb,
                                          hchunk, part, (size_t)w.M * Nb);
    debug_kernel("k_gemm_simt", s);
    count_launches(1);
    nsplit = (int)grid.z;
  }
  const int warps = w.Mpad * h->K;
  const int nfin = ceil_div(warps * 32, 256);
  const PriorArgs pa{h->Wp, h->bp, a->anchor, a->hidden, h->H, h->K, a->B, a->z_temperature,
                     a->seed, a->pos, a->round, wsp<int32_t>(c, w.off_zhat),
                     wsp<float>(c, w.off_log2pi), wsp<uint32_t>(c, w.off_ties),
                     wsp<uint32_t>(c, w.off_ties) + w.N};
  cudaError_t le = launch_dep(
      k_codes_prior<Tin>, dim3(nfin + a->N), dim3(256), 0, s, part, nsplit, w.M, w.Mpad, h->K,
      h->r, w.rr, w.rp, c.has_e, wsp<float>(c, w.off_codes), wsp<float>(c, w.off_cscale),
      wsp<__half>(c, w.off_cop), nfin, pa);
  debug_kernel("k_codes_prior", s);
  count_launches(1);
  return le != cudaSuccess ? le : cudaGetLastError();
}

cudaError_t launch_codes(const StepCtx& c) {
  return c.head->dtype == DBLAST_F32 ? codes_typed<float>(c) : codes_typed<__nv_bfloat16>(c);
}

}  // namespace dblast
