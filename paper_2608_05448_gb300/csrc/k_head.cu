// Vocabulary-wide passes on CUDA cores (any dtype / shape), the target
// log-sum-exp pass, and the finalize kernels shared with the tensor-core path.
//
// Partial records per vocabulary tile of TILE_V tokens:
//   draft  : partd[t][z][m] = (m2, s), s * 2^m2 = sum_v 2^{l_{m,z,v} log2(e)/T}
//   target : partt[t][row]  = (m2, s) of the target row t/T
//   verify : partv[t][m]    = (sum_v min(p, q), sum_v [p - q]_+)
// The finalize kernels merge the records in vocabulary order and draw every
// token by an inverse-CDF scan: first over tiles, then inside the chosen tile
// by recomputing its TILE_V values.
#include "dblast_internal.cuh"

namespace dblast {

constexpr int RB = 16;  // rows (positions) per CTA of the CUDA-core passes

// ---------------------------------------------------------------------------
// draft pass on CUDA cores: stash = W h + b; partd per (tile, z, row)
template <typename Tin>
__global__ void __launch_bounds__(TILE_V)
    k_draft_simt(const Tin* __restrict__ W, const Tin* __restrict__ hid,
                 const float* __restrict__ vbias, const float* __restrict__ wu,
                 const float* __restrict__ codes, int V, int H, int K, int rr, int M, int Mpad,
                 float k2, float* __restrict__ stash, float2* __restrict__ partd) {
  extern __shared__ float smem[];
  float* hs = smem;                    // [RB][64]
  float* cs = smem + RB * 64;          // [K*rr]
  float2* red = reinterpret_cast<float2*>(cs + 32 * 65);  // [RB*K][4] (8-byte aligned offset)
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
    if (vok) stash[(size_t)m * V + v] = base;
    for (int idx = tid; idx < K * rr; idx += TILE_V) cs[idx] = codes[(size_t)m * K * rr + idx];
    __syncthreads();
    for (int z = 0; z < K; ++z) {
      float2 p = make_float2(-INFINITY, 0.f);
      if (vok) {
        float corr = 0.f;
        const float* wr = wu + ((size_t)v * K + z) * rr;
        for (int k = 0; k < rr; ++k) corr = fmaf(wr[k], cs[z * rr + k], corr);
        p = make_float2((base + corr) * k2, 1.f);
      }
      p = warp_lse_merge(p);
      if (lane == 0) red[(r * K + z) * 4 + warp] = p;
    }
    __syncthreads();
  }
  for (int idx = tid; idx < RB * K; idx += TILE_V) {
    const int r = idx / K, z = idx - r * K, m = m0 + r;
    if (m >= M) continue;
    float2 p = red[idx * 4];
    for (int j = 1; j < 4; ++j) p = lse_merge(p, red[idx * 4 + j]);
    partd[((size_t)t * K + z) * Mpad + m] = p;
  }
}

template <typename Tin> static cudaError_t draft_simt_typed(const StepCtx& c) {
  const dblast_head* h = c.head;
  const WsLayout& w = c.wl;
  dim3 grid(w.nt, ceil_div(w.M, RB));
  const size_t smem = (RB * 64 + 32 * 65) * sizeof(float) + RB * 32 * 4 * sizeof(float2);
  k_draft_simt<Tin><<<grid, TILE_V, smem, c.stream>>>(
      static_cast<const Tin*>(h->W), static_cast<const Tin*>(c.args->hidden), h->vbias,
      prp<float>(c, c.pl.off_wu), wsp<float>(c, w.off_codes), h->V, h->H, h->K, w.rr, w.M,
      w.Mpad, c.k2, wsp<float>(c, w.off_stash), wsp<float2>(c, w.off_partd));
  debug_kernel("k_draft_simt", c.stream);
  count_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_draft_pass_simt(const StepCtx& c) {
  return c.head->dtype == DBLAST_F32 ? draft_simt_typed<float>(c)
                                     : draft_simt_typed<__nv_bfloat16>(c);
}

// ---------------------------------------------------------------------------
// merge per-tile (m2, s) records of one row into log2-sum-exp2 (double)
__device__ double warp_merge_tiles(const float2* __restrict__ part, size_t stride, int nt) {
  const int lane = threadIdx.x & 31;
  float mx = -INFINITY;
  for (int t = lane; t < nt; t += 32) mx = fmaxf(mx, part[(size_t)t * stride].x);
  mx = warp_max(mx);
  double s = 0.0;
  if (mx != -INFINITY)
    for (int t = lane; t < nt; t += 32) {
      const float2 q = part[(size_t)t * stride];
      if (q.y > 0.f) s += (double)q.y * exp2((double)q.x - (double)mx);
    }
  s = warp_sum_d(s);
  return mx == -INFINITY ? -INFINITY : (double)mx + log2(s);
}

// one warp per (m, z): lse2[m][z]
__global__ void k_draft_lse(const float2* __restrict__ partd, int nt, int K, int M, int Mpad,
                            double* __restrict__ lse2) {
  const int gw = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  if (gw >= M * K) return;
  const int m = gw / K, z = gw - m * K;
  const double L = warp_merge_tiles(partd + (size_t)z * Mpad + m, (size_t)K * Mpad, nt);
  if ((threadIdx.x & 31) == 0) lse2[(size_t)m * K + z] = L;
}

// Result of an inverse-CDF scan: the chosen item (-1 if none), the mass
// before it, the last item with positive mass, and the decision margin.
struct ScanHit {
  int idx;
  int last;
  double before;
  double margin;
};

// Inverse-CDF scan over `n` items of non-negative mass `mass(i)` (a functor
// holding its data by value): the first item whose inclusive cumulative mass
// exceeds `target`.
template <typename F>
__device__ __forceinline__ ScanHit warp_scan_find(int n, const F mass, double target) {
  const int lane = threadIdx.x & 31;
  double cum = 0.0;
  int lastp = -1;
  for (int base = 0; base < n; base += 32) {
    const int i = base + lane;
    const double p = (i < n) ? mass(i) : 0.0;
    const unsigned posb = __ballot_sync(0xffffffffu, p > 0.0);
    if (posb) lastp = base + 31 - __clz(posb);
    const double incl = warp_incl_scan_d(p) + cum;
    const unsigned hit = __ballot_sync(0xffffffffu, incl > target);
    if (hit) {
      const int l = __ffs(hit) - 1;
      const double il = __shfl_sync(0xffffffffu, incl, l);
      const double pl = __shfl_sync(0xffffffffu, p, l);
      return ScanHit{base + l, lastp, il - pl, 1.0};
    }
    cum = __shfl_sync(0xffffffffu, incl, 31);
  }
  return ScanHit{-1, lastp, cum, 0.0};
}

// Inside one vocabulary tile: masses of its TILE_V tokens from `elem(v)` (4 per
// lane, in order), cumulative mass starting at `before`.  Returns the first
// token whose cumulative mass exceeds `target` (idx -1 if none), the last
// token with positive mass, and the margin of the decision in units of `total`.
template <typename F>
__device__ __forceinline__ ScanHit warp_tile_find(int tile, int V, const F elem, double before,
                                                  double target, double total) {
  const int lane = threadIdx.x & 31;
  double e[4];
  double loc = 0.0;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const int v = tile * TILE_V + lane * 4 + j;
    e[j] = (v < V) ? elem(v) : 0.0;
    loc += e[j];
  }
  const double incl = warp_incl_scan_d(loc) + before;
  double c = incl - loc;
  int found = -1;
  double m = 0.0;
  int lastp = -1;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const double lo = c;
    c += e[j];
    if (e[j] > 0.0) lastp = tile * TILE_V + lane * 4 + j;
    if (found < 0 && c > target) {
      found = tile * TILE_V + lane * 4 + j;
      m = fmin(target - lo, c - target) / total;
    }
  }
  const unsigned hit = __ballot_sync(0xffffffffu, found >= 0);
  int lp = lastp;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) lp = max(lp, __shfl_xor_sync(0xffffffffu, lp, o));
  if (!hit) return ScanHit{-1, lp, before, 0.0};
  const int l = __ffs(hit) - 1;
  return ScanHit{__shfl_sync(0xffffffffu, found, l), lp, before,
                 __shfl_sync(0xffffffffu, m, l)};
}

__device__ __forceinline__ float corr_at(const float* __restrict__ wu, const float* __restrict__ c,
                                         int v, int z, int K, int rr) {
  const float* wr = wu + ((size_t)v * K + z) * rr;
  float acc = 0.f;
  for (int k = 0; k < rr; ++k) acc = fmaf(wr[k], c[k], acc);
  return acc;
}

// Functors for the scans (all data held by value).
struct TileMassLse {  // mass of tile t of a (m2, s) record row: s 2^(m2 - L)
  const float2* rec;
  size_t stride;
  double L;
  __device__ double operator()(int t) const {
    const float2 q = rec[(size_t)t * stride];
    return q.y > 0.f ? (double)q.y * exp2((double)q.x - L) : 0.0;
  }
};
struct TileMassRes {  // residual mass record of tile t (clamped at 0)
  const float2* rec;
  size_t stride;
  __device__ double operator()(int t) const {
    return (double)fmaxf(rec[(size_t)t * stride].y, 0.f);
  }
};
struct BranchProb {  // q_i(v|z) = 2^{(base_v + corr_z(v)) k2 - L}
  const float* srow;
  const float* wu;
  const float* cz;
  int z, K, rr;
  float k2;
  double L;
  __device__ double operator()(int v) const {
    const float s = (srow[v] + corr_at(wu, cz, v, z, K, rr)) * k2;
    return exp2((double)s - L);
  }
};
template <typename Tin> struct TargetProb {  // p_i(v) = 2^{t_v k2 - Lt}
  const Tin* trow;
  float k2;
  double Lt;
  __device__ double operator()(int v) const { return exp2((double)(ldf(trow + v) * k2) - Lt); }
};
template <typename Tin> struct ResidualMass {  // [p(v) - q(v|x_<i)]_+
  TargetProb<Tin> p;
  const float* srow;
  const float* wu;
  const float* cm;
  const double* lse2m;  // [K]
  const double* w2m;    // [K]
  int K, rr;
  float k2;
  __device__ double operator()(int v) const {
    double q = 0.0;
    for (int z = 0; z < K; ++z) {
      const double wz = w2m[z];
      if (wz == -INFINITY) continue;
      const float s = (srow[v] + corr_at(wu, cm + z * rr, v, z, K, rr)) * k2;
      q += exp2((double)s - lse2m[z] + wz);
    }
    return fmax(p(v) - q, 0.0);
  }
};

// one warp per row m = (n, i): draft token x from the z-hat branch (stream 1)
// and log2 q_z(x) for every branch
__global__ void k_draft_token(const float2* __restrict__ partd, const double* __restrict__ lse2,
                              const float* __restrict__ stash, const float* __restrict__ wu,
                              const float* __restrict__ codes, const int32_t* __restrict__ zhat,
                              int nt, int V, int K, int rr, int B, int M, int Mpad, float k2,
                              uint64_t seed, const int64_t* __restrict__ pos,
                              const uint32_t* __restrict__ rnd, int32_t* __restrict__ tok,
                              double* __restrict__ lq2, uint32_t* __restrict__ ties) {
  const int m = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (m >= M) return;
  const int n = m / B, i = m - n * B;
  const int z = zhat[n];
  const double L = lse2[(size_t)m * K + z];
  const float* cm = codes + (size_t)m * K * rr;
  const float* srow = stash + (size_t)m * V;
  const double u = decision_uniform(seed, 1u, rnd[n], (uint32_t)n, (uint32_t)(pos[n] + i));
  const TileMassLse tiles{partd + (size_t)z * Mpad + m, (size_t)K * Mpad, L};
  ScanHit th = warp_scan_find(nt, tiles, u);
  bool tie = false;
  if (th.idx < 0) {  // rounding left u above the total: the last tile with mass
    th.idx = th.last;
    th.before = 0.0;
    tie = true;
  }
  int x = -1;
  if (th.idx >= 0) {
    const BranchProb q{srow, wu, cm + z * rr, z, K, rr, k2, L};
    const ScanHit vh = warp_tile_find(th.idx, V, q, th.before, u, 1.0);
    x = vh.idx;
    if (x < 0) {
      x = vh.last;
      tie = true;
    } else if (vh.margin < (double)TIE_TOL) {
      tie = true;
    }
  }
  if (x < 0) x = 0;
  if (lane == 0) {
    tok[m] = x;
    if (tie) atomicOr(&ties[n], (uint32_t)TIE_DRAFT);
  }
  if (lane < K) {
    const float s = (srow[x] + corr_at(wu, cm + lane * rr, x, lane, K, rr)) * k2;
    lq2[(size_t)m * K + lane] = (double)s - lse2[(size_t)m * K + lane];
  }
}

// one warp per sequence: posterior (Eq. category-posterior) and q(x_i|x_<i)
// (Eq. dep-next-token); user-visible draft outputs
__global__ void k_posterior(const double* __restrict__ lq2, const double* __restrict__ lse2,
                            const float* __restrict__ log2pi, const int32_t* __restrict__ zhat,
                            const int32_t* __restrict__ tok, int N, int B, int K,
                            double* __restrict__ w2, dblast_draft_out out) {
  const int n = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (n >= N) return;
  double acc = (lane < K) ? (double)log2pi[n * K + lane] : -INFINITY;
  if (out.z_hat && lane == 0) out.z_hat[n] = zhat[n];
  if (out.pi && lane < K) out.pi[n * K + lane] = (float)exp2(acc);
  for (int i = 0; i < B; ++i) {
    const size_t m = (size_t)n * B + i;
    double mx = acc;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = fmax(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    const double e = (lane < K && acc != -INFINITY) ? exp2(acc - mx) : 0.0;
    const double lz = mx + log2(warp_sum_d(e));
    const double wz = (lane < K && acc != -INFINITY) ? acc - lz : -INFINITY;
    const double lq = (lane < K) ? lq2[m * K + lane] : -INFINITY;
    const double qt = warp_sum_d((lane < K && wz != -INFINITY) ? exp2(wz + lq) : 0.0);
    if (lane < K) {
      w2[m * K + lane] = wz;
      if (out.logw) out.logw[m * K + lane] = (float)(wz * (double)LN2);
      if (out.lse) out.lse[m * K + lane] = (float)(lse2[m * K + lane] * (double)LN2);
    }
    if (lane == 0) {
      if (out.q_tok) out.q_tok[m] = (float)qt;
      if (out.tokens) out.tokens[m] = tok[m];
    }
    if (lane < K) acc += lq;
  }
}

cudaError_t launch_draft_finalize(const StepCtx& c, const dblast_draft_out* outp) {
  const WsLayout& w = c.wl;
  const dblast_block_args* a = c.args;
  const int K = c.head->K;
  k_draft_lse<<<ceil_div(w.M * K * 32, 256), 256, 0, c.stream>>>(
      wsp<float2>(c, w.off_partd), w.nt, K, w.M, w.Mpad, wsp<double>(c, w.off_lse2));
  debug_kernel("k_draft_lse", c.stream);
  k_draft_token<<<ceil_div(w.M * 32, 256), 256, 0, c.stream>>>(
      wsp<float2>(c, w.off_partd), wsp<double>(c, w.off_lse2), wsp<float>(c, w.off_stash),
      prp<float>(c, c.pl.off_wu), wsp<float>(c, w.off_codes), wsp<int32_t>(c, w.off_zhat), w.nt,
      w.V, K, w.rr, w.B, w.M, w.Mpad, c.k2, a->seed, a->pos, a->round, wsp<int32_t>(c, w.off_tok),
      wsp<double>(c, w.off_lq2), wsp<uint32_t>(c, w.off_ties));
  debug_kernel("k_draft_token", c.stream);
  dblast_draft_out out{};
  if (outp) out = *outp;
  k_posterior<<<ceil_div(w.N * 32, 256), 256, 0, c.stream>>>(
      wsp<double>(c, w.off_lq2), wsp<double>(c, w.off_lse2), wsp<float>(c, w.off_log2pi),
      wsp<int32_t>(c, w.off_zhat), wsp<int32_t>(c, w.off_tok), w.N, w.B, K,
      wsp<double>(c, w.off_w2), out);
  debug_kernel("k_posterior", c.stream);
  count_launches(3);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// target rows: per-tile (m2, s) of t/T, then lse2t per row.  One warp per
// (row, tile); rows are laid out n*(B+1) + i in the workspace.
template <typename Tin>
__global__ void k_target_tiles(const Tin* __restrict__ target, int V, int nt, int B, int Bt,
                               int rows, int Rt, float k2, float2* __restrict__ partt) {
  const int gw = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (gw >= rows * nt) return;
  const int row = gw / nt, t = gw - row * nt;
  const int n = row / Bt, i = row - n * Bt;
  const Tin* tr = target + (size_t)row * V;
  float2 p = make_float2(-INFINITY, 0.f);
  float s[4];
  float mx = -INFINITY;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const int v = t * TILE_V + lane * 4 + j;
    s[j] = (v < V) ? ldf(tr + v) * k2 : -INFINITY;
    mx = fmaxf(mx, s[j]);
  }
  if (mx != -INFINITY) {
    float sum = 0.f;
#pragma unroll
    for (int j = 0; j < 4; ++j) sum += (s[j] != -INFINITY) ? exp2f(s[j] - mx) : 0.f;
    p = make_float2(mx, sum);
  }
  p = warp_lse_merge(p);
  if (lane == 0) partt[(size_t)t * Rt + (size_t)n * (B + 1) + i] = p;
}

__global__ void k_target_lse(const float2* __restrict__ partt, int nt, int B, int Bt, int rows,
                             int Rt, double* __restrict__ lse2t, float* __restrict__ lse_out) {
  const int gw = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  if (gw >= rows) return;
  const int n = gw / Bt, i = gw - n * Bt;
  const int rl = n * (B + 1) + i;
  const double L = warp_merge_tiles(partt + rl, (size_t)Rt, nt);
  if ((threadIdx.x & 31) == 0) {
    lse2t[rl] = L;
    if (lse_out) lse_out[(size_t)n * Bt + i] = (float)(L * (double)LN2);
  }
}

template <typename Tin> static cudaError_t target_typed(const StepCtx& c, const dblast_verify_out* o) {
  const WsLayout& w = c.wl;
  const int Bt = w.B + (o->has_bonus ? 1 : 0);
  const int rows = w.N * Bt;
  const long long warps = (long long)rows * w.nt;
  const unsigned blocks = (unsigned)((warps * 32 + 255) / 256);
  k_target_tiles<Tin><<<blocks, 256, 0, c.stream>>>(static_cast<const Tin*>(o->target), w.V, w.nt, w.B, Bt, rows,
                                    w.Rt, c.k2, wsp<float2>(c, w.off_partt));
  debug_kernel("k_target_tiles", c.stream);
  k_target_lse<<<ceil_div(rows * 32, 256), 256, 0, c.stream>>>(
      wsp<float2>(c, w.off_partt), w.nt, w.B, Bt, rows, w.Rt, wsp<double>(c, w.off_lse2t),
      o->lse_target);
  debug_kernel("k_target_lse", c.stream);
  count_launches(2);
  return cudaGetLastError();
}

cudaError_t launch_target_stats(const StepCtx& c, const dblast_verify_out* o) {
  return c.head->dtype == DBLAST_F32 ? target_typed<float>(c, o)
                                     : target_typed<__nv_bfloat16>(c, o);
}

// ---------------------------------------------------------------------------
// verify pass on CUDA cores: partv[t][m] = (sum min(p, q), sum [p - q]_+)
template <typename Tin>
__global__ void __launch_bounds__(TILE_V)
    k_verify_simt(const Tin* __restrict__ target, const float* __restrict__ stash,
                  const float* __restrict__ wu, const float* __restrict__ codes,
                  const double* __restrict__ lse2, const double* __restrict__ w2,
                  const double* __restrict__ lse2t, int V, int K, int rr, int B, int Bt, int M,
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
    if (tid < K) off[tid] = (float)(w2[(size_t)m * K + tid] - lse2[(size_t)m * K + tid]);
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
      const double Lt = lse2t[(size_t)n * (B + 1) + i];
      const float p = (float)exp2((double)(ldf(target + ((size_t)n * Bt + i) * V + v) * k2) - Lt);
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
      wsp<float>(c, w.off_codes), wsp<double>(c, w.off_lse2), wsp<double>(c, w.off_w2),
      wsp<double>(c, w.off_lse2t), w.V, c.head->K, w.rr, w.B, c.Bt, w.M, w.Mpad, c.k2,
      wsp<float2>(c, w.off_partv));
  debug_kernel("k_verify_simt", c.stream);
  count_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_verify_pass_simt(const StepCtx& c) {
  return c.head->dtype == DBLAST_F32 ? verify_simt_typed<float>(c)
                                     : verify_simt_typed<__nv_bfloat16>(c);
}

// ---------------------------------------------------------------------------
// one warp per row: alpha_m = sum_t A_t, residual mass R_m = sum_t R_t
__global__ void k_verify_merge(const float2* __restrict__ partv, int nt, int M, int Mpad,
                               double2* __restrict__ av) {
  const int m = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (m >= M) return;
  double a = 0.0, r = 0.0;
  for (int t = lane; t < nt; t += 32) {
    const float2 q = partv[(size_t)t * Mpad + m];
    a += q.x;
    r += q.y;
  }
  a = warp_sum_d(a);
  r = warp_sum_d(r);
  if (lane == 0) av[m] = make_double2(a, r);
}

// one warp per sequence: acceptance scan (stream 2), residual or bonus draw
// (stream 3), expected lengths, emitted tokens, state update
template <typename Tin>
__global__ void k_verify_final(const Tin* __restrict__ target, const float* __restrict__ stash,
                               const float* __restrict__ wu, const float* __restrict__ codes,
                               const double* __restrict__ lse2, const double* __restrict__ w2,
                               const double* __restrict__ lq2, const double* __restrict__ lse2t,
                               const float2* __restrict__ partv, const float2* __restrict__ partt,
                               const double2* __restrict__ av, const int32_t* __restrict__ tok,
                               const uint32_t* __restrict__ ties_draft, int N, int V, int K,
                               int rr, int B, int Bt, int nt, int Mpad, int Rt, float k2,
                               uint64_t seed, int64_t* __restrict__ pos, uint32_t* __restrict__ rnd,
                               dblast_verify_out out) {
  const int n = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (n >= N) return;
  const int64_t p0 = pos[n];
  const uint32_t rd = rnd[n];
  uint32_t ties = ties_draft[n];
  // per-position p_tok, q_tok, acceptance (lane i handles position i)
  double A = 0.0, alpha = 0.0, ptok = 0.0, qtok = 1.0, u2 = 0.0;
  bool acc_ok = false;
  if (lane < B) {
    const int m = n * B + lane;
    const int x = min(max(tok[m], 0), V - 1);  // tokens come from k_draft_token, always in [0, V)
    const double Lt = lse2t[(size_t)n * (B + 1) + lane];
    ptok = exp2((double)(ldf(target + ((size_t)n * Bt + lane) * V + x) * k2) - Lt);
    qtok = 0.0;
    for (int z = 0; z < K; ++z) {
      const double wz = w2[(size_t)m * K + z];
      if (wz != -INFINITY) qtok += exp2(wz + lq2[(size_t)m * K + z]);
    }
    const double ratio = ptok / qtok;
    A = fmin(1.0, ratio);
    alpha = av[m].x;
    u2 = decision_uniform(seed, 2u, rd, (uint32_t)n, (uint32_t)(p0 + lane));
    acc_ok = u2 < ratio;
    if (out.p_tok) out.p_tok[m] = (float)ptok;
    if (out.accept_prob) out.accept_prob[m] = (float)A;
    if (out.alpha) out.alpha[m] = (float)alpha;
  }
  const unsigned acc_mask = __ballot_sync(0xffffffffu, acc_ok);
  const unsigned rej = ~acc_mask & ((B >= 32) ? 0xffffffffu : ((1u << B) - 1u));
  const int L = rej ? (__ffs(rej) - 1) : B;
  // accept ties only for the positions that were tested (i <= L)
  const bool atie = lane < B && lane <= L && fabs(u2 * qtok - ptok) < (double)TIE_TOL * qtok;
  if (__ballot_sync(0xffffffffu, atie)) ties |= TIE_ACCEPT;
  // E[L|x] = sum_i prod_{j<=i} A_j and the same over alpha (products in lane order)
  double cA = (lane < B) ? A : 1.0, cAl = (lane < B) ? alpha : 1.0;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const double ta = __shfl_up_sync(0xffffffffu, cA, o);
    const double tl = __shfl_up_sync(0xffffffffu, cAl, o);
    if (lane >= o) {
      cA *= ta;
      cAl *= tl;
    }
  }
  const double expl = warp_sum_d(lane < B ? cA : 0.0);
  const double alen = warp_sum_d(lane < B ? cAl : 0.0);

  int extra = -1;
  bool tie = false;
  const int irow = (L < B) ? L : B;  // target row of the extra token
  const bool draw = (L < B) || (Bt > B);
  if (draw) {
    const double u3 = decision_uniform(seed, 3u, rd, (uint32_t)n, (uint32_t)(p0 + irow));
    const int rl = n * (B + 1) + irow;
    const double Lt = lse2t[rl];
    const TargetProb<Tin> pv{target + ((size_t)n * Bt + irow) * V, k2, Lt};
    bool from_p = (L >= B);
    if (L < B) {
      const int m = n * B + L;
      const double Rm = av[m].y;
      if (Rm < (double)TIE_TOL) ties |= TIE_RMASS;
      if (Rm > 0.0) {
        const double tm = u3 * Rm;
        ScanHit th = warp_scan_find(nt, TileMassRes{partv + m, (size_t)Mpad}, tm);
        if (th.idx < 0) {
          th.idx = th.last;
          th.before = 0.0;
          tie = true;
        }
        if (th.idx >= 0) {
          const ResidualMass<Tin> rm{pv, stash + (size_t)m * V, wu, codes + (size_t)m * K * rr,
                                     lse2 + (size_t)m * K, w2 + (size_t)m * K, K, rr, k2};
          const ScanHit vh = warp_tile_find(th.idx, V, rm, th.before, tm, Rm);
          extra = vh.idx;
          if (extra < 0) {
            extra = vh.last;
            tie = true;
          } else if (vh.margin < (double)TIE_TOL) {
            tie = true;
          }
        }
      }
      if (extra < 0) {  // no positive residual mass left by rounding: draw from p
        from_p = true;
        tie = true;
        ties |= TIE_RMASS;
      }
    }
    if (from_p) {
      ScanHit th = warp_scan_find(nt, TileMassLse{partt + rl, (size_t)Rt, Lt}, u3);
      if (th.idx < 0) {
        th.idx = th.last;
        th.before = 0.0;
        tie = true;
      }
      extra = 0;
      if (th.idx >= 0) {
        const ScanHit vh = warp_tile_find(th.idx, V, pv, th.before, u3, 1.0);
        extra = vh.idx;
        if (extra < 0) {
          extra = vh.last >= 0 ? vh.last : 0;
          tie = true;
        } else if (vh.margin < (double)TIE_TOL) {
          tie = true;
        }
      }
    }
  }
  if (tie) ties |= TIE_RESID;
  const int ne = L + (extra >= 0 ? 1 : 0);
  if (out.emitted) {
    for (int j = lane; j < B + 1; j += 32) {
      int val = -1;
      if (j < L) val = tok[n * B + j];
      else if (j == L && extra >= 0) val = extra;
      out.emitted[(size_t)n * (B + 1) + j] = val;
    }
  }
  if (lane == 0) {
    if (out.accepted) out.accepted[n] = L;
    if (out.n_emitted) out.n_emitted[n] = ne;
    if (out.exp_len) out.exp_len[n] = (float)expl;
    if (out.alpha_len) out.alpha_len[n] = (float)alen;
    if (out.tie_flags) out.tie_flags[n] = ties;
    pos[n] = p0 + ne;
    rnd[n] = rd + 1u;
  }
}

template <typename Tin>
static cudaError_t verify_final_typed(const StepCtx& c, const dblast_verify_out* o) {
  const int Bt = c.Bt;
  const WsLayout& w = c.wl;
  k_verify_merge<<<ceil_div(w.M * 32, 256), 256, 0, c.stream>>>(
      wsp<float2>(c, w.off_partv), w.nt, w.M, w.Mpad, wsp<double2>(c, w.off_av));
  debug_kernel("k_verify_merge", c.stream);
  k_verify_final<Tin><<<ceil_div(w.N * 32, 128), 128, 0, c.stream>>>(
      static_cast<const Tin*>(o->target), wsp<float>(c, w.off_stash), prp<float>(c, c.pl.off_wu),
      wsp<float>(c, w.off_codes), wsp<double>(c, w.off_lse2), wsp<double>(c, w.off_w2),
      wsp<double>(c, w.off_lq2), wsp<double>(c, w.off_lse2t), wsp<float2>(c, w.off_partv),
      wsp<float2>(c, w.off_partt), wsp<double2>(c, w.off_av), wsp<int32_t>(c, w.off_tok),
      wsp<uint32_t>(c, w.off_ties), w.N, w.V, c.head->K, w.rr, w.B, Bt, w.nt, w.Mpad, w.Rt, c.k2,
      c.args->seed, c.args->pos, c.args->round, *o);
  debug_kernel("k_verify_final", c.stream);
  count_launches(2);
  return cudaGetLastError();
}

cudaError_t launch_verify_finalize(const StepCtx& c, const dblast_verify_out* o) {
  return c.head->dtype == DBLAST_F32 ? verify_final_typed<float>(c, o)
                                     : verify_final_typed<__nv_bfloat16>(c, o);
}

}  // namespace dblast
