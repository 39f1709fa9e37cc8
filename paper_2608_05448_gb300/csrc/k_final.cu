// Finalize kernels of the step, shared by the CUDA-core and tensor-core
// vocabulary passes.  They merge the per-tile records of the passes
//   draft  : partd[t][z][m] = (m2, s), s * 2^m2 = sum_v 2^{l_{m,z,v} log2(e)/T}
//   target : partt[t][row]  = (tmax, s), s = sum_v 2^{(t_v - tmax) log2(e)/T}
//   verify : partv[t][m]    = (sum_v min(p, q), sum_v [p - q]_+)
// and take every decision of the step: the draft tokens (Sec. 3.1), the
// category posterior and q(x_i|x_<i) (Eqs. category-posterior and
// dep-next-token), acceptance with min(1, p/q) (Eq. 2), the residual or bonus
// token (Algorithm 1, App. A) and the expected lengths (Eq. 3).
//
// Every token draw is an inverse CDF over the vocabulary in two levels: a
// block-wide scan of the tile masses finds the tile, then the tile's TILE_V
// masses are recomputed and scanned.
//
// Precision without FP64: sums, scans, log-sum-exps and log-weights are
// float-float pairs (FF); exponents subtract a normaliser held as a pair, so
// the rounded part of every exponent is the small difference, not the large
// logit.
#include <type_traits>

#include "dblast_internal.cuh"

namespace dblast {

constexpr unsigned FULLMASK = 0xffffffffu;

// ------------------------------------------------------------ float-float
__device__ __forceinline__ FF ff_shfl_up(FF a, int o) {
  return FF{__shfl_up_sync(FULLMASK, a.hi, o), __shfl_up_sync(FULLMASK, a.lo, o)};
}
__device__ __forceinline__ FF ff_shfl_xor(FF a, int o) {
  return FF{__shfl_xor_sync(FULLMASK, a.hi, o), __shfl_xor_sync(FULLMASK, a.lo, o)};
}

// ------------------------------------------------------------ block helpers
struct BlockScan {
  FF excl, incl, total;  // excl of thread j equals incl of thread j-1 bit for bit
};

template <int NT> __device__ BlockScan block_scan_ff(FF v, FF* sh) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  FF wi = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const FF t = ff_shfl_up(wi, o);
    if (lane >= o) wi = ff_add(t, wi);
  }
  FF we = ff_shfl_up(wi, 1);
  if (lane == 0) we = FF{0.f, 0.f};
  if (lane == 31) sh[warp] = wi;
  __syncthreads();
  FF off{0.f, 0.f}, tot{0.f, 0.f};
#pragma unroll
  for (int w = 0; w < NT / 32; ++w) {
    if (w == warp) off = tot;
    tot = ff_add(tot, sh[w]);
  }
  __syncthreads();
  return BlockScan{ff_add(off, we), ff_add(off, wi), tot};
}

template <int NT> __device__ int block_min_i(int v, int* sh) {
  v = __reduce_min_sync(FULLMASK, v);
  if ((threadIdx.x & 31) == 0) sh[threadIdx.x >> 5] = v;
  __syncthreads();
  int r = sh[0];
#pragma unroll
  for (int w = 1; w < NT / 32; ++w) r = min(r, sh[w]);
  __syncthreads();
  return r;
}

template <int NT> __device__ int block_max_i(int v, int* sh) {
  return -block_min_i<NT>(-v, sh);
}

// (W U_z)_v . c: the branch correction of token v (rr % 4 == 0: 16-byte loads,
// the WU rows and the code rows then start on 16-byte boundaries)
__device__ __forceinline__ float corr_at(const float* __restrict__ wu, const float* __restrict__ c,
                                         int v, int z, int K, int rr) {
  const float* wr = wu + ((size_t)v * K + z) * rr;
  float acc = 0.f;
  if ((rr & 3) == 0) {
    const float4* w4 = reinterpret_cast<const float4*>(wr);
    const float4* c4 = reinterpret_cast<const float4*>(c);
    for (int k = 0; k < (rr >> 2); ++k) {
      const float4 a = w4[k], b = c4[k];
      acc = fmaf(a.x, b.x, acc);
      acc = fmaf(a.y, b.y, acc);
      acc = fmaf(a.z, b.z, acc);
      acc = fmaf(a.w, b.w, acc);
    }
    return acc;
  }
  for (int k = 0; k < rr; ++k) acc = fmaf(wr[k], c[k], acc);
  return acc;
}

// 2^{(x k2 - C)} for a float logit x and a split normaliser C = c.hi + c.lo:
// the product is exact inside the fma, so only the small difference rounds.
__device__ __forceinline__ float exp2_rel(float x, float k2, FF c) {
  return exp2f(fmaf(x, k2, -c.hi) - c.lo);
}
// 2^{(base + corr) k2 - C} with the same care for the two-term logit
__device__ __forceinline__ float exp2_rel2(float base, float corr, float k2, FF c) {
  return exp2f(fmaf(corr, k2, fmaf(base, k2, -c.hi)) - c.lo);
}

// ------------------------------------------------------- two-level draw
template <int NT> struct FindShared {
  FF d[NT / 32];
  int i[NT / 32];
  FF before;
  int tile, x, tie, near;
};

struct FindOut {
  int x;      // chosen token, -1 if no token has mass
  bool tie;   // the decision is within TIE_TOL of its threshold, or rounding forced a fallback
  bool near;  // within TIE_TOL + near_abs / total (near_abs: an absolute mass allowance)
};

// A token-mass functor may stage the chosen tile first, with every thread of
// the block (an overload of em_prepare for its type); the others read their
// tokens directly.
template <typename EM> __device__ __forceinline__ void em_prepare(const EM&, int) {}

// Smallest token whose cumulative mass (in vocabulary order) exceeds `target`.
// tmass(t): mass of tile t; emass(v): mass of token v (floats); `total` scales
// the decision margin.  With `frac`, target.hi is a fraction u of the summed
// tile masses, and that sum scales the margin.
template <int NT, typename TM, typename EM>
__device__ FindOut block_find(int nt, int V, const TM tmass, const EM emass, FF target,
                              float total, FindShared<NT>& fs, bool frac = false,
                              float near_abs = NEAR_DRAW) {
  static_assert(NT >= TILE_V, "one thread per token of a tile");
  const int tid = threadIdx.x, lane = tid & 31;
  const int chunk = ceil_div(nt, NT);
  const int t0 = min(nt, tid * chunk), t1 = min(nt, t0 + chunk);
  // level 1: this thread's chunk of tiles, loads issued eight at a time
  FF loc{0.f, 0.f};
  int lastp = -1;
  for (int c0 = 0; c0 < chunk; c0 += 8) {
    float w[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int t = t0 + c0 + j;
      w[j] = tmass(t < t1 ? t : 0);  // tile 0 always exists
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int t = t0 + c0 + j;
      if (t < t1) {
        loc = ff_addf(loc, w[j]);
        if (w[j] > 0.f) lastp = t;
      }
    }
  }
  const BlockScan sc = block_scan_ff<NT>(loc, fs.d);
  if (frac) {
    target = ff_mulf(sc.total, target.hi);
    total = ff_f(sc.total);
  }
  const int first = block_min_i<NT>(ff_gt(sc.incl, target) ? tid : NT, fs.i);
  const int lastall = block_max_i<NT>(lastp, fs.i);
  if (first < NT) {
    // the warp holding thread `first` rescans its chunk, 32 tiles per round,
    // starting from that thread's exclusive prefix
    if ((tid >> 5) == (first >> 5)) {
      const FF ex{__shfl_sync(FULLMASK, sc.excl.hi, first & 31),
                  __shfl_sync(FULLMASK, sc.excl.lo, first & 31)};
      const int f0 = first * chunk, f1 = min(nt, f0 + chunk);
      FF base = ex, lastlo{0.f, 0.f};
      int tt = -1, lp = -1;
      FF before{0.f, 0.f};
      for (int r0 = f0; r0 < f1 && tt < 0; r0 += 32) {
        const int t = r0 + lane;
        const float w = (t < f1) ? tmass(t) : 0.f;
        FF incl{w, 0.f};
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const FF u = ff_shfl_up(incl, o);
          if (lane >= o) incl = ff_add(u, incl);
        }
        FF ex1 = ff_shfl_up(incl, 1);
        if (lane == 0) ex1 = FF{0.f, 0.f};
        const FF hi = ff_add(base, incl), lo = ff_add(base, ex1);
        const unsigned hit = __ballot_sync(FULLMASK, t < f1 && ff_gt(hi, target));
        const unsigned pos = __ballot_sync(FULLMASK, t < f1 && w > 0.f);
        if (pos) {
          const int l = 31 - __clz(pos);
          lp = r0 + l;
          lastlo = FF{__shfl_sync(FULLMASK, lo.hi, l), __shfl_sync(FULLMASK, lo.lo, l)};
        }
        if (hit) {
          const int l = __ffs(hit) - 1;
          tt = r0 + l;
          before = FF{__shfl_sync(FULLMASK, lo.hi, l), __shfl_sync(FULLMASK, lo.lo, l)};
        }
        base = FF{__shfl_sync(FULLMASK, hi.hi, 31), __shfl_sync(FULLMASK, hi.lo, 31)};
      }
      if (lane == 0) {
        const bool miss = tt < 0;  // the rescan rounded below the target
        fs.tile = miss ? lp : tt;
        fs.before = miss ? lastlo : before;
        fs.tie = miss ? 1 : 0;
        fs.near = fs.tie;
      }
    }
  } else if (tid == 0) {  // rounding left the target at or above the total
    fs.tile = lastall;
    fs.before = lastall >= 0 ? ff_add(sc.total, FF{-tmass(lastall), 0.f}) : FF{0.f, 0.f};
    fs.tie = 1;
    fs.near = 1;
  }
  __syncthreads();
  const int tt = fs.tile;
  const FF before = fs.before;
  em_prepare(emass, tt);
  float e = 0.f;
  const int v = tt * TILE_V + tid;
  if (tt >= 0 && tid < TILE_V && v < V) e = emass(v);
  const BlockScan es = block_scan_ff<NT>(FF{e, 0.f}, fs.d);
  const FF lo = ff_add(before, es.excl), hi = ff_add(before, es.incl);
  const int fj = block_min_i<NT>((tt >= 0 && ff_gt(hi, target)) ? tid : NT, fs.i);
  const int lastv = block_max_i<NT>(e > 0.f ? tid : -1, fs.i);
  if (fj < NT) {
    if (tid == fj) {
      fs.x = tt * TILE_V + fj;
      const float margin = fminf(ff_f(ff_sub(target, lo)), ff_f(ff_sub(hi, target))) / total;
      if (margin < TIE_TOL) fs.tie = 1;
      if (margin < TIE_TOL + near_abs / total) fs.near = 1;
    }
  } else if (tid == 0) {
    fs.x = (tt >= 0 && lastv >= 0) ? tt * TILE_V + lastv : -1;
    fs.tie = 1;
    fs.near = 1;
  }
  __syncthreads();
  const FindOut r{fs.x, fs.tie != 0, fs.near != 0};
  __syncthreads();
  return r;
}

// Mass functors (data by value).
struct DraftTileMass {  // s 2^(m2 - L) of a draft record
  const float2* rec;
  size_t stride;
  FF L;
  __device__ float operator()(int t) const {
    const float2 q = rec[(size_t)t * stride];
    return q.y > 0.f ? q.y * exp2f((q.x - L.hi) - L.lo) : 0.f;
  }
};
struct TargetTileMass {  // s 2^(tmax k2 - Lt) of a target record
  const float2* rec;
  size_t stride;
  float k2;
  FF Lt;
  __device__ float operator()(int t) const {
    const float2 q = rec[(size_t)t * stride];
    return q.y > 0.f ? q.y * exp2_rel(q.x, k2, Lt) : 0.f;
  }
};
struct ResidTileMass {  // residual mass record, clamped at 0
  const float2* rec;
  size_t stride;
  __device__ float operator()(int t) const { return fmaxf(rec[(size_t)t * stride].y, 0.f); }
};
struct BranchTokenProb {  // q_i(v|z) = 2^{(base_v + corr_z(v)) k2 - L_z}
  const float* srow;
  const float* wu;
  const float* cz;
  int z, K, rr;
  float k2;
  FF L;
  __device__ float operator()(int v) const {
    return exp2_rel2(srow[v], corr_at(wu, cz, v, z, K, rr), k2, L);
  }
};
template <typename Tin> struct TargetTokenProb {  // p_i(v) = 2^{t_v k2 - Lt}
  const Tin* trow;
  float k2;
  FF Lt;
  __device__ float operator()(int v) const { return exp2_rel(ldf(trow + v), k2, Lt); }
};
// [p(v) - q(v|x_<i)]_+ of the tokens of one tile, computed by the whole
// block once the tile is known (prepare): thread j takes token j % 128 and
// the components z = g, g + G, ... with g = j / 128 and G = NT / 128, so
// a token's K correction loads are spread over G threads; the partial sums
// are then added in the order g = 0 .. G-1.
template <typename Tin> struct ResidualTokenMass {
  TargetTokenProb<Tin> p;
  const float* srow;
  const float* wu;
  const float* cm;  // codes of row m, [K, rr]
  const FF* C;      // [K] in shared memory: L_z - log2 w_z (+inf if w_z = 0)
  float* qpart;     // [G * TILE_V] shared: partial q sums
  float* pbuf;      // [TILE_V] shared: p(v) of the tile's tokens
  int K, rr, V, G;
  float k2;
  __device__ void prepare(int tt) const {  // every thread of the block
    const int tk = threadIdx.x % TILE_V, g = threadIdx.x / TILE_V;
    const int v = tt * TILE_V + tk;
    float q = 0.f;
    if (tt >= 0 && v < V && g < G) {
      if (g == 0) pbuf[tk] = p(v);
      const float base = srow[v];
      for (int z = g; z < K; z += G) {
        const FF c = C[z];
        if (c.hi == INFINITY) continue;
        q += exp2_rel2(base, corr_at(wu, cm + z * rr, v, z, K, rr), k2, c);
      }
    }
    if (g < G) qpart[threadIdx.x] = q;
    __syncthreads();
  }
  __device__ float operator()(int v) const {  // thread v % TILE_V, after prepare
    const int tk = threadIdx.x;
    float q = 0.f;
    for (int g = 0; g < G; ++g) q += qpart[g * TILE_V + tk];
    return fmaxf(pbuf[tk] - q, 0.f);
  }
};
template <typename Tin>
__device__ __forceinline__ void em_prepare(const ResidualTokenMass<Tin>& e, int tt) {
  e.prepare(tt);
}

// ---------------------------------------------------------------- draft side
// Partial log-sum-exps of the draft records: block (row group of 32, z, split);
// lane = row, warps and splits interleave over the tiles.
// lsep[sp][m][z] = (max, sum.hi, sum.lo, 0) with sum * 2^max the partial mass.
constexpr int LSE_WARPS = 16;
constexpr int LSE_BATCH = 19;  // records in flight per thread (1187 tiles: two batches)
__global__ void __launch_bounds__(LSE_WARPS * 32)
    k_draft_lse(const float2* __restrict__ partd, int nt, int K, int M, int Mpad,
                float4* __restrict__ lsep) {
  griddep_wait();  // launched as a dependent of the previous kernel
  __shared__ float smx[LSE_WARPS][32];
  __shared__ FF ssum[LSE_WARPS][32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int m = blockIdx.x * 32 + lane, z = blockIdx.y, sp = blockIdx.z;
  const int step = LSE_WARPS * LSE_SPLIT;
  float mx = -INFINITY;
  FF s{0.f, 0.f};
  if (m < M) {
    // batches of LSE_BATCH records, all loaded before any is used (one
    // memory round trip per batch); the batch's maximum, then its sum
    // against the running maximum
    const float2* p = partd + (size_t)z * Mpad + m;
    const size_t st = (size_t)K * Mpad;
    for (int t0 = sp * LSE_WARPS + warp; t0 < nt; t0 += LSE_BATCH * step) {
      float2 q[LSE_BATCH];
#pragma unroll
      for (int j = 0; j < LSE_BATCH; ++j) {
        const int t = t0 + j * step;
        q[j] = t < nt ? p[(size_t)t * st] : make_float2(-INFINITY, 0.f);
      }
      float bm = -INFINITY;
#pragma unroll
      for (int j = 0; j < LSE_BATCH; ++j)
        if (q[j].y > 0.f) bm = fmaxf(bm, q[j].x);
      if (bm > mx) {
        if (mx != -INFINITY) s = ff_mulf(s, exp2f(mx - bm));
        mx = bm;
      }
#pragma unroll
      for (int j = 0; j < LSE_BATCH; ++j)
        if (q[j].y > 0.f) s = ff_addf(s, q[j].y * exp2f(q[j].x - mx));
    }
  }
  smx[warp][lane] = mx;
  ssum[warp][lane] = s;
  __syncthreads();
  if (warp == 0 && m < M) {
    float M2 = -INFINITY;
#pragma unroll
    for (int w = 0; w < LSE_WARPS; ++w) M2 = fmaxf(M2, smx[w][lane]);
    FF S{0.f, 0.f};
    if (M2 != -INFINITY)
#pragma unroll
      for (int w = 0; w < LSE_WARPS; ++w) S = ff_add(S, ff_mulf(ssum[w][lane], exp2f(smx[w][lane] - M2)));
    lsep[((size_t)sp * M + m) * K + z] = make_float4(M2, S.hi, S.lo, 0.f);
  }
}

// The category posterior of one sequence n (Eq. category-posterior) and
// q(x_i|x_<i) (Eq. dep-next-token), run by one block of NT threads once every
// row of the sequence has its token: log2 w_{i,z} from the prefix sums over
// i of log2 q_z(x_j) (one thread per branch, positions in order), the
// per-row constants of the tensor-core verify pass and the user-visible
// draft outputs.  Rows of other blocks are read past L1 (ld.global.cg).
struct PostShared {
  FF A[32 * 32];   // log2 pi_z + sum_{j<i} log2 q_z(x_j), [B][K]
  FF Lq[32 * 32];  // log2 q_z(x_i)
  FF Lz[32 * 32];  // lse2 of every (i, z)
  float E[32 * 32];
  FF rowv[32];
  float rowb[32];
};
__device__ __forceinline__ FF ff_ldcg(const float2* p) {
  const float2 v = __ldcg(p);
  return FF{v.x, v.y};
}
template <int NT>
__device__ void posterior_seq(int n, const float2* __restrict__ lq2, const float2* __restrict__ lse2,
                              const float* __restrict__ log2pi, const int32_t* __restrict__ zhat,
                              const int32_t* __restrict__ tok, const float* __restrict__ cscale,
                              const float* __restrict__ sw, float k2, int B, int K,
                              float2* __restrict__ w2, float* __restrict__ qtok,
                              float2* __restrict__ vcz, float* __restrict__ vb0,
                              const dblast_draft_out& out, PostShared& ps) {
  const int t = threadIdx.x, BK = B * K;
  const size_t mb = (size_t)n * B;
  for (int e = t; e < BK; e += NT) {
    ps.Lq[e] = ff_ldcg(lq2 + mb * K + e);
    ps.Lz[e] = ff_ldcg(lse2 + mb * K + e);
  }
  __syncthreads();
  if (t < K) {  // exclusive prefix over positions, branch t
    const float lp = log2pi[n * K + t];
    FF run{0.f, 0.f};
    for (int i = 0; i < B; ++i) {
      ps.A[i * K + t] = (lp == -INFINITY || run.hi == -INFINITY) ? FF{-INFINITY, 0.f}
                                                                : ff_addf(run, lp);
      run = ff_add(run, ps.Lq[i * K + t]);
    }
  }
  __syncthreads();
  for (int i = t; i < B; i += NT) {  // log2 sum_z of row i, and B0 of the verify pass
    float mx = -INFINITY, lmx = -INFINITY;
    for (int k = 0; k < K; ++k) {
      mx = fmaxf(mx, ps.A[i * K + k].hi);
      lmx = fmaxf(lmx, ps.Lz[i * K + k].hi);
    }
    FF S{0.f, 0.f};
    if (mx != -INFINITY)
      for (int k = 0; k < K; ++k)
        if (ps.A[i * K + k].hi != -INFINITY) S = ff_addf(S, ff_exp2(ff_addf(ps.A[i * K + k], -mx)));
    ps.rowv[i] = (mx == -INFINITY) ? FF{-INFINITY, 0.f} : ff_add(FF{mx, 0.f}, ff_log2(S));
    ps.rowb[i] = floorf(lmx);  // keeps the verify pass's two factors in range
  }
  __syncthreads();
  for (int e = t; e < BK; e += NT) {
    const int i = e / K, z = e - i * K;
    const size_t m = mb + i;
    const FF acc = ps.A[e], lz = ps.rowv[i], lq = ps.Lq[e];
    const bool wdead = acc.hi == -INFINITY || lz.hi == -INFINITY;
    const FF wz = wdead ? FF{-INFINITY, 0.f} : ff_sub(acc, lz);
    ps.E[e] = (wdead || lq.hi == -INFINITY) ? 0.f : ff_exp2(ff_add(wz, lq));
    const FF Lz = ps.Lz[e];
    w2[m * K + z] = ff_st(wz);
    vcz[m * K + z] = make_float2(k2 / (cscale[m * K + z] * sw[z]),
                                 wdead ? -INFINITY : ff_f(ff_addf(ff_sub(wz, Lz), ps.rowb[i])));
    if (out.logw) out.logw[m * K + z] = wdead ? -INFINITY : ff_f(wz) * LN2;
    if (out.lse) out.lse[m * K + z] = ff_f(Lz) * LN2;
  }
  __syncthreads();
  for (int i = t; i < B; i += NT) {
    const size_t m = mb + i;
    FF qt{0.f, 0.f};
    for (int k = 0; k < K; ++k) qt = ff_addf(qt, ps.E[i * K + k]);
    qtok[m] = ff_f(qt);
    vb0[m] = ps.rowb[i];
    if (out.q_tok) out.q_tok[m] = ff_f(qt);
    if (out.tokens) out.tokens[m] = __ldcg(tok + m);
  }
  if (t < K && out.pi) out.pi[n * K + t] = exp2f(log2pi[n * K + t]);
  if (t == 0 && out.z_hat) out.z_hat[n] = zhat[n];
}

// One block per row m = (n, i): lse2 of every branch, the draft token
// x_i ~ q_i(.|z-hat) (stream 1), and log2 q_z(x_i) for every branch; the
// last block of a sequence to finish (a per-sequence counter, zeroed before
// the step) then runs that sequence's posterior.
constexpr int DT_NT = 256;
__global__ void __launch_bounds__(DT_NT)
    k_draft_token(const float2* __restrict__ partd, const float4* __restrict__ lsep,
                  const float* __restrict__ stash, const float* __restrict__ wu,
                  const float* __restrict__ codes, const int32_t* __restrict__ zhat, int nt, int V,
                  int K, int rr, int B, int M, int Mpad, float k2, uint64_t seed,
                  const int64_t* __restrict__ pos, const uint32_t* __restrict__ rnd,
                  const int32_t* __restrict__ given, float2* __restrict__ lse2,
                  int32_t* __restrict__ tok, float2* __restrict__ lq2,
                  uint32_t* __restrict__ ties, uint32_t* __restrict__ done,
                  const float* __restrict__ log2pi, const float* __restrict__ cscale,
                  const float* __restrict__ sw, float2* __restrict__ w2,
                  float* __restrict__ qtok, float2* __restrict__ vcz, float* __restrict__ vb0,
                  dblast_draft_out out, DevStatus* chk) {
  griddep_wait();  // launched as a dependent of the previous kernel
  __shared__ FindShared<DT_NT> fs;
  __shared__ FF sL[32];
  __shared__ int s_last;
  __shared__ PostShared ps;
  const int m = blockIdx.x, tid = threadIdx.x;
  const int n = m / B, i = m - n * B;
  // the sampled branch and the draw's uniform do not depend on the merge below
  const int z = zhat[n];
  const float u = decision_uniform(seed, 1u, rnd[n], (uint32_t)n, (uint32_t)(pos[n] + i));
  if (tid < K) {
    float4 q[LSE_SPLIT];
#pragma unroll
    for (int sp = 0; sp < LSE_SPLIT; ++sp) q[sp] = lsep[((size_t)sp * M + m) * K + tid];
    float mx = -INFINITY;
#pragma unroll
    for (int sp = 0; sp < LSE_SPLIT; ++sp) mx = fmaxf(mx, q[sp].x);
    FF S{0.f, 0.f};
    if (mx != -INFINITY)
#pragma unroll
      for (int sp = 0; sp < LSE_SPLIT; ++sp)
        S = ff_add(S, ff_mulf(FF{q[sp].y, q[sp].z}, exp2f(q[sp].x - mx)));
    const FF L = (mx == -INFINITY || !(S.hi > 0.f)) ? FF{-INFINITY, 0.f}
                                                   : ff_add(FF{mx, 0.f}, ff_log2(S));
    sL[tid] = L;
    lse2[(size_t)m * K + tid] = ff_st(L);
  }
  __syncthreads();
  const FF L = sL[z];
  const float* cm = codes + (size_t)m * K * rr;
  const float* srow = stash + (size_t)m * V;
  const DraftTileMass tm{partd + (size_t)z * Mpad + m, (size_t)K * Mpad, L};
  const BranchTokenProb em{srow, wu, cm + z * rr, z, K, rr, k2, L};
  int x;
  if (given) {  // a given block (training-side objectives): no draw
    x = checked_token(given[m], V, tid == 0 ? chk : nullptr, 1u);
    if (tid == 0) tok[m] = x;
  } else {
    const FindOut f = block_find<DT_NT>(nt, V, tm, em, FF{u, 0.f}, 1.f, fs);
    x = f.x >= 0 ? f.x : 0;
    if (tid == 0) {
      tok[m] = x;
      if (f.tie || f.x < 0) atomicOr(&ties[n], (uint32_t)TIE_DRAFT);
      if (f.near || f.x < 0) atomicOr(&ties[n], (uint32_t)TIE_DRAFT << NEAR_SHIFT);
    }
  }
  if (tid < K) {  // log2 q_z(x) = (base_x + corr_z(x)) k2 - L_z, products exact
    const FF s = ff_add(ff_prod(srow[x], k2), ff_prod(corr_at(wu, cm + tid * rr, x, tid, K, rr), k2));
    lq2[(size_t)m * K + tid] = ff_st(ff_sub(s, sL[tid]));
  }
  // this row's results are written: count it, and the sequence's last row
  // block runs the posterior
  __threadfence();
  __syncthreads();
  if (tid == 0) s_last = atomicAdd(&done[n], 1u) == (uint32_t)(B - 1);
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  posterior_seq<DT_NT>(n, lq2, lse2, log2pi, zhat, tok, cscale, sw, k2, B, K, w2, qtok, vcz, vb0,
                       out, ps);
}

cudaError_t launch_draft_finalize(const StepCtx& c, const dblast_draft_out* outp,
                                  const int32_t* given) {
  const WsLayout& w = c.wl;
  const dblast_block_args* a = c.args;
  const int K = c.head->K;
  cudaError_t le =
      launch_dep(k_draft_lse, dim3(ceil_div(w.M, 32), K, LSE_SPLIT), dim3(LSE_WARPS * 32), 0,
                 c.stream, wsp<float2>(c, w.off_partd), w.nt, K, w.M, w.Mpad, wsp<float4>(c, w.off_lsep));
  debug_kernel("k_draft_lse", c.stream);
  dblast_draft_out out{};
  if (outp) out = *outp;
  if (le == cudaSuccess) le = launch_dep(k_draft_token, dim3(w.M), dim3(DT_NT), 0, c.stream,
      wsp<float2>(c, w.off_partd), wsp<float4>(c, w.off_lsep), wsp<float>(c, w.off_stash),
      prp<float>(c, c.pl.off_wu), wsp<float>(c, w.off_codes), wsp<int32_t>(c, w.off_zhat), w.nt,
      w.V, K, w.rr, w.B, w.M, w.Mpad, c.k2, a->seed, a->pos, a->round, given,
      wsp<float2>(c, w.off_lse2),
      wsp<int32_t>(c, w.off_tok), wsp<float2>(c, w.off_lq2), wsp<uint32_t>(c, w.off_ties),
      wsp<uint32_t>(c, w.off_ties) + w.N, wsp<float>(c, w.off_log2pi),
      wsp<float>(c, w.off_cscale), prp<float>(c, c.pl.off_sw), wsp<float2>(c, w.off_w2),
      wsp<float>(c, w.off_qtok), wsp<float2>(c, w.off_vcz), wsp<float>(c, w.off_vb0), out, c.chk);
  debug_kernel("k_draft_token", c.stream);
  count_launches(2);
  return le != cudaSuccess ? le : cudaGetLastError();
}

// ---------------------------------------------------------------- target side
// One block per target row: a half-warp per tile of 128 tokens (8 per lane),
// the tile records partt and the row's lse2t = log2 sum_v 2^{t_v k2} (also as
// a float pair lt2 for the verify pass), and the row's collision probability
// coll = sum_v p(v)^2 (App. B), from the same exponentials squared.
constexpr int TS_NT = 256;
constexpr int TS_HW = TS_NT / 16;  // half-warps per block
constexpr int TS_NF = 4;           // tiles in flight per half-warp
static_assert(TS_HW <= 32, "one warp merges the half-warp partials");
template <typename Tin>
__global__ void __launch_bounds__(TS_NT)
    k_target_stats(const Tin* __restrict__ target, int V, int nt, int B, int Bt, int Rt, float k2,
                   bool vec, float2* __restrict__ partt, float2* __restrict__ lt2,
                   float* __restrict__ coll, float* __restrict__ lse_out) {
  __shared__ float smx[TS_HW];
  __shared__ FF ssum[TS_HW];
  __shared__ float ssq[TS_HW];
  const int row = blockIdx.x;
  const int n = row / Bt, i = row - n * Bt;
  const int rl = n * (B + 1) + i;
  const Tin* tr = target + (size_t)row * V;
  const int hw = threadIdx.x >> 4, hl = threadIdx.x & 15;
  float rmax = -INFINITY, rsq = 0.f;
  FF rsum{0.f, 0.f};
  // every lane of both half-warps runs the shuffles; `valid` gates the results
  auto tile = [&](int t, const float (&x)[8], bool valid) {
    float mx = x[0];
#pragma unroll
    for (int j = 1; j < 8; ++j) mx = fmaxf(mx, x[j]);
#pragma unroll
    for (int o = 8; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(FULLMASK, mx, o));
    float s = 0.f, s2 = 0.f;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const float e = exp2f((x[j] - mx) * k2);
      s += e;
      s2 = fmaf(e, e, s2);
    }
#pragma unroll
    for (int o = 8; o > 0; o >>= 1) {
      s += __shfl_xor_sync(FULLMASK, s, o);
      s2 += __shfl_xor_sync(FULLMASK, s2, o);
    }
    if (!valid) return;
    if (hl == 0) partt[(size_t)t * Rt + rl] = make_float2(mx, s);
    if (mx > rmax) {
      const float f = exp2f((rmax - mx) * k2);
      rsum = ff_mulf(rsum, f);
      rsq *= f * f;
      rmax = mx;
    }
    const float g = exp2f((mx - rmax) * k2);
    rsum = ff_addf(rsum, s * g);
    rsq = fmaf(s2, g * g, rsq);
  };
  // TS_NF tiles in flight per half-warp; the loop bounds are uniform over the block
  const int iters = ceil_div(nt, TS_HW);
  for (int k = 0; k < iters; k += TS_NF) {
    float x[TS_NF][8];
#pragma unroll
    for (int f = 0; f < TS_NF; ++f) {
      const int tf = (k + f) * TS_HW + hw;
      load8(tr, tf * TILE_V + hl * 8, (k + f < iters && tf < nt) ? V : 0, vec, x[f]);
    }
#pragma unroll
    for (int f = 0; f < TS_NF; ++f) {
      const int tf = (k + f) * TS_HW + hw;
      tile(tf, x[f], k + f < iters && tf < nt);
    }
  }
  if (hl == 0) {
    smx[hw] = rmax;
    ssum[hw] = rsum;
    ssq[hw] = rsq;
  }
  __syncthreads();
  if (threadIdx.x < 32) {
    const int l = threadIdx.x;
    const float ml = l < TS_HW ? smx[l] : -INFINITY;
    float M2 = ml;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) M2 = fmaxf(M2, __shfl_xor_sync(FULLMASK, M2, o));
    FF S{0.f, 0.f};
    float Q = 0.f;
    if (M2 != -INFINITY && ml != -INFINITY) {
      const float f = exp2f((ml - M2) * k2);
      S = ff_mulf(ssum[l], f);
      Q = ssq[l] * f * f;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      S = ff_add(S, ff_shfl_xor(S, o));
      Q += __shfl_xor_sync(FULLMASK, Q, o);
    }
    if (l == 0) {
      const FF L = (M2 == -INFINITY || !(S.hi > 0.f)) ? FF{-INFINITY, 0.f}
                                                     : ff_add(ff_prod(M2, k2), ff_log2(S));
      lt2[rl] = ff_st(L);
      const float sf = ff_f(S);
      coll[rl] = sf > 0.f ? Q / (sf * sf) : 0.f;
      if (lse_out) lse_out[row] = ff_f(L) * LN2;
    }
  }
}

// bf16 rows with V % 8 == 0 and 16-byte alignment: one block of TS2_NW warps
// per row.  A warp stages groups of 32 whole tiles (32 x 128 tokens, 8 KB) in
// shared memory with cp.async (double-buffered: the next group lands while
// this one is reduced), then every lane reduces one tile by itself, with no
// shuffles: the tile record (max, sum 2^{(t - max) k2}) and the lane's running
// (max, float-float sum) for the row's log-sum-exp.  Chunk j (16 bytes) of
// tile t sits at chunk j ^ (t & 7) of the tile's 256 bytes, so both the
// copies and the per-lane reads touch eight different bank groups per phase.
constexpr int TS2_NW = 3;
__device__ __forceinline__ float ex2a(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__global__ void __launch_bounds__(32 * TS2_NW)
    k_target_stats_tiles(const __nv_bfloat16* __restrict__ target, int V, int nt, int B, int Bt,
                         int Rt, float k2, float2* __restrict__ partt, float2* __restrict__ lt2,
                         float* __restrict__ coll, float* __restrict__ lse_out) {
  __shared__ __align__(16) uint4 stg[TS2_NW][2][32 * 16];  // 48 KB
  const int row = blockIdx.x;
  const int n = row / Bt, i = row - n * Bt;
  const int rl = n * (B + 1) + i;
  const uint4* tr = reinterpret_cast<const uint4*>(target + (size_t)row * V);
  const int nchunk = V >> 3;
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  const int groups = (nt + 31) >> 5;
  // lane l copies chunk (l & 15) of tiles 2k + (l >> 4) of group g into
  // buffer b; chunks past the row become bf16 -inf
  auto stage = [&](int g, int b) {
    uint4* ws = stg[w][b];
#pragma unroll
    for (int k = 0; k < 16; ++k) {
      const int tt = 2 * k + (l >> 4), j = l & 15;
      const int c = ((g << 5) + tt) * 16 + j;
      uint4* dst = ws + tt * 16 + (j ^ (tt & 7));
      if (c < nchunk) {
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(
                         static_cast<uint32_t>(__cvta_generic_to_shared(dst))),
                     "l"(tr + c)
                     : "memory");
      } else {
        *dst = make_uint4(0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u);
      }
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  };
  float rmax = -INFINITY, rsq = 0.f;
  FF rsum{0.f, 0.f};
  int buf = 0;
  if (w < groups) stage(w, 0);
  for (int g = w; g < groups; g += TS2_NW, buf ^= 1) {
    if (g + TS2_NW < groups) {
      stage(g + TS2_NW, buf ^ 1);
      asm volatile("cp.async.wait_group 1;" ::: "memory");
    } else {
      asm volatile("cp.async.wait_group 0;" ::: "memory");
    }
    __syncwarp();
    const uint4* ws = stg[w][buf];
    const int t = (g << 5) + l;
    // the tile's maximum on bf16 pairs, then the sum against it
    __nv_bfloat162 m2 = __float2bfloat162_rn(-INFINITY);
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      const uint4 q = ws[l * 16 + (j ^ (l & 7))];
      m2 = __hmax2(m2, __hmax2(__hmax2(*reinterpret_cast<const __nv_bfloat162*>(&q.x),
                                       *reinterpret_cast<const __nv_bfloat162*>(&q.y)),
                               __hmax2(*reinterpret_cast<const __nv_bfloat162*>(&q.z),
                                       *reinterpret_cast<const __nv_bfloat162*>(&q.w))));
    }
    const float mx = fmaxf(__low2float(m2), __high2float(m2));
    float s4[4] = {0.f, 0.f, 0.f, 0.f}, q4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      const uint4 q = ws[l * 16 + (j ^ (l & 7))];
      const uint32_t u[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
      for (int h = 0; h < 4; ++h) {
        const float a = __uint_as_float(u[h] << 16), b = __uint_as_float(u[h] & 0xFFFF0000u);
        const float ea = ex2a((a - mx) * k2), eb = ex2a((b - mx) * k2);
        s4[h] += ea + eb;
        q4[h] = fmaf(ea, ea, fmaf(eb, eb, q4[h]));
      }
    }
    __syncwarp();  // every lane has read this buffer before it is refilled
    if (t < nt) {
      const float s = (s4[0] + s4[1]) + (s4[2] + s4[3]);
      const float s2 = (q4[0] + q4[1]) + (q4[2] + q4[3]);
      partt[(size_t)t * Rt + rl] = make_float2(mx, s);
      if (mx > rmax) {
        const float f = exp2f((rmax - mx) * k2);
        rsum = ff_mulf(rsum, f);
        rsq *= f * f;
        rmax = mx;
      }
      const float g = exp2f((mx - rmax) * k2);
      rsum = ff_addf(rsum, s * g);
      rsq = fmaf(s2, g * g, rsq);
    }
  }
  // lanes, then warps
  float M1 = rmax;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) M1 = fmaxf(M1, __shfl_xor_sync(FULLMASK, M1, o));
  FF S1{0.f, 0.f};
  float Q1 = 0.f;
  if (M1 != -INFINITY && rmax != -INFINITY) {
    const float f = exp2f((rmax - M1) * k2);
    S1 = ff_mulf(rsum, f);
    Q1 = rsq * f * f;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    S1 = ff_add(S1, ff_shfl_xor(S1, o));
    Q1 += __shfl_xor_sync(FULLMASK, Q1, o);
  }
  // each warp's partial goes into the first entry of its own (now idle) buffer
  if (l == 0) stg[w][0][0] = make_uint4(__float_as_uint(M1), __float_as_uint(S1.hi),
                                        __float_as_uint(S1.lo), __float_as_uint(Q1));
  __syncthreads();
  if (threadIdx.x == 0) {
    float M2 = -INFINITY;
    for (int k = 0; k < TS2_NW; ++k) M2 = fmaxf(M2, __uint_as_float(stg[k][0][0].x));
    FF S{0.f, 0.f};
    float Q = 0.f;
    if (M2 != -INFINITY)
      for (int k = 0; k < TS2_NW; ++k) {
        const uint4 e = stg[k][0][0];
        const float mk = __uint_as_float(e.x);
        if (mk != -INFINITY) {
          const float f = exp2f((mk - M2) * k2);
          S = ff_add(S, ff_mulf(FF{__uint_as_float(e.y), __uint_as_float(e.z)}, f));
          Q = fmaf(__uint_as_float(e.w), f * f, Q);
        }
      }
    const FF L = (M2 == -INFINITY || !(S.hi > 0.f)) ? FF{-INFINITY, 0.f}
                                                   : ff_add(ff_prod(M2, k2), ff_log2(S));
    lt2[rl] = ff_st(L);
    const float sf = ff_f(S);
    coll[rl] = sf > 0.f ? Q / (sf * sf) : 0.f;
    if (lse_out) lse_out[row] = ff_f(L) * LN2;
  }
}

template <typename Tin>
static cudaError_t target_typed(const StepCtx& c, const dblast_verify_out* o) {
  const WsLayout& w = c.wl;
  const int Bt = w.B + (o->has_bonus ? 1 : 0);
  const int rows = w.N * Bt;
  const bool vec = (w.V % 8) == 0 && (reinterpret_cast<uintptr_t>(o->target) & 15u) == 0;
  if constexpr (std::is_same<Tin, __nv_bfloat16>::value) {
    if (vec) {
      k_target_stats_tiles<<<rows, 32 * TS2_NW, 0, c.stream>>>(
          static_cast<const __nv_bfloat16*>(o->target), w.V, w.nt, w.B, Bt, w.Rt, c.k2,
          wsp<float2>(c, w.off_partt), wsp<float2>(c, w.off_lt2), wsp<float>(c, w.off_coll),
          o->lse_target);
      debug_kernel("k_target_stats_tiles", c.stream);
      count_launches(1);
      return cudaGetLastError();
    }
  }
  k_target_stats<Tin><<<rows, TS_NT, 0, c.stream>>>(
      static_cast<const Tin*>(o->target), w.V, w.nt, w.B, Bt, w.Rt, c.k2, vec,
      wsp<float2>(c, w.off_partt), wsp<float2>(c, w.off_lt2), wsp<float>(c, w.off_coll),
      o->lse_target);
  debug_kernel("k_target_stats", c.stream);
  count_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_target_stats(const StepCtx& c, const dblast_verify_out* o) {
  return c.head->dtype == DBLAST_F32 ? target_typed<float>(c, o)
                                     : target_typed<__nv_bfloat16>(c, o);
}

// ---------------------------------------------------------------- verify side
// One block per sequence: the per-row sums of the verify records (alpha_i and
// the residual mass), acceptance (stream 2), residual or bonus draw (stream
// 3), expected lengths, emitted tokens, state update.  Warp 0 loads what the
// acceptance test needs (tokens, p and q at them, the uniforms, collision
// probabilities, the rows' branch normalisers) while warps 1.. add the
// records: thread (s, i) takes tiles s, s + S, ... of row i, consecutive
// threads on consecutive rows of a tile.
constexpr int VF_NT = 256;   // threads of the per-sequence kernels of the other modes
constexpr int VFS_NT = 512;  // threads of the stochastic-mode verify-final kernel
template <typename Tin>
__global__ void __launch_bounds__(VFS_NT, 1)
    k_verify_final(const Tin* __restrict__ target, const float* __restrict__ stash,
                   const float* __restrict__ wu, const float* __restrict__ codes,
                   const float2* __restrict__ lse2, const float2* __restrict__ w2,
                   const float* __restrict__ qtok_ws, const float2* __restrict__ lt2,
                   const float2* __restrict__ partv, const float2* __restrict__ partt,
                   const int32_t* __restrict__ tok,
                   const uint32_t* __restrict__ ties_draft, const float* __restrict__ coll, int V,
                   int K, int rr, int B, int Bt, int nt, int M, int Mpad, int Rt, float k2,
                   uint64_t seed,
                   int64_t* __restrict__ pos, uint32_t* __restrict__ rnd,
                   dblast_verify_out out, DevStatus* chk) {
  griddep_wait();  // launched as a dependent of the previous kernel
  constexpr int G = VFS_NT / TILE_V;
  __shared__ FindShared<VFS_NT> fs;
  __shared__ FF sC[32];
  __shared__ int sL;
  __shared__ uint32_t sties;
  __shared__ FF sR;
  __shared__ FF pa[VFS_NT], pr[VFS_NT];
  __shared__ FF rowA[32], rowR[32];
  __shared__ FF sCall[32 * 32];  // L_z - log2 w_z of every (i, z), +inf if w_z = 0
  __shared__ float qpart[G * TILE_V], pbuf[TILE_V];
  __shared__ float sacc[4][32];  // p(x_i), q(x_i|x_<i), u_i, coll_i
  const int n = blockIdx.x, tid = threadIdx.x, lane = tid & 31;
  const int64_t p0 = pos[n];
  const uint32_t rd = rnd[n];
  if (tid < 32) {
    // lane i: p(x_i) and q(x_i|x_<i), the acceptance uniform, coll_i, kept in
    // shared memory so that the loads complete while warps 1.. add records
    float ptok = 0.f, qtok = 1.f, u2 = 0.f, cC = 1.f;
    if (lane < B) {
      const int m = n * B + lane;
      const int x = checked_token(tok[m], V, chk, 3u);
      const FF Lt = ff_ld(lt2 + (size_t)n * (B + 1) + lane);
      const float tx = ldf(target + ((size_t)n * Bt + lane) * V + x);
      qtok = qtok_ws[m];
      cC = coll[(size_t)n * (B + 1) + lane];
      u2 = decision_uniform(seed, 2u, rd, (uint32_t)n, (uint32_t)(p0 + lane));
      ptok = (tx == -INFINITY) ? 0.f : ff_exp2(ff_sub(ff_prod(tx, k2), Lt));
    }
    sacc[0][lane] = ptok;
    sacc[1][lane] = qtok;
    sacc[2][lane] = u2;
    sacc[3][lane] = cC;
    if (lane == 0) sties = ties_draft[n];
    for (int j = lane; j < B * K; j += 32) {
      const size_t mz = (size_t)n * B * K + j;
      const FF wz = ff_ld(w2 + mz);
      sCall[j] = (wz.hi == -INFINITY) ? FF{INFINITY, 0.f} : ff_sub(ff_ld(lse2 + mz), wz);
    }
  } else {
    const int S = (VFS_NT - 32) / B;  // tile strides per row (B <= 32)
    const int t32 = tid - 32;
    FF a{0.f, 0.f}, r{0.f, 0.f};
    if (t32 < S * B) {
      const int i = t32 % B, s0 = t32 / B;
      const float2* pv = partv + (size_t)n * B + i;
      // 24 records in flight per thread
      for (int t = s0; t < nt; t += 24 * S) {
        float2 q[24];
#pragma unroll
        for (int j = 0; j < 24; ++j) {
          const int tj = t + j * S;
          q[j] = tj < nt ? pv[(size_t)tj * Mpad] : make_float2(0.f, 0.f);
        }
#pragma unroll
        for (int j = 0; j < 24; ++j) {
          a = ff_addf(a, q[j].x);
          r = ff_addf(r, q[j].y);
        }
      }
    }
    pa[tid] = a;
    pr[tid] = r;
  }
  __syncthreads();
  if (tid < B) {
    const int S = (VFS_NT - 32) / B;
    FF A{0.f, 0.f}, R{0.f, 0.f};
    for (int s0 = 0; s0 < S; ++s0) {
      A = ff_add(A, pa[32 + s0 * B + tid]);
      R = ff_add(R, pr[32 + s0 * B + tid]);
    }
    rowA[tid] = A;
    rowR[tid] = R;
  }
  __syncthreads();
  if (tid < 32) {
    // lane i: acceptance u < p/q
    const float ptok = sacc[0][lane], qtok = sacc[1][lane], u2 = sacc[2][lane];
    float cC = sacc[3][lane];
    uint32_t ties = sties;
    float A = 0.f, alpha = 0.f;
    bool acc_ok = false;
    if (lane < B) {
      const int m = n * B + lane;
      const float ratio = ptok / qtok;
      A = fminf(1.f, ratio);
      alpha = ff_f(rowA[lane]);
      acc_ok = u2 < ratio;
      if (out.p_tok) out.p_tok[m] = ptok;
      if (out.accept_prob) out.accept_prob[m] = A;
      if (out.alpha) out.alpha[m] = alpha;
      if (out.collision) out.collision[n * B + lane] = cC;
    }
    const unsigned acc_mask = __ballot_sync(FULLMASK, acc_ok);
    const unsigned rej = ~acc_mask & ((B >= 32) ? FULLMASK : ((1u << B) - 1u));
    const int L = rej ? (__ffs(rej) - 1) : B;
    // acceptance ties only for the positions that were tested (i <= L)
    const float amargin = fabsf(fmaf(u2, qtok, -ptok));
    const bool atie = lane < B && lane <= L && amargin < TIE_TOL * qtok;
    const bool anear = lane < B && lane <= L && amargin < (TIE_TOL + NEAR_ACCEPT) * qtok;
    if (__ballot_sync(FULLMASK, atie)) ties |= TIE_ACCEPT;
    if (__ballot_sync(FULLMASK, anear)) ties |= TIE_ACCEPT << NEAR_SHIFT;
    // E[L|x] = sum_i prod_{j<=i} A_j and the same over alpha; App. B: the
    // collision probabilities of the block's target rows and D_B = (1/B)
    // sum_j prod_{i<=j} coll_i (rows independent of the prefix).  Lane 0
    // forms the products and sums in position order from shared memory:
    // here that is much faster than shuffle scans of float pairs.
    sacc[0][lane] = A;
    sacc[1][lane] = alpha;
    if (L < B && lane < K) sC[lane] = sCall[L * K + lane];  // normalisers of the rejected row
    __syncwarp();
    if (lane == 0) {
      float pA = 1.f, pAl = 1.f, pC = 1.f;
      FF el{0.f, 0.f}, ea{0.f, 0.f}, ed{0.f, 0.f};
      for (int i = 0; i < B; ++i) {
        pA *= sacc[0][i];
        pAl *= sacc[1][i];
        pC *= sacc[3][i];
        el = ff_addf(el, pA);
        ea = ff_addf(ea, pAl);
        ed = ff_addf(ed, pC);
      }
      if (out.exp_len) out.exp_len[n] = ff_f(el);
      if (out.alpha_len) out.alpha_len[n] = ff_f(ea);
      if (out.determinism) out.determinism[n] = ff_f(ed) / (float)B;
      sL = L;
      sties = ties;
      sR = (L < B) ? rowR[L] : FF{0.f, 0.f};
    }
  }
  __syncthreads();
  const int L = sL;
  const FF Rm = sR;
  int extra = -1;
  bool tie = false, near = false;
  uint32_t tbits = 0;
  const int irow = (L < B) ? L : B;  // target row of the extra token
  if ((L < B) || (Bt > B)) {
    const float u3 = decision_uniform(seed, 3u, rd, (uint32_t)n, (uint32_t)(p0 + irow));
    const int rl = n * (B + 1) + irow;
    const FF Lt = ff_ld(lt2 + rl);
    const TargetTokenProb<Tin> pv{target + ((size_t)n * Bt + irow) * V, k2, Lt};
    bool from_p = (L >= B);
    if (L < B) {
      const int m = n * B + L;
      const float Rf = ff_f(Rm);
      if (Rf < TIE_TOL) tbits |= TIE_RMASS;
      if (Rf < TIE_TOL + NEAR_DRAW) tbits |= TIE_RMASS << NEAR_SHIFT;
      if (Rf > 0.f) {
        const ResidualTokenMass<Tin> rm{pv, stash + (size_t)m * V, wu, codes + (size_t)m * K * rr,
                                        sC, qpart, pbuf, K, rr, V, G, k2};
        const FindOut f = block_find<VFS_NT>(nt, V, ResidTileMass{partv + m, (size_t)Mpad}, rm,
                                             ff_mulf(Rm, u3), Rf, fs);
        extra = f.x;
        tie = f.tie;
        near = f.near;
      }
      if (extra < 0) {  // no positive residual mass left by rounding: draw from p
        from_p = true;
        tie = near = true;
        tbits |= TIE_RMASS;
      }
    }
    if (from_p) {
      const FindOut f = block_find<VFS_NT>(nt, V, TargetTileMass{partt + rl, (size_t)Rt, k2, Lt},
                                           pv, FF{u3, 0.f}, 1.f, fs);
      extra = f.x >= 0 ? f.x : 0;
      tie = tie || f.tie || f.x < 0;
      near = near || f.near || f.x < 0;
    }
  }
  if (tid == 0) {
    uint32_t tf = sties | tbits | (tie ? (uint32_t)TIE_RESID : 0u) |
                  (near ? (uint32_t)TIE_RESID << NEAR_SHIFT : 0u);
    tf |= (tf & 0xffu) << NEAR_SHIFT;  // a tie is also near
    const int ne = L + (extra >= 0 ? 1 : 0);
    if (out.accepted) out.accepted[n] = L;
    if (out.n_emitted) out.n_emitted[n] = ne;
    if (out.tie_flags) out.tie_flags[n] = tf;
    pos[n] = p0 + ne;
    rnd[n] = rd + 1u;
  }
  if (out.emitted) {
    for (int j = tid; j < B + 1; j += VFS_NT) {
      int val = -1;
      if (j < L) val = tok[n * B + j];
      else if (j == L && extra >= 0) val = extra;
      out.emitted[(size_t)n * (B + 1) + j] = val;
    }
  }
}

template <typename Tin>
static cudaError_t verify_final_typed(const StepCtx& c, const dblast_verify_out* o) {
  const int Bt = c.Bt;
  const WsLayout& w = c.wl;
  cudaError_t le = launch_dep(k_verify_final<Tin>, dim3(w.N), dim3(VFS_NT), 0, c.stream,
      static_cast<const Tin*>(o->target), wsp<float>(c, w.off_stash), prp<float>(c, c.pl.off_wu),
      wsp<float>(c, w.off_codes), wsp<float2>(c, w.off_lse2), wsp<float2>(c, w.off_w2),
      wsp<float>(c, w.off_qtok), wsp<float2>(c, w.off_lt2), wsp<float2>(c, w.off_partv),
      wsp<float2>(c, w.off_partt), wsp<int32_t>(c, w.off_tok),
      wsp<uint32_t>(c, w.off_ties), wsp<float>(c, w.off_coll), w.V, c.head->K, w.rr, w.B, Bt,
      w.nt, w.M, w.Mpad, w.Rt, c.k2, c.args->seed, c.args->pos, c.args->round, *o, c.chk);
  debug_kernel("k_verify_final", c.stream);
  count_launches(1);
  return le != cudaSuccess ? le : cudaGetLastError();
}

cudaError_t launch_verify_finalize(const StepCtx& c, const dblast_verify_out* o) {
  return c.head->dtype == DBLAST_F32 ? verify_final_typed<float>(c, o)
                                     : verify_final_typed<__nv_bfloat16>(c, o);
}

// ---------------------------------------------------------------- greedy-branch mode
// Sec. 3.1 ("Drafter sampling during inference") and App. A: the draft pass
// leaves per-tile records partd[t][z][m] = (max logit, token) of every
// branch; these kernels take x-hat_{i,z}, the block x_i = x-hat_{i,z-hat}, the
// consistent-branch sets C_i and q_greedy (Eq. appendix-greedy-conditional),
// and verify with it.  q_greedy has at most K atoms per position, so p is
// needed only at those tokens, plus the target tile records for the residual
// and bonus draws.
// top-two merge of (max, index, second) with a record (v, i, vs): ties to
// the lower index; the second of the union is the larger of the losing max
// and the winner's own second
__device__ __forceinline__ void arg_keep2(float& mx, int& ix, float& sc, float v, int i, float vs) {
  if (v > mx || (v == mx && i < ix)) {
    sc = fmaxf(mx, vs);
    mx = v;
    ix = i;
  } else {
    sc = fmaxf(sc, v);
  }
}

// Partial argmax of the draft records: block (row group of 32, z, split), lane
// = row, warps and splits interleave over the tiles (as k_draft_lse).
// lsep[sp][m][z] = (max, token bits, second-largest logit, 0).
__global__ void __launch_bounds__(LSE_WARPS * 32)
    k_greedy_argmax(const float2* __restrict__ partd, const float* __restrict__ partg, int nt,
                    int K, int M, int Mpad, float4* __restrict__ lsep) {
  griddep_wait();  // launched as a dependent of the previous kernel
  __shared__ float smx[LSE_WARPS][32], ssc[LSE_WARPS][32];
  __shared__ int six[LSE_WARPS][32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int m = blockIdx.x * 32 + lane, z = blockIdx.y, sp = blockIdx.z;
  const int step = LSE_WARPS * LSE_SPLIT;
  float mx = -INFINITY, sc = -INFINITY;
  int ix = 0x7fffffff;
  if (m < M) {
    const float2* p = partd + (size_t)z * Mpad + m;
    const float* g = partg + (size_t)z * Mpad + m;
    const size_t st = (size_t)K * Mpad;
    int t = sp * LSE_WARPS + warp;
    for (; t + 3 * step < nt; t += 4 * step) {
      const float2 q0 = p[(size_t)t * st], q1 = p[(size_t)(t + step) * st];
      const float2 q2 = p[(size_t)(t + 2 * step) * st], q3 = p[(size_t)(t + 3 * step) * st];
      const float g0 = g[(size_t)t * st], g1 = g[(size_t)(t + step) * st];
      const float g2 = g[(size_t)(t + 2 * step) * st], g3 = g[(size_t)(t + 3 * step) * st];
      arg_keep2(mx, ix, sc, q0.x, __float_as_int(q0.y), g0);
      arg_keep2(mx, ix, sc, q1.x, __float_as_int(q1.y), g1);
      arg_keep2(mx, ix, sc, q2.x, __float_as_int(q2.y), g2);
      arg_keep2(mx, ix, sc, q3.x, __float_as_int(q3.y), g3);
    }
    for (; t < nt; t += step) {
      const float2 q = p[(size_t)t * st];
      arg_keep2(mx, ix, sc, q.x, __float_as_int(q.y), g[(size_t)t * st]);
    }
  }
  smx[warp][lane] = mx;
  six[warp][lane] = ix;
  ssc[warp][lane] = sc;
  __syncthreads();
  if (warp == 0 && m < M) {
#pragma unroll
    for (int w = 1; w < LSE_WARPS; ++w) arg_keep2(mx, ix, sc, smx[w][lane], six[w][lane], ssc[w][lane]);
    lsep[((size_t)sp * M + m) * K + z] = make_float4(mx, __int_as_float(ix), sc, 0.f);
  }
}

// One block per sequence, thread t = (i, z) with i = t / K: x-hat_{i,z}, the
// block, C_i (bit z of cmask[m]: branch z drafted x_j at every j < i),
// pi~_{i,z} and q_greedy(x_i|x_<i), and the user-visible draft outputs.
// The draft side of one sequence, for any block size: x-hat_{i,z} (thread
// (i, z), strided), the block, C_i (bit z of cmask[m]: branch z drafted x_j at
// every j < i), pi~_{i,z} and q_greedy(x_i|x_<i), and the draft outputs.
// An argmax of a branch in C_i whose top-two logit gap is below
// GREEDY_TIE_TOL sets the draft tie bit of the sequence (ties_ws[n]).
// Shared arrays: X [B K], tokS, eqS, nearS, cmS, piS, sumS [32].
__device__ void greedy_draft_body(const float4* __restrict__ lsep, const float* __restrict__ log2pi,
                                  const int32_t* __restrict__ zhat, int n, int B, int K, int M,
                                  int V, int32_t* __restrict__ xhat_ws, int32_t* __restrict__ tok_ws,
                                  float* __restrict__ qtok_ws, uint32_t* __restrict__ cmask_ws,
                                  uint32_t* __restrict__ ties_ws, const dblast_draft_out& out,
                                  int* X, int* tokS, uint32_t* eqS, uint32_t* nearS, uint32_t* cmS,
                                  float* piS, float* sumS, float* qS) {
  const int nt = blockDim.x;
  if (threadIdx.x < 32) {
    eqS[threadIdx.x] = 0u;
    nearS[threadIdx.x] = 0u;
  }
  __syncthreads();
  for (int t = threadIdx.x; t < B * K; t += nt) {
    const int i = t / K, z = t - i * K;
    const size_t m = (size_t)n * B + i;
    float mx = -INFINITY, sc = -INFINITY;
    int ix = 0x7fffffff;
#pragma unroll
    for (int sp = 0; sp < LSE_SPLIT; ++sp) {
      const float4 q = lsep[((size_t)sp * M + m) * K + z];
      arg_keep2(mx, ix, sc, q.x, __float_as_int(q.y), q.z);
    }
    // top-two gap (0 for equal logits; NaN logits compare false and count as near)
    if (!(mx - sc >= GREEDY_TIE_TOL)) atomicOr(&nearS[i], 1u << z);
    ix = min(max(ix, 0), V - 1);  // every logit NaN: not a token, keep the index valid
    X[t] = ix;
    xhat_ws[m * K + z] = ix;
    if (out.branch_tokens) out.branch_tokens[m * K + z] = ix;
  }
  if ((int)threadIdx.x < K) piS[threadIdx.x] = exp2f(log2pi[n * K + threadIdx.x]);  // -inf gives 0
  __syncthreads();
  const int zh = zhat[n];
  if ((int)threadIdx.x < B) tokS[threadIdx.x] = X[threadIdx.x * K + zh];
  __syncthreads();
  for (int t = threadIdx.x; t < B * K; t += nt) {
    const int i = t / K, z = t - i * K;
    if (X[t] == tokS[i]) atomicOr(&eqS[i], 1u << z);
  }
  __syncthreads();
  if ((int)threadIdx.x < B) {  // C_t = branches that drafted x_j at every j < t
    const int t = threadIdx.x;
    uint32_t c = (K >= 32) ? 0xffffffffu : ((1u << K) - 1u);
    for (int j = 0; j < t; ++j) c &= eqS[j];
    cmS[t] = c;
    if (c & nearS[t]) atomicOr(&ties_ws[n], (uint32_t)TIE_DRAFT | ((uint32_t)TIE_DRAFT << NEAR_SHIFT));
    float S = 0.f, Q = 0.f;
    for (int k = 0; k < K; ++k) {
      if ((c >> k) & 1u) {
        S += piS[k];
        if ((eqS[t] >> k) & 1u) Q += piS[k];
      }
    }
    sumS[t] = S;
    const size_t mt = (size_t)n * B + t;
    const float qt = S > 0.f ? Q / S : 0.f;
    tok_ws[mt] = tokS[t];
    qtok_ws[mt] = qt;
    qS[t] = qt;
    cmask_ws[mt] = c;
    if (out.tokens) out.tokens[mt] = tokS[t];
    if (out.q_tok) out.q_tok[mt] = qt;
  }
  __syncthreads();
  if (out.logw)
    for (int t = threadIdx.x; t < B * K; t += nt) {
      const int i = t / K, z = t - i * K;
      const bool in = (cmS[i] >> z) & 1u;
      const float w = (in && sumS[i] > 0.f) ? piS[z] / sumS[i] : 0.f;
      out.logw[((size_t)n * B + i) * K + z] = w > 0.f ? logf(w) : -INFINITY;
    }
  if ((int)threadIdx.x < K && out.pi) out.pi[n * K + threadIdx.x] = piS[threadIdx.x];
  if (threadIdx.x == 0 && out.z_hat) out.z_hat[n] = zh;
}

__global__ void __launch_bounds__(1024)
    k_greedy_draft(const float4* __restrict__ lsep, const float* __restrict__ log2pi,
                   const int32_t* __restrict__ zhat, int B, int K, int M, int V,
                   int32_t* __restrict__ xhat_ws, int32_t* __restrict__ tok_ws,
                   float* __restrict__ qtok_ws, uint32_t* __restrict__ cmask_ws,
                   uint32_t* __restrict__ ties_ws, dblast_draft_out out) {
  griddep_wait();  // launched as a dependent of the previous kernel
  __shared__ int X[1024];
  __shared__ int tokS[32];
  __shared__ uint32_t eqS[32], nearS[32], cmS[32];
  __shared__ float piS[32], sumS[32], qS[32];
  greedy_draft_body(lsep, log2pi, zhat, blockIdx.x, B, K, M, V, xhat_ws, tok_ws, qtok_ws, cmask_ws,
                    ties_ws, out, X, tokS, eqS, nearS, cmS, piS, sumS, qS);
}

cudaError_t launch_greedy_draft_finalize(const StepCtx& c, const dblast_draft_out* outp) {
  const WsLayout& w = c.wl;
  const int K = c.head->K;
  cudaError_t le =
      launch_dep(k_greedy_argmax, dim3(ceil_div(w.M, 32), K, LSE_SPLIT), dim3(LSE_WARPS * 32), 0,
                 c.stream, wsp<float2>(c, w.off_partd), wsp<float>(c, w.off_partg), w.nt, K, w.M,
                 w.Mpad, wsp<float4>(c, w.off_lsep));
  debug_kernel("k_greedy_argmax", c.stream);
  dblast_draft_out out{};
  if (outp) out = *outp;
  const int pt = ceil_div(w.B * K, 32) * 32;
  if (le == cudaSuccess) le = launch_dep(k_greedy_draft, dim3(w.N), dim3(pt), 0, c.stream,
      wsp<float4>(c, w.off_lsep), wsp<float>(c, w.off_log2pi), wsp<int32_t>(c, w.off_zhat), w.B,
      K, w.M, w.V, wsp<int32_t>(c, w.off_xhat), wsp<int32_t>(c, w.off_tok),
      wsp<float>(c, w.off_qtok), wsp<uint32_t>(c, w.off_cmask), wsp<uint32_t>(c, w.off_ties), out);
  debug_kernel("k_greedy_draft", c.stream);
  count_launches(2);
  return le != cudaSuccess ? le : cudaGetLastError();
}

// Residual masses of the greedy conditional at the rejected row: the target
// tile records, except for tiles holding an atom, whose masses are summed
// token by token in shared memory (no cancellation of p_tile - q).
struct GreedyResidTileMass {
  TargetTileMass pt;
  const int* atile;   // tile of atom k, -1 if an earlier atom has the same tile
  const float* amass; // token-level residual mass of that tile
  int na;
  __device__ float operator()(int t) const {
    for (int k = 0; k < na; ++k)
      if (atile[k] == t) return amass[k];
    return pt(t);
  }
};
template <typename Tin> struct GreedyResidTokenMass {  // [p(v) - q_greedy(v)]_+
  TargetTokenProb<Tin> p;
  const int* atok;
  const float* aq;
  int na;
  __device__ float operator()(int v) const {
    float q = 0.f;
    for (int k = 0; k < na; ++k)
      if (atok[k] == v) q += aq[k];
    return fmaxf(p(v) - q, 0.f);
  }
};

// One block per sequence: p at the atoms of q_greedy, acceptance (stream 2),
// alpha_i = sum over atoms of min(p, q), residual or bonus draw (stream 3),
// expected lengths, emitted tokens, state update.
// The draft side when the verify kernel also takes the greedy draft (fused
// step): the argmax partials in, the draft outputs and workspace rows out.
struct GreedyDraftArgs {
  const float4* lsep;
  const int32_t* zhat;
  int M;
  int32_t* xhat_ws;
  int32_t* tok_ws;
  float* qtok_ws;
  uint32_t* cmask_ws;
  uint32_t* ties_ws;
  dblast_draft_out out;
};

template <typename Tin, bool WITH_DRAFT>
__global__ void __launch_bounds__(VF_NT)
    k_greedy_verify(const Tin* __restrict__ target, const float* __restrict__ log2pi,
                    const int32_t* xhat, const uint32_t* cmask, const float* qtok_ws,
                    const float2* __restrict__ lt2, const float2* __restrict__ partt,
                    const int32_t* tok, const uint32_t* ties_draft, const float* __restrict__ coll,
                    int V, int K, int B, int Bt, int nt, int Rt, float k2, uint64_t seed,
                    int64_t* __restrict__ pos, uint32_t* __restrict__ rnd, dblast_verify_out out,
                    GreedyDraftArgs gd, DevStatus* chk) {
  griddep_wait();  // launched as a dependent of the previous kernel
  __shared__ FindShared<VF_NT> fs;
  __shared__ int X[1024];
  __shared__ float piS[32];
  __shared__ int atok[32], atile[32];
  __shared__ float aq[32], amass[32];
  __shared__ uint32_t cmS[32];
  __shared__ float SS[32];
  __shared__ int tokS[32];
  __shared__ uint32_t eqS[32], nearS[32];
  __shared__ float qS[32];
  __shared__ float T[1024];  // min(p, q) of each distinct atom, at its first branch
  __shared__ int sL, sna;
  __shared__ uint32_t sties;
  __shared__ float sR;
  const int n = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t p0 = pos[n];
  const uint32_t rd = rnd[n];
  if constexpr (WITH_DRAFT) {
    greedy_draft_body(gd.lsep, log2pi, gd.zhat, n, B, K, gd.M, V, gd.xhat_ws, gd.tok_ws,
                      gd.qtok_ws, gd.cmask_ws, gd.ties_ws, gd.out, X, tokS, eqS, nearS, cmS, piS,
                      SS, qS);
    __syncthreads();
  } else {
    for (int j = tid; j < B * K; j += VF_NT) X[j] = xhat[(size_t)n * B * K + j];
    if (tid < K) piS[tid] = exp2f(log2pi[n * K + tid]);
    if (tid < B) {
      cmS[tid] = cmask[(size_t)n * B + tid];
      tokS[tid] = tok[(size_t)n * B + tid];
      qS[tid] = qtok_ws[(size_t)n * B + tid];
    }
    __syncthreads();
    if (tid < B) {
      float S = 0.f;
      for (int k = 0; k < K; ++k)
        if ((cmS[tid] >> k) & 1u) S += piS[k];
      SS[tid] = S;
    }
    __syncthreads();
  }
  // one term min(p(a), q(a)) per distinct token a of the branches in C_i, a
  // thread per (i, z): the first branch of C_i with that token carries it
  for (int t = tid; t < B * K; t += VF_NT) {
    const int i = t / K, z = t - i * K;
    const uint32_t c = cmS[i];
    float term = 0.f;
    if ((c >> z) & 1u) {
      const int a = X[t];
      bool first = true;
      float qa = 0.f;
      for (int k = 0; k < K; ++k) {
        if (!((c >> k) & 1u) || X[i * K + k] != a) continue;
        if (k < z) first = false;
        qa += piS[k];
      }
      if (first) {
        const float ta = ldf(target + ((size_t)n * Bt + i) * V + a);
        const FF Lt = ff_ld(lt2 + (size_t)n * (B + 1) + i);
        const float pa = (ta == -INFINITY) ? 0.f : ff_exp2(ff_sub(ff_prod(ta, k2), Lt));
        term = fminf(pa, SS[i] > 0.f ? qa / SS[i] : 0.f);
      }
    }
    T[t] = term;
  }
  __syncthreads();
  if (tid < 32) {
    uint32_t ties = ties_draft[n];
    float A = 0.f, alpha = 0.f, ptok = 0.f, qtok = 1.f, u2 = 0.f;
    bool acc_ok = false;
    uint32_t c = 0u;
    float S = 0.f;
    if (lane < B) {
      const int m = n * B + lane;
      const int x = checked_token(tokS[lane], V, chk, 4u);
      const FF Lt = ff_ld(lt2 + (size_t)n * (B + 1) + lane);
      const float tx = ldf(target + ((size_t)n * Bt + lane) * V + x);
      ptok = (tx == -INFINITY) ? 0.f : ff_exp2(ff_sub(ff_prod(tx, k2), Lt));
      qtok = qS[lane];
      const float ratio = ptok / qtok;
      A = fminf(1.f, ratio);
      c = cmS[lane];
      S = SS[lane];
      FF al{0.f, 0.f};
      for (int k = 0; k < K; ++k) al = ff_addf(al, T[lane * K + k]);
      alpha = ff_f(al);
      u2 = decision_uniform(seed, 2u, rd, (uint32_t)n, (uint32_t)(p0 + lane));
      acc_ok = u2 < ratio;
      if (out.p_tok) out.p_tok[m] = ptok;
      if (out.accept_prob) out.accept_prob[m] = A;
      if (out.alpha) out.alpha[m] = alpha;
    }
    const unsigned acc_mask = __ballot_sync(FULLMASK, acc_ok);
    const unsigned rej = ~acc_mask & ((B >= 32) ? FULLMASK : ((1u << B) - 1u));
    const int L = rej ? (__ffs(rej) - 1) : B;
    const float amargin = fabsf(fmaf(u2, qtok, -ptok));
    const bool atie = lane < B && lane <= L && amargin < TIE_TOL * qtok;
    const bool anear = lane < B && lane <= L && amargin < (TIE_TOL + NEAR_ACCEPT) * qtok;
    if (__ballot_sync(FULLMASK, atie)) ties |= TIE_ACCEPT;
    if (__ballot_sync(FULLMASK, anear)) ties |= TIE_ACCEPT << NEAR_SHIFT;
    // App. B: collision probabilities of the block's target rows and
    // D_B = (1/B) sum_j prod_{i<=j} coll_i (rows independent of the prefix)
    float cC = 1.f;
    if (lane < B) {
      cC = coll[(size_t)n * (B + 1) + lane];
      if (out.collision) out.collision[n * B + lane] = cC;
    }
    float cA = (lane < B) ? A : 1.f, cAl = (lane < B) ? alpha : 1.f;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const float ta = __shfl_up_sync(FULLMASK, cA, o);
      const float tl = __shfl_up_sync(FULLMASK, cAl, o);
      const float tc = __shfl_up_sync(FULLMASK, cC, o);
      if (lane >= o) {
        cA *= ta;
        cAl *= tl;
        cC *= tc;
      }
    }
    FF el{lane < B ? cA : 0.f, 0.f}, ea{lane < B ? cAl : 0.f, 0.f};
    FF ed{lane < B ? cC : 0.f, 0.f};
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      el = ff_add(el, ff_shfl_xor(el, o));
      ea = ff_add(ea, ff_shfl_xor(ea, o));
      ed = ff_add(ed, ff_shfl_xor(ed, o));
    }
    // the atoms of the rejected row: token, q_greedy, the tile (first atom of a tile only)
    if (L < B && lane == L) {
      int na = 0;
      for (int k = 0; k < K; ++k) {
        if (!((c >> k) & 1u)) continue;
        const int a = X[L * K + k];
        int j = 0;
        while (j < na && atok[j] != a) ++j;
        if (j == na) {
          atok[na] = a;
          aq[na] = 0.f;
          ++na;
        }
        aq[j] += S > 0.f ? piS[k] / S : 0.f;
      }
      for (int j = 0; j < na; ++j) {
        const int tj = atok[j] / TILE_V;
        bool first = true;
        for (int j2 = 0; j2 < j; ++j2) first = first && (atok[j2] / TILE_V != tj);
        atile[j] = first ? tj : -1;
      }
      sna = na;
      sR = 1.f - alpha;  // residual mass, for the tie flag
    }
    if (lane == 0) {
      if (out.exp_len) out.exp_len[n] = ff_f(el);
      if (out.alpha_len) out.alpha_len[n] = ff_f(ea);
      if (out.determinism) out.determinism[n] = ff_f(ed) / (float)B;
      sL = L;
      sties = ties;
    }
  }
  __syncthreads();
  const int L = sL;
  int extra = -1;
  bool tie = false, near = false;
  uint32_t tbits = 0;
  const int irow = (L < B) ? L : B;  // target row of the extra token
  if ((L < B) || (Bt > B)) {
    const float u3 = decision_uniform(seed, 3u, rd, (uint32_t)n, (uint32_t)(p0 + irow));
    const int rl = n * (B + 1) + irow;
    const FF Lt = ff_ld(lt2 + rl);
    const TargetTokenProb<Tin> pv{target + ((size_t)n * Bt + irow) * V, k2, Lt};
    const TargetTileMass ptm{partt + rl, (size_t)Rt, k2, Lt};
    bool from_p = (L >= B);
    if (L < B) {
      const int na = sna;
      const GreedyResidTokenMass<Tin> rm{pv, atok, aq, na};
      // token-level residual mass of every tile that holds an atom, one warp per tile
      for (int j = warp; j < na; j += VF_NT / 32) {
        if (atile[j] < 0) continue;
        FF sm{0.f, 0.f};
        for (int o = lane; o < TILE_V; o += 32) {
          const int v = atile[j] * TILE_V + o;
          if (v < V) sm = ff_addf(sm, rm(v));
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) sm = ff_add(sm, ff_shfl_xor(sm, o));
        if (lane == 0) amass[j] = ff_f(sm);
      }
      __syncthreads();
      if (sR < TIE_TOL) tbits |= TIE_RMASS;
      if (sR < TIE_TOL + NEAR_DRAW) tbits |= TIE_RMASS << NEAR_SHIFT;
      const FindOut f = block_find<VF_NT>(nt, V, GreedyResidTileMass{ptm, atile, amass, na}, rm,
                                          FF{u3, 0.f}, 1.f, fs, true);
      extra = f.x;
      tie = f.tie;
      near = f.near;
      if (extra < 0) {  // no positive residual mass left by rounding: draw from p
        from_p = true;
        tie = near = true;
        tbits |= TIE_RMASS;
      }
    }
    if (from_p) {
      const FindOut f = block_find<VF_NT>(nt, V, ptm, pv, FF{u3, 0.f}, 1.f, fs);
      extra = f.x >= 0 ? f.x : 0;
      tie = tie || f.tie || f.x < 0;
      near = near || f.near || f.x < 0;
    }
  }
  if (tid == 0) {
    uint32_t ties = sties | tbits | (tie ? (uint32_t)TIE_RESID : 0u) |
                    (near ? (uint32_t)TIE_RESID << NEAR_SHIFT : 0u);
    ties |= (ties & 0xffu) << NEAR_SHIFT;  // a tie is also near
    const int ne = L + (extra >= 0 ? 1 : 0);
    if (out.accepted) out.accepted[n] = L;
    if (out.n_emitted) out.n_emitted[n] = ne;
    if (out.tie_flags) out.tie_flags[n] = ties;
    pos[n] = p0 + ne;
    rnd[n] = rd + 1u;
  }
  if (out.emitted) {
    for (int j = tid; j < B + 1; j += VF_NT) {
      int val = -1;
      if (j < L) val = tokS[j];
      else if (j == L && extra >= 0) val = extra;
      out.emitted[(size_t)n * (B + 1) + j] = val;
    }
  }
}

template <typename Tin, bool WITH_DRAFT>
static cudaError_t greedy_verify_typed(const StepCtx& c, const dblast_verify_out* o,
                                       const dblast_draft_out* dout) {
  const WsLayout& w = c.wl;
  GreedyDraftArgs gd{};
  if (WITH_DRAFT) {
    gd.lsep = wsp<float4>(c, w.off_lsep);
    gd.zhat = wsp<int32_t>(c, w.off_zhat);
    gd.M = w.M;
    gd.xhat_ws = wsp<int32_t>(c, w.off_xhat);
    gd.tok_ws = wsp<int32_t>(c, w.off_tok);
    gd.qtok_ws = wsp<float>(c, w.off_qtok);
    gd.cmask_ws = wsp<uint32_t>(c, w.off_cmask);
    gd.ties_ws = wsp<uint32_t>(c, w.off_ties);
    if (dout) gd.out = *dout;
  }
  cudaError_t le = launch_dep(k_greedy_verify<Tin, WITH_DRAFT>, dim3(w.N), dim3(VF_NT), 0, c.stream,
      static_cast<const Tin*>(o->target), wsp<float>(c, w.off_log2pi),
      wsp<int32_t>(c, w.off_xhat), wsp<uint32_t>(c, w.off_cmask), wsp<float>(c, w.off_qtok),
      wsp<float2>(c, w.off_lt2), wsp<float2>(c, w.off_partt), wsp<int32_t>(c, w.off_tok),
      wsp<uint32_t>(c, w.off_ties), wsp<float>(c, w.off_coll), w.V, c.head->K, w.B, c.Bt, w.nt,
      w.Rt, c.k2, c.args->seed, c.args->pos, c.args->round, *o, gd, c.chk);
  debug_kernel("k_greedy_verify", c.stream);
  count_launches(1);
  return le != cudaSuccess ? le : cudaGetLastError();
}

cudaError_t launch_greedy_verify_finalize(const StepCtx& c, const dblast_verify_out* o) {
  return c.head->dtype == DBLAST_F32 ? greedy_verify_typed<float, false>(c, o, nullptr)
                                     : greedy_verify_typed<__nv_bfloat16, false>(c, o, nullptr);
}

// Fused step, greedy mode without a filter: the argmax partials, then one
// kernel per sequence that takes the greedy draft and verifies it.
cudaError_t launch_greedy_step_finalize(const StepCtx& c, const dblast_draft_out* dout,
                                        const dblast_verify_out* o) {
  const WsLayout& w = c.wl;
  const int K = c.head->K;
  cudaError_t le =
      launch_dep(k_greedy_argmax, dim3(ceil_div(w.M, 32), K, LSE_SPLIT), dim3(LSE_WARPS * 32), 0,
                 c.stream, wsp<float2>(c, w.off_partd), wsp<float>(c, w.off_partg), w.nt, K, w.M,
                 w.Mpad, wsp<float4>(c, w.off_lsep));
  debug_kernel("k_greedy_argmax", c.stream);
  count_launches(1);
  if (le != cudaSuccess) return le;
  return c.head->dtype == DBLAST_F32 ? greedy_verify_typed<float, true>(c, o, dout)
                                     : greedy_verify_typed<__nv_bfloat16, true>(c, o, dout);
}

// ---------------------------------------------------------------- early determinism
// App. B.  The target statistics give every row's tile records, log-sum-exp
// and collision probability; k_target_sample draws x_i^(m) ~ p_i (one block
// per (i, m, n), the two-level inverse CDF of the bonus draw with the
// stream-4 uniform) and keeps p_i(x_i^(m)); k_determinism_reduce forms
// D_exact from the collision probabilities and D-hat from the samples.
template <typename Tin>
__global__ void __launch_bounds__(VF_NT)
    k_target_sample(const Tin* __restrict__ target, const float2* __restrict__ partt,
                    const float2* __restrict__ lt2, int V, int nt, int rows, int b, int M, int Rt,
                    float k2, uint64_t seed, float* __restrict__ pval, int32_t* __restrict__ samples) {
  griddep_wait();  // launched as a dependent of the previous kernel
  __shared__ FindShared<VF_NT> fs;
  const int i = blockIdx.x, m = blockIdx.y, n = blockIdx.z;
  const int rl = n * rows + i;
  const FF Lt = ff_ld(lt2 + rl);
  const TargetTokenProb<Tin> pv{target + (size_t)rl * V, k2, Lt};
  const float u = decision_uniform(seed, 4u, (uint32_t)m, (uint32_t)n, (uint32_t)i);
  const FindOut f = block_find<VF_NT>(nt, V, TargetTileMass{partt + rl, (size_t)Rt, k2, Lt}, pv,
                                      FF{u, 0.f}, 1.f, fs);
  if (threadIdx.x == 0) {
    const int x = f.x >= 0 ? f.x : 0;
    const size_t o = ((size_t)n * M + m) * b + i;
    pval[o] = pv(x);
    if (samples) samples[o] = x;
  }
}

// All M draws of one target row in one block: the inclusive prefix of the
// tile masses is scanned once into shared memory; each warp then takes a
// draw, finds its tile by binary search and scans the tile's 128 tokens
// (four per lane).  The decisions are those of the block-wide two-level draw
// of k_target_sample.
constexpr int TSR_MAX_TILES = 5120;  // prefix in shared memory (40 KB)
template <typename Tin>
__global__ void __launch_bounds__(VF_NT)
    k_target_sample_row(const Tin* __restrict__ target, const float2* __restrict__ partt,
                        const float2* __restrict__ lt2, int V, int nt, int rows, int b, int M,
                        int Rt, float k2, uint64_t seed, float* __restrict__ pval,
                        int32_t* __restrict__ samples) {
  griddep_wait();  // launched as a dependent of the previous kernel
  extern __shared__ FF pre[];  // [nt] inclusive prefix of the tile masses
  __shared__ FF sh[VF_NT / 32];
  const int i = blockIdx.x, n = blockIdx.y;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int rl = n * rows + i;
  const FF Lt = ff_ld(lt2 + rl);
  const TargetTokenProb<Tin> pv{target + (size_t)rl * V, k2, Lt};
  const TargetTileMass tm{partt + rl, (size_t)Rt, k2, Lt};
  const int chunk = ceil_div(nt, VF_NT);
  const int t0 = min(nt, tid * chunk), t1 = min(nt, t0 + chunk);
  FF loc{0.f, 0.f};
  for (int t = t0; t < t1; ++t) {
    const float w = tm(t);
    loc = ff_addf(loc, w);
    pre[t] = FF{w, 0.f};  // the mass for now, the prefix below
  }
  const BlockScan sc = block_scan_ff<VF_NT>(loc, sh);
  FF run = sc.excl;
  for (int t = t0; t < t1; ++t) {
    run = ff_add(run, pre[t]);
    pre[t] = run;
  }
  __syncthreads();
  for (int m = warp; m < M; m += VF_NT / 32) {
    const FF target{decision_uniform(seed, 4u, (uint32_t)m, (uint32_t)n, (uint32_t)i), 0.f};
    int lo = 0, hi = nt;
    while (lo < hi) {
      const int mid = (lo + hi) >> 1;
      if (ff_gt(pre[mid], target)) hi = mid;
      else lo = mid + 1;
    }
    int tt = lo;
    if (tt >= nt) {  // rounding left the target at the total: the last tile with mass
      tt = nt - 1;
      while (tt > 0 && !(ff_gt(pre[tt], pre[tt - 1]))) --tt;
    }
    const FF before = tt > 0 ? pre[tt - 1] : FF{0.f, 0.f};
    float e[4];
    FF cum[4];
    FF acc{0.f, 0.f};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int v = tt * TILE_V + lane * 4 + j;
      e[j] = v < V ? pv(v) : 0.f;
      acc = ff_addf(acc, e[j]);
      cum[j] = acc;
    }
    FF incl = acc;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const FF t = ff_shfl_up(incl, o);
      if (lane >= o) incl = ff_add(t, incl);
    }
    FF excl = ff_shfl_up(incl, 1);
    if (lane == 0) excl = FF{0.f, 0.f};
    const FF base = ff_add(before, excl);
    int jj = 4;
#pragma unroll
    for (int j = 3; j >= 0; --j)
      if (ff_gt(ff_add(base, cum[j]), target)) jj = j;
    const unsigned hit = __ballot_sync(FULLMASK, jj < 4);
    int x;
    if (hit) {
      const int l = __ffs(hit) - 1;
      x = tt * TILE_V + l * 4 + __shfl_sync(FULLMASK, jj, l);
    } else {  // the last token with mass
      int lj = -1;
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (e[j] > 0.f) lj = j;
      const unsigned pos = __ballot_sync(FULLMASK, lj >= 0);
      const int l = pos ? 31 - __clz(pos) : 0;
      x = tt * TILE_V + l * 4 + max(__shfl_sync(FULLMASK, lj, l), 0);
    }
    if (lane == 0) {
      x = min(x, V - 1);
      const size_t o = ((size_t)n * M + m) * b + i;
      pval[o] = pv(x);
      if (samples) samples[o] = x;
    }
  }
}

constexpr int DR_NT = 256;
__global__ void __launch_bounds__(DR_NT)
    k_determinism_reduce(const float* __restrict__ coll, const float* __restrict__ pval, int rows,
                         int b, int M, float* __restrict__ collision, float* __restrict__ d_exact,
                         float* __restrict__ d_hat) {
  griddep_wait();  // launched as a dependent of the previous kernel
  __shared__ FF red[DR_NT / 32];
  const int n = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (tid == 0) {
    FF d{0.f, 0.f};
    float c = 1.f;
    for (int i = 0; i < b; ++i) {
      const float ci = coll[(size_t)n * rows + i];
      if (collision) collision[n * b + i] = ci;
      c *= ci;
      d = ff_addf(d, c);
    }
    if (d_exact) d_exact[n] = ff_f(d) / (float)b;
  }
  if (!d_hat) return;  // uniform over the block
  FF acc{0.f, 0.f};
  for (int m = tid; m < M; m += DR_NT) {
    const float* pv = pval + ((size_t)n * M + m) * b;
    float c = 1.f;
    for (int i = 0; i < b; ++i) {
      c *= pv[i];
      acc = ff_addf(acc, c);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc = ff_add(acc, ff_shfl_xor(acc, o));
  if (lane == 0) red[warp] = acc;
  __syncthreads();
  if (tid == 0) {
    FF t{0.f, 0.f};
    for (int w = 0; w < DR_NT / 32; ++w) t = ff_add(t, red[w]);
    d_hat[n] = ff_f(t) / ((float)M * (float)b);
  }
}

template <typename Tin>
static cudaError_t determinism_typed(const StepCtx& c, const dblast_verify_out* o, int rows, int b,
                                     int M, uint64_t seed, float* collision, float* d_exact,
                                     float* d_hat, int32_t* samples, size_t off_pval) {
  const WsLayout& w = c.wl;
  cudaError_t e = launch_target_stats(c, o);
  if (e == cudaSuccess && (d_hat || samples)) {
    if (w.nt <= TSR_MAX_TILES) {
      const size_t sm = (size_t)w.nt * sizeof(FF);
      e = sm > 48 * 1024 ? cudaFuncSetAttribute(k_target_sample_row<Tin>,
                                                 cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm)
                         : cudaSuccess;
      if (e == cudaSuccess)
        e = launch_dep(k_target_sample_row<Tin>, dim3(b, w.N), dim3(VF_NT), sm, c.stream,
                       static_cast<const Tin*>(o->target), wsp<float2>(c, w.off_partt),
                       wsp<float2>(c, w.off_lt2), w.V, w.nt, rows, b, M, w.Rt, c.k2, seed,
                       wsp<float>(c, off_pval), samples);
      debug_kernel("k_target_sample_row", c.stream);
    } else {
      e = launch_dep(k_target_sample<Tin>, dim3(b, M, w.N), dim3(VF_NT), 0, c.stream,
                     static_cast<const Tin*>(o->target), wsp<float2>(c, w.off_partt),
                     wsp<float2>(c, w.off_lt2), w.V, w.nt, rows, b, M, w.Rt, c.k2, seed,
                     wsp<float>(c, off_pval), samples);
      debug_kernel("k_target_sample", c.stream);
    }
    count_launches(1);
  }
  if (e == cudaSuccess) {
    e = launch_dep(k_determinism_reduce, dim3(w.N), dim3(DR_NT), 0, c.stream,
                   wsp<float>(c, w.off_coll), wsp<float>(c, off_pval), rows, b, M, collision,
                   d_exact, d_hat);
    debug_kernel("k_determinism_reduce", c.stream);
    count_launches(1);
  }
  return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t launch_determinism(const StepCtx& c, const dblast_verify_out* o, int rows, int b,
                               int M, uint64_t seed, float* collision, float* d_exact,
                               float* d_hat, int32_t* samples, size_t off_pval) {
  return c.head->dtype == DBLAST_F32
             ? determinism_typed<float>(c, o, rows, b, M, seed, collision, d_exact, d_hat,
                                        samples, off_pval)
             : determinism_typed<__nv_bfloat16>(c, o, rows, b, M, seed, collision, d_exact, d_hat,
                                                samples, off_pval);
}

// ---------------------------------------------------------------- target filter
// Sec. 3.2 / Sec. 4: verification against the target after temperature,
// top-k and top-p.  k_target_filter (one block per target row) finds the kept
// set from the tile records of the target statistics: the k largest logits
// (ties to the lower index) lie in the tiles whose maximum is at least the
// k-th largest tile maximum, so only those tiles are read.  A radix select
// on order-preserving keys gives the k-th largest value and how many of its
// equal values are needed; an ordered compaction (two passes over per-warp
// segments, ballots for the in-order ranks) lists the kept tokens by index.
// top-p ranks the k tokens by (logit desc, index asc) and keeps those whose
// preceding mass is below top_p.  Output per row: kept tokens by index,
// p' renormalised over them, sum p'^2, and a flag for a top-p cut within
// TIE_TOL.  k_filtered_verify then verifies against p' (its support has at
// most k tokens, so no vocabulary-wide pass is needed in either mode).
constexpr int TF_NT = 256;
constexpr int TF_W = TF_NT / 32;

__device__ __forceinline__ uint32_t fkey(float f) {
  if (f == 0.f) f = 0.f;  // -0 ranks with +0
  const uint32_t b = __float_as_uint(f);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

struct FilterShared {
  int hist[256];
  int wcnt[TF_W][2];
  int wbase[TF_W][2];
  int digit, above;
  int C;
  uint32_t tie;
  FF red[TF_W];
  float smax;
};

// The key of the k-th largest (1-based) of n keys get(i), and in *rem how many
// elements equal to that key belong to the k largest.
// Digits from bit 31 down to lo_shift (keys whose lower bits are all zero
// need fewer passes: 16 for keys of bf16 values).
template <typename GET>
__device__ uint32_t radix_kth_largest(int n, int k, const GET& get, FilterShared& sh, int* rem,
                                      int lo_shift) {
  const int tid = threadIdx.x, lane = tid & 31;
  uint32_t prefix = 0u, mask = 0u;
  int r = k;
  for (int shift = 24; shift >= lo_shift; shift -= 8) {
    for (int b = tid; b < 256; b += TF_NT) sh.hist[b] = 0;
    __syncthreads();
    for (int i = tid; i < n; i += TF_NT) {
      const uint32_t key = get(i);
      if ((key & mask) == prefix) atomicAdd(&sh.hist[(key >> shift) & 255u], 1);
    }
    __syncthreads();
    if (tid < 32) {
      // lane l owns digits 255 - 8l ... 248 - 8l (descending)
      int c[8], loc = 0;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        c[j] = sh.hist[255 - 8 * lane - j];
        loc += c[j];
      }
      int incl = loc;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int t = __shfl_up_sync(FULLMASK, incl, o);
        if (lane >= o) incl += t;
      }
      const int excl = incl - loc;
      const unsigned hit = __ballot_sync(FULLMASK, incl >= r);
      const int l0 = hit ? __ffs(hit) - 1 : 31;
      if (lane == l0) {
        int acc = excl, j = 0;
        while (j < 7 && acc + c[j] < r) acc += c[j++];
        sh.digit = 255 - 8 * lane - j;
        sh.above = acc;
      }
    }
    __syncthreads();
    prefix |= (uint32_t)sh.digit << shift;
    mask |= 255u << shift;
    r -= sh.above;
    __syncthreads();
  }
  *rem = r;
  return prefix;
}

// Ordered compaction in two passes over per-warp segments of n elements:
// cls(i) = 0 (drop), 1 (keep), 2 (keep if among the first `E` of class 2 in
// index order); emit(i, pos) is called for every kept element with its rank.
template <typename CLS, typename EMIT>
__device__ int ordered_compact(int n, int E, const CLS& cls, const EMIT& emit, FilterShared& sh) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int seg = ceil_div(ceil_div(n, TF_W), 32) * 32;
  const int s0 = min(n, warp * seg), s1 = min(n, s0 + seg);
  int c1 = 0, c2 = 0;
  for (int b = s0; b < s1; b += 32) {
    const int i = b + lane;
    const int c = i < s1 ? cls(i) : 0;
    c1 += __popc(__ballot_sync(FULLMASK, c == 1));
    c2 += __popc(__ballot_sync(FULLMASK, c == 2));
  }
  if (lane == 0) {
    sh.wcnt[warp][0] = c1;
    sh.wcnt[warp][1] = c2;
  }
  __syncthreads();
  if (tid == 0) {
    int a = 0, b = 0;
    for (int w = 0; w < TF_W; ++w) {
      sh.wbase[w][0] = a;
      sh.wbase[w][1] = b;
      a += sh.wcnt[w][0];
      b += sh.wcnt[w][1];
    }
    sh.C = a + min(b, E);
  }
  __syncthreads();
  int b1 = sh.wbase[warp][0], b2 = sh.wbase[warp][1];
  const unsigned lt = (1u << lane) - 1u;
  for (int b = s0; b < s1; b += 32) {
    const int i = b + lane;
    const int c = i < s1 ? cls(i) : 0;
    const unsigned m1 = __ballot_sync(FULLMASK, c == 1), m2 = __ballot_sync(FULLMASK, c == 2);
    const int r1 = b1 + __popc(m1 & lt), r2 = b2 + __popc(m2 & lt);
    if (c == 1 || (c == 2 && r2 < E)) emit(i, r1 + min(r2, E));
    b1 += __popc(m1);
    b2 += __popc(m2);
  }
  const int total = sh.C;
  __syncthreads();
  return total;
}

template <typename Tin>
__global__ void __launch_bounds__(TF_NT)
    k_target_filter(const Tin* __restrict__ target, const float2* __restrict__ partt, int V,
                    int nt, int B, int Bt, int Rt, int kf, float top_p, float k2,
                    int32_t* __restrict__ ftok, float* __restrict__ fp, int32_t* __restrict__ fcnt,
                    float* __restrict__ coll, uint32_t* __restrict__ ftie) {
  __shared__ FilterShared sh;
  __shared__ uint32_t tkey[FILTER_MAX_TILES];  // keys of the row's tile maxima
  __shared__ int clist[FILTER_MAX_TILES];
  __shared__ uint32_t ckey[FILTER_STAGE];      // keys of the candidate tokens, when they fit
  __shared__ int stok[FILTER_MAX_K];
  __shared__ float sval[FILTER_MAX_K];
  __shared__ float sw[FILTER_MAX_K];
  __shared__ FF scum[FILTER_MAX_K];
  __shared__ int skeep[FILTER_MAX_K];
  const int row = blockIdx.x, tid = threadIdx.x;
  const int n = row / Bt, i = row - n * Bt;
  const int rl = n * (B + 1) + i;
  const Tin* tr = target + (size_t)row * V;
  const int k = min(kf, V);
  // keys of bf16 values have 16 significant bits: two radix digits
  constexpr bool BF = std::is_same<Tin, __nv_bfloat16>::value;
  constexpr uint32_t KMASK = BF ? 0xFFFF0000u : 0xFFFFFFFFu;
  constexpr int LO = BF ? 16 : 0;
  for (int t = tid; t < nt; t += TF_NT) tkey[t] = fkey(partt[(size_t)t * Rt + rl].x) & KMASK;
  __syncthreads();
  // candidate tiles: maximum >= the k-th largest tile maximum
  uint32_t theta = 0u;
  if (k < nt) {
    int rem;
    theta = radix_kth_largest(nt, k, [&](int t) { return tkey[t]; }, sh, &rem, LO);
  }
  const int C = ordered_compact(
      nt, 0, [&](int t) { return tkey[t] >= theta ? 1 : 0; },
      [&](int t, int pos) { clist[pos] = t; }, sh);
  // the k-th largest logit of the candidate tiles, and its equal values needed
  auto gkey = [&](int j) {
    const int v = clist[j >> 7] * TILE_V + (j & (TILE_V - 1));
    return v < V ? (fkey(ldf(tr + v)) & KMASK) : 0u;
  };
  const bool staged = C * TILE_V <= FILTER_STAGE;
  if (staged)
    for (int j = tid; j < C * TILE_V; j += TF_NT) ckey[j] = gkey(j);
  __syncthreads();
  auto cand = [&](int j) { return staged ? ckey[j] : gkey(j); };
  int E;
  const uint32_t tau = radix_kth_largest(C * TILE_V, k, cand, sh, &E, LO);
  // kept tokens in index order
  const int cnt = ordered_compact(
      C * TILE_V, E,
      [&](int j) {
        const int v = clist[j >> 7] * TILE_V + (j & (TILE_V - 1));
        if (v >= V) return 0;
        const uint32_t key = cand(j);
        return key > tau ? 1 : (key == tau ? 2 : 0);
      },
      [&](int j, int pos) {
        const int v = clist[j >> 7] * TILE_V + (j & (TILE_V - 1));
        stok[pos] = v;
        sval[pos] = ldf(tr + v);
      },
      sh);
  __syncthreads();
  // weights relative to the largest kept logit
  if (tid < 32) {
    float m = -INFINITY;
    for (int j = tid; j < cnt; j += 32) m = fmaxf(m, sval[j]);
    m = warp_max(m);
    if (tid == 0) sh.smax = m;
  }
  __syncthreads();
  const FF cmax = ff_prod(sh.smax, k2);
  for (int j = tid; j < cnt; j += TF_NT)
    sw[j] = (sval[j] == -INFINITY || sh.smax == -INFINITY) ? 0.f : exp2_rel(sval[j], k2, cmax);
  __syncthreads();
  // top-p: rank by (logit desc, index asc), cumulative mass before each rank
  const bool use_p = top_p > 0.f && top_p < 1.f;
  if (tid == 0) sh.tie = 0u;
  if (use_p) {
    for (int j = tid; j < cnt; j += TF_NT) {
      int rk = 0;
      for (int l = 0; l < cnt; ++l)
        rk += (sval[l] > sval[j] || (sval[l] == sval[j] && stok[l] < stok[j])) ? 1 : 0;
      skeep[j] = rk;
    }
    __syncthreads();
    for (int j = tid; j < cnt; j += TF_NT) scum[skeep[j]] = FF{sw[j], 0.f};
    __syncthreads();
    // exclusive prefix sums in rank order (cnt <= FILTER_MAX_K == TF_NT)
    static_assert(FILTER_MAX_K <= TF_NT, "one thread per rank");
    const BlockScan bs = block_scan_ff<TF_NT>(tid < cnt ? scum[tid] : FF{0.f, 0.f}, sh.red);
    if (tid < cnt) scum[tid] = bs.excl;
    __syncthreads();
    const FF W = bs.total;
    const FF thr = ff_mulf(W, top_p);
    const float Wf = ff_f(W);
    for (int j = tid; j < cnt; j += TF_NT) {
      const FF before = scum[skeep[j]];
      skeep[j] = ff_gt(thr, before) ? 1 : 0;
      if (fabsf(ff_f(ff_sub(before, thr))) < TIE_TOL * Wf) atomicOr(&sh.tie, 1u);
    }
  } else {
    for (int j = tid; j < cnt; j += TF_NT) skeep[j] = 1;
  }
  __syncthreads();
  // renormalise over the kept tokens, collision probability, ordered output
  if (tid < 32) {
    FF Wk{0.f, 0.f};
    for (int j = tid; j < cnt; j += 32)
      if (skeep[j]) Wk = ff_addf(Wk, sw[j]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) Wk = ff_add(Wk, ff_shfl_xor(Wk, o));
    const float inv = 1.f / ff_f(Wk);
    float c2 = 0.f;
    int base = 0;
    for (int j0 = 0; j0 < cnt; j0 += 32) {
      const int j = j0 + tid;
      const bool kp = j < cnt && skeep[j];
      const unsigned m = __ballot_sync(FULLMASK, kp);
      if (kp) {
        const int pos = base + __popc(m & ((1u << tid) - 1u));
        const float pj = sw[j] * inv;
        ftok[(size_t)rl * FILTER_MAX_K + pos] = stok[j];
        fp[(size_t)rl * FILTER_MAX_K + pos] = pj;
        c2 = fmaf(pj, pj, c2);
      }
      base += __popc(m);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) c2 += __shfl_xor_sync(FULLMASK, c2, o);
    if (tid == 0) {
      fcnt[rl] = base;
      coll[rl] = c2;
      ftie[rl] = sh.tie;
    }
  }
}

// q(v|x_<i) at one token for the verify kernels: the soft mixture from the
// stash and the branch corrections, or q_greedy from the consistent branches.
struct SoftQ {
  const float* srow;  // stash row of position i
  const float* wu;
  const float* cm;    // codes of position i, [K, rr]
  const FF* Cz;       // [K] L_z - log2 w_z (+inf if w_z = 0)
  int K, rr;
  float k2;
  __device__ float operator()(int v) const {
    float q = 0.f;
    const float base = srow[v];
    for (int z = 0; z < K; ++z) {
      const FF c = Cz[z];
      if (c.hi == INFINITY) continue;
      q += exp2_rel2(base, corr_at(wu, cm + z * rr, v, z, K, rr), k2, c);
    }
    return q;
  }
};
struct GreedyQ {
  const int* X;       // x-hat of position i, [K]
  const float* pi;
  uint32_t c;         // C_i
  float S;            // sum of pi over C_i
  int K;
  __device__ float operator()(int v) const {
    float q = 0.f;
    for (int z = 0; z < K; ++z)
      if (((c >> z) & 1u) && X[z] == v) q += pi[z];
    return S > 0.f ? q / S : 0.f;
  }
};

// Inverse CDF over at most FILTER_MAX_K masses in index order by one warp:
// the smallest j whose cumulative mass exceeds u times the total (the
// total is the warp's own sum).  Returns j (-1 if the total is 0) and the
// margin of the decision relative to the total.
template <typename MASS>
__device__ int warp_inverse_cdf(int cnt, const MASS& mass, float u, float* margin, float* total) {
  const int lane = threadIdx.x & 31;
  FF tot{0.f, 0.f};
  for (int j = lane; j < cnt; j += 32) tot = ff_addf(tot, mass(j));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) tot = ff_add(tot, ff_shfl_xor(tot, o));
  *total = ff_f(tot);
  *margin = 0.f;
  if (!(tot.hi > 0.f)) return -1;
  const FF target = ff_mulf(tot, u);
  FF base{0.f, 0.f};
  int last = -1;
  for (int j0 = 0; j0 < cnt; j0 += 32) {
    const int j = j0 + lane;
    const float w = j < cnt ? mass(j) : 0.f;
    FF incl{w, 0.f};
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const FF t = ff_shfl_up(incl, o);
      if (lane >= o) incl = ff_add(t, incl);
    }
    FF ex1 = ff_shfl_up(incl, 1);
    if (lane == 0) ex1 = FF{0.f, 0.f};
    const FF hi = ff_add(base, incl), lo = ff_add(base, ex1);
    const unsigned hit = __ballot_sync(FULLMASK, j < cnt && ff_gt(hi, target));
    const unsigned pos = __ballot_sync(FULLMASK, j < cnt && w > 0.f);
    if (pos) last = j0 + 31 - __clz(pos);
    if (hit) {
      const int l = __ffs(hit) - 1;
      const float m = fminf(ff_f(ff_sub(target, lo)), ff_f(ff_sub(hi, target))) / ff_f(tot);
      *margin = __shfl_sync(FULLMASK, m, l);
      return j0 + l;
    }
    base = FF{__shfl_sync(FULLMASK, hi.hi, 31), __shfl_sync(FULLMASK, hi.lo, 31)};
  }
  return last;  // rounding left the target at the total: the last positive mass
}

// One block per sequence: verification against the filtered target p'.
// alpha_i and the residual mass need q only at the kept tokens of row i.
template <bool GREEDY>
__global__ void __launch_bounds__(VF_NT)
    k_filtered_verify(const int32_t* __restrict__ ftok, const float* __restrict__ fp,
                      const int32_t* __restrict__ fcnt, const uint32_t* __restrict__ ftie,
                      const float* __restrict__ coll, const float* __restrict__ stash,
                      const float* __restrict__ wu, const float* __restrict__ codes,
                      const float2* __restrict__ lse2, const float2* __restrict__ w2,
                      const int32_t* __restrict__ xhat, const uint32_t* __restrict__ cmask,
                      const float* __restrict__ log2pi, const float* __restrict__ qtok_ws,
                      const int32_t* __restrict__ tok, const uint32_t* __restrict__ ties_draft,
                      int V, int K, int rr, int B, int Bt, int kf, float k2, uint64_t seed,
                      int64_t* __restrict__ pos, uint32_t* __restrict__ rnd,
                      dblast_verify_out out) {
  griddep_wait();  // launched as a dependent of the previous kernel
  extern __shared__ float qS[];   // [B][kf]: q(v|x_<i) at the kept tokens of row i
  __shared__ FF Cz[32][32];       // soft: per position, L_z - log2 w_z
  __shared__ int X[1024];         // greedy: x-hat [B, K]
  __shared__ float piS[32], Ssum[32];
  __shared__ float alphaS[32];
  __shared__ int sL, sx;
  __shared__ uint32_t sties;
  const int n = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t p0 = pos[n];
  const uint32_t rd = rnd[n];
  const size_t m0 = (size_t)n * B;
  if (GREEDY) {
    for (int j = tid; j < B * K; j += VF_NT) X[j] = xhat[m0 * K + j];
    if (tid < K) piS[tid] = exp2f(log2pi[n * K + tid]);
  } else {
    for (int j = tid; j < B * K; j += VF_NT) {
      const int i = j / K, z = j - i * K;
      const FF wz = ff_ld(w2 + (m0 + i) * K + z);
      Cz[i][z] = (wz.hi == -INFINITY) ? FF{INFINITY, 0.f} : ff_sub(ff_ld(lse2 + (m0 + i) * K + z), wz);
    }
  }
  __syncthreads();
  if (GREEDY && tid < B) {
    const uint32_t c = cmask[m0 + tid];
    float S = 0.f;
    for (int z = 0; z < K; ++z)
      if ((c >> z) & 1u) S += piS[z];
    Ssum[tid] = S;
  }
  __syncthreads();
  auto qfun = [&](int i, int v) -> float {
    if constexpr (GREEDY) {
      return GreedyQ{X + i * K, piS, cmask[m0 + i], Ssum[i], K}(v);
    } else {
      return SoftQ{stash + (m0 + i) * V, wu, codes + (m0 + i) * K * rr, Cz[i], K, rr, k2}(v);
    }
  };
  // q at every (position, kept token), all threads; then
  // alpha_i = sum over the kept tokens of min(p'(v), q(v)): one warp per position
  for (int pq = tid; pq < B * kf; pq += VF_NT) {
    const int i = pq / kf, j = pq - i * kf;
    const int rl = n * (B + 1) + i;
    if (j < fcnt[rl]) qS[pq] = qfun(i, ftok[(size_t)rl * FILTER_MAX_K + j]);
  }
  __syncthreads();
  for (int i = warp; i < B; i += VF_NT / 32) {
    const int rl = n * (B + 1) + i;
    const int cnt = fcnt[rl];
    FF a{0.f, 0.f};
    for (int j = lane; j < cnt; j += 32)
      a = ff_addf(a, fminf(fp[(size_t)rl * FILTER_MAX_K + j], qS[i * kf + j]));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) a = ff_add(a, ff_shfl_xor(a, o));
    if (lane == 0) alphaS[i] = ff_f(a);
  }
  __syncthreads();
  if (tid < 32) {
    uint32_t ties = ties_draft[n];
    float A = 0.f, alpha = 0.f, ptok = 0.f, qtok = 1.f, u2 = 0.f;
    bool acc_ok = false;
    uint32_t ftb = 0u;
    for (int r = lane; r < Bt; r += 32) ftb |= ftie[n * (B + 1) + r];
    if (__any_sync(FULLMASK, ftb != 0u)) ties |= TIE_TOPP;
    if (lane < B) {
      const int m = n * B + lane;
      const int rl = n * (B + 1) + lane;
      const int x = tok[m];
      // p'(x_i): binary search among the kept tokens (sorted by index)
      int lo = 0, hi = fcnt[rl];
      while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (ftok[(size_t)rl * FILTER_MAX_K + mid] < x) lo = mid + 1;
        else hi = mid;
      }
      ptok = (lo < fcnt[rl] && ftok[(size_t)rl * FILTER_MAX_K + lo] == x)
                 ? fp[(size_t)rl * FILTER_MAX_K + lo] : 0.f;
      qtok = qtok_ws[m];
      const float ratio = ptok / qtok;
      A = fminf(1.f, ratio);
      alpha = alphaS[lane];
      u2 = decision_uniform(seed, 2u, rd, (uint32_t)n, (uint32_t)(p0 + lane));
      acc_ok = u2 < ratio;
      if (out.p_tok) out.p_tok[m] = ptok;
      if (out.accept_prob) out.accept_prob[m] = A;
      if (out.alpha) out.alpha[m] = alpha;
    }
    const unsigned acc_mask = __ballot_sync(FULLMASK, acc_ok);
    const unsigned rej = ~acc_mask & ((B >= 32) ? FULLMASK : ((1u << B) - 1u));
    const int L = rej ? (__ffs(rej) - 1) : B;
    const float amargin = fabsf(fmaf(u2, qtok, -ptok));
    const bool atie = lane < B && lane <= L && amargin < TIE_TOL * qtok;
    const bool anear = lane < B && lane <= L && amargin < (TIE_TOL + NEAR_ACCEPT) * qtok;
    if (__ballot_sync(FULLMASK, atie)) ties |= TIE_ACCEPT;
    if (__ballot_sync(FULLMASK, anear)) ties |= TIE_ACCEPT << NEAR_SHIFT;
    float cC = 1.f;
    if (lane < B) {
      cC = coll[(size_t)n * (B + 1) + lane];
      if (out.collision) out.collision[n * B + lane] = cC;
    }
    float cA = (lane < B) ? A : 1.f, cAl = (lane < B) ? alpha : 1.f;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const float ta = __shfl_up_sync(FULLMASK, cA, o);
      const float tl = __shfl_up_sync(FULLMASK, cAl, o);
      const float tc = __shfl_up_sync(FULLMASK, cC, o);
      if (lane >= o) {
        cA *= ta;
        cAl *= tl;
        cC *= tc;
      }
    }
    FF el{lane < B ? cA : 0.f, 0.f}, ea{lane < B ? cAl : 0.f, 0.f}, ed{lane < B ? cC : 0.f, 0.f};
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      el = ff_add(el, ff_shfl_xor(el, o));
      ea = ff_add(ea, ff_shfl_xor(ea, o));
      ed = ff_add(ed, ff_shfl_xor(ed, o));
    }
    // the residual or bonus token, by this warp
    int extra = -1;
    if (L < B || Bt > B) {
      const int irow = L < B ? L : B;
      const int rl = n * (B + 1) + irow;
      const int cnt = fcnt[rl];
      const int32_t* tk = ftok + (size_t)rl * FILTER_MAX_K;
      const float* pk = fp + (size_t)rl * FILTER_MAX_K;
      const float u3 = decision_uniform(seed, 3u, rd, (uint32_t)n, (uint32_t)(p0 + irow));
      float margin = 0.f, total = 0.f;
      int j = -1;
      bool from_p = L >= B;
      if (L < B) {
        j = warp_inverse_cdf(cnt, [&](int jj) { return fmaxf(pk[jj] - qS[L * kf + jj], 0.f); },
                             u3, &margin, &total);
        if (total < TIE_TOL) ties |= TIE_RMASS;
        if (total < TIE_TOL + NEAR_DRAW) ties |= TIE_RMASS << NEAR_SHIFT;
        if (j < 0) {
          from_p = true;
          ties |= TIE_RMASS;
        }
      }
      if (from_p) j = warp_inverse_cdf(cnt, [&](int jj) { return pk[jj]; }, u3, &margin, &total);
      if (margin < TIE_TOL) ties |= TIE_RESID;
      if (!(total > 0.f) || margin < TIE_TOL + NEAR_DRAW / total) ties |= TIE_RESID << NEAR_SHIFT;
      extra = j >= 0 ? tk[j] : (cnt > 0 ? tk[0] : 0);
    }
    if (lane == 0) {
      if (out.exp_len) out.exp_len[n] = ff_f(el);
      if (out.alpha_len) out.alpha_len[n] = ff_f(ea);
      if (out.determinism) out.determinism[n] = ff_f(ed) / (float)B;
      sL = L;
      sx = extra;
      sties = ties;
    }
  }
  __syncthreads();
  const int L = sL, extra = sx;
  if (tid == 0) {
    const int ne = L + (extra >= 0 ? 1 : 0);
    if (out.accepted) out.accepted[n] = L;
    if (out.n_emitted) out.n_emitted[n] = ne;
    if (out.tie_flags) out.tie_flags[n] = sties | ((sties & 0xffu) << NEAR_SHIFT);
    pos[n] = p0 + ne;
    rnd[n] = rd + 1u;
  }
  if (out.emitted) {
    for (int j = tid; j < B + 1; j += VF_NT) {
      int val = -1;
      if (j < L) val = tok[n * B + j];
      else if (j == L && extra >= 0) val = extra;
      out.emitted[(size_t)n * (B + 1) + j] = val;
    }
  }
}

template <typename Tin>
static cudaError_t filter_typed(const StepCtx& c, const dblast_verify_out* o) {
  const WsLayout& w = c.wl;
  const int rows = w.N * c.Bt;
  k_target_filter<Tin><<<rows, TF_NT, 0, c.stream>>>(
      static_cast<const Tin*>(o->target), wsp<float2>(c, w.off_partt), w.V, w.nt, w.B, c.Bt, w.Rt,
      o->top_k > 0 ? o->top_k : w.V, o->top_p, c.k2, wsp<int32_t>(c, w.off_ftok),
      wsp<float>(c, w.off_fp), wsp<int32_t>(c, w.off_fcnt), wsp<float>(c, w.off_coll),
      wsp<uint32_t>(c, w.off_ftie));
  debug_kernel("k_target_filter", c.stream);
  count_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_target_filter(const StepCtx& c, const dblast_verify_out* o) {
  return c.head->dtype == DBLAST_F32 ? filter_typed<float>(c, o) : filter_typed<__nv_bfloat16>(c, o);
}

cudaError_t launch_filtered_verify(const StepCtx& c, const dblast_verify_out* o) {
  const WsLayout& w = c.wl;
  auto k = c.greedy ? k_filtered_verify<true> : k_filtered_verify<false>;
  const int kf = o->top_k;  // the kept tokens per row at most (clamped by the caller)
  cudaError_t le = launch_dep(k, dim3(w.N), dim3(VF_NT), (size_t)w.B * kf * sizeof(float), c.stream,
      wsp<int32_t>(c, w.off_ftok), wsp<float>(c, w.off_fp), wsp<int32_t>(c, w.off_fcnt),
      wsp<uint32_t>(c, w.off_ftie), wsp<float>(c, w.off_coll), wsp<float>(c, w.off_stash),
      prp<float>(c, c.pl.off_wu), wsp<float>(c, w.off_codes), wsp<float2>(c, w.off_lse2),
      wsp<float2>(c, w.off_w2), wsp<int32_t>(c, w.off_xhat), wsp<uint32_t>(c, w.off_cmask),
      wsp<float>(c, w.off_log2pi), wsp<float>(c, w.off_qtok), wsp<int32_t>(c, w.off_tok),
      wsp<uint32_t>(c, w.off_ties), w.V, c.head->K, w.rr, w.B, c.Bt, kf, c.k2, c.args->seed,
      c.args->pos, c.args->round, *o);
  debug_kernel("k_filtered_verify", c.stream);
  count_launches(1);
  return le != cudaSuccess ? le : cudaGetLastError();
}

// ---------------------------------------------------------------- training-side objectives
// Sec. 3.2, forward only, on a given target block x*: the draft pass and the
// draft finalize kernels run with the given tokens in place of draws, so
// q(x*_i|x*_<i) (Eqs. category-posterior, dep-next-token) and log2 q_z(x*_i)
// come from the step's own kernels; one warp per sequence then forms
// p(x*_i) (filtered like verification), A_i, r_l, S_l, l_tau, J_AL and the
// block NLL (Eq. dependent-nll) from sum_i log2 q_z(x*_i) and the prior.
template <typename Tin>
__global__ void __launch_bounds__(32)
    k_al_objective(const Tin* __restrict__ target, const int32_t* __restrict__ tok,
                   const float* __restrict__ qtok_ws, const float2* __restrict__ lq2,
                   const float* __restrict__ log2pi, const float2* __restrict__ lt2,
                   const int32_t* __restrict__ ftok, const float* __restrict__ fp,
                   const int32_t* __restrict__ fcnt, const uint32_t* __restrict__ ftie,
                   bool filtered, int V, int K, int B, int Bt, float k2, float tau,
                   dblast_al_args al) {
  griddep_wait();  // launched as a dependent of the previous kernel
  const int n = blockIdx.x, lane = threadIdx.x;
  const size_t m0 = (size_t)n * B;
  const bool on = lane < B;
  uint32_t ties = 0u;
  float p = 1.f, q = 1.f;
  if (on) {
    const int m = (int)m0 + lane;
    const int rl = n * (B + 1) + lane;
    const int x = tok[m];
    q = qtok_ws[m];
    if (filtered) {
      int lo = 0, hi = fcnt[rl];
      while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (ftok[(size_t)rl * FILTER_MAX_K + mid] < x) lo = mid + 1;
        else hi = mid;
      }
      p = (lo < fcnt[rl] && ftok[(size_t)rl * FILTER_MAX_K + lo] == x)
              ? fp[(size_t)rl * FILTER_MAX_K + lo] : 0.f;
      if (ftie[rl]) ties |= TIE_TOPP;
    } else {
      const float tx = ldf(target + ((size_t)n * Bt + lane) * V + x);
      p = (tx == -INFINITY) ? 0.f : ff_exp2(ff_sub(ff_prod(tx, k2), ff_ld(lt2 + rl)));
    }
  }
  const float A = on ? fminf(1.f, p / q) : 1.f;
  // log2 r_l: prefix sums of log2 q - log2 p; S_l: prefix sums of prod A
  FF lr{on ? log2f(q) - log2f(p) : 0.f, 0.f};
  float cA = A;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const FF t = ff_shfl_up(lr, o);
    const float ta = __shfl_up_sync(FULLMASK, cA, o);
    if (lane >= o) {
      lr = ff_add(t, lr);
      cA *= ta;
    }
  }
  FF S{on ? cA : 0.f, 0.f};
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const FF t = ff_shfl_up(S, o);
    if (lane >= o) S = ff_add(t, S);
  }
  const float l2tau = tau > 0.f ? log2f(tau) : -INFINITY;
  const float lrf = ff_f(lr);
  const unsigned below = __ballot_sync(FULLMASK, on && lrf < l2tau);
  const int l_tau = below ? __ffs(below) : B;
  const bool in = lane < l_tau;
  if (__ballot_sync(FULLMASK, in && tau > 0.f && fabsf(lrf - l2tau) * LN2 < TIE_TOL))
    ties |= TIE_TAU;
  // r_l multiplies l + 1 ratios, each within NEAR_ACCEPT (relative)
  if (__ballot_sync(FULLMASK, in && tau > 0.f &&
                                  fabsf(lrf - l2tau) * LN2 < TIE_TOL + NEAR_ACCEPT * (lane + 1)))
    ties |= TIE_TAU << NEAR_SHIFT;
  FF jt{in ? lrf + ff_f(ff_log2(S)) : 0.f, 0.f};
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) jt = ff_add(jt, ff_shfl_xor(jt, o));
  // block NLL: -log sum_z pi_z prod_i q_z(x*_i), in base 2 over the lanes z
  FF sz{-INFINITY, 0.f};
  if (lane < K) {
    const float lp = log2pi[n * K + lane];
    if (lp != -INFINITY) {
      sz = FF{lp, 0.f};
      for (int i = 0; i < B; ++i) sz = ff_add(sz, ff_ld(lq2 + (m0 + i) * K + lane));
    }
  }
  const float mx = warp_max(sz.hi);
  float e = (sz.hi == -INFINITY || mx == -INFINITY) ? 0.f : ff_exp2(ff_addf(sz, -mx));
  e = warp_sum(e);
  ties = __reduce_or_sync(FULLMASK, ties);
  if (on) {
    const int m = (int)m0 + lane;
    if (al.r) al.r[m] = exp2f(lrf);
    if (al.S) al.S[m] = ff_f(S);
    if (al.accept_prob) al.accept_prob[m] = A;
    if (al.q_cond) al.q_cond[m] = q;
    if (al.p_tok) al.p_tok[m] = p;
  }
  if (lane == 0) {
    if (al.j_al) al.j_al[n] = ff_f(jt) * LN2;
    if (al.l_tau) al.l_tau[n] = l_tau;
    if (al.nll) al.nll[n] = (mx == -INFINITY) ? INFINITY : -(mx + log2f(e)) * LN2;
    if (al.tie_flags) al.tie_flags[n] = ties | ((ties & 0xffu) << NEAR_SHIFT);
  }
}

cudaError_t launch_al_objective(const StepCtx& c, const dblast_al_args* al, bool filtered) {
  const WsLayout& w = c.wl;
  cudaError_t le;
  if (c.head->dtype == DBLAST_F32)
    le = launch_dep(k_al_objective<float>, dim3(w.N), dim3(32), 0, c.stream,
                    static_cast<const float*>(al->target), wsp<int32_t>(c, w.off_tok),
                    wsp<float>(c, w.off_qtok), wsp<float2>(c, w.off_lq2),
                    wsp<float>(c, w.off_log2pi), wsp<float2>(c, w.off_lt2),
                    wsp<int32_t>(c, w.off_ftok), wsp<float>(c, w.off_fp),
                    wsp<int32_t>(c, w.off_fcnt), wsp<uint32_t>(c, w.off_ftie), filtered, w.V,
                    c.head->K, w.B, c.Bt, c.k2, al->tau, *al);
  else
    le = launch_dep(k_al_objective<__nv_bfloat16>, dim3(w.N), dim3(32), 0, c.stream,
                    static_cast<const __nv_bfloat16*>(al->target), wsp<int32_t>(c, w.off_tok),
                    wsp<float>(c, w.off_qtok), wsp<float2>(c, w.off_lq2),
                    wsp<float>(c, w.off_log2pi), wsp<float2>(c, w.off_lt2),
                    wsp<int32_t>(c, w.off_ftok), wsp<float>(c, w.off_fp),
                    wsp<int32_t>(c, w.off_fcnt), wsp<uint32_t>(c, w.off_ftie), filtered, w.V,
                    c.head->K, w.B, c.Bt, c.k2, al->tau, *al);
  debug_kernel("k_al_objective", c.stream);
  count_launches(1);
  return le != cudaSuccess ? le : cudaGetLastError();
}

}  // namespace dblast
