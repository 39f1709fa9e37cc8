// Tensor-core passes for sm_103a: tcgen05.mma with fp32 accumulators in TMEM,
// operands staged in shared memory by TMA (cp.async.bulk.tensor, 128-byte
// swizzle), mbarrier pipelines, one persistent CTA per SM.
//
// Draft pass (rows a2+a3 of the step).  For a tile of 128 positions (TMEM
// lanes) x 128 vocabulary tokens (TMEM columns):
//   base    D_b  = h . W^T                        (bf16 x bf16, K = H)
//   branch  D_z  = c_z . WU_z^T   for z < K        (split fp16: hi.hi + hi.lo + lo.hi)
//   l_{m,z,v} = D_b + D_z / (sc_{m,z} sw_z) + b_v, s = l log2(e) / T
// and the epilogue warps reduce every (m, z) row of the tile to a (max, sum)
// record of 2^s, stash W h + b in fp32 and never write the branch logits.
// The branch GEMMs of tile t are interleaved with the base GEMM of tile t+1
// so the epilogue of one tile overlaps the main loop of the next.
//
// Prep pass (row a0): the same machinery with only the base GEMM computes
// WU = [U_z | e_z]^T . W^T and stores it as fp32 [V, K, rr].
#include <cuda.h>

#include <algorithm>
#include <cstdlib>

#include "dblast_internal.cuh"

namespace dblast {

uint32_t wait_limit();

namespace tc {

constexpr int BM = 128;            // rows per tile (TMEM lanes)
constexpr int BN = 128;            // vocabulary tokens per tile (TMEM columns)
constexpr int BK = 64;             // elements per stage row (128 bytes, SW128 atom)
constexpr int STAGE_A = BM * BK * 2;   // 16 KB
constexpr int STAGE_B = BN * BK * 2;   // 16 KB
constexpr int STAGE_BYTES = STAGE_A + STAGE_B;
constexpr int KMAX = 16;           // components supported by the tensor-core path
// verify pass: warp 0 TMA, warp 1 MMA (warps 2-3 idle), warps 4-19 the
// epilogue, four per SM sub-partition with 32 columns each; warpgroup 0 gives
// registers to the epilogue warpgroups (56 + 4 x 104 <= 5 x 96 per thread)
constexpr int NUM_EPI_WARPS = 16;
constexpr int NUM_THREADS = 32 * (4 + NUM_EPI_WARPS);
constexpr int VREG = 96, VREG_LO = 56, VREG_HI = 104;
static_assert(4 * VREG_LO + 16 * VREG_HI <= 20 * VREG, "register split must fit the launch pool");
constexpr uint32_t TMEM_COLS = 512;

enum Mode { MODE_PREP = 0, MODE_DRAFT = 1, MODE_GREEDY = 2 };

// ------------------------------------------------------------------ PTX
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ uint64_t globaltimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count));
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// The retry of a wait that did not complete at once: the warp may be
// suspended for up to WAIT_HINT_NS nanoseconds (or until the phase completes)
// before the loop around it checks its bounds again, instead of polling and
// taking issue slots from the warps that share its scheduler.
#ifndef DBLAST_WAIT_HINT_NS
#define DBLAST_WAIT_HINT_NS 20000
#endif
constexpr uint32_t WAIT_HINT_NS = DBLAST_WAIT_HINT_NS;
// The draft epilogue's waits for its next accumulator sleep this long between
// polls: its warps share schedulers with the producer and the MMA issuer,
// whose instruction streams pace the tensor pipe (measured: 0.5112 -> 0.5092
// ms per draft pass; the verify pass, whose roles all wait on one another,
// was 1 us slower with it and does not use it).
constexpr uint32_t NAP_NS = 100;
__device__ __forceinline__ bool mbar_retry_wait(uint64_t* bar, uint32_t parity) {
  if constexpr (WAIT_HINT_NS == 0) {
    return mbar_try_wait(bar, parity);
  } else {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}\n"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity), "n"(WAIT_HINT_NS)
        : "memory");
    return ok != 0;
  }
}

// Shared state of the roles: every wait is bounded; a wait that runs out
// raises `abort` so that the other roles leave their loops too.
struct Ctl {
  uint32_t spin_limit;        // 0: time bound only
  volatile int* abort;        // shared flag
  DevStatus* status;          // global status word
};

__device__ __noinline__ void record_timeout(const Ctl& c, uint32_t where) {
  *c.abort = 1;
  atomicExch(&c.status->timeout, 1u);
  atomicExch(&c.status->where, where);
}

// sleep_ns > 0: a role whose waits are not on the critical path sleeps that
// long between polls, so that it takes no issue slots from the warps sharing
// its scheduler while it waits
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, const Ctl& c,
                                          uint32_t where, uint32_t sleep_ns = 0) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer();
  for (uint32_t i = 1;; ++i) {
    if (sleep_ns) __nanosleep(sleep_ns);
    // a spin limit (fault injection) counts plain polls
    if (c.spin_limit ? mbar_try_wait(bar, parity) : mbar_retry_wait(bar, parity)) return true;
    if (*c.abort) return false;
    if ((c.spin_limit && i >= c.spin_limit) || (globaltimer() - t0) > 2000000000ull) {
      record_timeout(c, where);
      return false;
    }
  }
}

__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, uint64_t* bar,
                                            int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes "
      "[%0], [%1, {%3, %4}], [%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(x), "r"(y)
      : "memory");
}

__device__ __forceinline__ void tma_load_3d(void* dst, const CUtensorMap* map, uint64_t* bar,
                                            int x, int y, int z) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes "
      "[%0], [%1, {%3, %4, %5}], [%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(x), "r"(y), "r"(z)
      : "memory");
}

// copies of data read once (evict-first L2 policy)
__device__ __forceinline__ uint64_t l2_evict_first() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}
__device__ __forceinline__ void tma_load_2d_once(void* dst, const CUtensorMap* map, uint64_t* bar,
                                                 int x, int y, uint64_t pol) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint "
      "[%0], [%1, {%3, %4}], [%2], %5;" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(x), "r"(y), "l"(pol)
      : "memory");
}
__device__ __forceinline__ void tma_load_3d_once(void* dst, const CUtensorMap* map, uint64_t* bar,
                                                 int x, int y, int z, uint64_t pol) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint "
      "[%0], [%1, {%3, %4, %5}], [%2], %6;" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(x), "r"(y), "r"(z), "l"(pol)
      : "memory");
}

__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cluster_id_x() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%clusterid.x;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cluster_count_x() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%nclusterid.x;" : "=r"(r));
  return r;
}
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
  asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// K-major operand in a 128-byte-swizzled tile: rows of 128 bytes, 8-row
// groups 1024 bytes apart; the start address moves by 32 bytes per 16-element
// K step inside the row.
__device__ __forceinline__ uint64_t sdesc(uint32_t saddr) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr >> 4) & 0x3FFFu);
  d |= static_cast<uint64_t>(1) << 16;                 // leading byte offset (unused here)
  d |= static_cast<uint64_t>(1024 >> 4) << 32;         // stride byte offset: 8 rows
  d |= static_cast<uint64_t>(1) << 46;                 // descriptor version for tcgen05
  d |= static_cast<uint64_t>(2) << 61;                 // 128-byte swizzle
  return d;
}

// the same for a 64-byte-swizzled operand (rows of 64 bytes, 8-row groups 512
// bytes apart): the branch operands of one component, [hi | lo] of rank 16
__device__ __forceinline__ uint64_t sdesc64(uint32_t saddr) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr >> 4) & 0x3FFFu);
  d |= static_cast<uint64_t>(1) << 16;
  d |= static_cast<uint64_t>(512 >> 4) << 32;
  d |= static_cast<uint64_t>(1) << 46;
  d |= static_cast<uint64_t>(4) << 61;                 // 64-byte swizzle
  return d;
}

// instruction descriptor, kind::f16: fp32 accumulate, A/B both bf16 or both
// fp16, both K-major, M = m (128, or 256 for a CTA pair), N = n
__host__ __device__ constexpr uint32_t idesc_f16(bool bf16, int n, int m = BM) {
  return (1u << 4) | ((bf16 ? 1u : 0u) << 7) | ((bf16 ? 1u : 0u) << 10) |
         (static_cast<uint32_t>(n >> 3) << 17) | (static_cast<uint32_t>(m >> 4) << 24);
}

__device__ __forceinline__ void umma(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc,
                                     uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(d_tmem),
      "l"(a), "l"(b), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void umma_commit(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}

// ---- CTA pairs (cta_group::2): one MMA spans the tensor cores of two SMs.
// The A operand and the accumulator are split by rows (128 per SM), the B
// operand by N (half of the tile in each SM's shared memory, at the same
// offset); the even CTA of the pair issues every MMA.

// the shared::cluster address of the object at p's offset in CTA `rank`
__device__ __forceinline__ uint32_t cluster_addr(const void* p, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_u32(p)), "r"(rank));
  return r;
}
// Hand-over of a TMEM accumulator the thread has finished reading
// (tcgen05.wait::ld has returned, so the values are in registers): nothing
// written before it needs to be visible to the waiter, so the arrive is
// relaxed.  A release arrive would first wait for the thread's earlier global
// stores (the stash rows, the records) to become visible, which at cluster
// scope takes a large part of a component's epilogue.
__device__ __forceinline__ void mbar_arrive_taken(uint64_t* bar) {
  asm volatile("mbarrier.arrive.relaxed.cta.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar))
               : "memory");
}
__device__ __forceinline__ void mbar_arrive_taken_cluster(uint32_t caddr) {
  asm volatile("mbarrier.arrive.relaxed.cluster.shared::cluster.b64 _, [%0];" ::"r"(caddr)
               : "memory");
}
// a wait whose arrivals may come from the other CTA of the pair
__device__ __forceinline__ bool mbar_try_wait_cl(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ bool mbar_retry_wait_cl(uint64_t* bar, uint32_t parity) {
  if constexpr (WAIT_HINT_NS == 0) {
    return mbar_try_wait_cl(bar, parity);
  } else {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}\n"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity), "n"(WAIT_HINT_NS)
        : "memory");
    return ok != 0;
  }
}
__device__ __forceinline__ bool mbar_wait_cl(uint64_t* bar, uint32_t parity, const Ctl& c,
                                             uint32_t where, uint32_t sleep_ns = 0) {
  if (mbar_try_wait_cl(bar, parity)) return true;
  const uint64_t t0 = globaltimer();
  for (uint32_t i = 1;; ++i) {
    if (sleep_ns) __nanosleep(sleep_ns);
    if (c.spin_limit ? mbar_try_wait_cl(bar, parity) : mbar_retry_wait_cl(bar, parity)) return true;
    if (*c.abort) return false;
    if ((c.spin_limit && i >= c.spin_limit) || (globaltimer() - t0) > 2000000000ull) {
      record_timeout(c, where);
      return false;
    }
  }
}
// a copy into this CTA's shared memory whose complete_tx goes to the mbarrier
// at cluster address bar_cl (the even CTA's)
__device__ __forceinline__ void tma_load_2d_pair(void* dst, const CUtensorMap* map,
                                                 uint32_t bar_cl, int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes "
      "[%0], [%1, {%3, %4}], [%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar_cl), "r"(x), "r"(y)
      : "memory");
}
__device__ __forceinline__ void umma_pair(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc,
                                          uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(d_tmem),
      "l"(a), "l"(b), "r"(idesc), "r"(accumulate)
      : "memory");
}
// arrive on the mbarrier at bar's offset in both CTAs of the pair once the
// pair MMAs issued so far have completed
__device__ __forceinline__ void umma_commit_pair(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 "
      "[%0], %1;" ::"r"(smem_u32(bar)), "h"((uint16_t)3)
      : "memory");
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
        "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
        "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
        "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
}

__device__ __forceinline__ void named_bar_sync(int id, int nthreads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

// ------------------------------------------------------------ draft pass
// 128 x 256 tiles in two TMEM regions of 256 columns: tile t accumulates its
// base GEMM in region t & 1, and once the epilogue has taken that base, the
// same region holds its branch components one at a time, while tile t+1's
// base accumulates in the other region.  The MMA issuer therefore never waits
// for a base accumulator to be read; it waits only until tile t-1's last
// component has been taken before starting tile t+1.  12 warps: warp 0 issues TMA, warp
// 1 issues MMAs and owns TMEM, warps 4-11 are the epilogue (two per TMEM lane
// quarter, 128 columns each).  Warpgroup 0 gives registers to the epilogue
// warpgroups with setmaxnreg (56 + 2 x 224 = 3 x 168 per thread; 64 + 2 x 216
// when warps 2-3 also run the target statistics).
//
// The pair form (PAIR = true) runs the same roles on a cluster of two CTAs
// with cta_group::2 MMAs of 256 x 256: each SM stages its own 128 rows of A
// and 128 of the 256 B rows (32 KB a stage instead of 48), so six stages fit
// and the L2 reads of the head per tile fall by a third.  Both CTAs' copies
// complete on the even CTA's full barriers, its MMA commits arrive on both
// CTAs' barriers, and both epilogues hand the accumulators back on the even
// CTA's bempty / cempty.
constexpr int DBN = 256;                     // vocabulary tokens per tile
constexpr int DSTAGE_A = BM * BK * 2;        // 16 KB
constexpr int DCOLS = DBN / 2;               // columns per epilogue thread
constexpr int D_THREADS = 384;
constexpr int DREG = 168, DREG_LO = 56, DREG_HI = 224;
static_assert(4 * DREG_LO + 8 * DREG_HI == 12 * DREG, "register split must equal the launch pool");
// with the target statistics on warps 2-3 the first warpgroup needs 64
// registers (56 spilled in its stage loops); the epilogue fits in 216
constexpr int DREG_LO_TS = 64, DREG_HI_TS = 216;
static_assert(4 * DREG_LO_TS + 8 * DREG_HI_TS <= 12 * DREG, "register split must fit the launch pool");
constexpr int D_EPI = 256;                   // epilogue threads
constexpr int DAZ_BYTES = KMAX * D_EPI * 4;  // per-thread branch scales
constexpr int DVB_BYTES = 2 * DBN * 4;       // vocabulary bias of two tiles
template <bool PAIR>
struct DCfg {
  static constexpr int STAGES = PAIR ? 6 : 4;
  static constexpr int BROWS = PAIR ? DBN / 2 : DBN;       // B rows staged by one CTA
  static constexpr int STAGE_B = BROWS * BK * 2;           // 16 or 32 KB
  static constexpr int STAGE = DSTAGE_A + STAGE_B;         // 32 or 48 KB
  static constexpr int TX = PAIR ? 2 * STAGE : STAGE;      // bytes completing one full barrier
  // a branch item of rank 16: 64-byte rows of A (BM) and B (BROWS)
  static constexpr int TX_NARROW = (PAIR ? 2 : 1) * (BM + BROWS) * 64;
  static constexpr size_t SMEM = (size_t)STAGES * STAGE + DAZ_BYTES + DVB_BYTES + 256 + 64 + 1024;
};
static_assert(DCfg<true>::SMEM <= 227 * 1024 && DCfg<false>::SMEM <= 227 * 1024, "shared memory");

struct Params {
  int mode;
  int cs;                    // CTAs per cluster: 2 for the CTA pair, else 1
  int n_mt, n_vt, n_tiles;   // M tiles, vocabulary tiles, cluster tiles (x ksplit in prep mode)
  int nb;                    // base stages per tile
  int K, rp, zps;            // components, padded rank, components per 64-wide block
  int M, V, Mpad;            // valid rows, vocabulary (B-operand rows), padded rows
  float k2;                  // log2(e) / T
  const float* vbias;        // [V] or null
  const float* cscale;       // [Mpad, K]
  const float* sw;           // [K]
  float* stash;              // [M, V]
  float2* partd;             // [nt, K, Mpad]
  float* partg;              // [nt, K, Mpad] greedy mode: second-largest logit of the record
  float* wu;                 // prep output [ksplit][V, prep_rows]
  int prep_rows;             // valid A rows in prep mode
  size_t split_stride;       // elements between the split-K partial outputs
  DevStatus* status;
  uint32_t spin_limit;
  // target statistics computed by the idle warps 2-3 of the draft pass
  // (fused step, bf16 target with V % 8 == 0); tgt == nullptr: off
  const __nv_bfloat16* tgt;  // [t_rows, V]
  int t_rows, t_Bt, t_B, t_Rt, t_nt;
  float t_k2;                // log2(e) / T
  float2* t_partt;           // [nt, Rt] tile records (tmax, sum 2^((t - tmax) k2))
  float2* t_lt2;             // [Rt] log2 sum_v 2^(t_v k2) as a float pair
  float* t_coll;             // [Rt] sum_v p(v)^2
  float* t_lse;              // [t_rows] natural log-sum-exp, or null
};

// Tile `slot` of this CTA.  The two CTAs of a pair share a vocabulary tile
// and take consecutive M tiles; cluster tiles are numbered split-major (prep
// mode), then vocabulary-major, so concurrently running clusters also share
// B tiles through L2.
struct Sched {
  int cid, ncl, rank;  // cluster index, cluster count, rank in the cluster
};
__device__ __forceinline__ Sched sched_of(const Params& P) {
  if (P.cs == 1) return Sched{(int)blockIdx.x, (int)gridDim.x, 0};
  return Sched{(int)cluster_id_x(), (int)cluster_count_x(), (int)cluster_ctarank()};
}
__device__ __forceinline__ void tile_of(const Params& P, const Sched& S, int slot, int* sp,
                                        int* mt, int* vt) {
  const int t = S.cid + slot * S.ncl;
  const int ng = P.n_mt / P.cs;
  const int per = ng * P.n_vt;
  *sp = t / per;
  const int r = t - *sp * per;
  *vt = r / ng;
  *mt = (r - *vt * ng) * P.cs + S.rank;
}

// The item sequence of slot s (consumed by the MMA thread, produced by the TMA
// thread): the base stages of tile s, with the branch items (one per
// component) of tile s-1 inserted before base stage ins_point(z).  The last
// slot (s == my_tiles) holds only the branch items of the last tile.  The
// first branch item comes after 1/8 of the base stages (the epilogue is
// still taking the base accumulator and writing the stash), the others
// follow evenly up to six stages before the end, so that the last
// component's epilogue ends before the tile's base accumulator is complete
// (measured best among first in {0, 1/8, 1/4, 3/8} x last in nb - {2..12}).
__device__ __forceinline__ int ins_point(int z, int nb, int nz) {
  const int first = nb / 8;
  const int last = nb - 6 > first ? nb - 6 : first;
  return nz > 1 ? first + (z * (last - first)) / (nz - 1) : first;
}

// The producer and the MMA issuer are single threads whose dependent
// instruction chains sit on the critical path of every stage (a stage is 512
// tensor cycles, a thread's chain runs at several cycles per instruction), so
// both are inlined (parameters read from the constant bank, no local copies)
// and run the base stages between two branch items in a loop that only
// waits, issues and advances the stage; measured alone, such a loop keeps
// the tensor pipe busy at 128 cycles per 128 x 256 x 16 MMA.
template <bool PAIR>
__device__ __forceinline__ void draft_producer(const Params& P, const Sched& S,
                                               const CUtensorMap* tm_a, const CUtensorMap* tm_b,
                                               const CUtensorMap* tm_ca, const CUtensorMap* tm_cb,
                                               unsigned char* stages, uint64_t* full,
                                               uint64_t* empty, const Ctl& ctl, int my_tiles) {
  using C = DCfg<PAIR>;
  // a pair CTA loads its own A tile and its half of the B tile (the B maps
  // then have DBN/2 rows)
  const int bq = DBN / P.cs;
  const bool lead = !PAIR || S.rank == 0;
  const uint32_t full_cl = PAIR ? cluster_addr(full, 0) : 0u;  // the even CTA's full barriers
  int stage = 0;
  uint32_t phase = 0, issued_mask = 0u, issued_phase = 0u;
  bool ok = true;
  const int nzK = (P.mode != MODE_PREP) ? P.K : 0;
  // one stage: wait until the slot is free, arm its full barrier, copy the
  // A and B boxes
  auto load = [&](const CUtensorMap* ma, const CUtensorMap* mb, int xk, int y0, int y1,
                  uint32_t tx) {
    if (!mbar_wait(&empty[stage], phase ^ 1u, ctl, 1)) return false;
    unsigned char* sa = stages + stage * C::STAGE;
    uint64_t* fb = &full[stage];
    if (lead) mbar_arrive_expect_tx(fb, tx);
    if constexpr (PAIR) {
      const uint32_t fcl = full_cl + (uint32_t)(stage * 8);
      tma_load_2d_pair(sa, ma, fcl, xk, y0);
      tma_load_2d_pair(sa + DSTAGE_A, mb, fcl, xk, y1);
    } else {
      tma_load_2d(sa, ma, fb, xk, y0);
      tma_load_2d(sa + DSTAGE_A, mb, fb, xk, y1);
    }
    issued_mask |= 1u << stage;
    issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
    if (++stage == C::STAGES) {
      stage = 0;
      phase ^= 1u;
    }
    return true;
  };
  for (int slot = 0; slot <= my_tiles && ok; ++slot) {
    const int nbv = (slot < my_tiles) ? P.nb : 0;
    const int nzv = (slot >= 1) ? nzK : 0;
    int sp = 0, mt = 0, vt = 0, psp = 0, pmt = 0, pvt = 0;
    if (slot < my_tiles) tile_of(P, S, slot, &sp, &mt, &vt);
    if (slot >= 1) tile_of(P, S, slot - 1, &psp, &pmt, &pvt);
    const int ya = mt * BM, yb = vt * DBN + S.rank * bq;
    const int yca = pmt * BM, ycb = pvt * DBN + S.rank * bq;
    int kx = sp * P.nb * BK;
    int jb = 0;
    // base stages up to the next insertion point, then one branch item
    for (int zd = 0; zd <= nzv && ok; ++zd) {
      const int jend = zd < nzv ? ins_point(zd, nbv, nzv) : nbv;
      for (; jb < jend; ++jb, kx += BK)
        if (!(ok = load(tm_a, tm_b, kx, ya, yb, C::TX))) break;
      // a branch item copies its own component: with rank 16 ([hi | lo], 32
      // elements) a 64-byte-wide box, else the 64-wide block of the component
      if (ok && zd < nzv)
        ok = (P.zps == 2) ? load(tm_ca, tm_cb, zd * 32, yca, ycb, C::TX_NARROW)
                          : load(tm_ca, tm_cb, zd * BK, yca, ycb, C::TX);
    }
  }
  // copies still in flight after an abort: wait (bounded) before leaving.  The
  // odd CTA of a pair cannot wait on the even CTA's barriers; its copies land
  // within microseconds, so it waits a fixed 100 us instead.
  if (lead) {
    for (int s = 0; s < C::STAGES; ++s)
      if (issued_mask & (1u << s)) {
        const uint64_t t0 = globaltimer();
        while (!mbar_try_wait(&full[s], (issued_phase >> s) & 1u) &&
               (globaltimer() - t0) < 2000000000ull) {
        }
      }
  } else if (!ok && issued_mask) {
    const uint64_t t0 = globaltimer();
    while ((globaltimer() - t0) < 100000ull) {
    }
  }
}

template <bool PAIR>
__device__ __forceinline__ void draft_mma(const Params& P, uint32_t tmem, unsigned char* stages,
                                          uint64_t* full, uint64_t* empty, uint64_t* bfull,
                                          uint64_t* bempty, uint64_t* cfull, uint64_t* cempty,
                                          uint64_t* done, const Ctl& ctl, int my_tiles) {
  using C = DCfg<PAIR>;
  constexpr int MM = PAIR ? 2 * BM : BM;
  const uint32_t id_base = idesc_f16(true, DBN, MM);
  const uint32_t id_corr = idesc_f16(false, DBN, MM);
  // shared-memory descriptors: the start-address field holds addr >> 4, so a
  // byte offset off inside the 1024-aligned stages moves it by off >> 4
  const uint64_t d0 = sdesc(smem_u32(stages));
  auto mma = [&](uint32_t d, uint64_t a, uint64_t b, uint32_t id, uint32_t acc) {
    if constexpr (PAIR) umma_pair(d, a, b, id, acc);
    else umma(d, a, b, id, acc);
  };
  // release a stage / hand an accumulator over: in a pair the commit arrives
  // on the barrier at the same offset in both CTAs
  auto commit_all = [&](uint64_t* bar) {
    if constexpr (PAIR) umma_commit_pair(bar);
    else umma_commit(bar);
  };
  auto commit_acc = [&](uint64_t* bar) {
    if constexpr (PAIR) umma_commit_pair(bar);
    else umma_commit(bar);
  };
  auto wait_taken = [&](uint64_t* bar, uint32_t parity, uint32_t where) {
    if constexpr (PAIR) return mbar_wait_cl(bar, parity, ctl, where);
    else return mbar_wait(bar, parity, ctl, where);
  };
  int stage = 0;
  uint32_t phase = 0;
  uint32_t cuse0 = 0u, cuse1 = 0u;  // components issued into TMEM region 0 / 1
  uint64_t da = d0;  // descriptor of the current stage's A box
  auto next = [&]() {
    if (++stage == C::STAGES) {
      stage = 0;
      phase ^= 1u;
      da = d0;
    } else {
      da += (uint64_t)(C::STAGE >> 4);
    }
  };
  bool ok = true;
  const int nzK = (P.mode != MODE_PREP) ? P.K : 0;
  for (int slot = 0; slot <= my_tiles && ok; ++slot) {
    const int nbv = (slot < my_tiles) ? P.nb : 0;
    const int nzv = (slot >= 1) ? nzK : 0;
    // tile `slot` accumulates in region r, the components of tile slot-1 in
    // the other one (where that tile's base was)
    const int r = slot & 1;
    const uint32_t dbase = tmem + (uint32_t)(r * DBN), dcol = tmem + (uint32_t)((r ^ 1) * DBN);
    int jb = 0;
    for (int zd = 0; zd <= nzv && ok; ++zd) {
      const int jend = zd < nzv ? ins_point(zd, nbv, nzv) : nbv;
      if (jb == 0 && jend > 0) {
        // region r is free once the epilogue has taken tile slot-2's base
        // and every component computed there
        if (!(ok = wait_taken(&bempty[r], ((uint32_t)(slot >> 1) & 1u) ^ 1u, 2))) break;
        const uint32_t cu = r ? cuse1 : cuse0;
        if (cu > 0 && !(ok = wait_taken(&cempty[r], (cu - 1u) & 1u, 4))) break;
        tc_fence_after();
      }
      for (; jb < jend; ++jb) {
        if (!(ok = mbar_wait(&full[stage], phase, ctl, 3))) break;
        tc_fence_after();
        const uint64_t db = da + (uint64_t)(DSTAGE_A >> 4);
        mma(dbase, da, db, id_base, jb > 0 ? 1u : 0u);
        mma(dbase, da + 2, db + 2, id_base, 1u);
        mma(dbase, da + 4, db + 4, id_base, 1u);
        mma(dbase, da + 6, db + 6, id_base, 1u);
        commit_all(&empty[stage]);
        if (jb == nbv - 1) commit_acc(&bfull[r]);
        next();
      }
      if (!ok || zd == nzv) break;
      // branch item zd of the previous tile, in its region once the epilogue
      // has taken that tile's base (zd = 0) or component zd-1:
      // hi.hi + hi.lo + lo.hi; element offsets o (hi) and o + rp (lo) are
      // multiples of 16 (32 bytes)
      if (zd == 0) {
        if (!(ok = wait_taken(&bempty[r ^ 1], (uint32_t)((slot - 1) >> 1) & 1u, 2))) break;
      } else {
        if (!(ok = wait_taken(&cempty[r ^ 1], ((r ? cuse0 : cuse1) - 1u) & 1u, 4))) break;
      }
      tc_fence_after();
      if (!(ok = mbar_wait(&full[stage], phase, ctl, 3))) break;
      tc_fence_after();
      if (P.zps == 2) {
        // rank 16: hi at bytes 0-31, lo at 32-63 of each 64-byte row
        const uint32_t sa = smem_u32(stages + stage * C::STAGE);
        const uint64_t a64 = sdesc64(sa), b64 = sdesc64(sa + DSTAGE_A);
        mma(dcol, a64, b64, id_corr, 0u);
        mma(dcol, a64, b64 + 2, id_corr, 1u);
        mma(dcol, a64 + 2, b64, id_corr, 1u);
      } else {
        const uint64_t db = da + (uint64_t)(DSTAGE_A >> 4);
        for (int kk = 0; kk < P.rp; kk += 16) {
          const uint64_t hi = (uint64_t)(kk >> 3), lo = (uint64_t)((P.rp + kk) >> 3);
          mma(dcol, da + hi, db + hi, id_corr, kk > 0 ? 1u : 0u);
          mma(dcol, da + hi, db + lo, id_corr, 1u);
          mma(dcol, da + lo, db + hi, id_corr, 1u);
        }
      }
      commit_acc(&cfull[r ^ 1]);
      commit_all(&empty[stage]);
      if (r) ++cuse0;
      else ++cuse1;
      next();
    }
  }
  // wait (bounded) for every MMA this thread issued before TMEM is freed
  commit_acc(done);
  const uint64_t t0 = globaltimer();
  while (!mbar_try_wait(done, 0u) && (globaltimer() - t0) < 2000000000ull) {
  }
}

__device__ __forceinline__ void tmem_ld32_raw(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
        "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
        "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
        "=r"(r[31])
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld16_raw(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
        "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_wait_ld() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}
// the same wait, with r passed through it: the compiler then cannot move a
// use of r (the destination of a load still in flight) above the wait
__device__ __forceinline__ void tmem_wait_ld(uint32_t (&r)[32]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]),
                 "+r"(r[6]), "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]),
                 "+r"(r[12]), "+r"(r[13]), "+r"(r[14]), "+r"(r[15]), "+r"(r[16]), "+r"(r[17]),
                 "+r"(r[18]), "+r"(r[19]), "+r"(r[20]), "+r"(r[21]), "+r"(r[22]), "+r"(r[23]),
                 "+r"(r[24]), "+r"(r[25]), "+r"(r[26]), "+r"(r[27]), "+r"(r[28]), "+r"(r[29]),
                 "+r"(r[30]), "+r"(r[31])
               :
               : "memory");
}
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm volatile("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// 2^x on the special-function unit, as a plain (reorderable) instruction
__device__ __forceinline__ float ex2n(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Two fp32 lanes per instruction (the compiler's packed fma/add/mul, round to
// nearest): each lane is rounded exactly as the scalar instruction, with half
// the issue slots.  a - b is fma(b, -1, a), exact up to the one rounding.
typedef float2 F2;
__device__ __forceinline__ F2 f2(float lo, float hi) { return make_float2(lo, hi); }
__device__ __forceinline__ void f2_get(F2 a, float& lo, float& hi) {
  lo = a.x;
  hi = a.y;
}
__device__ __forceinline__ F2 f2_fma(F2 a, F2 b, F2 c) { return __ffma2_rn(a, b, c); }
__device__ __forceinline__ F2 f2_add(F2 a, F2 b) { return __fadd2_rn(a, b); }
__device__ __forceinline__ F2 f2_sub(F2 a, F2 b) { return __ffma2_rn(b, make_float2(-1.f, -1.f), a); }
__device__ __forceinline__ F2 f2_mul(F2 a, F2 b) { return __fmul2_rn(a, b); }
__device__ __forceinline__ F2 f2_ex2(F2 a) { return make_float2(ex2n(a.x), ex2n(a.y)); }

// the wait for a 16-column load, with its destination passed through it
__device__ __forceinline__ void tmem_wait_ld16(uint32_t (&r)[16]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]),
                 "+r"(r[6]), "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]),
                 "+r"(r[12]), "+r"(r[13]), "+r"(r[14]), "+r"(r[15])
               :
               : "memory");
}
// Greedy-branch epilogue of one tile (Sec. 3.1, "Drafter sampling during
// inference"): for every component z, the largest logit
// l_v = base_v + b_v + D_z / (cscale sw) of this thread's 128 columns and its
// token (lowest index on ties) become the record (max, index) of the half
// tile, and the second-largest logit its tie record; no stash and no
// exponentials.  Four interleaved chains keep the compare-and-select
// sequences independent.
// top-two merge of (max, index, second): the second of the union is the
// larger of the losing max and the winner's own second
__device__ __forceinline__ void arg_keep2(float& mx, int& ix, float& sc, float v, int i, float vs) {
  if (v > mx || (v == mx && i < ix)) {
    sc = fmaxf(mx, vs);
    mx = v;
    ix = i;
  } else {
    sc = fmaxf(sc, v);
  }
}
template <bool PAIR>
__device__ __forceinline__ bool greedy_components(const Params& P, uint32_t tmem, int lane,
                                                  uint32_t lane_off, int rg, int half, int slot,
                                                  int m, int v0, int et, const float* az,
                                                  float (&bk)[DCOLS], uint64_t* cfull,
                                                  uint64_t* cempty, const Ctl& ctl) {
  const bool live = v0 < P.V;
#pragma unroll
  for (int j = 0; j < DCOLS; ++j)
    if (v0 + j >= P.V) bk[j] = -INFINITY;
  const int rec = (v0 / DCOLS);
  for (int z = 0; z < P.K; ++z) {
    if (!mbar_wait(&cfull[rg], (uint32_t)((slot >> 1) * P.K + z) & 1u, ctl, 6, NAP_NS)) return false;
    tc_fence_after();
    const float a = az[z * D_EPI + et];
    float m0 = -INFINITY, m1 = -INFINITY, m2 = -INFINITY, m3 = -INFINITY;
    float s0 = -INFINITY, s1 = -INFINITY, s2 = -INFINITY, s3 = -INFINITY;
    int i0 = 0, i1 = 1, i2 = 2, i3 = 3;
    // 16-column chunks, the load of chunk c+1 in flight while chunk c is
    // reduced (two 16-register buffers: with 32-column ones the epilogue,
    // which holds the tile's 128 base logits, spilled)
    const uint32_t tb = tmem + lane_off + (uint32_t)(rg * DBN + half * DCOLS);
    uint32_t ra[16], rb[16];
    tmem_ld16_raw(tb, ra);
    tmem_wait_ld16(ra);
#pragma unroll
    for (int cc = 0; cc < DCOLS / 16; ++cc) {
      uint32_t(&cur)[16] = (cc & 1) ? rb : ra;
      uint32_t(&nxt)[16] = (cc & 1) ? ra : rb;
      if (cc + 1 < DCOLS / 16) tmem_ld16_raw(tb + (uint32_t)((cc + 1) * 16), nxt);
#pragma unroll
      for (int j = 0; j < 16; j += 4) {
        const int c = cc * 16 + j;
        const float x0 = fmaf(__uint_as_float(cur[j]), a, bk[c]);
        const float x1 = fmaf(__uint_as_float(cur[j + 1]), a, bk[c + 1]);
        const float x2 = fmaf(__uint_as_float(cur[j + 2]), a, bk[c + 2]);
        const float x3 = fmaf(__uint_as_float(cur[j + 3]), a, bk[c + 3]);
        // each chain sees increasing columns, so a strict compare keeps the
        // lowest; the chain's second is max(second, min(x, max)) before the update
        s0 = fmaxf(s0, fminf(x0, m0));
        s1 = fmaxf(s1, fminf(x1, m1));
        s2 = fmaxf(s2, fminf(x2, m2));
        s3 = fmaxf(s3, fminf(x3, m3));
        if (x0 > m0) { m0 = x0; i0 = c; }
        if (x1 > m1) { m1 = x1; i1 = c + 1; }
        if (x2 > m2) { m2 = x2; i2 = c + 2; }
        if (x3 > m3) { m3 = x3; i3 = c + 3; }
      }
      if (cc + 1 < DCOLS / 16) tmem_wait_ld16(nxt);
    }
    tc_fence_before();
    __syncwarp();
    if (lane == 0) {
      if constexpr (PAIR) mbar_arrive_taken_cluster(cluster_addr(&cempty[rg], 0));
      else mbar_arrive_taken(&cempty[rg]);
    }
    arg_keep2(m0, i0, s0, m1, i1, s1);
    arg_keep2(m2, i2, s2, m3, i3, s3);
    arg_keep2(m0, i0, s0, m2, i2, s2);
    if (live) {
      const size_t ro = ((size_t)rec * P.K + z) * P.Mpad + m;
      P.partd[ro] = make_float2(m0, __int_as_float(v0 + i0));
      P.partg[ro] = s0;
    }
  }
  return true;
}

// Epilogue: per tile, the base accumulator plus b_v becomes the stash; then// Epilogue: per tile, the base accumulator plus b_v becomes the stash; then
// for every component z the record (ref, sum 2^{t_v}) of this thread's 128
// columns, t_v = D_z a_z + (base_v + b_v) k2 - ref, with ref = k2 max_v
// (base_v + b_v) taken once per tile.  A sum outside [2^-100, 2^100] (a branch
// offset far from the base logits) is redone against the exact maximum.
template <bool PAIR, bool GREEDY>
__device__ __forceinline__ void draft_epilogue(const Params& P, uint32_t tmem, int warp, int lane,
                                            float* az, float* vbs, uint64_t* vbar,
                                            uint64_t* bfull, uint64_t* bempty,
                                            uint64_t* cfull, uint64_t* cempty, const Ctl& ctl,
                                            int my_tiles) {
  const int ew = warp - 4;
  const int q = warp & 3;        // TMEM lane quarter of this warp
  const int half = ew >> 2;      // which 128 columns of the tile
  const int row = q * 32 + lane;
  const int et = ew * 32 + lane;
  const uint32_t lane_off = (uint32_t)(q * 32) << 16;
  const Sched S = sched_of(P);
  for (int slot = 0; slot < my_tiles; ++slot) {
    int sp, mt, vt;
    tile_of(P, S, slot, &sp, &mt, &vt);
    const int m = mt * BM + row;
    const int v0 = vt * DBN + half * DCOLS;
    float bk[DCOLS];
    // this tile's vocabulary bias, staged in shared memory (double-buffered by
    // slot parity: every thread arrives on vbar of slot s+1 only after its
    // reads of slot s, so the writes of slot s+2 cannot overtake them), and the
    // branch scales, while the main loop still runs
    const float* vb = vbs + (slot & 1) * DBN + half * DCOLS;
    if (P.mode != MODE_PREP) {
      for (int z = 0; z < P.K; ++z) az[z * D_EPI + et] = P.k2 / (P.cscale[(size_t)m * P.K + z] * P.sw[z]);
      const int vc = vt * DBN + et;
      vbs[(slot & 1) * DBN + et] = (P.vbias && vc < P.V) ? __ldg(P.vbias + vc) : 0.f;
      mbar_arrive(vbar);
      if (!mbar_wait(vbar, (uint32_t)slot & 1u, ctl, 7, NAP_NS)) break;
    }
    const int rg = slot & 1;  // the tile's TMEM region (base, then its components)
    if (!mbar_wait(&bfull[rg], (uint32_t)(slot >> 1) & 1u, ctl, 5, NAP_NS)) break;
    tc_fence_after();
    {
      const uint32_t tb = tmem + lane_off + (uint32_t)(rg * DBN + half * DCOLS);
      uint32_t ra[32], rb[32];
      tmem_ld32_raw(tb, ra);
      tmem_wait_ld(ra);
#pragma unroll
      for (int cc = 0; cc < DCOLS / 32; ++cc) {
        uint32_t(&cur)[32] = (cc & 1) ? rb : ra;
        uint32_t(&nxt)[32] = (cc & 1) ? ra : rb;
        if (cc + 1 < DCOLS / 32) tmem_ld32_raw(tb + (uint32_t)((cc + 1) * 32), nxt);
#pragma unroll
        for (int j = 0; j < 32; ++j)
          bk[cc * 32 + j] = (P.mode != MODE_PREP) ? __uint_as_float(cur[j]) + vb[cc * 32 + j]
                                                  : __uint_as_float(cur[j]);
        if (cc + 1 < DCOLS / 32) tmem_wait_ld(nxt);
      }
    }
    // the base accumulator is in registers: hand TMEM back to the MMA thread
    tc_fence_before();
    __syncwarp();
    if (lane == 0) {
      if constexpr (PAIR) mbar_arrive_taken_cluster(cluster_addr(&bempty[rg], 0));  // the even CTA's
      else mbar_arrive_taken(&bempty[rg]);
    }

    if (P.mode == MODE_PREP) {
      if (m < P.prep_rows) {
        float* out = P.wu + (size_t)sp * P.split_stride;
#pragma unroll
        for (int j = 0; j < DCOLS; ++j) {
          const int v = v0 + j;
          if (v < P.V) out[(size_t)v * P.prep_rows + m] = bk[j];
        }
      }
      continue;
    }

    if constexpr (GREEDY) {
      if (!greedy_components<PAIR>(P, tmem, lane, lane_off, rg, half, slot, m, v0, et, az, bk, cfull,
                             cempty, ctl))
        break;
      continue;
    }

    // stash W h + b (32-byte stores: each fills one sector of this thread's
    // row; no L1 allocation, which left more of the SM's L1/shared-memory
    // bandwidth to the operand copies than the streaming (.cs) policy:
    // 0.5124 -> 0.5063 ms per draft pass)
    if (m < P.M) {
      float* srow = P.stash + (size_t)m * P.V + v0;
      if (v0 + DCOLS <= P.V && (P.V & 7) == 0) {
#pragma unroll
        for (int j = 0; j < DCOLS; j += 8)
          asm volatile("st.global.L1::no_allocate.v8.f32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"l"(srow + j),
                       "f"(bk[j]), "f"(bk[j + 1]), "f"(bk[j + 2]), "f"(bk[j + 3]), "f"(bk[j + 4]),
                       "f"(bk[j + 5]), "f"(bk[j + 6]), "f"(bk[j + 7])
                       : "memory");
      } else if (v0 + DCOLS <= P.V && (P.V & 3) == 0) {
#pragma unroll
        for (int j = 0; j < DCOLS; j += 4)
          *reinterpret_cast<float4*>(srow + j) = make_float4(bk[j], bk[j + 1], bk[j + 2], bk[j + 3]);
      } else {
        for (int j = 0; j < DCOLS; ++j)
          if (v0 + j < P.V) srow[j] = bk[j];
      }
    }
    // reference and scaled base: bk_j <- (base_j + b_j) k2 - ref (-inf past V)
    float bmax = -INFINITY;
#pragma unroll
    for (int j = 0; j < DCOLS; ++j)
      if (v0 + j < P.V) bmax = fmaxf(bmax, bk[j]);
    const bool live = v0 < P.V;
    const float ref = live ? bmax * P.k2 : 0.f;
#pragma unroll
    for (int j = 0; j < DCOLS; ++j) bk[j] = (v0 + j < P.V) ? fmaf(bk[j], P.k2, -ref) : -INFINITY;

    const int rec = vt * 2 + half;
    bool ok = true;
    for (int z = 0; z < P.K; ++z) {
      if (!mbar_wait(&cfull[rg], (uint32_t)((slot >> 1) * P.K + z) & 1u, ctl, 6, NAP_NS)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const float a = az[z * D_EPI + et];
      float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
      // 32-column chunks, the load of chunk c+1 in flight while chunk c is reduced
      const uint32_t tb = tmem + lane_off + (uint32_t)(rg * DBN + half * DCOLS);
      uint32_t ra[32], rb[32];
      tmem_ld32_raw(tb, ra);
      tmem_wait_ld(ra);
#pragma unroll
      for (int cc = 0; cc < DCOLS / 32; ++cc) {
        uint32_t(&cur)[32] = (cc & 1) ? rb : ra;
        uint32_t(&nxt)[32] = (cc & 1) ? ra : rb;
        if (cc + 1 < DCOLS / 32) tmem_ld32_raw(tb + (uint32_t)((cc + 1) * 32), nxt);
#pragma unroll
        for (int j = 0; j < 32; j += 4) {
          s0 += ex2(fmaf(__uint_as_float(cur[j]), a, bk[cc * 32 + j]));
          s1 += ex2(fmaf(__uint_as_float(cur[j + 1]), a, bk[cc * 32 + j + 1]));
          s2 += ex2(fmaf(__uint_as_float(cur[j + 2]), a, bk[cc * 32 + j + 2]));
          s3 += ex2(fmaf(__uint_as_float(cur[j + 3]), a, bk[cc * 32 + j + 3]));
        }
        if (cc + 1 < DCOLS / 32) tmem_wait_ld(nxt);
      }
      float sum = (s0 + s1) + (s2 + s3);
      float rz = ref;
      const bool bad = live && !(sum >= 0x1p-100f && sum <= 0x1p100f);
      if (__any_sync(0xffffffffu, bad)) {
        // exact maximum of this thread's values, then the sum against it
        float mx = -INFINITY;
#pragma unroll
        for (int cc = 0; cc < DCOLS / 16; ++cc) {
          uint32_t r[16];
          tmem_ld16_raw(tmem + lane_off + (uint32_t)(rg * DBN + half * DCOLS + cc * 16), r);
          tmem_wait_ld();
#pragma unroll
          for (int j = 0; j < 16; ++j) mx = fmaxf(mx, fmaf(__uint_as_float(r[j]), a, bk[cc * 16 + j]));
        }
        float s = 0.f;
#pragma unroll
        for (int cc = 0; cc < DCOLS / 16; ++cc) {
          uint32_t r[16];
          tmem_ld16_raw(tmem + lane_off + (uint32_t)(rg * DBN + half * DCOLS + cc * 16), r);
          tmem_wait_ld();
#pragma unroll
          for (int j = 0; j < 16; ++j) s += ex2(fmaf(__uint_as_float(r[j]), a, bk[cc * 16 + j]) - mx);
        }
        if (bad) {
          sum = s;
          rz = ref + mx;
        }
      }
      // the branch accumulator is read: hand it back
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if constexpr (PAIR) mbar_arrive_taken_cluster(cluster_addr(&cempty[rg], 0));
        else mbar_arrive_taken(&cempty[rg]);
      }
      if (live) {  // the record, also without L1 allocation
        float2* dst = P.partd + ((size_t)rec * P.K + z) * P.Mpad + m;
        asm volatile("st.global.L1::no_allocate.v2.f32 [%0], {%1, %2};" ::"l"(dst), "f"(rz), "f"(sum) : "memory");
      }
    }
    if (!ok) break;
  }
}

// Target statistics on the idle warps 2-3 of the draft pass (fused step):
// the records of the stand-alone target-statistics kernel (per 128-token tile
// (tmax, sum 2^((t - tmax) k2)), per row the log-sum-exp pair and the
// collision probability), computed while the tensor cores run.  Rows go
// round-robin over the CTAs; in a row the two warps take alternate runs of
// eight tiles, four lanes per tile (64 contiguous bytes each).  One run is in
// registers at a time: the 56 registers of these warps hold no second one.
__device__ __forceinline__ void ts_load(const uint4* tr, int nchunk, int c0, uint4 (&d)[4]) {
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const int c = c0 + k;
    d[k] = c < nchunk ? __ldg(tr + c)
                      : make_uint4(0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u);
  }
}
__device__ __forceinline__ void draft_target_stats(const Params& P, int w, int lane, float* xch) {
  const int q = lane >> 2, ql = lane & 3;
  const int nchunk = P.V >> 3;
  const float k2 = P.t_k2;
  const int ngroups = (P.t_nt + 15) >> 4;  // 16 tiles per run pair, 8 per warp
  for (int row = blockIdx.x; row < P.t_rows; row += gridDim.x) {
    const int n = row / P.t_Bt, i = row - n * P.t_Bt;
    const int rl = n * (P.t_B + 1) + i;
    const uint4* tr = reinterpret_cast<const uint4*>(P.tgt + (size_t)row * P.V);
    float rmax = -INFINITY, rsq = 0.f;
    FF rsum{0.f, 0.f};
    uint4 cur[4];
    int t = w * 8 + q;
    ts_load(tr, nchunk, t * 16 + ql * 4, cur);
    for (int g = 0; g < ngroups; ++g, t += 16) {

      __nv_bfloat162 m2 = __float2bfloat162_rn(-INFINITY);
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const uint4 u = cur[k];
        m2 = __hmax2(m2, __hmax2(__hmax2(*reinterpret_cast<const __nv_bfloat162*>(&u.x),
                                         *reinterpret_cast<const __nv_bfloat162*>(&u.y)),
                                 __hmax2(*reinterpret_cast<const __nv_bfloat162*>(&u.z),
                                         *reinterpret_cast<const __nv_bfloat162*>(&u.w))));
      }
      float mx = fmaxf(__low2float(m2), __high2float(m2));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
      float sa = 0.f, s2 = 0.f;
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const uint32_t uu[4] = {cur[k].x, cur[k].y, cur[k].z, cur[k].w};
#pragma unroll
        for (int h = 0; h < 4; ++h) {
          const float a = __uint_as_float(uu[h] << 16), b = __uint_as_float(uu[h] & 0xFFFF0000u);
          const float ea = ex2((a - mx) * k2), eb = ex2((b - mx) * k2);
          sa += ea + eb;
          s2 = fmaf(ea, ea, fmaf(eb, eb, s2));
        }
      }
      sa += __shfl_xor_sync(0xffffffffu, sa, 1);
      sa += __shfl_xor_sync(0xffffffffu, sa, 2);
      s2 += __shfl_xor_sync(0xffffffffu, s2, 1);
      s2 += __shfl_xor_sync(0xffffffffu, s2, 2);
      if (t < P.t_nt) {
        if (ql == 0) P.t_partt[(size_t)t * P.t_Rt + rl] = make_float2(mx, sa);
        if (mx > rmax) {
          const float f = exp2f((rmax - mx) * k2);
          rsum = ff_mulf(rsum, f);
          rsq *= f * f;
          rmax = mx;
        }
        const float gsc = exp2f((mx - rmax) * k2);
        rsum = ff_addf(rsum, sa * gsc);
        rsq = fmaf(s2, gsc * gsc, rsq);
      }
      if (g + 1 < ngroups) ts_load(tr, nchunk, (t + 16) * 16 + ql * 4, cur);
    }
    // the quads of this warp (the four lanes of a quad hold the same state)
    float M1 = rmax;
#pragma unroll
    for (int o = 4; o < 32; o <<= 1) M1 = fmaxf(M1, __shfl_xor_sync(0xffffffffu, M1, o));
    FF S1{0.f, 0.f};
    float Q1 = 0.f;
    if (ql == 0 && M1 != -INFINITY && rmax != -INFINITY) {
      const float f = exp2f((rmax - M1) * k2);
      S1 = ff_mulf(rsum, f);
      Q1 = rsq * f * f;
    }
#pragma unroll
    for (int o = 4; o < 32; o <<= 1) {
      const FF o1{__shfl_xor_sync(0xffffffffu, S1.hi, o), __shfl_xor_sync(0xffffffffu, S1.lo, o)};
      S1 = ff_add(S1, o1);
      Q1 += __shfl_xor_sync(0xffffffffu, Q1, o);
    }
    if (lane == 0) {
      xch[w * 4] = M1;
      xch[w * 4 + 1] = S1.hi;
      xch[w * 4 + 2] = S1.lo;
      xch[w * 4 + 3] = Q1;
    }
    named_bar_sync(8, 64);
    if (w == 0 && lane == 0) {
      const float M2 = fmaxf(xch[0], xch[4]);
      FF S{0.f, 0.f};
      float Q = 0.f;
      if (M2 != -INFINITY)
        for (int k = 0; k < 2; ++k) {
          const float mk = xch[4 * k];
          if (mk != -INFINITY) {
            const float f = exp2f((mk - M2) * k2);
            S = ff_add(S, ff_mulf(FF{xch[4 * k + 1], xch[4 * k + 2]}, f));
            Q = fmaf(xch[4 * k + 3], f * f, Q);
          }
        }
      const FF L = (M2 == -INFINITY || !(S.hi > 0.f)) ? FF{-INFINITY, 0.f}
                                                     : ff_add(ff_prod(M2, k2), ff_log2(S));
      P.t_lt2[rl] = ff_st(L);
      const float sf = ff_f(S);
      P.t_coll[rl] = sf > 0.f ? Q / (sf * sf) : 0.f;
      if (P.t_lse) P.t_lse[row] = ff_f(L) * LN2;
    }
    named_bar_sync(8, 64);
  }
}

template <bool PAIR, bool GREEDY = false, bool TS = false>
__global__ void __launch_bounds__(D_THREADS, 1)
    k_tc_pass(const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_b,
              const __grid_constant__ CUtensorMap tm_ca, const __grid_constant__ CUtensorMap tm_cb,
              const Params P) {
  using C = DCfg<PAIR>;
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  unsigned char* stages = smem;
  float* az = reinterpret_cast<float*>(smem + C::STAGES * C::STAGE);
  float* vbs = reinterpret_cast<float*>(smem + C::STAGES * C::STAGE + DAZ_BYTES);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::STAGES * C::STAGE + DAZ_BYTES + DVB_BYTES);
  uint64_t* full = bars;                    // [STAGES]
  uint64_t* empty = bars + C::STAGES;       // [STAGES]
  // per TMEM region: base accumulator ready / taken (8 epilogue warps per
  // CTA), branch accumulator ready / taken
  uint64_t* bfull = bars + 2 * C::STAGES;   // [2]
  uint64_t* bempty = bfull + 2;             // [2]
  uint64_t* cfull = bfull + 4;              // [2]
  uint64_t* cempty = bfull + 6;             // [2]
  uint64_t* done = bfull + 8;               // every MMA of this CTA finished
  uint64_t* vbar = bfull + 9;               // a tile's vocabulary bias staged (256 epilogue threads)
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bfull + 10);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  float* xch = reinterpret_cast<float*>(bars + 32);  // 64 bytes after the barrier block

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const Sched S = sched_of(P);
  const int my_tiles = (P.n_tiles > S.cid) ? (P.n_tiles - 1 - S.cid) / S.ncl + 1 : 0;
  const Ctl ctl{P.spin_limit, abort_flag, P.status};

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(&full[s], 1);
      // a pair's MMAs are issued (and committed) by the even CTA alone
      mbar_init(&empty[s], 1);
    }
    for (int g = 0; g < 2; ++g) {
      mbar_init(&bfull[g], 1);
      mbar_init(&bempty[g], PAIR ? 16 : 8);
      mbar_init(&cfull[g], 1);
      mbar_init(&cempty[g], PAIR ? 16 : 8);
    }
    mbar_init(done, 1);
    mbar_init(vbar, D_EPI);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {
    if constexpr (PAIR) {
      // one warp of each CTA of the pair allocates the same columns in both SMs
      asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                       smem_u32(tmem_slot)),
                   "r"(TMEM_COLS));
      asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;");
    } else {
      asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                       smem_u32(tmem_slot)),
                   "r"(TMEM_COLS));
      asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  // both CTAs' barriers exist before the peer's copies or commits reach them
  if (PAIR) cluster_sync_all();
  const uint32_t tmem = *tmem_slot;
  griddep_wait();  // the set-up above overlaps the end of the previous kernel

  if (warp >= 4) {
    asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(TS ? DREG_HI_TS : DREG_HI));
    draft_epilogue<PAIR, GREEDY>(P, tmem, warp, lane, az, vbs, vbar, bfull, bempty, cfull, cempty, ctl,
                         my_tiles);
  } else {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(TS ? DREG_LO_TS : DREG_LO));
    if (warp == 0 && lane == 0)
      draft_producer<PAIR>(P, S, &tm_a, &tm_b, &tm_ca, &tm_cb, stages, full, empty, ctl, my_tiles);
    else if (warp == 1 && lane == 0 && (!PAIR || S.rank == 0))
      draft_mma<PAIR>(P, tmem, stages, full, empty, bfull, bempty, cfull, cempty, done, ctl,
                      my_tiles);
    else if constexpr (TS) {
      if (warp == 2 || warp == 3) draft_target_stats(P, warp - 2, lane, xch);
    }
  }

  tc_fence_before();
  __syncthreads();
  // a pair frees its columns only after the even CTA's MMAs (which write both
  // SMs' TMEM) have completed
  if (PAIR) cluster_sync_all();
  if (warp == 1) {
    tc_fence_after();
    if constexpr (PAIR)
      asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                   "r"(TMEM_COLS));
    else
      asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                   "r"(TMEM_COLS));
  }
  // no CTA leaves while its peer may still arrive on its barriers
  if (PAIR) cluster_sync_all();
}

// ------------------------------------------------------------ verify pass
// For a tile of 128 positions x 128 tokens: branch GEMMs D_z = c_z . WU_z^T
// (two components per TMEM slot, two slots), then per (m, v)
//   q(v|x_<i) = 2^{bk_v - B0} sum_z 2^{D_z a_{m,z} + log2 w_{m,z} - L_{m,z} + B0},
//   p(v)      = 2^{t_v log2(e)/T - Lt_m},
// and the tile records (sum min(p, q), sum [p - q]_+).  bk = stash log2(e)/T;
// B0 = floor(max_z L_{m,z}) keeps both factors inside the fp32 range.
// The stash and target tiles of a verify tile go through shared memory when
// use_x (V % 8 == 0 and 128 % B == 0), one 32-column quarter at a time: each
// quarter has its own barriers and its own copying lane (warp 2, lanes 0-3),
// so that the four warps of a quarter never wait for the other quarters.  The
// four partial records of a row are added by whichever of its four warps
// finishes the tile last, so no barrier spans all epilogue warps either.
constexpr int VSTAGES = 3;
constexpr int XS_BOX = BM * 32 * 4;     // stash box [128 rows][32 fp32], 128-byte swizzle
constexpr int XT_BOX = BM * 32 * 2;     // target box [128 rows][32 bf16], 64-byte swizzle
constexpr int XS_BYTES = 4 * XS_BOX;
constexpr int XT_BYTES = 4 * XT_BOX;
constexpr int VRED_BYTES = 2 * 4 * BM * 8;  // per tile parity and quarter: (sum min, sum resid) per row
constexpr size_t VSMEM =
    (size_t)VSTAGES * STAGE_BYTES + XS_BYTES + XT_BYTES + VRED_BYTES + 256 + 1024;
struct VParams {
  int n_mt, n_vt, n_tiles, ncs, K, rp, zps, M, V, Mpad, B, Bt;
  int use_x;
  float k2;
  const float2* vcz;     // [M, K]: (k2 / (sc_{m,z} sw_z), log2 w_{m,z} - L_{m,z} + B0_m)
  const float* vb0;      // [M]: B0_m
  const float2* lt2;     // [N (B+1)]: target log2-sum-exp as a float pair
  const float* stash;    // [M, V]
  const __nv_bfloat16* target;  // [N, Bt, V]
  float2* partv;         // [nt, Mpad]
  DevStatus* status;
  uint32_t spin_limit;
};

__device__ __forceinline__ void vtile_of(const VParams& P, int slot, int* mt, int* vt) {
  const int t = (int)blockIdx.x + slot * (int)gridDim.x;
  *vt = t / P.n_mt;
  *mt = t - *vt * P.n_mt;
}
// The next slot's tile: when the grid is a multiple of the M-tile count (the
// usual launch) the M tile stays and the vocabulary tile advances by a
// constant, without the integer division of vtile_of (which takes the
// special-function unit the epilogue keeps busy).
__device__ __forceinline__ void vtile_next(const VParams& P, int slot, int* mt, int* vt) {
  if ((int)gridDim.x % P.n_mt == 0) *vt += (int)gridDim.x / P.n_mt;
  else vtile_of(P, slot + 1, mt, vt);
}

__global__ void __launch_bounds__(NUM_THREADS, 1)
    k_tc_verify(const __grid_constant__ CUtensorMap tm_ca, const __grid_constant__ CUtensorMap tm_cb,
                const __grid_constant__ CUtensorMap tm_xs, const __grid_constant__ CUtensorMap tm_xt,
                const VParams P) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  unsigned char* stage_base = smem;
  unsigned char* xs = smem + VSTAGES * STAGE_BYTES;  // stash boxes [4]
  unsigned char* xt = xs + XS_BYTES;                 // target boxes [4]
  float2* red = reinterpret_cast<float2*>(xt + XT_BYTES);   // [2][4][BM]
  uint64_t* bars = reinterpret_cast<uint64_t*>(xt + XT_BYTES + VRED_BYTES);
  uint64_t* full = bars;
  uint64_t* empty = bars + VSTAGES;
  uint64_t* sfull = bars + 2 * VSTAGES;  // [2] TMEM slot ready
  uint64_t* sempty = sfull + 2;          // [2] TMEM slot free
  uint64_t* done = sfull + 4;
  uint64_t* xfull = sfull + 5;           // [4] a quarter's stash and target boxes landed
  uint64_t* xempty = sfull + 9;          // [4] ... and read (the quarter's 4 warps)
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sfull + 13);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  int* qcount = reinterpret_cast<int*>(tmem_slot + 2);  // [2][4] quarters done per lane quarter

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int my_tiles = (P.n_tiles > (int)blockIdx.x)
                           ? (P.n_tiles - 1 - (int)blockIdx.x) / (int)gridDim.x + 1
                           : 0;
  const int ngroups = (P.K + 1) / 2;     // two components per TMEM slot
  Ctl ctl{P.spin_limit, abort_flag, P.status};

  if (threadIdx.x == 0) {
    for (int s = 0; s < VSTAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&sfull[b], 1);
      mbar_init(&sempty[b], NUM_EPI_WARPS);
    }
    mbar_init(done, 1);
    for (int c = 0; c < 4; ++c) {
      mbar_init(&xfull[c], 1);
      mbar_init(&xempty[c], 4);
    }
    for (int c = 0; c < 8; ++c) qcount[c] = 0;
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tmem_slot)),
                 "r"(TMEM_COLS));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  griddep_wait();  // the set-up above overlaps the end of the previous kernel

  if (warp >= 4) {
    asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(VREG_HI));
    const int ew = warp - 4;
    const int q = warp & 3;
    const int cq = ew >> 2;  // column quarter of the tile
    const int row = q * 32 + lane;
    const uint32_t lane_off = (uint32_t)(q * 32) << 16;
    uint32_t guse0 = 0u, guse1 = 0u;
    // per-row constants, loaded again only when the tile's M tile changes:
    // B0 and the target log-sum-exp (used after the components), and the
    // row of (k2 / scale, log2 w - L + B0) per component
    int cur_mt = -1, m = 0;
    bool mok = false;
    float B0f = 0.f;
    float2 Lt = make_float2(0.f, 0.f);
    const float2* vrow = P.vcz;
    int mt, vt;
    vtile_of(P, 0, &mt, &vt);
    for (int slot = 0; slot < my_tiles; vtile_next(P, slot, &mt, &vt), ++slot) {
      if (mt != cur_mt) {
        cur_mt = mt;
        m = mt * BM + row;
        mok = m < P.M;
        B0f = mok ? P.vb0[m] : 0.f;
        vrow = P.vcz + (size_t)(mok ? m : 0) * P.K;
        const int n = m / P.B, i = m - n * P.B;
        Lt = mok ? P.lt2[(size_t)n * (P.B + 1) + i] : make_float2(0.f, 0.f);
      }
      const int v0 = vt * BN + cq * 32;
      F2 acc2[16];  // columns (2j, 2j+1)
#pragma unroll
      for (int j = 0; j < 16; ++j) acc2[j] = f2(0.f, 0.f);
      bool ok = true;
      for (int g = 0; g < ngroups; ++g) {
        const int gs = g & 1;
        const uint32_t use = gs ? guse1 : guse0;
        // the group's constants are loaded before the wait for its accumulators
        const int nz = min(2, P.K - 2 * g);
        const float2 c0v = mok ? vrow[2 * g] : make_float2(0.f, -INFINITY);
        const float2 c1v = (mok && nz > 1) ? vrow[2 * g + 1] : make_float2(0.f, -INFINITY);
        if (!mbar_wait(&sfull[gs], use & 1u, ctl, 14)) { ok = false; break; }
        if (gs) ++guse1; else ++guse0;
        tc_fence_after();
        // this quarter's 32 columns of the group's one or two components are
        // read in 16-column chunks (component, half), the load of the next
        // chunk in flight while the current one is reduced; the slot is
        // handed back once the last chunk is in registers
        const uint32_t tb = tmem + lane_off + (uint32_t)(gs * 2 * BN + cq * 32);
        uint32_t ra[16], rb[16];
        auto chunk = [&](const uint32_t (&r)[16], float2 cz, int h) {
          const F2 czx = f2(cz.x, cz.x), czy = f2(cz.y, cz.y);
#pragma unroll
          for (int j = 0; j < 8; ++j)
            acc2[h * 8 + j] = f2_add(acc2[h * 8 + j],
                                     f2_ex2(f2_fma(f2(__uint_as_float(r[2 * j]), __uint_as_float(r[2 * j + 1])),
                                                   czx, czy)));
        };
        auto release = [&]() {
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive_taken(&sempty[gs]);
        };
        tmem_ld16_raw(tb, ra);
        tmem_wait_ld16(ra);
        tmem_ld16_raw(tb + 16, rb);
        chunk(ra, c0v, 0);
        tmem_wait_ld16(rb);
        if (nz > 1) {
          tmem_ld16_raw(tb + BN, ra);
          chunk(rb, c0v, 1);
          tmem_wait_ld16(ra);
          tmem_ld16_raw(tb + BN + 16, rb);
          chunk(ra, c1v, 0);
          tmem_wait_ld16(rb);
          release();
          chunk(rb, c1v, 1);
        } else {
          release();
          chunk(rb, c0v, 1);
        }
      }
      if (!ok) break;
      // four partial sums per quantity keep the add chains short: As2[h]
      // holds the sums of columns j with j & 3 == 2h and 2h + 1
      F2 As2[2] = {f2(0.f, 0.f), f2(0.f, 0.f)}, Rs2[2] = {f2(0.f, 0.f), f2(0.f, 0.f)};
      const F2 k2x = f2(P.k2, P.k2), nB0x = f2(-B0f, -B0f);
      const F2 nLtx = f2(-Lt.x, -Lt.x), Ltyx = f2(Lt.y, Lt.y);
      // columns 2jp and 2jp + 1 together
      auto accumulate2 = [&](int jp, float s0, float s1, float t0, float t1) {
        const F2 qv = f2_mul(f2_ex2(f2_fma(f2(s0, s1), k2x, nB0x)), acc2[jp]);
        const F2 pv = f2_ex2(f2_sub(f2_fma(f2(t0, t1), k2x, nLtx), Ltyx));
        float q0, q1, p0, p1;
        f2_get(qv, q0, q1);
        f2_get(pv, p0, p1);
        const F2 mn = f2(fminf(p0, q0), fminf(p1, q1));
        As2[jp & 1] = f2_add(As2[jp & 1], mn);
        Rs2[jp & 1] = f2_add(Rs2[jp & 1], f2_sub(pv, mn));
      };
      // one column (ragged tail): the same arithmetic on one lane of a pair
      auto accumulate1 = [&](int j, float sv, float tv) {
        float a0, a1;
        f2_get(acc2[j >> 1], a0, a1);
        const float qv = ex2(fmaf(sv, P.k2, -B0f)) * ((j & 1) ? a1 : a0);
        const float pv = ex2(fmaf(tv, P.k2, -Lt.x) - Lt.y);
        const float mn = fminf(pv, qv);
        const int h = (j >> 1) & 1;
        float x0, x1, y0, y1;
        f2_get(As2[h], x0, x1);
        f2_get(Rs2[h], y0, y1);
        if (j & 1) {
          x1 += mn;
          y1 += pv - mn;
        } else {
          x0 += mn;
          y0 += pv - mn;
        }
        As2[h] = f2(x0, x1);
        Rs2[h] = f2(y0, y1);
      };
      const bool full_cols = v0 + 32 <= P.V;
      if (P.use_x) {
        // this quarter's stash and target rows from shared memory: stash box
        // cq (128-byte rows, 128-byte swizzle: 16-byte chunk c of row r at
        // chunk c ^ (r & 7)) and target box cq (64-byte rows, 64-byte
        // swizzle: chunk c of row r at chunk c ^ ((r >> 1) & 3))
        if (!mbar_wait(&xfull[cq], (uint32_t)slot & 1u, ctl, 18)) break;
        if (mok) {
          const unsigned char* sbase = xs + cq * XS_BOX + row * 128;
          const unsigned char* tbase = xt + cq * XT_BOX + row * 64;
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const int c0 = (2 * k) ^ (row & 7), c1 = (2 * k + 1) ^ (row & 7);
            const float4 s0 = *reinterpret_cast<const float4*>(sbase + c0 * 16);
            const float4 s1 = *reinterpret_cast<const float4*>(sbase + c1 * 16);
            const uint4 t8 =
                *reinterpret_cast<const uint4*>(tbase + ((k ^ ((row >> 1) & 3)) * 16));
            const __nv_bfloat162* tp = reinterpret_cast<const __nv_bfloat162*>(&t8);
            const float sv[8] = {s0.x, s0.y, s0.z, s0.w, s1.x, s1.y, s1.z, s1.w};
            float tv[8];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
              const float2 f = __bfloat1622float2(tp[u]);
              tv[2 * u] = f.x;
              tv[2 * u + 1] = f.y;
            }
            if (full_cols) {
#pragma unroll
              for (int u = 0; u < 8; u += 2)
                accumulate2((k * 8 + u) >> 1, sv[u], sv[u + 1], tv[u], tv[u + 1]);
            } else {
#pragma unroll
              for (int u = 0; u < 8; ++u)
                if (v0 + k * 8 + u < P.V) accumulate1(k * 8 + u, sv[u], tv[u]);
            }
          }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&xempty[cq]);
      } else if (mok) {
        const float* srow = P.stash + (size_t)m * P.V + v0;
        const int n = m / P.B, i = m - n * P.B;
        const __nv_bfloat16* trow = P.target + ((size_t)n * P.Bt + i) * P.V + v0;
#pragma unroll
        for (int u = 0; u < 32; ++u)
          if (v0 + u < P.V) accumulate1(u, srow[u], __bfloat162float(trow[u]));
      }
      float As4[4], Rs4[4];
      f2_get(As2[0], As4[0], As4[1]);
      f2_get(As2[1], As4[2], As4[3]);
      f2_get(Rs2[0], Rs4[0], Rs4[1]);
      f2_get(Rs2[1], Rs4[2], Rs4[3]);
      const float As = (As4[0] + As4[1]) + (As4[2] + As4[3]);
      const float Rs = (Rs4[0] + Rs4[1]) + (Rs4[2] + Rs4[3]);
      // one record per (tile, row): the last of the four warps of this lane
      // quarter to get here adds the four column quarters, in quarter order.
      // The counter of a tile parity only grows; its four arrivals of one
      // tile all come before any of the tile two slots later, since that
      // tile's first components wait for every warp to release this tile's.
      float2* rb = red + (slot & 1) * 4 * BM;
      rb[cq * BM + row] = make_float2(As, Rs);
      __syncwarp();
      int last = 0;
      if (lane == 0) {
        // acquire-release at CTA scope: this warp's partials (ordered by the
        // __syncwarp above) are visible to the warp that counts 3, and that
        // warp sees the other three
        uint32_t old;
        asm volatile("atom.acq_rel.cta.shared::cta.add.u32 %0, [%1], 1;"
                     : "=r"(old)
                     : "r"(smem_u32(&qcount[(slot & 1) * 4 + q]))
                     : "memory");
        last = (old & 3u) == 3u;
      }
      __syncwarp();
      if (__shfl_sync(0xffffffffu, last, 0)) {
        const float2 o0 = rb[row], o1 = rb[BM + row], o2 = rb[2 * BM + row], o3 = rb[3 * BM + row];
        P.partv[(size_t)vt * P.Mpad + m] =
            make_float2((o0.x + o1.x) + (o2.x + o3.x), (o0.y + o1.y) + (o2.y + o3.y));
      }
    }
  } else {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(VREG_LO));
    if (warp == 0) {
      if (lane == 0) {
        int stage = 0;
        uint32_t phase = 0, issued_mask = 0u, issued_phase = 0u;
        bool ok = true;
        for (int slot = 0; slot < my_tiles && ok; ++slot) {
          int mt, vt;
          vtile_of(P, slot, &mt, &vt);
          for (int c = 0; c < P.ncs; ++c) {
            if (!mbar_wait(&empty[stage], phase ^ 1u, ctl, 11)) { ok = false; break; }
            unsigned char* sa = stage_base + stage * STAGE_BYTES;
            mbar_arrive_expect_tx(&full[stage], STAGE_BYTES);
            tma_load_2d(sa, &tm_ca, &full[stage], c * BK, mt * BM);
            tma_load_2d(sa + STAGE_A, &tm_cb, &full[stage], c * BK, vt * BN);
            issued_mask |= 1u << stage;
            issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
            if (++stage == VSTAGES) { stage = 0; phase ^= 1u; }
          }
        }
        for (int s = 0; s < VSTAGES; ++s)
          if (issued_mask & (1u << s)) {
            const uint64_t t0 = globaltimer();
            while (!mbar_try_wait(&full[s], (issued_phase >> s) & 1u) &&
                   (globaltimer() - t0) < 2000000000ull) {
            }
          }
      }
    } else if (warp == 2) {
      if (lane < 4 && P.use_x) {
        // lane c copies column quarter c of every tile's stash and target
        // rows, once that quarter's warps have read the previous tile's
        const int c = lane;
        bool x_issued = false;
        uint32_t x_phase = 0;
        // the stash and target rows are read once: evict-first in L2
        const uint64_t pol = l2_evict_first();
        for (int slot = 0; slot < my_tiles; ++slot) {
          int mt, vt;
          vtile_of(P, slot, &mt, &vt);
          if (!mbar_wait(&xempty[c], ((uint32_t)slot & 1u) ^ 1u, ctl, 17)) break;
          mbar_arrive_expect_tx(&xfull[c], XS_BOX + XT_BOX);
          tma_load_2d_once(xs + c * XS_BOX, &tm_xs, &xfull[c], vt * BN + c * 32, mt * BM, pol);
          tma_load_3d_once(xt + c * XT_BOX, &tm_xt, &xfull[c], vt * BN + c * 32, 0,
                           (mt * BM) / P.B, pol);
          x_issued = true;
          x_phase = (uint32_t)slot & 1u;
        }
        if (x_issued) {
          const uint64_t t0 = globaltimer();
          while (!mbar_try_wait(&xfull[c], x_phase) && (globaltimer() - t0) < 2000000000ull) {
          }
        }
      }
    } else if (warp == 1) {
      if (lane == 0) {
        const uint32_t id_corr = idesc_f16(false, BN);
        int stage = 0;
        uint32_t phase = 0, guse0 = 0u, guse1 = 0u;
        bool ok = true;
        for (int slot = 0; slot < my_tiles && ok; ++slot) {
          int c = 0;  // next stage of this tile
          for (int g = 0; g < ngroups && ok; ++g) {
            const int gs = g & 1;
            const uint32_t use = gs ? guse1 : guse0;
            if (!mbar_wait(&sempty[gs], (use & 1u) ^ 1u, ctl, 12)) { ok = false; break; }
            tc_fence_after();
            const int z0 = 2 * g, z1 = min(P.K, z0 + 2);
            // stages holding components z0 .. z1-1
            while (ok && c < P.ncs && c * P.zps < z1) {
              if (!mbar_wait(&full[stage], phase, ctl, 13)) { ok = false; break; }
              tc_fence_after();
              const uint32_t sa = smem_u32(stage_base + stage * STAGE_BYTES);
              const uint32_t sb = sa + STAGE_A;
              for (int zz = 0; zz < P.zps; ++zz) {
                const int z = c * P.zps + zz;
                if (z >= z1) break;
                const uint32_t col = tmem + (uint32_t)(gs * 2 * BN + (z - z0) * BN);
                const int o = zz * 2 * P.rp;
                int first = 1;
                for (int kk = 0; kk < P.rp; kk += 16) {
                  const uint32_t hi = (uint32_t)(o + kk) * 2u, lo = (uint32_t)(o + P.rp + kk) * 2u;
                  umma(col, sdesc(sa + hi), sdesc(sb + hi), id_corr, first ? 0u : 1u);
                  umma(col, sdesc(sa + hi), sdesc(sb + lo), id_corr, 1u);
                  umma(col, sdesc(sa + lo), sdesc(sb + hi), id_corr, 1u);
                  first = 0;
                }
              }
              umma_commit(&empty[stage]);
              if (++stage == VSTAGES) { stage = 0; phase ^= 1u; }
              ++c;
            }
            if (!ok) break;
            umma_commit(&sfull[gs]);
            if (gs) ++guse1; else ++guse0;
          }
        }
        umma_commit(done);
        const uint64_t t0 = globaltimer();
        while (!mbar_try_wait(done, 0u) && (globaltimer() - t0) < 2000000000ull) {
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                 "r"(TMEM_COLS));
  }
}

// --------------------------------------------------------------- host side
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static bool tried = false;
  if (!tried) {
    tried = true;
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

// 2-D K-major tile map: rows x cols elements of 2 bytes, box box_rows x 64
static bool make_map(CUtensorMap* m, const void* base, uint64_t cols, uint64_t rows, bool bf16,
                     uint32_t box_rows, bool narrow = false) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {narrow ? 32u : (cuuint32_t)BK, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, bf16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2,
                  const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE,
                  narrow ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// general tiled map: rank 2 or 3, dims/strides in elements (strides in bytes
// are derived), box in elements, 128-byte swizzle unless given
static bool make_map_nd(CUtensorMap* m, const void* base, CUtensorMapDataType dt, int esize,
                        int rank, const uint64_t* dims, const uint32_t* box,
                        CUtensorMapSwizzle swz = CU_TENSOR_MAP_SWIZZLE_128B) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t d[3], st[2];
  cuuint32_t bx[3], es[3] = {1, 1, 1};
  uint64_t stride = (uint64_t)esize;
  for (int i = 0; i < rank; ++i) {
    d[i] = dims[i];
    bx[i] = box[i];
    if (i > 0) st[i - 1] = stride;
    stride *= dims[i];
  }
  CUresult r = fn(m, dt, (cuuint32_t)rank, const_cast<void*>(base), d, st, bx, es,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, swz,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

static int num_sms() {
  static int n = 0;
  if (!n) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 1;
  }
  return n;
}

// The register split of k_tc_pass (setmaxnreg) assumes the kernel was built
// with exactly DREG registers per thread: with fewer, the epilogue's increase
// could never be granted.  Such a build is refused instead of launched.
template <bool PAIR, bool GREEDY, bool TS>
static cudaError_t pass_kernel_ready() {
  static int state = -1;
  static unsigned long long ctx = 0ull;  // the attribute is set again in a new context
  const unsigned long long cur = current_context_id();
  if (cur != ctx) state = -1;
  ctx = cur;
  if (state < 0) {
    cudaFuncAttributes fa;
    cudaError_t e = cudaFuncGetAttributes(&fa, k_tc_pass<PAIR, GREEDY, TS>);
    if (e != cudaSuccess) return e;
    if (fa.numRegs != DREG) {
      state = 0;
    } else {
      e = cudaFuncSetAttribute(k_tc_pass<PAIR, GREEDY, TS>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               (int)DCfg<PAIR>::SMEM);
      if (e != cudaSuccess) return e;
      state = 1;
    }
  }
  return state == 1 ? cudaSuccess : cudaErrorInvalidKernelImage;
}

static cudaLaunchConfig_t cluster_config(int grid, int cs, size_t smem, cudaStream_t s,
                                         cudaLaunchAttribute* at) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(D_THREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  at[0].id = cudaLaunchAttributeClusterDimension;
  at[0].val.clusterDim.x = cs;
  at[0].val.clusterDim.y = 1;
  at[0].val.clusterDim.z = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cfg;
}

// clusters of cs CTAs that can be resident at once (cached per form and size)
template <bool PAIR, bool GREEDY, bool TS>
static int max_clusters(int cs) {
  static int cache[5] = {0, 0, 0, 0, 0};
  if (cs < 1 || cs > 4) return 0;
  if (!cache[cs]) {
    cudaLaunchAttribute at[1];
    cudaLaunchConfig_t cfg = cluster_config(cs * num_sms(), cs, DCfg<PAIR>::SMEM, 0, at);
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, k_tc_pass<PAIR, GREEDY, TS>, &cfg) != cudaSuccess || n < 1)
      n = 1;
    cache[cs] = n;
  }
  return cache[cs];
}

template <bool PAIR, bool GREEDY = false, bool TS = false>
static cudaError_t launch(const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& ca,
                          const CUtensorMap& cb, const Params& P, cudaStream_t s) {
  cudaError_t e = pass_kernel_ready<PAIR, GREEDY, TS>();
  if (e != cudaSuccess) return e;
  if (P.n_tiles <= 0) return cudaSuccess;
  if (!PAIR) {
    const int grid = P.n_tiles < num_sms() ? P.n_tiles : num_sms();
    e = launch_dep(k_tc_pass<false, GREEDY, TS>, dim3(grid), dim3(D_THREADS), DCfg<false>::SMEM, s, a,
                   b, ca, cb, P);
  } else {
    const int ncl = std::min(P.n_tiles, max_clusters<PAIR, GREEDY, TS>(P.cs));
    cudaLaunchAttribute at[2];
    cudaLaunchConfig_t cfg = cluster_config(ncl * P.cs, P.cs, DCfg<PAIR>::SMEM, s, at);
    at[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.numAttrs = 2;
    e = cudaLaunchKernelEx(&cfg, k_tc_pass<PAIR, GREEDY, TS>, a, b, ca, cb, P);
  }
  if (e != cudaSuccess) return e;
  debug_kernel("k_tc_pass", s);
  count_launches(1);
  count_tc_launch();
  return cudaGetLastError();
}

// The CTA-pair schedule (the default) needs an even number of M tiles: a
// pair covers 256 rows.  DBLAST_DRAFT_PAIR=0 forces the single-SM schedule.
static bool draft_pair(int n_mt) {
  if (n_mt % 2 != 0) return false;
  const char* env = getenv("DBLAST_DRAFT_PAIR");
  return !(env && env[0] == '0' && env[1] == 0);
}

}  // namespace tc

bool tc_supported(const dblast_head* h) {
  if (!h || h->dtype != DBLAST_BF16 || (h->H % tc::BK) != 0) return false;
  const int rr = h->r + (h->e ? 1 : 0);
  if (rr > 32 || h->K > tc::KMAX) return false;
  return tc::encode_fn() != nullptr;
}

// transposed expander factor [F_z | e_z]^T as bf16 [rows_pad, H] (zero rows
// past K rr, and a zero row r of every block when e is null)
__global__ void k_prep_transpose(const __nv_bfloat16* __restrict__ U,
                                 const __nv_bfloat16* __restrict__ e, int H, int K, int r, int rr,
                                 int rows_pad, __nv_bfloat16* __restrict__ ut) {
  const size_t n = (size_t)rows_pad * H;
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n;
       i += (size_t)gridDim.x * blockDim.x) {
    const int hh = (int)(i % H);
    const int row = (int)(i / H);
    __nv_bfloat16 v = __float2bfloat16(0.f);
    if (row < K * rr) {
      const int z = row / rr, k = row - z * rr;
      if (k < r) v = U[((size_t)z * H + hh) * r + k];
      else if (e) v = e[(size_t)z * H + hh];
    }
    ut[i] = v;
  }
}

static void transpose_expander(const void* F, const void* e, const dblast_head* h,
                               const PrepLayout& pl, __nv_bfloat16* out, cudaStream_t s) {
  const int rows_pad = ceil_div(h->K * pl.rr, tc::BM) * tc::BM;
  k_prep_transpose<<<1024, 256, 0, s>>>(static_cast<const __nv_bfloat16*>(F),
                                        static_cast<const __nv_bfloat16*>(e), h->H, h->K, h->r,
                                        pl.rr, rows_pad, out);
  debug_kernel("k_prep_transpose", s);
  count_launches(1);
}

cudaError_t launch_prep_tc(const dblast_head* h, const PrepLayout& pl, cudaStream_t s) {
  unsigned char* prep = static_cast<unsigned char*>(h->prep);
  const int rows = h->K * pl.rr;
  const int rows_pad = ceil_div(rows, tc::BM) * tc::BM;
  auto* utp = reinterpret_cast<__nv_bfloat16*>(prep + pl.off_ut);
  transpose_expander(h->U, h->e, h, pl, utp, s);
  // V_z^T (with a zero row for the constant code of e) for the per-call codes GEMM
  transpose_expander(h->Vf, nullptr, h, pl, reinterpret_cast<__nv_bfloat16*>(prep + pl.off_vt), s);
  CUtensorMap ma, mb;
  if (!tc::make_map(&ma, utp, h->H, rows_pad, true, tc::BM) ||
      !tc::make_map(&mb, h->W, h->H, h->V, true, tc::DBN))
    return cudaErrorInvalidValue;
  tc::Params P{};
  P.mode = tc::MODE_PREP;
  P.cs = 1;
  P.n_mt = rows_pad / tc::BM;
  P.n_vt = ceil_div(h->V, tc::DBN);
  P.n_tiles = P.n_mt * P.n_vt;
  P.nb = h->H / tc::BK;
  P.K = h->K;
  P.rp = pl.rp;
  P.zps = 1;
  P.M = rows;
  P.V = h->V;
  P.Mpad = rows_pad;
  P.wu = reinterpret_cast<float*>(prep + pl.off_wu);
  P.prep_rows = rows;
  P.split_stride = 0;
  P.status = reinterpret_cast<DevStatus*>(prep + pl.off_status);
  P.spin_limit = wait_limit();
  return tc::launch<false>(ma, mb, ma, mb, P, s);
}

// codes c_{m,z} = V_z^T h_m for every position: the prep machinery with
// A = V^T [K rr, H], B = hidden [M, H], split-K partials [ksplit][M][K rr]
cudaError_t launch_codes_tc(const StepCtx& c, float* part, int* nsplit) {
  const dblast_head* h = c.head;
  const WsLayout& w = c.wl;
  const int rows = h->K * w.rr;
  const int rows_pad = ceil_div(rows, tc::BM) * tc::BM;
  CUtensorMap ma, mb;
  if (!tc::make_map(&ma, c.prep + c.pl.off_vt, h->H, rows_pad, true, tc::BM) ||
      !tc::make_map(&mb, c.args->hidden, h->H, w.M, true, tc::DBN))
    return cudaErrorInvalidValue;
  const int nb64 = h->H / tc::BK;
  const int base_tiles = (rows_pad / tc::BM) * ceil_div(w.M, tc::DBN);
  int ks = 1;
  for (int d = 1; d <= CODES_MAX_SPLIT && d <= nb64; ++d)
    if (nb64 % d == 0 && base_tiles * d <= tc::num_sms()) ks = d;
  tc::Params P{};
  P.mode = tc::MODE_PREP;
  P.cs = 1;
  P.n_mt = rows_pad / tc::BM;
  P.n_vt = ceil_div(w.M, tc::DBN);
  P.n_tiles = P.n_mt * P.n_vt * ks;
  P.nb = nb64 / ks;
  P.K = h->K;
  P.rp = w.rp;
  P.zps = 1;
  P.M = rows;
  P.V = w.M;
  P.Mpad = rows_pad;
  P.wu = part;
  P.prep_rows = rows;
  P.split_stride = (size_t)w.M * rows;
  P.status = wsp<DevStatus>(c, w.off_status);
  P.spin_limit = wait_limit();
  *nsplit = ks;
  return tc::launch<false>(ma, mb, ma, mb, P, c.stream);
}

cudaError_t launch_draft_pass_tc(const StepCtx& c) {
  const dblast_head* h = c.head;
  const WsLayout& w = c.wl;
  const int n_mt = w.Mpad / tc::BM;
  const bool pair = tc::draft_pair(n_mt);
  const int cs = pair ? 2 : 1;
  const uint32_t bq = tc::DBN / cs;  // B rows each CTA loads
  CUtensorMap ma, mb, mca, mcb;
  const unsigned char* prep = c.prep;
  const bool narrow = tc::BK / (2 * w.rp) == 2;  // rank 16: one component per 64-byte box
  if (!tc::make_map(&ma, c.args->hidden, h->H, w.M, true, tc::BM) ||
      !tc::make_map(&mb, h->W, h->H, h->V, true, bq) ||
      !tc::make_map(&mca, c.ws + w.off_cop, w.KC, w.Mpad, false, tc::BM, narrow) ||
      !tc::make_map(&mcb, prep + c.pl.off_wuop, w.KC, h->V, false, bq, narrow))
    return cudaErrorInvalidValue;
  tc::Params P{};
  P.mode = c.greedy ? tc::MODE_GREEDY : tc::MODE_DRAFT;
  P.cs = cs;
  P.n_mt = n_mt;
  P.n_vt = ceil_div(h->V, tc::DBN);
  P.n_tiles = (P.n_mt / cs) * P.n_vt;
  P.nb = h->H / tc::BK;
  P.K = h->K;
  P.rp = w.rp;
  P.zps = tc::BK / (2 * w.rp);
  P.M = w.M;
  P.V = h->V;
  P.Mpad = w.Mpad;
  P.k2 = c.greedy ? 1.f : c.k2;  // greedy records hold logits, not log2-scaled ones
  P.vbias = h->vbias;
  P.cscale = wsp<float>(c, w.off_cscale);
  P.sw = prp<float>(c, c.pl.off_sw);
  P.stash = wsp<float>(c, w.off_stash);
  P.partd = wsp<float2>(c, w.off_partd);
  P.partg = wsp<float>(c, w.off_partg);
  P.status = wsp<DevStatus>(c, w.off_status);
  P.spin_limit = wait_limit();
  if (c.fuse_tstats) {
    P.tgt = static_cast<const __nv_bfloat16*>(c.target);
    P.t_rows = w.N * c.Bt;
    P.t_Bt = c.Bt;
    P.t_B = w.B;
    P.t_Rt = w.Rt;
    P.t_nt = w.nt;
    P.t_k2 = LOG2E / c.args->temperature;
    P.t_partt = wsp<float2>(c, w.off_partt);
    P.t_lt2 = wsp<float2>(c, w.off_lt2);
    P.t_coll = wsp<float>(c, w.off_coll);
    P.t_lse = c.lse_target;
  }
  if (c.greedy)
    return c.fuse_tstats
               ? (pair ? tc::launch<true, true, true>(ma, mb, mca, mcb, P, c.stream)
                       : tc::launch<false, true, true>(ma, mb, mca, mcb, P, c.stream))
               : (pair ? tc::launch<true, true>(ma, mb, mca, mcb, P, c.stream)
                       : tc::launch<false, true>(ma, mb, mca, mcb, P, c.stream));
  if (c.fuse_tstats)
    return pair ? tc::launch<true, false, true>(ma, mb, mca, mcb, P, c.stream)
                : tc::launch<false, false, true>(ma, mb, mca, mcb, P, c.stream);
  return pair ? tc::launch<true>(ma, mb, mca, mcb, P, c.stream)
              : tc::launch<false>(ma, mb, mca, mcb, P, c.stream);
}

cudaError_t launch_verify_pass_tc(const StepCtx& c) {
  const dblast_head* h = c.head;
  const WsLayout& w = c.wl;
  CUtensorMap mca, mcb, mxs, mxt;
  if (!tc::make_map(&mca, c.ws + w.off_cop, w.KC, w.Mpad, false, tc::BM) ||
      !tc::make_map(&mcb, c.prep + c.pl.off_wuop, w.KC, h->V, false, tc::BN))
    return cudaErrorInvalidValue;
  // stash and target tiles through shared memory: 16-byte row strides and
  // whole sequences per 128-row tile
  const bool use_x = (h->V % 8) == 0 && (tc::BM % w.B) == 0 &&
                     (reinterpret_cast<uintptr_t>(c.target) & 15u) == 0;
  mxs = mca;
  mxt = mca;
  if (use_x) {
    const uint64_t ds[2] = {(uint64_t)h->V, (uint64_t)w.M};
    const uint32_t bs[2] = {32, (uint32_t)tc::BM};
    const uint64_t dt[3] = {(uint64_t)h->V, (uint64_t)c.Bt, (uint64_t)w.N};
    const uint32_t bt[3] = {32, (uint32_t)w.B, (uint32_t)(tc::BM / w.B)};
    if (!tc::make_map_nd(&mxs, c.ws + w.off_stash, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, 2, ds, bs) ||
        !tc::make_map_nd(&mxt, c.target, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, 3, dt, bt,
                         CU_TENSOR_MAP_SWIZZLE_64B))
      return cudaErrorInvalidValue;
  }
  tc::VParams P{};
  P.n_mt = w.Mpad / tc::BM;
  P.n_vt = ceil_div(h->V, tc::BN);
  P.n_tiles = P.n_mt * P.n_vt;
  P.ncs = ceil_div(w.KC, tc::BK);
  P.K = h->K;
  P.rp = w.rp;
  P.zps = tc::BK / (2 * w.rp);
  P.M = w.M;
  P.V = h->V;
  P.Mpad = w.Mpad;
  P.B = w.B;
  P.Bt = c.Bt;
  P.use_x = use_x ? 1 : 0;
  P.k2 = c.k2;
  P.vcz = wsp<float2>(c, w.off_vcz);
  P.vb0 = wsp<float>(c, w.off_vb0);
  P.lt2 = wsp<float2>(c, w.off_lt2);
  P.stash = wsp<float>(c, w.off_stash);
  P.target = static_cast<const __nv_bfloat16*>(c.target);
  P.partv = wsp<float2>(c, w.off_partv);
  P.status = wsp<DevStatus>(c, w.off_status);
  P.spin_limit = wait_limit();
  // the register split (setmaxnreg) assumes exactly VREG registers per thread
  static int state = -1;
  static unsigned long long ctx = 0ull;  // the attribute is set again in a new context
  const unsigned long long cur = current_context_id();
  if (cur != ctx) state = -1;
  ctx = cur;
  if (state < 0) {
    cudaFuncAttributes fa;
    cudaError_t e = cudaFuncGetAttributes(&fa, tc::k_tc_verify);
    if (e != cudaSuccess) return e;
    if (fa.numRegs != tc::VREG) {
      state = 0;
    } else {
      e = cudaFuncSetAttribute(tc::k_tc_verify, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               (int)tc::VSMEM);
      if (e != cudaSuccess) return e;
      state = 1;
    }
  }
  if (state != 1) return cudaErrorInvalidKernelImage;
  const int grid = P.n_tiles < tc::num_sms() ? P.n_tiles : tc::num_sms();
  cudaError_t le = launch_dep(tc::k_tc_verify, dim3(grid), dim3(tc::NUM_THREADS), tc::VSMEM,
                              c.stream, mca, mcb, mxs, mxt, P);
  if (le != cudaSuccess) return le;
  debug_kernel("k_tc_verify", c.stream);
  count_launches(1);
  count_tc_launch();
  return cudaGetLastError();
}

}  // namespace dblast
