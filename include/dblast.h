/*
 * dblast.h - C ABI of the DBLast draft+verify step on one GPU (sm_103a).
 *
 * The step (paper: "DBLast: Dependent Block Drafting for Stochastic
 * Speculative Decoding") drafts a block of B tokens from a K-component
 * latent-mixture proposal and verifies it against given target logits:
 *
 *   draft   - category prior and latent draw z-hat (Sec. 3.1, "Drafter
 *             sampling during inference"), branch distributions through the
 *             reused vocabulary head (Sec. 3.1, Architecture; Eq. 5), one
 *             draft token per position from the z-hat branch, the category
 *             posterior (Eq. category-posterior) and the mixture conditional
 *             q(x_i|x_<i) (Eq. dep-next-token, equal to Eq. 1).
 *   verify  - acceptance with probability min(1, p/q) (Eq. 2), stop at the
 *             first rejection, residual draw from norm([p - q]_+) or the
 *             bonus token when all B are accepted (Algorithm 1; Appendix A,
 *             "Distributional correctness"), the overlap
 *             alpha_i = sum_v min(p_i(v), q(v|x_<i)) and the expected accepted
 *             length of the drafted block sum_i prod_{j<=i} A_j (Eq. 3).
 *
 * Greedy-branch mode (args->mode = DBLAST_MODE_GREEDY; Sec. 3.1, "Drafter
 * sampling during inference"; Appendix A, "Greedy-Branch Proposal",
 * "Prefix-Marginalized Conditional" and its verification algorithm): every
 * branch is decoded greedily, x-hat_{i,z} = argmax_v l_{i,z,v} (lowest index
 * on ties), the block is the z-hat branch, and verification uses the sparse
 * conditional q_greedy(v|x_<i) = sum_{z in C_i} pi~_{i,z} 1{v = x-hat_{i,z}}
 * over the consistent branches C_i = {z : x-hat_{j,z} = x_j for all j < i},
 * pi~ = pi restricted to C_i and renormalised.  Acceptance, residual
 * [p - q_greedy]_+, bonus, alpha and Eq. 3 are as above.  Stream 1 is not
 * used in this mode.
 *
 * The expander is rank r: h_{i,z} = h_i + U_z (V_z^T h_i) + e_z.
 * Temperatures: q_i(.|z) = softmax(l_{i,z}/T), p_i = softmax(t_i/T),
 * prior softmax(l/Z_T) (Z_T = 0 selects the highest-prior category).
 *
 * Conventions for every entry point:
 *   - All array pointers are DEVICE pointers to caller-owned, row-major,
 *     contiguous memory, 16-byte aligned.  The library never allocates or
 *     frees device memory; scratch space comes from the caller ("prep" and
 *     "workspace" buffers, sized by the *_bytes queries).
 *   - Calls are asynchronous on `stream`.  Argument errors are returned
 *     immediately, before any launch.  Errors found on the device (a bounded
 *     wait that ran out) are recorded in the workspace and reported by
 *     dblast_device_status().
 *   - Shapes: 1 <= K <= 32, 1 <= r <= 64, 1 <= B <= 32, N >= 1, V >= 1,
 *     H >= 8 with H % 8 == 0; T > 0; Z_T >= 0.
 *   - Random decisions use one uniform each from Philox4x32-10 (Salmon et al.,
 *     SC'11) with key (seed lo, seed hi) and counter
 *     (0, pos_abs, n, (stream << 24) | (round & 0xffffff)); u = ((w0>>9)+0.5)
 *     * 2^-23.  Streams: 0 latent category (pos_abs = pos[n]), 1 draft token,
 *     2 acceptance, 3 residual/bonus (pos_abs = pos[n] + i).  Every draw is an
 *     inverse-CDF draw in vocabulary order: the smallest index whose
 *     cumulative mass exceeds u times the total.
 */
#ifndef DBLAST_H_
#define DBLAST_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* dblast_stream_t; /* a cudaStream_t; NULL = legacy default stream */

typedef enum {
  DBLAST_OK = 0,
  DBLAST_ERR_INVALID_ARG = 1,  /* NULL pointer, bad shape, bad temperature */
  DBLAST_ERR_UNSUPPORTED = 2,  /* shape/dtype the requested implementation cannot run */
  DBLAST_ERR_WORKSPACE = 3,    /* prep or workspace buffer too small / misaligned */
  DBLAST_ERR_CUDA = 4,         /* a CUDA runtime call failed */
  DBLAST_ERR_TIMEOUT = 5,      /* a device-side bounded wait ran out (see dblast_device_status) */
  DBLAST_ERR_NO_DEVICE = 6,    /* no usable sm_103 device */
  DBLAST_ERR_BOUNDS = 7        /* a device-side index check failed (see dblast_set_checks) */
} dblast_status;

typedef enum { DBLAST_BF16 = 0, DBLAST_F32 = 1 } dblast_dtype;

/* Kernel family for the two vocabulary-wide passes.  AUTO picks TCGEN05 for
 * bf16 inputs with H % 64 == 0, else SIMT (plain CUDA cores, any shape). */
typedef enum { DBLAST_IMPL_AUTO = 0, DBLAST_IMPL_SIMT = 1, DBLAST_IMPL_TCGEN05 = 2 } dblast_impl;

/* Drafting mode.  SOFT: draft tokens sampled from the z-hat branch
 * distribution, dense mixture conditional (Eq. dep-next-token).  GREEDY: the
 * greedy-branch decoder of Appendix A (see the top of this file). */
typedef enum { DBLAST_MODE_SOFT = 0, DBLAST_MODE_GREEDY = 1 } dblast_mode;

/* Drafter head (Sec. 3.1, Architecture; Table 1 with a rank-r expander).
 * W is the reused vocabulary head, U/Vf the expander factors, e its optional
 * bias, Wp/bp the category-prior head, vbias an optional vocabulary bias.
 * W, U, Vf, e, Wp have `dtype`; bp and vbias are fp32. */
typedef struct {
  int V, H, K, r;
  dblast_dtype dtype;
  const void* W;      /* [V, H]    */
  const void* U;      /* [K, H, r] */
  const void* Vf;     /* [K, H, r] */
  const void* e;      /* [K, H] or NULL */
  const void* Wp;     /* [K, H]    */
  const float* bp;    /* [K] or NULL */
  const float* vbias; /* [V] or NULL */
  void* prep;         /* device buffer, dblast_prep_bytes() bytes, filled by dblast_head_prepare() */
  size_t prep_bytes;
} dblast_head;

/* One block per sequence n.  pos[n] is the absolute position of the first
 * block token and round[n] counts the sequence's draft/verify rounds; both
 * feed the Philox counters and are advanced by the verify step
 * (pos += n_emitted, round += 1). */
typedef struct {
  int N, B;
  float temperature;     /* T > 0, for drafter and target token distributions */
  float z_temperature;   /* Z_T >= 0, category temperature */
  uint64_t seed;
  const void* hidden;    /* [N, B, H] block hidden states h_i (head dtype) */
  const void* anchor;    /* [N, H] block-anchor state for the prior, or NULL = hidden[:, 0, :] */
  int64_t* pos;          /* [N] in/out */
  uint32_t* round;       /* [N] in/out */
  dblast_impl impl;
  dblast_mode mode;      /* SOFT (0) or GREEDY (1); draft and verify of one block use the same */
} dblast_block_args;

/* Draft outputs.  Every pointer may be NULL (not written). */
typedef struct {
  int32_t* z_hat;  /* [N]       latent category */
  float* pi;       /* [N, K]    tempered prior softmax(l/Z_T) */
  int32_t* tokens; /* [N, B]    draft block */
  float* lse;      /* [N, B, K] natural log of sum_v exp(l_{i,z,v}/T) (SOFT mode; not written
                                in GREEDY mode) */
  float* logw;     /* [N, B, K] natural log of the posterior q(z|y,x_<i); GREEDY: log pi~_{i,z},
                                -inf for z outside C_i */
  float* q_tok;    /* [N, B]    q(x_i|y,x_<i) (GREEDY: q_greedy) */
  int32_t* branch_tokens; /* [N, B, K] GREEDY: x-hat_{i,z} of every branch (not written in SOFT
                                mode) */
} dblast_draft_out;

/* Verify inputs/outputs.  target is required; every output may be NULL. */
typedef struct {
  const void* target;   /* [N, B + has_bonus, V] target logits (head dtype) */
  int has_bonus;        /* 1: row B holds the bonus-position logits */
  float* p_tok;         /* [N, B]     p_i(x_i) */
  float* accept_prob;   /* [N, B]     A_i = min(1, p/q) (Eq. 2) */
  float* alpha;         /* [N, B]     sum_v min(p_i(v), q(v|x_<i)) */
  float* lse_target;    /* [N, B+has_bonus] natural log of sum_v exp(t/T) */
  int32_t* accepted;    /* [N]        accepted draft tokens L (bonus/residual excluded) */
  int32_t* emitted;     /* [N, B+1]   accepted tokens then the residual/bonus token, -1 padded */
  int32_t* n_emitted;   /* [N]        number of valid entries in emitted */
  float* exp_len;       /* [N]        sum_i prod_{j<=i} A_j (Eq. 3) */
  float* alpha_len;     /* [N]        sum_i prod_{j<=i} alpha_j */
  uint32_t* tie_flags;  /* [N]        bit0 z-hat, bit1 draft, bit2 accept, bit3 residual/bonus,
                                       bit4 residual mass < 1e-6: a decision within 1e-6 of its threshold
                                       by the kernels' own arithmetic.  Bits 8-14: the same kinds,
                                       "near": within 1e-6 plus the kernels' precision allowance
                                       (5e-5 of probability mass for a draw, 1e-4 relative for the
                                       acceptance ratio p/q), so every decision that may be a tie of
                                       the exact arithmetic is flagged; a tie bit implies its near bit.
                                       GREEDY mode: bit1 (and bit9) = the greedy argmax of a branch in
                                       C_i whose top-two logit gap is below 1e-4 (the logits are fp32) */
  float* collision;     /* [N, B]     sum_v p_i(v)^2, the collision probability of target row i (App. B) */
  float* determinism;   /* [N]        target-block early determinism D_B = (1/B) sum_j prod_{i<=j}
                                       collision_i (App. B, Eq. appendix-early-determinism, for
                                       target rows that do not depend on the drafted prefix) */
  /* Target filter (inputs), applied to every target row after the temperature
   * and before verification (Sec. 3.2, Sec. 4: temperature, top-k, top-p):
   * top-k keeps the k largest logits, ties at the k-th value to the lower
   * token index (0 or >= V: off); top-p then keeps, in the order (logit desc,
   * index asc), every token whose preceding mass renormalised over the
   * top-k set is below top_p (0 or >= 1: off).  p' is renormalised over the
   * kept set and used for p_tok, acceptance, alpha, the residual, the bonus
   * token and collision/determinism; lse_target stays the unfiltered
   * log-sum-exp.  With a filter on, at most 256 tokens may stay (top-p needs
   * top_k in 1..256, or V <= 256) and V <= 262144; else DBLAST_ERR_UNSUPPORTED.
   * tie_flags bit5 (and bit13): a top-p cut within 1e-6 of top_p on some row. */
  int top_k;
  float top_p;
} dblast_verify_out;

/* Bytes of the prep buffer for this head (depends on V, K, r, e != NULL). */
size_t dblast_prep_bytes(const dblast_head* head);

/* Bytes of the per-call workspace for N sequences of block B.  Its first 256
 * bytes are the device status word that dblast_device_status() reads and
 * clears: zero them once before the workspace's first call (the rest needs
 * no initialisation). */
size_t dblast_workspace_bytes(const dblast_head* head, int N, int B, int has_bonus);

/* Once per weight set: fills head->prep with W U_z (and W e_z) in fp32 and in
 * the split-fp16 operand layout of the tensor-core pass.  Asynchronous. */
dblast_status dblast_head_prepare(const dblast_head* head, dblast_stream_t stream);

/* Draft: prior, z-hat, branch statistics, draft block, posterior and q_tok.
 * Leaves in `workspace` what dblast_verify_block needs. */
dblast_status dblast_draft_block(const dblast_head* head, const dblast_block_args* args,
                                 dblast_draft_out* out, void* workspace, size_t workspace_bytes,
                                 dblast_stream_t stream);

/* Verify a block drafted by dblast_draft_block with the same head, args and
 * workspace (unmodified in between).  Advances pos and round. */
dblast_status dblast_verify_block(const dblast_head* head, const dblast_block_args* args,
                                  dblast_verify_out* out, void* workspace, size_t workspace_bytes,
                                  dblast_stream_t stream);

/* Both, in one call. */
dblast_status dblast_draft_and_verify(const dblast_head* head, const dblast_block_args* args,
                                      dblast_draft_out* dout, dblast_verify_out* vout,
                                      void* workspace, size_t workspace_bytes,
                                      dblast_stream_t stream);

/* Synchronises `stream`, returns DBLAST_ERR_TIMEOUT if a device-side wait of
 * a previous call on this workspace ran out, else DBLAST_ERR_BOUNDS if an
 * index check of such a call failed (checks on), and clears the record. */
dblast_status dblast_device_status(void* workspace, dblast_stream_t stream);

/* Host-side fault injection for tests: spin limit of the device-side bounded
 * waits of later calls (0 = default).  A limit of 1 makes waits give up. */
void dblast_set_wait_limit(uint32_t spins);

/* Device-side index checks of later calls (process-wide; 0 = off, the
 * default unless the environment sets DBLAST_CHECK=1).  With checks on, every
 * data-dependent token index a kernel reads (the given tokens of
 * dblast_al_objective, the drafted tokens the verify kernels look up) is
 * tested against [0, V); a value outside it is recorded in the workspace
 * status word and reported as DBLAST_ERR_BOUNDS by dblast_device_status().
 * There is no trap: with checks on or off the access itself uses the index
 * clamped into [0, V), so an out-of-range value never reads outside the
 * target or stash rows.  Not a paper operation: a debugging aid. */
void dblast_set_checks(int enable);

/* Measurement counters of this process.  dblast_stats_reset(n) zeroes them
 * and sets per-pass timing: with n > 0, CUDA events are recorded on the
 * caller's stream around every n-th draft pass (the vocabulary-head
 * contraction with its fused softmax epilogue) and every n-th verify pass
 * (the fused target-streaming kernel) from the reset on; n = 0 turns it off.
 * An event between two kernels keeps the later one from starting while the
 * earlier one drains, so a timed call runs a little slower than an untimed
 * one; n > 1 leaves the other calls as they are.  dblast_stats_get() waits
 * for the recorded events and returns the summed pass times (ms), the number
 * of timed passes and the number of kernel launches issued by the library
 * since the reset. */
typedef struct {
  uint64_t calls;            /* draft/verify entry-point calls */
  uint64_t kernel_launches;  /* kernels launched by the library */
  uint64_t tc_launches;      /* of which tensor-core (tcgen05) kernels */
  uint64_t timed_draft, timed_verify;
  double draft_pass_ms, verify_pass_ms;
} dblast_stats;
void dblast_stats_reset(int enable_pass_timing);
dblast_status dblast_stats_get(dblast_stats* out);

/* No-allocation variant of the target log-sum-exp pass.  The paper has no
 * counterpart; this is a service for callers that cannot allocate device
 * memory when they call in, such as a plugin run inside another engine's
 * enqueue step (cudaMalloc would synchronise the device and bypass that
 * engine's memory pool) or code with a fixed device-memory budget.
 *
 *   lse_out[row] = log sum_v exp(target[row, v] / temperature)
 *
 * target: [rows, V] logits of `dtype` (device); lse_out: [rows] fp32 (device).
 * Its only scratch is a static device array of DBLAST_NOALLOC_MAX_RECORDS
 * 8-byte records (8 MiB on every GPU that loads the library, held until the
 * process exits); rows * ceil(V / 128) must not exceed it, otherwise
 * DBLAST_ERR_WORKSPACE is returned and nothing is launched.  It calls no
 * allocation routine.  The first call on a device, with that device current,
 * looks up the array's device address (cudaGetSymbolAddress); make that first
 * call before any stream capture.  After a cudaDeviceReset the next call sees
 * the device's new context and looks the address up again (so, again, before
 * any capture).  `stream` must belong to the current device.  Every call reuses the same array, so calls that overlap on the GPU
 * (other streams or threads) race; serialise them. */
#define DBLAST_NOALLOC_MAX_RECORDS (1u << 20)
dblast_status dblast_target_lse_noalloc(const void* target, int rows, int V, dblast_dtype dtype,
                                        float temperature, float* lse_out,
                                        dblast_stream_t stream);

/* Training-side objectives, forward only, on given target blocks (Sec. 3.2).
 * For each sequence n the target block x*_{1:B} = tokens[n] (sampled from the
 * target) is scored under the soft latent-mixture proposal (Eq. 5; the
 * prior at args->z_temperature, branch distributions at args->temperature):
 *   q_cond[n, i] = q(x*_i|y, x*_<i) (Eqs. category-posterior, dep-next-token)
 *   p_tok[n, i]  = p(x*_i), the target after the filter top_k / top_p (as in
 *                  dblast_verify_out)
 *   accept_prob  = A_i = min(1, p/q) (Eq. 2)
 *   r[n, l]      = prod_{j<=l} q_cond_j / p_tok_j, the prefix importance ratio
 *   S[n, l]      = sum_{i<=l} prod_{j<=i} A_j
 *   l_tau[n]     = the first l (1-based) with r_l < tau, else B
 *   j_al[n]      = sum_{l<=l_tau} (log r_l + log S_l) (Eq. subblock-objective;
 *                  the training loss is -j_al, Eq. training-loss)
 *   nll[n]       = -log sum_z q(z|y) prod_i q_i(x*_i|y,z) (Eq. dependent-nll;
 *                  K = 1: Eq. independent-nll)
 *   tie_flags[n] bit5: a top-p cut within 1e-6; bit6: an r_l within 1e-6
 *                (relative) of tau among l <= l_tau; bits 13, 14: the same
 *                within the precision allowance (1e-4 relative per factor of r_l).
 * Natural logarithms.  args->mode must be DBLAST_MODE_SOFT; args->seed, pos
 * and round are read (the latent draw of the shared draft kernels) but not
 * advanced.  Uses the step workspace (dblast_workspace_bytes with the same
 * N, B, has_bonus).  Every output may be NULL. */
typedef struct {
  const int32_t* tokens; /* [N, B] target block x*_{1:B} */
  const void* target;    /* [N, B + has_bonus, V] target logits (head dtype) */
  int has_bonus;
  int top_k;
  float top_p;
  float tau;             /* truncation threshold, >= 0 (the paper: 0.1) */
  float* nll;            /* [N] */
  float* j_al;           /* [N] */
  int32_t* l_tau;        /* [N] */
  float* r;              /* [N, B] */
  float* S;              /* [N, B] */
  float* accept_prob;    /* [N, B] */
  float* q_cond;         /* [N, B] */
  float* p_tok;          /* [N, B] */
  uint32_t* tie_flags;   /* [N] */
} dblast_al_args;
dblast_status dblast_al_objective(const dblast_head* head, const dblast_block_args* args,
                                  const dblast_al_args* al, void* workspace,
                                  size_t workspace_bytes, dblast_stream_t stream);

/* Target-block early determinism of given target rows (App. B).
 *   collision[n, i] = sum_v p_{n,i}(v)^2 for the first b rows of sequence n,
 *   d_exact[n]      = (1/b) sum_j prod_{i<=j} collision[n, i]
 *                     (Eq. appendix-early-determinism when the rows do not
 *                     depend on the sampled prefix),
 *   d_hat[n]        = 1/(M b) sum_m sum_j prod_{i<=j} p_{n,i}(x_i^(m)), the
 *                     M-sample estimator (Eq. appendix-early-determinism-estimator)
 *                     with x_i^(m) ~ p_{n,i} drawn by inverse CDF from the
 *                     stream-4 uniform (round field = m, sequence n, pos_abs = i),
 *   samples[n, m, i] = x_i^(m).
 * target: [N, rows, V] device logits of `dtype`, p = softmax(t / temperature);
 * 1 <= b <= min(rows, 32).  Every output is a device pointer or NULL; d_hat
 * and samples need M >= 1.  Scratch: `workspace` of
 * dblast_determinism_workspace_bytes(N, rows, b, V, M) bytes, 16-byte aligned.
 * Asynchronous on `stream`; argument errors return before any launch. */
size_t dblast_determinism_workspace_bytes(int N, int rows, int b, int V, int M);
dblast_status dblast_target_determinism(const void* target, dblast_dtype dtype, int N, int rows,
                                        int b, int V, float temperature, int M, uint64_t seed,
                                        float* collision, float* d_exact, float* d_hat,
                                        int32_t* samples, void* workspace,
                                        size_t workspace_bytes, dblast_stream_t stream);

const char* dblast_status_string(dblast_status s);
const char* dblast_version(void);

#ifdef __cplusplus
}
#endif
#endif /* DBLAST_H_ */
