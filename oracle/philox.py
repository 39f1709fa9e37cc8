"""Counter-based uniforms for the oracle: Philox4x32-10 and the decision uniforms.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path imports this module;
only tests/, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may use it.

Philox4x32-10 is the counter-based generator of Salmon, Moraes, Dror and Shaw,
"Parallel random numbers: as easy as 1, 2, 3" (SC'11).  One round maps the
counter (c0, c1, c2, c3) under the key (k0, k1) to

    (hi(M1*c2) ^ c1 ^ k0,  lo(M1*c2),  hi(M0*c0) ^ c3 ^ k1,  lo(M0*c0))

with the published multipliers M0 = 0xD2511F53, M1 = 0xCD9E8D57; after each
round the key is bumped by the Weyl constants (0x9E3779B9, 0xBB67AE85).  Ten
rounds make Philox4x32-10.  Written here from that definition with plain
Python integers (slow and obviously exact).

The paper draws its randomness abstractly (category, draft block, acceptance,
residual; Sec. 3.1 and Algorithm 1).  The build fixes one uniform per decision,
keyed by (seed; stream, round, sequence, absolute position):

    key     = (seed & 0xffffffff, seed >> 32)
    counter = (draw, pos_abs & 0xffffffff, seq, (stream << 24) | (round & 0xffffff))
    u       = ((word0 >> 9) + 0.5) * 2**-23

so u lies in (0, 1) and is exactly representable in fp32 and fp64.

Parity pin: this generator is compared against an independent library
implementation of Philox4x32-10 (Triton's, run on the CPU in interpreter mode)
in tests/test_oracle_philox.py, and against cuRAND's Philox4_32_10 on the GPU.
"""

MASK32 = 0xFFFFFFFF
PHILOX_M0 = 0xD2511F53
PHILOX_M1 = 0xCD9E8D57
PHILOX_W0 = 0x9E3779B9
PHILOX_W1 = 0xBB67AE85

# decision streams (one uniform per decision)
STREAM_PRIOR = 0     # latent category z-hat, once per block
STREAM_DRAFT = 1     # draft token x_i at position i
STREAM_ACCEPT = 2    # accept / reject x_i
STREAM_RESIDUAL = 3  # residual draw at the first rejection, or the bonus token
STREAM_TARGET = 4    # target block samples of the early-determinism estimator
                     # (round field = sample index m, pos_abs = position i)


def philox4x32_10(ctr, key):
    """Return the four 32-bit output words of Philox4x32-10(ctr, key)."""
    c0, c1, c2, c3 = (int(c) & MASK32 for c in ctr)
    k0, k1 = (int(k) & MASK32 for k in key)
    for _ in range(10):
        p0 = PHILOX_M0 * c0
        p1 = PHILOX_M1 * c2
        c0, c1, c2, c3 = (((p1 >> 32) ^ c1 ^ k0) & MASK32, p1 & MASK32,
                          ((p0 >> 32) ^ c3 ^ k1) & MASK32, p0 & MASK32)
        k0 = (k0 + PHILOX_W0) & MASK32
        k1 = (k1 + PHILOX_W1) & MASK32
    return (c0, c1, c2, c3)


def word_to_uniform(w):
    """Map a 32-bit word to u = ((w >> 9) + 0.5) * 2^-23, a value in (0, 1)."""
    return ((int(w) >> 9) + 0.5) * (2.0 ** -23)


def decision_uniform(seed, stream, round_, seq, pos_abs, draw=0):
    """The uniform for one decision (see the module docstring for the key/counter)."""
    seed = int(seed)
    key = (seed & MASK32, (seed >> 32) & MASK32)
    ctr = (int(draw) & MASK32, int(pos_abs) & MASK32, int(seq) & MASK32,
           ((int(stream) & 0xFF) << 24) | (int(round_) & 0xFFFFFF))
    return word_to_uniform(philox4x32_10(ctr, key)[0])
