"""Philox4x32-10 counter-based generator, written from its published definition.

TEST INFRASTRUCTURE ONLY (see oracle/__init__.py): the oracle's own copy of the generator that
supplies the uniforms of speculative sampling.  The CUDA library carries an independent
implementation; the two share no code and are checked against the known-answer vectors that the
generator's authors published (Salmon, Moraes, Dror, Shaw, "Parallel random numbers: as easy as
1, 2, 3", SC'11; Random123 known-answer tests) and against each other.

Definition (SC'11, Sec. 3.2 / Fig. 2): a Philox-4x32 round maps counter (c0, c1, c2, c3) under
key (k0, k1) to (hi(M1*c2) ^ c1 ^ k0, lo(M1*c2), hi(M0*c0) ^ c3 ^ k1, lo(M0*c0)), with
multipliers M0 = 0xD2511F53, M1 = 0xCD9E8D57; between rounds the key is bumped by the Weyl
constants (0x9E3779B9, 0xBB67AE85).  Philox4x32-10 applies 10 rounds (9 key bumps).

Uniform mapping used by the verifier: u = (x >> 8) * 2**-24 for the first output word x, i.e. a
24-bit uniform on [0, 1) that is exact in fp32.
"""
import numpy as np

M0 = 0xD2511F53
M1 = 0xCD9E8D57
W0 = 0x9E3779B9
W1 = 0xBB67AE85
_MASK = 0xFFFFFFFF


def philox4x32_10(counter, key):
    """Vectorised Philox4x32-10.

    counter: array-like [..., 4] of uint32 words; key: array-like [..., 2].
    Returns uint32 array [..., 4].
    """
    c = np.asarray(counter, dtype=np.uint64) & _MASK
    k = np.asarray(key, dtype=np.uint64) & _MASK
    c0, c1, c2, c3 = (c[..., i].copy() for i in range(4))
    k0 = np.broadcast_to(k[..., 0], c0.shape).copy()
    k1 = np.broadcast_to(k[..., 1], c0.shape).copy()
    for r in range(10):
        if r > 0:
            k0 = (k0 + W0) & _MASK
            k1 = (k1 + W1) & _MASK
        p0 = c0 * np.uint64(M0)  # < 2**64, exact in uint64
        p1 = c2 * np.uint64(M1)
        hi0, lo0 = p0 >> np.uint64(32), p0 & _MASK
        hi1, lo1 = p1 >> np.uint64(32), p1 & _MASK
        c0, c1, c2, c3 = (hi1 ^ c1 ^ k0) & _MASK, lo1, (hi0 ^ c3 ^ k1) & _MASK, lo0
    return np.stack([c0, c1, c2, c3], axis=-1).astype(np.uint32)


def to_uniform24(x):
    """u = (x >> 8) * 2**-24, exact in fp32."""
    return (np.asarray(x, dtype=np.uint32) >> np.uint32(8)).astype(np.float64) * (2.0 ** -24)


def verify_uniforms(seed: int, offset: int, req: int, n_slots: int):
    """Uniforms u[slot] for one request of one verify step.

    Counter = (slot, request, offset_lo, offset_hi), key = (seed_lo, seed_hi); the first output
    word is mapped by to_uniform24.  Returned as float64 (exact fp32 values).
    """
    slots = np.arange(n_slots, dtype=np.uint64)
    ctr = np.stack([slots,
                    np.full(n_slots, req, np.uint64),
                    np.full(n_slots, offset & _MASK, np.uint64),
                    np.full(n_slots, (offset >> 32) & _MASK, np.uint64)], axis=-1)
    key = np.array([seed & _MASK, (seed >> 32) & _MASK], dtype=np.uint64)
    out = philox4x32_10(ctr, key)
    return to_uniform24(out[:, 0])
