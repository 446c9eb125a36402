"""Philox4x32-10 and the uniforms SD^2 draws from it (oracle; test infrastructure only).

Philox4x32 is the counter-based generator of Salmon, Moraes, Dror and Shaw, "Parallel
random numbers: as easy as 1, 2, 3" (SC'11): a 4x32-bit counter is encrypted under a 2x32-bit
key by 10 rounds of multiply-high/low mixing with a Weyl-sequence key schedule. Written here
from that definition. Pinned by the published known-answer vectors (tests/golden/philox_kat.txt).

Counter layout used by the SD^2 path (the paper fixes none; every random draw of the method
is named by what it is for):
  key     = (seed mod 2^32, seed >> 32)
  counter = (c0, purpose << 16 | i, b, step)
    c0      = v >> 2 for a draw per vocabulary entry v (word v & 3 of the output), else 0
    purpose = DRAFT (sample draft token i), ACCEPT (uniform for draft i), RESAMPLE (residual /
              bonus / prefill sample from block row i)
    b       = sequence index in the batch, step = iteration index (0 = prefill)
Uniform from a 32-bit word x: u = (2*(x >> 9) + 1) * 2^-24, an odd multiple of 2^-24 in (0,1),
exact in fp32.
"""
from __future__ import annotations

import numpy as np

MUL0 = 0xD2511F53
MUL1 = 0xCD9E8D57
WEYL0 = 0x9E3779B9
WEYL1 = 0xBB67AE85
MASK32 = 0xFFFFFFFF

DRAFT = 0
ACCEPT = 1
RESAMPLE = 2


def philox4x32_10(counters, key) -> np.ndarray:
    """Encrypt counters [N,4] (uint32) under key (k0, k1); returns [N,4] uint32."""
    c = np.asarray(counters, dtype=np.uint64).reshape(-1, 4) & MASK32
    x0, x1, x2, x3 = (c[:, j].copy() for j in range(4))
    k0, k1 = int(key[0]) & MASK32, int(key[1]) & MASK32
    for rnd in range(10):
        if rnd:  # key schedule: add the Weyl constants before every round but the first
            k0 = (k0 + WEYL0) & MASK32
            k1 = (k1 + WEYL1) & MASK32
        p0 = x0 * np.uint64(MUL0)          # 32x32 -> 64-bit product, exact in uint64
        p1 = x2 * np.uint64(MUL1)
        hi0, lo0 = p0 >> np.uint64(32), p0 & np.uint64(MASK32)
        hi1, lo1 = p1 >> np.uint64(32), p1 & np.uint64(MASK32)
        x0, x1, x2, x3 = hi1 ^ x1 ^ np.uint64(k0), lo1, hi0 ^ x3 ^ np.uint64(k1), lo0
    return np.stack([x0, x1, x2, x3], axis=1).astype(np.uint32)


def seed_key(seed: int):
    seed = int(seed) & 0xFFFFFFFFFFFFFFFF
    return (seed & MASK32, seed >> 32)


def bits_to_uniform(x) -> np.ndarray:
    """u = (2*(x >> 9) + 1) * 2^-24 in fp32 (exact)."""
    x = np.asarray(x, dtype=np.uint32)
    odd = (x >> np.uint32(9)).astype(np.uint32) * np.uint32(2) + np.uint32(1)
    return odd.astype(np.float32) * np.float32(2.0 ** -24)


def vocab_uniforms(seed: int, purpose: int, i: int, b: int, step: int, vocab: int) -> np.ndarray:
    """One uniform per vocabulary entry v in [0, vocab), from counter (v>>2, purpose<<16|i, b, step)."""
    n4 = (vocab + 3) // 4
    ctr = np.zeros((n4, 4), dtype=np.uint64)
    ctr[:, 0] = np.arange(n4, dtype=np.uint64)
    ctr[:, 1] = (purpose << 16) | i
    ctr[:, 2] = b
    ctr[:, 3] = step
    words = philox4x32_10(ctr, seed_key(seed)).reshape(-1)[:vocab]
    return bits_to_uniform(words)


def accept_uniform(seed: int, i: int, b: int, step: int) -> np.float32:
    """The uniform u_i of the acceptance test for draft i: word 0 of counter (0, ACCEPT<<16|i, b, step)."""
    ctr = np.array([[0, (ACCEPT << 16) | i, b, step]], dtype=np.uint64)
    return bits_to_uniform(philox4x32_10(ctr, seed_key(seed))[0, 0])
