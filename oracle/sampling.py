"""Sampling and speculative acceptance (oracle; test infrastructure only).

Restates Sec. 3.1 ("Verification"): the verifier's distribution p is compared with the
drafter's q by rejection sampling (Leviathan et al. 2023; Chen et al. 2023): draft x_i is kept
with probability min(1, p_{i-1}(x_i) / q_i(x_i)); at the first rejection a replacement is drawn
from norm(max(0, p - q)); if all k drafts are kept, one more token is drawn from p_k, so a block
yields (accepted + 1) tokens (Sec. 4 "Metrics"). At T = 0 (greedy, Sec. 4 "Decoding
Parameters") a draft is kept iff it is the verifier's argmax, and the emitted token is the argmax.

Readings where the paper is silent (each listed in the design notes):
  * p = softmax(z * (1/T)) with 1/T rounded to fp32 once; both models use the same T.
  * The normaliser is exact: each e_v = exp(s_v - max s) is truncated to a multiple of 2^-45
    and summed as a 64-bit integer (order-free), then rounded once to fp32.
  * Accept iff u * q(x) <= p(x), u from Philox (see philox.py), compared in fp32.
  * Sampling is an exponential race: y = argmax_v w_v / E_v with E_v = -ln u_v, ties to the
    lowest v, entries with w_v = 0 excluded. With w = p this draws from p; in log form
    argmax_v (z_v/T - ln E_v) draws from softmax(z/T) with no normaliser. If the residual is
    zero everywhere (only possible through rounding) the replacement is drawn from p instead.

Pinned in tests/test_oracle_sampling.py: the analytic acceptance reproduces the verifier's
autoregressive distribution exactly (brute force, tiny vocabularies), the sampled acceptance
matches the analytic one (Monte Carlo, chi-square), the acceptance rate equals
sum_v min(p_v, q_v) (Leviathan et al., Thm. 3.5), and races match their target distributions.
"""
from __future__ import annotations

from typing import List, Optional, Sequence, Tuple

import numpy as np

from . import philox
from .fpmath import exp_cw, log_at

F32 = np.float32
FIX_SHIFT = 45          # the normaliser's fixed point: multiples of 2^-45


def inv_temperature(temp: float) -> np.float32:
    """1/T rounded once to fp32 (T > 0)."""
    return F32(1.0) / F32(temp)


def u64_to_f32_nearest_even(x: int) -> np.float32:
    """Round a non-negative integer to the nearest fp32 (ties to even), exactly."""
    x = int(x)
    nb = x.bit_length()
    if nb <= 24:
        return F32(x)
    sh = nb - 24
    q, r = x >> sh, x & ((1 << sh) - 1)
    half = 1 << (sh - 1)
    if r > half or (r == half and (q & 1)):
        q += 1
    return np.ldexp(F32(q), sh).astype(F32)


def softmax_exact_norm(z, inv_t) -> Tuple[np.ndarray, np.ndarray, np.float32]:
    """p = softmax(z * inv_t) in fp32 with the fixed-point normaliser; returns (p, e, S)."""
    s = (np.asarray(z, dtype=F32) * F32(inv_t)).astype(F32)
    t = (s - s.max()).astype(F32)
    e = exp_cw(t)
    fixed = (e * F32(2.0 ** FIX_SHIFT)).astype(F32).astype(np.uint64)   # exact scale, truncation
    total = int(fixed.sum(dtype=np.uint64))
    S = (u64_to_f32_nearest_even(total) * F32(2.0 ** -FIX_SHIFT)).astype(F32)
    p = (e / S).astype(F32)
    return p, e, S


def race_log(z, inv_t, u) -> int:
    """argmax_v (z_v * inv_t - ln(-ln u_v)): a draw from softmax(z * inv_t)."""
    s = (np.asarray(z, dtype=F32) * F32(inv_t)).astype(F32)
    E = (-log_at(u)).astype(F32)
    key = (s - log_at(E)).astype(F32)
    return int(np.argmax(key))


def race_ratio(w, u) -> Optional[int]:
    """argmax_v w_v / (-ln u_v) over w_v > 0: a draw from w / sum(w); None if w == 0 everywhere."""
    w = np.asarray(w, dtype=F32)
    E = (-log_at(u)).astype(F32)
    key = (w / E).astype(F32)
    if not np.any(key > 0):
        return None
    return int(np.argmax(key))


def argmax(z) -> int:
    """Greedy choice: the largest logit, ties to the lowest index."""
    return int(np.argmax(np.asarray(z, dtype=F32)))


def sample_draft(z, temp: float, seed: int, b: int, step: int, i: int) -> int:
    """Draft token i (1-based) of sequence b: argmax at T = 0, else a race on softmax(z/T)."""
    if temp == 0.0:
        return argmax(z)
    u = philox.vocab_uniforms(seed, philox.DRAFT, i, b, step, len(z))
    return race_log(z, inv_temperature(temp), u)


def sample_from_target(z, temp: float, seed: int, b: int, step: int, row: int) -> int:
    """A token from the verifier's row (bonus token, or the first token after the prompt)."""
    if temp == 0.0:
        return argmax(z)
    u = philox.vocab_uniforms(seed, philox.RESAMPLE, row, b, step, len(z))
    return race_log(z, inv_temperature(temp), u)


def accept_block(target, draft, xhat: Sequence[int], temp: float, seed: int, b: int,
                 step: int) -> Tuple[List[int], int]:
    """Speculative acceptance of one block (Sec. 3.1).

    target: [k+1, V] verifier logits; row i is the distribution of the token after the i-th
            block input (row 0 follows the last committed token, row i follows draft i).
    draft:  [k, V] drafter logits; row i-1 is q_i, the distribution draft i was sampled from.
    Returns (emitted tokens, j): the j accepted drafts followed by one verifier token.
    """
    target = np.asarray(target, dtype=F32)
    draft = np.asarray(draft, dtype=F32)
    k = len(xhat)
    V = target.shape[-1]
    if temp == 0.0:
        for i in range(1, k + 1):
            if int(xhat[i - 1]) != argmax(target[i - 1]):
                return [int(x) for x in xhat[:i - 1]] + [argmax(target[i - 1])], i - 1
        return [int(x) for x in xhat] + [argmax(target[k])], k
    inv_t = inv_temperature(temp)
    for i in range(1, k + 1):
        x = int(xhat[i - 1])
        p, _, _ = softmax_exact_norm(target[i - 1], inv_t)
        q, _, _ = softmax_exact_norm(draft[i - 1], inv_t)
        u = philox.accept_uniform(seed, i, b, step)
        if F32(u * q[x]) <= p[x]:
            continue
        j = i - 1
        resid = np.maximum((p - q).astype(F32), F32(0.0))
        uv = philox.vocab_uniforms(seed, philox.RESAMPLE, j, b, step, V)
        y = race_ratio(resid, uv)
        if y is None:
            y = race_log(target[j], inv_t, uv)
        return [int(x) for x in xhat[:j]] + [y], j
    uv = philox.vocab_uniforms(seed, philox.RESAMPLE, k, b, step, V)
    return [int(x) for x in xhat] + [race_log(target[k], inv_t, uv)], k


# ---------------------------------------------------------------------------------------------
# Analytic (fp64) form of the same rules, used to pin the sampled form above.
# ---------------------------------------------------------------------------------------------

def accept_probability(p, q, x: int) -> float:
    """Probability that draft x is kept: min(1, p(x)/q(x)) (Sec. 3.1)."""
    return 1.0 if q[x] <= p[x] else float(p[x]) / float(q[x])


def residual_distribution(p, q) -> np.ndarray:
    """norm(max(0, p - q)); p itself when the residual vanishes."""
    r = np.maximum(np.asarray(p, np.float64) - np.asarray(q, np.float64), 0.0)
    s = r.sum()
    return np.asarray(p, np.float64) if s <= 0 else r / s


def block_outcomes(p_rows, q_rows, xhat: Sequence[int]):
    """All outcomes of accepting one fixed draft block, with their probabilities.

    p_rows: k+1 target distributions, q_rows: k draft distributions (fp64 arrays).
    Returns a list of (emitted token tuple, probability).
    """
    k = len(xhat)
    out = []
    alive = 1.0
    for i in range(1, k + 1):
        a = accept_probability(p_rows[i - 1], q_rows[i - 1], xhat[i - 1])
        rej = alive * (1.0 - a)
        if rej > 0:
            r = residual_distribution(p_rows[i - 1], q_rows[i - 1])
            for y, py in enumerate(r):
                if py > 0:
                    out.append((tuple(int(x) for x in xhat[:i - 1]) + (y,), rej * py))
        alive *= a
    if alive > 0:
        for y, py in enumerate(np.asarray(p_rows[k], np.float64)):
            if py > 0:
                out.append((tuple(int(x) for x in xhat) + (y,), alive * py))
    return out
