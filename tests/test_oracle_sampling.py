"""Pins for the oracle's sampling and speculative acceptance (CPU only).

O1: the analytic acceptance rule reproduces the verifier's autoregressive distribution exactly
    (brute-force enumeration on tiny vocabularies, fp64), across block boundaries.
O6: the acceptance rate equals sum_v min(p_v, q_v) (Leviathan et al. 2023, Thm. 3.5; the paper's
    Sec. 3.3 cites the equivalence of total-variation distance and rejection rate).
The sampled fp32/Philox form is checked against the analytic form by Monte Carlo (chi-square).
"""
import itertools
import math
from collections import Counter, defaultdict

import numpy as np
import pytest
from scipy import stats

from oracle import philox, sampling


def _toy_tables(V, seed):
    """Context-dependent toy distributions p(.|prefix), q(.|prefix) (fp64), some zeros allowed."""
    cache = {}

    def dist(which, prefix):
        key = (which, tuple(prefix))
        if key not in cache:
            h = hash((seed, 0 if which == "p" else 1) + tuple(prefix)) & 0xFFFFFFFF
            rng = np.random.default_rng(h)
            w = rng.gamma(0.7, size=V)
            if rng.random() < 0.3:
                w[rng.integers(V)] = 0.0          # a zero-probability entry
            cache[key] = w / w.sum()
        return cache[key]

    return (lambda pre: dist("p", pre)), (lambda pre: dist("q", pre))


def _sd_output_distribution(p, q, V, k, m, prefix=()):
    """Exact distribution of the next m emitted tokens of chain SD (draft k, then accept)."""
    if m == 0:
        return {(): 1.0}
    out = defaultdict(float)
    for xhat in itertools.product(range(V), repeat=k):
        pd = 1.0
        for i in range(k):
            pd *= q(prefix + xhat[:i])[xhat[i]]
        if pd == 0.0:
            continue
        p_rows = [p(prefix + xhat[:i]) for i in range(k + 1)]
        q_rows = [q(prefix + xhat[:i]) for i in range(k)]
        for emitted, pr in sampling.block_outcomes(p_rows, q_rows, xhat):
            if len(emitted) >= m:
                out[emitted[:m]] += pd * pr
            else:
                rest = _sd_output_distribution(p, q, V, k, m - len(emitted), prefix + emitted)
                for r, prr in rest.items():
                    out[emitted + r] += pd * pr * prr
    return out


def _ar_distribution(p, V, m, prefix=()):
    out = {}
    for ys in itertools.product(range(V), repeat=m):
        pr = 1.0
        for i in range(m):
            pr *= p(prefix + ys[:i])[ys[i]]
        out[ys] = pr
    return out


@pytest.mark.parametrize("V,k,m,seed", [(3, 1, 3, 0), (3, 2, 3, 1), (3, 3, 4, 2), (5, 1, 2, 3),
                                        (5, 2, 3, 4), (2, 3, 5, 5)])
def test_losslessness_bruteforce(V, k, m, seed):
    p, q = _toy_tables(V, seed)
    sd = _sd_output_distribution(p, q, V, k, m)
    ar = _ar_distribution(p, V, m)
    assert abs(sum(sd.values()) - 1.0) < 1e-12
    for ys, pr in ar.items():
        assert abs(sd.get(ys, 0.0) - pr) < 1e-12, (ys, sd.get(ys, 0.0), pr)


def test_bruteforce_detects_a_wrong_rule():
    """The enumeration is sensitive: accepting with min(1, q/p) instead breaks losslessness."""
    V, k, m = 3, 2, 2
    p, q = _toy_tables(V, 11)
    orig = sampling.accept_probability
    try:
        sampling.accept_probability = lambda pp, qq, x: 1.0 if pp[x] <= qq[x] else qq[x] / pp[x]
        sd = _sd_output_distribution(p, q, V, k, m)
    finally:
        sampling.accept_probability = orig
    ar = _ar_distribution(p, V, m)
    assert max(abs(sd.get(y, 0.0) - pr) for y, pr in ar.items()) > 1e-3


def test_softmax_exact_norm_matches_fp64():
    rng = np.random.default_rng(0)
    for V, scale, inv_t in [(4096, 1.0, 1.0), (32000, 3.0, 1.0), (1000, 5.0, 1 / 0.7)]:
        z = (rng.standard_normal(V) * scale).astype(np.float32)
        p, e, S = sampling.softmax_exact_norm(z, sampling.inv_temperature(1 / inv_t))
        s32 = (z * sampling.inv_temperature(1 / inv_t)).astype(np.float32)
        t32 = (s32 - s32.max()).astype(np.float32)
        # normaliser and exp against the exact exp of the same fp32 exponents
        ref = np.exp(t32.astype(np.float64))
        ref /= ref.sum()
        assert np.max(np.abs(p - ref) / ref) < 4e-7
        # end to end against fp64 softmax: bounded by the rounding of the exponent itself
        s = z.astype(np.float64) * float(sampling.inv_temperature(1 / inv_t))
        ref64 = np.exp(s - s.max())
        ref64 /= ref64.sum()
        bound = (np.abs(s) + np.abs(s).max() + 8) * 2.0 ** -24
        assert np.all(np.abs(p - ref64) / ref64 < bound)
        assert abs(p.astype(np.float64).sum() - 1.0) < 1e-5
        assert np.max(e) == 1.0


def test_u64_to_f32_rounding():
    for x in [0, 1, 2 ** 24 - 1, 2 ** 24 + 1, 2 ** 24 + 3, 2 ** 45 + 2 ** 21, 2 ** 62 + 12345,
              (2 ** 24 + 1) << 20, ((2 ** 24 + 1) << 20) + (1 << 19), ((2 ** 24 + 1) << 20) + (1 << 19) + 1]:
        f = sampling.u64_to_f32_nearest_even(x)
        # nearest-even: no other fp32 is closer, ties go to the even significand
        lo, hi = np.nextafter(f, np.float32(0)), np.nextafter(f, np.float32(np.inf))
        d = abs(int(f) - x)
        assert d <= abs(int(lo) - x) and d <= abs(int(hi) - x)


def _chi2_ok(counts, probs, n):
    probs = np.asarray(probs, np.float64)
    keep = probs * n >= 5
    obs = np.array([counts.get(i, 0) for i in range(len(probs))], np.float64)
    o = np.append(obs[keep], obs[~keep].sum())
    e = np.append(probs[keep] * n, probs[~keep].sum() * n)
    assert o[e == 0].sum() == 0, "draws where the target probability is zero"
    o, e = o[e > 0], e[e > 0]
    e = e * (o.sum() / e.sum())
    return stats.chisquare(o, e).pvalue > 1e-3


def test_race_log_draws_softmax():
    rng = np.random.default_rng(1)
    V = 12
    z = (rng.standard_normal(V) * 1.5).astype(np.float32)
    inv_t = sampling.inv_temperature(0.7)
    s = z.astype(np.float64) * float(inv_t)
    target = np.exp(s - s.max())
    target /= target.sum()
    n = 20000
    cnt = Counter(sampling.race_log(z, inv_t, philox.vocab_uniforms(5, 0, 1, b, 0, V)) for b in range(n))
    assert _chi2_ok(cnt, target, n)


def test_race_ratio_draws_weights_and_skips_zeros():
    w = np.array([0.0, 0.1, 0.0, 0.4, 0.2, 0.3], np.float32)
    n = 20000
    cnt = Counter(sampling.race_ratio(w, philox.vocab_uniforms(6, 2, 0, b, 1, 6)) for b in range(n))
    assert cnt[0] == 0 and cnt[2] == 0
    assert _chi2_ok(cnt, w / w.sum(), n)
    assert sampling.race_ratio(np.zeros(6, np.float32), philox.vocab_uniforms(6, 2, 0, 0, 1, 6)) is None


def test_greedy_acceptance():
    V, k = 10, 4
    target = np.zeros((k + 1, V), np.float32)
    for i, a in enumerate([3, 1, 4, 1, 5]):
        target[i, a] = 1.0
    draft = np.zeros((k, V), np.float32)
    assert sampling.accept_block(target, draft, [3, 1, 4, 1], 0.0, 0, 0, 1) == ([3, 1, 4, 1, 5], 4)
    assert sampling.accept_block(target, draft, [3, 1, 7, 1], 0.0, 0, 0, 1) == ([3, 1, 4], 2)
    assert sampling.accept_block(target, draft, [0, 1, 4, 1], 0.0, 0, 0, 1) == ([3], 0)
    target[2, 9] = 1.0      # tie between 4 and 9 -> lowest index 4
    assert sampling.accept_block(target, draft, [3, 1, 4, 1], 0.0, 0, 0, 1)[1] == 4


def _sampled_block_distribution(target, draft, xhat, temp, n, b0=0):
    cnt = Counter()
    for t in range(n):
        emitted, _ = sampling.accept_block(target, draft, xhat, temp, 77, b0 + t % 97, 1 + t // 97)
        cnt[tuple(emitted)] += 1
    return cnt


def test_sampled_acceptance_matches_analytic():
    """Monte Carlo: fp32/Philox acceptance of a fixed block vs the analytic outcome distribution."""
    rng = np.random.default_rng(3)
    V, k, T = 5, 2, 1.0
    target = rng.standard_normal((k + 1, V)).astype(np.float32)
    draft = rng.standard_normal((k, V)).astype(np.float32)
    xhat = [1, 3]
    p_rows = [sampling.softmax_exact_norm(r, 1.0)[0].astype(np.float64) for r in target]
    q_rows = [sampling.softmax_exact_norm(r, 1.0)[0].astype(np.float64) for r in draft]
    analytic = dict(sampling.block_outcomes(p_rows, q_rows, xhat))
    keys = sorted(analytic)
    n = 20000
    cnt = _sampled_block_distribution(target, draft, xhat, T, n)
    assert set(cnt) <= set(keys)
    idx = {kk: i for i, kk in enumerate(keys)}
    assert _chi2_ok({idx[kk]: c for kk, c in cnt.items()}, [analytic[kk] for kk in keys], n)


def test_acceptance_rate_is_overlap():
    """O6: a draft sampled from q is accepted with probability sum_v min(p_v, q_v)."""
    rng = np.random.default_rng(4)
    V = 40
    zt = (rng.standard_normal(V) * 2).astype(np.float32)
    zd = (rng.standard_normal(V) * 2).astype(np.float32)
    p = sampling.softmax_exact_norm(zt, 1.0)[0].astype(np.float64)
    q = sampling.softmax_exact_norm(zd, 1.0)[0].astype(np.float64)
    alpha = np.minimum(p, q).sum()
    n, acc = 20000, 0
    for t in range(n):
        b, step = t % 101, 1 + t // 101
        x = sampling.sample_draft(zd, 1.0, 9, b, step, 1)
        _, j = sampling.accept_block(np.stack([zt, zt]), zd[None], [x], 1.0, 9, b, step)
        acc += j
    sigma = math.sqrt(alpha * (1 - alpha) / n)
    assert abs(acc / n - alpha) < 4.5 * sigma
