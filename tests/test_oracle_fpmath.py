"""Pins for the oracle's Philox generator and its exp/log methods (CPU only)."""
import numpy as np
import pytest

from conftest import golden_rows
from oracle import philox
from oracle.fpmath import exp_cw, log_at


def test_philox_known_answers():
    rows = golden_rows("philox_kat.txt")
    assert len(rows) == 3
    for r in rows:
        v = [int(x, 16) for x in r]
        out = philox.philox4x32_10([v[0:4]], v[4:6])[0]
        assert [int(x) for x in out] == v[6:10]


def test_philox_vectorised_matches_single():
    ctr = np.array([[i, 7, 3, 11] for i in range(16)], dtype=np.uint64)
    many = philox.philox4x32_10(ctr, (123, 456))
    for i in range(16):
        one = philox.philox4x32_10(ctr[i:i + 1], (123, 456))
        assert np.array_equal(many[i], one[0])


def test_uniform_range_and_grid():
    x = np.array([0, 1, 511, 512, 0xFFFFFFFF, 0x80000000], dtype=np.uint32)
    u = philox.bits_to_uniform(x)
    assert u.dtype == np.float32
    assert np.all(u > 0) and np.all(u < 1)
    assert u[0] == np.float32(2.0 ** -24) and u[2] == u[0]
    assert u[3] == np.float32(3 * 2.0 ** -24)
    assert u[4] == np.float32(1 - 2.0 ** -24)
    # every value is an odd multiple of 2^-24
    k = (u.astype(np.float64) * 2 ** 24)
    assert np.all(k == np.round(k)) and np.all(k.astype(np.int64) % 2 == 1)


def test_vocab_uniforms_layout():
    # entry v comes from word v & 3 of counter (v >> 2, purpose << 16 | i, b, step)
    u = philox.vocab_uniforms(99, philox.RESAMPLE, 3, 5, 17, 10)
    for v in (0, 3, 4, 9):
        w = philox.philox4x32_10([[v >> 2, (philox.RESAMPLE << 16) | 3, 5, 17]], philox.seed_key(99))
        assert u[v] == philox.bits_to_uniform(w[0, v & 3])
    # uniform over (0,1): mean and spread of many draws
    big = philox.vocab_uniforms(1, 0, 1, 0, 0, 200000)
    assert abs(big.mean() - 0.5) < 0.005 and abs(big.var() - 1 / 12) < 0.002


def _ulps(approx, exact64):
    ulp = np.spacing(np.abs(exact64).astype(np.float32)).astype(np.float64)
    return np.abs(approx.astype(np.float64) - exact64) / ulp


def test_exp_cw_accuracy():
    t = np.concatenate([np.linspace(-80, 0, 400001), -np.logspace(-12, 1.9, 20001), [0.0]]).astype(np.float32)
    e = exp_cw(t)
    assert e.dtype == np.float32
    assert _ulps(e, np.exp(t.astype(np.float64))).max() <= 1.5
    assert exp_cw(np.float32(0.0)) == np.float32(1.0)          # the row maximum contributes exactly 1
    assert np.all(exp_cw(np.array([-80.5, -200.0, -1e30], np.float32)) == 0)
    assert np.all(np.diff(exp_cw(np.linspace(-30, 0, 10001).astype(np.float32))) >= 0)  # monotone


def test_log_at_accuracy():
    x = np.concatenate([np.linspace(1e-7, 1, 300001), np.linspace(1, 40, 300001),
                        np.logspace(-30, 30, 20001)]).astype(np.float32)
    l = log_at(x)
    ref = np.log(x.astype(np.float64))
    nz = ref != 0
    assert _ulps(l[nz], ref[nz]).max() <= 2.5
    assert log_at(np.float32(1.0)) == 0
    # the uniforms of the method: -ln u > 0 for every grid point, including the largest
    u = philox.bits_to_uniform(np.array([0, 0xFFFFFFFF], np.uint32))
    assert np.all(-log_at(u) > 0)
