"""exp and log as fixed sequences of correctly rounded fp32 operations (oracle; test only).

The sampling and acceptance decisions of SD^2 are integers (a token id, accept/reject) decided
by floating point. So that the oracle and the GPU take every such decision identically, both
evaluate the transcendental functions by the same published methods, using only operations
IEEE 754 rounds correctly (fp32 multiply, add, subtract, divide, round-to-integer, exact
power-of-two scaling) in a fixed order with no fused multiply-add. numpy's float32 array
arithmetic is exactly that.

exp_cw: Cody & Waite argument reduction (Cody and Waite, "Software Manual for the
  Elementary Functions", 1980): n = rint(t / ln 2), r = t - n*ln2_hi - n*ln2_lo with ln 2
  split so that n*ln2_hi is exact, then the degree-7 Taylor polynomial of e^r (coefficients
  1/j! rounded to fp32) in Horner form, then scaling by 2^n. Inputs below -80 return 0.
log_at: x = 2^e * m with m in [sqrt(1/2), sqrt(2)); ln m = 2 atanh(s), s = (m-1)/(m+1),
  by the odd series 2(s + s^3/3 + ... + s^11/11) (Abramowitz & Stegun 4.1.27); then
  ln x = e*ln2_hi + (e*ln2_lo + ln m).

Pinned against numpy's float64 exp/log (error bound in ulps) in tests/test_oracle_fpmath.py.
"""
from __future__ import annotations

import numpy as np

F32 = np.float32
_h = float.fromhex

LOG2E = F32(_h("0x1.715476p+0"))     # fp32 nearest 1/ln 2
LN2_HI = F32(_h("0x1.62e400p-1"))    # ln 2 with the low 8 significand bits cleared
LN2_LO = F32(_h("0x1.7f7d1cp-20"))   # fp32 nearest (ln 2 - LN2_HI)
SQRT2 = F32(_h("0x1.6a09e6p+0"))     # fp32 nearest sqrt 2
EXP_CUTOFF = F32(-80.0)

# 1/j!, j = 7..0, fp32 nearest
EXP_COEF = [F32(_h(x)) for x in ("0x1.a01a02p-13", "0x1.6c16c2p-10", "0x1.111112p-7",
                                 "0x1.555556p-5", "0x1.555556p-3", "0x1p-1", "0x1p+0", "0x1p+0")]
# 1/j, j = 11, 9, 7, 5, 3, fp32 nearest
LOG_COEF = [F32(_h(x)) for x in ("0x1.745d18p-4", "0x1.c71c72p-4", "0x1.24924ap-3",
                                 "0x1.99999ap-3", "0x1.555556p-2")]


def exp_cw(t) -> np.ndarray:
    """e^t for fp32 t <= ~0 (Cody-Waite reduction + degree-7 Taylor); t < -80 gives 0."""
    t = np.asarray(t, dtype=F32)
    with np.errstate(over="ignore", invalid="ignore"):
        return _exp_cw(t)


def _exp_cw(t):
    n = np.rint(t * LOG2E).astype(F32)
    r = (t - n * LN2_HI).astype(F32)
    r = (r - n * LN2_LO).astype(F32)
    p = np.full_like(r, EXP_COEF[0])
    for c in EXP_COEF[1:]:
        p = (p * r).astype(F32)
        p = (p + c).astype(F32)
    out = np.ldexp(p, np.where(t < EXP_CUTOFF, 0, n).astype(np.int32)).astype(F32)
    return np.where(t < EXP_CUTOFF, F32(0.0), out).astype(F32)


def log_at(x) -> np.ndarray:
    """ln x for positive normal fp32 x (atanh series on the reduced significand)."""
    x = np.asarray(x, dtype=F32)
    bits = x.view(np.uint32)
    e = (bits >> np.uint32(23)).astype(np.int32) - 127
    m = ((bits & np.uint32(0x7FFFFF)) | np.uint32(0x3F800000)).view(F32)
    big = m > SQRT2
    m = np.where(big, (m * F32(0.5)).astype(F32), m)
    e = np.where(big, e + 1, e)
    s = ((m - F32(1.0)).astype(F32) / (m + F32(1.0)).astype(F32)).astype(F32)
    s2 = (s * s).astype(F32)
    q = np.full_like(s, LOG_COEF[0])
    for c in LOG_COEF[1:]:
        q = (q * s2).astype(F32)
        q = (q + c).astype(F32)
    two_s = (s * F32(2.0)).astype(F32)
    ln_m = (two_s + (two_s * (s2 * q).astype(F32)).astype(F32)).astype(F32)
    ef = e.astype(F32)
    return ((ef * LN2_HI).astype(F32) + ((ef * LN2_LO).astype(F32) + ln_m).astype(F32)).astype(F32)
