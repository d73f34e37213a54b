"""The lane draft kernel forms the temporal-encoding angle a_j + b_j t and
reduces it mod 2 pi in fp32-pair arithmetic instead of fp64.  This CPU test
takes the constants that kernel uses (read from its source), checks them
against 2 pi, and runs the same float32 steps in numpy (two-sum, fast
two-sum, FMA-exact products, k * 2 pi removed as a pair) against the angle
formed and reduced in fp64, over the frequency ranges of the THP, SAHP and
AttNHP encodings (App. D.4) and times up to 10^4.  The reduced fp32 angle
must lie within a few fp32 ulps of the fp64 one."""
import os
import re

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
f32 = np.float32


def _constants():
    src = open(os.path.join(ROOT, "paper_2507_09252_gb300", "csrc", "draft.cu")).read()
    m = re.search(r"P_HI = ([0-9.eE+-]+)f, P_LO = ([0-9.eE+-]+)f, INV = ([0-9.eE+-]+)f", src)
    assert m, "constants of reduced_angle not found"
    return tuple(f32(float(g)) for g in m.groups())


def _fma(a, b, c):
    # exact product of two floats fits a double; one rounding to float32 after the add
    return (a.astype(np.float64) * b.astype(np.float64) + c.astype(np.float64)).astype(f32)


def _two_sum(a, b):
    s = a + b
    bb = s - a
    return s, (a - (s - bb)) + (b - bb)


def _fast_two_sum(a, b):
    s = a + b
    return s, b - (s - a)


def _split(x):
    hi = x.astype(f32)
    return hi, (x - hi.astype(np.float64)).astype(f32)


def _pair_angle(a, b, t, P_HI, P_LO, INV):
    (ah, al), (bh, bl), (th, tl) = _split(a), _split(b), _split(t)
    p = bh * th
    e = _fma(bh, th, -p)
    e = _fma(bh, tl, e)
    e = _fma(bl, th, e)
    s, sl = _two_sum(ah, p)
    ang_h, ang_l = _fast_two_sum(s, sl + (e + al))
    k = np.rint(ang_h * INV).astype(f32)
    q = k * P_HI
    qe = _fma(k, np.full_like(k, P_HI), -q)
    r = ang_h - q
    r = r - qe
    r = r + ang_l
    return _fma(-k, np.full_like(k, P_LO), r)


def test_constants_are_two_pi():
    P_HI, P_LO, INV = _constants()
    two_pi = 2.0 * np.pi
    assert P_HI == f32(two_pi)
    assert P_LO == f32(two_pi - float(P_HI))
    assert abs(float(P_HI) + float(P_LO) - two_pi) < 1e-14
    assert INV == f32(1.0 / two_pi)


def test_pair_reduction_matches_fp64():
    P_HI, P_LO, INV = _constants()
    rng = np.random.default_rng(3)
    d = 32
    je = np.arange(d) - (np.arange(d) & 1)
    thp_b = 10000.0 ** (-je / d)
    sahp_a = np.arange(d) / 10000.0 ** (je / d)
    sahp_b = rng.normal(0.0, 0.5, d)
    att_b = 1.0 / (0.1 * (5.0 * 1000.0 / 0.1) ** (je / d))
    n = 4000
    t = np.concatenate([rng.uniform(0.0, 1e4, n), rng.exponential(5.0, n)])
    worst = 0.0
    for a, b in ((np.zeros(d), thp_b), (sahp_a, sahp_b), (np.zeros(d), att_b)):
        A = np.broadcast_to(a, (t.size, d)).ravel()
        Bv = np.broadcast_to(b, (t.size, d)).ravel()
        T = np.repeat(t, d)
        ang = A + Bv * T
        ref = ang - 2.0 * np.pi * np.rint(ang / (2.0 * np.pi))
        got = _pair_angle(A, Bv, T, P_HI, P_LO, INV).astype(np.float64)
        diff = np.angle(np.exp(1j * (got - ref)))  # wrapped to (-pi, pi]
        worst = max(worst, float(np.abs(diff).max()))
        # k = rint(angle / 2 pi) is rounded in float32, so near a half turn the
        # remainder may pass pi by a little (still the right angle mod 2 pi)
        assert np.abs(got).max() <= np.pi + 1e-2
    # a float32 angle near pi is within 1.2e-7 of any real one; the pair
    # arithmetic adds well under that
    assert worst < 4e-7, worst
