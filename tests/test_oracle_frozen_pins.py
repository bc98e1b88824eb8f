"""Pins of the oracle's frozen-statistics maps (the inference mode that applies the L1BN and
Q_A constants of a calibration batch to later batches; the paper defines no running
estimate, so this is a stated reading of its L1BN at inference).

  * With the constants of the same batch, the frozen L1BN maps reproduce or_bn_fwd's X and A
    codes exactly, and frozen SQ with the batch's own maximum reproduces SQ.
  * On other batches -- including accumulators far beyond the calibration range -- the maps
    equal floor((F acc + B) / 2^P) and floor((G X + H) / 2^P') evaluated with Python's
    unbounded integers, clipped to the code ranges."""
import numpy as np
import pytest

import oracle as O
from paper_2011_14504_gb300 import synthetic as S


def _batch(g, m, c, spread):
    return (g.standard_normal((m, c)) * spread + g.integers(-3000, 3001, c)).astype(np.int32)


@pytest.mark.parametrize("k_a", [8, 4])
def test_frozen_bn_with_own_constants_is_the_forward(k_a):
    g = S.rng(61 + k_a)
    m, c = 700, 48
    acc = _batch(g, m, c, 20000.0)
    gam, bet = S.bn_gamma_beta_codes(g, c)
    r = O.bn_fwd(acc, 2.0 ** -13, gam, bet, k_a=k_a)
    X, A = O.bn_apply_fixed(acc, r.F, r.B, r.G, r.H, r.p_x, r.p_a, 16, k_a)
    assert np.array_equal(X, r.X) and np.array_equal(A, r.A)


def test_frozen_bn_on_other_batches_matches_big_integers():
    g = S.rng(63)
    m, c = 300, 16
    acc0 = _batch(g, m, c, 5000.0)
    gam, bet = S.bn_gamma_beta_codes(g, c)
    r = O.bn_fwd(acc0, 2.0 ** -12, gam, bet)
    # a later batch: shifted, and some accumulators 1000 x beyond the calibration maximum
    acc = _batch(g, m, c, 9000.0)
    acc[::37] = (acc[::37].astype(np.int64) * 1000).clip(-2 ** 31 + 1, 2 ** 31 - 1).astype(np.int32)
    X, A = O.bn_apply_fixed(acc, r.F, r.B, r.G, r.H, r.p_x, r.p_a)
    for i in range(0, m, 7):
        for j in range(c):
            t = int(r.F[j]) * int(acc[i, j]) + int(r.B[j])
            xw = max(-32767, min(32767, t >> r.p_x))          # Python >> is floor division
            u = int(r.G[j]) * xw + int(r.H[j])
            aw = max(0, min(127, u >> r.p_a))
            assert X[i, j] == xw and A[i, j] == aw, (i, j)


def test_frozen_sq_is_sq_with_the_calibration_maximum():
    g = S.rng(64)
    q = g.integers(-10 ** 6, 10 ** 6, 5000)
    for relu in (False, True):
        M = int((np.maximum(q, 0) if relu else np.abs(q)).max())
        full, s_full = O.sq_int(q, 0.5, 8, relu)
        frozen, s_frozen = O.sq_at(q, M, 0.5, 8, relu)
        assert np.array_equal(frozen, full) and s_frozen == s_full
    # values beyond the frozen maximum clip to the top code
    c, _ = O.sq_at(np.array([3 * M, -3 * M, M]), M, 0.5, 8, False)
    assert c.tolist() == [127, -127, 127]
