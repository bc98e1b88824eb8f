"""Pins of the oracle's per-channel Scale variant (Eqs. (ScaleFactor), (ScaleQ) with the
maximum taken over each channel's elements instead of the whole tensor).

The variant is pinned to properties it must have whatever its arithmetic:
  * with one channel it is the per-tensor SQ (itself pinned to exact rationals);
  * every channel's codes and scale are the per-tensor SQ of that channel's elements alone;
  * multiplying one channel by a positive integer leaves every code unchanged (the ratio
    q / Scale does not move) and multiplies that channel's scale only;
  * codes are monotone in q within a channel, and a channel's largest |q| takes the top code.
"""
import numpy as np
import pytest

import oracle as O


def _tensor(g, outer, C, inner, hi):
    return g.integers(-hi, hi + 1, size=(outer, C, inner), dtype=np.int64)


@pytest.mark.parametrize("k", [4, 8, 16])
@pytest.mark.parametrize("relu", [False, True])
def test_single_channel_is_per_tensor_sq(k, relu):
    g = np.random.default_rng(11 + k)
    q = _tensor(g, 7, 1, 9, 5000)
    codes, sc = O.sq_per_channel(q, 7, 1, 9, 0.37, k, relu)
    want, s = O.sq_int(q, 0.37, k, relu)
    assert np.array_equal(codes, want)
    assert sc[0] == s


@pytest.mark.parametrize("shape", [(5, 6, 1), (2, 3, 17), (1, 8, 40), (4, 1, 4)])
@pytest.mark.parametrize("relu", [False, True])
def test_each_channel_is_sq_of_its_slice(shape, relu):
    outer, C, inner = shape
    g = np.random.default_rng(sum(shape) + relu)
    q = _tensor(g, outer, C, inner, 1 << 20)
    q[:, C // 2, :] = 0                            # an all-zero channel
    codes, sc = O.sq_per_channel(q, outer, C, inner, 2.0 ** -9, 8, relu)
    for c in range(C):
        want, s = O.sq_int(q[:, c, :], 2.0 ** -9, 8, relu)
        assert np.array_equal(codes[:, c, :], want), c
        assert sc[c] == s, c


def test_channel_scaling_leaves_codes():
    g = np.random.default_rng(5)
    outer, C, inner = 6, 5, 7
    q = _tensor(g, outer, C, inner, 3000)
    codes, sc = O.sq_per_channel(q, outer, C, inner, 1.0, 8)
    t = np.array([1, 3, 7, 1, 1000], dtype=np.int64)
    q2 = q * t[None, :, None]
    codes2, sc2 = O.sq_per_channel(q2, outer, C, inner, 1.0, 8)
    assert np.array_equal(codes, codes2)
    assert np.array_equal(sc2, sc * t)


@pytest.mark.parametrize("k", [4, 8])
def test_monotone_and_top_code(k):
    g = np.random.default_rng(23)
    outer, C, inner = 3, 4, 50
    q = _tensor(g, outer, C, inner, 10 ** 6)
    codes, _ = O.sq_per_channel(q, outer, C, inner, 1.0, k)
    top = (1 << (k - 1)) - 1
    for c in range(C):
        v = q[:, c, :].ravel()
        cc = codes[:, c, :].ravel()
        order = np.argsort(v, kind="stable")
        assert np.all(np.diff(cc[order]) >= 0)
        i = np.argmax(np.abs(v))
        assert abs(int(cc[i])) == top
        assert np.abs(cc).max() <= top


# ---------------------------------------------------------------- weight decay
# The decoupled decay step m - rhu(m / 2^shift) is pinned to: the closed form on exact
# multiples m = t 2^shift (m -> t (2^shift - 1)); no growth and no change of sign for any m;
# the rounding tie m / 2^shift = j + 1/2 going to j + 1 (half up, also for negative m); and
# W_q as the plain UQ of the new masters (Eq. (WQ1), pinned elsewhere).

@pytest.mark.parametrize("shift", [1, 5, 17])
def test_weight_decay_closed_form_and_monotone(shift):
    g = np.random.default_rng(shift)
    t = g.integers(-(1 << (23 - min(shift, 22))), 1 << (23 - min(shift, 22)), size=500)
    m = (t << shift).astype(np.int64)
    m = m[np.abs(m) < (1 << 23)].astype(np.int32)
    m2, _ = O.weight_decay(m, shift)
    assert np.array_equal(m2.astype(np.int64), (m.astype(np.int64) >> shift) * ((1 << shift) - 1))
    r = g.integers(-(1 << 23) + 1, 1 << 23, size=5000).astype(np.int32)
    r2, wq = O.weight_decay(r, shift)
    assert np.all(np.abs(r2.astype(np.int64)) <= np.abs(r.astype(np.int64)))
    assert np.all((np.sign(r2) == np.sign(r)) | (r2 == 0))
    assert np.array_equal(wq, O.requant_master(r2, 24, 8))


def test_weight_decay_ties_round_half_up():
    shift = 4
    m = np.array([8, 24, -8, -24, 7, -7, 9, -9], dtype=np.int32)      # m / 16 = +-0.5, +-1.5
    m2, _ = O.weight_decay(m, shift)
    # rhu(0.5) = 1, rhu(1.5) = 2, rhu(-0.5) = 0, rhu(-1.5) = -1; +-7/16 round to 0, 9/16 to 1,
    # -9/16 to -1
    assert m2.tolist() == [7, 22, -8, -23, 7, -7, 8, -8]
