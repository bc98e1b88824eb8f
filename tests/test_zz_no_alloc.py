"""The allocation-free integer-BN forward (iq_bn_int_fwd_noalloc) against the workspace
version (iq_bn_int_fwd), through the C ABI, on two calls in a row.

It exists for callers that cannot allocate device memory themselves; its scratch is a
file-scope device array shared by all calls.  Both entry points run the same integer
computation, so their outputs must be identical.  This file is collected last so that a
run stopping at the first failure has run every other test before it.
"""
import numpy as np
import pytest
import torch

from paper_2011_14504_gb300 import iq
from paper_2011_14504_gb300 import synthetic as S

pytestmark = pytest.mark.gpu

DEV = "cuda"


def _run(fn, acc, s_acc, gam, bet, **kw):
    m, c = acc.shape
    X = torch.empty((m, c), dtype=torch.int16, device=DEV)
    A = torch.empty((m, c), dtype=torch.int8, device=DEV)
    codes = torch.empty(2 * c, dtype=torch.int32, device=DEV)
    scal = torch.empty(iq.IQ_BN_SCALES, dtype=torch.float64, device=DEV)
    fixed = torch.empty(4 * c + 2, dtype=torch.int64, device=DEV)
    s_a = torch.zeros(1, dtype=torch.float64, device=DEV)
    fn(acc, s_acc, gam, bet, A, s_a, xhat=X, bn_codes=codes, bn_scales=scal, bn_fixed=fixed, **kw)
    torch.cuda.synchronize()
    return [t.cpu().numpy() for t in (X, A, codes, scal, fixed, s_a)]


def _case(g, m, c, spread, call):
    acc = torch.from_numpy((g.standard_normal((m, c)) * spread +
                            g.integers(-2000, 2001, c)).astype(np.int32)).to(DEV)
    gam, bet = (torch.from_numpy(v).to(DEV) for v in S.bn_gamma_beta_codes(g, c))
    s_acc = torch.tensor([2.0 ** -14 * (call + 1.5)], dtype=torch.float64, device=DEV)
    return acc, s_acc, gam, bet


def test_noalloc_matches_workspace_version_twice():
    """A larger channel count, then a smaller one: the second call reuses the bytes the
    first one left in the shared array."""
    g = S.rng(2024)
    for call, (m, c, spread) in enumerate([(777, 4096, 90000.0), (4096, 256, 3000.0)]):
        acc, s_acc, gam, bet = _case(g, m, c, spread, call)
        want = _run(iq.iq_bn_int_fwd, acc, s_acc, gam, bet)
        got = _run(iq.iq_bn_int_fwd_noalloc, acc, s_acc, gam, bet)
        for w, h in zip(want, got):
            assert np.array_equal(w, h), call


def test_noalloc_identical_calls_in_a_row():
    """The same call twice: a statistic that is not reset between calls (a sum that
    doubles, an extreme that sticks) would change the second result."""
    g = S.rng(7)
    acc, s_acc, gam, bet = _case(g, 3000, 512, 20000.0, 0)
    want = _run(iq.iq_bn_int_fwd, acc, s_acc, gam, bet)
    for rep in range(2):
        got = _run(iq.iq_bn_int_fwd_noalloc, acc, s_acc, gam, bet)
        for w, h in zip(want, got):
            assert np.array_equal(w, h), rep


def test_noalloc_rejects_too_many_channels():
    acc = torch.zeros((8, 4100), dtype=torch.int32, device=DEV)
    g = torch.zeros(4100, dtype=torch.int32, device=DEV)
    with pytest.raises(iq.IqError) as e:
        _run(iq.iq_bn_int_fwd_noalloc, acc, torch.ones(1, dtype=torch.float64, device=DEV), g, g)
    assert e.value.code == iq.IQ_ERR_UNSUPPORTED
