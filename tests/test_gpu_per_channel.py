"""GPU parity of the per-channel Scale variant (Eqs. (ScaleFactor), (ScaleQ) with the maximum
taken per channel), through the C ABI, bit-exact against the oracle: NHWC-, NCHW- and
filter-shaped views, int32 and int64 inputs, 4-, 8- and 16-bit codes, with and without ReLU,
an all-zero channel, and the argument checks."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2011_14504_gb300 import iq

pytestmark = pytest.mark.gpu

DEV = "cuda"

CASES = [
    # outer, c, inner, in dtype, k, out dtype, relu
    (16 * 33 * 31, 256, 1, np.int32, 8, torch.int8, True),      # NHWC conv output
    (2 * 65 * 65, 2048, 1, np.int32, 8, torch.int8, False),
    (4, 96, 37 * 29, np.int32, 8, torch.int8, False),            # NCHW
    (1, 64, 3 * 3 * 128, np.int64, 8, torch.int8, False),        # KRSC filter gradient
    (1000, 24, 1, np.int64, 16, torch.int16, True),
    (777, 13, 5, np.int32, 4, torch.int32, False),
]


@pytest.mark.parametrize("ci", range(len(CASES)))
def test_per_channel_sq_matches_oracle(ci):
    outer, c, inner, idt, k, odt, relu = CASES[ci]
    g = np.random.default_rng(300 + ci)
    hi = (1 << 30) if idt == np.int64 else (1 << 24)
    q = g.integers(-hi, hi, size=(outer, c, inner), dtype=np.int64)
    q[:, c // 3, :] = 0                                          # an all-zero channel
    q[:, -1, :] //= 1000                                         # a small-valued channel
    q = q.astype(idt)
    codes = torch.empty(q.shape, dtype=odt, device=DEV)
    s_out = torch.empty(c, dtype=torch.float64, device=DEV)
    s_in = torch.tensor([3.5e-6], dtype=torch.float64, device=DEV)
    iq.iq_requantize_per_channel(torch.from_numpy(q).to(DEV), outer, c, inner, s_in, k, codes,
                                 s_out, relu=relu)
    want, sw = O.sq_per_channel(q, outer, c, inner, 3.5e-6, k, relu)
    torch.cuda.synchronize()
    assert np.array_equal(codes.cpu().numpy().astype(np.int32), want)
    assert np.array_equal(s_out.cpu().numpy(), sw)


def test_per_channel_sq_argument_checks():
    q = torch.zeros((4, 8, 1), dtype=torch.int32, device=DEV)
    codes = torch.empty((4, 8, 1), dtype=torch.int8, device=DEV)
    s_out = torch.empty(8, dtype=torch.float64, device=DEV)
    s_in = torch.ones(1, dtype=torch.float64, device=DEV)
    with pytest.raises(iq.IqError):                              # 16-bit codes in int8
        iq.iq_requantize_per_channel(q, 4, 8, 1, s_in, 16, codes, s_out)
    with pytest.raises(iq.IqError):
        iq.iq_requantize_per_channel(q, 4, 8, 1, s_in, 1, codes, s_out)
    iq.iq_requantize_per_channel(q, 4, 8, 1, s_in, 8, codes, s_out)
    torch.cuda.synchronize()
    assert not codes.cpu().numpy().any()
    assert np.all(s_out.cpu().numpy() == 2.0 ** -7)


@pytest.mark.parametrize("shift", [1, 11, 17, 30])
def test_weight_decay_matches_oracle(shift):
    """The decoupled L2 weight decay of the masters (decay step 2^-shift) and the regenerated
    forward codes, against the oracle."""
    g = np.random.default_rng(shift)
    m = g.integers(-(1 << 23) + 1, 1 << 23, size=100003).astype(np.int32)
    dm = torch.from_numpy(m).to(DEV)
    wq = torch.empty(m.shape, dtype=torch.int8, device=DEV)
    iq.iq_weight_decay(dm, wq, shift)
    m2, w2 = O.weight_decay(m, shift)
    torch.cuda.synchronize()
    assert np.array_equal(dm.cpu().numpy(), m2)
    assert np.array_equal(wq.cpu().numpy().astype(np.int32), w2)
