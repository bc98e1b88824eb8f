"""The oracle and the library defaults against the few numbers the paper prints
(tests/golden/paper_values.json, each entry with its section and equation)."""
import json
import os

import numpy as np

import oracle as O
from paper_2011_14504_gb300 import iq

GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_values.json")))


def test_step_of_8_bit_quantizer_is_the_printed_value():
    # the UQ grid at k = 8: adjacent codes of inputs one step apart differ by exactly one,
    # and the step rounds to the printed 0.008
    g = GOLD["delta_k8"]
    delta = 2.0 ** (1 - 8)
    codes = O.uq(np.array([0.0, delta, 2 * delta, -delta], np.float32), 8)
    assert codes.tolist() == [0, 1, 2, -1]
    assert round(delta, g["printed_digits"]) == g["value"]


def test_uq_clip_range_is_one_step_inside_plus_minus_one():
    # Eq. (UQ): values beyond +-1 clip to +-(1 - Delta)
    delta = 2.0 ** -7
    codes = O.uq(np.array([1.0, 5.0, -1.0, -7.5, 1 - delta], np.float32), 8)
    vals = codes * delta
    assert vals.tolist() == [1 - delta, 1 - delta, -1 + delta, -1 + delta, 1 - delta]
    assert GOLD["uq_range_k8"]["hi"] == "1-Delta" and GOLD["uq_range_k8"]["lo"] == "-1+Delta"


def test_x2_scaled_quantizer_covers_plus_minus_two():
    # Sec. 3.1.1: the BN parameters use 2 UQ(x / 2, k), whose range is +-2 (1 - Delta)
    r = GOLD["x2_scaled_range"]["value"]
    k = 8
    codes = O.uq2(np.array([r, -r, 1.5, 0.5], np.float32), k)
    step = 2.0 ** (2 - k)
    assert (codes * step).tolist() == [r * (1 - 2.0 ** (1 - k)), -r * (1 - 2.0 ** (1 - k)), 1.5, 0.5]


def test_library_bn_bit_widths_follow_the_deeplab_setting():
    b = GOLD["deeplab_bits"]
    bits = iq.bn_bits()
    assert (bits.k_mu, bits.k_sigma, bits.k_xhat, bits.k_gamma, bits.k_beta) == \
        (b["k_mu"], b["k_sigma"], b["k_xhat"], b["k_gamma"], b["k_beta"])
    assert bits.k_a == b["k_A"]
    from oracle import deeplab as OD
    assert OD.K_E2 in b["k_E2"]


def test_weight_master_width_is_k_u():
    # Eq. (WQ1): W_q = UQ8 of the k_U = 24 bit master, i.e. the top 8 bits rounded half up
    assert GOLD["fcn_bits"]["k_U"] == GOLD["deeplab_bits"]["k_U"] == 24
    m = np.array([0, 2 ** 15 - 1, 2 ** 15, 3 * 2 ** 16, -(2 ** 15), -(2 ** 15) - 1,
                  2 ** 23 - 1], np.int32)
    assert O.requant_master(m).tolist() == [0, 0, 1, 3, 0, -1, 127]
