"""GPU parity of the nibble-split fp8 GEMM (tcgen05 kind::f8f6f4, four MMAs per k-step on the
e4m3 nibbles of the int8 codes), through the C ABI: exact against the int64 product of the
same int8 matrices, including all-extreme operands (every code -128 or 127, the largest
partial sums) and the longest reduction the route keeps exact (k = 65536), and against the
fp16-carrier route of the library's 1x1 convolution on the same operands."""
import numpy as np
import pytest
import torch

from paper_2011_14504_gb300 import iq

pytestmark = pytest.mark.gpu

DEV = "cuda"


def run(a, b):
    c = torch.empty((a.shape[0], b.shape[0]), dtype=torch.int32, device=DEV)
    iq.iq_gemm_s8_nibble(torch.from_numpy(a).to(DEV), torch.from_numpy(b).to(DEV), c)
    torch.cuda.synchronize()
    return c.cpu().numpy()


@pytest.mark.parametrize("m,n,k", [(128, 128, 128), (256, 384, 640), (1024, 512, 2304)])
def test_nibble_gemm_exact(m, n, k):
    g = np.random.default_rng(m + n + k)
    a = g.integers(-128, 128, size=(m, k), dtype=np.int64).astype(np.int8)
    b = g.integers(-128, 128, size=(n, k), dtype=np.int64).astype(np.int8)
    want = a.astype(np.int64) @ b.astype(np.int64).T
    assert np.array_equal(run(a, b).astype(np.int64), want)


def test_nibble_gemm_extremes_and_longest_k():
    g = np.random.default_rng(7)
    m, n, k = 128, 128, 65536
    a = np.where(g.random((m, k)) < 0.5, -128, 127).astype(np.int8)
    b = np.where(g.random((n, k)) < 0.5, -128, 127).astype(np.int8)
    a[0, :] = -128
    b[0, :] = -128                                 # c[0][0] = 65536 * 16384 = 2^30
    want = a.astype(np.int64) @ b.astype(np.int64).T
    assert np.array_equal(run(a, b).astype(np.int64), want)


def test_nibble_gemm_matches_conv_route():
    g = np.random.default_rng(9)
    m, n, k = 512, 256, 1024
    a = g.integers(-127, 128, size=(m, k), dtype=np.int64).astype(np.int8)
    b = g.integers(-127, 128, size=(n, k), dtype=np.int64).astype(np.int8)
    d = iq.conv_desc(1, 1, m, k, n, 1, 1)
    acc = torch.empty((1, 1, m, n), dtype=torch.int32, device=DEV)
    a_out = torch.empty((1, 1, m, n), dtype=torch.int8, device=DEV)
    iq.iq_conv_fwd(d, torch.from_numpy(a).to(DEV), torch.ones(1, dtype=torch.float64, device=DEV),
                   torch.from_numpy(b).to(DEV), a_out, torch.empty(1, dtype=torch.float64, device=DEV),
                   relu=False, acc_out=acc)
    torch.cuda.synchronize()
    assert np.array_equal(run(a, b), acc.cpu().numpy().reshape(m, n))


def test_nibble_gemm_argument_checks():
    a = torch.zeros((100, 128), dtype=torch.int8, device=DEV)
    b = torch.zeros((128, 128), dtype=torch.int8, device=DEV)
    c = torch.empty((100, 128), dtype=torch.int32, device=DEV)
    with pytest.raises(iq.IqError):
        iq.iq_gemm_s8_nibble(a, b, c)
