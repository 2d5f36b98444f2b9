"""MemoryBridge output on the GPU against the fp64 oracle: LayerNorm,
nu tanh and the 2 nu norm cap, row by row (fp32 on the GPU: within 2e-5 of
nu relative), with and without the cap active, in place, and over more rows
than the grid (grid-stride)."""

import numpy as np
import pytest
import torch

import oracle
import paper_2609_25537_gb300 as cmc

pytestmark = pytest.mark.gpu


def _case(rows, D, nu, scale, affine, dev, seed=0, in_place=False):
    rng = np.random.default_rng(seed)
    x = (rng.standard_normal((rows, D)) * scale + 0.3).astype(np.float32)
    g = (1 + 0.2 * rng.standard_normal(D)).astype(np.float32) if affine else None
    b = (0.2 * rng.standard_normal(D)).astype(np.float32) if affine else None
    xd = torch.from_numpy(x).to(dev)
    gd = None if g is None else torch.from_numpy(g).to(dev)
    bd = None if b is None else torch.from_numpy(b).to(dev)
    out = cmc.bridge_epilogue(xd, nu, gamma=gd, beta=bd, out=xd if in_place else None)
    got = out.cpu().numpy().astype(np.float64)
    ref = oracle.bridge_epilogue(x, np.ones(D) if g is None else g, np.zeros(D) if b is None else b, nu)
    np.testing.assert_allclose(got, ref, rtol=2e-5, atol=2e-5 * nu)
    assert np.all(np.linalg.norm(got, axis=1) <= 2 * nu * (1 + 1e-5))
    return ref


# rows in registers, one 128-thread CTA per row: D = 64 and 36 take one float4
# per thread, 1028 three (the last one partial), 2048 four, 2600 six, 3072 six,
# 3588 eight (partial), 4096 eight; 16384: rows staged in shared memory
@pytest.mark.parametrize("rows,D", [(1024, 4096), (300, 64), (7, 16384), (50, 36), (33, 2048),
                                    (17, 3072), (29, 1028), (21, 2600), (13, 3588)])
@pytest.mark.parametrize("affine", [False, True])
def test_bridge_epilogue_shapes(cuda_device, rows, D, affine):
    ref = _case(rows, D, 0.8, 2.0, affine, cuda_device)
    # at D >= 16 these rows are capped: the norm is exactly 2 nu
    if D >= 64:
        np.testing.assert_allclose(np.linalg.norm(ref, axis=1), 1.6, rtol=1e-12)


def test_bridge_epilogue_below_the_cap_and_in_place(cuda_device):
    # a tiny gamma keeps nu tanh(m_hat) well inside the 2 nu ball: no rescale
    rng = np.random.default_rng(3)
    D = 512
    x = rng.standard_normal((64, D)).astype(np.float32)
    g = np.full(D, 0.01, dtype=np.float32)
    xd = torch.from_numpy(x).to(cuda_device)
    out = cmc.bridge_epilogue(xd, 1.5, gamma=torch.from_numpy(g).to(cuda_device), out=xd)
    assert out.data_ptr() == xd.data_ptr()
    ref = oracle.bridge_epilogue(x, g, np.zeros(D), 1.5)
    np.testing.assert_allclose(out.cpu().numpy(), ref, rtol=2e-5, atol=3e-5)
    assert np.all(np.linalg.norm(ref, axis=1) < 3.0)


def test_bridge_epilogue_many_rows(cuda_device):
    _case(20000, 64, 0.5, 1.0, True, cuda_device, seed=9)
