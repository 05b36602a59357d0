"""Parity of rdn_qk_prologue / rdn_qk_prologue_bwd (SiLU, then L2 normalisation
of q and k rows) with the fp64 oracle, through the C ABI."""
import numpy as np
import pytest
import torch

import oracle
import paper_2509_25223_gb300 as rdn
from tests.parity_util import as64, assert_close

pytestmark = pytest.mark.gpu

DT = {"bf16": torch.bfloat16, "f32": torch.float32}


def _rows(shape, dtype, seed, scale=2.0):
    g = torch.Generator(device="cpu").manual_seed(seed)
    return (scale * torch.randn(shape, generator=g)).to(DT[dtype]).cuda()


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("D", [64, 128])
@pytest.mark.parametrize("shape", [(1, 1, 1), (2, 37, 3), (3, 130, 4)])
def test_prologue_forward_and_backward(dtype, D, shape):
    """q and k in one launch (row counts that leave partial groups of rows per
    warp), and the backward with upstream gradients of both outputs."""
    q = _rows(shape + (D,), dtype, 1)
    k = _rows(shape + (D,), dtype, 2)
    yq, yk = rdn.qk_prologue(q, k)
    dyq = _rows(shape + (D,), dtype, 3, 1.0)
    dyk = _rows(shape + (D,), dtype, 4, 1.0)
    dq, dk = rdn.qk_prologue_bwd(q, k, dyq, dyk)
    torch.cuda.synchronize()
    for x, y, dy, dx, name in [(q, yq, dyq, dq, "q"), (k, yk, dyk, dk, "k")]:
        assert_close(y, oracle.qk_prologue(as64(x)), dtype, "y" + name)
        assert_close(dx, oracle.qk_prologue_bwd(as64(x), as64(dy)), dtype, "dx" + name)


def test_prologue_single_tensor_and_unit_norm():
    q = _rows((2, 300, 16, 128), "f32", 5)
    yq, yk = rdn.qk_prologue(q)
    assert yk is None
    torch.cuda.synchronize()
    n = torch.linalg.vector_norm(yq.double(), dim=-1)
    assert float((n - 1).abs().max()) < 1e-5
    dq, _ = rdn.qk_prologue_bwd(q, None, torch.ones_like(q))
    torch.cuda.synchronize()
    assert_close(dq, oracle.qk_prologue_bwd(as64(q), np.ones(q.shape)), "f32", "dq")


def test_prologue_norm_floor():
    """Rows whose SiLU norm is below eps are scaled by 1/eps (forward) and the
    backward takes the floor's branch: all-zero rows and tiny rows."""
    eps = 1e-3
    x = torch.zeros(4, 128)
    x[1] = 1e-5 * torch.arange(128) / 128.0
    x[2, 3] = -2e-4
    x[3] = torch.randn(128, generator=torch.Generator().manual_seed(9))  # a regular row
    x = x.cuda()
    dy = torch.randn(4, 128, generator=torch.Generator().manual_seed(10)).cuda()
    y, _ = rdn.qk_prologue(x, eps=eps)
    dx, _ = rdn.qk_prologue_bwd(x, None, dy, eps=eps)
    torch.cuda.synchronize()
    np.testing.assert_allclose(as64(y), oracle.qk_prologue(as64(x), eps=eps), atol=1e-6, rtol=1e-5)
    np.testing.assert_allclose(as64(dx), oracle.qk_prologue_bwd(as64(x), as64(dy), eps=eps),
                               atol=1e-5, rtol=1e-4)
    assert float(y[0].abs().max()) == 0.0


def test_prologue_full_size_sampled():
    """The bench workload's q, k shape (8 x 4096 x 16 rows of 128, bf16), in the
    launch configuration the bench times; sampled rows against the oracle."""
    B, T, H, D = 8, 4096, 16, 128
    q = _rows((B, T, H, D), "bf16", 11)
    k = _rows((B, T, H, D), "bf16", 12)
    dyq = _rows((B, T, H, D), "bf16", 13, 1.0)
    dyk = _rows((B, T, H, D), "bf16", 14, 1.0)
    yq, yk = rdn.qk_prologue(q, k)
    dq, dk = rdn.qk_prologue_bwd(q, k, dyq, dyk)
    torch.cuda.synchronize()
    rng = np.random.default_rng(0)
    idx = [(int(rng.integers(B)), int(rng.integers(T)), int(rng.integers(H))) for _ in range(64)]
    idx += [(0, 0, 0), (B - 1, T - 1, H - 1)]
    for t_in, t_out, t_dy, t_dx in [(q, yq, dyq, dq), (k, yk, dyk, dk)]:
        xs = torch.stack([t_in[i] for i in idx])
        assert_close(torch.stack([t_out[i] for i in idx]), oracle.qk_prologue(as64(xs)), "bf16", "y")
        dys = torch.stack([t_dy[i] for i in idx])
        assert_close(torch.stack([t_dx[i] for i in idx]),
                     oracle.qk_prologue_bwd(as64(xs), as64(dys)), "bf16", "dx")
