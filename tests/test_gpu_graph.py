"""The entry points under CUDA graph capture: a training step (forward with
chunk states and saved intermediates, backward reading them) captured once
and replayed on new inputs copied into the captured tensors gives the same
results as the eager calls on those inputs."""
import pytest
import torch

import paper_2509_25223_gb300 as rdn
from rdn_synthetic import make_inputs
from tests.parity_util import assert_close

pytestmark = pytest.mark.gpu

NAMES = ("q", "k", "v", "g", "beta", "gamma")


@pytest.mark.parametrize("dtype,D,variant", [("bf16", 128, "rdn"), ("f32", 64, "rla")])
def test_step_replays_under_cuda_graph(dtype, D, variant):
    B, T, H = 2, 200, 2
    static = make_inputs(B, T, H, D, dtype=dtype, with_grad_out=True, device="cuda", seed=1)
    fwd = rdn.rdn_fwd if variant == "rdn" else rdn.rla_fwd
    bwd = rdn.rdn_bwd if variant == "rdn" else rdn.rla_bwd
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    save = variant == "rdn"
    wsf = torch.empty(rdn.workspace_bytes(f"{variant}_fwd", B, T, H, D, tdt, save_for_bwd=save),
                      dtype=torch.uint8, device="cuda")

    def step(x):
        o, ST, RT, Sc, Rc = fwd(*(x[n] for n in NAMES), clip=1.0, return_chunk_states=True,
                                workspace=wsf, save_for_bwd=save)
        kw = dict(fwd_saved=True) if save else {}
        d = bwd(*(x[n] for n in NAMES), x["dO"], clip=1.0, S_chunks=Sc, R_chunks=Rc,
                fwd_workspace=wsf, **kw)
        return o, ST, d

    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):  # warm-up outside the capture (first-use lookups)
        step(static)
    torch.cuda.current_stream().wait_stream(s)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        o_g, ST_g, d_g = step(static)
    for seed in (2, 3):
        new = make_inputs(B, T, H, D, dtype=dtype, with_grad_out=True, device="cuda", seed=seed)
        for n in NAMES + ("dO",):
            static[n].copy_(new[n])
        g.replay()
        torch.cuda.synchronize()
        o_e, ST_e, d_e = step(new)
        torch.cuda.synchronize()
        assert torch.equal(o_g, o_e) and torch.equal(ST_g, ST_e)
        for name in ("dq", "dk", "dv", "dg", "dbeta", "dgamma"):
            assert_close(d_g[name], d_e[name].float(), dtype, name)
