"""One token through M LittleBit linears of one shape in one launch
(littlebit_linear_forward_multi) against the oracle, against M calls of the
single-linear entry point, and against itself (repeated calls on one
workspace are bit-identical)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2506_13771_gb300 import build as lb_build
from paper_2506_13771_gb300 import inputs
from paper_2506_13771_gb300 import littlebit as lb

pytestmark = pytest.mark.gpu

DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _built():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    lb_build.build()
    lb.lib()


def rel(a, b) -> float:
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / np.linalg.norm(b))


MULTI = [
    # d_in, d_out, ranks, M
    (512, 136, (64, 32), 3),        # ragged output octets over the CTAs
    (256, 1000, (16, 8), 7),        # 8 input words: most CTAs hold none
    (1024, 512, (256,), 5),         # one path
    (4096, 11008, (128, 128), 2),   # gate / up of the 7B shape
    (11008, 4096, (512, 512), 3),   # several input words per CTA
    (4096, 4096, (64, 64), 24),     # the most linears per launch; the ring wraps 4 times
]


@pytest.mark.parametrize("d_in,d_out,rs,M", MULTI)
@pytest.mark.parametrize("out_dtype", [torch.float32, torch.bfloat16])
def test_multi_vs_oracle_and_single(d_in, d_out, rs, M, out_dtype):
    rng = inputs.rng_for(113, salt=d_in + d_out + M)
    layers = [inputs.make_linear(rng, d_in, d_out, list(rs), len(rs), 0.05) for _ in range(M)]
    x = inputs.bf16_normal(rng, (1, d_in))
    D = [lb.DeviceLinear(L, DEV) for L in layers]
    xt = lb.bf16_tensor(x, DEV)[0]
    ws = lb.new_workspace(lb.multi_workspace_size(D), DEV)
    y = torch.full((M, d_out), float("nan"), dtype=out_dtype, device=DEV)
    for rep in range(3):   # the launch epoch flips the exchange buffers every call
        lb.linear_forward_multi(D, xt, y=y, ws=ws)
        torch.cuda.synchronize()
        yg = y.float().cpu().numpy().astype(np.float64)
        assert np.all(np.isfinite(yg))
        if rep == 0:
            y0 = yg.copy()
        else:
            assert np.array_equal(yg, y0)
    for m in range(M):
        e = rel(yg[m], oracle.forward_factored(layers[m], x)[0])
        assert e <= (1e-4 if out_dtype == torch.float32 else 2e-3), (m, e)
    # bit for bit the single-linear path at T = 1 (the same exact fixed-point
    # exchange and the same fp32 sums in the same order)
    for m in (0, M - 1):
        ys = torch.full((1, d_out), float("nan"), dtype=out_dtype, device=DEV)
        lb.linear_forward(D[m], xt[None, :], y=ys)
        torch.cuda.synchronize()
        assert torch.equal(ys[0], y[m])
    st = lb.lib().littlebit_poll_error(ws.data_ptr(), None)
    assert st == lb.LB_OK
