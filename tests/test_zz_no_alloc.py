"""littlebit_linear_forward_noalloc against littlebit_linear_forward.

The allocation-free entry point serves callers that cannot allocate device
memory (their memory is owned by a host framework, or their hot path may
not call cudaMalloc).  It runs on a scratch array built into the library,
shared by every call.  These checks call it through the C ABI twice in a
row, so the second call starts from the first call's leftovers, and compare
both results with the workspace entry point.  This file is collected last.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2506_13771_gb300 import build as lb_build
from paper_2506_13771_gb300 import inputs
from paper_2506_13771_gb300 import littlebit as lb

pytestmark = pytest.mark.gpu

TOL_FP32 = 1e-4  # the fp32-output bound of the parity tests
TOL_BF16 = 2e-3  # the bf16-output bound of the parity tests
DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _built():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    lb_build.build()
    lb.lib()


def rel(a, b):
    a = a.double().cpu().numpy()
    b = b.double().cpu().numpy()
    return float(np.linalg.norm(a - b) / np.linalg.norm(b))


def call_noalloc(D, x, y, code):
    return lb.lib().littlebit_linear_forward_noalloc(
        ctypes.byref(D.c), x.data_ptr(), x.shape[0], y.data_ptr(), code,
        torch.cuda.current_stream().cuda_stream)


def layer_for(cfg):
    """(layer, x bf16 bits) of a parity case."""
    if cfg == "512_r16_T4":
        return inputs.config1()
    if cfg.startswith("4096_r64"):
        return inputs.config2(8 if cfg.endswith("T8") else 1)
    rng = inputs.rng_for(300, salt=len(cfg))
    if cfg == "unequal_ranks_T5":  # Eq. 6 with paths of rank 48 and 16
        L = inputs.make_linear(rng, 1024, 768, [48, 16], 2, 0.05)
        return L, inputs.bf16_normal(rng, (5, 1024))
    assert cfg == "one_path_T3"
    L = inputs.make_linear(rng, 1024, 768, 32, 1, 0.05)
    return L, inputs.bf16_normal(rng, (3, 1024))


@pytest.mark.parametrize("out_dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("cfg", ["512_r16_T4", "4096_r64_T8", "4096_r64_T1", "unequal_ranks_T5",
                                 "one_path_T3"])
def test_noalloc_matches_workspace_entry_point(cfg, out_dtype):
    layer, x_bits = layer_for(cfg)
    D = lb.DeviceLinear(layer, DEV)
    x = lb.bf16_tensor(x_bits, DEV)
    ref = lb.linear_forward(D, x, out_dtype=out_dtype)
    code = lb.LB_OUT_FP32 if out_dtype == torch.float32 else lb.LB_OUT_BF16
    outs = []
    for _ in range(2):  # the second call reuses the scratch the first one left behind
        y = torch.full_like(ref, float("nan"))
        st = call_noalloc(D, x, y, code)
        assert st == lb.LB_OK, lb.status_string(st)
        torch.cuda.synchronize()
        outs.append(y)
    tol = TOL_FP32 if out_dtype == torch.float32 else TOL_BF16
    for y in outs:
        assert torch.isfinite(y.float()).all()
        assert rel(y, ref) <= tol


def test_noalloc_at_its_limit_and_one_token_beyond():
    """T * (sum of ranks) == 65536 fp32 sums is accepted and matches the
    workspace entry point; one more token is refused with LB_ERR_WORKSPACE
    before anything is launched."""
    layer, _ = inputs.config1()  # two paths of rank 16: 2048 tokens fill the scratch
    D = lb.DeviceLinear(layer, DEV)
    x = lb.bf16_tensor(inputs.bf16_normal(inputs.rng_for(301), (2049, 512)), DEV)
    ref = lb.linear_forward(D, x[:2048], out_dtype=torch.float32)
    for _ in range(2):
        y = torch.full_like(ref, float("nan"))
        st = call_noalloc(D, x[:2048], y, lb.LB_OUT_FP32)
        assert st == lb.LB_OK, lb.status_string(st)
        torch.cuda.synchronize()
        assert rel(y, ref) <= TOL_FP32
    y = torch.full((2049, 512), float("nan"), dtype=torch.float32, device=DEV)
    assert call_noalloc(D, x, y, lb.LB_OUT_FP32) == lb.LB_ERR_WORKSPACE
    torch.cuda.synchronize()
    assert torch.isnan(y).all()


def test_noalloc_rejects_requests_beyond_its_scratch():
    layer, x_bits = inputs.config2(1)
    D = lb.DeviceLinear(layer, DEV)
    # 600 tokens x 128 ranks = 76800 fp32 sums > 65536
    x = torch.zeros((600, 4096), dtype=torch.bfloat16, device=DEV)
    y = torch.zeros((600, 4096), dtype=torch.float32, device=DEV)
    st = lb.lib().littlebit_linear_forward_noalloc(ctypes.byref(D.c), x.data_ptr(), 600,
                                                   y.data_ptr(), lb.LB_OUT_FP32, None)
    assert st == lb.LB_ERR_WORKSPACE
