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


@pytest.mark.parametrize("cfg", ["512_r16_T4", "4096_r64_T8", "4096_r64_T1"])
def test_noalloc_matches_workspace_entry_point(cfg):
    if cfg == "512_r16_T4":
        layer, x_bits = inputs.config1()
    else:
        layer, x_bits = inputs.config2(8 if cfg.endswith("T8") else 1)
    D = lb.DeviceLinear(layer, DEV)
    x = lb.bf16_tensor(x_bits, DEV)
    ref = lb.linear_forward(D, x, out_dtype=torch.float32)
    outs = []
    for _ in range(2):  # the second call reuses the scratch the first one left behind
        y = torch.full_like(ref, float("nan"))
        st = lb.lib().littlebit_linear_forward_noalloc(
            ctypes.byref(D.c), x.data_ptr(), x.shape[0], y.data_ptr(), lb.LB_OUT_FP32,
            torch.cuda.current_stream().cuda_stream)
        assert st == lb.LB_OK, lb.status_string(st)
        torch.cuda.synchronize()
        outs.append(y)
    for y in outs:
        assert torch.isfinite(y).all()
        assert rel(y, ref) <= TOL_FP32


def test_noalloc_rejects_requests_beyond_its_scratch():
    layer, x_bits = inputs.config2(1)
    D = lb.DeviceLinear(layer, DEV)
    # 600 tokens x 128 ranks = 76800 fp32 sums > 65536
    x = torch.zeros((600, 4096), dtype=torch.bfloat16, device=DEV)
    y = torch.zeros((600, 4096), dtype=torch.float32, device=DEV)
    st = lb.lib().littlebit_linear_forward_noalloc(ctypes.byref(D.c), x.data_ptr(), 600,
                                                   y.data_ptr(), lb.LB_OUT_FP32, None)
    assert st == lb.LB_ERR_WORKSPACE
