"""The decode step at position p (the paper's end-to-end decoding setting:
LittleBit linears inside a Llama-shaped decoder with RMS norms, rotary
embedding and softmax attention over a KV cache) on the GPU, through the C
ABI, against the fp64 oracle run on the same tokens.

Bar: the activations are fp32 on the GPU and exact in the oracle (no bf16
rounding points between the linears), so the differences are fp32 versus
fp64 arithmetic: ~1e-6 per layer on these chains (the 70B-shaped stack holds
1e-4 over 80 layers).  Outputs and caches are held to 1e-4 relative L2."""
import numpy as np
import pytest
import torch

import oracle
from paper_2506_13771_gb300 import build as lb_build
from paper_2506_13771_gb300 import inputs
from paper_2506_13771_gb300 import littlebit as lb

pytestmark = pytest.mark.gpu

DEV = "cuda"
TOL = 1e-4


@pytest.fixture(scope="module", autouse=True)
def _built():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    lb_build.build()
    lb.lib()


@pytest.fixture(scope="module")
def orc():
    return oracle.Oracle()


def rel(a, b) -> float:
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / np.linalg.norm(b))


def small(rng, n_layers=2, n_heads=4, n_kv_heads=2, head_dim=64, d_ff=384, r=(64, 32, 64)):
    d, dkv = n_heads * head_dim, n_kv_heads * head_dim
    layers = []
    for _ in range(n_layers):
        for (di, do, rr) in inputs.stack_shapes(d, dkv, d_ff, *r):
            layers.append(inputs.make_linear(rng, di, do, rr, 2, inputs.unit_gain_scale(di, rr)))
    return layers, {"n_heads": n_heads, "n_kv_heads": n_kv_heads, "head_dim": head_dim,
                    "rope_base": 10000.0}


def run_and_compare(orc, layers, shape, xs, max_pos, graph=False):
    n_layers = len(layers) // 7
    dec = lb.DeviceDecoder(layers, shape["n_heads"], shape["n_kv_heads"], shape["head_dim"],
                           max_pos, shape["rope_base"], DEV)
    d, dkv = dec.d_model, dec.d_kv
    kc = np.zeros((n_layers, max_pos, dkv))
    vc = np.zeros((n_layers, max_pos, dkv))
    x_static = torch.zeros(d, dtype=torch.bfloat16, device=DEV)
    out = torch.full((d,), float("nan"), dtype=torch.float32, device=DEV)
    g = None
    if graph:
        # one step captured once; every replay decodes the next position
        x_static.copy_(lb.bf16_tensor(xs[0], DEV))
        dec.step(x_static, out)             # warm-up outside the capture (position 0)
        torch.cuda.synchronize()
        dec.pos.zero_()
        dec.kcache.zero_()
        dec.vcache.zero_()
        s = torch.cuda.Stream()
        with torch.cuda.stream(s):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=s):
                dec.step(x_static, out, stream=s)
        torch.cuda.synchronize()
    worst = 0.0
    for p, x in enumerate(xs):
        x_static.copy_(lb.bf16_tensor(x, DEV))
        if graph:
            g.replay()
        else:
            dec.step(x_static, out)
        torch.cuda.synchronize()
        want, _, _ = orc.decoder_step(layers, shape, p, x, kc, vc, round_inputs=False)
        got = out.cpu().numpy().astype(np.float64)
        assert np.all(np.isfinite(got))
        e = rel(got, want)
        worst = max(worst, e)
        assert e <= TOL, (p, e)
    assert int(dec.pos.item()) == len(xs)
    P = len(xs)
    kg = dec.kcache.cpu().numpy().astype(np.float64)
    vg = dec.vcache.cpu().numpy().astype(np.float64)
    assert rel(kg[:, :P], kc[:, :P]) <= TOL and rel(vg[:, :P], vc[:, :P]) <= TOL
    assert not kg[:, P:].any() and not vg[:, P:].any()
    assert dec.poll_error() == lb.LB_OK
    return worst


def test_decoder_steps_vs_oracle(orc):
    """Nine tokens from position 0 through a 2-layer GQA decoder (4 query
    heads sharing 2 kv heads of 64): each step's output and, at the end, every
    cache row against the oracle; rows after the last position stay zero."""
    rng = inputs.rng_for(110)
    layers, shape = small(rng)
    xs = inputs.bf16_normal(rng, (9, 256))
    run_and_compare(orc, layers, shape, xs, max_pos=16)


def test_decoder_step_replays_as_a_graph(orc):
    """The step captured once as a CUDA graph: each replay reads the device
    position, decodes the next token and advances the position."""
    rng = inputs.rng_for(111)
    layers, shape = small(rng, n_layers=3, n_heads=4, n_kv_heads=4, head_dim=64, d_ff=256,
                          r=(32, 32, 64))
    xs = inputs.bf16_normal(rng, (6, 256))
    run_and_compare(orc, layers, shape, xs, max_pos=6, graph=True)


def test_decoder_long_context(orc):
    """200 tokens through one GQA layer with heads of 128 (the benchmark's head
    size): attention over up to 200 cached positions, many times the positions
    one pass of the attention kernel's warps covers, checked at every step."""
    rng = inputs.rng_for(112)
    layers, shape = small(rng, n_layers=1, n_heads=4, n_kv_heads=2, head_dim=128, d_ff=256,
                          r=(32, 32, 32))
    xs = inputs.bf16_normal(rng, (200, 512))
    run_and_compare(orc, layers, shape, xs, max_pos=256)


def test_decoder_7b_shape_first_tokens(orc):
    """The Llama2-7B-shaped workload of the benchmark (32 layers, 32 heads of
    128, d_ff 11008, two LittleBit paths per linear): its first three tokens."""
    layers, xs = inputs.decoder7b(3)
    S = inputs.DECODER_7B
    shape = {"n_heads": S["n_heads"], "n_kv_heads": S["n_kv_heads"], "head_dim": S["head_dim"],
             "rope_base": 10000.0}
    run_and_compare(orc, layers, shape, xs, max_pos=8)


def test_decoder_position_out_of_range_is_refused():
    """A step at position max_pos records LB_ERR_RANGE and writes nothing."""
    rng = inputs.rng_for(112)
    layers, shape = small(rng, n_layers=1)
    dec = lb.DeviceDecoder(layers, shape["n_heads"], shape["n_kv_heads"], shape["head_dim"], 4,
                           10000.0, DEV)
    dec.pos.fill_(4)
    x = lb.bf16_tensor(inputs.bf16_normal(rng, (256,)), DEV)
    out = torch.full((256,), float("nan"), dtype=torch.float32, device=DEV)
    dec.step(x, out)
    assert dec.poll_error() == lb.LB_ERR_RANGE
    assert torch.isnan(out).all() and not dec.kcache.any() and int(dec.pos.item()) == 4
    assert dec.poll_error() == lb.LB_OK
