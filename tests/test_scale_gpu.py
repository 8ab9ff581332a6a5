"""Input magnitude: the single-token kernels against the fp64 oracle when x, g
and l are far from unit scale (needs a GB300).

Prop. 1 is linear, Y(c x) = c Y(x), so a correct kernel's relative error must
not depend on the overall magnitude of its inputs.  The single-token kernels
all-reduce the rank-r partial sums t across the CTAs through fixed-point
exchange words; these tests hold them to the same bars as the unit-scale
parity tests (relative L2 1e-4 for fp32 outputs, 2e-3 for bf16) with x scaled
by 2^-16, 2^-8 and 2^8, with g and l drawn 1000x smaller, and with a decoder
whose residual stream has an RMS of 1e-3.  Because the exchange sums are
exact, scaling x by a power of two must also scale the fp32 output of a
single linear by exactly that power, bit for bit.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2506_13771_gb300 import build as lb_build
from paper_2506_13771_gb300 import inputs
from paper_2506_13771_gb300 import littlebit as lb

pytestmark = pytest.mark.gpu

TOL = 2e-3
TOL_FP32 = 1e-4
DEV = "cuda"
SHIFTS = [-16, -8, 8]


@pytest.fixture(scope="module", autouse=True)
def _built():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    lb_build.build()
    lb.lib()


def rel(a, b) -> float:
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / np.linalg.norm(b))


def shift_bf16(bits: np.ndarray, k: int) -> np.ndarray:
    """bf16 bit patterns of the values times 2^k (exact: normal values only)."""
    f = (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64) * 2.0 ** k
    out = (f.astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)
    assert np.array_equal((out.astype(np.uint32) << 16).view(np.float32).astype(np.float64), f)
    return out


def forward(D, x_bits, out_dtype):
    x = lb.bf16_tensor(x_bits, DEV)
    y = torch.full((x.shape[0], D.d_out), float("nan"), dtype=out_dtype, device=DEV)
    lb.linear_forward(D, x, y=y)
    torch.cuda.synchronize()
    return y


def check(y, ref, out_dtype):
    got = y.float().cpu().numpy().astype(np.float64)
    assert np.all(np.isfinite(got))
    e = rel(got, ref)
    assert e <= (TOL_FP32 if out_dtype == torch.float32 else TOL), e
    return e


def one_token_cases():
    L2, _ = inputs.config2(1)
    lins3, _, _ = inputs.config3(128, 1)
    return {"cfg2_q": L2, "cfg3_gate": lins3["gate"], "cfg3_down": lins3["down"]}


@pytest.fixture(scope="module")
def cases():
    return {k: (L, lb.DeviceLinear(L, DEV)) for k, L in one_token_cases().items()}


@pytest.mark.parametrize("name", ["cfg2_q", "cfg3_gate", "cfg3_down"])
@pytest.mark.parametrize("k", SHIFTS)
@pytest.mark.parametrize("out_dtype", [torch.float32, torch.bfloat16])
def test_single_token_scaled_input(cases, name, k, out_dtype):
    L, D = cases[name]
    x = inputs.bf16_normal(inputs.rng_for(200, salt=k + 100), (1, L["d_in"]), 2.0 ** k)
    check(forward(D, x, out_dtype), oracle.forward_factored(L, x), out_dtype)


@pytest.mark.parametrize("name", ["cfg2_q", "cfg3_down"])
def test_single_token_scale_equivariance_is_exact(cases, name):
    """y(2^k x) == 2^k y(x) bit for bit for the fp32 output."""
    L, D = cases[name]
    x = inputs.bf16_normal(inputs.rng_for(201), (1, L["d_in"]))
    y0 = forward(D, x, torch.float32)
    for k in SHIFTS:
        yk = forward(D, shift_bf16(x, k), torch.float32)
        assert torch.equal(yk, y0 * 2.0 ** k), k


@pytest.mark.parametrize("d_in,d_out,r", [(4096, 4096, 64), (4096, 11008, 128),
                                          (11008, 4096, 128)])
@pytest.mark.parametrize("out_dtype", [torch.float32, torch.bfloat16])
def test_single_token_small_g_and_l(d_in, d_out, r, out_dtype):
    """g and l 1000x smaller than the workloads' |N(0,1)| * 0.02 (fp16 subnormals
    among them, decoded exactly on both sides)."""
    rng = inputs.rng_for(202, salt=d_out + r)
    L = inputs.make_linear(rng, d_in, d_out, r, 2, 0.02, g_mul=1e-3, l_mul=1e-3)
    x = inputs.bf16_normal(rng, (1, d_in))
    check(forward(lb.DeviceLinear(L, DEV), x, out_dtype), oracle.forward_factored(L, x),
          out_dtype)


@pytest.mark.parametrize("k", SHIFTS)
def test_multi_linear_scaled_input(k):
    """Several same-shape linears on one token in one launch (the grouped q / k / v
    and gate / up of the decode step)."""
    rng = inputs.rng_for(203, salt=k + 100)
    Ls = [inputs.make_linear(rng, 4096, 4096, 64, 2, 0.02,
                             g_mul=1e-3 if m == 1 else 1.0, l_mul=1e-3 if m == 1 else 1.0)
          for m in range(3)]
    x = inputs.bf16_normal(rng, (4096,), 2.0 ** k)
    Ds = [lb.DeviceLinear(L, DEV) for L in Ls]
    y = lb.linear_forward_multi(Ds, lb.bf16_tensor(x, DEV), out_dtype=torch.float32)
    torch.cuda.synchronize()
    got = y.cpu().numpy().astype(np.float64)
    for m, L in enumerate(Ls):
        ref = oracle.forward_factored(L, x[None, :])[0]
        assert rel(got[m], ref) <= TOL_FP32, (m, rel(got[m], ref))


# ------------------------------------------------------------------ stack


def run_stack(layers, x0, head_dim):
    S = lb.DeviceStack(layers, head_dim, DEV)
    ws = S.prepare()
    out, q, kv = lb.stack_forward(S, lb.bf16_tensor(x0, DEV), ws=ws)
    assert lb.poll_error(ws) == lb.LB_OK
    return tuple(t.cpu().numpy().astype(np.float64) for t in (out, q, kv))


def check_stack(got, ref):
    out, q, kv = got
    r_out, r_q, r_kv = ref
    for g in got:
        assert np.all(np.isfinite(g))
    assert rel(out, r_out) <= TOL_FP32, rel(out, r_out)
    for l in range(q.shape[0]):
        assert rel(q[l], r_q[l]) <= TOL_FP32, (l, "q", rel(q[l], r_q[l]))
        assert rel(kv[l, 0], r_kv[l, 0]) <= TOL_FP32, (l, "k", rel(kv[l, 0], r_kv[l, 0]))
        assert rel(kv[l, 1], r_kv[l, 1]) <= TOL_FP32, (l, "v", rel(kv[l, 1], r_kv[l, 1]))


SMALL = dict(d_model=1024, d_kv=256, d_ff=2048, r_qo=48, r_kv=16, r_mlp=64, head_dim=64)


@pytest.mark.parametrize("k", SHIFTS)
def test_stack_two_layers_scaled_input(k):
    layers, x0 = inputs.make_stack(n_layers=2, config_id=204, **SMALL)
    x0 = shift_bf16(x0, k)
    check_stack(run_stack(layers, x0, 64), oracle.stack_forward(layers, x0, head_dim=64))


def test_stack_two_layers_small_scales():
    """g and l 1000x smaller in every linear: every exchanged t (and every
    q, k, v output) is ~1000x smaller than at unit gain."""
    layers, x0 = inputs.make_stack(n_layers=2, config_id=205, g_mul=1e-3, l_mul=1e-3, **SMALL)
    check_stack(run_stack(layers, x0, 64), oracle.stack_forward(layers, x0, head_dim=64))


@pytest.mark.parametrize("bad", [0x7F80, 0xFFC0])  # bf16 +inf, NaN
def test_nonfinite_input_reports_range(bad):
    """An infinite or NaN input entry leaves every exchange's range: the stack
    and the single-token kernel record LB_ERR_RANGE (the exchanges still
    complete -- out-of-range contributions are sent as zero, so nothing
    waits), and a workspace prepared again afterwards computes the finite
    input correctly."""
    layers, x0 = inputs.make_stack(n_layers=2, config_id=207, **SMALL)
    xb = x0.copy()
    xb[17] = bad
    S = lb.DeviceStack(layers, 64, DEV)
    ws = S.prepare()
    lb.stack_forward(S, lb.bf16_tensor(xb, DEV), ws=ws)
    assert lb.poll_error(ws) == lb.LB_ERR_RANGE
    S.prepare(ws)
    out, q, kv = lb.stack_forward(S, lb.bf16_tensor(x0, DEV), ws=ws)
    assert lb.poll_error(ws) == lb.LB_OK
    got = tuple(t.cpu().numpy().astype(np.float64) for t in (out, q, kv))
    check_stack(got, oracle.stack_forward(layers, x0, head_dim=64))

    L, _ = inputs.config2(1)
    D = lb.DeviceLinear(L, DEV)
    x = inputs.bf16_normal(inputs.rng_for(208), (1, L["d_in"]))
    x[0, 5] = bad
    ws1 = lb.new_workspace(lb.workspace_size(D, 1), DEV)
    y = torch.empty((1, D.d_out), dtype=torch.float32, device=DEV)
    lb.linear_forward(D, lb.bf16_tensor(x, DEV), y=y, ws=ws1)
    assert lb.poll_error(ws1) == lb.LB_ERR_RANGE


@pytest.fixture(scope="module")
def stack70b():
    layers, x0 = inputs.config5()
    return layers, x0, lb.DeviceStack(layers, 128, DEV)


@pytest.mark.parametrize("k", SHIFTS)
def test_stack_70b_scaled_input(stack70b, k):
    """The 80-layer Llama2-70B-shaped stack on x0 times 2^k."""
    layers, x0, S = stack70b
    xk = shift_bf16(x0, k)
    ws = S.prepare()
    out, q, kv = lb.stack_forward(S, lb.bf16_tensor(xk, DEV), ws=ws)
    assert lb.poll_error(ws) == lb.LB_OK
    got = tuple(t.cpu().numpy().astype(np.float64) for t in (out, q, kv))
    check_stack(got, oracle.stack_forward(layers, xk, head_dim=128))


def test_stack_70b_small_scales():
    layers, x0 = inputs.make_stack(n_layers=80, config_id=206, g_mul=1e-3, l_mul=1e-3,
                                   **{k: v for k, v in inputs.STACK_70B.items()
                                      if k != "n_layers"})
    check_stack(run_stack(layers, x0, 128), oracle.stack_forward(layers, x0, head_dim=128))


# ------------------------------------------------------------------ decode step


def test_decoder_small_hidden_state():
    """The decode step at positions 0..5 with token embeddings of RMS 1e-3 and
    the o / down outputs 1000x smaller, so the residual stream -- the input of
    every grouped q / k / v and gate / up launch, whose 1 / rms rides the
    exchange -- keeps an RMS near 1e-3."""
    orc = oracle.Oracle()
    rng = inputs.rng_for(207)
    n_heads, n_kv, hd, d_ff = 4, 2, 64, 384
    d, dkv = n_heads * hd, n_kv * hd
    layers = []
    for _ in range(2):
        for k, (di, do, rr) in enumerate(inputs.stack_shapes(d, dkv, d_ff, 64, 32, 64)):
            layers.append(inputs.make_linear(rng, di, do, rr, 2, inputs.unit_gain_scale(di, rr),
                                             h_mul=1e-3 if k in (3, 6) else 1.0))
    shape = {"n_heads": n_heads, "n_kv_heads": n_kv, "head_dim": hd, "rope_base": 10000.0}
    xs = inputs.bf16_normal(rng, (6, d), 1e-3)
    max_pos = 8
    dec = lb.DeviceDecoder(layers, n_heads, n_kv, hd, max_pos, 10000.0, DEV)
    kc = np.zeros((2, max_pos, dkv))
    vc = np.zeros((2, max_pos, dkv))
    out = torch.full((d,), float("nan"), dtype=torch.float32, device=DEV)
    for p, x in enumerate(xs):
        dec.step(lb.bf16_tensor(x, DEV), out)
        torch.cuda.synchronize()
        want, _, _ = orc.decoder_step(layers, shape, p, x, kc, vc, round_inputs=False)
        got = out.cpu().numpy().astype(np.float64)
        assert np.all(np.isfinite(got))
        assert float(np.sqrt(np.mean(want ** 2))) < 1e-2
        assert rel(got, want) <= TOL_FP32, (p, rel(got, want))
    assert dec.poll_error() == lb.LB_OK
