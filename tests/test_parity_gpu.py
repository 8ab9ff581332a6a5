"""CUDA path vs the fp64 CPU oracle, through the C ABI (needs a GB300).

Bars: sign packing bit-exact; float outputs within relative L2 2e-3 of the
oracle (bf16 inputs, fp32 accumulation), the tolerance the workload states.
fp32 outputs are also held to 1e-4: fp32 sums of n sign-weighted terms of
unit-scale data carry a relative error of order 2^-24 * sqrt(n) (about 1e-5
for the largest reduction here, n = 28672), so 1e-4 leaves a 10x margin;
bf16 outputs carry the bf16 rounding itself (relative RMS about 1.2e-3).
"""
import ctypes
import os

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


@pytest.fixture(scope="module", autouse=True)
def _built():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    lb_build.build()
    lb.lib()


def rel(a, b) -> float:
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / np.linalg.norm(b))


def oracle_layer(layer: dict) -> dict:
    """The oracle's view of a layer: explicit signs packed by the ORACLE packer."""
    paths = []
    for P in layer["paths"]:
        if "v_words" in P:
            paths.append(P)
        else:
            paths.append(dict(r=P["r"], v_words=oracle.pack_v(P["v_signs"]),
                              u_words=oracle.pack_u(P["u_signs"]), g=P["g"], l=P["l"], h=P["h"]))
    return {"d_in": layer["d_in"], "d_out": layer["d_out"], "paths": paths}


def gpu_forward(D: lb.DeviceLinear, x_bits: np.ndarray, out_dtype) -> np.ndarray:
    x = lb.bf16_tensor(x_bits, DEV)
    y = torch.full((x.shape[0], D.d_out), float("nan"), dtype=out_dtype, device=DEV)
    lb.linear_forward(D, x, y=y)
    torch.cuda.synchronize()
    return y.float().cpu().numpy().astype(np.float64)


def check(y_gpu, y_ref, out_dtype, fp32_tol=TOL_FP32):
    assert np.all(np.isfinite(y_gpu)), "unwritten (NaN sentinel) or non-finite outputs"
    e = rel(y_gpu, y_ref)
    assert e <= TOL, e
    if out_dtype == torch.float32:
        assert e <= fp32_tol, e
    return e


# ------------------------------------------------------------------ packing (Eq. 2)


@pytest.mark.parametrize("rows,cols", [(1, 1), (5, 16), (33, 70), (64, 192), (100, 33),
                                       (512, 512), (4096, 64)])
def test_pack_bit_exact(rows, cols):
    rng = np.random.default_rng(rows * 1000 + cols)
    s = inputs.random_signs(rng, rows, cols)
    d = torch.from_numpy(s).to(DEV)
    wu = lb.pack(d, lb.LB_PACK_U).cpu().numpy().view(np.uint32)
    wv = lb.pack(d, lb.LB_PACK_V).cpu().numpy().view(np.uint32)
    assert np.array_equal(wu, oracle.pack_u(s))
    assert np.array_equal(wv, oracle.pack_v(s))


def test_pack_flags_invalid_sign():
    s = np.ones((8, 40), np.int8)
    s[3, 17] = 0
    bad = torch.zeros(1, dtype=torch.int32, device=DEV)
    lb.pack(torch.from_numpy(s).to(DEV), lb.LB_PACK_U, bad=bad)
    assert int(bad.item()) == 1
    ok = torch.zeros(1, dtype=torch.int32, device=DEV)
    lb.pack(torch.from_numpy(np.ones((8, 40), np.int8)).to(DEV), lb.LB_PACK_V, bad=ok)
    assert int(ok.item()) == 0


# ------------------------------------------------------------------ single linears


@pytest.mark.parametrize("out_dtype", [torch.float32, torch.bfloat16])
def test_config1_512_r16_T4(out_dtype):
    L, x = inputs.config1()
    D = lb.DeviceLinear(L, DEV)
    y = gpu_forward(D, x, out_dtype)
    OL = oracle_layer(L)
    check(y, oracle.forward_factored(OL, x), out_dtype)
    check(y, oracle.forward_dense(OL, x), out_dtype)


@pytest.mark.parametrize("T", [1, 8])
@pytest.mark.parametrize("out_dtype", [torch.float32, torch.bfloat16])
def test_config2_4096_r64(T, out_dtype):
    L, x = inputs.config2(T)
    D = lb.DeviceLinear(L, DEV)
    check(gpu_forward(D, x, out_dtype), oracle.forward_factored(L, x), out_dtype)


@pytest.mark.parametrize("r", [128, 512])
@pytest.mark.parametrize("T", [1, 16, 64])
def test_config3_ffn_triple(r, T):
    lins, x, x_down = inputs.config3(r, T)
    # T >= 16 runs on the tensor cores with fp16 operands (z rounded to fp16)
    tol = 1e-3 if T >= 16 else TOL_FP32
    for name in ("gate", "up", "down"):
        L = lins[name]
        xin = x_down if name == "down" else x
        D = lb.DeviceLinear(L, DEV)
        check(gpu_forward(D, xin, torch.float32), oracle.forward_factored(L, xin), torch.float32,
              tol)
    D = lb.DeviceLinear(lins["down"], DEV)
    check(gpu_forward(D, x_down, torch.bfloat16), oracle.forward_factored(lins["down"], x_down),
          torch.bfloat16)


@pytest.mark.parametrize("shape", list(inputs.PREFILL_SHAPES))
@pytest.mark.parametrize("T", [2048, 8192])
def test_config4_prefill_sampled_tokens(shape, T):
    """Full-size prefill on the GPU; the oracle recomputes sampled tokens."""
    L, x = inputs.config4(shape, T)
    D = lb.DeviceLinear(L, DEV)
    y = gpu_forward(D, x, torch.bfloat16)
    assert np.all(np.isfinite(y))
    rng = np.random.default_rng(T)
    rows = np.unique(np.concatenate([[0, T - 1], rng.choice(T, 14, replace=False)]))
    check(y[rows], oracle.forward_factored(L, x[rows]), torch.bfloat16)


STRESS = [
    # d_in, d_out, ranks, T
    (32, 17, (1,), 1), (32, 1000, (16, 33), 2), (4128, 17, (96, 1), 3), (4128, 1000, (33, 96), 7),
    (64, 64, (96,), 8), (4128, 1000, (16,), 9), (1024, 300, (33, 16), 65), (4128, 40, (1, 1), 1),
    (96, 2048, (1000, 24), 1), (8192, 8, (64, 64), 1),
    # T >= 16 but d_out % 8 != 0 or r > 512: the CUDA-core path
    (512, 2100, (192,), 300), (256, 512, (576,), 40),
]


@pytest.mark.parametrize("d_in,d_out,rs,T", STRESS)
def test_stress_shapes(d_in, d_out, rs, T):
    rng = inputs.rng_for(100, salt=d_in + d_out + T)
    L = inputs.make_linear(rng, d_in, d_out, list(rs), len(rs), 0.1)
    x = inputs.bf16_normal(rng, (T, d_in))
    D = lb.DeviceLinear(L, DEV)
    tol = 1e-3 if _tensor_path(d_in, rs, T) else TOL_FP32
    check(gpu_forward(D, x, torch.float32), oracle.forward_factored(L, x), torch.float32, tol)


PREFILL = [
    # d_in, d_out, ranks, T   (the tensor-core path: T >= 16 and T x sum of ranks
    # above 8192, ranks multiples of 64 up to 512, d_out a multiple of 8)
    (64, 256, (64,), 160), (128, 512, (64, 64), 256), (4096, 4096, (64, 64), 200),
    (256, 1000, (128, 64), 77), (512, 2104, (192,), 300), (1024, 768, (512, 512), 130),
    (4096, 11008, (128, 128), 64), (64, 8, (64, 64), 65), (512, 1000, (512,), 17),
    # stage 1 split along d_in into K slices (long d_in, few token tiles)
    (11008, 4096, (128, 128), 48), (4096, 2048, (512, 512), 300), (2048, 64, (64, 64), 72),
    # four token tiles or more with stage-1 tiles at most 128 wide: fp16 x in
    # a TMEM ring (N1 = 128: six stages, N1 = 64: eight)
    (1024, 520, (64, 64), 700), (2048, 1000, (64,), 900),
    # outputs narrower than one TMA store box (64 bf16 / 32 fp32 columns): the
    # stores clip the columns beyond d_out
    (1024, 8, (64, 64), 400), (512, 24, (64,), 512), (256, 40, (128, 128), 700),
]


@pytest.mark.parametrize("d_in,d_out,rs,T", PREFILL)
@pytest.mark.parametrize("out_dtype", [torch.float32, torch.bfloat16])
def test_prefill_tensor_core_shapes(d_in, d_out, rs, T, out_dtype):
    """Ragged token counts and output widths, one and two paths, on tcgen05."""
    rng = inputs.rng_for(104, salt=d_in + d_out + T)
    L = inputs.make_linear(rng, d_in, d_out, list(rs), len(rs), 0.05)
    x = inputs.bf16_normal(rng, (T, d_in))
    D = lb.DeviceLinear(L, DEV)
    y = gpu_forward(D, x, out_dtype)
    # fp16 operands (x converted exactly, z = l.t rounded to fp16): ~3e-4
    e = rel(y, oracle.forward_factored(L, x))
    assert np.all(np.isfinite(y)) and e <= (TOL if out_dtype == torch.bfloat16 else 1e-3), e


PAIR = [
    # d_in, d_out, ranks, T: N1 a multiple of 512 and at least 96 column-pair
    # tiles, ragged last token tile
    (1024, 264, (512, 512), 6100), (512, 136, (256, 256), 12200), (4096, 512, (512,), 12290),
]


@pytest.mark.parametrize("d_in,d_out,rs,T", PAIR)
@pytest.mark.parametrize("two_sm", [True, False])
def test_prefill_column_pair_tiles(d_in, d_out, rs, T, two_sm):
    """Long token runs with N1 a multiple of 512 take stage 1 in column-pair
    tiles: by default on SM pairs (tcgen05 cta_group::2, 256 x 512 tiles,
    then stage 2 in 256 x 256 pair tiles, three launches), with
    LB_PREFILL_2SM=0 in the one-launch 1-SM form (128 x 512 tiles, 64-byte
    swizzle).  Sampled rows of the forward and of both latent types against
    the oracle."""
    old = os.environ.get("LB_PREFILL_2SM")
    os.environ["LB_PREFILL_2SM"] = "1" if two_sm else "0"
    try:
        _column_pair_case(d_in, d_out, rs, T)
    finally:
        if old is None:
            os.environ.pop("LB_PREFILL_2SM", None)
        else:
            os.environ["LB_PREFILL_2SM"] = old


def _column_pair_case(d_in, d_out, rs, T):
    rng = inputs.rng_for(109, salt=d_in + T)
    L = inputs.make_linear(rng, d_in, d_out, list(rs), len(rs), 0.05)
    x = inputs.bf16_normal(rng, (T, d_in))
    D = lb.DeviceLinear(L, DEV)
    ws = lb.new_workspace(lb.workspace_size(D, T), DEV)
    xin = lb.bf16_tensor(x, DEV)
    rows = np.unique(np.concatenate([[0, 1, 127, 128, T - 85, T - 1],
                                     rng.choice(T, 10, replace=False)]))
    y = torch.full((T, d_out), float("nan"), dtype=torch.float32, device=DEV)
    lb.linear_forward(D, xin, y=y, ws=ws)
    torch.cuda.synchronize()
    yg = y.cpu().numpy().astype(np.float64)
    assert np.all(np.isfinite(yg))
    e = rel(yg[rows], oracle.forward_factored(L, x[rows]))
    assert e <= 1e-3, e
    z_ref = oracle.latent(L, x[rows])
    for zt, tol in ((torch.float32, 1e-4), (torch.float16, 1e-3)):
        z = torch.full((T, sum(rs)), float("nan"), dtype=zt, device=DEV)
        lb.linear_latent(D, xin, z=z, ws=ws)
        torch.cuda.synchronize()
        zg = z.float().cpu().numpy().astype(np.float64)
        assert np.all(np.isfinite(zg))
        e = rel(zg[rows], z_ref)
        assert e <= tol, e
    # the expansion alone (stage 2 on its own) from seeded fp16 latents
    z16 = rng.standard_normal((T, sum(rs))).astype(np.float16)
    ye = torch.full((T, d_out), float("nan"), dtype=torch.float32, device=DEV)
    lb.linear_expand(D, torch.from_numpy(z16).to(DEV), y=ye, ws=ws)
    torch.cuda.synchronize()
    yeg = ye.cpu().numpy().astype(np.float64)
    assert np.all(np.isfinite(yeg))
    e = rel(yeg[rows], oracle.expand(L, z16[rows].astype(np.float64)))
    assert e <= 1e-4, e
    assert lb.poll_error(ws) == lb.LB_OK


@pytest.mark.parametrize("T", [1, 4])
def test_padding_bits_are_ignored(T):
    """U words with every padding bit set (r = 33, 16) give the same output."""
    rng = inputs.rng_for(101, salt=T)
    L = inputs.make_linear(rng, 256, 96, [33, 16], 2, 0.1)
    x = inputs.bf16_normal(rng, (T, 256))
    y_ref = oracle.forward_factored(L, x)
    for P, pad in zip(L["paths"], (0xFFFFFFFE, 0xFFFF0000)):
        P["u_words"] = P["u_words"].copy()
        P["u_words"][:, -1] |= np.uint32(pad)
    D = lb.DeviceLinear(L, DEV)
    check(gpu_forward(D, x, torch.float32), y_ref, torch.float32)


# ------------------------------------------------------------------ latent states (Sec. 5)

LATENT = [
    # d_in, d_out, ranks, T   (CUDA-core stages unless T >= 16 and the ranks and
    # d_in are multiples of 64)
    (256, 96, (33, 16), 1), (512, 40, (7,), 3), (4128, 1000, (96, 1), 9), (1024, 300, (33, 16), 65),
    (8192, 1024, (32, 32), 1), (8192, 1024, (32, 32), 64),
    (128, 512, (64, 64), 256), (256, 1000, (128, 64), 77), (4096, 2048, (512, 512), 300),
    (11008, 4096, (128, 128), 48), (4096, 4096, (64, 64), 600), (4096, 1000, (128,), 16),
]


def _tensor_path(d_in, rs, T):
    return (T >= 16 and T * sum(rs) > 8192 and d_in % 64 == 0
            and all(r % 64 == 0 and r <= 512 for r in rs))


@pytest.mark.parametrize("d_in,d_out,rs,T", LATENT)
@pytest.mark.parametrize("z_dtype", [torch.float32, torch.float16])
def test_latent_and_expand(d_in, d_out, rs, T, z_dtype):
    """z = l . ((X . g) V_sign) per path as [T][r_0 + r_1], and its expansion,
    each against the oracle; expanding the GPU latent gives the forward."""
    rng = inputs.rng_for(106, salt=d_in + d_out + T)
    L = inputs.make_linear(rng, d_in, d_out, list(rs), len(rs), 0.05)
    x = inputs.bf16_normal(rng, (T, d_in))
    D = lb.DeviceLinear(L, DEV)
    ws = lb.new_workspace(lb.workspace_size(D, T), DEV)
    xin = lb.bf16_tensor(x, DEV)
    z = torch.full((T, sum(rs)), float("nan"), dtype=z_dtype, device=DEV)
    lb.linear_latent(D, xin, z=z, ws=ws)
    torch.cuda.synchronize()
    zg = z.float().cpu().numpy().astype(np.float64)
    z_ref = oracle.latent(L, x)
    assert np.all(np.isfinite(zg))
    # fp32: fp32 sums (1e-4 as for the forward); fp16: the fp16 rounding of z
    # itself, relative RMS 2^-11 / sqrt(3) ~ 2.8e-4
    e = rel(zg, z_ref)
    assert e <= (1e-4 if z_dtype == torch.float32 else 1e-3), e
    # the expansion alone, on the oracle's latent in the same element type
    z_in = torch.from_numpy(z_ref.astype(np.float32)).to(z_dtype)
    z_exp = z_in.double().numpy()
    y = torch.full((T, d_out), float("nan"), dtype=torch.float32, device=DEV)
    lb.linear_expand(D, z_in.to(DEV), y=y, ws=ws)
    torch.cuda.synchronize()
    yg = y.cpu().numpy().astype(np.float64)
    assert np.all(np.isfinite(yg))
    # the tensor-core stage rounds an fp32 z to fp16 operands
    tol = 1e-3 if (_tensor_path(d_in, rs, T) and z_dtype == torch.float32) else 1e-4
    e = rel(yg, oracle.expand(L, z_exp))
    assert e <= tol, e
    # expand(latent(X)) against the oracle's forward (fp32 output: with a few
    # hundred outputs the bf16 rounding alone can exceed 2e-3 by chance)
    yc = torch.full((T, d_out), float("nan"), dtype=torch.float32, device=DEV)
    lb.linear_expand(D, z, y=yc, ws=ws)
    torch.cuda.synchronize()
    tol = 1e-3 if (_tensor_path(d_in, rs, T) or z_dtype == torch.float16) else 1e-4
    check(yc.cpu().numpy().astype(np.float64), oracle.forward_factored(L, x), torch.float32, tol)


def test_latent_kv_cache_70b_kv_projection():
    """The 70B key projection (8192 -> 1024, two paths of rank 32): a 512-token
    fp16 latent cache is 16x smaller than the bf16 keys, and its expansion
    matches the forward of each cached token."""
    rng = inputs.rng_for(107)
    T, d, dkv, r = 512, 8192, 1024, 32
    L = inputs.make_linear(rng, d, dkv, [r, r], 2, 0.02)
    x = inputs.bf16_normal(rng, (T, d))
    D = lb.DeviceLinear(L, DEV)
    xin = lb.bf16_tensor(x, DEV)
    z = lb.linear_latent(D, xin, z_dtype=torch.float16)
    keys = lb.linear_forward(D, xin, out_dtype=torch.bfloat16)
    assert z.numel() * z.element_size() * 16 == keys.numel() * keys.element_size()
    y = lb.linear_expand(D, z, out_dtype=torch.float32)
    torch.cuda.synchronize()
    rows = np.array([0, 1, 77, 300, T - 1])
    zg = z.float().cpu().numpy().astype(np.float64)
    assert rel(zg[rows], oracle.latent(L, x[rows])) <= 1e-3
    ref = oracle.forward_factored(L, x[rows])
    assert rel(y.cpu().numpy().astype(np.float64)[rows], ref) <= TOL
    assert rel(keys.float().cpu().numpy().astype(np.float64)[rows], ref) <= TOL


def test_latent_full_size_prefill_sampled_tokens():
    """4096 x 4096, two paths of rank 512, 2048 tokens: the tensor-core
    latent (split along d_in or not, as the forward) on sampled tokens."""
    L, x = inputs.config4("4096x4096_r512", 2048)
    D = lb.DeviceLinear(L, DEV)
    xin = lb.bf16_tensor(x, DEV)
    for z_dtype, tol in ((torch.float32, 1e-4), (torch.float16, 1e-3)):
        z = lb.linear_latent(D, xin, z_dtype=z_dtype)
        torch.cuda.synchronize()
        rows = np.array([0, 5, 127, 128, 1000, 2047])
        zg = z.float().cpu().numpy().astype(np.float64)[rows]
        assert rel(zg, oracle.latent(L, x[rows])) <= tol


# ------------------------------------------------------------------ Dual-SVID (Sec. 3.2, 3.3)


def _svid_weights(layer):
    """W_hat of each path of a host layer dict (oracle unpacker and decoders)."""
    out = []
    for P in layer["paths"]:
        r = P["r"]
        us = oracle.unpack_u(P["u_words"], layer["d_out"], r)
        vs = oracle.unpack_v(P["v_words"], layer["d_in"], r)
        dec = lambda b: np.asarray(b, np.uint16).view(np.float16).astype(np.float64)
        out.append((us, vs, oracle.path_weight(us, vs, dec(P["h"]), dec(P["g"]), dec(P["l"]))))
    return out


@pytest.mark.parametrize("d_out,d_in,ranks", [(256, 384, (16, 16)), (384, 256, (24,)),
                                              (200, 136, (8, 40)), (96, 96, (96,))])
def test_dual_svid_vs_oracle(d_out, d_in, ranks):
    """Dual-SVID on the GPU (subspace iteration) against the oracle (exact
    Jacobi SVD) on weights whose singular values fall by 0.85 per index:
    path-0 signs equal wherever |U'| and |V'| are not tiny, scales within
    fp16 rounding, each path's W_hat and the total reconstruction error match."""
    rng = inputs.rng_for(108, salt=d_out + d_in)
    W = inputs.spectral_weight(rng, d_out, d_in, 0.85 ** np.arange(min(d_out, d_in)))
    ref = oracle.dual_svid(W, ranks)
    got = lb.layer_to_host(lb.dual_svid(torch.from_numpy(W.astype(np.float32)).to(DEV), ranks,
                                        iters=10))
    torch.cuda.synchronize()
    gw, rw = _svid_weights(got), _svid_weights(ref)
    r0 = ranks[0]
    s, U, V = oracle.svd_top(W, r0)
    Up, Vp = U * np.sqrt(s), V * np.sqrt(s)
    for mine, theirs, F in ((gw[0][0], ref["signs"][0][0], Up), (gw[0][1], ref["signs"][0][1], Vp)):
        bad = mine != theirs
        assert np.all(np.abs(F[bad]) < 1e-3 * np.abs(F).max()), int(bad.sum())
    dec = lambda b: np.asarray(b, np.uint16).view(np.float16).astype(np.float64)
    for key in ("h", "g", "l"):
        a, b = dec(got["paths"][0][key]), dec(ref["paths"][0][key])
        assert rel(a, b) <= 2e-3, (key, rel(a, b))
    assert rel(gw[0][2], rw[0][2]) <= 2e-3, rel(gw[0][2], rw[0][2])
    Wg = sum(p[2] for p in gw)
    Wr = sum(p[2] for p in rw)
    eg, er = rel(Wg, W), rel(Wr, W)
    assert abs(eg - er) <= 0.02 * er + 1e-4, (eg, er)
    if len(ranks) == 2:
        assert rel(Wg, W) < rel(gw[0][2], W)  # the residual path helps


def test_dual_svid_exact_cases():
    """A Sylvester-Hadamard LittleBit weight (h = g = 1) is recovered (signs up
    to one joint flip per column, W_hat = W within fp16 scale rounding); an
    all-zero weight gives +1 signs and zero scales."""
    d, r = 64, 8
    H = np.array([[1.0]])
    while H.shape[0] < d:
        H = np.block([[H, H], [H, -H]])
    H = H[:, :r]
    lam = np.array([9.0, 7.5, 6.0, 5.0, 4.0, 3.0, 2.0, 1.5])
    W = (H * lam) @ H.T
    got = lb.layer_to_host(lb.dual_svid(torch.from_numpy(W.astype(np.float32)).to(DEV), [r]))
    ((us, vs, Wg),) = _svid_weights(got)
    flip = (us[0] * H[0]).astype(np.int8)
    assert np.array_equal(us, (H * flip).astype(np.int8))
    assert np.array_equal(vs, (H * flip).astype(np.int8))
    assert rel(Wg, W) <= 2e-3
    Z = torch.zeros((48, 80), dtype=torch.float32, device=DEV)
    got = lb.layer_to_host(lb.dual_svid(Z, [4, 4]))
    for P in got["paths"]:
        assert not P["u_words"].any() and not P["v_words"].any()
        for key in ("h", "g", "l"):
            assert np.all(np.asarray(P[key], np.uint16).view(np.float16) == 0)


def test_dual_svid_512x384_two_paths():
    """A larger weight, 512 x 384 with ranks (40, 40): the same checks as the
    small cases against the oracle's exact SVD (a few seconds of CPU work)."""
    test_dual_svid_vs_oracle(512, 384, (40, 40))


# ------------------------------------------------------------------ QAT backward (SmoothSign)

# TF32 rounds the non-sign GEMM operands to 10 mantissa bits (relative error
# up to 2^-11 per element, about 2^-11 / sqrt(3) ~ 2.8e-4 RMS); a product
# with two rounded operands (dY^T z, X^T dt) carries about 4e-4 relative L2.
# fp32 accumulation adds ~1e-6.  Bar: 2e-3 relative L2 per gradient.
TOL_TF32 = 2e-3


def _train_case(rng, d_in, d_out, rs):
    paths = []
    for r in rs:
        paths.append({"r": r,
                      "u": (rng.standard_normal((d_out, r)) * 0.02).astype(np.float32),
                      "v": (rng.standard_normal((d_in, r)) * 0.02).astype(np.float32),
                      "g": (0.5 + rng.random(d_in)).astype(np.float32),
                      "l": (0.5 + rng.random(r)).astype(np.float32),
                      "h": (0.5 + rng.random(d_out)).astype(np.float32)})
    return {"d_in": d_in, "d_out": d_out, "paths": paths}


@pytest.mark.parametrize("d_in,d_out,rs,T", [(256, 192, (16, 16), 64), (512, 1024, (64,), 130),
                                             (1000, 520, (33, 7), 37), (4096, 4096, (64, 64), 256)])
def test_train_forward_backward_vs_oracle(d_in, d_out, rs, T):
    """QAT forward and every gradient of the backward against the fp64 oracle
    on the same fp32 latent factors (signs decided on identical values)."""
    rng = inputs.rng_for(109, salt=d_in + d_out + T)
    layer = _train_case(rng, d_in, d_out, rs)
    x = rng.standard_normal((T, d_in)).astype(np.float32)
    dy = rng.standard_normal((T, d_out)).astype(np.float32)
    TL = lb.TrainLinear(layer, DEV)
    xd, dyd = torch.from_numpy(x).to(DEV), torch.from_numpy(dy).to(DEV)
    y = lb.train_forward(TL, xd)
    grads, dx = lb.train_backward(TL, xd, dyd, k=100.0)
    torch.cuda.synchronize()
    L64 = {"d_in": d_in, "d_out": d_out,
           "paths": [{k: (P[k].astype(np.float64) if k != "r" else P[k]) for k in P}
                     for P in layer["paths"]]}
    y_ref = oracle.train_forward(L64, x.astype(np.float64))
    g_ref, dx_ref = oracle.train_backward(L64, x.astype(np.float64), dy.astype(np.float64), k=100.0)
    assert rel(y.cpu().numpy(), y_ref) <= TOL_TF32
    assert rel(dx.cpu().numpy(), dx_ref) <= TOL_TF32
    for p in range(len(rs)):
        for key in ("du", "dv", "dg", "dl", "dh"):
            e = rel(grads[p][key].cpu().numpy(), g_ref[p][key])
            assert e <= TOL_TF32, (p, key, e)


def test_train_backward_saved_matches_and_checks_its_forward():
    """The backward that reuses its forward's workspace state gives the same
    bits as the one that recomputes it, also after another backward in
    between; on a workspace whose last forward had another input it records
    LB_ERR_PLAN."""
    rng = inputs.rng_for(110)
    d_in, d_out, rs, T = 512, 384, (32, 24), 96
    layer = _train_case(rng, d_in, d_out, rs)
    TL = lb.TrainLinear(layer, DEV)
    x = torch.from_numpy(rng.standard_normal((T, d_in)).astype(np.float32)).to(DEV)
    x2 = torch.from_numpy(rng.standard_normal((T, d_in)).astype(np.float32)).to(DEV)
    dy = torch.from_numpy(rng.standard_normal((T, d_out)).astype(np.float32)).to(DEV)
    ws = TL.workspace(T, DEV)
    lb.train_forward(TL, x, ws=ws)
    g_ref, dx_ref = lb.train_backward(TL, x, dy, ws=ws)
    g_sav, dx_sav = lb.train_backward(TL, x, dy, ws=ws, saved=True)
    torch.cuda.synchronize()
    assert lb.poll_error(ws) == lb.LB_OK
    assert torch.equal(dx_sav, dx_ref)
    for p in range(len(rs)):
        for key in ("du", "dv", "dg", "dl", "dh"):
            assert torch.equal(g_sav[p][key], g_ref[p][key]), (p, key)
    lb.train_forward(TL, x2, ws=ws)
    lb.train_backward(TL, x, dy, ws=ws, saved=True)
    assert lb.poll_error(ws) == lb.LB_ERR_PLAN


# ------------------------------------------------------------------ stack


def run_stack(layers, x0, head_dim):
    S = lb.DeviceStack(layers, head_dim, DEV)
    x = lb.bf16_tensor(x0, DEV)
    out = torch.full((S.d_model,), float("nan"), device=DEV)
    q = torch.full((S.n_layers, S.d_model), float("nan"), device=DEV)
    kv = torch.full((S.n_layers, 2, S.d_kv), float("nan"), device=DEV)
    ws = S.prepare()
    lb.stack_forward(S, x, out=out, q_out=q, kv_out=kv, ws=ws)
    assert lb.poll_error(ws) == lb.LB_OK
    return (out.cpu().numpy().astype(np.float64), q.cpu().numpy().astype(np.float64),
            kv.cpu().numpy().astype(np.float64))


def check_stack(got, ref):
    out, q, kv = got
    r_out, r_q, r_kv = ref
    for g, r in ((out, r_out), (q, r_q), (kv, r_kv)):
        assert np.all(np.isfinite(g))
    assert rel(out, r_out) <= TOL_FP32, rel(out, r_out)
    for l in range(q.shape[0]):
        assert rel(q[l], r_q[l]) <= TOL_FP32, (l, rel(q[l], r_q[l]))
        assert rel(kv[l, 0], r_kv[l, 0]) <= TOL_FP32, (l, "k")
        assert rel(kv[l, 1], r_kv[l, 1]) <= TOL_FP32, (l, "v")


def test_stack_small():
    layers, x0 = inputs.make_stack(n_layers=3, d_model=1024, d_kv=256, d_ff=2048, r_qo=48,
                                   r_kv=16, r_mlp=64, head_dim=64, config_id=102)
    check_stack(run_stack(layers, x0, 64), oracle.stack_forward(layers, x0, head_dim=64))


def test_stack_ragged_slices():
    """d_model / 32 and d_ff / 32 not multiples of the CTA count; one path."""
    layers, x0 = inputs.make_stack(n_layers=2, d_model=640, d_kv=160, d_ff=1696, r_qo=40,
                                   r_kv=8, r_mlp=56, head_dim=32, config_id=103)
    for L in layers:
        L["paths"] = L["paths"][:1]
    check_stack(run_stack(layers, x0, 32), oracle.stack_forward(layers, x0, head_dim=32))


def test_stack_mixed_paths_and_ranks():
    """Per-linear path counts and unequal path ranks (Eq. 6 allows both): one-path
    linears split their words across the half-warps, a gate of two paths meets an
    up of one, and paths of unequal rank run side by side with masked words."""
    rng = inputs.rng_for(104)
    d, dkv, dff = 512, 128, 1024
    spec = [(d, d, [40]), (d, dkv, [8, 24]), (d, dkv, [16, 8]), (d, d, [48, 16]),
            (d, dff, [56, 24]), (d, dff, [40]), (dff, d, [32, 64])]
    layers = []
    for _ in range(2):
        for di, do, rs in spec:
            c = inputs.unit_gain_scale(di, sum(rs) // len(rs), len(rs))
            layers.append(inputs.make_linear(rng, di, do, rs, len(rs), c))
    x0 = inputs.bf16_normal(rng, (d,))
    check_stack(run_stack(layers, x0, 64), oracle.stack_forward(layers, x0, head_dim=64))


def test_stack_workspace_reuse_and_plan_check():
    """Back-to-back launches on one prepared workspace agree (the launch leaves
    it clean); a workspace prepared for other linears is refused on the
    device with LB_ERR_PLAN and no output is written."""
    layers, x0 = inputs.make_stack(n_layers=2, d_model=512, d_kv=128, d_ff=1024, r_qo=32,
                                   r_kv=8, r_mlp=48, head_dim=64, config_id=104)
    S = lb.DeviceStack(layers, 64, DEV)
    x = lb.bf16_tensor(x0, DEV)
    ws = S.prepare()
    outs = []
    for _ in range(3):
        out, _, _ = lb.stack_forward(S, x, ws=ws)
        outs.append(out.cpu().numpy().astype(np.float64))
    assert lb.poll_error(ws) == lb.LB_OK
    ref = oracle.stack_forward(layers, x0, head_dim=64)[0]
    for o in outs:
        assert rel(o, ref) <= TOL_FP32
    other_layers, _ = inputs.make_stack(n_layers=2, d_model=512, d_kv=128, d_ff=1024, r_qo=32,
                                        r_kv=8, r_mlp=48, head_dim=64, config_id=105)
    S2 = lb.DeviceStack(other_layers, 64, DEV)
    out2 = torch.full((512,), float("nan"), device=DEV)
    lb.stack_forward(S2, x, out=out2, want_q=False, want_kv=False, ws=ws)
    assert lb.poll_error(ws) == lb.LB_ERR_PLAN
    assert torch.isnan(out2).all()
    S2.prepare(ws)
    lb.stack_forward(S2, x, out=out2, want_q=False, want_kv=False, ws=ws)
    assert lb.poll_error(ws) == lb.LB_OK
    assert rel(out2.cpu().numpy(), oracle.stack_forward(other_layers, x0, head_dim=64)[0]) <= TOL_FP32


def test_stack_70b_full():
    """The full 80-layer Llama2-70B-shaped stack, every output checked."""
    layers, x0 = inputs.config5()
    check_stack(run_stack(layers, x0, 128), oracle.stack_forward(layers, x0, head_dim=128))


def test_stack_cluster_pairs():
    """The two-CTA cluster variant (LB_STACK_CLUSTER=2: the stage-1 partials of
    each CTA pair meet in distributed shared memory and one contribution per
    pair goes to the exchange) against the oracle, on the 80-layer 70B shape
    and on a small stack with ragged slices; a workspace prepared for one
    cluster size is refused by the other with LB_ERR_PLAN."""
    old = os.environ.get("LB_STACK_CLUSTER")
    try:
        os.environ["LB_STACK_CLUSTER"] = "2"
        layers, x0 = inputs.config5()
        check_stack(run_stack(layers, x0, 128), oracle.stack_forward(layers, x0, head_dim=128))
        layers, x0 = inputs.make_stack(n_layers=2, d_model=640, d_kv=160, d_ff=1696, r_qo=40,
                                       r_kv=8, r_mlp=56, head_dim=32, config_id=103)
        check_stack(run_stack(layers, x0, 32), oracle.stack_forward(layers, x0, head_dim=32))
        S = lb.DeviceStack(layers, 32, DEV)
        ws = S.prepare()
        os.environ["LB_STACK_CLUSTER"] = "1"
        out = torch.full((S.d_model,), float("nan"), device=DEV)
        lb.stack_forward(S, lb.bf16_tensor(x0, DEV), out=out, want_q=False, want_kv=False, ws=ws)
        assert lb.poll_error(ws) == lb.LB_ERR_PLAN
        assert torch.isnan(out).all()
    finally:
        if old is None:
            os.environ.pop("LB_STACK_CLUSTER", None)
        else:
            os.environ["LB_STACK_CLUSTER"] = old


def test_fused_launch_reuses_workspace():
    """From four token tiles on, the forward (and each of latent / expand) is
    one cooperative launch whose grid barriers count on workspace words 1 and
    2.  Repeated calls on one workspace give bit-identical outputs and leave
    both words at zero; after a timed-out wait and its poll (which clears
    them) the launch works again."""
    rng = inputs.rng_for(108, salt=0)
    # 4 token tiles x 4 column tiles: stage 1 is split into K slices, so the
    # launch runs three grid barriers (expansion, slices, stage 2)
    T, d_in, d_out = 512, 4096, 2048
    L = inputs.make_linear(rng, d_in, d_out, [512, 512], 2, 0.05)
    x = inputs.bf16_normal(rng, (T, d_in))
    D = lb.DeviceLinear(L, DEV)
    ws = lb.new_workspace(lb.workspace_size(D, T), DEV)
    xin = lb.bf16_tensor(x, DEV)

    def forward():
        y = torch.full((T, d_out), float("nan"), dtype=torch.float32, device=DEV)
        lb.linear_forward(D, xin, y=y, ws=ws)
        torch.cuda.synchronize()
        return y

    def words():
        return ws[:16].view(torch.int32).cpu().tolist()

    y0 = forward()
    rows = np.array([0, 1, 127, 128, 300, T - 1])
    check(y0.cpu().numpy().astype(np.float64)[rows], oracle.forward_factored(L, x[rows]),
          torch.float32, 1e-3)
    assert words()[:3] == [0, 0, 0]
    z = torch.empty((T, 1024), dtype=torch.float16, device=DEV)
    for _ in range(3):
        lb.linear_latent(D, xin, z=z, ws=ws)
        yc = torch.empty((T, d_out), dtype=torch.float32, device=DEV)
        lb.linear_expand(D, z, y=yc, ws=ws)
        torch.cuda.synchronize()
        assert torch.equal(yc, y0)
        assert torch.equal(forward(), y0)
    assert lb.poll_error(ws) == lb.LB_OK
    assert words()[:3] == [0, 0, 0]
    lb.selftest_wait_timeout(ws)
    y = torch.full((T, d_out), float("nan"), dtype=torch.float32, device=DEV)
    lb.linear_forward(D, xin, y=y, ws=ws)
    assert lb.poll_error(ws) == lb.LB_ERR_TIMEOUT
    assert torch.isnan(y).all(), "a kernel wrote outputs while the error word was set"
    assert words()[:3] == [0, 0, 0]
    assert torch.equal(forward(), y0)
    assert lb.poll_error(ws) == lb.LB_OK


# ------------------------------------------------------------------ bounded waits


def test_grid_wait_times_out_and_is_sticky():
    """A wait nobody releases gives up after its limit with LB_ERR_TIMEOUT; until
    polled, kernels on that workspace return without writing; after the poll
    the workspace works again."""
    L, x = inputs.config2(1)
    D = lb.DeviceLinear(L, DEV)
    ws = lb.new_workspace(lb.workspace_size(D, 1), DEV)
    lb.selftest_wait_timeout(ws)
    xin = lb.bf16_tensor(x, DEV)
    y = torch.full((1, D.d_out), float("nan"), dtype=torch.float32, device=DEV)
    lb.linear_forward(D, xin, y=y, ws=ws)
    assert lb.poll_error(ws) == lb.LB_ERR_TIMEOUT
    assert torch.isnan(y).all(), "a kernel wrote outputs while the error word was set"
    assert lb.poll_error(ws) == lb.LB_OK
    lb.linear_forward(D, xin, y=y, ws=ws)
    torch.cuda.synchronize()
    check(y.cpu().numpy().astype(np.float64), oracle.forward_factored(L, x), torch.float32)


def test_exchange_diagnostic_runs_clean():
    """The exchange-chain diagnostic (the stack's all-reduce with nothing around
    it) completes every round in both encodings, with and without the two-CTA
    clusters, and
    rejects sizes it cannot hold."""
    for words in (1, 2):
        for cluster in (1, 2):
            ws = lb.selftest_exchange(40, [65, 384, 1281, 640], cluster, words, device=DEV)
            assert lb.poll_error(ws) == lb.LB_OK
    arr = (ctypes.c_int32 * 1)(4096)
    assert lb.lib().littlebit_selftest_exchange(4, arr, 1, 2, 1, ws.data_ptr(), ws.numel(),
                                                None) == lb.LB_ERR_INVALID_ARG
    arr = (ctypes.c_int32 * 1)(64)
    assert lb.lib().littlebit_selftest_exchange(4, arr, 1, 1, 3, ws.data_ptr(), ws.numel(),
                                                None) == lb.LB_ERR_INVALID_ARG
