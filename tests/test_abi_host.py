"""Host-side checks of the C ABI (no GPU needed): the library builds, loads and
exports every entry point include/littlebit.h declares, and argument
validation answers with status codes before any CUDA call is made."""
import ctypes
import os
import re

import pytest

from paper_2506_13771_gb300 import build as lb_build
from paper_2506_13771_gb300 import littlebit as lb

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include",
                      "littlebit.h")


@pytest.fixture(scope="module")
def L():
    lb_build.build()
    return lb.lib()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(littlebit_\w+)\s*\(", text)))


def test_exports_every_declared_symbol(L):
    names = declared_functions()
    assert len(names) >= 8
    for n in names:
        assert hasattr(L, n), f"{n} declared in littlebit.h but not exported"
    assert sorted(lb.EXPORTED) == names


def test_status_strings(L):
    for code, name in [(lb.LB_OK, "LB_OK"), (lb.LB_ERR_INVALID_ARG, "LB_ERR_INVALID_ARG"),
                       (lb.LB_ERR_UNSUPPORTED, "LB_ERR_UNSUPPORTED"), (lb.LB_ERR_CUDA, "LB_ERR_CUDA"),
                       (lb.LB_ERR_TIMEOUT, "LB_ERR_TIMEOUT"), (lb.LB_ERR_WORKSPACE, "LB_ERR_WORKSPACE"),
                       (lb.LB_ERR_PLAN, "LB_ERR_PLAN"), (lb.LB_ERR_RANGE, "LB_ERR_RANGE")]:
        assert lb.status_string(code) == name
    assert lb.status_string(99) == "LB_ERR_UNKNOWN"


FAKE = 0x10000000  # a 16-byte aligned address; never dereferenced on these paths


def fake_linear(d_in=4096, d_out=4096, rs=(64, 64)):
    c = lb.lb_linear()
    c.d_in, c.d_out, c.n_paths = d_in, d_out, len(rs)
    for p, r in enumerate(rs):
        c.path[p].r = r
        for k, f in enumerate(["v_bits", "u_bits", "g", "l", "h"]):
            setattr(c.path[p], f, FAKE + 0x100000 * (5 * p + k))
    return c


def fwd(L, c, T=1, x=FAKE, y=FAKE, dtype=0, ws=FAKE, ws_bytes=1 << 30):
    return L.littlebit_linear_forward(ctypes.byref(c) if c is not None else None, x, T, y, dtype,
                                      ws, ws_bytes, None)


def test_workspace_sizes(L):
    c = fake_linear()
    n1 = L.littlebit_workspace_size(ctypes.byref(c), 1)
    n8 = L.littlebit_workspace_size(ctypes.byref(c), 8)
    assert n1 >= 256 + 4 * 128 and n8 >= 256 + 4 * 8 * 128
    assert n1 % 256 == 0 and n8 % 256 == 0
    assert L.littlebit_workspace_size(None, 1) == 0
    bad = fake_linear(rs=(0, 64))
    assert L.littlebit_workspace_size(ctypes.byref(bad), 1) == 0


def test_forward_argument_validation(L):
    assert fwd(L, None) == lb.LB_ERR_INVALID_ARG
    c = fake_linear()
    assert fwd(L, c, T=-1) == lb.LB_ERR_INVALID_ARG
    assert fwd(L, c, dtype=7) == lb.LB_ERR_INVALID_ARG
    assert fwd(L, c, x=0) == lb.LB_ERR_INVALID_ARG
    assert fwd(L, c, y=FAKE + 4) == lb.LB_ERR_INVALID_ARG          # misaligned output
    assert fwd(L, c, ws=0) == lb.LB_ERR_WORKSPACE
    assert fwd(L, c, ws=FAKE + 16) == lb.LB_ERR_WORKSPACE           # ws must be 256-aligned
    assert fwd(L, c, ws_bytes=64) == lb.LB_ERR_WORKSPACE
    assert fwd(L, c, T=0) == lb.LB_OK                               # no-op
    c3 = fake_linear()
    c3.n_paths = 3
    assert fwd(L, c3) == lb.LB_ERR_INVALID_ARG
    cz = fake_linear(d_in=0)
    assert fwd(L, cz) == lb.LB_ERR_INVALID_ARG
    cmis = fake_linear()
    cmis.path[1].g = FAKE + 2
    assert fwd(L, cmis) == lb.LB_ERR_INVALID_ARG
    cnull = fake_linear()
    cnull.path[0].u_bits = None
    assert fwd(L, cnull) == lb.LB_ERR_INVALID_ARG
    assert fwd(L, fake_linear(d_in=40)) == lb.LB_ERR_UNSUPPORTED    # d_in % 32
    assert fwd(L, fake_linear(rs=(2000, 64))) == lb.LB_ERR_UNSUPPORTED


def test_latent_and_expand_argument_validation(L):
    c = fake_linear()
    lat, exp = L.littlebit_linear_latent, L.littlebit_linear_expand
    ref = ctypes.byref(c)
    assert lat(None, FAKE, 1, FAKE, 0, FAKE, 1 << 30, None) == lb.LB_ERR_INVALID_ARG
    assert lat(ref, FAKE, -1, FAKE, 0, FAKE, 1 << 30, None) == lb.LB_ERR_INVALID_ARG
    assert lat(ref, FAKE, 1, FAKE, 2, FAKE, 1 << 30, None) == lb.LB_ERR_INVALID_ARG  # z dtype
    assert lat(ref, FAKE, 0, FAKE, 0, FAKE, 1 << 30, None) == lb.LB_OK              # T = 0
    assert lat(ref, FAKE, 1, 0, 0, FAKE, 1 << 30, None) == lb.LB_ERR_INVALID_ARG
    assert lat(ref, FAKE, 1, FAKE + 8, 1, FAKE, 1 << 30, None) == lb.LB_ERR_INVALID_ARG
    assert lat(ref, FAKE, 1, FAKE, 0, FAKE, 64, None) == lb.LB_ERR_WORKSPACE
    assert lat(ctypes.byref(fake_linear(d_in=40)), FAKE, 1, FAKE, 0, FAKE, 1 << 30,
               None) == lb.LB_ERR_UNSUPPORTED
    assert exp(None, FAKE, 0, 1, FAKE, 0, FAKE, 1 << 30, None) == lb.LB_ERR_INVALID_ARG
    assert exp(ref, FAKE, 2, 1, FAKE, 0, FAKE, 1 << 30, None) == lb.LB_ERR_INVALID_ARG  # z dtype
    assert exp(ref, FAKE, 0, 1, FAKE, 5, FAKE, 1 << 30, None) == lb.LB_ERR_INVALID_ARG  # y dtype
    assert exp(ref, FAKE, 0, 0, FAKE, 0, FAKE, 1 << 30, None) == lb.LB_OK              # T = 0
    assert exp(ref, FAKE + 4, 0, 1, FAKE, 0, FAKE, 1 << 30, None) == lb.LB_ERR_INVALID_ARG
    assert exp(ref, FAKE, 0, 1, FAKE, 0, FAKE + 16, 1 << 30, None) == lb.LB_ERR_WORKSPACE


def test_dual_svid_argument_validation(L):
    arr = (lb.lb_path_init * 2)()
    for p in range(2):
        arr[p].r = 16
        arr[p].v_bits = arr[p].u_bits = arr[p].g = arr[p].l = arr[p].h = FAKE
    ws_size = L.littlebit_dual_svid_workspace_size
    n = ws_size(256, 384, 2, arr)
    assert n > 256 * 384 * 4                       # holds the residual copy of W
    assert ws_size(256, 384, 3, arr) == 0          # n_paths
    assert ws_size(0, 384, 2, arr) == 0
    assert ws_size(256, 384, 2, None) == 0
    arr[1].r = 300
    assert ws_size(256, 384, 2, arr) == 0          # r > min(d_out, d_in)
    arr[1].r = 16
    svid = L.littlebit_dual_svid
    assert svid(None, 256, 384, 2, arr, 8, FAKE, n, None) == lb.LB_ERR_INVALID_ARG
    assert svid(FAKE + 4, 256, 384, 2, arr, 8, FAKE, n, None) == lb.LB_ERR_INVALID_ARG
    assert svid(FAKE, 256, 384, 2, arr, 0, FAKE, n, None) == lb.LB_ERR_INVALID_ARG   # iters
    assert svid(FAKE, 256, 384, 2, arr, 8, FAKE, n - 256, None) == lb.LB_ERR_WORKSPACE
    assert svid(FAKE, 256, 384, 2, arr, 8, FAKE + 16, n, None) == lb.LB_ERR_WORKSPACE
    arr[0].h = 0
    assert svid(FAKE, 256, 384, 2, arr, 8, FAKE, n, None) == lb.LB_ERR_INVALID_ARG


def test_train_argument_validation(L):
    c = lb.lb_train_linear()
    c.d_in, c.d_out, c.n_paths = 64, 32, 1
    c.path[0].r = 8
    c.path[0].u = c.path[0].v = c.path[0].g = c.path[0].l = c.path[0].h = FAKE
    ref = ctypes.byref(c)
    n = L.littlebit_train_workspace_size(ref, 16)
    assert n > 0
    g = (lb.lb_train_grad * 1)()
    g[0].du = g[0].dv = g[0].dg = g[0].dl = g[0].dh = FAKE
    fwd, bwd = L.littlebit_train_forward, L.littlebit_train_backward
    assert fwd(ref, FAKE, 0, FAKE, FAKE, n, None) == lb.LB_OK                    # T = 0
    assert fwd(ref, FAKE + 4, 16, FAKE, FAKE, n, None) == lb.LB_ERR_INVALID_ARG
    assert fwd(ref, FAKE, 16, FAKE, FAKE, 64, None) == lb.LB_ERR_WORKSPACE
    assert bwd(ref, FAKE, FAKE, 16, 0.0, g, None, FAKE, n, None) == lb.LB_ERR_INVALID_ARG  # k
    assert bwd(ref, FAKE, FAKE, 16, 100.0, None, None, FAKE, n, None) == lb.LB_ERR_INVALID_ARG
    sav = L.littlebit_train_backward_saved
    assert sav(ref, FAKE, FAKE, 16, 0.0, g, None, FAKE, n, None) == lb.LB_ERR_INVALID_ARG
    assert sav(ref, FAKE, FAKE, 16, 100.0, g, None, FAKE, 64, None) == lb.LB_ERR_WORKSPACE
    g[0].dl = 0
    assert bwd(ref, FAKE, FAKE, 16, 100.0, g, None, FAKE, n, None) == lb.LB_ERR_INVALID_ARG
    assert sav(ref, FAKE, FAKE, 16, 100.0, g, None, FAKE, n, None) == lb.LB_ERR_INVALID_ARG
    c.n_paths = 3
    assert L.littlebit_train_workspace_size(ref, 16) == 0


def fake_stack(n_layers=2, d=256, dkv=64, dff=512, rq=16, rk=8, rm=24):
    shapes = [(d, d, rq), (d, dkv, rk), (d, dkv, rk), (d, d, rq), (d, dff, rm), (d, dff, rm),
              (dff, d, rm)]
    arr = (lb.lb_linear * (7 * n_layers))()
    for l in range(n_layers):
        for i, (di, do, r) in enumerate(shapes):
            arr[7 * l + i] = fake_linear(di, do, (r, r))
    return arr


def test_stack_argument_validation(L):
    arr = fake_stack()
    hd = 32
    n = L.littlebit_stack_workspace_size(arr, 2, hd)
    assert n > 256 and n % 256 == 0
    st = L.littlebit_stack_forward
    ok = dict(x0=FAKE, out=FAKE, q=None, kv=None, ws=FAKE, nb=n)

    def call(a=arr, layers=2, head_dim=hd, **kw):
        v = dict(ok, **kw)
        return st(a, layers, head_dim, v["x0"], v["out"], v["q"], v["kv"], v["ws"], v["nb"], None)

    assert call(layers=0) == lb.LB_ERR_INVALID_ARG
    assert call(head_dim=0) == lb.LB_ERR_INVALID_ARG
    assert call(head_dim=48) == lb.LB_ERR_INVALID_ARG               # 256 % 48 != 0
    assert call(x0=0) == lb.LB_ERR_INVALID_ARG
    assert call(kv=FAKE + 8) == lb.LB_ERR_INVALID_ARG
    assert call(q=FAKE + 4) == lb.LB_ERR_INVALID_ARG
    assert call(nb=n - 256) == lb.LB_ERR_WORKSPACE
    broken = fake_stack()
    broken[3] = fake_linear(256, 128, (16, 16))                      # o must be d -> d
    assert L.littlebit_stack_workspace_size(broken, 2, hd) == 0
    assert call(a=broken) == lb.LB_ERR_INVALID_ARG
    uneven = fake_stack()
    uneven[7] = fake_linear(256, 256, (32, 16))                      # layer 1 q differs
    assert call(a=uneven) == lb.LB_ERR_UNSUPPORTED
    prep = L.littlebit_stack_prepare
    assert prep(arr, 2, 0, FAKE, n, None) == lb.LB_ERR_INVALID_ARG
    assert prep(arr, 2, hd, FAKE, n - 256, None) == lb.LB_ERR_WORKSPACE
    assert prep(uneven, 2, hd, FAKE, n, None) == lb.LB_ERR_UNSUPPORTED


def test_decoder_argument_validation(L):
    arr = fake_stack()                 # d 256 = 4 heads x 64, d_kv 64 = 1 kv head
    S = lb.lb_decoder_shape(2, 4, 1, 64, 64, 10000.0)
    n = L.littlebit_decoder_workspace_size(arr, ctypes.byref(S))
    assert n > 256 and n % 256 == 0
    st = L.littlebit_decoder_step
    ok = dict(x=FAKE, k=FAKE, v=FAKE, pos=FAKE, out=FAKE, ws=FAKE, nb=n)

    def call(a=arr, shape=S, **kw):
        v = dict(ok, **kw)
        return st(a, ctypes.byref(shape), v["x"], v["k"], v["v"], v["pos"], v["out"], v["ws"],
                  v["nb"], None)

    def shape(**kw):
        f = dict(n_layers=2, n_heads=4, n_kv_heads=1, head_dim=64, max_pos=64, rope_base=10000.0)
        f.update(kw)
        return lb.lb_decoder_shape(*f.values())

    assert call(shape=shape(n_layers=0)) == lb.LB_ERR_INVALID_ARG
    assert call(shape=shape(n_kv_heads=3)) == lb.LB_ERR_INVALID_ARG     # 4 % 3 != 0
    assert call(shape=shape(n_heads=8, head_dim=32)) == lb.LB_ERR_INVALID_ARG  # 64, 128 or 256
    assert call(shape=shape(max_pos=0)) == lb.LB_ERR_INVALID_ARG
    assert call(shape=shape(max_pos=8193)) == lb.LB_ERR_INVALID_ARG
    assert call(shape=shape(rope_base=1.0)) == lb.LB_ERR_INVALID_ARG
    assert call(x=0) == lb.LB_ERR_INVALID_ARG
    assert call(x=FAKE + 8) == lb.LB_ERR_INVALID_ARG
    assert call(pos=0) == lb.LB_ERR_INVALID_ARG
    assert call(pos=FAKE + 2) == lb.LB_ERR_INVALID_ARG
    assert call(ws=FAKE + 16) == lb.LB_ERR_WORKSPACE
    assert call(nb=n - 256) == lb.LB_ERR_WORKSPACE
    broken = fake_stack()
    broken[1] = fake_linear(256, 128, (8, 8))                         # k must be d -> d_kv
    assert L.littlebit_decoder_workspace_size(broken, ctypes.byref(S)) == 0
    assert call(a=broken) == lb.LB_ERR_UNSUPPORTED
    uneven = fake_stack()
    uneven[7] = fake_linear(256, 256, (32, 16))                       # layer 1 q differs
    assert call(a=uneven) == lb.LB_ERR_UNSUPPORTED
    assert L.littlebit_decoder_poll_error(arr, ctypes.byref(shape(n_layers=0)), FAKE, None) == \
        lb.LB_ERR_INVALID_ARG
    assert L.littlebit_decoder_poll_error(arr, ctypes.byref(S), None, None) == lb.LB_ERR_WORKSPACE


def test_multi_argument_validation(L):
    arr = (lb.lb_linear * 3)(*[fake_linear(1024, 512, (64, 64)) for _ in range(3)])
    n = L.littlebit_multi_workspace_size(arr, 3)
    assert n > 256 and n % 256 == 0
    f = L.littlebit_linear_forward_multi
    assert f(arr, 0, FAKE, FAKE, 0, FAKE, n, None) == lb.LB_ERR_INVALID_ARG
    assert f(arr, 25, FAKE, FAKE, 0, FAKE, n, None) == lb.LB_ERR_INVALID_ARG
    assert f(arr, 3, 0, FAKE, 0, FAKE, n, None) == lb.LB_ERR_INVALID_ARG
    assert f(arr, 3, FAKE, FAKE + 4, 0, FAKE, n, None) == lb.LB_ERR_INVALID_ARG
    assert f(arr, 3, FAKE, FAKE, 2, FAKE, n, None) == lb.LB_ERR_INVALID_ARG
    assert f(arr, 3, FAKE, FAKE, 0, FAKE, n - 256, None) == lb.LB_ERR_WORKSPACE
    assert f(arr, 3, FAKE, FAKE, 0, FAKE + 128, n, None) == lb.LB_ERR_WORKSPACE
    assert L.littlebit_multi_workspace_size(arr, 0) == 0
    assert L.littlebit_multi_workspace_size(arr, 25) == 0


def test_pack_argument_validation(L):
    p = L.littlebit_pack
    assert p(None, 4, 4, lb.LB_PACK_U, FAKE, 4, None, None) == lb.LB_ERR_INVALID_ARG
    assert p(FAKE, 0, 4, lb.LB_PACK_U, FAKE, 4, None, None) == lb.LB_ERR_INVALID_ARG
    assert p(FAKE, 4, 4, 5, FAKE, 4, None, None) == lb.LB_ERR_INVALID_ARG
    assert p(FAKE, 4, 40, lb.LB_PACK_U, FAKE, 7, None, None) == lb.LB_ERR_INVALID_ARG  # needs 8
    assert p(FAKE, 40, 4, lb.LB_PACK_V, FAKE, 7, None, None) == lb.LB_ERR_INVALID_ARG  # needs 8
    assert p(FAKE + 1, 4, 4, lb.LB_PACK_U, FAKE, 4, None, None) == lb.LB_ERR_INVALID_ARG
    assert L.littlebit_poll_error(None, None) == lb.LB_ERR_WORKSPACE
    assert L.littlebit_selftest_wait_timeout(FAKE + 16, None) == lb.LB_ERR_WORKSPACE


def test_product_path_has_no_cpu_fallback(tmp_path):
    """The binding refuses to run without the compiled library."""
    with pytest.raises(OSError):
        lb.lib(str(tmp_path / "liblittlebit.so"))
