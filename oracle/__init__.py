"""CPU oracle for the LittleBit linear forward (arXiv 2506.13771).

TEST INFRASTRUCTURE ONLY.  This package is the independent fp64 reference the
CUDA path is checked against.  Only ``tests/``, ``__graft_entry__.smoke()`` and
the ``cpu_baseline`` / ``--impl reference`` leg of ``bench.py`` may import it;
the product package never does, and this package never imports the product.

The arithmetic lives in ``lb_oracle.c`` (plain C, fp64, one function per
definition of the paper: Eq. 2 packing, Eq. 4-6 dense weight, Prop. 1 factored
forward, latent states, Dual-SVID initialisation, App. E bit accounting).  This module only builds it with gcc and
marshals numpy arrays through ctypes.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "lb_oracle.c")
_HDR = os.path.join(_HERE, "lb_oracle.h")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liblboracle.so")

_lib = None
_lock = threading.Lock()


def build(force: bool = False) -> str:
    """Compile lb_oracle.c into _build/liblboracle.so with gcc (+OpenMP)."""
    os.makedirs(_BUILD, exist_ok=True)
    newest_src = max(os.path.getmtime(_SRC), os.path.getmtime(_HDR))
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= newest_src):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-std=c11", "-O2", "-fPIC", "-shared", "-fopenmp",
           "-ffp-contract=off", "-Wall", "-Wextra", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


class Path(ctypes.Structure):
    _fields_ = [("r", ctypes.c_int32),
                ("v_words", ctypes.c_void_p),
                ("u_words", ctypes.c_void_p),
                ("g", ctypes.c_void_p),
                ("l", ctypes.c_void_p),
                ("h", ctypes.c_void_p)]


class Linear(ctypes.Structure):
    _fields_ = [("d_in", ctypes.c_int32),
                ("d_out", ctypes.c_int32),
                ("n_paths", ctypes.c_int32),
                ("path", Path * 2)]


def _bind(lib):
    d, i64, u16, vp = ctypes.c_double, ctypes.c_int64, ctypes.c_uint16, ctypes.c_void_p
    lib.lbo_half_to_double.argtypes = [u16]
    lib.lbo_half_to_double.restype = d
    lib.lbo_bf16_to_double.argtypes = [u16]
    lib.lbo_bf16_to_double.restype = d
    for name in ("lbo_pack_u", "lbo_pack_v"):
        getattr(lib, name).argtypes = [vp, i64, i64, vp]
        getattr(lib, name).restype = ctypes.c_int
    for name in ("lbo_unpack_u", "lbo_unpack_v"):
        getattr(lib, name).argtypes = [vp, i64, i64, vp]
        getattr(lib, name).restype = None
    lib.lbo_forward_dense.argtypes = [ctypes.POINTER(Linear), vp, i64, vp]
    lib.lbo_forward_dense.restype = ctypes.c_int
    lib.lbo_forward_factored.argtypes = [ctypes.POINTER(Linear), vp, i64, vp]
    lib.lbo_forward_factored.restype = ctypes.c_int
    lib.lbo_apply_factored.argtypes = [ctypes.POINTER(Linear), vp, i64, vp, vp]
    lib.lbo_apply_factored.restype = ctypes.c_int
    lib.lbo_latent.argtypes = [ctypes.POINTER(Linear), vp, i64, vp]
    lib.lbo_latent.restype = ctypes.c_int
    lib.lbo_expand.argtypes = [ctypes.POINTER(Linear), vp, i64, vp]
    lib.lbo_expand.restype = None
    lib.lbo_svd_top.argtypes = [vp, i64, i64, i64, vp, vp, vp]
    lib.lbo_svd_top.restype = ctypes.c_int
    lib.lbo_dual_svid_path.argtypes = [vp, i64, i64, i64, vp, vp, vp, vp, vp]
    lib.lbo_dual_svid_path.restype = ctypes.c_int
    lib.lbo_path_weight.argtypes = [vp, vp, vp, vp, vp, i64, i64, i64, vp]
    lib.lbo_path_weight.restype = None
    lib.lbo_train_forward.argtypes = [ctypes.POINTER(TrainLinear), vp, i64, vp, ctypes.c_int]
    lib.lbo_train_forward.restype = ctypes.c_int
    lib.lbo_train_backward.argtypes = [ctypes.POINTER(TrainLinear), vp, vp, i64, d, ctypes.c_int,
                                       ctypes.POINTER(TrainGrad), vp]
    lib.lbo_train_backward.restype = ctypes.c_int
    lib.lbo_stack_forward.argtypes = [ctypes.POINTER(Linear), ctypes.c_int32, ctypes.c_int32,
                                      vp, vp, vp, vp]
    lib.lbo_stack_forward.restype = ctypes.c_int
    lib.lbo_round_bf16.argtypes = [d]
    lib.lbo_round_bf16.restype = d
    lib.lbo_rope.argtypes = [vp, i64, i64, d]
    lib.lbo_rope.restype = None
    i32 = ctypes.c_int32
    lib.lbo_decoder_step.argtypes = [ctypes.POINTER(Linear), i32, i32, i32, i32, d, i64, i64, i32,
                                     vp, vp, vp, vp, vp, vp]
    lib.lbo_decoder_step.restype = ctypes.c_int
    lib.lbo_bpw.argtypes = [i64, i64, i64, ctypes.c_int32]
    lib.lbo_bpw.restype = d
    lib.lbo_rank_for_bpw.argtypes = [d, i64, i64, ctypes.c_int32]
    lib.lbo_rank_for_bpw.restype = d
    lib.lbo_flops.argtypes = [i64, i64, i64, i64, ctypes.c_int32]
    lib.lbo_flops.restype = d
    lib.lbo_set_threads.argtypes = [ctypes.c_int32]
    lib.lbo_set_threads.restype = None
    lib.lbo_get_threads.argtypes = []
    lib.lbo_get_threads.restype = ctypes.c_int32
    return lib


def _ptr(a: np.ndarray) -> int:
    return a.ctypes.data


def _c(a, dtype) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=dtype)


class _Holder:
    """Keeps the numpy buffers referenced by a ctypes Linear alive."""

    def __init__(self, layer: dict):
        self.keep = []
        self.c = Linear()
        self.c.d_in = int(layer["d_in"])
        self.c.d_out = int(layer["d_out"])
        paths = layer["paths"]
        self.c.n_paths = len(paths)
        for p, P in enumerate(paths):
            arrs = {
                "v_words": _c(P["v_words"], np.uint32),
                "u_words": _c(P["u_words"], np.uint32),
                "g": _c(P["g"], np.uint16),
                "l": _c(P["l"], np.uint16),
                "h": _c(P["h"], np.uint16),
            }
            self.keep.append(arrs)
            cp = self.c.path[p]
            cp.r = int(P["r"])
            for k, a in arrs.items():
                setattr(cp, k, _ptr(a))


class TrainPath(ctypes.Structure):
    _fields_ = [("r", ctypes.c_int32), ("u", ctypes.c_void_p), ("v", ctypes.c_void_p),
                ("g", ctypes.c_void_p), ("l", ctypes.c_void_p), ("h", ctypes.c_void_p)]


class TrainLinear(ctypes.Structure):
    _fields_ = [("d_in", ctypes.c_int32), ("d_out", ctypes.c_int32), ("n_paths", ctypes.c_int32),
                ("path", TrainPath * 2)]


class TrainGrad(ctypes.Structure):
    _fields_ = [("du", ctypes.c_void_p), ("dv", ctypes.c_void_p), ("dg", ctypes.c_void_p),
                ("dl", ctypes.c_void_p), ("dh", ctypes.c_void_p)]


class _TrainHolder:
    """Keeps the fp64 arrays referenced by a ctypes TrainLinear alive."""

    def __init__(self, layer: dict):
        self.keep = []
        self.c = TrainLinear()
        self.c.d_in, self.c.d_out = int(layer["d_in"]), int(layer["d_out"])
        self.c.n_paths = len(layer["paths"])
        for p, P in enumerate(layer["paths"]):
            arrs = {k: _c(P[k], np.float64) for k in ("u", "v", "g", "l", "h")}
            self.keep.append(arrs)
            cp = self.c.path[p]
            cp.r = int(P["r"])
            for k, a in arrs.items():
                setattr(cp, k, _ptr(a))


class Oracle:
    """The oracle functions bound to one compiled copy of lb_oracle.c."""

    def __init__(self, lib_path: str | None = None):
        self.lib = _bind(ctypes.CDLL(lib_path or build()))

    # ------------------------------------------------------------ formats
    def half_to_double(self, bits: int) -> float:
        """IEEE binary16 bit pattern -> value (from the format definition)."""
        return self.lib.lbo_half_to_double(int(bits))

    def bf16_to_double(self, bits: int) -> float:
        """bfloat16 bit pattern -> value (from the format definition)."""
        return self.lib.lbo_bf16_to_double(int(bits))

    # ------------------------------------------------------------ packing (Eq. 2)
    def pack_u(self, signs: np.ndarray) -> np.ndarray:
        """U_sign [d_out][r] (+-1 int8) -> words [d_out][ceil(r/32)]."""
        s = _c(signs, np.int8)
        rows, cols = s.shape
        out = np.zeros((rows, (cols + 31) // 32), dtype=np.uint32)
        if self.lib.lbo_pack_u(_ptr(s), rows, cols, _ptr(out)) != 0:
            raise ValueError("signs must be +1 or -1")
        return out

    def pack_v(self, signs: np.ndarray) -> np.ndarray:
        """V_sign [d_in][r] (+-1 int8) -> words [ceil(d_in/32)][r]."""
        s = _c(signs, np.int8)
        rows, cols = s.shape
        out = np.zeros(((rows + 31) // 32, cols), dtype=np.uint32)
        if self.lib.lbo_pack_v(_ptr(s), rows, cols, _ptr(out)) != 0:
            raise ValueError("signs must be +1 or -1")
        return out

    def unpack_u(self, words: np.ndarray, rows: int, cols: int) -> np.ndarray:
        w = _c(words, np.uint32)
        out = np.zeros((rows, cols), dtype=np.int8)
        self.lib.lbo_unpack_u(_ptr(w), rows, cols, _ptr(out))
        return out

    def unpack_v(self, words: np.ndarray, rows: int, cols: int) -> np.ndarray:
        w = _c(words, np.uint32)
        out = np.zeros((rows, cols), dtype=np.int8)
        self.lib.lbo_unpack_v(_ptr(w), rows, cols, _ptr(out))
        return out

    # ------------------------------------------------------------ forward
    def forward_dense(self, layer: dict, x_bf16: np.ndarray) -> np.ndarray:
        """Eq. 4-6 then Y = X W^T, fp64.  x_bf16: uint16 bit patterns [T][d_in]."""
        hold = _Holder(layer)
        x = _c(x_bf16, np.uint16)
        y = np.zeros((x.shape[0], layer["d_out"]), dtype=np.float64)
        if self.lib.lbo_forward_dense(ctypes.byref(hold.c), _ptr(x), x.shape[0], _ptr(y)):
            raise MemoryError("oracle dense forward failed")
        return y

    def forward_factored(self, layer: dict, x_bf16: np.ndarray) -> np.ndarray:
        """Prop. 1 per path, paths summed (Eq. 6), fp64."""
        hold = _Holder(layer)
        x = _c(x_bf16, np.uint16)
        y = np.zeros((x.shape[0], layer["d_out"]), dtype=np.float64)
        if self.lib.lbo_forward_factored(ctypes.byref(hold.c), _ptr(x), x.shape[0], _ptr(y)):
            raise MemoryError("oracle factored forward failed")
        return y

    def apply_factored(self, layer: dict, x: np.ndarray, want_t: bool = False):
        """Prop. 1 on an fp64 input [T][d_in]; optionally also the stage-1 t_p."""
        hold = _Holder(layer)
        X = _c(x, np.float64)
        T = X.shape[0]
        y = np.zeros((T, layer["d_out"]), dtype=np.float64)
        rs = [int(P["r"]) for P in layer["paths"]]
        t = np.zeros(T * sum(rs), dtype=np.float64) if want_t else None
        if self.lib.lbo_apply_factored(ctypes.byref(hold.c), _ptr(X), T, _ptr(y),
                                       _ptr(t) if want_t else None):
            raise MemoryError("oracle factored forward failed")
        if not want_t:
            return y
        ts, off = [], 0
        for r in rs:
            ts.append(t[off:off + T * r].reshape(T, r))
            off += T * r
        return y, ts

    def latent(self, layer: dict, x_bf16: np.ndarray) -> np.ndarray:
        """Latent states z [T][r_0 + r_1] (l_p . (X . g_p) V_p,sign per path), fp64."""
        hold = _Holder(layer)
        x = _c(x_bf16, np.uint16)
        n1 = sum(int(P["r"]) for P in layer["paths"])
        z = np.zeros((x.shape[0], n1), dtype=np.float64)
        if self.lib.lbo_latent(ctypes.byref(hold.c), _ptr(x), x.shape[0], _ptr(z)):
            raise MemoryError("oracle latent failed")
        return z

    def expand(self, layer: dict, z: np.ndarray) -> np.ndarray:
        """Y [T][d_out] = sum_p h_p . (U_p,sign z_p) from latents in latent()'s layout."""
        hold = _Holder(layer)
        Z = _c(z, np.float64)
        n1 = sum(int(P["r"]) for P in layer["paths"])
        assert Z.ndim == 2 and Z.shape[1] == n1
        y = np.zeros((Z.shape[0], layer["d_out"]), dtype=np.float64)
        self.lib.lbo_expand(ctypes.byref(hold.c), _ptr(Z), Z.shape[0], _ptr(y))
        return y

    def stack_forward(self, layers: list, x0_bf16: np.ndarray, head_dim: int = 128,
                      want_q: bool = True, want_kv: bool = True):
        """Decode step at position 0 through n_layers x (q,k,v,o,gate,up,down);
        returns (out [d], q [n_layers][d] or None, kv [n_layers][2][d_kv] or None)."""
        assert len(layers) % 7 == 0
        n_layers = len(layers) // 7
        holders = [_Holder(L) for L in layers]
        arr = (Linear * len(layers))(*[h.c for h in holders])
        x0 = _c(x0_bf16, np.uint16)
        d = layers[0]["d_in"]
        out = np.zeros(d, dtype=np.float64)
        q = np.zeros((n_layers, d), dtype=np.float64) if want_q else None
        kv = np.zeros((n_layers, 2, layers[1]["d_out"]), dtype=np.float64) if want_kv else None
        if self.lib.lbo_stack_forward(arr, n_layers, int(head_dim), _ptr(x0), _ptr(out),
                                      _ptr(q) if want_q else None,
                                      _ptr(kv) if want_kv else None):
            raise MemoryError("oracle stack forward failed")
        return out, q, kv

    # ------------------------------------------------------------ decode step at position p (App. I.3)
    def round_bf16(self, v) -> np.ndarray:
        """The nearest bf16 value of each element (ties to even), as float64."""
        v = np.asarray(v, dtype=np.float64)
        return np.array([self.lib.lbo_round_bf16(float(e)) for e in v.ravel()]).reshape(v.shape)

    def rope(self, x: np.ndarray, p: int, base: float = 10000.0) -> np.ndarray:
        """One head rotated to position p (half-split pairing)."""
        y = _c(np.array(x, dtype=np.float64), np.float64)
        self.lib.lbo_rope(_ptr(y), y.shape[0], int(p), float(base))
        return y

    def decoder_step(self, layers: list, shape: dict, pos: int, x_bf16: np.ndarray,
                     kcache: np.ndarray, vcache: np.ndarray, round_inputs: bool = True,
                     want_attn: bool = False, want_qk: bool = False):
        """One decode step at position pos; kcache / vcache [n_layers][max_pos][d_kv]
        (float64, updated in place at row pos).  shape: n_heads, n_kv_heads,
        head_dim, rope_base.  Returns (out [d], attn [n_layers][d] or None,
        qk [n_layers][d + d_kv] or None)."""
        assert len(layers) % 7 == 0
        n_layers = len(layers) // 7
        holders = [_Holder(L) for L in layers]
        arr = (Linear * len(layers))(*[h.c for h in holders])
        H, G, D = shape["n_heads"], shape["n_kv_heads"], shape["head_dim"]
        d, dkv = H * D, G * D
        assert kcache.dtype == np.float64 and kcache.flags.c_contiguous
        assert vcache.dtype == np.float64 and vcache.flags.c_contiguous
        assert kcache.shape == vcache.shape and kcache.shape[0] == n_layers and kcache.shape[2] == dkv
        x = _c(x_bf16, np.uint16)
        out = np.zeros(d, dtype=np.float64)
        attn = np.zeros((n_layers, d)) if want_attn else None
        qk = np.zeros((n_layers, d + dkv)) if want_qk else None
        if self.lib.lbo_decoder_step(arr, n_layers, H, G, D, float(shape.get("rope_base", 10000.0)),
                                     int(pos), kcache.shape[1], 1 if round_inputs else 0,
                                     _ptr(x), _ptr(kcache), _ptr(vcache), _ptr(out),
                                     _ptr(attn) if want_attn else None,
                                     _ptr(qk) if want_qk else None):
            raise ValueError("decoder_step: position out of range, bad shape or no memory")
        return out, attn, qk

    # ------------------------------------------------------------ Dual-SVID (Sec. 3.2, 3.3)
    def svd_top(self, A: np.ndarray, r: int):
        """The r largest singular triples of A by one-sided Jacobi: (s[r], U[m][r], V[n][r])."""
        A = _c(A, np.float64)
        m, n = A.shape
        s = np.zeros(r)
        U = np.zeros((m, r))
        V = np.zeros((n, r))
        if self.lib.lbo_svd_top(_ptr(A), m, n, r, _ptr(s), _ptr(U), _ptr(V)):
            raise ValueError("svd_top: rank out of range or no memory")
        return s, U, V

    def dual_svid_path(self, R: np.ndarray, r: int):
        """Dual-SVID of one path (Sec. 3.2): (usign [d_out][r], vsign [d_in][r], h, g, l) in fp64."""
        R = _c(R, np.float64)
        d_out, d_in = R.shape
        us = np.zeros((d_out, r), np.int8)
        vs = np.zeros((d_in, r), np.int8)
        h, g, l = np.zeros(d_out), np.zeros(d_in), np.zeros(r)
        if self.lib.lbo_dual_svid_path(_ptr(R), d_out, d_in, r, _ptr(us), _ptr(vs), _ptr(h),
                                       _ptr(g), _ptr(l)):
            raise ValueError("dual_svid_path: rank out of range or no memory")
        return us, vs, h, g, l

    def path_weight(self, us, vs, h, g, l) -> np.ndarray:
        """W_hat = diag(h) U_sign diag(l) V_sign^T diag(g) (Eq. 4), fp64."""
        us, vs = _c(us, np.int8), _c(vs, np.int8)
        h, g, l = _c(h, np.float64), _c(g, np.float64), _c(l, np.float64)
        d_out, r = us.shape
        d_in = vs.shape[0]
        W = np.zeros((d_out, d_in))
        self.lib.lbo_path_weight(_ptr(us), _ptr(vs), _ptr(h), _ptr(g), _ptr(l), d_out, d_in, r,
                                 _ptr(W))
        return W

    def dual_svid(self, W: np.ndarray, ranks) -> dict:
        """Dual-SVID initialisation with Residual Compensation (Sec. 3.2, 3.3): path 0 from
        W, each further path from the residual W - sum of the previous paths' W_hat, where a
        path's W_hat uses its scales as stored (rounded to fp16, nearest even).  Returns a
        layer dict (packed words, fp16 scale bits) plus 'signs' (usign, vsign per path)."""
        W = _c(W, np.float64)
        R = W.copy()
        paths, signs = [], []
        for r in ranks:
            us, vs, h, g, l = self.dual_svid_path(R, int(r))
            h16, g16, l16 = (np.asarray(a, np.float64).astype(np.float16) for a in (h, g, l))
            paths.append({"r": int(r), "u_words": self.pack_u(us), "v_words": self.pack_v(vs),
                          "h": h16.view(np.uint16), "g": g16.view(np.uint16),
                          "l": l16.view(np.uint16)})
            signs.append((us, vs))
            R = R - self.path_weight(us, vs, h16.astype(np.float64), g16.astype(np.float64),
                                     l16.astype(np.float64))
        return {"d_in": W.shape[1], "d_out": W.shape[0], "paths": paths, "signs": signs}

    # ------------------------------------------------------------ QAT with SmoothSign
    def train_forward(self, layer: dict, x: np.ndarray, relaxed: bool = False) -> np.ndarray:
        """Y = sum_p Prop. 1 with sign(U), sign(V) of the latent factors (identity if relaxed)."""
        hold = _TrainHolder(layer)
        X = _c(x, np.float64)
        Y = np.zeros((X.shape[0], layer["d_out"]))
        if self.lib.lbo_train_forward(ctypes.byref(hold.c), _ptr(X), X.shape[0], _ptr(Y),
                                      1 if relaxed else 0):
            raise MemoryError("oracle train forward failed")
        return Y

    def train_backward(self, layer: dict, x: np.ndarray, dy: np.ndarray, k: float = 100.0,
                       relaxed: bool = False):
        """Gradients of sum(Y . dY): (list of per-path dicts du, dv, dg, dl, dh; dX)."""
        hold = _TrainHolder(layer)
        X, DY = _c(x, np.float64), _c(dy, np.float64)
        T = X.shape[0]
        grads = (TrainGrad * len(layer["paths"]))()
        out = []
        for p, P in enumerate(layer["paths"]):
            r = int(P["r"])
            g = {"du": np.zeros((layer["d_out"], r)), "dv": np.zeros((layer["d_in"], r)),
                 "dg": np.zeros(layer["d_in"]), "dl": np.zeros(r), "dh": np.zeros(layer["d_out"])}
            out.append(g)
            for key, a in g.items():
                setattr(grads[p], key, _ptr(a))
        dX = np.zeros((T, layer["d_in"]))
        if self.lib.lbo_train_backward(ctypes.byref(hold.c), _ptr(X), _ptr(DY), T, float(k),
                                       1 if relaxed else 0, grads, _ptr(dX)):
            raise MemoryError("oracle train backward failed")
        return out, dX

    # ------------------------------------------------------------ accounting (App. E, I.1)
    def bpw(self, d_out: int, d_in: int, r: int, n_paths: int = 2) -> float:
        return self.lib.lbo_bpw(d_out, d_in, r, n_paths)

    def rank_for_bpw(self, b: float, d_out: int, d_in: int, n_paths: int = 2) -> float:
        return self.lib.lbo_rank_for_bpw(b, d_out, d_in, n_paths)

    def flops(self, T: int, d_out: int, d_in: int, r: int, n_paths: int = 2) -> float:
        return self.lib.lbo_flops(T, d_out, d_in, r, n_paths)

    def set_threads(self, n: int) -> None:
        self.lib.lbo_set_threads(int(n))

    def get_threads(self) -> int:
        return int(self.lib.lbo_get_threads())


def default() -> Oracle:
    """The oracle built from the committed lb_oracle.c (built on first use)."""
    global _lib
    with _lock:
        if _lib is None:
            _lib = Oracle()
        return _lib


def _forward(name):
    def f(*args, **kwargs):
        return getattr(default(), name)(*args, **kwargs)
    f.__name__ = name
    f.__doc__ = getattr(Oracle, name).__doc__
    return f


for _name in ("half_to_double", "bf16_to_double", "pack_u", "pack_v", "unpack_u", "unpack_v",
              "forward_dense", "forward_factored", "apply_factored", "latent", "expand",
              "svd_top", "dual_svid_path", "path_weight", "dual_svid", "train_forward",
              "train_backward", "stack_forward",
              "bpw", "rank_for_bpw", "flops", "set_threads", "get_threads"):
    globals()[_name] = _forward(_name)
del _name
