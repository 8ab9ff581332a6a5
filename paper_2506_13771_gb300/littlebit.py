"""Python binding of liblittlebit.so (include/littlebit.h).

Argument marshalling only: torch owns device memory and streams, every step
of the LittleBit forward runs in the library's CUDA kernels.  There is no
CPU fallback: if the library is missing or fails to load, ``lib()`` raises.
"""
from __future__ import annotations

import ctypes
import os
import threading

import numpy as np
import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "liblittlebit.so")

(LB_OK, LB_ERR_INVALID_ARG, LB_ERR_UNSUPPORTED, LB_ERR_CUDA, LB_ERR_TIMEOUT, LB_ERR_WORKSPACE,
 LB_ERR_PLAN, LB_ERR_RANGE) = range(8)
LB_OUT_BF16, LB_OUT_FP32 = 0, 1
LB_LATENT_FP32, LB_LATENT_FP16 = 0, 1
LB_PACK_U, LB_PACK_V = 0, 1

EXPORTED = ["littlebit_status_string", "littlebit_pack", "littlebit_workspace_size",
            "littlebit_linear_forward", "littlebit_linear_latent", "littlebit_linear_expand",
            "littlebit_dual_svid_workspace_size", "littlebit_dual_svid",
            "littlebit_train_workspace_size", "littlebit_train_forward",
            "littlebit_train_backward", "littlebit_train_backward_saved",
            "littlebit_stack_workspace_size",
            "littlebit_stack_prepare", "littlebit_stack_forward", "littlebit_poll_error",
            "littlebit_selftest_wait_timeout", "littlebit_linear_forward_noalloc",
            "littlebit_decoder_workspace_size", "littlebit_decoder_step",
            "littlebit_decoder_poll_error", "littlebit_multi_workspace_size",
            "littlebit_linear_forward_multi", "littlebit_selftest_exchange_workspace_size",
            "littlebit_selftest_exchange"]


class lb_decoder_shape(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int32), ("n_heads", ctypes.c_int32),
                ("n_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("max_pos", ctypes.c_int32), ("rope_base", ctypes.c_float)]


class LittleBitError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__(f"{what}: {status_string(status)}")


class lb_path(ctypes.Structure):
    _fields_ = [("r", ctypes.c_int32),
                ("v_bits", ctypes.c_void_p),
                ("u_bits", ctypes.c_void_p),
                ("g", ctypes.c_void_p),
                ("l", ctypes.c_void_p),
                ("h", ctypes.c_void_p)]


class lb_linear(ctypes.Structure):
    _fields_ = [("d_in", ctypes.c_int32),
                ("d_out", ctypes.c_int32),
                ("n_paths", ctypes.c_int32),
                ("path", lb_path * 2)]


class lb_train_path(ctypes.Structure):
    _fields_ = [("r", ctypes.c_int32), ("u", ctypes.c_void_p), ("v", ctypes.c_void_p),
                ("g", ctypes.c_void_p), ("l", ctypes.c_void_p), ("h", ctypes.c_void_p)]


class lb_train_linear(ctypes.Structure):
    _fields_ = [("d_in", ctypes.c_int32), ("d_out", ctypes.c_int32), ("n_paths", ctypes.c_int32),
                ("path", lb_train_path * 2)]


class lb_train_grad(ctypes.Structure):
    _fields_ = [("du", ctypes.c_void_p), ("dv", ctypes.c_void_p), ("dg", ctypes.c_void_p),
                ("dl", ctypes.c_void_p), ("dh", ctypes.c_void_p)]


class lb_path_init(ctypes.Structure):
    """Output buffers of one path for littlebit_dual_svid (device pointers)."""
    _fields_ = [("r", ctypes.c_int32), ("v_bits", ctypes.c_void_p), ("u_bits", ctypes.c_void_p),
                ("g", ctypes.c_void_p), ("l", ctypes.c_void_p), ("h", ctypes.c_void_p)]


_lib = None
_lock = threading.Lock()


def lib(path: str | None = None):
    """Load liblittlebit.so (raises OSError if it is not built)."""
    global _lib
    with _lock:
        if _lib is not None and path is None:
            return _lib
        p = path or LIB_PATH
        if not os.path.exists(p):
            raise OSError(f"{p} is missing: build it with paper_2506_13771_gb300.build.build()")
        L = ctypes.CDLL(p)
        vp, i64, i32, sz = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_size_t
        L.littlebit_status_string.argtypes = [ctypes.c_int]
        L.littlebit_status_string.restype = ctypes.c_char_p
        L.littlebit_pack.argtypes = [vp, i64, i64, i32, vp, i64, vp, vp]
        L.littlebit_pack.restype = ctypes.c_int
        L.littlebit_workspace_size.argtypes = [ctypes.POINTER(lb_linear), i64]
        L.littlebit_workspace_size.restype = sz
        L.littlebit_linear_forward.argtypes = [ctypes.POINTER(lb_linear), vp, i64, vp, i32, vp,
                                               sz, vp]
        L.littlebit_linear_forward.restype = ctypes.c_int
        L.littlebit_linear_latent.argtypes = [ctypes.POINTER(lb_linear), vp, i64, vp, i32, vp,
                                              sz, vp]
        L.littlebit_linear_latent.restype = ctypes.c_int
        L.littlebit_linear_expand.argtypes = [ctypes.POINTER(lb_linear), vp, i32, i64, vp, i32,
                                              vp, sz, vp]
        L.littlebit_linear_expand.restype = ctypes.c_int
        L.littlebit_dual_svid_workspace_size.argtypes = [i32, i32, i32, ctypes.POINTER(lb_path_init)]
        L.littlebit_dual_svid_workspace_size.restype = sz
        L.littlebit_dual_svid.argtypes = [vp, i32, i32, i32, ctypes.POINTER(lb_path_init), i32, vp,
                                          sz, vp]
        L.littlebit_dual_svid.restype = ctypes.c_int
        L.littlebit_train_workspace_size.argtypes = [ctypes.POINTER(lb_train_linear), i64]
        L.littlebit_train_workspace_size.restype = sz
        L.littlebit_train_forward.argtypes = [ctypes.POINTER(lb_train_linear), vp, i64, vp, vp, sz,
                                              vp]
        L.littlebit_train_forward.restype = ctypes.c_int
        L.littlebit_train_backward.argtypes = [ctypes.POINTER(lb_train_linear), vp, vp, i64,
                                               ctypes.c_float, ctypes.POINTER(lb_train_grad), vp,
                                               vp, sz, vp]
        L.littlebit_train_backward.restype = ctypes.c_int
        L.littlebit_train_backward_saved.argtypes = L.littlebit_train_backward.argtypes
        L.littlebit_train_backward_saved.restype = ctypes.c_int
        L.littlebit_stack_workspace_size.argtypes = [ctypes.POINTER(lb_linear), i32, i32]
        L.littlebit_stack_workspace_size.restype = sz
        L.littlebit_stack_prepare.argtypes = [ctypes.POINTER(lb_linear), i32, i32, vp, sz, vp]
        L.littlebit_stack_prepare.restype = ctypes.c_int
        L.littlebit_stack_forward.argtypes = [ctypes.POINTER(lb_linear), i32, i32, vp, vp, vp, vp,
                                              vp, sz, vp]
        L.littlebit_stack_forward.restype = ctypes.c_int
        L.littlebit_decoder_workspace_size.argtypes = [ctypes.POINTER(lb_linear),
                                                       ctypes.POINTER(lb_decoder_shape)]
        L.littlebit_decoder_workspace_size.restype = sz
        L.littlebit_decoder_step.argtypes = [ctypes.POINTER(lb_linear),
                                             ctypes.POINTER(lb_decoder_shape), vp, vp, vp, vp, vp,
                                             vp, sz, vp]
        L.littlebit_decoder_step.restype = ctypes.c_int
        L.littlebit_decoder_poll_error.argtypes = [ctypes.POINTER(lb_linear),
                                                   ctypes.POINTER(lb_decoder_shape), vp, vp]
        L.littlebit_decoder_poll_error.restype = ctypes.c_int
        L.littlebit_multi_workspace_size.argtypes = [ctypes.POINTER(lb_linear), i32]
        L.littlebit_multi_workspace_size.restype = sz
        L.littlebit_linear_forward_multi.argtypes = [ctypes.POINTER(lb_linear), i32, vp, vp, i32,
                                                     vp, sz, vp]
        L.littlebit_linear_forward_multi.restype = ctypes.c_int
        L.littlebit_poll_error.argtypes = [vp, vp]
        L.littlebit_poll_error.restype = ctypes.c_int
        L.littlebit_selftest_wait_timeout.argtypes = [vp, vp]
        L.littlebit_selftest_wait_timeout.restype = ctypes.c_int
        L.littlebit_linear_forward_noalloc.argtypes = [ctypes.POINTER(lb_linear), vp, i64, vp,
                                                       i32, vp]
        L.littlebit_linear_forward_noalloc.restype = ctypes.c_int
        L.littlebit_selftest_exchange_workspace_size.argtypes = [i32, vp, i32]
        L.littlebit_selftest_exchange_workspace_size.restype = sz
        L.littlebit_selftest_exchange.argtypes = [i32, vp, i32, i32, i32, vp, sz, vp]
        L.littlebit_selftest_exchange.restype = ctypes.c_int
        if path is None:
            _lib = L
        return L


def status_string(status: int) -> str:
    return lib().littlebit_status_string(int(status)).decode()


def _check(status: int, what: str) -> None:
    if status != LB_OK:
        raise LittleBitError(status, what)


def _stream(stream) -> int | None:
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


# ------------------------------------------------------------------ tensors


def to_device_bits(a: np.ndarray, device) -> torch.Tensor:
    """Copy a numpy bit-pattern array (uint16 / uint32) to the device unchanged."""
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint32:
        return torch.from_numpy(a.view(np.int32)).to(device)
    if a.dtype == np.uint16:
        return torch.from_numpy(a.view(np.int16)).to(device)
    raise TypeError(f"unsupported bit array dtype {a.dtype}")


def bf16_tensor(x_bits: np.ndarray, device) -> torch.Tensor:
    """bf16 bit patterns (uint16) -> torch.bfloat16 tensor on device."""
    return to_device_bits(x_bits, device).view(torch.bfloat16)


class DeviceLinear:
    """One LittleBit linear resident on the device, and its lb_linear struct.

    Built from a layer dict of ``inputs.make_linear``: packed words are copied
    as they are; explicit +-1 signs are packed on the device by littlebit_pack.
    """

    def __init__(self, layer: dict, device="cuda", stream=None):
        self.d_in = int(layer["d_in"])
        self.d_out = int(layer["d_out"])
        self.paths = []
        self.ranks = []
        self.c = lb_linear()
        self.c.d_in = self.d_in
        self.c.d_out = self.d_out
        self.c.n_paths = len(layer["paths"])
        for p, P in enumerate(layer["paths"]):
            r = int(P["r"])
            if "v_words" in P:
                v = to_device_bits(P["v_words"], device)
                u = to_device_bits(P["u_words"], device)
            else:
                v = pack(torch.from_numpy(P["v_signs"]).to(device), LB_PACK_V, stream=stream)
                u = pack(torch.from_numpy(P["u_signs"]).to(device), LB_PACK_U, stream=stream)
            t = {"v_bits": v, "u_bits": u, "g": to_device_bits(P["g"], device),
                 "l": to_device_bits(P["l"], device), "h": to_device_bits(P["h"], device)}
            self.paths.append(t)
            self.ranks.append(r)
            cp = self.c.path[p]
            cp.r = r
            for k, ten in t.items():
                setattr(cp, k, ten.data_ptr())

    @property
    def nbytes(self) -> int:
        return sum(t.numel() * t.element_size() for P in self.paths for t in P.values())


# ------------------------------------------------------------------ entry points


def pack(signs: torch.Tensor, layout: int, out: torch.Tensor | None = None,
         bad: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """Eq. 2 packing of a device int8 [rows][cols] +-1 matrix -> int32 words
    (uint32 bit patterns) in the U or V layout."""
    assert signs.dtype == torch.int8 and signs.dim() == 2 and signs.is_contiguous()
    rows, cols = signs.shape
    shape = (rows, (cols + 31) // 32) if layout == LB_PACK_U else ((rows + 31) // 32, cols)
    if out is None:
        out = torch.empty(shape, dtype=torch.int32, device=signs.device)
    _check(lib().littlebit_pack(signs.data_ptr(), rows, cols, layout, out.data_ptr(), out.numel(),
                                bad.data_ptr() if bad is not None else None, _stream(stream)),
           "littlebit_pack")
    return out


def workspace_size(L: DeviceLinear, T: int) -> int:
    return int(lib().littlebit_workspace_size(ctypes.byref(L.c), int(T)))


def new_workspace(nbytes: int, device="cuda") -> torch.Tensor:
    """A zero-filled workspace (uint8), as the ABI requires before first use."""
    return torch.zeros(max(int(nbytes), 256), dtype=torch.uint8, device=device)


def _forward_args(L: DeviceLinear, x: torch.Tensor, out_dtype, y: torch.Tensor | None):
    """Checks x (bf16 [T][d_in] on the current CUDA device) and the output y
    ([T][d_out], bf16 or fp32, contiguous, on x's device), allocating y when
    it is None; returns (contiguous x, y)."""
    assert x.dtype == torch.bfloat16 and x.dim() == 2 and x.shape[1] == L.d_in
    assert x.is_cuda and x.device.index == torch.cuda.current_device(), \
        "x must be on the current CUDA device"
    x = x.contiguous()
    T = x.shape[0]
    if y is None:
        y = torch.empty((T, L.d_out), dtype=out_dtype, device=x.device)
    assert tuple(y.shape) == (T, L.d_out), (tuple(y.shape), (T, L.d_out))
    assert y.dtype in (torch.bfloat16, torch.float32) and y.is_contiguous()
    assert y.device == x.device
    return x, y


def linear_forward(L: DeviceLinear, x: torch.Tensor, out_dtype=torch.bfloat16,
                   y: torch.Tensor | None = None, ws: torch.Tensor | None = None,
                   stream=None) -> torch.Tensor:
    """Y = X W^T (Prop. 1 per path, Eq. 6 sum) for x bf16 [T][d_in] on device."""
    x, y = _forward_args(L, x, out_dtype, y)
    T = x.shape[0]
    y_dtype = LB_OUT_FP32 if y.dtype == torch.float32 else LB_OUT_BF16
    if ws is None:
        ws = new_workspace(workspace_size(L, T), x.device)
    _check(lib().littlebit_linear_forward(ctypes.byref(L.c), x.data_ptr(), T, y.data_ptr(),
                                          y_dtype, ws.data_ptr(), ws.numel(), _stream(stream)),
           "littlebit_linear_forward")
    return y


def linear_latent(L: DeviceLinear, x: torch.Tensor, z_dtype=torch.float32,
                  z: torch.Tensor | None = None, ws: torch.Tensor | None = None,
                  stream=None) -> torch.Tensor:
    """Latent states z [T][r_0 + r_1] = l_p . ((X . g_p) V_p,sign) per path
    (Sec. 5, KV cache compression) for x bf16 [T][d_in] on device."""
    assert x.dtype == torch.bfloat16 and x.dim() == 2 and x.shape[1] == L.d_in
    x = x.contiguous()
    T = x.shape[0]
    if z is None:
        z = torch.empty((T, sum(L.ranks)), dtype=z_dtype, device=x.device)
    assert z.dtype in (torch.float32, torch.float16) and z.is_contiguous()
    code = LB_LATENT_FP16 if z.dtype == torch.float16 else LB_LATENT_FP32
    if ws is None:
        ws = new_workspace(workspace_size(L, T), x.device)
    _check(lib().littlebit_linear_latent(ctypes.byref(L.c), x.data_ptr(), T, z.data_ptr(), code,
                                         ws.data_ptr(), ws.numel(), _stream(stream)),
           "littlebit_linear_latent")
    return z


def linear_expand(L: DeviceLinear, z: torch.Tensor, out_dtype=torch.bfloat16,
                  y: torch.Tensor | None = None, ws: torch.Tensor | None = None,
                  stream=None) -> torch.Tensor:
    """Y [T][d_out] = sum_p h_p . (U_p,sign z_p) from latents z [T][r_0 + r_1]
    (fp32 or fp16) on device."""
    assert z.dtype in (torch.float32, torch.float16) and z.dim() == 2
    assert z.shape[1] == sum(L.ranks)
    z = z.contiguous()
    T = z.shape[0]
    code = LB_LATENT_FP16 if z.dtype == torch.float16 else LB_LATENT_FP32
    if y is None:
        y = torch.empty((T, L.d_out), dtype=out_dtype, device=z.device)
    y_dtype = LB_OUT_FP32 if y.dtype == torch.float32 else LB_OUT_BF16
    if ws is None:
        ws = new_workspace(workspace_size(L, T), z.device)
    _check(lib().littlebit_linear_expand(ctypes.byref(L.c), z.data_ptr(), code, T, y.data_ptr(),
                                         y_dtype, ws.data_ptr(), ws.numel(), _stream(stream)),
           "littlebit_linear_expand")
    return y


def dual_svid(W: torch.Tensor, ranks, iters: int = 8, ws: torch.Tensor | None = None,
              stream=None) -> dict:
    """Dual-SVID initialisation (Sec. 3.2) with Residual Compensation (Sec. 3.3) of a dense
    fp32 weight W [d_out][d_in] on the device.  Returns a layer dict of device tensors:
    {'d_in', 'd_out', 'paths': [{'r', 'v_words', 'u_words', 'g', 'l', 'h'}]} (int32 words,
    int16 fp16 bit patterns)."""
    assert W.dtype == torch.float32 and W.dim() == 2 and W.is_cuda
    W = W.contiguous()
    d_out, d_in = W.shape
    outs = []
    arr = (lb_path_init * len(ranks))()
    for p, r in enumerate(ranks):
        t = {"r": int(r),
             "v_words": torch.empty(((d_in + 31) // 32, r), dtype=torch.int32, device=W.device),
             "u_words": torch.empty((d_out, (r + 31) // 32), dtype=torch.int32, device=W.device),
             "g": torch.empty(d_in, dtype=torch.int16, device=W.device),
             "l": torch.empty(r, dtype=torch.int16, device=W.device),
             "h": torch.empty(d_out, dtype=torch.int16, device=W.device)}
        outs.append(t)
        arr[p].r = int(r)
        arr[p].v_bits, arr[p].u_bits = t["v_words"].data_ptr(), t["u_words"].data_ptr()
        arr[p].g, arr[p].l, arr[p].h = t["g"].data_ptr(), t["l"].data_ptr(), t["h"].data_ptr()
    n = int(lib().littlebit_dual_svid_workspace_size(d_out, d_in, len(ranks), arr))
    if n == 0:
        raise LittleBitError(LB_ERR_INVALID_ARG, "littlebit_dual_svid_workspace_size")
    if ws is None:
        ws = torch.empty(n, dtype=torch.uint8, device=W.device)
    _check(lib().littlebit_dual_svid(W.data_ptr(), d_out, d_in, len(ranks), arr, int(iters),
                                     ws.data_ptr(), ws.numel(), _stream(stream)),
           "littlebit_dual_svid")
    return {"d_in": d_in, "d_out": d_out, "paths": outs}


def layer_to_host(layer: dict) -> dict:
    """A layer dict of device tensors as numpy arrays in the inputs.make_linear layout."""
    paths = []
    for P in layer["paths"]:
        paths.append({"r": P["r"],
                      "v_words": P["v_words"].cpu().numpy().view(np.uint32),
                      "u_words": P["u_words"].cpu().numpy().view(np.uint32),
                      "g": P["g"].cpu().numpy().view(np.uint16),
                      "l": P["l"].cpu().numpy().view(np.uint16),
                      "h": P["h"].cpu().numpy().view(np.uint16)})
    return {"d_in": layer["d_in"], "d_out": layer["d_out"], "paths": paths}


class TrainLinear:
    """A LittleBit linear in QAT form on the device: latent fp32 factors and scales.
    Built from {'d_in', 'd_out', 'paths': [{'r', 'u', 'v', 'g', 'l', 'h'}]} (numpy or torch)."""

    def __init__(self, layer: dict, device="cuda"):
        self.d_in, self.d_out = int(layer["d_in"]), int(layer["d_out"])
        self.c = lb_train_linear()
        self.c.d_in, self.c.d_out, self.c.n_paths = self.d_in, self.d_out, len(layer["paths"])
        self.paths, self.ranks = [], []
        for p, P in enumerate(layer["paths"]):
            t = {k: torch.as_tensor(np.asarray(P[k]) if not torch.is_tensor(P[k]) else P[k],
                                    dtype=torch.float32).to(device).contiguous()
                 for k in ("u", "v", "g", "l", "h")}
            self.paths.append(t)
            self.ranks.append(int(P["r"]))
            cp = self.c.path[p]
            cp.r = int(P["r"])
            for k, ten in t.items():
                setattr(cp, k, ten.data_ptr())

    def workspace(self, T: int, device="cuda") -> torch.Tensor:
        n = int(lib().littlebit_train_workspace_size(ctypes.byref(self.c), int(T)))
        return torch.empty(max(n, 256), dtype=torch.uint8, device=device)


def train_forward(L: TrainLinear, x: torch.Tensor, ws: torch.Tensor | None = None,
                  stream=None) -> torch.Tensor:
    """QAT forward (signs of the latent factors), fp32 x [T][d_in] -> y [T][d_out]."""
    assert x.dtype == torch.float32 and x.dim() == 2 and x.shape[1] == L.d_in
    x = x.contiguous()
    T = x.shape[0]
    y = torch.empty((T, L.d_out), dtype=torch.float32, device=x.device)
    ws = ws if ws is not None else L.workspace(T, x.device)
    _check(lib().littlebit_train_forward(ctypes.byref(L.c), x.data_ptr(), T, y.data_ptr(),
                                         ws.data_ptr(), ws.numel(), _stream(stream)),
           "littlebit_train_forward")
    return y


def train_backward(L: TrainLinear, x: torch.Tensor, dy: torch.Tensor, k: float = 100.0,
                   want_dx: bool = True, ws: torch.Tensor | None = None, stream=None,
                   saved: bool = False):
    """QAT backward with SmoothSign: (per-path dicts du, dv, dg, dl, dh; dX or None).
    saved: reuse what train_forward(L, x) left in ws (littlebit_train_backward_saved)."""
    x, dy = x.contiguous(), dy.contiguous()
    T = x.shape[0]
    grads = (lb_train_grad * len(L.paths))()
    out = []
    for p, P in enumerate(L.paths):
        g = {"du": torch.empty_like(P["u"]), "dv": torch.empty_like(P["v"]),
             "dg": torch.empty_like(P["g"]), "dl": torch.empty_like(P["l"]),
             "dh": torch.empty_like(P["h"])}
        out.append(g)
        for key, ten in g.items():
            setattr(grads[p], key, ten.data_ptr())
    dx = torch.empty_like(x) if want_dx else None
    ws = ws if ws is not None else L.workspace(T, x.device)
    fn = lib().littlebit_train_backward_saved if saved else lib().littlebit_train_backward
    _check(fn(ctypes.byref(L.c), x.data_ptr(), dy.data_ptr(), T, float(k), grads,
              dx.data_ptr() if want_dx else None, ws.data_ptr(), ws.numel(), _stream(stream)),
           "littlebit_train_backward")
    return out, dx


class DeviceStack:
    """n_layers x (q, k, v, o, gate, up, down) LittleBit linears on the device."""

    def __init__(self, layers: list, head_dim: int = 128, device="cuda"):
        assert len(layers) % 7 == 0
        self.n_layers = len(layers) // 7
        self.head_dim = int(head_dim)
        self.linears = [DeviceLinear(L, device) for L in layers]
        self.carray = (lb_linear * len(self.linears))(*[L.c for L in self.linears])
        self.d_model = self.linears[0].d_in
        self.d_kv = self.linears[1].d_out

    @property
    def nbytes(self) -> int:
        return sum(L.nbytes for L in self.linears)

    def workspace_size(self) -> int:
        return int(lib().littlebit_stack_workspace_size(self.carray, self.n_layers, self.head_dim))

    def prepare(self, ws: torch.Tensor | None = None, stream=None) -> torch.Tensor:
        """Prepare (and return) a workspace for this stack."""
        if ws is None:
            ws = new_workspace(self.workspace_size(), self.linears[0].paths[0]["g"].device)
        _check(lib().littlebit_stack_prepare(self.carray, self.n_layers, self.head_dim,
                                             ws.data_ptr(), ws.numel(), _stream(stream)),
               "littlebit_stack_prepare")
        return ws


def stack_forward(S: DeviceStack, x0: torch.Tensor, out: torch.Tensor | None = None,
                  q_out: torch.Tensor | None = None, kv_out: torch.Tensor | None = None,
                  want_q: bool = True, want_kv: bool = True, ws: torch.Tensor | None = None,
                  stream=None):
    """One decode step through the stack; returns (out fp32 [d_model],
    q fp32 [n_layers][d_model] or None, kv fp32 [n_layers][2][d_kv] or None).
    ws: a workspace prepared by ``S.prepare()`` (one is made if None)."""
    assert x0.dtype == torch.bfloat16 and x0.numel() == S.d_model
    dev = x0.device
    if out is None:
        out = torch.empty(S.d_model, dtype=torch.float32, device=dev)
    if q_out is None and want_q:
        q_out = torch.empty((S.n_layers, S.d_model), dtype=torch.float32, device=dev)
    if kv_out is None and want_kv:
        kv_out = torch.empty((S.n_layers, 2, S.d_kv), dtype=torch.float32, device=dev)
    if ws is None:
        ws = S.prepare(stream=stream)
    _check(lib().littlebit_stack_forward(S.carray, S.n_layers, S.head_dim, x0.data_ptr(),
                                         out.data_ptr(),
                                         q_out.data_ptr() if q_out is not None else None,
                                         kv_out.data_ptr() if kv_out is not None else None,
                                         ws.data_ptr(), ws.numel(), _stream(stream)),
           "littlebit_stack_forward")
    return out, q_out, kv_out


def poll_error(ws: torch.Tensor, stream=None) -> int:
    """Synchronise and return (and clear) the workspace's sticky error status."""
    return int(lib().littlebit_poll_error(ws.data_ptr(), _stream(stream)))


def selftest_wait_timeout(ws: torch.Tensor, stream=None) -> None:
    """Launch the bounded-wait diagnostic (records LB_ERR_TIMEOUT in ws)."""
    _check(lib().littlebit_selftest_wait_timeout(ws.data_ptr(), _stream(stream)),
           "littlebit_selftest_wait_timeout")


def selftest_exchange(n_rounds: int, sizes, cluster: int = 1, words: int = 1,
                      ws: torch.Tensor | None = None, device="cuda", stream=None) -> torch.Tensor:
    """Launch the exchange-chain diagnostic (n_rounds dependent all-reduces of
    sizes[k % len(sizes)] elements; words = 1: the stack's encoding, 2: the
    single-linear kernels'); returns the workspace (poll it)."""
    arr = (ctypes.c_int32 * len(sizes))(*[int(v) for v in sizes])
    need = int(lib().littlebit_selftest_exchange_workspace_size(int(n_rounds), arr, len(sizes)))
    if need == 0:
        raise LittleBitError(LB_ERR_INVALID_ARG, "littlebit_selftest_exchange_workspace_size")
    if ws is None:
        ws = new_workspace(need, device)
    _check(lib().littlebit_selftest_exchange(int(n_rounds), arr, len(sizes), int(cluster),
                                             int(words), ws.data_ptr(), ws.numel(),
                                             _stream(stream)),
           "littlebit_selftest_exchange")
    return ws


def linear_forward_noalloc(L: DeviceLinear, x: torch.Tensor, out_dtype=torch.bfloat16,
                           y: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """Y = X W^T without a workspace: the library's built-in scratch is used
    (for callers that cannot allocate device memory; see littlebit.h)."""
    x, y = _forward_args(L, x, out_dtype, y)
    T = x.shape[0]
    y_dtype = LB_OUT_FP32 if y.dtype == torch.float32 else LB_OUT_BF16
    _check(lib().littlebit_linear_forward_noalloc(ctypes.byref(L.c), x.data_ptr(), T, y.data_ptr(),
                                                  y_dtype, _stream(stream)),
           "littlebit_linear_forward_noalloc")
    return y


# ------------------------------------------------------------------ decode at position p (App. I.3)


class DeviceDecoder:
    """A Llama-shaped decoder whose n_layers x (q, k, v, o, gate, up, down)
    linears are LittleBit linears on the device, with its fp32 KV cache
    ([n_layers][max_pos][d_kv] each for keys and values), the device position
    counter and a workspace (all zero-filled: the cache starts empty)."""

    def __init__(self, layers: list, n_heads: int, n_kv_heads: int, head_dim: int = 128,
                 max_pos: int = 512, rope_base: float = 10000.0, device="cuda"):
        assert len(layers) % 7 == 0
        self.n_layers = len(layers) // 7
        self.linears = [DeviceLinear(L, device) for L in layers]
        self.carray = (lb_linear * len(self.linears))(*[L.c for L in self.linears])
        self.shape = lb_decoder_shape(self.n_layers, int(n_heads), int(n_kv_heads), int(head_dim),
                                      int(max_pos), float(rope_base))
        self.d_model = int(n_heads) * int(head_dim)
        self.d_kv = int(n_kv_heads) * int(head_dim)
        nbytes = int(lib().littlebit_decoder_workspace_size(self.carray, ctypes.byref(self.shape)))
        if nbytes == 0:
            raise LittleBitError(LB_ERR_INVALID_ARG, "littlebit_decoder_workspace_size")
        self.ws = new_workspace(nbytes, device)
        self.kcache = torch.zeros((self.n_layers, max_pos, self.d_kv), dtype=torch.float32,
                                  device=device)
        self.vcache = torch.zeros_like(self.kcache)
        self.pos = torch.zeros(1, dtype=torch.int32, device=device)

    @property
    def nbytes(self) -> int:
        return sum(L.nbytes for L in self.linears)

    def step(self, x: torch.Tensor, out: torch.Tensor | None = None, stream=None) -> torch.Tensor:
        """Decodes the token x (bf16 [d_model]) at the current position and
        advances it; returns the last hidden state (fp32 [d_model])."""
        assert x.dtype == torch.bfloat16 and x.numel() == self.d_model and x.is_contiguous()
        if out is None:
            out = torch.empty(self.d_model, dtype=torch.float32, device=x.device)
        _check(lib().littlebit_decoder_step(self.carray, ctypes.byref(self.shape), x.data_ptr(),
                                            self.kcache.data_ptr(), self.vcache.data_ptr(),
                                            self.pos.data_ptr(), out.data_ptr(), self.ws.data_ptr(),
                                            self.ws.numel(), _stream(stream)),
               "littlebit_decoder_step")
        return out

    def poll_error(self, stream=None) -> int:
        return int(lib().littlebit_decoder_poll_error(self.carray, ctypes.byref(self.shape),
                                                      self.ws.data_ptr(), _stream(stream)))


# ------------------------------------------------------------------ several linears, one token


def multi_workspace_size(linears: list) -> int:
    arr = (lb_linear * len(linears))(*[L.c for L in linears])
    return int(lib().littlebit_multi_workspace_size(arr, len(linears)))


def linear_forward_multi(linears: list, x: torch.Tensor, out_dtype=torch.bfloat16,
                         y: torch.Tensor | None = None, ws: torch.Tensor | None = None,
                         stream=None) -> torch.Tensor:
    """y[m] = x W_m^T for M DeviceLinears of one shape and one bf16 token x [d_in]:
    one launch; returns [M][d_out]."""
    assert x.dtype == torch.bfloat16 and x.is_contiguous()
    M = len(linears)
    arr = (lb_linear * M)(*[L.c for L in linears])
    if y is None:
        y = torch.empty((M, linears[0].d_out), dtype=out_dtype, device=x.device)
    assert y.dtype in (torch.bfloat16, torch.float32) and y.is_contiguous()
    if ws is None:
        ws = new_workspace(multi_workspace_size(linears), x.device)
    code = LB_OUT_FP32 if y.dtype == torch.float32 else LB_OUT_BF16
    _check(lib().littlebit_linear_forward_multi(arr, M, x.data_ptr(), y.data_ptr(), code,
                                                ws.data_ptr(), ws.numel(), _stream(stream)),
           "littlebit_linear_forward_multi")
    return y
