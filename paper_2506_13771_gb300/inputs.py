"""Seeded synthetic inputs for the LittleBit forward, shared by the CUDA path's
tests and benchmarks and by the CPU oracle's tests.

This module holds none of the method's arithmetic: it only draws random
numbers (numpy PCG64), rounds them to the storage formats the paper fixes
(FP16 scales, Eq. 3; bf16 activations), and lays random sign bits out in the
packed word format.  Packing of explicit +-1 matrices is NOT done here: each
side packs with its own packer.

Distributions (the paper's trained weights and datasets are not available, so
these stand in for the Llama2 linear shapes of Table 11 / App. I):
  * signs   : Bernoulli(0.5) over {-1,+1}
  * h, g, l : |N(0,1)| * c, drawn in fp64, rounded once to fp16 (RNE)
  * x       : N(0,1), drawn in fp64, rounded to fp32 then to bf16 (RNE)
Seeds are 20250600 + config id.
"""
from __future__ import annotations

import numpy as np

SEED_BASE = 20250600


def rng_for(config_id: int, salt: int = 0) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(SEED_BASE + int(config_id) + 1000 * int(salt)))


def f32_to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round fp32 values to bfloat16 (round to nearest even); returns uint16 bits."""
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32).astype(np.uint64)
    rounded = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return rounded.astype(np.uint16)


def bf16_normal(rng: np.random.Generator, shape, scale: float = 1.0) -> np.ndarray:
    """N(0,1) * scale activations stored as bf16 bit patterns."""
    return f32_to_bf16_bits((rng.standard_normal(shape) * scale).astype(np.float32))


def fp16_abs_normal(rng: np.random.Generator, n: int, c: float) -> np.ndarray:
    """|N(0,1)| * c scales stored as fp16 bit patterns."""
    v = np.abs(rng.standard_normal(n)) * c
    return v.astype(np.float16).view(np.uint16)


def random_signs(rng: np.random.Generator, rows: int, cols: int) -> np.ndarray:
    """Bernoulli(0.5) +-1 matrix, int8."""
    b = rng.integers(0, 2, size=(rows, cols), dtype=np.int8)
    return (1 - 2 * b).astype(np.int8)


def random_u_words(rng: np.random.Generator, d_out: int, r: int) -> np.ndarray:
    """Random sign bits directly in the U word layout [d_out][ceil(r/32)];
    padding bits (beyond r) are zero."""
    nw = (r + 31) // 32
    w = rng.integers(0, 1 << 32, size=(d_out, nw), dtype=np.uint64).astype(np.uint32)
    tail = r - 32 * (nw - 1)
    if tail < 32:
        w[:, -1] &= np.uint32((1 << tail) - 1)
    return w


def random_v_words(rng: np.random.Generator, d_in: int, r: int) -> np.ndarray:
    """Random sign bits directly in the V word layout [ceil(d_in/32)][r];
    padding bits (beyond d_in) are zero."""
    nw = (d_in + 31) // 32
    w = rng.integers(0, 1 << 32, size=(nw, r), dtype=np.uint64).astype(np.uint32)
    tail = d_in - 32 * (nw - 1)
    if tail < 32:
        w[-1, :] &= np.uint32((1 << tail) - 1)
    return w


def make_linear(rng: np.random.Generator, d_in: int, d_out: int, r, n_paths: int = 2,
                scale: float = 0.02, explicit_signs: bool = False, g_mul: float = 1.0,
                l_mul: float = 1.0, h_mul: float = 1.0) -> dict:
    """One LittleBit linear.  With explicit_signs=True each path carries
    'u_signs' [d_out][r] and 'v_signs' [d_in][r] (+-1 int8) and no words;
    otherwise it carries random 'u_words' / 'v_words' in the packed layout.
    r may be an int or a per-path list.  g, l and h are drawn at scale times
    g_mul, l_mul and h_mul."""
    rs = list(r) if isinstance(r, (list, tuple)) else [int(r)] * n_paths
    paths = []
    for p in range(n_paths):
        rp = rs[p]
        P = {"r": rp}
        if explicit_signs:
            P["v_signs"] = random_signs(rng, d_in, rp)
            P["u_signs"] = random_signs(rng, d_out, rp)
        else:
            P["v_words"] = random_v_words(rng, d_in, rp)
            P["u_words"] = random_u_words(rng, d_out, rp)
        P["g"] = fp16_abs_normal(rng, d_in, scale * g_mul)
        P["l"] = fp16_abs_normal(rng, rp, scale * l_mul)
        P["h"] = fp16_abs_normal(rng, d_out, scale * h_mul)
        paths.append(P)
    return {"d_in": int(d_in), "d_out": int(d_out), "paths": paths}


# --------------------------------------------------------------------------
# The workloads (Llama2 linear shapes; App. I / Table 11 setting)
# --------------------------------------------------------------------------

def config1(explicit_signs: bool = True):
    """512 x 512, two paths of rank 16, scales |N|*0.05, 4 tokens."""
    rng = rng_for(1)
    L = make_linear(rng, 512, 512, 16, 2, 0.05, explicit_signs)
    x = bf16_normal(rng, (4, 512))
    return L, x


def config2(T: int = 1):
    """Llama2-7B q_proj shape 4096 x 4096, two paths of rank 64, scales |N|*0.02."""
    rng = rng_for(2)
    L = make_linear(rng, 4096, 4096, 64, 2, 0.02)
    x = bf16_normal(rng_for(2, salt=T), (T, 4096))
    return L, x


def config3(r: int = 128, T: int = 1):
    """Llama2-7B FFN triple: gate, up 4096->11008 and down 11008->4096."""
    rng = rng_for(3, salt=r)
    gate = make_linear(rng, 4096, 11008, r, 2, 0.02)
    up = make_linear(rng, 4096, 11008, r, 2, 0.02)
    down = make_linear(rng, 11008, 4096, r, 2, 0.02)
    x = bf16_normal(rng_for(3, salt=10000 + T), (T, 4096))
    x_down = bf16_normal(rng_for(3, salt=20000 + T), (T, 11008))
    return {"gate": gate, "up": up, "down": down}, x, x_down


PREFILL_SHAPES = {
    "4096x4096_r64": (4096, 4096, 64),
    "4096x4096_r512": (4096, 4096, 512),
    "4096x11008_r128": (4096, 11008, 128),
}


def config4(shape: str = "4096x4096_r64", T: int = 2048):
    """Prefill: many-token LittleBit linears (d_in, d_out, r), two paths."""
    d_in, d_out, r = PREFILL_SHAPES[shape]
    rng = rng_for(4, salt=r)
    L = make_linear(rng, d_in, d_out, r, 2, 0.02)
    x = bf16_normal(rng_for(4, salt=10000 + T), (T, d_in))
    return L, x


STACK_70B = {
    "d_model": 8192, "d_kv": 1024, "d_ff": 28672, "n_layers": 80,
    "r_qo": 192, "r_kv": 32, "r_mlp": 320, "head_dim": 128,
}


def stack_shapes(d_model, d_kv, d_ff, r_qo, r_kv, r_mlp):
    """(d_in, d_out, r) of q, k, v, o, gate, up, down in chain order."""
    return [(d_model, d_model, r_qo), (d_model, d_kv, r_kv), (d_model, d_kv, r_kv),
            (d_model, d_model, r_qo), (d_model, d_ff, r_mlp), (d_model, d_ff, r_mlp),
            (d_ff, d_model, r_mlp)]


def unit_gain_scale(d_in: int, r: int, n_paths: int = 2) -> float:
    """Scale c of |N(0,1)|*c for h, g and l such that a linear maps an input of
    rms 1 to an output of rms about 1 (each output is a sum of n_paths*r*d_in
    sign-weighted products of three scales: rms ~ c^3 sqrt(n_paths r d_in))."""
    return float((n_paths * r * d_in) ** (-1.0 / 6.0))


def make_stack(n_layers: int = 80, d_model: int = 8192, d_kv: int = 1024, d_ff: int = 28672,
               r_qo: int = 192, r_kv: int = 32, r_mlp: int = 320, head_dim: int = 128,
               config_id: int = 5, x_scale: float = 1.0, g_mul: float = 1.0,
               l_mul: float = 1.0, out_h_mul: float = 1.0):
    """Llama2-70B-shaped decode stack: n_layers x (q,k,v,o,gate,up,down), two
    paths each, random sign words, unit-gain scales (g and l times g_mul and
    l_mul, the h of o and down -- the branches that write the residual
    stream -- times out_h_mul).
    Returns (list of 7*n_layers linears, x0 bf16 bits [d_model], N(0,1) * x_scale)."""
    rng = rng_for(config_id)
    shapes = stack_shapes(d_model, d_kv, d_ff, r_qo, r_kv, r_mlp)
    layers = []
    for _ in range(n_layers):
        for k, (di, do, r) in enumerate(shapes):
            layers.append(make_linear(rng, di, do, r, 2, unit_gain_scale(di, r, 2), g_mul=g_mul,
                                      l_mul=l_mul, h_mul=out_h_mul if k in (3, 6) else 1.0))
    x0 = bf16_normal(rng, (d_model,), x_scale)
    return layers, x0


# Llama2-7B-shaped decoder (the model of the paper's end-to-end decoding
# table, shape only): 32 layers, d_model 4096 = 32 heads x 128, MHA, d_ff
# 11008, with the ranks of the single-linear workloads (q/k/v/o 4096^2 at
# r = 64 per path, ~0.08 BPW; the MLP at r = 128, ~0.1 BPW).
DECODER_7B = dict(n_layers=32, d_model=4096, d_kv=4096, d_ff=11008, r_qo=64, r_kv=64, r_mlp=128,
                  n_heads=32, n_kv_heads=32, head_dim=128)


def decoder7b(n_tokens: int, n_layers: int = 32, config_id: int = 9):
    """The 7B-shaped decoder's linears (two paths each, random sign words,
    unit-gain scales) and n_tokens token embeddings, bf16 N(0,1) [n_tokens][4096]."""
    kw = {k: v for k, v in DECODER_7B.items()
          if k not in ("n_layers", "n_heads", "n_kv_heads", "head_dim")}
    layers, _ = make_stack(n_layers=n_layers, config_id=config_id, **kw)
    xs = bf16_normal(rng_for(config_id, salt=1), (n_tokens, DECODER_7B["d_model"]))
    return layers, xs


def config5(n_layers: int = 80):
    kw = {k: v for k, v in STACK_70B.items() if k not in ("n_layers", "head_dim")}
    return make_stack(n_layers=n_layers, **kw)


def spectral_weight(rng: np.random.Generator, d_out: int, d_in: int,
                    spectrum: np.ndarray) -> np.ndarray:
    """A dense fp64 weight A diag(spectrum) B^T with random orthonormal A, B
    (QR of Gaussian matrices): a synthetic stand-in for a trained weight with
    a prescribed singular spectrum (the Dual-SVID workloads)."""
    k = min(d_out, d_in)
    A, _ = np.linalg.qr(rng.standard_normal((d_out, k)))
    B, _ = np.linalg.qr(rng.standard_normal((d_in, k)))
    return (A * np.asarray(spectrum, np.float64)[:k]) @ B.T
