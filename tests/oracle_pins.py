"""Pins of the CPU oracle against facts that do not come from the oracle itself.

Each pin takes an ``oracle.Oracle`` and raises AssertionError on a mismatch.
They are collected by test_oracle_pins.py, and re-run against deliberately
broken copies of the oracle by test_oracle_mutations.py to show that a
plausible mistake (dropped term, wrong sign, wrong index, transposed operand)
fails at least one of them.

Sources of truth used here, none of which is the oracle:
  * numpy's own float16 / float32 decoders (exhaustive over all 2^16 patterns)
  * numpy.packbits (an independent bit packer)
  * closed forms of Prop. 1 / Eq. 4 for special parameter choices (rank 1,
    all-equal signs, Sylvester-Hadamard factors with unit scales)
  * a hand-expanded quadruple sum over every sign pattern of a tiny layer
  * the worked examples of App. E and App. I.1, and Table 4's KV-cache ranks
    (tests/golden/)
  * algebraic invariants: path-swap symmetry of Eq. 6, h_res = 0 reducing to
    one path
  * numpy's LAPACK SVD for the Dual-SVID steps; exact recovery of a rank-1
    matrix and of a Sylvester-Hadamard LittleBit weight
  * for the decoder chain: textbook softmax attention over the one cached
    position, and closed forms with branches switched off or made the identity
"""
from __future__ import annotations

import os

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")

# ------------------------------------------------------------------ helpers


def np_half(bits) -> np.ndarray:
    return np.asarray(bits, dtype=np.uint16).view(np.float16).astype(np.float64)


def np_bf16(bits) -> np.ndarray:
    u = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16
    with np.errstate(invalid="ignore"):
        return u.view(np.float32).astype(np.float64)


def half_bits(v) -> np.ndarray:
    return np.asarray(v, dtype=np.float64).astype(np.float16).view(np.uint16)


def bf16_bits_exact(v) -> np.ndarray:
    """bf16 bits of values that are exactly representable (checked)."""
    f = np.asarray(v, dtype=np.float32)
    u = f.view(np.uint32)
    assert np.all((u & 0xFFFF) == 0), "value not exactly representable in bf16"
    return (u >> 16).astype(np.uint16)


def rel(a, b) -> float:
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    den = np.linalg.norm(b)
    return float(np.linalg.norm(a - b) / (den if den > 0 else 1.0))


def layer_from_signs(orc, d_in, d_out, paths):
    """paths: list of dicts with u_signs, v_signs, g, l, h (fp16 bits)."""
    out = []
    for P in paths:
        out.append({"r": P["u_signs"].shape[1],
                    "u_words": orc.pack_u(P["u_signs"]),
                    "v_words": orc.pack_v(P["v_signs"]),
                    "g": P["g"], "l": P["l"], "h": P["h"]})
    return {"d_in": d_in, "d_out": d_out, "paths": out}


def rand_path(rng, d_in, d_out, r, c=0.3):
    return {"u_signs": (1 - 2 * rng.integers(0, 2, (d_out, r))).astype(np.int8),
            "v_signs": (1 - 2 * rng.integers(0, 2, (d_in, r))).astype(np.int8),
            "g": half_bits(np.abs(rng.standard_normal(d_in)) * c + 0.05),
            "l": half_bits(np.abs(rng.standard_normal(r)) * c + 0.05),
            "h": half_bits(np.abs(rng.standard_normal(d_out)) * c + 0.05)}


def rand_x(rng, T, d_in):
    f = rng.standard_normal((T, d_in)).astype(np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    return ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)


def sylvester(n: int) -> np.ndarray:
    H = np.ones((1, 1), dtype=np.int8)
    while H.shape[0] < n:
        H = np.block([[H, H], [H, -H]]).astype(np.int8)
    return H


def fwht(v: np.ndarray) -> np.ndarray:
    """Textbook in-place fast Walsh-Hadamard transform (Sylvester order)."""
    a = np.array(v, dtype=np.float64)
    h = 1
    n = a.shape[-1]
    while h < n:
        for i in range(0, n, 2 * h):
            x = a[..., i:i + h].copy()
            y = a[..., i + h:i + 2 * h].copy()
            a[..., i:i + h] = x + y
            a[..., i + h:i + 2 * h] = x - y
        h *= 2
    return a


# ------------------------------------------------------------------ pins: formats


def pin_fp16_exhaustive(orc):
    bits = np.arange(65536, dtype=np.uint32)
    ref = np_half(bits.astype(np.uint16))
    got = np.array([orc.half_to_double(int(b)) for b in bits])
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(got), nan)
    assert np.array_equal(got[~nan], ref[~nan])


def pin_bf16_exhaustive(orc):
    bits = np.arange(65536, dtype=np.uint32)
    ref = np_bf16(bits.astype(np.uint16))
    got = np.array([orc.bf16_to_double(int(b)) for b in bits])
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(got), nan)
    assert np.array_equal(got[~nan], ref[~nan])


# ------------------------------------------------------------------ pins: packing (Eq. 2)


def pin_pack_structured(orc):
    ones = np.ones((3, 64), np.int8)
    assert np.all(orc.pack_u(ones) == 0)
    assert np.all(orc.pack_u(-ones) == 0xFFFFFFFF)
    alt = np.tile(np.array([1, -1], np.int8), (3, 32))
    assert np.all(orc.pack_u(alt) == 0xAAAAAAAA)
    # rank 16: half a word, padding bits zero
    assert np.all(orc.pack_u(-np.ones((5, 16), np.int8)) == 0x0000FFFF)
    # V packs along rows
    assert np.all(orc.pack_v(-np.ones((64, 3), np.int8)) == 0xFFFFFFFF)
    assert np.all(orc.pack_v(np.tile(np.array([[1], [-1]], np.int8), (32, 3))) == 0xAAAAAAAA)
    assert np.all(orc.pack_v(-np.ones((40, 2), np.int8))[1] == 0x000000FF)
    # a lone -1 at element (o, j) sets exactly bit j%32 of word j//32 in row o
    s = np.ones((4, 70), np.int8)
    s[2, 37] = -1
    w = orc.pack_u(s)
    exp = np.zeros_like(w)
    exp[2, 1] = 1 << 5
    assert np.array_equal(w, exp)
    try:
        orc.pack_u(np.zeros((2, 8), np.int8))
    except ValueError:
        pass
    else:
        raise AssertionError("pack accepted a 0 sign")


def _np_pack_rows(signs: np.ndarray) -> np.ndarray:
    """Independent packer: numpy.packbits, little bit order, bytes -> uint32 LE."""
    rows, cols = signs.shape
    nw = (cols + 31) // 32
    bits = np.zeros((rows, nw * 32), np.uint8)
    bits[:, :cols] = (signs == -1)
    by = np.packbits(bits, axis=1, bitorder="little")
    return by.reshape(rows, nw, 4).astype(np.uint32) @ np.array([1, 1 << 8, 1 << 16, 1 << 24],
                                                                 dtype=np.uint32)


def pin_pack_vs_numpy(orc):
    rng = np.random.default_rng(7)
    for rows, cols in [(5, 1), (7, 31), (3, 32), (9, 33), (17, 100), (64, 192)]:
        s = (1 - 2 * rng.integers(0, 2, (rows, cols))).astype(np.int8)
        wu = orc.pack_u(s)
        assert np.array_equal(wu, _np_pack_rows(s))
        wv = orc.pack_v(s)
        assert np.array_equal(wv, _np_pack_rows(s.T).T)
        assert np.array_equal(orc.unpack_u(wu, rows, cols), s)
        assert np.array_equal(orc.unpack_v(wv, rows, cols), s)


# ------------------------------------------------------------------ pins: forward


def pin_dense_equals_factored(orc):
    """Prop. 1 is an identity: factored (Prop. 1) == dense (Eq. 4-6)."""
    rng = np.random.default_rng(11)
    for (d_in, d_out, rs, T) in [(40, 24, (3, 5), 3), (70, 33, (33, 1), 2), (64, 64, (16, 16), 4),
                                 (96, 17, (40,), 1)]:
        L = layer_from_signs(orc, d_in, d_out, [rand_path(rng, d_in, d_out, r) for r in rs])
        x = rand_x(rng, T, d_in)
        yd = orc.forward_dense(L, x)
        yf = orc.forward_factored(L, x)
        assert rel(yf, yd) <= 1e-12, rel(yf, yd)


def pin_rank1_closed_form(orc):
    """r = 1: W = h u l v^T g, so Y[t][o] = h_o u_o l * sum_i v_i g_i X[t][i]."""
    rng = np.random.default_rng(12)
    d_in, d_out, T = 77, 45, 3
    P = rand_path(rng, d_in, d_out, 1)
    L = layer_from_signs(orc, d_in, d_out, [P])
    x = rand_x(rng, T, d_in)
    X = np_bf16(x)
    u = P["u_signs"][:, 0].astype(np.float64)
    v = P["v_signs"][:, 0].astype(np.float64)
    s = X @ (v * np_half(P["g"]))
    ref = np.outer(s, np_half(P["h"]) * u * np_half(P["l"])[0])
    for y in (orc.forward_factored(L, x), orc.forward_dense(L, x)):
        assert rel(y, ref) <= 1e-14, rel(y, ref)


def pin_all_equal_signs(orc):
    """All +1 signs: Y[t][o] = h_o (sum_j l_j)(sum_i g_i X[t][i]); U all -1 negates it;
    U and V both all -1 leaves it unchanged."""
    rng = np.random.default_rng(13)
    d_in, d_out, r, T = 50, 20, 9, 2
    x = rand_x(rng, T, d_in)
    X = np_bf16(x)
    for su, sv, sign in [(1, 1, 1.0), (-1, 1, -1.0), (-1, -1, 1.0), (1, -1, -1.0)]:
        P = rand_path(rng, d_in, d_out, r)
        P["u_signs"] = np.full((d_out, r), su, np.int8)
        P["v_signs"] = np.full((d_in, r), sv, np.int8)
        L = layer_from_signs(orc, d_in, d_out, [P])
        ref = sign * np.outer(X @ np_half(P["g"]), np_half(P["h"])) * np_half(P["l"]).sum()
        y = orc.forward_factored(L, x)
        assert rel(y, ref) <= 1e-14, rel(y, ref)


def pin_hadamard_identity(orc):
    """Unit scales and U = V = H (Sylvester, r = d = 512): W = H H^T = d I, so
    Y = 512 X exactly.  With r < d, W x = H_r H_r^T x = FWHT(mask_r(FWHT(x)))."""
    d = 512
    H = sylvester(d)
    one = np.full(d, 0x3C00, np.uint16)  # fp16 1.0
    P = {"u_signs": H, "v_signs": H, "g": one, "l": one, "h": one}
    L = layer_from_signs(orc, d, d, [P])
    rng = np.random.default_rng(14)
    x = rand_x(rng, 3, d)
    y = orc.forward_factored(L, x)
    assert np.array_equal(y, 512.0 * np_bf16(x))
    d, r = 256, 200
    H = sylvester(d)
    P = {"u_signs": H[:, :r].copy(), "v_signs": H[:, :r].copy(),
         "g": np.full(d, 0x3C00, np.uint16), "l": np.full(r, 0x3C00, np.uint16),
         "h": np.full(d, 0x3C00, np.uint16)}
    L = layer_from_signs(orc, d, d, [P])
    x = rand_x(rng, 2, d)
    c = fwht(np_bf16(x))
    c[:, r:] = 0.0
    ref = fwht(c)
    assert np.array_equal(orc.forward_factored(L, x), ref)
    assert np.array_equal(orc.forward_dense(L, x), ref)


def pin_brute_force(orc):
    """Every sign pattern of a 2 -> 3 layer of rank 2: the oracle agrees with a
    hand-expanded sum_j sum_i h_o U[o][j] l_j V[i][j] g_i X[t][i]."""
    rng = np.random.default_rng(15)
    d_in, d_out, r, T = 2, 3, 2, 2
    P = rand_path(rng, d_in, d_out, r)
    x = rand_x(rng, T, d_in)
    X = np_bf16(x)
    g, l, h = np_half(P["g"]), np_half(P["l"]), np_half(P["h"])
    nbits = d_out * r + d_in * r
    for pattern in range(1 << nbits):
        bits = [(pattern >> k) & 1 for k in range(nbits)]
        U = np.array([1 - 2 * b for b in bits[:d_out * r]], np.int8).reshape(d_out, r)
        V = np.array([1 - 2 * b for b in bits[d_out * r:]], np.int8).reshape(d_in, r)
        Q = dict(P, u_signs=U, v_signs=V)
        L = layer_from_signs(orc, d_in, d_out, [Q])
        ref = np.zeros((T, d_out))
        for t in range(T):
            for o in range(d_out):
                acc = 0.0
                for j in range(r):
                    for i in range(d_in):
                        acc += h[o] * U[o, j] * l[j] * V[i, j] * g[i] * X[t, i]
                ref[t, o] = acc
        yf = orc.forward_factored(L, x)
        yd = orc.forward_dense(L, x)
        assert rel(yf, ref) <= 1e-14 and rel(yd, ref) <= 1e-14, pattern


def pin_residual_paths(orc):
    """Eq. 6: swapping the primary and residual paths leaves Y unchanged; a
    residual path with h_res = 0 reduces Y to the primary path alone."""
    rng = np.random.default_rng(16)
    d_in, d_out, T = 48, 40, 3
    A = rand_path(rng, d_in, d_out, 7)
    B = rand_path(rng, d_in, d_out, 12)
    x = rand_x(rng, T, d_in)
    y_ab = orc.forward_factored(layer_from_signs(orc, d_in, d_out, [A, B]), x)
    y_ba = orc.forward_factored(layer_from_signs(orc, d_in, d_out, [B, A]), x)
    assert rel(y_ab, y_ba) <= 1e-15
    y_a = orc.forward_factored(layer_from_signs(orc, d_in, d_out, [A]), x)
    y_b = orc.forward_factored(layer_from_signs(orc, d_in, d_out, [B]), x)
    assert rel(y_ab, y_a + y_b) <= 1e-15
    assert rel(y_a, y_b) > 0.1
    Z = dict(B, h=np.zeros(d_out, np.uint16))
    y_a0 = orc.forward_factored(layer_from_signs(orc, d_in, d_out, [A, Z]), x)
    assert np.array_equal(y_a0, y_a)


def pin_padding_ignored(orc):
    """Bits beyond r (U words) and beyond d_in (V words) carry no signs."""
    rng = np.random.default_rng(17)
    d_in, d_out, r, T = 40, 24, 16, 2
    P = rand_path(rng, d_in, d_out, r)
    L = layer_from_signs(orc, d_in, d_out, [P])
    x = rand_x(rng, T, d_in)
    y = orc.forward_factored(L, x)
    Lp = {"d_in": d_in, "d_out": d_out, "paths": [dict(L["paths"][0])]}
    Lp["paths"][0]["u_words"] = L["paths"][0]["u_words"] | np.uint32(0xFFFF0000)
    vw = L["paths"][0]["v_words"].copy()
    vw[-1] |= np.uint32(0xFFFFFF00)
    Lp["paths"][0]["v_words"] = vw
    assert np.array_equal(orc.forward_factored(Lp, x), y)
    assert np.array_equal(orc.forward_dense(Lp, x), orc.forward_dense(L, x))


# ------------------------------------------------------------------ pins: latent states


def pin_latent_hadamard(orc):
    """Unit scales, V = U = the first r columns of a Sylvester matrix H: the
    latent is the first r Walsh-Hadamard coefficients of X, and expanding
    coefficients c gives FWHT(c padded with zeros).  With two paths that
    split the columns of H (r_0 + r_1 = d), the latent is the whole transform
    in column order and expanding it gives d X (H H^T = d I)."""
    rng = np.random.default_rng(21)
    d = 256
    H = sylvester(d)
    one = lambda n: np.full(n, 0x3C00, np.uint16)  # fp16 1.0
    x = rand_x(rng, 3, d)
    c = fwht(np_bf16(x))
    for r in (200, 1):
        L = layer_from_signs(orc, d, d, [{"u_signs": H[:, :r].copy(), "v_signs": H[:, :r].copy(),
                                          "g": one(d), "l": one(r), "h": one(d)}])
        z = orc.latent(L, x)
        assert np.array_equal(z, c[:, :r])
        zp = np.zeros_like(c)
        zp[:, :r] = z
        assert np.array_equal(orc.expand(L, z), fwht(zp))
    r0 = 72
    L = layer_from_signs(orc, d, d, [
        {"u_signs": H[:, :r0].copy(), "v_signs": H[:, :r0].copy(), "g": one(d), "l": one(r0),
         "h": one(d)},
        {"u_signs": H[:, r0:].copy(), "v_signs": H[:, r0:].copy(), "g": one(d),
         "l": one(d - r0), "h": one(d)}])
    z = orc.latent(L, x)
    assert np.array_equal(z, c)
    assert np.array_equal(orc.expand(L, z), d * np_bf16(x))


def pin_latent_closed_forms(orc):
    """r = 1: z[t] = l v.(g X[t]); all-equal V signs s: z[t][j] = s l_j sum_i g_i X[t][i];
    expanding a one-hot latent e_j gives the column h . U[:, j] * 1."""
    rng = np.random.default_rng(22)
    d_in, d_out, T = 61, 29, 3
    x = rand_x(rng, T, d_in)
    X = np_bf16(x)
    P = rand_path(rng, d_in, d_out, 1)
    L = layer_from_signs(orc, d_in, d_out, [P])
    v = P["v_signs"][:, 0].astype(np.float64)
    ref = (X @ (v * np_half(P["g"])))[:, None] * np_half(P["l"])[0]
    assert rel(orc.latent(L, x), ref) <= 1e-14
    for sv in (1, -1):
        P = rand_path(rng, d_in, d_out, 9)
        P["v_signs"] = np.full((d_in, 9), sv, np.int8)
        L = layer_from_signs(orc, d_in, d_out, [P])
        ref = sv * np.outer(X @ np_half(P["g"]), np_half(P["l"]))
        assert rel(orc.latent(L, x), ref) <= 1e-14
        for j in (0, 4, 8):
            e = np.zeros((1, 9))
            e[0, j] = 1.0
            col = np_half(P["h"]) * P["u_signs"][:, j]
            assert np.array_equal(orc.expand(L, e)[0], col)


def pin_latent_brute_force(orc):
    """Every V sign pattern of a 2-input rank-2 path: the latent agrees with a
    hand-expanded l_j sum_i V[i][j] g_i X[t][i]; every U pattern of a 2 x 2 U:
    the expansion agrees with h_o sum_j U[o][j] z[t][j]."""
    rng = np.random.default_rng(23)
    d_in, d_out, r, T = 2, 2, 2, 2
    P = rand_path(rng, d_in, d_out, r)
    x = rand_x(rng, T, d_in)
    X = np_bf16(x)
    g, l, h = np_half(P["g"]), np_half(P["l"]), np_half(P["h"])
    Z = rng.standard_normal((T, r))
    for pattern in range(1 << (d_in * r)):
        S = np.array([1 - 2 * ((pattern >> k) & 1) for k in range(d_in * r)],
                     np.int8).reshape(d_in, r)
        L = layer_from_signs(orc, d_in, d_out, [dict(P, v_signs=S, u_signs=S)])
        zref = np.zeros((T, r))
        yref = np.zeros((T, d_out))
        for t in range(T):
            for j in range(r):
                for i in range(d_in):
                    zref[t, j] += l[j] * S[i, j] * g[i] * X[t, i]
            for o in range(d_out):
                for j in range(r):
                    yref[t, o] += h[o] * S[o, j] * Z[t, j]
        assert rel(orc.latent(L, x), zref) <= 1e-15, pattern
        assert rel(orc.expand(L, Z), yref) <= 1e-15, pattern


def pin_latent_expand_composition(orc):
    """Expanding the latent gives the forward (Prop. 1 split at its latent),
    checked against the dense Eq. 4-6 weight; a two-path latent is the two
    one-path latents side by side, and its expansion the sum of theirs."""
    rng = np.random.default_rng(24)
    for (d_in, d_out, rs, T) in [(40, 24, (3, 5), 3), (96, 17, (40,), 2), (64, 33, (17, 16), 2)]:
        paths = [rand_path(rng, d_in, d_out, r) for r in rs]
        L = layer_from_signs(orc, d_in, d_out, paths)
        x = rand_x(rng, T, d_in)
        z = orc.latent(L, x)
        assert z.shape == (T, sum(rs))
        y = orc.expand(L, z)
        yd = orc.forward_dense(L, x)
        assert rel(y, yd) <= 1e-12, rel(y, yd)
        if len(rs) == 2:
            L0 = layer_from_signs(orc, d_in, d_out, paths[:1])
            L1 = layer_from_signs(orc, d_in, d_out, paths[1:])
            z0, z1 = orc.latent(L0, x), orc.latent(L1, x)
            assert np.array_equal(z, np.concatenate([z0, z1], axis=1))
            ys = orc.expand(L0, z[:, :rs[0]]) + orc.expand(L1, z[:, rs[0]:])
            assert rel(y, ys) <= 1e-15


# ------------------------------------------------------------------ pins: accounting


def _golden_rows(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                rows.append(line.split())
    return rows


def pin_bpw_worked_examples(orc):
    for d_out, d_in, b, r, b_at_r in _golden_rows("bpw_worked_examples.txt"):
        d_out, d_in, b, r = int(d_out), int(d_in), float(b), int(r)
        r_real = orc.rank_for_bpw(b, d_out, d_in, 2)
        assert round(r_real) == r, (r_real, r)
        assert abs(orc.bpw(d_out, d_in, round(r_real), 2) - b) < 0.01
        if b_at_r != "-":
            # the paper prints b cut to 4 decimals (0.54987 -> "0.5498")
            assert 0.0 <= orc.bpw(d_out, d_in, r, 2) - float(b_at_r) < 1e-4
    # the rank solve inverts the accounting exactly, and one path halves the
    # sign and scale bits (App. E note on dropping Residual Compensation)
    for (d_out, d_in, r) in [(512, 512, 16), (8192, 28672, 320), (1024, 8192, 32)]:
        assert abs(orc.rank_for_bpw(orc.bpw(d_out, d_in, r, 2), d_out, d_in, 2) - r) < 1e-9
        assert abs(orc.bpw(d_out, d_in, r, 1) * 2 - orc.bpw(d_out, d_in, r, 2)) < 1e-15


def pin_theoretical_cost(orc):
    for T, d_out, d_in, r, mflops in _golden_rows("theoretical_cost.txt"):
        f = orc.flops(int(T), int(d_out), int(d_in), int(r), 1)
        assert abs(f / 1e6 - float(mflops)) < 0.05, f


# ------------------------------------------------------------------ pins: Dual-SVID (Sec. 3.2, 3.3)


def pin_svd_top_vs_numpy(orc):
    """The Jacobi SVD's r largest singular triples against numpy's LAPACK SVD
    (values, vectors up to the joint sign), orthonormality, the sign
    convention, and Eckart-Young: the rank-r error is the tail of the spectrum."""
    rng = np.random.default_rng(25)
    for m, n, r in [(40, 30, 5), (30, 40, 7), (24, 24, 24), (50, 17, 1)]:
        A = rng.standard_normal((m, n))
        s, U, V = orc.svd_top(A, r)
        Un, sn, Vtn = np.linalg.svd(A)
        assert np.allclose(s, sn[:r], rtol=1e-12, atol=0), (m, n, r)
        assert np.allclose(np.abs(np.sum(U * Un[:, :r], axis=0)), 1.0, atol=1e-10)
        assert np.allclose(np.abs(np.sum(V * Vtn[:r].T, axis=0)), 1.0, atol=1e-10)
        assert np.allclose(U.T @ U, np.eye(r), atol=1e-12)
        assert np.allclose(V.T @ V, np.eye(r), atol=1e-12)
        for j in range(r):
            k = int(np.argmax(np.abs(V[:, j])))
            assert V[k, j] > 0
        err = np.linalg.norm(A - (U * s) @ V.T) ** 2
        tail = float(np.sum(sn[r:] ** 2))
        assert abs(err - tail) <= 1e-10 * max(1.0, tail), (err, tail)


def pin_dual_svid_rank1(orc):
    """A rank-1 W = a b^T: the signs are those of a and b (jointly flipped so
    that the largest |b_i| is positive), |U'| and |V'| are rank-1 already, and
    the primary path reproduces W; the residual path then has nothing left."""
    rng = np.random.default_rng(26)
    a = rng.standard_normal(23)
    a[5] = 0.0  # a zero row of W: U' is 0 there, sign(0) = +1 and h = 0
    b = rng.standard_normal(19)
    W = np.outer(a, b)
    us, vs, h, g, l = orc.dual_svid_path(W, 1)
    flip = 1 if b[np.argmax(np.abs(b))] > 0 else -1
    assert us[5, 0] == 1 and h[5] == 0.0
    assert np.array_equal(us[:, 0], np.where(flip * a < 0, -1, 1).astype(np.int8))
    assert np.array_equal(vs[:, 0], np.where(flip * b < 0, -1, 1).astype(np.int8))
    assert rel(orc.path_weight(us, vs, h, g, l), W) <= 1e-13
    L = orc.dual_svid(W, [1, 1])
    h1 = np_half(L["paths"][1]["h"])
    g1 = np_half(L["paths"][1]["g"])
    # the residual is W minus the fp16-rounded primary path: small, and the
    # second path's W_hat is of its size, not of W's
    us1, vs1 = L["signs"][1]
    W1 = orc.path_weight(us1, vs1, h1, g1, np_half(L["paths"][1]["l"]))
    assert np.linalg.norm(W1) <= 5e-3 * np.linalg.norm(W)


def pin_dual_svid_hadamard(orc):
    """W = H_r diag(lam) H_r^T (Sylvester columns, distinct lam > 0) is a
    LittleBit weight with h = g = 1: Dual-SVID finds U_sign = V_sign = H_r up
    to one joint sign per column (all entries of a column tie in magnitude,
    so the sign convention falls to rounding there) and W_hat = W."""
    d, r = 64, 8
    H = sylvester(d)[:, :r].astype(np.float64)
    lam = np.array([9.0, 7.5, 6.0, 5.0, 4.0, 3.0, 2.0, 1.5])
    W = (H * lam) @ H.T
    us, vs, h, g, l = orc.dual_svid_path(W, r)
    flip = (us[0] * H[0]).astype(np.int8)
    assert np.array_equal(us, (H * flip).astype(np.int8))
    assert np.array_equal(vs, (H * flip).astype(np.int8))
    assert rel(orc.path_weight(us, vs, h, g, l), W) <= 1e-12
    # the scales factor the magnitudes: h and g constant, l proportional to lam
    assert np.ptp(h) <= 1e-12 * h.mean() and np.ptp(g) <= 1e-12 * g.mean()
    assert np.allclose(l / l[0], lam / lam[0], rtol=1e-12)


def pin_dual_svid_vs_lapack(orc):
    """Dual-SVID assembled from numpy's SVD (truncated SVD, then the leading
    singular pair of |U'| and |V'|) gives the same signs and W_hat as the
    oracle's Jacobi / power-iteration steps; and scaling W by c scales W_hat by
    c with the same signs."""
    rng = np.random.default_rng(27)
    m, n, r = 36, 28, 6
    A = rng.standard_normal((m, n)) * np.linspace(2.0, 0.5, n)
    us, vs, h, g, l = orc.dual_svid_path(A, r)
    Un, sn, Vtn = np.linalg.svd(A)
    Ur, Vr = Un[:, :r] * np.sqrt(sn[:r]), Vtn[:r].T * np.sqrt(sn[:r])
    for j in range(r):  # the oracle's joint sign convention
        if Vr[np.argmax(np.abs(Vr[:, j])), j] < 0:
            Ur[:, j], Vr[:, j] = -Ur[:, j], -Vr[:, j]
    assert np.array_equal(us, np.where(Ur < 0, -1, 1).astype(np.int8))
    assert np.array_equal(vs, np.where(Vr < 0, -1, 1).astype(np.int8))

    def rank1(M):
        u, s1, vt = np.linalg.svd(M)
        a, b = np.abs(u[:, 0]) * np.sqrt(s1[0]), np.abs(vt[0]) * np.sqrt(s1[0])
        return a, b
    hu, lu = rank1(np.abs(Ur))
    gv, lv = rank1(np.abs(Vr))
    W_ref = (hu[:, None] * np.where(Ur < 0, -1.0, 1.0) * (lu * lv)) @ \
        (gv[:, None] * np.where(Vr < 0, -1.0, 1.0)).T
    assert rel(orc.path_weight(us, vs, h, g, l), W_ref) <= 1e-9
    assert rel(h * g.mean() * l.mean(), hu * gv.mean() * (lu * lv).mean()) <= 1e-9
    us2, vs2, h2, g2, l2 = orc.dual_svid_path(3.0 * A, r)
    assert np.array_equal(us2, us) and np.array_equal(vs2, vs)
    assert rel(orc.path_weight(us2, vs2, h2, g2, l2), 3.0 * orc.path_weight(us, vs, h, g, l)) <= 1e-12


# ------------------------------------------------------------------ pins: QAT backward (SmoothSign)


def _train_layer(rng, d_in, d_out, rs, signs_only=False):
    paths = []
    for r in rs:
        u = rng.standard_normal((d_out, r))
        v = rng.standard_normal((d_in, r))
        if signs_only:
            u, v = np.where(u < 0, -1.0, 1.0), np.where(v < 0, -1.0, 1.0)
        paths.append({"r": r, "u": u, "v": v, "g": 0.2 + rng.random(d_in),
                      "l": 0.2 + rng.random(r), "h": 0.2 + rng.random(d_out)})
    return {"d_in": d_in, "d_out": d_out, "paths": paths}


def pin_train_forward_is_inference(orc):
    """The training forward on latent factors equals the inference forward
    (Prop. 1, pinned above) on their packed signs, for scales and inputs that
    fp16 / bf16 hold exactly."""
    rng = np.random.default_rng(28)
    d_in, d_out, T = 64, 40, 3
    L = _train_layer(rng, d_in, d_out, (8, 5))
    for P in L["paths"]:
        for key in ("g", "l", "h"):
            P[key] = np.asarray(P[key]).astype(np.float16).astype(np.float64)
    x = rand_x(rng, T, d_in)
    inf = {"d_in": d_in, "d_out": d_out, "paths": [
        {"r": P["r"], "u_words": orc.pack_u(np.where(P["u"] < 0, -1, 1).astype(np.int8)),
         "v_words": orc.pack_v(np.where(P["v"] < 0, -1, 1).astype(np.int8)),
         "g": half_bits(P["g"]), "l": half_bits(P["l"]), "h": half_bits(P["h"])}
        for P in L["paths"]]}
    assert rel(orc.train_forward(L, np_bf16(x)), orc.forward_factored(inf, x)) <= 1e-13


def pin_train_backward_central_differences(orc):
    """With the signs relaxed to the identity the loss sum(Y . dY) is linear in
    every single entry of h, g, l, X, S(U) and S(V), so a central difference
    of the forward gives each gradient entry up to rounding."""
    rng = np.random.default_rng(29)
    d_in, d_out, T = 24, 18, 5
    L = _train_layer(rng, d_in, d_out, (4, 3))
    X = rng.standard_normal((T, d_in))
    dY = rng.standard_normal((T, d_out))
    grads, dX = orc.train_backward(L, X, dY, relaxed=True)
    loss = lambda LL, XX: float(np.sum(orc.train_forward(LL, XX, relaxed=True) * dY))
    eps = 1e-3
    for p in range(2):
        for key, gkey in (("h", "dh"), ("g", "dg"), ("l", "dl"), ("u", "du"), ("v", "dv")):
            arr = L["paths"][p][key]
            for _ in range(3):
                idx = tuple(rng.integers(0, n) for n in arr.shape)
                old = arr[idx]
                arr[idx] = old + eps
                lp = loss(L, X)
                arr[idx] = old - eps
                lm = loss(L, X)
                arr[idx] = old
                fd = (lp - lm) / (2 * eps)
                assert abs(fd - grads[p][gkey][idx]) <= 1e-8 * max(1.0, abs(fd)), (p, key, fd)
    for _ in range(4):
        idx = (rng.integers(0, T), rng.integers(0, d_in))
        Xp, Xm = X.copy(), X.copy()
        Xp[idx] += eps
        Xm[idx] -= eps
        fd = (loss(L, Xp) - loss(L, Xm)) / (2 * eps)
        assert abs(fd - dX[idx]) <= 1e-8 * max(1.0, abs(fd))


def pin_smoothsign_factor(orc):
    """Through the sign the gradient is the sign-matrix gradient times the
    derivative of tanh(k x), k = 100: at latent U' = S(U) . a (a > 0, so the
    signs and the forward do not change) the backward equals the relaxed
    backward at S(U) times a central difference of numpy's tanh at U'."""
    rng = np.random.default_rng(30)
    d_in, d_out, T, k = 20, 16, 4, 100.0
    L = _train_layer(rng, d_in, d_out, (5,), signs_only=True)
    X = rng.standard_normal((T, d_in))
    dY = rng.standard_normal((T, d_out))
    ref, _ = orc.train_backward(L, X, dY, k=k, relaxed=True)
    P = L["paths"][0]
    au = rng.uniform(0.001, 0.03, P["u"].shape)
    av = rng.uniform(0.001, 0.03, P["v"].shape)
    L2 = {"d_in": d_in, "d_out": d_out, "paths": [dict(P, u=P["u"] * au, v=P["v"] * av)]}
    got, _ = orc.train_backward(L2, X, dY, k=k)
    hstep = 1e-7
    for lat, key in ((L2["paths"][0]["u"], "du"), (L2["paths"][0]["v"], "dv")):
        dtanh = (np.tanh(k * (lat + hstep)) - np.tanh(k * (lat - hstep))) / (2 * hstep)
        assert rel(got[0][key], ref[0][key] * dtanh) <= 1e-6, key
    for key in ("dg", "dl", "dh"):
        assert rel(got[0][key], ref[0][key]) <= 1e-13, key


def pin_kv_cache_table4(orc):
    """Table 4: the single-path rank for each target bits per weight of a
    d_model x d_model key/value projection (rounded up to a multiple of 8)
    and the reduction d_model / r of the cache when the latent replaces the
    d_model-wide key or value."""
    for d, b, r, factor in _golden_rows("kv_cache_table4.txt"):
        d, b, r, factor = int(d), float(b), int(r), float(factor)
        r_real = orc.rank_for_bpw(b, d, d, 1)
        assert int(np.ceil(r_real / 8.0)) * 8 == r, (b, r_real, r)
        assert orc.bpw(d, d, r, 1) >= b
        assert round(d / r, 1) == factor


# ------------------------------------------------------------------ pins: decode chain


def small_stack(rng, n_layers=3, d=64, dkv=16, dff=96, rq=8, rkv=4, rm=12):
    from paper_2506_13771_gb300 import inputs
    shapes = inputs.stack_shapes(d, dkv, dff, rq, rkv, rm)
    layers = []
    for _ in range(n_layers):
        for (di, do, r) in shapes:
            layers.append(inputs.make_linear(rng, di, do, r, 2, inputs.unit_gain_scale(di, r)))
    x0 = inputs.bf16_normal(rng, (d,))
    return layers, x0


def _rho(v):
    return v / np.sqrt(np.mean(v * v))


def _attention(q, k_cache, v_cache, head_dim):
    """Textbook grouped-query attention of one query over a cached sequence:
    per query head, softmax(q_h . k_{g,s} / sqrt(head_dim)) over positions s,
    then the weighted sum of v_{g,s}; g = the kv head the query head shares."""
    n_q = q.shape[0] // head_dim
    n_kv = k_cache.shape[1] // head_dim
    out = np.zeros_like(q)
    for hq in range(n_q):
        g = hq // (n_q // n_kv)
        qh = q[hq * head_dim:(hq + 1) * head_dim]
        ks = k_cache[:, g * head_dim:(g + 1) * head_dim]
        vs = v_cache[:, g * head_dim:(g + 1) * head_dim]
        s = ks @ qh / np.sqrt(head_dim)
        w = np.exp(s - s.max())
        w /= w.sum()
        out[hq * head_dim:(hq + 1) * head_dim] = w @ vs
    return out


def pin_stack_chain(orc):
    """The decoder chain re-built from single-linear oracle calls, numpy RMS
    normalisation, SiLU and textbook attention over the one cached position."""
    rng = np.random.default_rng(18)
    hd = 8
    layers, x0 = small_stack(rng)
    out, qs, kv = orc.stack_forward(layers, x0, head_dim=hd)
    a = np_bf16(x0)
    for l in range(len(layers) // 7):
        Q, K, V, O, G, Up, D = layers[7 * l:7 * l + 7]
        n = _rho(a)[None, :]
        q = orc.apply_factored(Q, n)[0]
        k = orc.apply_factored(K, n)[0]
        v = orc.apply_factored(V, n)[0]
        assert rel(qs[l], q) <= 1e-12 and rel(kv[l, 0], k) <= 1e-12 and rel(kv[l, 1], v) <= 1e-12
        attn = _attention(q, k[None, :], v[None, :], hd)
        h = a + orc.apply_factored(O, attn[None, :])[0]
        n = _rho(h)[None, :]
        gt = orc.apply_factored(G, n)[0]
        m = gt / (1.0 + np.exp(-gt)) * orc.apply_factored(Up, n)[0]
        a = h + orc.apply_factored(D, m[None, :])[0]
    assert rel(out, a) <= 1e-12, rel(out, a)


def pin_stack_zero_branches(orc):
    """With h = 0 in every O and Down path no branch reaches the residual
    stream: the output is x0 exactly, while q, k, v are still produced."""
    rng = np.random.default_rng(19)
    layers, x0 = small_stack(rng)
    for l in range(len(layers) // 7):
        for idx in (3, 6):
            for P in layers[7 * l + idx]["paths"]:
                P["h"] = np.zeros_like(P["h"])
    out, qs, kv = orc.stack_forward(layers, x0, head_dim=8)
    assert np.array_equal(out, np_bf16(x0))
    n = _rho(np_bf16(x0))[None, :]
    for l in range(len(layers) // 7):
        assert rel(qs[l], orc.apply_factored(layers[7 * l], n)[0]) <= 1e-12
        assert rel(kv[l, 1], orc.apply_factored(layers[7 * l + 2], n)[0]) <= 1e-12


def pin_stack_attention_closed_form(orc):
    """Down switched off (h = 0) and O = the unit-scale Sylvester-Hadamard
    linear (W = d I): every layer adds exactly d * broadcast(v) to the stream."""
    rng = np.random.default_rng(20)
    d, dkv, hd = 64, 16, 8
    layers, x0 = small_stack(rng, d=d, dkv=dkv)
    H = sylvester(d)
    one = np.full(d, 0x3C00, np.uint16)
    for l in range(len(layers) // 7):
        layers[7 * l + 3] = layer_from_signs(orc, d, d, [{"u_signs": H, "v_signs": H,
                                                           "g": one, "l": one, "h": one}])
        for P in layers[7 * l + 6]["paths"]:
            P["h"] = np.zeros_like(P["h"])
    out, _, kv = orc.stack_forward(layers, x0, head_dim=hd)
    a = np_bf16(x0)
    for l in range(len(layers) // 7):
        v = orc.apply_factored(layers[7 * l + 2], _rho(a)[None, :])[0]
        assert rel(kv[l, 1], v) <= 1e-12
        bcast = np.concatenate([v[(hq // (d // dkv)) * hd:(hq // (d // dkv) + 1) * hd]
                                for hq in range(d // hd)])
        a = a + d * bcast
    assert rel(out, a) <= 1e-13, rel(out, a)


# ------------------------------------------------------------------ pins: decode step at position p


def _bf16_rne_of_f32(f32: np.ndarray) -> np.ndarray:
    """bf16 rounding of float32 values by the integer carry trick (ties to even)."""
    u = np.asarray(f32, dtype=np.float32).view(np.uint32).astype(np.uint64)
    r = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16) << 16
    return r.astype(np.uint32).view(np.float32).astype(np.float64)


def pin_round_bf16(orc):
    """Nearest-even bf16 rounding: equal to the integer carry trick on float32
    inputs (random values, exact ties with even and odd kept bits, tiny and
    subnormal magnitudes); for float64 inputs between float32 values the
    result is a bf16 value within half a bf16 step, and just above a tie it
    rounds away from the tie's even neighbour."""
    rng = np.random.default_rng(30)
    f = np.concatenate([rng.standard_normal(3000) * 10.0 ** rng.integers(-30, 30, 3000),
                        rng.standard_normal(200) * 1e-39]).astype(np.float32)
    # exact ties: the low 16 bits of finite float32 values set to 0x8000, with
    # the last kept bit both even and odd
    u = (rng.standard_normal(400).astype(np.float32).view(np.uint32) & 0xFFFF0000) | 0x8000
    ties = np.concatenate([u, u ^ 0x00010000]).view(np.float32)
    f = np.concatenate([f, ties])
    assert np.array_equal(orc.round_bf16(f.astype(np.float64)), _bf16_rne_of_f32(f))
    v = rng.standard_normal(500) * 3.0
    r = orc.round_bf16(v)
    assert np.array_equal(_bf16_rne_of_f32(r.astype(np.float32)), r)  # representable
    e = np.floor(np.log2(np.abs(v)))
    assert np.all(np.abs(v - r) <= np.ldexp(1.0, (e - 8).astype(int)) * (1 + 1e-12))
    # 1 + 2^-8 is a tie between 1 and 1 + 2^-7 (kept bit even: down); a hair above it rounds up
    assert orc.round_bf16(1 + 2.0 ** -8) == 1.0
    assert orc.round_bf16(1 + 2.0 ** -8 + 2.0 ** -40) == 1 + 2.0 ** -7


def pin_rope(orc):
    """Rotary embedding: the half-split pairing and frequencies on unit vectors
    (closed forms), identity at position 0, norm preservation, composition of
    rotations, and scores that depend only on the position difference."""
    c1, s1 = np.cos(1.0), np.sin(1.0)
    assert np.allclose(orc.rope([1.0, 0.0], 1), [c1, s1], rtol=0, atol=1e-15)
    assert np.allclose(orc.rope([1.0, 0.0, 0.0, 0.0], 1), [c1, 0.0, s1, 0.0], rtol=0, atol=1e-15)
    th = 10000.0 ** -0.5
    assert np.allclose(orc.rope([0.0, 1.0, 0.0, 0.0], 1), [0.0, np.cos(th), 0.0, np.sin(th)],
                       rtol=0, atol=1e-15)
    assert np.allclose(orc.rope([0.0, 0.0, 0.0, 1.0], 3), [0.0, -np.sin(3 * th), 0.0, np.cos(3 * th)],
                       rtol=0, atol=1e-15)
    rng = np.random.default_rng(31)
    x, y = rng.standard_normal(128), rng.standard_normal(128)
    assert np.array_equal(orc.rope(x, 0), x)
    assert abs(np.linalg.norm(orc.rope(x, 77)) - np.linalg.norm(x)) <= 1e-12
    assert np.allclose(orc.rope(orc.rope(x, 5), 9), orc.rope(x, 14), rtol=0, atol=1e-12)
    for p, t, sh in ((9, 3, 40), (100, 0, 7), (5, 5, 1000)):
        a = orc.rope(x, p) @ orc.rope(y, t)
        b = orc.rope(x, p + sh) @ orc.rope(y, t + sh)
        assert abs(a - b) <= 1e-10 * (1 + abs(a)), (a, b)


DEC = {"n_heads": 8, "n_kv_heads": 2, "head_dim": 8, "rope_base": 10000.0}


def _decode_tokens(orc, layers, xs, max_pos, round_inputs=True):
    n_layers = len(layers) // 7
    dkv = layers[1]["d_out"]
    kc = np.zeros((n_layers, max_pos, dkv))
    vc = np.zeros((n_layers, max_pos, dkv))
    outs = []
    for p, x in enumerate(xs):
        outs.append(orc.decoder_step(layers, DEC, p, x, kc, vc, round_inputs)[0])
    return outs, kc, vc


def pin_decoder_pos0_is_stack(orc):
    """At position 0 (exact inputs) the rotation is the identity and the
    softmax of one score is 1: the step equals the position-0 stack chain."""
    rng = np.random.default_rng(32)
    layers, x0 = small_stack(rng)
    out_s, _, kv = orc.stack_forward(layers, x0, head_dim=8)
    kc = np.zeros((3, 4, 16))
    vc = np.zeros((3, 4, 16))
    out, _, _ = orc.decoder_step(layers, DEC, 0, x0, kc, vc, round_inputs=False)
    assert rel(out, out_s) <= 1e-12, rel(out, out_s)
    assert rel(kc[:, 0], kv[:, 0]) <= 1e-12 and rel(vc[:, 0], kv[:, 1]) <= 1e-12
    assert not kc[:, 1:].any() and not vc[:, 1:].any()


def pin_decoder_composition(orc):
    """Step 3 rebuilt from single-linear oracle calls, numpy RMS, the pinned
    bf16 rounding and rotation, and textbook attention over cache rows 0..3."""
    rng = np.random.default_rng(33)
    layers, _ = small_stack(rng)
    xs = [inputs_bf16(rng, 64) for _ in range(4)]
    _, kc, vc = _decode_tokens(orc, layers, xs[:3], 6)
    kc0, vc0 = kc.copy(), vc.copy()
    out, attn, qk = orc.decoder_step(layers, DEC, 3, xs[3], kc, vc, True, True, True)
    a = np_bf16(xs[3])
    D = DEC["head_dim"]
    for l in range(3):
        Q, K, V, O, G, Up, Dn = layers[7 * l:7 * l + 7]
        n = orc.round_bf16(_rho(a))[None, :]
        q = orc.apply_factored(Q, n)[0]
        k = orc.apply_factored(K, n)[0]
        v = orc.apply_factored(V, n)[0]
        q = np.concatenate([orc.rope(q[h * D:(h + 1) * D], 3) for h in range(8)])
        k = np.concatenate([orc.rope(k[g * D:(g + 1) * D], 3) for g in range(2)])
        assert rel(qk[l], np.concatenate([q, k])) <= 1e-12
        assert rel(kc[l, 3], k) <= 1e-12 and rel(vc[l, 3], v) <= 1e-12
        assert np.array_equal(kc[l, :3], kc0[l, :3]) and not kc[l, 4:].any()
        at = _attention(q, np.vstack([kc0[l, :3], k]), np.vstack([vc0[l, :3], v]), D)
        assert rel(attn[l], at) <= 1e-12, rel(attn[l], at)
        h = a + orc.apply_factored(O, orc.round_bf16(at)[None, :])[0]
        n = orc.round_bf16(_rho(h))[None, :]
        gt = orc.apply_factored(G, n)[0]
        m = orc.round_bf16(gt / (1.0 + np.exp(-gt)) * orc.apply_factored(Up, n)[0])
        a = h + orc.apply_factored(Dn, m[None, :])[0]
    assert rel(out, a) <= 1e-12, rel(out, a)


def inputs_bf16(rng, n):
    return rand_x(rng, 1, n)[0]


def pin_decoder_attention_closed_forms(orc):
    """One layer, two kv heads shared by four query heads each.  (a) Cached
    keys equal to the new key: uniform weights, each head reads the mean of
    its kv head's values.  (b) Position 1 with a zero key at row 0: the
    weights are a logistic function of q . k / sqrt(head_dim)."""
    rng = np.random.default_rng(34)
    layers, _ = small_stack(rng, n_layers=1)
    x = inputs_bf16(rng, 64)
    D, p = DEC["head_dim"], 5
    kc = np.zeros((1, 8, 16))
    vc = rng.standard_normal((1, 8, 16))
    _, _, qk = orc.decoder_step(layers, DEC, p, x, kc.copy(), vc.copy(), True, False, True)
    kc[0, :p] = qk[0, 64:]
    _, attn, _ = orc.decoder_step(layers, DEC, p, x, kc, vc, True, True, False)
    for h in range(8):
        g = h // 4
        want = vc[0, :p + 1, g * D:(g + 1) * D].mean(axis=0)
        assert rel(attn[0, h * D:(h + 1) * D], want) <= 1e-12
    kc = np.zeros((1, 4, 16))
    vc = np.zeros((1, 4, 16))
    vc[0, 0] = rng.standard_normal(16)
    _, attn, qk = orc.decoder_step(layers, DEC, 1, x, kc, vc, True, True, True)
    q, k = qk[0, :64], qk[0, 64:]
    for h in range(8):
        g = h // 4
        s = q[h * D:(h + 1) * D] @ k[g * D:(g + 1) * D] / np.sqrt(D)
        w1 = 1.0 / (1.0 + np.exp(-s))
        want = (1 - w1) * vc[0, 0, g * D:(g + 1) * D] + w1 * vc[0, 1, g * D:(g + 1) * D]
        assert rel(attn[0, h * D:(h + 1) * D], want) <= 1e-12


def pin_decoder_causal(orc):
    """Cache rows after the current position are never read (NaN there
    changes nothing), and position max_pos is refused."""
    rng = np.random.default_rng(35)
    layers, _ = small_stack(rng, n_layers=2)
    xs = [inputs_bf16(rng, 64) for _ in range(3)]
    outs, kc, vc = _decode_tokens(orc, layers, xs, 5)
    kc2, vc2 = kc.copy(), vc.copy()
    kc2[:, 3:] = np.nan
    vc2[:, 3:] = np.nan
    kc[:, 2:] = 0.0
    vc[:, 2:] = 0.0
    kc2[:, 2] = 0.0
    vc2[:, 2] = 0.0
    a = orc.decoder_step(layers, DEC, 2, xs[2], kc, vc)[0]
    b = orc.decoder_step(layers, DEC, 2, xs[2], kc2, vc2)[0]
    assert np.all(np.isfinite(b)) and np.array_equal(a, b) and np.array_equal(a, outs[2])
    try:
        orc.decoder_step(layers, DEC, 5, xs[0], kc, vc)
    except ValueError:
        pass
    else:
        raise AssertionError("position max_pos accepted")


ALL_PINS = [pin_fp16_exhaustive, pin_bf16_exhaustive, pin_pack_structured, pin_pack_vs_numpy,
            pin_dense_equals_factored, pin_rank1_closed_form, pin_all_equal_signs,
            pin_hadamard_identity, pin_brute_force, pin_residual_paths, pin_padding_ignored,
            pin_latent_hadamard, pin_latent_closed_forms, pin_latent_brute_force,
            pin_latent_expand_composition, pin_bpw_worked_examples, pin_theoretical_cost,
            pin_kv_cache_table4, pin_svd_top_vs_numpy, pin_dual_svid_rank1,
            pin_dual_svid_hadamard, pin_dual_svid_vs_lapack, pin_train_forward_is_inference,
            pin_train_backward_central_differences, pin_smoothsign_factor, pin_stack_chain,
            pin_stack_zero_branches, pin_stack_attention_closed_form, pin_round_bf16, pin_rope,
            pin_decoder_pos0_is_stack, pin_decoder_composition,
            pin_decoder_attention_closed_forms, pin_decoder_causal]
