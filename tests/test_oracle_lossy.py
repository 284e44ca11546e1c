"""Pins of the lossy-comparator oracle against cases whose answer is known
without it: a row with planted large entries (top-k), ties, a row of +-c (sign
quantization is then exact), an exactly low-rank batch (the truncated SVD
recovers it), the Eckart-Young error of the truncated SVD (the sum of the
discarded squared singular values, from numpy's eigvalsh of X^T X), the fp8
e4m3 encoding and decoding against torch's float8_e4m3fn casts (every tie of
the format included), int8 codes of a row whose scale is exactly 1 (rounding
half to even by hand), the row maximum mapping to +-qmax, and the rounding
error bounds of both 8-bit formats."""
import importlib.util
import os

import numpy as np
import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "..", "oracle", "lossy.py")


def load(text=None):
    spec = importlib.util.spec_from_loader("lossy_under_test", loader=None)
    mod = importlib.util.module_from_spec(spec)
    exec(compile(text if text is not None else open(SRC).read(), SRC, "exec"), mod.__dict__)
    return mod


def bf16(x):
    x = np.asarray(x, np.float32)
    u = x.view(np.uint32)
    return ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)


def pin_topk_planted(o):
    rng = np.random.default_rng(0)
    x = rng.uniform(-1, 1, (3, 40))
    planted = [[3, 17, 29], [0, 1, 39], [5, 6, 7]]
    for t, cs in enumerate(planted):
        for j, c in enumerate(cs):
            x[t, c] = (10 + j) * (-1) ** j
    cols = o.topk_columns(bf16(x), 3)
    return all(list(cols[t]) == sorted(planted[t]) for t in range(3))


def pin_topk_ties_lower_index(o):
    x = np.array([[1.0, -2.0, 2.0, 0.5, -2.0, 2.0]])
    return list(o.topk_columns(bf16(x), 2)[0]) == [1, 2]


def pin_topk_restore(o):
    vals = np.array([[5.0, -7.0]])
    X = o.topk_restore(vals, np.array([[1, 3]]), 5)
    return np.array_equal(X, np.array([[0, 5.0, 0, -7.0, 0]]))


def pin_sign_exact_on_pm_c(o):
    rng = np.random.default_rng(1)
    c = rng.uniform(0.5, 2, (4, 1))
    X = c * rng.choice([-1.0, 1.0], (4, 33))
    bits, scale = o.sign_compress(X)
    return np.allclose(o.sign_restore(bits, scale), X, rtol=0, atol=1e-15) and bits.dtype == np.uint8


def pin_sign_scale_is_mean_magnitude(o):
    bits, scale = o.sign_compress(np.array([[1.0, -3.0, 0.0, 4.0]]))
    return list(bits[0]) == [0, 1, 0, 0] and abs(scale[0] - 2.0) <= 1e-15


def pin_lowrank_recovers_rank_r(o):
    rng = np.random.default_rng(2)
    X = rng.standard_normal((50, 4)) @ rng.standard_normal((4, 30))
    return np.allclose(o.lowrank(X, 4), X, atol=1e-10)


def pin_lowrank_eckart_young(o):
    rng = np.random.default_rng(3)
    X = rng.standard_normal((40, 25))
    ev = np.sort(np.linalg.eigvalsh(X.T @ X))          # squared singular values, ascending
    err2 = np.sum((X - o.lowrank(X, 6)) ** 2)
    return abs(err2 - ev[:-6].sum()) <= 1e-8 * ev.sum()


def pin_wire_sizes(o):
    return (o.wire_bytes("subspace", 10, 8192, k=82) == 1640
            and o.wire_bytes("topk", 10, 8192, kk=41) == 1640
            and o.wire_bytes("sign", 10, 8192) == 10 * 1024 + 40
            and o.wire_bytes("lowrank", 10, 8192, r=2) == 4 * 8202
            and o.wire_bytes("int8", 10, 8192) == o.wire_bytes("e4m3", 10, 8192) == 10 * 8196)


def _e4m3_grid():
    """Every finite e4m3 magnitude (0 .. 448) from the format's definition:
    subnormals m * 2^-9 and normals (8 + m) * 2^(E - 10), E = 1..15."""
    sub = [m * 2.0 ** -9 for m in range(8)]
    nor = [(8 + m) * 2.0 ** (E - 10) for E in range(1, 16) for m in range(8)]
    return np.array(sorted(set(sub + nor[:-1])))           # S.1111.111 is NaN


def pin_e4m3_encode_matches_torch(o):
    torch = pytest.importorskip("torch")
    g = _e4m3_grid()
    mids = (g[1:] + g[:-1]) / 2                           # every tie
    rng = np.random.default_rng(4)
    rnd = rng.standard_normal(20000) * np.exp2(rng.uniform(-12, 9, 20000))
    v = np.concatenate([g, mids, -g, -mids, rnd, [1e-30, -1e-30, 447.9, 455.0, -463.0]])
    v = v[np.abs(v) < 464].astype(np.float32)
    ref = torch.from_numpy(v).to(torch.float8_e4m3fn).view(torch.uint8).numpy()
    got = o.e4m3_encode(v)
    return (np.array_equal(got, ref) and got[len(g) - 1] == 0x7E
            and o.e4m3_encode(np.float32([500.0, -1e4]))[1] == 0xFE)


def pin_e4m3_decode_matches_torch(o):
    torch = pytest.importorskip("torch")
    codes = np.arange(256, dtype=np.uint8)
    ref = torch.from_numpy(codes).view(torch.float8_e4m3fn).float().numpy().astype(np.float64)
    got = o.e4m3_decode(codes)
    return np.array_equal(np.isnan(got), np.isnan(ref)) and np.array_equal(
        got[~np.isnan(got)], ref[~np.isnan(ref)]) and got[0x7E] == 448.0


def pin_int8_codes_closed_form(o):
    # a = 127 makes r = 127 / a = 1 exactly, so the codes are x rounded half to even
    x = np.array([[127.0, -0.5, 0.5, 1.5, 2.5, -2.5, 126.5, 3.0, -127.0, 0.25]])
    codes, scale = o.quant_compress(bf16(x), "int8")
    want = np.array([127, 0, 0, 2, 2, -2, 126, 3, -127, 0], np.int8)
    return np.array_equal(codes.view(np.int8)[0], want) and scale[0] == np.float32(1.0)


def pin_quant_zero_row(o):
    z = bf16(np.zeros((2, 16)))
    ok = True
    for fmt in ("int8", "e4m3"):
        codes, scale = o.quant_compress(z, fmt)
        ok = ok and not codes.any() and not scale.any()
        ok = ok and not o.quant_restore(codes, scale, fmt).any()
    return ok


def pin_quant_row_max_is_exact(o):
    # the largest magnitude maps to +-qmax and restores to itself
    rng = np.random.default_rng(5)
    x = rng.standard_normal((6, 64)) * np.exp2(rng.uniform(-6, 6, (6, 1)))
    b = bf16(x)
    xf = o.bf16_bits_to_f32(b)
    j = np.argmax(np.abs(xf), axis=1)
    ok = True
    for fmt, top in (("int8", 127), ("e4m3", 448)):
        codes, scale = o.quant_compress(b, fmt)
        dq = o.quant_decode(codes, fmt)
        back = o.quant_restore(codes, scale, fmt)
        rows = np.arange(6)
        ok = ok and np.array_equal(np.abs(dq[rows, j]), np.full(6, float(top)))
        ok = ok and np.array_equal(back[rows, j], b[rows, j])
    return ok


def pin_quant_error_bounds(o):
    # int8: within half a code of x * r; e4m3: within half an ulp of the
    # format (2^-4 relative for normals, 2^-10 absolute on the subnormal grid)
    rng = np.random.default_rng(6)
    x = rng.standard_normal((8, 256)) * np.exp2(rng.uniform(-3, 3, (8, 256)))
    b = bf16(x)
    xf = o.bf16_bits_to_f32(b).astype(np.float64)
    ok = True
    for fmt in ("int8", "e4m3"):
        codes, scale = o.quant_compress(b, fmt)
        qmax = 127.0 if fmt == "int8" else 448.0
        u = xf * (qmax / np.abs(xf).max(axis=1))[:, None]       # x in code units
        err = np.abs(o.quant_decode(codes, fmt) - u)
        lim = 0.5 + 1e-4 if fmt == "int8" else np.maximum(2.0 ** -4 * np.abs(u), 2.0 ** -10) * (1 + 1e-4)
        ok = ok and bool(np.all(err <= lim))
    return ok


PINS = [pin_topk_planted, pin_topk_ties_lower_index, pin_topk_restore, pin_sign_exact_on_pm_c,
        pin_sign_scale_is_mean_magnitude, pin_lowrank_recovers_rank_r, pin_lowrank_eckart_young, pin_wire_sizes,
        pin_e4m3_encode_matches_torch, pin_e4m3_decode_matches_torch, pin_int8_codes_closed_form,
        pin_quant_zero_row, pin_quant_row_max_is_exact, pin_quant_error_bounds]


@pytest.mark.parametrize("pin", PINS, ids=[p.__name__ for p in PINS])
def test_lossy_oracle_pins(pin):
    assert pin(load())


MUTANTS = {
    "ties_higher_index": ("key=lambda c: (-mag[t, c], c)", "key=lambda c: (-mag[t, c], -c)"),
    "smallest_magnitudes": ("key=lambda c: (-mag[t, c], c)", "key=lambda c: (mag[t, c], c)"),
    "sign_of_positive": ("(X < 0).astype(np.uint8)", "(X > 0).astype(np.uint8)"),
    "scale_rms": ("np.abs(X).mean(axis=1)", "np.sqrt((X * X).mean(axis=1))"),
    "lowrank_off_by_one": ("(Uu[:, :r] * s[:r]) @ Vt[:r]", "(Uu[:, :r - 1] * s[:r - 1]) @ Vt[:r - 1]"),
    "index_bytes": ("return T * kk * (2 + 2)", "return T * kk * (2 + 4)"),
    "int8_round_down": ("np.clip(np.rint(p), -127, 127)", "np.clip(np.floor(p), -127, 127)"),
    "e4m3_ties_up": ("n = np.rint(v / np.exp2(e - 3.0))", "n = np.floor(v / np.exp2(e - 3.0) + 0.5)"),
    "e4m3_bias_8": ("(e + 7) * 8 + (n - 8)", "(e + 8) * 8 + (n - 8)"),
    "e4m3_no_subnormals": ("e = np.maximum(e, -6)", "e = np.maximum(e, -7)"),
    "scale_mean_not_max": ("a = np.abs(x).max(axis=1)", "a = np.abs(x).mean(axis=1)"),
    "restore_without_scale": ("f32_to_bf16_bits(q * np.asarray(scale, np.float32)[:, None])",
                              "f32_to_bf16_bits(q + 0 * np.asarray(scale, np.float32)[:, None])"),
    "decode_bias_6": ("(8 + M) * np.exp2(E - 10.0)", "(8 + M) * np.exp2(E - 9.0)"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_lossy_mutants_are_caught(name):
    a, b = MUTANTS[name]
    text = open(SRC).read()
    assert a in text
    mod = load(text.replace(a, b))
    failed = []
    for pin in PINS:
        try:
            ok = pin(mod)
        except Exception:
            ok = False
        if not ok:
            failed.append(pin.__name__)
    assert failed, "mutant %s passed every pin" % name
