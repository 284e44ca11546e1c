"""GPU parity: every boundary call of the C ABI against the fp64 oracle.

Bar (relative Frobenius error against the oracle's unrounded fp64 value):
1e-2 for bf16 outputs, 1e-5 for fp32 outputs; bit-exact for gathers, wire byte
counts and layouts.  Sizes span several 128-token tiles with ragged tails, k
from 1 to 128, d from 16 to 16384 (including widths that end in a partial
64-column chunk and 128-column block); guard bands around every output catch
out-of-bounds writes.
"""
import ctypes

import numpy as np
import pytest
import torch

from gpu_util import assert_parity, dev, dtname, guarded, guards_intact, host, widen
from paper_2506_01260_gb300 import workloads as W

pytestmark = pytest.mark.gpu

# (name, T, seq_len, d, k, vocab)
CASES = [
    ("ragged_d512_k20", 1000, 300, 512, 20, 3000),
    ("short_d256_k8", 333, 128, 256, 8, 1024),
    ("tiles_d1024_k41", 4173, 1024, 1024, 41, 5000),
    ("kmax_d2048_k128", 300, 100, 2048, 128, 777),
    ("wide_d8192_k82", 260, 4096, 8192, 82, 1000),
    ("one_token_d64_k1", 1, 7, 64, 1, 5),
    ("square_d16_k16", 70, 9, 16, 16, 33),
    ("exact_tile_d256_k16", 256, 128, 256, 16, 300),
    ("ragged_chunk_d200_k24", 300, 50, 200, 24, 700),      # d: 3 chunks of 64 + 8; blocks 128 + 72
    ("ragged_chunk_d2056_k33", 257, 64, 2056, 33, 900),
    ("wide_d12288_k96", 150, 64, 12288, 96, 400),
    ("wide_d16384_k128", 131, 32, 16384, 128, 300),
]
DTYPES = ["bf16", "f32"]


def case_inputs(name, T, n, d, k, vocab, dtype, seed=0):
    wl = W.Workload(name, 1, n, d, k, vocab, 1000 + seed + d + k, off_scale=1e-2, grad=True)
    return W.generate(wl, T=T, dtype=dtype)


@pytest.fixture(scope="module")
def bases():
    return {}


@pytest.mark.parametrize("dtype", DTYPES)
@pytest.mark.parametrize("case", CASES, ids=[c[0] for c in CASES])
def test_forward_round_trip(sn, oracle, case, dtype):
    name, T, n, d, k, vocab = case
    inp = case_inputs(name, T, n, d, k, vocab, dtype)
    basis = sn.Basis(dev(inp["U"]))
    X, tok, pe, ids = dev(inp["X"]), dev(inp["tok_emb"]), dev(inp["pos_emb"]), dev(inp["ids"])
    tdt = X.dtype
    fullC, C = guarded((T, k), tdt)
    sn.sn_compress_fwd(basis, X, ids, tok, n, pos_emb=pe, out=C)
    fullX, Xr = guarded((T, d), tdt)
    sn.sn_decompress_fwd(basis, C, ids, tok, n, pos_emb=pe, out=Xr)
    sn.sn_check_errors(basis)
    assert guards_intact(fullC) and guards_intact(fullX)
    _, C64, st = oracle.compress_fwd(inp["X"], inp["ids"], inp["tok_emb"], inp["U"], n,
                                     pos_emb=inp["pos_emb"])
    assert st == 0
    assert_parity(host(C), C64, dtype)
    _, X64, _ = oracle.decompress_fwd(host(C), inp["ids"], inp["tok_emb"], inp["U"], n,
                                      pos_emb=inp["pos_emb"])
    assert_parity(host(Xr), X64, dtype)
    # wire layout: C is a contiguous [T, k] slab, T*k elements, nothing else
    assert sn.sn_wire_bytes(basis, tdt, T) == T * k * (2 if dtype == "bf16" else 4)
    basis.destroy()


@pytest.mark.parametrize("dtype", DTYPES)
@pytest.mark.parametrize("case", CASES, ids=[c[0] for c in CASES])
def test_backward_round_trip(sn, oracle, case, dtype):
    name, T, n, d, k, vocab = case
    inp = case_inputs(name, T, n, d, k, vocab, dtype)
    basis = sn.Basis(dev(inp["U"]))
    G = dev(inp["G"])
    fullC, C = guarded((T, k), G.dtype)
    sn.sn_compress_bwd(basis, G, out=C)
    fullG, Gr = guarded((T, d), G.dtype)
    sn.sn_decompress_bwd(basis, C, out=Gr)
    sn.sn_check_errors(basis)
    assert guards_intact(fullC) and guards_intact(fullG)
    _, C64, _ = oracle.compress_bwd(inp["G"], inp["U"])
    assert_parity(host(C), C64, dtype)
    _, G64, _ = oracle.decompress_bwd(host(C), inp["U"])
    assert_parity(host(Gr), G64, dtype)
    basis.destroy()


@pytest.mark.parametrize("dtype", DTYPES)
def test_explicit_positions_and_no_positional_table(sn, oracle, dtype):
    T, n, d, k, vocab = 700, 50, 512, 24, 900
    inp = case_inputs("pos", T, n, d, k, vocab, dtype, seed=5)
    rng = np.random.default_rng(3)
    pos = rng.integers(0, n, T).astype(np.int32)
    basis = sn.Basis(dev(inp["U"]))
    X, tok, pe, ids = dev(inp["X"]), dev(inp["tok_emb"]), dev(inp["pos_emb"]), dev(inp["ids"])
    C = sn.sn_compress_fwd(basis, X, ids, tok, n, pos_emb=pe, pos=dev(pos))
    Xr = sn.sn_decompress_fwd(basis, C, ids, tok, n, pos_emb=pe, pos=dev(pos))
    C2 = sn.sn_compress_fwd(basis, X, ids, tok, n)
    Xr2 = sn.sn_decompress_fwd(basis, C2, ids, tok, n)
    sn.sn_check_errors(basis)
    _, C64, _ = oracle.compress_fwd(inp["X"], inp["ids"], inp["tok_emb"], inp["U"], n,
                                    pos_emb=inp["pos_emb"], pos=pos)
    assert_parity(host(C), C64, dtype)
    _, X64, _ = oracle.decompress_fwd(host(C), inp["ids"], inp["tok_emb"], inp["U"], n,
                                      pos_emb=inp["pos_emb"], pos=pos)
    assert_parity(host(Xr), X64, dtype)
    _, C64, _ = oracle.compress_fwd(inp["X"], inp["ids"], inp["tok_emb"], inp["U"], n)
    assert_parity(host(C2), C64, dtype)
    _, X64, _ = oracle.decompress_fwd(host(C2), inp["ids"], inp["tok_emb"], inp["U"], n)
    assert_parity(host(Xr2), X64, dtype)
    basis.destroy()


def test_gather_bit_exact(sn, oracle):
    """C = 0 reconstructs round(T_fixed[ids] + P[pos]) bit-for-bit (bf16)."""
    T, n, d, k, vocab = 1500, 256, 1024, 33, 4000
    inp = case_inputs("gather", T, n, d, k, vocab, "bf16", seed=9)
    basis = sn.Basis(dev(inp["U"]))
    C0 = np.zeros((T, k), np.uint16)
    Xr = sn.sn_decompress_fwd(basis, dev(C0), dev(inp["ids"]), dev(inp["tok_emb"]), n,
                              pos_emb=dev(inp["pos_emb"]))
    sn.sn_check_errors(basis)
    Xo, _, _ = oracle.decompress_fwd(C0, inp["ids"], inp["tok_emb"], inp["U"], n,
                                     pos_emb=inp["pos_emb"])
    assert np.array_equal(host(Xr), Xo)
    # without a positional table the output is the gathered row itself
    Xr = sn.sn_decompress_fwd(basis, dev(C0), dev(inp["ids"]), dev(inp["tok_emb"]), n)
    assert np.array_equal(host(Xr), inp["tok_emb"][inp["ids"]])
    basis.destroy()


@pytest.mark.parametrize("dtype", DTYPES)
def test_bad_ids_zero_rows_and_report(sn, oracle, dtype):
    T, n, d, k, vocab = 400, 64, 256, 12, 500
    inp = case_inputs("bad", T, n, d, k, vocab, dtype, seed=11)
    ids = inp["ids"].copy()
    ids[[5, 130, 399]] = [vocab, -3, 2**31 - 1]
    basis = sn.Basis(dev(inp["U"]))
    X, tok, pe = dev(inp["X"]), dev(inp["tok_emb"]), dev(inp["pos_emb"])
    C = sn.sn_compress_fwd(basis, X, dev(ids), tok, n, pos_emb=pe)
    with pytest.raises(sn.SNError) as e:
        sn.sn_check_errors(basis)
    assert e.value.status == sn.SN_ERR_BAD_ID
    sn.sn_check_errors(basis)            # the error word was cleared
    Ch = host(C)
    assert np.all(widen(Ch[[5, 130, 399]]) == 0)
    _, C64, st = oracle.compress_fwd(inp["X"], ids, inp["tok_emb"], inp["U"], n,
                                     pos_emb=inp["pos_emb"])
    assert st == 4
    assert_parity(Ch, C64, dtype)
    Xr = sn.sn_decompress_fwd(basis, C, dev(ids), tok, n, pos_emb=pe)
    with pytest.raises(sn.SNError):
        sn.sn_check_errors(basis)
    assert np.all(widen(host(Xr)[[5, 130, 399]]) == 0)
    # an explicit position outside [0, seq_len) is reported the same way
    pos = (np.arange(T) % n).astype(np.int32)
    pos[77] = n
    C = sn.sn_compress_fwd(basis, X, dev(inp["ids"]), tok, n, pos_emb=pe, pos=dev(pos))
    with pytest.raises(sn.SNError):
        sn.sn_check_errors(basis)
    assert np.all(widen(host(C)[77]) == 0)
    basis.destroy()


@pytest.mark.parametrize("dtype", DTYPES)
@pytest.mark.parametrize("d,k,cols,ld", [(512, 20, 1000, 1000), (256, 8, 300, 304),
                                         (1024, 41, 77, 80), (2048, 128, 129, 136),
                                         (16, 16, 8, 8)])
def test_project_weight(sn, oracle, dtype, d, k, cols, ld):
    rng = np.random.default_rng(d + k + cols)
    U = W.orthonormal_basis(d, k, rng).astype(np.float32)
    full = 0.02 * rng.standard_normal((d, ld))
    Wh = W.to_bf16(full) if dtype == "bf16" else full.astype(np.float32)
    basis = sn.Basis(dev(U))
    Wd = dev(Wh)[:, :cols]
    out_full = torch.full((d, ld), 7.0, dtype=Wd.dtype, device=Wd.device)
    out = out_full[:, :cols]
    sn.sn_project_weight(basis, Wd, out=out)
    sn.sn_check_errors(basis)
    _, W64, _ = oracle.project_weight(np.ascontiguousarray(Wh[:, :cols]), U)
    assert_parity(host(out), W64, dtype)
    if cols < ld:      # the padding columns beyond `cols` are untouched
        assert bool((out_full[:, cols:] == 7.0).all())
    # in place, on a strided view with the same leading dimension
    Wd2 = dev(Wh)[:, :cols]
    sn.sn_project_weight(basis, Wd2, out=Wd2)
    assert torch.equal(Wd2, out)
    basis.destroy()


@pytest.mark.parametrize("d,k,cols", [(8192, 82, 8192), (4096, 41, 14336)])
def test_project_weight_in_place_full_size(sn, d, k, cols):
    """At the benchmark's weight shapes the projection's three passes overlap
    their neighbours' start-up (programmatic dependent launch); projecting in
    place must give exactly the out-of-place result, so no pass may write W'
    before the first pass has read all of W."""
    rng = np.random.default_rng(d + cols)
    U = W.orthonormal_basis(d, k, rng).astype(np.float32)
    basis = sn.Basis(dev(U))
    g = torch.Generator(device="cuda").manual_seed(3)
    Wd = (0.02 * torch.randn(d, cols, generator=g, device="cuda")).to(torch.bfloat16)
    ref = sn.sn_project_weight(basis, Wd)
    for _ in range(3):
        Wi = Wd.clone()
        sn.sn_project_weight(basis, Wi, out=Wi)
        sn.sn_check_errors(basis)
        assert torch.equal(Wi, ref)
    basis.destroy()


def test_project_weight_repeated_and_very_wide(sn, oracle):
    """The first pass writes fp32 partials over several d-ranges per column tile
    into the caller's workspace and the second sums them: calls with other
    column counts in between give identical results, and a W of 4097 column
    tiles (half a million columns) matches the oracle."""
    d, k = 2048, 41                         # 32 chunks of d: several splits per tile
    rng = np.random.default_rng(17)
    U = W.orthonormal_basis(d, k, rng).astype(np.float32)
    basis = sn.Basis(dev(U))
    g = torch.Generator(device="cuda").manual_seed(5)
    Wa = (0.02 * torch.randn(d, 1000, generator=g, device="cuda")).to(torch.bfloat16)
    Wb = (0.02 * torch.randn(d, 304, generator=g, device="cuda")).to(torch.bfloat16)
    ref = sn.sn_project_weight(basis, Wa)
    for _ in range(3):
        sn.sn_project_weight(basis, Wb)
        assert torch.equal(sn.sn_project_weight(basis, Wa), ref)
    sn.sn_check_errors(basis)
    _, W64, _ = oracle.project_weight(host(Wa), U)
    assert_parity(host(ref), W64, "bf16")
    basis.destroy()
    # 4097 tiles of 128 columns
    d, k, cols = 64, 8, 4097 * 128
    U = W.orthonormal_basis(d, k, rng).astype(np.float32)
    basis = sn.Basis(dev(U))
    Wh = W.to_bf16(0.02 * rng.standard_normal((d, cols)))
    out = sn.sn_project_weight(basis, dev(Wh))
    sn.sn_check_errors(basis)
    _, W64, _ = oracle.project_weight(Wh, U)
    assert_parity(host(out), W64, "bf16")
    basis.destroy()


@pytest.mark.parametrize("dtype", DTYPES)
def test_projection_identities(sn, dtype):
    """P^2 = P and P U = U on the GPU output (Sec. 4.3; U^T U = I, App. A)."""
    d, k, cols = 1024, 41, 512
    rng = np.random.default_rng(5)
    U64 = W.orthonormal_basis(d, k, rng)
    basis = sn.Basis(dev(U64.astype(np.float32)))
    Wh = W.to_bf16(0.02 * rng.standard_normal((d, cols))) if dtype == "bf16" else \
        (0.02 * rng.standard_normal((d, cols))).astype(np.float32)
    W1 = sn.sn_project_weight(basis, dev(Wh))
    W2 = sn.sn_project_weight(basis, W1)
    assert_parity(host(W2), widen(host(W1)), dtype)
    B = rng.standard_normal((k, cols))
    In = U64 @ B
    Inh = W.to_bf16(In) if dtype == "bf16" else In.astype(np.float32)
    Pin = sn.sn_project_weight(basis, dev(Inh))
    assert_parity(host(Pin), widen(Inh), dtype, scale=2)
    basis.destroy()


def test_gradient_identity_app_a(sn):
    """(G P) W' = G W' with W' = P W (App. A): projecting the incoming gradient
    loses nothing below a projected residual-writing weight."""
    d, k, m, T = 2048, 20, 512, 640
    rng = np.random.default_rng(6)
    U = W.orthonormal_basis(d, k, rng).astype(np.float32)
    basis = sn.Basis(dev(U))
    Wp = sn.sn_project_weight(basis, dev(W.to_bf16(0.02 * rng.standard_normal((d, m)))))
    G = dev(W.to_bf16(rng.standard_normal((T, d))))
    Gp = sn.sn_decompress_bwd(basis, sn.sn_compress_bwd(basis, G))
    sn.sn_check_errors(basis)
    lhs = Gp.float() @ Wp.float()
    rhs = G.float() @ Wp.float()
    err = float((lhs - rhs).norm() / rhs.norm())
    assert err <= 1e-2, err
    basis.destroy()


def test_residual_closure(sn):
    """With W' = P W, X = E + h W'^T lies in E + S and round-trips (Sec. 4.2-4.3)."""
    T, n, d, k, vocab, m = 900, 300, 1024, 24, 2000, 256
    rng = np.random.default_rng(12)
    U = W.orthonormal_basis(d, k, rng).astype(np.float32)
    basis = sn.Basis(dev(U))
    Wp = sn.sn_project_weight(basis, dev(W.to_bf16(0.05 * rng.standard_normal((d, m)))))
    h = torch.from_numpy(rng.standard_normal((T, m)).astype(np.float32)).cuda()
    tok = dev(W.to_bf16(0.02 * rng.standard_normal((vocab, d))))
    pe = dev(W.to_bf16(0.02 * rng.standard_normal((n, d))))
    ids = dev(rng.integers(0, vocab, T).astype(np.int32))
    pos = torch.arange(T, device="cuda") % n
    Y = h @ Wp.float().T
    X = (tok[ids].float() + pe[pos].float() + Y).to(torch.bfloat16)
    Xr = sn.sn_decompress_fwd(basis, sn.sn_compress_fwd(basis, X, ids, tok, n, pos_emb=pe), ids,
                              tok, n, pos_emb=pe)
    sn.sn_check_errors(basis)
    err = float((Xr.float() - X.float()).norm() / Y.norm())
    assert err <= 1e-2, err
    basis.destroy()


def test_wire_round_trip(sn):
    """compress -> pinned host wire -> device -> reconstruct equals the direct
    reconstruction bit-for-bit; the wire carries exactly T*k*2 bytes."""
    T, n, d, k, vocab = 2048, 512, 2048, 20, 3000
    inp = case_inputs("wire", T, n, d, k, vocab, "bf16", seed=13)
    basis = sn.Basis(dev(inp["U"]))
    X, tok, pe, ids = dev(inp["X"]), dev(inp["tok_emb"]), dev(inp["pos_emb"]), dev(inp["ids"])
    C = sn.sn_compress_fwd(basis, X, ids, tok, n, pos_emb=pe)
    nbytes = sn.sn_wire_bytes(basis, torch.bfloat16, T)
    assert nbytes == T * k * 2 == C.numel() * 2
    wire = torch.empty(nbytes, dtype=torch.uint8, pin_memory=True)
    sn.sn_wire_send(C, wire)
    C_rx = torch.empty_like(C)
    sn.sn_wire_recv(wire, C_rx)
    X1 = sn.sn_decompress_fwd(basis, C_rx, ids, tok, n, pos_emb=pe)
    X2 = sn.sn_decompress_fwd(basis, C, ids, tok, n, pos_emb=pe)
    sn.sn_check_errors(basis)
    assert torch.equal(C_rx, C)
    assert torch.equal(X1, X2)
    assert np.array_equal(wire.numpy(), host(C).view(np.uint8).reshape(-1))
    basis.destroy()


def test_zero_tokens_is_a_no_op(sn):
    basis = sn.Basis(dev(W.orthonormal_basis(64, 4, np.random.default_rng(0)).astype(np.float32)))
    X = torch.empty(0, 64, dtype=torch.bfloat16, device="cuda")
    ids = torch.empty(0, dtype=torch.int32, device="cuda")
    tok = torch.zeros(10, 64, dtype=torch.bfloat16, device="cuda")
    C = sn.sn_compress_fwd(basis, X, ids, tok, 8)
    assert C.shape == (0, 4)
    G = sn.sn_decompress_bwd(basis, C)
    assert G.shape == (0, 64)
    sn.sn_check_errors(basis)
    basis.destroy()


def test_argument_errors(sn):
    U = dev(W.orthonormal_basis(64, 4, np.random.default_rng(0)).astype(np.float32))
    basis = sn.Basis(U)
    X = torch.zeros(10, 64, dtype=torch.bfloat16, device="cuda")
    tok = torch.zeros(10, 64, dtype=torch.bfloat16, device="cuda")
    ids = torch.zeros(10, dtype=torch.int32, device="cuda")
    with pytest.raises(sn.SNError) as e:      # misaligned X
        raw = torch.zeros(10 * 64 + 1, dtype=torch.bfloat16, device="cuda")[1:].view(10, 64)
        sn.sn_compress_fwd(basis, raw, ids, tok, 8)
    assert e.value.status == sn.SN_ERR_ALIGNMENT
    with pytest.raises(sn.SNError) as e:      # seq_len = 0
        sn.sn_compress_fwd(basis, X, ids, tok, 0)
    assert e.value.status == sn.SN_ERR_INVALID_ARG
    with pytest.raises(sn.SNError) as e:      # output overlapping the input
        sn.sn_compress_bwd(basis, X, out=X.view(-1)[:40].view(10, 4))
    assert e.value.status == sn.SN_ERR_INVALID_ARG
    with pytest.raises(sn.SNError):           # k > d
        sn.Basis(torch.zeros(16, 17, device="cuda"))
    basis.destroy()


@pytest.mark.parametrize("layout", ["ragged", "position_major"])
def test_more_tiles_than_sms(sn, oracle, layout):
    """More row tiles than SMs, so every persistent CTA takes several tiles and
    a few take one more (ragged last tile, and the position-block-major tile
    order); every row of C must come out."""
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    if layout == "ragged":
        T, n = (sms + 9) * 128 - 50, 128          # 9 tiles past one per SM, the last ragged
    else:
        T, n = (sms + 8) * 128, 256               # 2-tile sequences, tiles run position-major
    d, k, vocab = 128, 24, 600
    inp = case_inputs("tail_" + layout, T, n, d, k, vocab, "bf16", seed=11)
    basis = sn.Basis(dev(inp["U"]))
    X, tok, pe, ids, G = (dev(inp["X"]), dev(inp["tok_emb"]), dev(inp["pos_emb"]),
                          dev(inp["ids"]), dev(inp["G"]))
    fullC, C = guarded((T, k), X.dtype)
    sn.sn_compress_fwd(basis, X, ids, tok, n, pos_emb=pe, out=C)
    fullCg, Cg = guarded((T, k), X.dtype)
    sn.sn_compress_bwd(basis, G, out=Cg)
    sn.sn_check_errors(basis)
    assert guards_intact(fullC) and guards_intact(fullCg)
    _, C64, st = oracle.compress_fwd(inp["X"], inp["ids"], inp["tok_emb"], inp["U"], n,
                                     pos_emb=inp["pos_emb"])
    assert st == 0
    assert_parity(host(C), C64, "bf16")
    _, Cg64, _ = oracle.compress_bwd(inp["G"], inp["U"])
    assert_parity(host(Cg), Cg64, "bf16")
    # every row is covered: no row of C left at the guard fill or zero
    assert np.all(np.abs(widen(host(C))).sum(axis=1) > 0)
    basis.destroy()


@pytest.mark.parametrize("layout", ["ragged", "few_tiles", "position_major"])
def test_split_last_round(sn, oracle, layout):
    """When the persistent grid's last round would hold only a few row tiles,
    those tiles run as d-range items whose fp32 partials are summed afterwards
    (d = 2048: 32 chunks, so 2 to 4 items a tile): a ragged last tile, fewer
    tiles than half the SMs (every tile split), and the position-major tile
    order.  Bad ids inside split tiles are zeroed and reported as anywhere else,
    explicit positions are honoured, and the projected-table compress splits the
    same way."""
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    if layout == "ragged":
        T, n = (sms + 10) * 128 - 37, 128
    elif layout == "few_tiles":
        T, n = 40 * 128, 128
    else:
        T, n = (sms + 8) * 128, 256
    d, k, vocab = 2048, 24, 600
    inp = case_inputs("split_" + layout, T, n, d, k, vocab, "bf16", seed=13)
    ids = inp["ids"].copy()
    bad = [T - 1, T - 130, 3]
    ids[bad] = [vocab, -1, vocab + 7]
    basis = sn.Basis(dev(inp["U"]))
    X, tok, pe, G = dev(inp["X"]), dev(inp["tok_emb"]), dev(inp["pos_emb"]), dev(inp["G"])
    fullC, C = guarded((T, k), X.dtype)
    sn.sn_compress_fwd(basis, X, dev(ids), tok, n, pos_emb=pe, out=C)
    with pytest.raises(sn.SNError) as e:
        sn.sn_check_errors(basis)
    assert e.value.status == sn.SN_ERR_BAD_ID
    fullCg, Cg = guarded((T, k), X.dtype)
    sn.sn_compress_bwd(basis, G, out=Cg)
    sn.sn_check_errors(basis)
    assert guards_intact(fullC) and guards_intact(fullCg)
    Ch = host(C)
    assert np.all(widen(Ch[bad]) == 0)
    _, C64, st = oracle.compress_fwd(inp["X"], ids, inp["tok_emb"], inp["U"], n,
                                     pos_emb=inp["pos_emb"])
    assert st == 4
    assert_parity(Ch, C64, "bf16")
    good = np.setdiff1d(np.arange(T), bad)
    assert np.all(np.abs(widen(Ch[good])).sum(axis=1) > 0)
    _, Cg64, _ = oracle.compress_bwd(inp["G"], inp["U"])
    assert_parity(host(Cg), Cg64, "bf16")
    # the projected-table compress over the same tiles
    TU, PU = sn.sn_project_tables(basis, tok, pos_emb=pe)
    Cp = sn.sn_compress_fwd_projected(basis, X, dev(ids), TU, n, PU=PU)
    with pytest.raises(sn.SNError):
        sn.sn_check_errors(basis)
    assert np.all(widen(host(Cp)[bad]) == 0)
    assert_parity(host(Cp), C64, "bf16")
    if layout == "ragged":
        # explicit positions (not one contiguous run per tile: gathered rows)
        pos = np.random.default_rng(4).integers(0, n, T).astype(np.int32)
        C = sn.sn_compress_fwd(basis, X, dev(inp["ids"]), tok, n, pos_emb=pe, pos=dev(pos))
        sn.sn_check_errors(basis)
        _, C64, _ = oracle.compress_fwd(inp["X"], inp["ids"], inp["tok_emb"], inp["U"], n,
                                        pos_emb=inp["pos_emb"], pos=pos)
        assert_parity(host(C), C64, "bf16")
    basis.destroy()


def test_host_pointers_are_refused(sn):
    """Every tensor argument must be device memory of the current device: host
    memory (pageable or pinned) is refused with SN_ERR_INVALID_ARG before any
    launch, in the binding and at the C ABI."""
    T, d, k, n, vocab = 256, 256, 8, 128, 1024
    U = torch.linalg.qr(torch.randn(d, k, dtype=torch.float64))[0].float().contiguous().cuda()
    basis = sn.Basis(U)
    with pytest.raises(ValueError):
        sn.Basis(U.cpu())
    st = sn._lib.sn_basis_create(ctypes.c_void_p(U.cpu().data_ptr()), d, k,
                                 ctypes.byref(ctypes.c_void_p()), None)
    assert st == sn.SN_ERR_INVALID_ARG
    X = torch.zeros(T, d, dtype=torch.bfloat16, device="cuda")
    ids = torch.zeros(T, dtype=torch.int32, device="cuda")
    tok = torch.zeros(vocab, d, dtype=torch.bfloat16, device="cuda")
    C = torch.empty(T, k, dtype=torch.bfloat16, device="cuda")
    launches = sn.sn_launch_count()
    with pytest.raises(ValueError):
        sn.sn_compress_fwd(basis, X.cpu(), ids, tok, n, out=C)
    lib, P = sn._lib, ctypes.c_void_p
    for host in (X.cpu(), X.cpu().pin_memory()):
        st = lib.sn_compress_fwd(basis.handle, sn.SN_BF16, P(host.data_ptr()), P(ids.data_ptr()),
                                 None, T, n, P(tok.data_ptr()), vocab, None, P(C.data_ptr()),
                                 None)
        assert st == sn.SN_ERR_INVALID_ARG
        st = lib.sn_decompress_fwd(basis.handle, sn.SN_BF16, P(C.data_ptr()), P(ids.data_ptr()),
                                   None, T, n, P(tok.data_ptr()), vocab, None,
                                   P(host.data_ptr()), None)
        assert st == sn.SN_ERR_INVALID_ARG
        st = lib.sn_compress_bwd(basis.handle, sn.SN_BF16, P(host.data_ptr()), T,
                                 P(C.data_ptr()), None)
        assert st == sn.SN_ERR_INVALID_ARG
        codes = torch.empty(T, d, dtype=torch.uint8, device="cuda")
        scale = torch.empty(T, dtype=torch.float32, device="cuda")
        st = lib.sn_quant_compress(P(host.data_ptr()), T, d, 0, P(codes.data_ptr()),
                                   P(scale.data_ptr()), None)
        assert st == sn.SN_ERR_INVALID_ARG
    ids_host = ids.cpu()
    st = lib.sn_compress_fwd(basis.handle, sn.SN_BF16, P(X.data_ptr()), P(ids_host.data_ptr()),
                             None, T, n, P(tok.data_ptr()), vocab, None, P(C.data_ptr()), None)
    assert st == sn.SN_ERR_INVALID_ARG
    assert sn.sn_launch_count() == launches        # nothing was launched
    sn.sn_compress_fwd(basis, X, ids, tok, n, out=C)  # device memory still works
    sn.sn_check_errors(basis)
    basis.destroy()


def test_binding_refuses_short_tables_and_wrong_outputs(sn):
    """The kernels index the positional table by position and write T rows of
    the output without bounds information, so the binding refuses a positional
    table with fewer than seq_len rows, a pos array of the wrong length and an
    output of the wrong shape before anything is launched."""
    T, n, d, k, vocab = 256, 128, 256, 8, 1024
    U = torch.linalg.qr(torch.randn(d, k, dtype=torch.float64))[0].float().contiguous().cuda()
    basis = sn.Basis(U)
    X = torch.zeros(T, d, dtype=torch.bfloat16, device="cuda")
    ids = torch.zeros(T, dtype=torch.int32, device="cuda")
    tok = torch.zeros(vocab, d, dtype=torch.bfloat16, device="cuda")
    pe = torch.zeros(n, d, dtype=torch.bfloat16, device="cuda")
    C = torch.zeros(T, k, dtype=torch.bfloat16, device="cuda")
    launches = sn.sn_launch_count()
    bad_calls = [
        lambda: sn.sn_compress_fwd(basis, X, ids, tok, n + 1, pos_emb=pe),           # short table
        lambda: sn.sn_decompress_fwd(basis, C, ids, tok, n + 1, pos_emb=pe),
        lambda: sn.sn_compress_fwd(basis, X, ids, tok, n, pos_emb=pe[:, :128]),      # narrow table
        lambda: sn.sn_compress_fwd(basis, X, ids, tok, n, pos_emb=pe,
                                   pos=ids[:100]),                                    # short pos
        lambda: sn.sn_compress_fwd(basis, X, ids, tok, n, out=C[:100]),               # short out
        lambda: sn.sn_decompress_fwd(basis, C, ids, tok, n, out=X[:, :128]),
        lambda: sn.sn_compress_bwd(basis, X, out=C[:, :4]),
        lambda: sn.sn_decompress_bwd(basis, C, out=X[:10]),
    ]
    for call in bad_calls:
        with pytest.raises(ValueError):
            call()
    assert sn.sn_launch_count() == launches
    sn.sn_compress_fwd(basis, X, ids, tok, n, pos_emb=pe, out=C)     # the valid call runs
    sn.sn_check_errors(basis)
    basis.destroy()
