"""GPU parity of the GQA append + decode path against the oracle, through the
C ABI: bit-exact codes/scales/zeros, fp64-oracle tolerance on outputs, over
every stored format, ragged lengths spanning several tiles, split counts,
sharing, eviction lists and the error paths."""
import math

import numpy as np
import pytest
import torch

from _parity import (assert_close, check_codes, f32, gqa_expected, oracle_state)

pytestmark = pytest.mark.gpu

FORMATS = [
    dict(bits=16, group=64, key_axis="token"),
    dict(bits=8, group=64, key_axis="token"),
    dict(bits=4, group=32, key_axis="token"),
    dict(bits=8, group=32, key_axis="token"),
    dict(bits=4, group=64, key_axis="token"),
    dict(bits=8, group=64, key_axis="channel"),
    dict(bits=4, group=32, key_axis="channel"),
]


def _cache(B, Hq, Hkv, D, T, layers, max_splits=16):
    from paper_2609_37988_gb300.cache import Cache, Layer
    return Cache(n_layers=len(layers), n_q_heads=Hq, n_kv_heads=Hkv, head_dim=D, max_batch=B,
                 max_ctx=T, layers=[Layer(**l) for l in layers], max_splits=max_splits)


def _fill(cache, layer, B, Hkv, D, chunks, dtype, seed):
    """Append ``chunks`` = list of per-sequence counts; returns the full
    inputs [B, T, H, D] (host float32, rows past each length unused) and lens."""
    g = torch.Generator(device="cpu").manual_seed(seed)
    total = [0] * B
    ks, vs = [], []
    T = sum(max(c) for c in chunks)
    K = torch.zeros((B, T, Hkv, D)); V = torch.zeros((B, T, Hkv, D))
    for counts in chunks:
        n = max(counts)
        k = (torch.randn((B, n, Hkv, D), generator=g) * 1.5 + 0.3).to(dtype)
        v = torch.randn((B, n, Hkv, D), generator=g).to(dtype)
        npb = torch.tensor(counts, dtype=torch.int32, device="cuda")
        cache.append(layer, k.cuda(), v.cuda(), n_per_seq=npb)
        for b in range(B):
            K[b, total[b]:total[b] + counts[b]] = k[b, :counts[b]].float()
            V[b, total[b]:total[b] + counts[b]] = v[b, :counts[b]].float()
            total[b] += counts[b]
    return K.numpy(), V.numpy(), np.array(total)


@pytest.mark.parametrize("D", [128, 64])
@pytest.mark.parametrize("fmt", FORMATS, ids=lambda f: f"{f['bits']}b-g{f['group']}-{f['key_axis']}")
@pytest.mark.parametrize("in_dtype", [torch.bfloat16, torch.float32], ids=["bf16in", "f32in"])
def test_append_codes_bit_exact(fmt, D, in_dtype):
    B, Hkv = 3, 2
    chunks = [[1, 33, 70], [31, 0, 64], [100, 2, 63]]   # ragged, crosses groups and tiles
    c = _cache(B, 4, Hkv, D, 300, [dict(**fmt)])
    K, V, lens = _fill(c, 0, B, Hkv, D, chunks, in_dtype, seed=D + fmt["bits"])
    assert c.lengths(0).cpu().tolist() == lens.tolist()
    st = oracle_state(K, V, lens, fmt)
    check_codes(c.export(0), st, lens, fmt)
    assert c.device_error() == 0


@pytest.mark.parametrize("D", [128, 64])
@pytest.mark.parametrize("fmt", FORMATS, ids=lambda f: f"{f['bits']}b-g{f['group']}-{f['key_axis']}")
@pytest.mark.parametrize("G", [1, 5, 8])
def test_decode_parity(fmt, D, G):
    B, Hkv = 3, 2
    Hq = G * Hkv
    chunks = [[1, 257, 33], [0, 140, 31]]
    c = _cache(B, Hq, Hkv, D, 600, [dict(**fmt)])
    K, V, lens = _fill(c, 0, B, Hkv, D, chunks, torch.bfloat16, seed=3 * G + D)
    st = oracle_state(K, V, lens, fmt)
    sigma = 1.0 / math.sqrt(D)
    for qdt in (torch.bfloat16, torch.float32):
        q = torch.randn((B, Hq, D), generator=torch.Generator().manual_seed(G)).to(qdt)
        ref = gqa_expected(q, st, lens, sigma)
        for ns in (0, 1, 3, 7):
            out = c.decode(0, q.cuda(), sigma, n_splits=ns)
            assert_close(f32(out), ref, what=f"{fmt} D{D} G{G} {qdt} splits={ns}")
    assert c.device_error() == 0


def test_edge_lengths_and_empty_sequences():
    # T = 0 for one sequence, T = 1, exact tile and group multiples
    fmt = dict(bits=4, group=32, key_axis="token")
    for counts in ([0, 1, 64], [128, 32, 2]):
        c = _cache(3, 8, 2, 128, 256, [fmt])
        K, V, lens = _fill(c, 0, 3, 2, 128, [counts], torch.bfloat16, seed=sum(counts))
        st = oracle_state(K, V, lens, fmt)
        q = torch.randn((3, 8, 128)).to(torch.bfloat16)
        out = f32(c.decode(0, q.cuda(), 0.1, n_splits=2))
        ref = gqa_expected(q, st, lens, 0.1)
        for b in range(3):
            if lens[b] == 0:
                assert (out[b] == 0).all()
            else:
                assert_close(out[b], ref[b], what=f"lens {counts}")


def test_inheritor_reads_source_bytes_bit_identical():
    layers = [dict(bits=4, group=32), dict(inherit=True), dict(bits=16), dict(inherit=True)]
    c = _cache(2, 10, 2, 128, 300, layers)
    _fill(c, 0, 2, 2, 128, [[200, 150]], torch.bfloat16, 1)
    _fill(c, 2, 2, 2, 128, [[200, 150]], torch.bfloat16, 2)
    assert [c.source(l) for l in range(4)] == [0, 0, 2, 2]
    q = torch.randn((2, 10, 128)).to(torch.bfloat16).cuda()
    for src, inh in ((0, 1), (2, 3)):
        a = c.decode(src, q, 0.09, n_splits=3)
        b = c.decode(inh, q, 0.09, n_splits=3)
        assert torch.equal(a, b)
    from paper_2609_37988_gb300.cache import KVKError
    with pytest.raises(KVKError, match="INHERITED_LAYER"):
        c.append(1, torch.zeros((2, 1, 2, 128), dtype=torch.bfloat16, device="cuda"),
                 torch.zeros((2, 1, 2, 128), dtype=torch.bfloat16, device="cuda"))


def test_capacity_is_checked_on_the_host():
    from paper_2609_37988_gb300.cache import KVKError
    c = _cache(1, 4, 1, 64, 100, [dict(bits=8, group=64)])
    x = torch.zeros((1, 90, 1, 64), dtype=torch.bfloat16, device="cuda")
    c.append(0, x, x)
    with pytest.raises(KVKError, match="CAPACITY"):
        c.append(0, x[:, :20], x[:, :20])
    assert c.lengths(0).cpu().tolist() == [90]


def test_softmax_scale_must_be_positive():
    from paper_2609_37988_gb300.cache import KVKError
    c = _cache(1, 4, 1, 64, 64, [dict(bits=4, group=32)])
    x = torch.zeros((1, 8, 1, 64), dtype=torch.bfloat16, device="cuda")
    c.append(0, x, x)
    q = torch.zeros((1, 4, 64), dtype=torch.bfloat16, device="cuda")
    for bad in (0.0, -0.125, float("nan"), float("inf")):
        with pytest.raises(KVKError, match="INVALID_ARG"):
            c.decode(0, q, bad)
    assert c.decode(0, q, 0.125).isfinite().all()


@pytest.mark.parametrize("fmt", [dict(bits=4, group=32, key_axis="token"),
                                 dict(bits=8, group=64, key_axis="token"),
                                 dict(bits=16, group=64, key_axis="token")], ids=["int4", "int8", "bf16"])
def test_kept_list_gather(fmt):
    B, Hkv, G, D, T = 3, 2, 5, 128, 700
    cap = 160
    c = _cache(B, G * Hkv, Hkv, D, T, [dict(evict_capacity=cap, **fmt)])
    K, V, lens = _fill(c, 0, B, Hkv, D, [[700, 400, 90]], torch.bfloat16, seed=9)
    st = oracle_state(K, V, lens, fmt)
    rng = np.random.default_rng(0)
    n_kept = np.array([160, 77, 90], np.int32)
    idx = np.zeros((B, cap), np.int32)
    kept = []
    for b in range(B):
        sel = np.sort(rng.choice(int(lens[b]), int(n_kept[b]), replace=False)).astype(np.int32)
        idx[b, :len(sel)] = sel
        kept.append(sel)
    q = torch.randn((B, G * Hkv, D)).to(torch.bfloat16)
    plain = c.decode(0, q.cuda(), 0.1, n_splits=2).clone()
    c.set_kept(0, torch.from_numpy(idx).cuda(), torch.from_numpy(n_kept).cuda())
    for ns in (0, 1, 3):
        out = c.decode(0, q.cuda(), 0.1, n_splits=ns)
        assert_close(f32(out), gqa_expected(q, st, lens, 0.1, kept), what=f"gather splits={ns}")
    # keeping every position (sequence 2 keeps all 90) equals no eviction
    assert torch.equal(c.decode(0, q.cuda(), 0.1, n_splits=2)[2], plain[2])
    assert c.device_error() == 0
    # a kept position past the length is reported, skipped, and does not fault
    bad = idx.copy(); bad[1, 3] = 5000
    c.set_kept(0, torch.from_numpy(bad).cuda(), torch.from_numpy(n_kept).cuda())
    out = c.decode(0, q.cuda(), 0.1, n_splits=2)
    assert torch.isfinite(out).all()
    assert c.device_error() == 1
    c.set_kept(0)  # clear
    assert torch.equal(c.decode(0, q.cuda(), 0.1, n_splits=2), plain)


def test_partials_and_reduce_equal_decode():
    from paper_2609_37988_gb300.cache import splitk_reduce
    c = _cache(2, 16, 2, 128, 1000, [dict(bits=4, group=32)])
    _fill(c, 0, 2, 2, 128, [[1000, 517]], torch.bfloat16, 4)
    q = torch.randn((2, 16, 128)).to(torch.bfloat16).cuda()
    for ns in (2, 5, 16):
        p = c.decode_partial(0, q, 0.1, ns)
        assert p.shape == (ns, 32, 130)
        merged = splitk_reduce(p).view(2, 16, 128)
        assert torch.equal(merged, c.decode(0, q, 0.1, n_splits=ns))
    # more splits than tiles: the extra partials are empty (m = -inf, l = 0)
    p = c.decode_partial(0, q, 0.1, 16)
    assert torch.isinf(p[15, 16:, 128]).all() and (p[15, 16:, 129] == 0).all()


@pytest.mark.parametrize("S,dim", [(1, 128), (5, 128), (8, 64), (9, 96), (16, 130), (17, 512),
                                   (40, 128), (64, 32)])
def test_splitk_reduce_matches_log_sum_exp(S, dim):
    """The merge against the log-sum-exp identity in fp64, with empty splits
    (m = -inf, l = 0) and rows whose splits are all empty."""
    from paper_2609_37988_gb300.cache import splitk_reduce
    rng = np.random.default_rng(S * 1000 + dim)
    rows = 37
    P = np.zeros((S, rows, dim + 2), np.float32)
    P[:, :, :dim] = rng.normal(size=(S, rows, dim))
    P[:, :, dim] = rng.normal(scale=6.0, size=(S, rows))
    P[:, :, dim + 1] = rng.uniform(1.0, 50.0, size=(S, rows))
    empty = rng.uniform(size=(S, rows)) < 0.3
    empty[:, 5] = True  # a row with no positions at all
    P[:, :, dim][empty] = -np.inf
    P[:, :, dim + 1][empty] = 0.0
    P[:, :, :dim][empty] = 0.0
    got = splitk_reduce(torch.from_numpy(P).cuda()).cpu().numpy()
    P64 = P.astype(np.float64)
    m = P64[:, :, dim]
    M = m.max(axis=0)
    w = np.where(np.isinf(m), 0.0, np.exp2(m - np.where(np.isinf(M), 0.0, M)))
    L = (w * P64[:, :, dim + 1]).sum(axis=0)
    A = (w[:, :, None] * P64[:, :, :dim]).sum(axis=0)
    want = np.where(L[:, None] > 0, A / np.where(L > 0, L, 1.0)[:, None], 0.0)
    np.testing.assert_allclose(got, want, rtol=2e-6, atol=2e-6)
    assert (got[5] == 0).all()


def test_per_channel_keys_one_position_at_a_time():
    # the open group moves through the residual plane and is quantised when
    # it fills, exactly as a bulk append of the same positions
    fmt = dict(bits=4, group=32, key_axis="channel")
    a = _cache(2, 4, 1, 128, 200, [fmt])
    b = _cache(2, 4, 1, 128, 200, [fmt])
    g = torch.Generator().manual_seed(5)
    k = torch.randn((2, 70, 1, 128), generator=g).to(torch.bfloat16).cuda()
    v = torch.randn((2, 70, 1, 128), generator=g).to(torch.bfloat16).cuda()
    a.append(0, k, v)
    for t in range(70):
        b.append(0, k[:, t:t + 1].contiguous(), v[:, t:t + 1].contiguous())
    ea, eb = a.export(0), b.export(0)
    # positions 0..63 are two full key groups; 64..69 are still bf16 residual
    assert torch.equal(ea["k_codes"][:, :, :64], eb["k_codes"][:, :, :64])
    for key in ("v_codes", "v_scale", "v_zero"):
        assert torch.equal(ea[key][:, :, :70], eb[key][:, :, :70]), key
    assert torch.equal(ea["k_scale"][:, :, :2], eb["k_scale"][:, :, :2])
    assert torch.equal(ea["k_residual"][:, :, :6], eb["k_residual"][:, :, :6])
    q = torch.randn((2, 4, 128)).to(torch.bfloat16).cuda()
    assert torch.equal(a.decode(0, q, 0.1, n_splits=1), b.decode(0, q, 0.1, n_splits=1))


def _tie_rows(B, n, Hkv, D, group, levels, symmetric, seed):
    """Rows whose quantiser quotients land exactly on half-integers and one
    float32 ulp either side of them: each group (or row, for the symmetric
    quantiser) spans a range that makes the scale a power of two, so
    (x - min) / scale or x / scale is exactly k + 1/2 for the tie channels."""
    rng = np.random.default_rng(seed)
    x = np.zeros((B, n, Hkv, D), np.float32)
    span = D if symmetric else group
    for idx in np.ndindex(B, n, Hkv):
        e = float(2.0 ** rng.integers(-6, 6))
        for g0 in range(0, D, span):
            k = rng.integers(0, levels, size=span).astype(np.float32)
            vals = (k + 0.5) * e
            if symmetric:
                vals *= rng.choice([-1.0, 1.0], size=span).astype(np.float32)
                vals[0], vals[1] = levels * e, -levels * e   # max |x| = q 2^e: scale 2^e
                base = 0.0
            else:
                base = float(rng.normal()) * 4.0 * e
                vals[0], vals[1] = 0.0, levels * e            # range = levels 2^e: scale 2^e
            nudge = rng.integers(-1, 2, size=span)            # a third exact, a third 1 ulp off
            vals = np.where(nudge > 0, np.nextafter(vals, np.float32(np.inf)),
                            np.where(nudge < 0, np.nextafter(vals, np.float32(-np.inf)), vals))
            vals[0] = 0.0 if not symmetric else vals[0]
            vals[1] = levels * e if not symmetric else vals[1]
            x[idx][g0:g0 + span] = (np.float32(base) + vals.astype(np.float32)) if not symmetric else vals
    return x


@pytest.mark.parametrize("fmt", [dict(bits=4, group=32, key_axis="token"),
                                 dict(bits=8, group=64, key_axis="token"),
                                 dict(bits=4, scheme="symmetric"), dict(bits=8, scheme="symmetric")],
                         ids=["int4g32", "int8g64", "sym4", "sym8"])
def test_append_rounding_ties(fmt):
    # float32 inputs exactly on the quantiser's rounding boundaries (and one
    # ulp away): the codes must still equal the oracle's (round half to even
    # of the correctly rounded quotient), on the bulk append path
    B, Hkv, D, n = 2, 2, 128, 40
    sym = fmt.get("scheme") == "symmetric"
    levels = (1 << (fmt["bits"] - 1)) - 1 if sym else (1 << fmt["bits"]) - 1
    group = fmt.get("group", D)
    k = _tie_rows(B, n, Hkv, D, group, levels, sym, seed=fmt["bits"] + 10 * sym)
    v = _tie_rows(B, n, Hkv, D, group, levels, sym, seed=fmt["bits"] + 10 * sym + 1)
    c = _cache(B, 4, Hkv, D, n, [dict(**fmt)])
    c.append(0, torch.from_numpy(k).cuda(), torch.from_numpy(v).cuda())
    lens = np.full(B, n)
    cfg = dict(fmt, key_axis="token")
    st = oracle_state(k, v, lens, cfg)
    check_codes(c.export(0), st, lens, cfg)
    assert c.device_error() == 0
