"""GPU parity of the symmetric per-vector scheme (the paper's own quantiser,
Appendix C.3: one bf16 scale per token-head row, codes in [-q, q]) at 8, 4
and 2 bits, through the C ABI: codes and scales bit-exact against the
oracle, decode outputs within the fp64-oracle tolerance over ragged lengths,
split counts, sharing, eviction lists and empty sequences."""
import math

import numpy as np
import pytest
import torch

from _parity import assert_close, check_codes, f32, gqa_expected, oracle_state

pytestmark = pytest.mark.gpu

BITS = [8, 4, 2]


def _fmt(bits, **kw):
    return dict(bits=bits, group=64, key_axis="token", scheme="symmetric", **kw)


def _cache(B, Hq, Hkv, T, layers, max_splits=16):
    from paper_2609_37988_gb300.cache import Cache, Layer
    return Cache(n_layers=len(layers), n_q_heads=Hq, n_kv_heads=Hkv, head_dim=128, max_batch=B,
                 max_ctx=T, layers=[Layer(**l) for l in layers], max_splits=max_splits)


def _fill(cache, layer, B, Hkv, chunks, dtype, seed, special=False):
    """Append ``chunks`` (per-sequence counts per call); returns host float32
    inputs [B, T, H, 128] and the lengths.  ``special`` plants a zero row,
    rows of dyadic values (exact rounding ties) and one huge-range row."""
    g = torch.Generator(device="cpu").manual_seed(seed)
    total = [0] * B
    T = sum(max(c) for c in chunks)
    K = torch.zeros((B, T, Hkv, 128)); V = torch.zeros((B, T, Hkv, 128))
    for counts in chunks:
        n = max(counts)
        k = torch.randn((B, n, Hkv, 128), generator=g) * 1.5 + 0.3
        v = torch.randn((B, n, Hkv, 128), generator=g)
        if special and n >= 4:
            k[0, 0, 0] = 0.0
            v[0, 0, 0] = 0.0
            k[0, 1] = torch.round(k[0, 1] * 4) / 4
            v[0, 2] = torch.round(v[0, 2] * 8) / 8
            k[0, 3, 0, 5] = 900.0
        k, v = k.to(dtype), v.to(dtype)
        npb = torch.tensor(counts, dtype=torch.int32, device="cuda")
        cache.append(layer, k.cuda(), v.cuda(), n_per_seq=npb)
        for b in range(B):
            K[b, total[b]:total[b] + counts[b]] = k[b, :counts[b]].float()
            V[b, total[b]:total[b] + counts[b]] = v[b, :counts[b]].float()
            total[b] += counts[b]
    return K.numpy(), V.numpy(), np.array(total)


@pytest.mark.parametrize("bits", BITS)
@pytest.mark.parametrize("in_dtype", [torch.bfloat16, torch.float32], ids=["bf16in", "f32in"])
def test_sym_append_codes_bit_exact(bits, in_dtype):
    B, Hkv = 3, 2
    chunks = [[4, 33, 70], [31, 0, 64], [100, 2, 63]]   # ragged, crosses tiles
    fmt = _fmt(bits)
    c = _cache(B, 4, Hkv, 300, [fmt])
    K, V, lens = _fill(c, 0, B, Hkv, chunks, in_dtype, seed=bits, special=True)
    assert c.lengths(0).cpu().tolist() == lens.tolist()
    st = oracle_state(K, V, lens, fmt)
    ex = c.export(0)
    check_codes(ex, st, lens, fmt)
    q = (1 << (bits - 1)) - 1
    kc = ex["k_codes"][0, :, :lens[0]].cpu()
    assert int(kc.min()) >= -q and int(kc.max()) <= q
    if bits == 2:
        assert set(torch.unique(kc).tolist()) == {-1, 0, 1}
    assert float(ex["k_scale"][0, 0, 0]) == 0.0        # the zero row
    assert c.device_error() == 0


@pytest.mark.parametrize("bits", BITS)
@pytest.mark.parametrize("G", [1, 5, 8])
def test_sym_decode_parity(bits, G):
    B, Hkv = 3, 2
    Hq = G * Hkv
    chunks = [[1, 257, 33], [0, 140, 31]]
    fmt = _fmt(bits)
    c = _cache(B, Hq, Hkv, 600, [fmt])
    K, V, lens = _fill(c, 0, B, Hkv, chunks, torch.bfloat16, seed=7 * G + bits, special=True)
    st = oracle_state(K, V, lens, fmt)
    sigma = 1.0 / math.sqrt(128)
    for qdt in (torch.bfloat16, torch.float32):
        q = torch.randn((B, Hq, 128), generator=torch.Generator().manual_seed(G)).to(qdt)
        ref = gqa_expected(q, st, lens, sigma)
        for ns in (0, 1, 3, 7):
            out = c.decode(0, q.cuda(), sigma, n_splits=ns)
            assert_close(f32(out), ref, what=f"sym{bits} G{G} {qdt} splits={ns}")
    assert c.device_error() == 0


@pytest.mark.parametrize("bits", BITS)
def test_sym_edge_lengths_and_sharing(bits):
    # T = 0, T = 1, exact tile multiples; an inheritor reads the same bytes
    fmt = _fmt(bits)
    for counts in ([0, 1, 64], [128, 256, 2]):
        c = _cache(3, 8, 2, 300, [fmt, dict(inherit=True)])
        K, V, lens = _fill(c, 0, 3, 2, [counts], torch.bfloat16, seed=sum(counts) + bits)
        st = oracle_state(K, V, lens, fmt)
        q = torch.randn((3, 8, 128)).to(torch.bfloat16)
        out = c.decode(0, q.cuda(), 0.1, n_splits=2)
        assert torch.equal(out, c.decode(1, q.cuda(), 0.1, n_splits=2))
        out = f32(out)
        ref = gqa_expected(q, st, lens, 0.1)
        for b in range(3):
            if lens[b] == 0:
                assert (out[b] == 0).all()
            else:
                assert_close(out[b], ref[b], what=f"sym{bits} lens {counts}")


@pytest.mark.parametrize("bits", BITS)
def test_sym_kept_list_gather(bits):
    B, Hkv, G, T = 3, 2, 5, 700
    cap = 160
    fmt = _fmt(bits)
    c = _cache(B, G * Hkv, Hkv, T, [dict(evict_capacity=cap, **fmt)])
    K, V, lens = _fill(c, 0, B, Hkv, [[700, 400, 90]], torch.bfloat16, seed=19 + bits)
    st = oracle_state(K, V, lens, fmt)
    rng = np.random.default_rng(bits)
    n_kept = np.array([160, 77, 90], np.int32)
    idx = np.zeros((B, cap), np.int32)
    kept = []
    for b in range(B):
        sel = np.sort(rng.choice(int(lens[b]), int(n_kept[b]), replace=False)).astype(np.int32)
        idx[b, :len(sel)] = sel
        kept.append(sel)
    q = torch.randn((B, G * Hkv, 128)).to(torch.bfloat16)
    plain = c.decode(0, q.cuda(), 0.1, n_splits=2).clone()
    c.set_kept(0, torch.from_numpy(idx).cuda(), torch.from_numpy(n_kept).cuda())
    for ns in (0, 1, 3):
        out = c.decode(0, q.cuda(), 0.1, n_splits=ns)
        assert_close(f32(out), gqa_expected(q, st, lens, 0.1, kept), what=f"sym{bits} gather {ns}")
    # sequence 2 keeps all of its positions: gathered equals streamed
    assert_close(f32(c.decode(0, q.cuda(), 0.1, n_splits=2)[2]), f32(plain[2]), max_abs=1e-5,
                 rel_l2=1e-6, what="keep-all")
    assert c.device_error() == 0
    bad = idx.copy(); bad[1, 3] = 5000
    c.set_kept(0, torch.from_numpy(bad).cuda(), torch.from_numpy(n_kept).cuda())
    assert torch.isfinite(c.decode(0, q.cuda(), 0.1, n_splits=2)).all()
    assert c.device_error() == 1


def test_sym_two_bit_one_position_at_a_time():
    # appending positions one by one gives the same records as one bulk append
    fmt = _fmt(2)
    a = _cache(2, 4, 1, 200, [fmt])
    b = _cache(2, 4, 1, 200, [fmt])
    g = torch.Generator().manual_seed(5)
    k = torch.randn((2, 70, 1, 128), generator=g).to(torch.bfloat16).cuda()
    v = torch.randn((2, 70, 1, 128), generator=g).to(torch.bfloat16).cuda()
    a.append(0, k, v)
    for t in range(70):
        b.append(0, k[:, t:t + 1].contiguous(), v[:, t:t + 1].contiguous())
    ea, eb = a.export(0), b.export(0)
    for key in ("k_codes", "v_codes", "k_scale", "v_scale"):
        assert torch.equal(ea[key][:, :, :70], eb[key][:, :, :70]), key
    q = torch.randn((2, 4, 128)).to(torch.bfloat16).cuda()
    assert torch.equal(a.decode(0, q, 0.1, n_splits=1), b.decode(0, q, 0.1, n_splits=1))
