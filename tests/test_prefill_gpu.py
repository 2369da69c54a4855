"""GPU parity of causal chunk attention (pre-fill) over the compressed cache,
through the C ABI: every stored format, chunks spanning several row blocks
and tiles, ragged lengths (including sequences shorter than the chunk),
bf16 and fp32 queries, an inheriting layer, and the error paths.  Expected
values: the fp64 oracle on the dequantised state of the same inputs."""
import math

import numpy as np
import pytest
import torch

from _parity import assert_close, f32, oracle_state
from oracle import attention as oatt

pytestmark = pytest.mark.gpu

FORMATS = [
    dict(bits=16, group=64, key_axis="token"),
    dict(bits=8, group=64, key_axis="token"),
    dict(bits=4, group=32, key_axis="token"),
    dict(bits=8, group=32, key_axis="token"),
    dict(bits=4, group=64, key_axis="token"),
    dict(bits=8, group=64, key_axis="token", scheme="symmetric"),
    dict(bits=4, group=64, key_axis="token", scheme="symmetric"),
    dict(bits=2, group=64, key_axis="token", scheme="symmetric"),
    dict(bits=8, group=64, key_axis="channel"),
    dict(bits=4, group=32, key_axis="channel"),
]


def _fid(f):
    return f"{f.get('scheme', 'grouped')[:3]}{f['bits']}g{f['group']}{'-kpc' if f['key_axis'] == 'channel' else ''}"


def _cache(B, Hq, Hkv, T, layers):
    from paper_2609_37988_gb300.cache import Cache, Layer
    return Cache(n_layers=len(layers), n_q_heads=Hq, n_kv_heads=Hkv, head_dim=128, max_batch=B,
                 max_ctx=T, layers=[Layer(**l) for l in layers], max_splits=16)


def _fill(cache, B, Hkv, counts, seed, dtype=torch.bfloat16):
    g = torch.Generator().manual_seed(seed)
    n = max(counts)
    k = (torch.randn((B, n, Hkv, 128), generator=g) * 1.5 + 0.3).to(dtype)
    v = torch.randn((B, n, Hkv, 128), generator=g).to(dtype)
    cache.append(0, k.cuda(), v.cuda(), n_per_seq=torch.tensor(counts, dtype=torch.int32, device="cuda"))
    return k.float().numpy(), v.float().numpy(), np.array(counts)


def _queries(B, n_q, Hq, seed, dtype):
    g = torch.Generator().manual_seed(seed)
    return torch.randn((B, n_q, Hq, 128), generator=g).to(dtype)


def _expected(q, st, lens, sigma):
    return oatt.gqa_prefill(f32(q), st["k_hat"], st["v_hat"], lens, sigma)


@pytest.mark.parametrize("fmt", FORMATS, ids=_fid)
@pytest.mark.parametrize("G,n_q", [(5, 40), (4, 70)], ids=["g5-nq40", "g4-nq70"])
def test_prefill_parity(fmt, G, n_q):
    # rows per unit: 200 (two row blocks) / 280 (three); lengths ragged, one
    # sequence shorter than the chunk
    B, Hkv, T = 3, 2, 700
    Hq = G * Hkv
    c = _cache(B, Hq, Hkv, T, [fmt])
    K, V, lens = _fill(c, B, Hkv, [650, 300, n_q // 2], seed=fmt["bits"] * 7 + G)
    st = oracle_state(K, V, lens, fmt)
    sigma = 1.0 / math.sqrt(128)
    for qdt in (torch.bfloat16, torch.float32):
        q = _queries(B, n_q, Hq, seed=G, dtype=qdt)
        out = c.prefill(0, q.cuda(), sigma)
        ref = _expected(q, st, lens, sigma)
        assert_close(f32(out), ref, what=f"{_fid(fmt)} G{G} n_q{n_q} {qdt}")
        # queries before position 0 give zeros
        assert (f32(out[2, : n_q - n_q // 2]) == 0).all()
    assert c.device_error() == 0


@pytest.mark.parametrize("fmt", [FORMATS[0], FORMATS[2], FORMATS[6], FORMATS[9]], ids=_fid)
def test_prefill_long_chunk_many_tiles(fmt):
    # a 256-query chunk over 1000 positions: 1280 rows (ten row blocks) per
    # unit, 16 tiles of 64 positions for the last block
    B, Hkv, G, T = 1, 2, 5, 1024
    c = _cache(B, G * Hkv, Hkv, T, [fmt])
    K, V, lens = _fill(c, B, Hkv, [1000], seed=11)
    st = oracle_state(K, V, lens, fmt)
    q = _queries(B, 256, G * Hkv, seed=3, dtype=torch.bfloat16)
    out = c.prefill(0, q.cuda(), 0.09)
    assert_close(f32(out), _expected(q, st, lens, 0.09), what=f"{_fid(fmt)} long chunk")


def test_prefill_one_query_is_decode_and_inheritor_reads_anchor():
    B, Hkv, G, T = 2, 4, 5, 600
    fmt = dict(bits=4, group=32, key_axis="token")
    c = _cache(B, G * Hkv, Hkv, T, [fmt, dict(inherit=True)])
    K, V, lens = _fill(c, B, Hkv, [513, 77], seed=4)
    q = _queries(B, 1, G * Hkv, seed=8, dtype=torch.bfloat16).cuda()
    pre = c.prefill(0, q, 0.1)
    dec = c.decode(0, q[:, 0].contiguous(), 0.1)
    # two roundings of the same value (different operand splits): far inside
    # either one's distance to the fp64 oracle
    assert_close(f32(pre[:, 0]), f32(dec), max_abs=2e-4, rel_l2=1e-4, what="one query = decode")
    q2 = _queries(B, 33, G * Hkv, seed=9, dtype=torch.bfloat16).cuda()
    assert torch.equal(c.prefill(1, q2, 0.1), c.prefill(0, q2, 0.1))
    assert c.device_error() == 0


def test_prefill_rejections():
    from paper_2609_37988_gb300._lib import KVKError
    c = _cache(2, 4, 2, 300, [dict(bits=8, group=64, key_axis="channel"), dict(bits=16)])
    q = torch.zeros((2, 8, 4, 128), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(KVKError):
        c.prefill(1, q, 0.0)  # scale
    with pytest.raises(KVKError):
        c.prefill(1, torch.zeros((2, 0, 4, 128), dtype=torch.bfloat16, device="cuda"), 0.1)
    from paper_2609_37988_gb300.cache import Cache, Layer
    m = Cache(kind="mla", n_layers=1, n_q_heads=16, head_dim=128, latent_dim=512, rope_dim=64,
              max_batch=1, max_ctx=64, layers=[Layer(bits=16, width=512)])
    with pytest.raises((KVKError, ValueError)):
        m.prefill(0, torch.zeros((1, 4, 16, 128), dtype=torch.bfloat16, device="cuda"), 0.1)


@pytest.mark.slow
def test_prefill_full_size_sampled():
    """The bench's pre-fill call (14B shape: int4 g32 anchor, B=4 x 8192
    positions, 40 q / 8 KV heads, a 2048-query chunk) with the bench's
    inputs; sampled queries of the first and last sequence against the
    oracle (each one a decode over its causal prefix)."""
    import bench
    from paper_2609_37988_gb300 import workloads as W
    B, T, n_q = 4, 8192, bench.PREFILL_CHUNK
    w, c, q = bench._prefill_setup(B, T, n_q, torch.device("cuda", 0))
    out = f32(c.prefill(0, q, w.sigma))
    assert c.device_error() == 0
    fmt = dict(bits=4, group=32, key_axis="token")
    for b in (0, B - 1):
        k = torch.cat([W.kv_inputs(w, 0, t0, min(T, t0 + 4096), device="cuda")[0][b:b + 1].cpu()
                       for t0 in range(0, T, 4096)], 1)
        v = torch.cat([W.kv_inputs(w, 0, t0, min(T, t0 + 4096), device="cuda")[1][b:b + 1].cpu()
                       for t0 in range(0, T, 4096)], 1)
        st = oracle_state(f32(k), f32(v), np.array([T]), fmt)
        for i in (0, 1, 777, n_q - 2, n_q - 1):
            p = T - n_q + i
            ref = oatt.gqa_decode(f32(q[b:b + 1, i]), st["k_hat"], st["v_hat"], [p + 1], w.sigma)
            assert_close(out[b:b + 1, i], ref, what=f"sequence {b} query {i}")
