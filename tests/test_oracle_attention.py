"""Pins for oracle/attention.py and oracle/cache.py (no GPU): brute force,
a library routine (torch SDPA in float64), special cases with closed forms,
and the MLA absorption identity."""
import math

import numpy as np
import pytest
import torch

from oracle import attention, cache, quant


def test_sources_nearest_preceding_anchor():
    assert attention.resolve_sources([1, 0, 0, 1, 0, 1, 1, 0]) == [0, 0, 0, 3, 3, 5, 6, 6]
    with pytest.raises(ValueError):
        attention.resolve_sources([0, 1, 1])


def _brute_gqa(q, K, V, lens, sigma):
    B, Hq, D = q.shape
    G = Hq // K.shape[1]
    out = np.zeros_like(q, dtype=np.float64)
    for b in range(B):
        for h in range(Hq):
            j = h // G
            sc = [sigma * sum(float(q[b, h, i]) * float(K[b, j, t, i]) for i in range(D))
                  for t in range(lens[b])]
            m = max(sc)
            w = [math.exp(s - m) for s in sc]
            tot = sum(w)
            for i in range(D):
                out[b, h, i] = sum(w[t] * float(V[b, j, t, i]) for t in range(lens[b])) / tot
    return out


def test_gqa_matches_brute_force():
    rng = np.random.default_rng(0)
    B, Hq, Hkv, T, D = 2, 6, 2, 9, 5
    q = rng.standard_normal((B, Hq, D))
    K = rng.standard_normal((B, Hkv, T, D))
    V = rng.standard_normal((B, Hkv, T, D))
    lens = [9, 4]
    got = attention.gqa_decode(q, K, V, lens, 0.7)
    np.testing.assert_allclose(got, _brute_gqa(q, K, V, lens, 0.7), rtol=1e-12, atol=1e-12)


def test_gqa_matches_torch_sdpa():
    rng = np.random.default_rng(1)
    B, Hq, Hkv, T, D = 3, 8, 2, 33, 16
    q = rng.standard_normal((B, Hq, D))
    K = rng.standard_normal((B, Hkv, T, D))
    V = rng.standard_normal((B, Hkv, T, D))
    sigma = 1 / math.sqrt(D)
    got = attention.gqa_decode(q, K, V, [T] * B, sigma)
    G = Hq // Hkv
    tq = torch.from_numpy(q)[:, :, None, :]
    tk = torch.from_numpy(K).repeat_interleave(G, dim=1)
    tv = torch.from_numpy(V).repeat_interleave(G, dim=1)
    ref = torch.nn.functional.scaled_dot_product_attention(tq, tk, tv, scale=sigma)[:, :, 0]
    np.testing.assert_allclose(got, ref.numpy(), rtol=1e-12, atol=1e-12)


def test_single_position_returns_value_and_constant_keys_average():
    rng = np.random.default_rng(2)
    q = rng.standard_normal((1, 4, 8))
    K = rng.standard_normal((1, 1, 5, 8))
    V = rng.standard_normal((1, 1, 5, 8))
    out1 = attention.gqa_decode(q, K, V, [1], 1.0)
    np.testing.assert_allclose(out1[0], np.repeat(V[0, 0, :1], 4, 0), rtol=0, atol=0)
    Kc = np.repeat(K[:, :, :1], 5, axis=2)
    outc = attention.gqa_decode(q, Kc, V, [5], 1.0)
    np.testing.assert_allclose(outc[0], np.repeat(V[0, 0].mean(0)[None], 4, 0), atol=1e-14)


def test_kept_positions_equal_compacted_cache():
    rng = np.random.default_rng(3)
    B, Hq, Hkv, T, D = 2, 4, 2, 40, 8
    q = rng.standard_normal((B, Hq, D))
    K = rng.standard_normal((B, Hkv, T, D))
    V = rng.standard_normal((B, Hkv, T, D))
    kept = [np.sort(rng.choice(T, 11, replace=False)) for _ in range(B)]
    got = attention.gqa_decode(q, K, V, [T] * B, 0.3, kept)
    Kc = np.stack([K[b][:, kept[b]] for b in range(B)])
    Vc = np.stack([V[b][:, kept[b]] for b in range(B)])
    np.testing.assert_allclose(got, attention.gqa_decode(q, Kc, Vc, [11] * B, 0.3), atol=1e-14)
    allpos = [np.arange(T)] * B
    np.testing.assert_allclose(attention.gqa_decode(q, K, V, [T] * B, 0.3, allpos),
                               attention.gqa_decode(q, K, V, [T] * B, 0.3), atol=0)


def _mla_inputs(seed, B=2, H=3, T=7, Dn=8, dR=4, r=12):
    rng = np.random.default_rng(seed)
    return dict(q_nope=rng.standard_normal((B, H, Dn)), q_pe=rng.standard_normal((B, H, dR)),
                c=rng.standard_normal((B, T, r)), k_r=rng.standard_normal((B, T, dR)),
                w_uk=rng.standard_normal((H, Dn, r)), w_uv=rng.standard_normal((H, Dn, r)))


@pytest.mark.parametrize("d", [12, 6, 3])
def test_mla_absorbed_equals_unabsorbed(d):
    x = _mla_inputs(4)
    lens = [7, 5]
    got = attention.mla_decode_unabsorbed(**x, d=d, lens=lens, sigma=0.4)
    B, H, _ = x["q_nope"].shape
    for b in range(B):
        C = x["c"][b, :lens[b], :d]
        for h in range(H):
            q_lat = x["w_uk"][h, :, :d].T @ x["q_nope"][b, h]       # absorbed query
            s = 0.4 * (C @ q_lat + x["k_r"][b, :lens[b]] @ x["q_pe"][b, h])
            p = np.exp(s - s.max()); p /= p.sum()
            o_lat = p @ C
            np.testing.assert_allclose(got[b, h], x["w_uv"][h, :, :d] @ o_lat, rtol=1e-12, atol=1e-12)


def test_mla_full_rank_is_sdpa_on_reconstructed_cache_and_prefix_mask_equals_truncation():
    x = _mla_inputs(5)
    r = x["c"].shape[-1]
    B, H, Dn = x["q_nope"].shape
    T = x["c"].shape[1]
    got = attention.mla_decode_unabsorbed(**x, d=r, lens=[T] * B, sigma=0.25)
    K = np.concatenate([np.einsum("hnr,btr->bhtn", x["w_uk"], x["c"]),
                        np.repeat(x["k_r"][:, None], H, 1)], -1)
    V = np.einsum("hnr,btr->bhtn", x["w_uv"], x["c"])
    q = np.concatenate([x["q_nope"], x["q_pe"]], -1)
    ref = torch.nn.functional.scaled_dot_product_attention(
        torch.from_numpy(q)[:, :, None], torch.from_numpy(K), torch.from_numpy(V), scale=0.25)[:, :, 0]
    np.testing.assert_allclose(got, ref.numpy(), rtol=1e-12, atol=1e-12)
    # Appendix C.2: training zeroes coordinates past d (prefix mask); a
    # deployed kernel stores only the first d.  Both read the same scores.
    d = 5
    masked = dict(x); masked["c"] = x["c"].copy(); masked["c"][..., d:] = 0
    np.testing.assert_allclose(
        attention.mla_decode_unabsorbed(**masked, d=r, lens=[T] * B, sigma=0.25),
        attention.mla_decode_unabsorbed(**x, d=d, lens=[T] * B, sigma=0.25), rtol=1e-12, atol=1e-12)


def test_plan_inheritors_read_source_and_full_precision_is_plain_attention():
    rng = np.random.default_rng(6)
    B, Hq, Hkv, T, D = 2, 4, 2, 70, 64
    owns = [1, 0, 1, 0]
    k = {l: rng.standard_normal((B, Hkv, T, D)).astype(np.float32) for l in (0, 2)}
    v = {l: rng.standard_normal((B, Hkv, T, D)).astype(np.float32) for l in (0, 2)}
    lens = {0: np.array([70, 33]), 2: np.array([70, 33])}
    st = {0: cache.anchor_state(k[0], v[0], lens[0], 16),
          2: cache.anchor_state(k[2], v[2], lens[2], 8, 32, "channel")}
    qs = [rng.standard_normal((B, Hq, D)) for _ in range(4)]
    outs = cache.plan_outputs(owns, st, qs, lens, 0.125)
    np.testing.assert_allclose(outs[1], attention.gqa_decode(qs[1], k[0], v[0], lens[0], 0.125), atol=1e-13)
    # per-channel key state for sequence 1 (33 tokens): 1 full group + 1 residual
    assert st[2]["k_codes"][1].shape == (Hkv, 32, D) and st[2]["k_residual"][1].shape == (Hkv, 1, D)
    kh = quant.dequantise_per_channel(st[2]["k_codes"][1], st[2]["k_scale"][1], st[2]["k_zero"][1], 32,
                                      st[2]["k_residual"][1])
    np.testing.assert_allclose(st[2]["k_hat"][1, :, :33], kh, atol=0)


# ---- chunk (prefill) attention ----------------------------------------------
def _brute_prefill(q, K, V, lens, sigma):
    B, C, Hq, D = q.shape
    G = Hq // K.shape[1]
    out = np.zeros(q.shape, np.float64)
    for b in range(B):
        for i in range(C):
            p = int(lens[b]) - C + i
            if p < 0:
                continue
            for h in range(Hq):
                j = h // G
                sc = [sigma * sum(float(q[b, i, h, c]) * float(K[b, j, t, c]) for c in range(D))
                      for t in range(p + 1)]
                m = max(sc)
                w = [math.exp(x - m) for x in sc]
                tot = sum(w)
                for c in range(D):
                    out[b, i, h, c] = sum(w[t] * float(V[b, j, t, c]) for t in range(p + 1)) / tot
    return out


def test_prefill_matches_brute_force():
    rng = np.random.default_rng(3)
    B, C, Hq, Hkv, T, D = 2, 4, 4, 2, 9, 3
    q = rng.standard_normal((B, C, Hq, D))
    K = rng.standard_normal((B, Hkv, T, D))
    V = rng.standard_normal((B, Hkv, T, D))
    lens = [9, 3]  # sequence 1: the first query sits before position 0
    got = attention.gqa_prefill(q, K, V, lens, 0.7)
    np.testing.assert_allclose(got, _brute_prefill(q, K, V, lens, 0.7), rtol=1e-12, atol=1e-12)
    assert (got[1, 0] == 0).all()


def test_prefill_matches_library_causal_sdpa():
    # torch's scaled_dot_product_attention with an explicit causal mask whose
    # diagonal is shifted by the cached prefix, in float64
    rng = np.random.default_rng(4)
    B, C, Hq, Hkv, T, D = 1, 6, 6, 3, 20, 8
    q = rng.standard_normal((B, C, Hq, D))
    K = rng.standard_normal((B, Hkv, T, D))
    V = rng.standard_normal((B, Hkv, T, D))
    G = Hq // Hkv
    qt = torch.from_numpy(q).permute(0, 2, 1, 3)                      # [B, Hq, C, D]
    kt = torch.from_numpy(K).repeat_interleave(G, dim=1)               # [B, Hq, T, D]
    vt = torch.from_numpy(V).repeat_interleave(G, dim=1)
    mask = torch.arange(T)[None, :] <= (T - C + torch.arange(C))[:, None]
    ref = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, attn_mask=mask, scale=0.3)
    got = attention.gqa_prefill(q, K, V, [T], 0.3)
    np.testing.assert_allclose(got, ref.permute(0, 2, 1, 3).numpy(), rtol=1e-12, atol=1e-12)


def test_prefill_first_position_returns_its_value_and_last_query_is_decode():
    rng = np.random.default_rng(5)
    B, C, Hq, Hkv, D = 1, 5, 4, 1, 6
    q = rng.standard_normal((B, C, Hq, D))
    K = rng.standard_normal((B, Hkv, C, D))
    V = rng.standard_normal((B, Hkv, C, D))
    got = attention.gqa_prefill(q, K, V, [C], 1.0)
    # the chunk is the whole sequence: query 0 sees only position 0
    np.testing.assert_array_equal(got[0, 0], np.broadcast_to(V[0, 0, 0], (Hq, D)))
    # the last query sees every position: one decode step
    np.testing.assert_allclose(got[:, -1], attention.gqa_decode(q[:, -1], K, V, [C], 1.0),
                               rtol=1e-13, atol=1e-13)


# ---- MLA chunk (prefill) attention ------------------------------------------
def _mla_case(seed, B=2, C=5, H=3, Dn=4, dR=2, r=6, d=4, T=11):
    rng = np.random.default_rng(seed)
    return (rng.standard_normal((B, C, H, Dn)), rng.standard_normal((B, C, H, dR)),
            rng.standard_normal((B, T, r)), rng.standard_normal((B, T, dR)),
            rng.standard_normal((H, Dn, r)), rng.standard_normal((H, Dn + 1, r)), d)


def test_mla_prefill_matches_library_causal_sdpa():
    # per head: keys [W_UK c[:d] ; k^R], queries [q_nope ; q_pe], values
    # W_UV c[:d]; torch's scaled_dot_product_attention with the causal mask
    # shifted by the cached prefix, in float64
    qn, qp, c, kr, wk, wv, d = _mla_case(6)
    B, C, H, _ = qn.shape
    T = c.shape[1]
    lens = [T, T]
    Kc = np.einsum("hnk,btk->bhtn", wk[:, :, :d], c[:, :, :d])
    K = np.concatenate([Kc, np.broadcast_to(kr[:, None], (B, H) + kr.shape[1:])], -1)
    V = np.einsum("hvk,btk->bhtv", wv[:, :, :d], c[:, :, :d])
    Q = np.concatenate([qn, qp], -1).transpose(0, 2, 1, 3)
    mask = torch.arange(T)[None, :] <= (T - C + torch.arange(C))[:, None]
    ref = torch.nn.functional.scaled_dot_product_attention(
        torch.from_numpy(np.ascontiguousarray(Q)), torch.from_numpy(np.ascontiguousarray(K)),
        torch.from_numpy(V), attn_mask=mask, scale=0.4)
    got = attention.mla_prefill_unabsorbed(qn, qp, c, kr, wk, wv, d, lens, 0.4)
    np.testing.assert_allclose(got, ref.permute(0, 2, 1, 3).numpy(), rtol=1e-12, atol=1e-12)


def test_mla_prefill_short_sequence_and_last_query_is_decode():
    qn, qp, c, kr, wk, wv, d = _mla_case(7)
    C = qn.shape[1]
    lens = [c.shape[1], 3]  # sequence 1: its first C - 3 queries sit before position 0
    got = attention.mla_prefill_unabsorbed(qn, qp, c, kr, wk, wv, d, lens, 0.5)
    assert (got[1, :C - 3] == 0).all()
    dec = attention.mla_decode_unabsorbed(qn[:, -1], qp[:, -1], c, kr, wk, wv, d, lens, 0.5)
    np.testing.assert_allclose(got[:, -1], dec, rtol=1e-13, atol=1e-13)
    # query C - 3 of sequence 1 sits at position 0: it returns that position's value
    np.testing.assert_allclose(got[1, C - 3], np.einsum("hvk,k->hv", wv[:, :, :d], c[1, 0, :d]),
                               rtol=1e-12, atol=1e-12)
