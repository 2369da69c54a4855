"""GPU parity of the window-vote evictor composed with the compressed cache
(Sec. 3.4; Appendix, eviction implementations: votes summed over an
observation window of queries), through the C ABI.

The votes are compared with the fp64 oracle on the same dequantised keys;
the kept lists must equal the oracle's except where two votes sit within
the fp32 scoring error of the cut (a swap between near-equal votes is then
valid); decode over the installed per-(sequence, KV head) lists is compared
with the oracle's decode over the oracle's lists."""
import math

import numpy as np
import pytest
import torch

from _parity import assert_close, f32, gqa_expected, oracle_state
from oracle import evict as oev

pytestmark = pytest.mark.gpu

FORMATS = [
    dict(bits=16, group=64, key_axis="token"),
    dict(bits=8, group=64, key_axis="token"),
    dict(bits=4, group=32, key_axis="token"),
    dict(bits=8, group=64, key_axis="token", scheme="symmetric"),
    dict(bits=4, group=64, key_axis="token", scheme="symmetric"),
    dict(bits=2, group=64, key_axis="token", scheme="symmetric"),
]

# Votes against the fp64 oracle.  On the tensor cores each factor enters as
# bf16 hi + lo (residual <= 2^-18 of it) and the lo*lo product is dropped, so
# a score's error is at most 3 * 2^-18 * sigma * log2(e) * sum_i |q_i k_i|
# (~1.7e-4 in log2 units for these inputs) and a vote's relative error at
# most 2 ln 2 times that; with independent rounding errors it is ~10x less.
# The CUDA-core fallback (fp32 products) is tighter still.
VOTE_RTOL = 1e-4
VOTE_ATOL = 1e-7


def _fid(f):
    return f"{f.get('scheme', 'grouped')[:3]}{f['bits']}"


def _cache(B, Hq, Hkv, D, T, layers):
    from paper_2609_37988_gb300.cache import Cache, Layer
    return Cache(n_layers=len(layers), n_q_heads=Hq, n_kv_heads=Hkv, head_dim=D, max_batch=B,
                 max_ctx=T, layers=[Layer(**l) for l in layers], max_splits=16)


def _fill(cache, B, Hkv, D, counts, seed, spread=1.5):
    g = torch.Generator().manual_seed(seed)
    n = max(counts)
    k = (torch.randn((B, n, Hkv, D), generator=g) * spread + 0.3).to(torch.bfloat16)
    v = torch.randn((B, n, Hkv, D), generator=g).to(torch.bfloat16)
    cache.append(0, k.cuda(), v.cuda(), n_per_seq=torch.tensor(counts, dtype=torch.int32,
                                                                 device="cuda"))
    return k.float().numpy(), v.float().numpy(), np.array(counts)


def _qwin(B, n_win, Hq, D, seed, dtype=torch.bfloat16):
    g = torch.Generator().manual_seed(seed)
    return torch.randn((B, n_win, Hq, D), generator=g).to(dtype)


def _check_lists(cache, q, st, lens, sigma, budget, votes_gpu, what):
    """Votes within tolerance; lists equal to the oracle's up to near-ties at
    the cut; returns the oracle's lists and whether the lists were equal."""
    B, n_win = q.shape[0], q.shape[1]
    kept, votes = oev.snapkv_kept(f32(q), st["k_hat"], lens, sigma, budget)
    got = cache.kept_lists(0)
    assert got is not None and got[2], "per-head lists installed"
    idx, n = got[0].cpu().numpy(), got[1].cpu().numpy()
    vg = f32(votes_gpu)
    exact = True
    Hkv = idx.shape[1]
    for b in range(B):
        L = int(lens[b])
        for j in range(Hkv):
            ref = kept[b][j]
            assert int(n[b, j]) == len(ref), f"{what} b{b} j{j}: n_kept {n[b, j]} != {len(ref)}"
            sel = idx[b, j, :n[b, j]]
            assert (np.diff(sel) > 0).all(), f"{what}: list not strictly increasing"
            if L <= budget:
                np.testing.assert_array_equal(sel, np.arange(L))
                continue
            P = L - n_win
            np.testing.assert_array_equal(sel[-n_win:], np.arange(P, L))   # the window
            ov = votes[b][j]
            gv = vg[b, j, :P]
            err = np.abs(gv - ov)
            assert (err <= VOTE_RTOL * np.abs(ov) + VOTE_ATOL).all(), \
                f"{what} b{b} j{j}: vote error {err.max():.3e} (mass {ov.sum():.3f})"
            # attention mass: every window query puts at most mass 1 before the window
            assert gv.sum() <= n_win * (q.shape[2] // Hkv) * (1 + 1e-5)
            chosen, want = set(sel[:-n_win].tolist()), set(ref[:-n_win].tolist())
            if chosen != want:
                exact = False
                kth = np.sort(ov)[::-1][budget - n_win - 1]
                for t in chosen ^ want:
                    assert abs(ov[t] - kth) <= 4 * (VOTE_RTOL * kth + VOTE_ATOL), \
                        f"{what} b{b} j{j}: position {t} (vote {ov[t]:.6e}) swapped at cut {kth:.6e}"
    return kept, exact


@pytest.mark.parametrize("fmt", FORMATS, ids=_fid)
@pytest.mark.parametrize("G,n_win,qdt", [(4, 32, torch.bfloat16), (5, 32, torch.float32),
                                         (5, 64, torch.bfloat16)],
                         ids=["r128", "r160-f32q", "r320-cuda-cores"])
def test_evict_votes_and_lists(fmt, G, n_win, qdt):
    # R = n_win G window rows: 128 (one row chunk), 160 (two, the second
    # partly past the query rows), 320 (scored on the CUDA cores)
    B, Hkv, D, T = 3, 2, 128, 800
    Hq = G * Hkv
    cap, budget = 256, 200
    c = _cache(B, Hq, Hkv, D, T, [dict(evict_capacity=cap, **fmt)])
    K, V, lens = _fill(c, B, Hkv, D, [700, 333, 150], seed=fmt["bits"] + 3)
    st = oracle_state(K, V, lens, fmt)
    sigma = 1.0 / math.sqrt(D)
    q = _qwin(B, n_win, Hq, D, seed=11, dtype=qdt)
    votes = c.evict_window(0, q.cuda(), sigma, budget)
    torch.cuda.synchronize()
    kept, _ = _check_lists(c, q, st, lens, sigma, budget, votes, _fid(fmt))
    assert c.device_error() == 0


@pytest.mark.parametrize("fmt", [FORMATS[0], FORMATS[2], FORMATS[4]], ids=_fid)
def test_evict_then_decode_per_head(fmt):
    # decode over the installed per-head lists against the oracle's decode
    # over the oracle's lists (the seed gives no near-tie at the cut)
    B, Hkv, G, D, T = 2, 4, 5, 128, 1100
    Hq = G * Hkv
    cap, budget, n_win = 320, 288, 16
    c = _cache(B, Hq, Hkv, D, T, [dict(evict_capacity=cap, **fmt), dict(inherit=True)])
    K, V, lens = _fill(c, B, Hkv, D, [1030, 280], seed=5)
    st = oracle_state(K, V, lens, fmt)
    sigma = 1.0 / math.sqrt(D)
    q = _qwin(B, n_win, Hq, D, seed=2, dtype=torch.float32)
    plain = c.decode(0, _qwin(B, 1, Hq, D, 9)[:, 0].contiguous().cuda(), sigma, n_splits=2).clone()
    votes = c.evict_window(0, q.cuda(), sigma, budget)
    kept, exact = _check_lists(c, q, st, lens, sigma, budget, votes, _fid(fmt))
    assert exact, "this seed has no near-tie: the lists must equal the oracle's"
    qd = _qwin(B, 1, Hq, D, 9)[:, 0].contiguous()
    ref = gqa_expected(qd, st, lens, sigma, kept)
    for ns in (0, 1, 3):
        out = c.decode(0, qd.cuda(), sigma, n_splits=ns)
        assert_close(f32(out), ref, what=f"{_fid(fmt)} per-head gather splits={ns}")
        # the inheriting layer reads the same lists
        assert torch.equal(out, c.decode(1, qd.cuda(), sigma, n_splits=ns))
    # sequence 1 (280 <= budget) keeps everything: gathered equals streamed
    # up to the order of the fp32 sums (the two paths split the positions
    # differently)
    assert_close(f32(c.decode(0, qd.cuda(), sigma, n_splits=2)[1]), f32(plain[1]), max_abs=1e-5,
                 rel_l2=1e-5, what="keep-all")
    # set_kept(None) goes back to every position
    c.set_kept(0)
    assert c.kept_lists(0) is None
    assert torch.equal(c.decode(0, qd.cuda(), sigma, n_splits=2), plain)
    assert c.device_error() == 0


def test_evict_equal_votes_keep_smaller_positions():
    # every key the same: every vote is equal, so the first budget - n_win
    # positions are kept (Sec. 3.4 reading: ties go to the smaller position)
    B, Hkv, G, D = 2, 1, 3, 64
    c = _cache(B, G, Hkv, D, 600, [dict(bits=8, group=64, key_axis="token", evict_capacity=128)])
    k = torch.full((B, 500, Hkv, D), 0.25, dtype=torch.bfloat16, device="cuda")
    v = torch.randn((B, 500, Hkv, D), device="cuda").to(torch.bfloat16)
    c.append(0, k, v, n_per_seq=torch.tensor([500, 130], dtype=torch.int32, device="cuda"))
    q = _qwin(B, 8, G, D, 4).cuda()
    c.evict_window(0, q, 0.125, 100)
    idx, n, ph = c.kept_lists(0)
    idx, n = idx.cpu().numpy(), n.cpu().numpy()
    assert ph and n.tolist() == [[100], [100]]
    np.testing.assert_array_equal(idx[0, 0, :100], np.r_[np.arange(92), np.arange(492, 500)])
    np.testing.assert_array_equal(idx[1, 0, :100], np.r_[np.arange(92), np.arange(122, 130)])


def test_evict_window_only_and_planted_key():
    # budget == n_win keeps only the window; with one more slot the planted
    # key every window query attends to is the one kept
    B, Hkv, G, D = 1, 2, 2, 128
    fmt = dict(bits=4, group=32, key_axis="token", evict_capacity=64)
    c = _cache(B, Hkv * G, Hkv, D, 400, [fmt])
    g = torch.Generator().manual_seed(3)
    k = torch.randn((B, 300, Hkv, D), generator=g) * 0.3
    q = torch.randn((B, 8, Hkv * G, D), generator=g)
    k[0, 77, 0] = q[0, :, :G].mean(dim=(0, 1)) * 4      # head 0's window looks at 77
    k[0, 201, 1] = q[0, :, G:].mean(dim=(0, 1)) * 4     # head 1's at 201
    v = torch.randn((B, 300, Hkv, D), generator=g)
    c.append(0, k.to(torch.bfloat16).cuda(), v.to(torch.bfloat16).cuda())
    c.evict_window(0, q.to(torch.bfloat16).cuda(), 1 / math.sqrt(D), 8)
    idx, n, _ = c.kept_lists(0)
    assert n.cpu().tolist() == [[8, 8]]
    np.testing.assert_array_equal(idx[0, :, :8].cpu().numpy(), np.tile(np.arange(292, 300), (2, 1)))
    c.evict_window(0, q.to(torch.bfloat16).cuda(), 1 / math.sqrt(D), 9)
    idx, n, _ = c.kept_lists(0)
    idx = idx.cpu().numpy()
    np.testing.assert_array_equal(idx[0, 0, :9], np.r_[77, np.arange(292, 300)])
    np.testing.assert_array_equal(idx[0, 1, :9], np.r_[201, np.arange(292, 300)])


def test_evict_d64_and_empty_sequences():
    B, Hkv, G, D = 3, 2, 2, 64
    fmt = dict(bits=8, group=64, key_axis="token")
    c = _cache(B, Hkv * G, Hkv, D, 700, [dict(evict_capacity=200, **fmt)])
    K, V, lens = _fill(c, B, Hkv, D, [0, 640, 129], seed=8)
    st = oracle_state(K, V, lens, fmt)
    q = _qwin(B, 1, Hkv * G, D, 1)
    votes = c.evict_window(0, q.cuda(), 0.125, 100)
    _check_lists(c, q, st, lens, 0.125, 100, votes, "d64")
    out = c.decode(0, q[:, 0].contiguous().cuda(), 0.125)
    kept, _ = oev.snapkv_kept(f32(q), st["k_hat"], lens, 0.125, 100)
    assert (f32(out[0]) == 0).all()
    assert_close(f32(out[1:]), gqa_expected(q[:, 0], st, lens, 0.125, kept)[1:], what="d64 decode")


def test_evict_rejections():
    from paper_2609_37988_gb300._lib import KVKError
    c = _cache(2, 4, 2, 128, 300, [dict(bits=4, group=32, key_axis="token", evict_capacity=64),
                                   dict(inherit=True),
                                   dict(bits=8, group=64, key_axis="token"),
                                   dict(bits=8, group=64, key_axis="channel")])
    q = torch.zeros((2, 8, 4, 128), dtype=torch.bfloat16, device="cuda")
    for layer, budget, msg in ((0, 7, "below the window"), (0, 65, "above the capacity"),
                               (1, 16, "inheriting layer"), (2, 16, "no capacity"),
                               (3, 16, "per-channel keys")):
        with pytest.raises(KVKError):
            c.evict_window(layer, q, 0.1, budget)
    with pytest.raises(KVKError):
        c.evict_window(0, torch.zeros((2, 0, 4, 128), dtype=torch.bfloat16, device="cuda"), 0.1, 8)
    with pytest.raises(KVKError):
        c.evict_window(0, q, 0.0, 16)
    assert c.kept_lists(0) is None      # nothing was installed


@pytest.mark.slow
def test_evict_full_size_sampled():
    """The bench's eviction call (14B long-context shape: B=4, 8 KV / 40 q
    heads, 131072 positions, int4 g32, window 32, budget T/8) with the bench's
    inputs; two (sequence, KV head) units checked against the oracle: every
    vote, and the kept list up to near-ties at the cut."""
    import bench
    from paper_2609_37988_gb300 import workloads as W
    w, c, q = bench._evict_setup(4, 131072, torch.device("cuda", 0))
    budget, n_win = w.keep, bench.EVICT_WINDOW
    G = w.n_q_heads // w.n_kv_heads
    votes = f32(c.evict_window(0, q, w.sigma, budget))
    idx, n, _ = c.kept_lists(0)
    idx, n = idx.cpu().numpy(), n.cpu().numpy()
    assert c.device_error() == 0
    T = w.context
    P = T - n_win
    cfg = w.layers[0]
    for b, j in ((0, 0), (3, 7)):
        # the bench's inputs (drawn on the device), this unit's keys only
        k = torch.cat([W.kv_inputs(w, 0, b0, min(T, b0 + 16384), device="cuda")[0]
                       [b:b + 1, :, j:j + 1].cpu() for b0 in range(0, T, 16384)], 1)
        st = oracle_state(f32(k), f32(k), np.array([T]), cfg)
        qb = f32(q[b, :, j * G:(j + 1) * G])
        ov = oev.window_votes(qb, st["k_hat"][0], T, w.sigma, 0, G)
        gv = votes[b, j, :P]
        err = np.abs(gv - ov)
        assert (err <= VOTE_RTOL * ov + VOTE_ATOL).all(), f"unit ({b},{j}): vote error {err.max():.3e}"
        assert int(n[b, j]) == budget
        sel = idx[b, j, :budget]
        np.testing.assert_array_equal(sel[-n_win:], np.arange(P, T))
        want = set(oev.select(ov, budget - n_win).tolist())
        kth = np.sort(ov)[::-1][budget - n_win - 1]
        for t in set(sel[:-n_win].tolist()) ^ want:
            assert abs(ov[t] - kth) <= 4 * (VOTE_RTOL * kth + VOTE_ATOL), (b, j, t)
