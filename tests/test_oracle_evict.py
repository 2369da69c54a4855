"""Pins for oracle/evict.py (the window-vote evictor) against brute force,
a library softmax, conservation of attention mass and planted cases."""
import math

import numpy as np
import pytest

from oracle import attention, evict


def _brute_votes(q_win, K, L, sigma, j, G):
    # scalar loops: causal softmax of every window query, summed over the
    # queries and heads, read at the positions before the window
    n_win = len(q_win)
    P = L - n_win
    vote = [0.0] * P
    for w in range(n_win):
        pw = P + w
        for h in range(j * G, (j + 1) * G):
            s = [sigma * sum(float(q_win[w][h][d]) * float(K[j][u][d]) for d in range(len(K[j][u])))
                 for u in range(pw + 1)]
            m = max(s)
            e = [math.exp(x - m) for x in s]
            z = sum(e)
            for t in range(P):
                vote[t] += e[t] / z
    return vote


def test_votes_brute_force():
    rng = np.random.default_rng(1)
    n_win, Hq, Hkv, D, L = 3, 4, 2, 5, 11
    q = rng.standard_normal((n_win, Hq, D))
    K = rng.standard_normal((Hkv, L, D))
    for j in range(Hkv):
        got = evict.window_votes(q, K, L, 0.7, j, Hq // Hkv)
        want = _brute_votes(q, K, L, 0.7, j, Hq // Hkv)
        np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-15)


def test_single_query_equals_library_softmax():
    scipy_special = pytest.importorskip("scipy.special")
    rng = np.random.default_rng(2)
    L, D = 40, 16
    q = rng.standard_normal((1, 1, D))
    K = rng.standard_normal((1, L, D))
    got = evict.window_votes(q, K, L, 0.25, 0, 1)
    full = scipy_special.softmax(0.25 * (K[0] @ q[0, 0]))
    np.testing.assert_allclose(got, full[:L - 1], rtol=1e-12)


def test_attention_mass_is_conserved():
    # every window query spreads exactly 1 over positions <= itself: the
    # prefix votes plus the window's own share equal n_win * G
    rng = np.random.default_rng(3)
    n_win, Hq, Hkv, D, L = 6, 6, 2, 8, 50
    G = Hq // Hkv
    q = rng.standard_normal((n_win, Hq, D))
    K = rng.standard_normal((Hkv, L, D))
    P = L - n_win
    for j in range(Hkv):
        prefix = evict.window_votes(q, K, L, 0.4, j, G).sum()
        own = 0.0
        for w in range(n_win):
            for h in range(j * G, (j + 1) * G):
                a = attention.softmax_weights(0.4 * (K[j, :P + w + 1] @ q[w, h]))
                own += a[P:].sum()
        assert prefix + own == pytest.approx(n_win * G, rel=1e-12)


def test_planted_position_is_kept_and_lists_are_valid():
    rng = np.random.default_rng(4)
    B, n_win, Hq, Hkv, D, T = 2, 4, 4, 2, 16, 64
    q = rng.standard_normal((B, n_win, Hq, D))
    K = rng.standard_normal((B, Hkv, T, D)) * 0.1
    # position 7 of KV head 1, sequence 0: a key along every window query of
    # that head's group takes almost all of their attention
    K[0, 1, 7] = 40.0 * q[0, :, 2:4].sum(axis=(0, 1)) / np.linalg.norm(q[0, :, 2:4].sum(axis=(0, 1)))
    lens = [64, 20]
    kept, votes = evict.snapkv_kept(q, K, lens, 0.25, budget=24)
    assert 7 in kept[0][1]
    assert votes[0][1].argmax() == 7
    for b, L in enumerate(lens):
        for j in range(Hkv):
            kp = kept[b][j]
            assert len(kp) == min(L, 24)
            assert np.all(np.diff(kp) > 0) and kp[0] >= 0 and kp[-1] < L
            if L > 24:
                assert set(range(L - n_win, L)) <= set(kp.tolist())  # the window is kept
    # sequence 1 (20 positions <= budget) keeps everything
    assert all(np.array_equal(kept[1][j], np.arange(20)) for j in range(Hkv))


def test_select_breaks_ties_by_position():
    v = np.array([0.5, 0.9, 0.5, 0.9, 0.1, 0.5])
    assert evict.select(v, 3).tolist() == [0, 1, 3]   # 0.9, 0.9, then the first 0.5
    assert evict.select(v, 4).tolist() == [0, 1, 2, 3]
    assert evict.select(v, 10).tolist() == list(range(6))


def test_per_head_kept_lists_in_decode():
    # per-head lists that are all equal give the shared-list result; distinct
    # lists read distinct positions per KV head
    rng = np.random.default_rng(5)
    B, Hq, Hkv, T, D = 2, 4, 2, 30, 8
    q = rng.standard_normal((B, Hq, D))
    K = rng.standard_normal((B, Hkv, T, D))
    V = rng.standard_normal((B, Hkv, T, D))
    shared = [np.array([1, 4, 9, 20]), np.array([0, 2])]
    a = attention.gqa_decode(q, K, V, [T, T], 0.3, shared)
    b = attention.gqa_decode(q, K, V, [T, T], 0.3, [[s, s] for s in shared])
    np.testing.assert_array_equal(a, b)
    per = [[np.array([1, 4]), np.array([9, 20, 29])], [np.array([0]), np.array([2, 3])]]
    c = attention.gqa_decode(q, K, V, [T, T], 0.3, per)
    for bb in range(B):
        for h in range(Hq):
            j = h // 2
            d = attention.gqa_decode(q[bb:bb + 1, h:h + 1], K[bb:bb + 1, j:j + 1], V[bb:bb + 1, j:j + 1],
                                     [T], 0.3, [per[bb][j]])
            np.testing.assert_allclose(c[bb, h], d[0, 0], rtol=1e-13)
