"""Oracle of the attention-scored evictor (test infrastructure; see
``oracle/__init__.py``).

Sec. 3.4 composes token eviction with the cache plan: an evictor runs on
the same (compressed) cache and the reduction factors multiply.  The
evictors the paper runs (SnapKV and its relatives, Appendix "Eviction
implementations") score positions by summing attention over a 32-query
observation window.  The paper gives no formula; the reading used here (and
by the CUDA path):

* the window is the last ``n_win`` positions of the sequence; window query
  ``w`` sits at position ``p_w = len - n_win + w`` and attends causally to
  positions ``0 .. p_w`` with the layer's softmax scale;
* in a GQA layer the selection is per KV head ``j``: the vote of a position
  ``t < len - n_win`` sums the attention weights the window queries of every
  query head of ``j`` put on it,
      vote[j, t] = sum_w sum_{h in group j} softmax_{u <= p_w}(sigma <q_{w,h}, k_u>)[t];
* the ``budget - n_win`` positions with the largest votes are kept (equal
  votes: the smaller position first), together with the whole window; a
  sequence of at most ``budget`` positions keeps everything; the kept list
  is sorted;
* no pooling of the votes (the paper does not mention one).

Everything is float64 on dequantised keys.
"""
from __future__ import annotations

import numpy as np

from .attention import softmax_weights


def window_votes(q_win, k_hat, length, sigma, j, G):
    """Votes of the positions before the window for KV head ``j`` of one
    sequence.  ``q_win``: ``[n_win, H_q, D]``; ``k_hat``: ``[H_kv, T, D]``.
    Returns ``[length - n_win]`` float64."""
    q_win = np.asarray(q_win, np.float64)
    n_win = q_win.shape[0]
    P = length - n_win
    vote = np.zeros(max(P, 0), np.float64)
    for w in range(n_win):
        pw = P + w
        K = np.asarray(k_hat[j, :pw + 1], np.float64)
        for h in range(j * G, (j + 1) * G):
            a = softmax_weights(sigma * (K @ q_win[w, h]))
            vote += a[:P]
    return vote


def select(vote, keep):
    """Indices of the ``keep`` largest votes (equal votes: smaller index
    first), sorted ascending."""
    vote = np.asarray(vote, np.float64)
    if keep >= vote.size:
        return np.arange(vote.size)
    order = np.lexsort((np.arange(vote.size), -vote))  # by -vote, then index
    return np.sort(order[:keep])


def snapkv_kept(q_win, k_hat, lens, sigma, budget):
    """Kept lists per (sequence, KV head).

    q_win : ``[B, n_win, H_q, D]`` window queries
    k_hat : ``[B, H_kv, T, D]`` dequantised keys
    Returns ``kept[b][j]`` (int64 arrays, sorted) and the votes
    ``votes[b][j]`` (float64 over the positions before the window; empty
    when the sequence keeps everything).
    """
    q_win = np.asarray(q_win, np.float64)
    B, n_win, Hq, D = q_win.shape
    Hkv = k_hat.shape[1]
    G = Hq // Hkv
    if budget < n_win:
        raise ValueError("the budget must hold the window")
    kept, votes = [], []
    for b in range(B):
        L = int(lens[b])
        kb, vb = [], []
        for j in range(Hkv):
            if L <= budget:
                kb.append(np.arange(L))
                vb.append(np.zeros(0))
                continue
            v = window_votes(q_win[b], k_hat[b], L, sigma, j, G)
            sel = select(v, budget - n_win)
            kb.append(np.concatenate([sel, np.arange(L - n_win, L)]))
            vb.append(v)
        kept.append(kb)
        votes.append(vb)
    return kept, votes
