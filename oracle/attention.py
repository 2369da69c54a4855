"""Oracle decode attention (test infrastructure; see ``oracle/__init__.py``).

Everything here runs in float64 on already-dequantised caches.

* ``resolve_sources`` -- Sec. 2.1 (depth axis): a layer either owns a cache
  (an *anchor*) or inherits from the nearest anchor before it; layer 1 must
  own one (Sec. 2.2, below eq. compression).  Returns ``src[l]``.
* ``gqa_decode`` -- one decode step of grouped-query attention for every
  query head: query head ``h`` reads KV head ``h // G`` (contiguous groups of
  ``G = H_q / H_kv``), scores ``s_t = sigma * <q_h, k_t>``, softmax over the
  positions the layer reads, output ``sum_t p_t v_t``.  With a kept-position
  list (eviction composed with compression, Sec. 3.4) only the listed
  positions are read.
* ``gqa_prefill`` -- attention of a chunk of new queries over the
  compressed cache: the chunk is the last ``C`` positions of each sequence
  (already written to the cache), and query ``i`` at position
  ``len - C + i`` attends causally to positions ``0 .. len - C + i`` of the
  dequantised cache (the other side of the step the paper times as
  pre-fill, Sec. 4: the cache holds the compressed keys and values the
  decode steps then read).  Queries before position 0 give zeros.
* ``mla_decode_unabsorbed`` -- Appendix C.2: the MLA cache holds the latent
  ``c`` truncated to its first ``d`` coordinates and the post-RoPE positional
  key ``k^R`` shared by all heads.  Head ``h`` reconstructs its content key
  ``W_UK^h[:, :d] c[:d]`` and value ``W_UV^h[:, :d] c[:d]`` explicitly; the
  score adds ``<q_pe^h, k^R>``.  The GPU computes the absorbed form; the
  algebraic identity between the two is pinned by a test.
* ``mla_prefill_unabsorbed`` -- the chunk attention of an MLA layer: query
  ``i`` of the chunk (the last ``C`` positions of each sequence) at position
  ``len - C + i`` attends causally to positions ``0 .. len - C + i`` with the
  explicitly reconstructed keys and values of ``mla_decode_unabsorbed``.
"""
from __future__ import annotations

import numpy as np


def resolve_sources(owns):
    """``owns[l]`` true when layer ``l`` (0-based) owns a cache.

    Returns ``src`` with ``src[l] = l`` for anchors and the nearest anchor
    index ``< l`` for inheritors.  Raises ``ValueError`` if layer 0 inherits.
    """
    owns = [bool(o) for o in owns]
    if not owns or not owns[0]:
        raise ValueError("layer 0 must own a cache")
    src = []
    last = 0
    for l, o in enumerate(owns):
        if o:
            last = l
        src.append(last)
    return src


def softmax_weights(scores: np.ndarray) -> np.ndarray:
    """Numerically safe softmax along the last axis (float64)."""
    s = np.asarray(scores, dtype=np.float64)
    m = s.max(axis=-1, keepdims=True)
    e = np.exp(s - m)
    return e / e.sum(axis=-1, keepdims=True)


def gqa_decode(q, k_hat, v_hat, lens, sigma, kept=None):
    """One decode step over a GQA cache.

    q      : ``[B, H_q, D]``
    k_hat  : ``[B, H_kv, T, D]`` dequantised keys (positions >= lens[b] unused)
    v_hat  : ``[B, H_kv, T, D]``
    lens   : ``[B]`` valid positions per sequence
    sigma  : softmax scale
    kept   : optional list (per sequence) of position arrays to read instead
             of ``0..lens[b]-1``; an entry may instead be a list of arrays,
             one per KV head (per-head kept lists)
    Returns ``[B, H_q, D]`` float64.
    """
    q = np.asarray(q, np.float64)
    B, Hq, D = q.shape
    Hkv = k_hat.shape[1]
    if Hq % Hkv:
        raise ValueError("H_q must be a multiple of H_kv")
    G = Hq // Hkv
    out = np.zeros((B, Hq, D), np.float64)
    for b in range(B):
        per_head = kept is not None and isinstance(kept[b], (list, tuple))
        for h in range(Hq):
            j = h // G
            if kept is None:
                pos = np.arange(int(lens[b]))
            else:
                pos = np.asarray(kept[b][j] if per_head else kept[b], np.int64)
            if pos.size == 0:
                continue
            K = np.asarray(k_hat[b, j, pos], np.float64)
            V = np.asarray(v_hat[b, j, pos], np.float64)
            p = softmax_weights(sigma * (K @ q[b, h]))
            out[b, h] = p @ V
    return out


def gqa_prefill(q, k_hat, v_hat, lens, sigma):
    """Causal chunk attention over a GQA cache.

    q      : ``[B, C, H_q, D]`` the queries of each sequence's last ``C``
             positions
    k_hat  : ``[B, H_kv, T, D]`` dequantised keys, v_hat likewise
    lens   : ``[B]`` positions held (the chunk included)
    Returns ``[B, C, H_q, D]`` float64.
    """
    q = np.asarray(q, np.float64)
    B, C, Hq, D = q.shape
    Hkv = k_hat.shape[1]
    if Hq % Hkv:
        raise ValueError("H_q must be a multiple of H_kv")
    G = Hq // Hkv
    out = np.zeros((B, C, Hq, D), np.float64)
    for b in range(B):
        L = int(lens[b])
        for i in range(C):
            p = L - C + i  # position of query i
            if p < 0:
                continue
            for h in range(Hq):
                j = h // G
                K = np.asarray(k_hat[b, j, :p + 1], np.float64)
                V = np.asarray(v_hat[b, j, :p + 1], np.float64)
                w = softmax_weights(sigma * (K @ q[b, i, h]))
                out[b, i, h] = w @ V
    return out


def mla_decode_unabsorbed(q_nope, q_pe, c, k_r, w_uk, w_uv, d, lens, sigma):
    """MLA decode step, content keys and values reconstructed explicitly.

    q_nope : ``[B, H, Dn]``      q_pe : ``[B, H, dR]`` (post-RoPE)
    c      : ``[B, T, >=d]``     latent cache (only ``[:d]`` is read)
    k_r    : ``[B, T, dR]``      positional key (post-RoPE)
    w_uk   : ``[H, Dn, r]``      w_uv : ``[H, Dv, r]``
    Returns ``[B, H, Dv]`` float64.
    """
    q_nope = np.asarray(q_nope, np.float64)
    q_pe = np.asarray(q_pe, np.float64)
    B, H, _ = q_nope.shape
    Dv = w_uv.shape[1]
    out = np.zeros((B, H, Dv), np.float64)
    for b in range(B):
        T = int(lens[b])
        if T == 0:
            continue
        C = np.asarray(c[b, :T, :d], np.float64)          # [T, d]
        KR = np.asarray(k_r[b, :T], np.float64)           # [T, dR]
        for h in range(H):
            Wk = np.asarray(w_uk[h, :, :d], np.float64)   # [Dn, d]
            Wv = np.asarray(w_uv[h, :, :d], np.float64)   # [Dv, d]
            Kc = C @ Wk.T                                 # [T, Dn] content keys
            Vh = C @ Wv.T                                 # [T, Dv] values
            s = sigma * (Kc @ q_nope[b, h] + KR @ q_pe[b, h])
            out[b, h] = softmax_weights(s) @ Vh
    return out


def mla_prefill_unabsorbed(q_nope, q_pe, c, k_r, w_uk, w_uv, d, lens, sigma):
    """MLA chunk attention, content keys and values reconstructed explicitly.

    q_nope : ``[B, C, H, Dn]``   q_pe : ``[B, C, H, dR]`` (post-RoPE), the
             queries of each sequence's last ``C`` positions
    c, k_r, w_uk, w_uv : as for ``mla_decode_unabsorbed``; ``lens`` the
             positions held (the chunk included)
    Returns ``[B, C, H, Dv]`` float64; queries before position 0 give zeros.
    """
    q_nope = np.asarray(q_nope, np.float64)
    q_pe = np.asarray(q_pe, np.float64)
    B, C, H, _ = q_nope.shape
    Dv = w_uv.shape[1]
    out = np.zeros((B, C, H, Dv), np.float64)
    for b in range(B):
        L = int(lens[b])
        Cb = np.asarray(c[b, :L, :d], np.float64)           # [L, d]
        KR = np.asarray(k_r[b, :L], np.float64)             # [L, dR]
        for h in range(H):
            Wk = np.asarray(w_uk[h, :, :d], np.float64)     # [Dn, d]
            Wv = np.asarray(w_uv[h, :, :d], np.float64)     # [Dv, d]
            Kc = Cb @ Wk.T                                  # [L, Dn] content keys
            Vh = Cb @ Wv.T                                  # [L, Dv] values
            for i in range(C):
                p = L - C + i  # position of query i
                if p < 0:
                    continue
                s = sigma * (Kc[:p + 1] @ q_nope[b, i, h] + KR[:p + 1] @ q_pe[b, i, h])
                out[b, i, h] = softmax_weights(s) @ Vh[:p + 1]
    return out
