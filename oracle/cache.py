"""Oracle for a whole per-layer plan (test infrastructure).

A plan holds one action per layer (Sec. 2.2): inherit, or produce a cache at
some bit-width (and, for MLA, some kept width).  The plan is fixed for the
whole generation (Sec. 2.3), so an anchor's stored state depends only on the
tokens written to it.

``anchor_state`` turns the raw keys/values written to one anchor into what
the cache stores (codes, scales, zeros, residual) and into the float64
dequantised keys/values attention reads.  ``plan_outputs`` resolves every
layer's source (nearest preceding anchor, Sec. 2.1) and runs
``attention.gqa_decode`` with that layer's own query.
"""
from __future__ import annotations

import numpy as np

from . import quant
from .attention import gqa_decode, resolve_sources


def anchor_state(k, v, lens, bits, group=None, key_axis="token", value_axis="token",
                 scheme="grouped"):
    """Stored and dequantised state of one GQA anchor.

    k, v : ``[B, H_kv, T, D]`` values as written (float32-exact)
    lens : ``[B]`` tokens written per sequence
    scheme : ``"grouped"`` (asymmetric, scale and zero per group) or
             ``"symmetric"`` (the paper's per-vector quantiser: one bf16
             scale per token-head row of keys and of values, Appendix C.3)
    Returns a dict with ``k_hat``/``v_hat`` (float64, zero past ``lens``) and,
    for quantised layers, the stored ``k_codes``, ``k_scale``, ``k_zero``,
    ``v_codes``, ``v_scale``, ``v_zero`` and (per-channel keys)
    ``k_residual``; per-channel entries are lists indexed by sequence because
    each sequence's group count depends on its own length.  The symmetric
    scheme stores signed ``k_codes``/``v_codes`` and ``k_scale``/``v_scale``
    of shape ``[B, H_kv, T]``, no zeros.
    """
    k = np.asarray(k, np.float32)
    v = np.asarray(v, np.float32)
    B, H, T, D = k.shape
    st = {"bits": bits, "group": group, "key_axis": key_axis, "value_axis": value_axis,
          "scheme": scheme}
    k_hat = np.zeros(k.shape, np.float64)
    v_hat = np.zeros(v.shape, np.float64)
    if bits == 16:
        for b in range(B):
            n = int(lens[b])
            k_hat[b, :, :n] = k[b, :, :n]
            v_hat[b, :, :n] = v[b, :, :n]
        st.update(k_hat=k_hat, v_hat=v_hat)
        return st
    if scheme == "symmetric":
        kc, ks = quant.quantise_symmetric(k, bits)
        vc, vs = quant.quantise_symmetric(v, bits)
        kh = quant.dequantise_symmetric(kc, ks)
        vh = quant.dequantise_symmetric(vc, vs)
        for b in range(B):
            n = int(lens[b])
            k_hat[b, :, :n] = kh[b, :, :n]
            v_hat[b, :, :n] = vh[b, :, :n]
        st.update(k_codes=kc, k_scale=ks, v_codes=vc, v_scale=vs, k_hat=k_hat, v_hat=v_hat)
        return st
    if scheme != "grouped":
        raise ValueError(f"unknown quantisation scheme {scheme!r}")
    if value_axis != "token":
        raise ValueError("values are quantised per token")
    vc, vs, vz = quant.quantise_per_token(v, bits, group)
    st.update(v_codes=vc, v_scale=vs, v_zero=vz)
    vh = quant.dequantise_per_token(vc, vs, vz, group)
    if key_axis == "token":
        kc, ks, kz = quant.quantise_per_token(k, bits, group)
        st.update(k_codes=kc, k_scale=ks, k_zero=kz)
        kh = quant.dequantise_per_token(kc, ks, kz, group)
        for b in range(B):
            n = int(lens[b])
            k_hat[b, :, :n] = kh[b, :, :n]
    elif key_axis == "channel":
        st.update(k_codes=[], k_scale=[], k_zero=[], k_residual=[])
        for b in range(B):
            n = int(lens[b])
            c, s, z, r = quant.quantise_per_channel(k[b, :, :n], bits, group)
            st["k_codes"].append(c)
            st["k_scale"].append(s)
            st["k_zero"].append(z)
            st["k_residual"].append(r)
            k_hat[b, :, :n] = quant.dequantise_per_channel(c, s, z, group, r)
    else:
        raise ValueError(f"unknown key axis {key_axis!r}")
    for b in range(B):
        n = int(lens[b])
        v_hat[b, :, :n] = vh[b, :, :n]
    st.update(k_hat=k_hat, v_hat=v_hat)
    return st


def plan_outputs(owns, states, queries, lens, sigma, kept=None):
    """Decode output of every layer of a plan.

    owns    : per-layer bool (True = anchor)
    states  : dict anchor index -> ``anchor_state`` result
    queries : per-layer ``[B, H_q, D]``
    lens    : dict anchor index -> ``[B]`` lengths
    kept    : optional dict anchor index -> per-sequence kept positions
    """
    src = resolve_sources(owns)
    outs = []
    for l, s in enumerate(src):
        st = states[s]
        kp = None if kept is None else kept.get(s)
        outs.append(gqa_decode(queries[l], st["k_hat"], st["v_hat"], lens[s], sigma, kp))
    return outs


def mla_anchor_state(c, k_r, lens, width, bits, scheme="symmetric"):
    """Stored and dequantised state of one MLA anchor (all three axes: the
    latent truncated to its first ``width`` coordinates, Appendix C.2, and
    stored with a quantiser of Appendix C.3).

    c   : ``[B, T, >= width]`` latents as written (bf16-exact values)
    k_r : ``[B, T, d_R]`` post-RoPE positional keys
    Every position stores two vectors, the kept latent ``c[:width]`` and the
    positional key, each quantised as ONE vector:

    * ``"symmetric"`` (the paper's quantiser, bits 8/4/2): one bf16 scale per
      vector, signed codes in ``[-q, q]``;
    * ``"grouped"`` (asymmetric, bits 8/4): one float32 (scale, zero) pair
      per vector, the group spanning the whole vector.

    ``bits == 16`` stores the bf16 values (no codes).  Returns a dict with
    ``c_hat`` ``[B, T, width]`` and ``kr_hat`` ``[B, T, d_R]`` (float64,
    zero past each length) and, when quantised, ``c_codes``, ``c_scale``,
    ``kr_codes``, ``kr_scale`` (+ ``c_zero``, ``kr_zero`` for the grouped
    scheme), codes ``[B, T, n]`` and metadata ``[B, T]``.
    """
    c = np.asarray(c, np.float32)[:, :, :width]
    k_r = np.asarray(k_r, np.float32)
    B, T, _ = c.shape
    st = {"bits": bits, "scheme": scheme, "width": width}
    if bits == 16:
        c_hat, kr_hat = c.astype(np.float64), k_r.astype(np.float64)
    elif scheme == "symmetric":
        cc, cs = quant.quantise_symmetric(c, bits)
        rc, rs = quant.quantise_symmetric(k_r, bits)
        st.update(c_codes=cc, c_scale=cs, kr_codes=rc, kr_scale=rs)
        c_hat, kr_hat = quant.dequantise_symmetric(cc, cs), quant.dequantise_symmetric(rc, rs)
    elif scheme == "grouped":
        cc, cs, cz = quant.quantise_groups(c, bits)
        rc, rs, rz = quant.quantise_groups(k_r, bits)
        st.update(c_codes=cc, c_scale=cs, c_zero=cz, kr_codes=rc, kr_scale=rs, kr_zero=rz)
        c_hat = quant.dequantise_per_token(cc, cs[..., None], cz[..., None], width)
        kr_hat = quant.dequantise_per_token(rc, rs[..., None], rz[..., None], k_r.shape[-1])
    else:
        raise ValueError(f"unknown quantisation scheme {scheme!r}")
    c_hat = np.array(c_hat, np.float64)
    kr_hat = np.array(kr_hat, np.float64)
    for b in range(B):
        n = int(lens[b])
        c_hat[b, n:] = 0.0
        kr_hat[b, n:] = 0.0
    st.update(c_hat=c_hat, kr_hat=kr_hat)
    return st
