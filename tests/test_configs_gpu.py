"""The five benchmark workloads through the same calls bench.py times.

Reduced sizes are checked against the oracle in full (every layer, every
output).  Full sizes are checked on sampled (sequence, head) outputs the
oracle computes one by one, in the bench's launch configuration
(automatic split count)."""
import math

import numpy as np
import pytest
import torch

from _parity import assert_close, f32, gqa_expected, layers_from, oracle_state
from oracle import attention as oatt
from paper_2609_37988_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def _gqa_cache(w, max_ctx, max_splits=64):
    from paper_2609_37988_gb300.cache import Cache
    return Cache(n_layers=w.n_layers, n_q_heads=w.n_q_heads, n_kv_heads=w.n_kv_heads,
                 head_dim=w.head_dim, max_batch=w.batch, max_ctx=max_ctx, layers=layers_from(w),
                 max_splits=max_splits)


def _run_gqa(w, check_rows=None):
    """Fill every anchor (context - 1 positions, then one appended position
    when the workload appends per step), decode every layer, compare."""
    T = w.context
    c = _gqa_cache(w, T)
    states, inputs = {}, {}
    pre = T - 1 if w.append_per_step else T
    for a in w.anchors:
        k, v = W.kv_inputs(w, a, 0, pre, device="cuda")
        c.append(a, k, v)
        if w.append_per_step:
            k1, v1 = W.kv_inputs(w, a, pre, T, device="cuda")
            c.append(a, k1, v1)
            k, v = torch.cat([k, k1], 1), torch.cat([v, v1], 1)
        inputs[a] = (k, v)
    lens = np.full(w.batch, T)
    kept = {}
    if w.keep:
        for a in w.anchors:
            idx, n = W.kept_positions(w, a, lens, device="cuda")
            c.set_kept(a, idx, n)
            kept[a] = [idx[b, :int(n[b])].cpu().numpy() for b in range(w.batch)]
    src = w.sources()
    for l in range(w.n_layers):
        q = W.queries(w, l, device="cuda")
        out = f32(c.decode(l, q, w.sigma))
        a = src[l]
        cfg = w.layers[a]
        k, v = inputs[a]
        rows = range(w.batch) if check_rows is None else check_rows
        rows = list(rows)
        kb = f32(k[rows]); vb = f32(v[rows])
        st = oracle_state(kb, vb, lens[rows], cfg)
        kp = None if not kept else [kept[a][b] for b in rows]
        ref = gqa_expected(q[rows], st, lens[rows], w.sigma, kp)
        assert_close(out[rows], ref, what=f"{w.name} layer {l} (src {a})")
    assert c.device_error() == 0


@pytest.mark.parametrize("n,kw", [
    (1, {}),                                                   # the toy, in full
    (2, dict(batch=2, context=300, n_layers=6)),
    (3, dict(batch=2, context=200, n_layers=8)),
    (5, dict(batch=2, context=2048, n_layers=4)),
], ids=["cfg1", "cfg2-small", "cfg3-small", "cfg5-small"])
def test_gqa_workloads_reduced(n, kw):
    _run_gqa(W.config(n, **kw))


def test_mla_workload_reduced():
    w = W.config(4, batch=3, context=300, n_layers=4)
    from paper_2609_37988_gb300.cache import Cache
    c = Cache(kind="mla", n_layers=w.n_layers, n_q_heads=16, head_dim=128, latent_dim=512,
              rope_dim=64, max_batch=w.batch, max_ctx=w.context, layers=layers_from(w))
    lens = np.full(w.batch, w.context)
    for l in range(w.n_layers):
        cl, kr = W.mla_inputs(w, l, 0, w.context, device="cuda")
        c.append(l, cl, kr)
        wk, wv = W.mla_weights(w, l, device="cuda")
        qn, qp = W.mla_queries(w, l, device="cuda")
        out = c.decode_mla(l, qn, qp, wk, wv, w.sigma)
        d = w.layers[l]["width"]
        ref = oatt.mla_decode_unabsorbed(f32(qn), f32(qp), f32(cl), f32(kr), f32(wk), f32(wv), d,
                                         lens, w.sigma)
        assert_close(f32(out), ref, what=f"mla layer {l} d={d}")


def _one_anchor_of_each_kind(w):
    """The workload cut to the first anchor of each storage kind (bits,
    quantiser, key axis), each followed by an inheritor, in layer order; the
    per-layer input scales follow their anchors."""
    picked = {}
    for a in w.anchors:
        cfg = w.layers[a]
        picked.setdefault((cfg["bits"], cfg["scheme"], cfg["key_axis"]), a)
    layers, scale = [], {}
    for a in sorted(picked.values()):
        if a in w.kv_scale:
            scale[len(layers)] = w.kv_scale[a]
        layers.append(dict(w.layers[a]))
        layers.append(dict(w.layers[a], inherit=True))
    w.layers, w.n_layers, w.kv_scale = layers, len(layers), scale
    return w


@pytest.mark.slow
@pytest.mark.parametrize("n,sym", [(2, None), (3, None), (5, None), (3, 8), (3, 4), (3, 2)],
                         ids=["cfg2", "cfg3", "cfg5", "cfg3-sym8", "cfg3-sym4", "cfg3-sym2"])
def test_full_size_sampled(n, sym):
    """Full geometry (batch, context, heads, the bench's automatic split
    count), one anchor of every storage kind the workload holds (and an
    inheritor reading it), sampled sequences against the oracle."""
    w = _one_anchor_of_each_kind(W.config(n, sym_bits=sym))
    if sym is not None:  # the bf16 anchors are covered by the cfg3 case
        w.layers = [a for a in w.layers if a["bits"] != 16]
        w.n_layers = len(w.layers)
    _run_gqa(w, check_rows=[0, w.batch - 1])


@pytest.mark.slow
def test_mla_full_size_sampled():
    w = W.config(4, n_layers=2)
    from paper_2609_37988_gb300.cache import Cache
    c = Cache(kind="mla", n_layers=w.n_layers, n_q_heads=16, head_dim=128, latent_dim=512,
              rope_dim=64, max_batch=w.batch, max_ctx=w.context, layers=layers_from(w))
    rows = [0, 31, 63]
    for l in range(w.n_layers):
        cl, kr = W.mla_inputs(w, l, 0, w.context, device="cuda")
        c.append(l, cl, kr)
        wk, wv = W.mla_weights(w, l, device="cuda")
        qn, qp = W.mla_queries(w, l, device="cuda")
        out = f32(c.decode_mla(l, qn, qp, wk, wv, w.sigma))
        d = w.layers[l]["width"]
        ref = oatt.mla_decode_unabsorbed(f32(qn[rows]), f32(qp[rows]), f32(cl[rows]), f32(kr[rows]),
                                         f32(wk), f32(wv), d, [w.context] * 3, w.sigma)
        assert_close(out[rows], ref, what=f"mla full layer {l} d={d}")
