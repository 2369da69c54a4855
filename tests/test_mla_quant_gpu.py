"""GPU parity of quantised MLA latents, all three axes of a plan at once
(Appendix C.2 truncation with the quantisers of Appendix C.3): each
position's kept latent and positional key stored as one quantised vector
each.  Codes, scales and zeros bit-exact against the oracle; decode outputs
against the oracle's unabsorbed MLA decode on the dequantised cache, over
every kept width and each code width of both schemes."""
import math

import numpy as np
import pytest
import torch

from _parity import assert_close, f32
from oracle import attention as oatt
from oracle import cache as ocache

pytestmark = pytest.mark.gpu

FORMATS = [("grouped", 8), ("grouped", 4), ("symmetric", 8), ("symmetric", 4), ("symmetric", 2)]


def _fid(f):
    return f"{'sym' if f[0] == 'symmetric' else 'g'}{f[1]}"


def _cache(B, T, layers, H=16, max_splits=16):
    from paper_2609_37988_gb300.cache import Cache, Layer
    return Cache(kind="mla", n_layers=len(layers), n_q_heads=H, head_dim=128, latent_dim=512,
                 rope_dim=64, max_batch=B, max_ctx=T, layers=[Layer(**l) for l in layers],
                 max_splits=max_splits)


def _layer(width, fmt):
    return dict(bits=fmt[1], scheme=fmt[0], width=width)


def _inputs(B, n, seed, r=512):
    g = torch.Generator().manual_seed(seed)
    decay = torch.arange(r).add(1.0).rsqrt()
    c = (torch.randn((B, n, r), generator=g) * decay).to(torch.bfloat16)
    kr = torch.randn((B, n, 64), generator=g).to(torch.bfloat16)
    return c, kr


def _weights(H, seed, r=512):
    g = torch.Generator().manual_seed(seed)
    wk = (torch.randn((H, 128, r), generator=g) / math.sqrt(512)).to(torch.bfloat16)
    wv = (torch.randn((H, 128, r), generator=g) / math.sqrt(512)).to(torch.bfloat16)
    return wk, wv


def _queries(B, H, seed):
    g = torch.Generator().manual_seed(seed)
    return (torch.randn((B, H, 128), generator=g).to(torch.bfloat16),
            torch.randn((B, H, 64), generator=g).to(torch.bfloat16))


def _check_codes(ex, st, lens):
    for b, n in enumerate(lens):
        for name in ("c", "kr"):
            np.testing.assert_array_equal(ex[name + "_codes"][b, :n].cpu().numpy(),
                                          st[name + "_codes"][b, :n])
            np.testing.assert_array_equal(ex[name + "_scale"][b, :n].cpu().numpy(),
                                          st[name + "_scale"][b, :n].astype(np.float32))
            if st["scheme"] == "grouped":
                np.testing.assert_array_equal(ex[name + "_zero"][b, :n].cpu().numpy(),
                                              st[name + "_zero"][b, :n])


@pytest.mark.parametrize("fmt", FORMATS, ids=_fid)
@pytest.mark.parametrize("width", [512, 256, 128, 64])
def test_quantised_mla_codes_and_decode(width, fmt):
    B, H = 3, 16
    lens = [300, 65, 1]
    c_ = _cache(B, 320, [_layer(width, fmt)])
    c, kr = _inputs(B, 300, width + fmt[1])
    c_.append(0, c.cuda(), kr.cuda(), n_per_seq=torch.tensor(lens, dtype=torch.int32, device="cuda"))
    st = ocache.mla_anchor_state(f32(c), f32(kr), lens, width, fmt[1], fmt[0])
    _check_codes(c_.export(0), st, lens)
    wk, wv = _weights(H, 7)
    qn, qp = _queries(B, H, 11)
    sigma = 1.0 / math.sqrt(128 + 64)
    ref = oatt.mla_decode_unabsorbed(f32(qn), f32(qp), st["c_hat"], st["kr_hat"], f32(wk), f32(wv),
                                     width, lens, sigma)
    for ns in (0, 1, 3):
        out = c_.decode_mla(0, qn.cuda(), qp.cuda(), wk.cuda(), wv.cuda(), sigma, n_splits=ns)
        assert_close(f32(out), ref, what=f"mla {_fid(fmt)} d={width} splits={ns}")
    assert c_.device_error() == 0


@pytest.mark.parametrize("fmt", [FORMATS[1], FORMATS[4]], ids=_fid)
def test_quantised_mla_sharing_fewer_heads_empty_and_appended(fmt):
    # H = 5, an empty and a 1-position sequence, more splits than tiles, an
    # inheriting layer (bit-identical), appends in two chunks (codes of a
    # position do not depend on when it was written)
    B, H, width = 4, 5, 256
    lens = [0, 1, 200, 129]
    c_ = _cache(B, 256, [_layer(width, fmt), dict(inherit=True)], H=H)
    c, kr = _inputs(B, 200, 3)
    first = [0, 1, 120, 64]
    c_.append(0, c[:, :120].cuda(), kr[:, :120].cuda(),
              n_per_seq=torch.tensor(first, dtype=torch.int32, device="cuda"))
    rest = [l - f for l, f in zip(lens, first)]
    c2 = torch.stack([torch.cat([c[b, first[b]:lens[b]], c[b, :80 - rest[b]]]) for b in range(B)])
    k2 = torch.stack([torch.cat([kr[b, first[b]:lens[b]], kr[b, :80 - rest[b]]]) for b in range(B)])
    c_.append(0, c2.cuda(), k2.cuda(), n_per_seq=torch.tensor(rest, dtype=torch.int32, device="cuda"))
    st = ocache.mla_anchor_state(f32(c), f32(kr), lens, width, fmt[1], fmt[0])
    _check_codes(c_.export(0), st, lens)
    wk, wv = _weights(H, 13)
    qn, qp = _queries(B, H, 17)
    sigma = 1.0 / math.sqrt(192)
    ref = oatt.mla_decode_unabsorbed(f32(qn), f32(qp), st["c_hat"], st["kr_hat"], f32(wk), f32(wv),
                                     width, lens, sigma)
    for ns in (0, 7, 16):
        out = c_.decode_mla(0, qn.cuda(), qp.cuda(), wk.cuda(), wv.cuda(), sigma, n_splits=ns)
        assert torch.isfinite(out).all() and (out[0] == 0).all()
        assert_close(f32(out[1:]), ref[1:], what=f"mla {_fid(fmt)} H=5 splits={ns}")
        assert torch.equal(out, c_.decode_mla(1, qn.cuda(), qp.cuda(), wk.cuda(), wv.cuda(), sigma,
                                              n_splits=ns))
    assert c_.device_error() == 0


@pytest.mark.slow
@pytest.mark.parametrize("fmt", [FORMATS[1], FORMATS[3]], ids=_fid)
def test_quantised_mla_full_size_sampled(fmt):
    # the MLA workload's geometry (64 sequences x 4096 positions, 16 heads),
    # the widest latent, automatic splits; sampled sequences
    from paper_2609_37988_gb300 import workloads as W
    w = W.config(4, n_layers=1)
    c_ = _cache(w.batch, w.context, [_layer(512, fmt)])
    cl, kr = W.mla_inputs(w, 0, 0, w.context, device="cuda")
    c_.append(0, cl, kr)
    wk, wv = W.mla_weights(w, 0, device="cuda")
    qn, qp = W.mla_queries(w, 0, device="cuda")
    out = f32(c_.decode_mla(0, qn, qp, wk, wv, w.sigma))
    rows = [0, 31, 63]
    st = ocache.mla_anchor_state(f32(cl[rows]), f32(kr[rows]), [w.context] * 3, 512, fmt[1], fmt[0])
    ref = oatt.mla_decode_unabsorbed(f32(qn[rows]), f32(qp[rows]), st["c_hat"], st["kr_hat"], f32(wk),
                                     f32(wv), 512, [w.context] * 3, w.sigma)
    assert_close(out[rows], ref, what=f"mla full {_fid(fmt)}")
    assert c_.device_error() == 0
