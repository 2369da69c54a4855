"""GPU parity of MLA causal chunk attention (pre-fill) over the latent cache,
bf16 and quantised, through the C ABI: every query row of the chunk attends
to its own causal prefix with the absorbed query (the decode path per row),
against the oracle's unabsorbed chunk attention on the dequantised cache.
Ragged lengths, one sequence shorter than the chunk, an inheriting layer;
bf16 chunks of an even number of rows decode two rows per CTA at d >= 256
(a pair may hold an empty row beside a one-position row), odd ones one."""
import math

import numpy as np
import pytest
import torch

from _parity import assert_close, f32
from oracle import attention as oatt
from oracle import cache as ocache

pytestmark = pytest.mark.gpu

H = 16


def _setup(width, fmt, lens, T, seed, H=H):
    from paper_2609_37988_gb300.cache import Cache, Layer
    B = len(lens)
    layer = dict(bits=16, width=width) if fmt is None else dict(bits=fmt[1], scheme=fmt[0], width=width)
    c = Cache(kind="mla", n_layers=2, n_q_heads=H, head_dim=128, latent_dim=512, rope_dim=64,
              max_batch=B, max_ctx=T, layers=[Layer(**layer), Layer(inherit=True)], max_splits=16)
    g = torch.Generator().manual_seed(seed)
    decay = torch.arange(512).add(1.0).rsqrt()
    n = max(lens)
    cl = (torch.randn((B, n, 512), generator=g) * decay).to(torch.bfloat16)
    kr = torch.randn((B, n, 64), generator=g).to(torch.bfloat16)
    c.append(0, cl.cuda(), kr.cuda(), n_per_seq=torch.tensor(lens, dtype=torch.int32, device="cuda"))
    wk = (torch.randn((H, 128, 512), generator=g) / math.sqrt(512)).to(torch.bfloat16)
    wv = (torch.randn((H, 128, 512), generator=g) / math.sqrt(512)).to(torch.bfloat16)
    if fmt is None:
        c_hat, kr_hat = f32(cl), f32(kr)
    else:
        st = ocache.mla_anchor_state(f32(cl), f32(kr), lens, width, fmt[1], fmt[0])
        c_hat, kr_hat = st["c_hat"], st["kr_hat"]
    return c, wk, wv, c_hat, kr_hat


@pytest.mark.parametrize("width,fmt", [(512, None), (64, None), (256, ("grouped", 8)),
                                       (128, ("symmetric", 4)), (512, ("symmetric", 2))],
                         ids=["bf16-d512", "bf16-d64", "g8-d256", "sym4-d128", "sym2-d512"])
def test_mla_prefill_parity(width, fmt):
    lens, n_q = [300, 129, 20], 40
    c, wk, wv, c_hat, kr_hat = _setup(width, fmt, lens, 320, seed=width + (fmt[1] if fmt else 16))
    g = torch.Generator().manual_seed(5)
    qn = torch.randn((len(lens), n_q, H, 128), generator=g).to(torch.bfloat16)
    qp = torch.randn((len(lens), n_q, H, 64), generator=g).to(torch.bfloat16)
    sigma = 1.0 / math.sqrt(192)
    out = c.prefill_mla(0, qn.cuda(), qp.cuda(), wk.cuda(), wv.cuda(), sigma)
    ref = oatt.mla_prefill_unabsorbed(f32(qn), f32(qp), c_hat, kr_hat, f32(wk), f32(wv), width, lens, sigma)
    assert_close(f32(out), ref, what=f"mla prefill d={width} {fmt}")
    # queries before position 0 give zeros; the inheritor reads the anchor
    assert (f32(out[2, : n_q - lens[2]]) == 0).all()
    again = c.prefill_mla(1, qn.cuda(), qp.cuda(), wk.cuda(), wv.cuda(), sigma)
    assert torch.equal(out, again)
    # the last query of each sequence is one decode step
    dec = c.decode_mla(0, qn[:, -1].contiguous().cuda(), qp[:, -1].contiguous().cuda(), wk.cuda(),
                       wv.cuda(), sigma)
    assert_close(f32(out[:, -1]), f32(dec), max_abs=2e-4, rel_l2=1e-4, what="last query = decode")
    assert c.device_error() == 0


def test_mla_prefill_rejections():
    from paper_2609_37988_gb300._lib import KVKError
    c, wk, wv, _, _ = _setup(64, None, [10, 10], 64, seed=1)
    qn = torch.zeros((2, 4, H, 128), dtype=torch.bfloat16, device="cuda")
    qp = torch.zeros((2, 4, H, 64), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(KVKError):
        c.prefill_mla(0, qn, qp, wk.cuda(), wv.cuda(), 0.0)  # scale
    with pytest.raises(KVKError):
        c.prefill_mla(0, torch.zeros((2, 65, H, 128), dtype=torch.bfloat16, device="cuda"),
                      torch.zeros((2, 65, H, 64), dtype=torch.bfloat16, device="cuda"), wk.cuda(),
                      wv.cuda(), 0.1)  # n_q > max_ctx


@pytest.mark.parametrize("width,n_q,heads", [(512, 40, 10), (512, 39, 16), (256, 40, 5), (256, 2, 16),
                                              (128, 40, 16)],
                         ids=["d512-pairs-h10", "d512-odd-rows", "d256-pairs-h5", "d256-one-pair", "d128-rows"])
def test_mla_prefill_row_pairs(width, n_q, heads):
    """Two rows per CTA: each row masks its own causal end inside the shared
    tiles; fewer than 16 heads; an odd row count keeps one row per CTA."""
    lens = [301, 130, 21]
    c, wk, wv, c_hat, kr_hat = _setup(width, None, lens, 320, seed=width + n_q, H=heads)
    g = torch.Generator().manual_seed(6)
    qn = torch.randn((len(lens), n_q, heads, 128), generator=g).to(torch.bfloat16)
    qp = torch.randn((len(lens), n_q, heads, 64), generator=g).to(torch.bfloat16)
    sigma = 1.0 / math.sqrt(192)
    out = c.prefill_mla(0, qn.cuda(), qp.cuda(), wk.cuda(), wv.cuda(), sigma)
    ref = oatt.mla_prefill_unabsorbed(f32(qn), f32(qp), c_hat, kr_hat, f32(wk), f32(wv), width, lens, sigma)
    assert_close(f32(out), ref, what=f"mla prefill pairs d={width} n_q={n_q} H={heads}")
    empty = max(0, n_q - lens[2])
    assert (f32(out[2, :empty]) == 0).all()
    if empty < n_q:
        assert (np.abs(f32(out[2, empty])) > 0).any()  # the one-position row
    assert c.device_error() == 0
