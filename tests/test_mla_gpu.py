"""GPU parity of the MLA path (truncate on write, absorbed latent decode,
up-projection) against the oracle's unabsorbed MLA (Appendix C.2)."""
import math

import numpy as np
import pytest
import torch

from _parity import assert_close, f32
from oracle import attention as oatt

pytestmark = pytest.mark.gpu


def _mla_cache(B, T, widths, r=512, H=16, max_splits=16):
    from paper_2609_37988_gb300.cache import Cache, Layer
    return Cache(kind="mla", n_layers=len(widths), n_q_heads=H, head_dim=128, latent_dim=r,
                 rope_dim=64, max_batch=B, max_ctx=T,
                 layers=[Layer(inherit=(w == 0), bits=16, width=w) for w in widths],
                 max_splits=max_splits)


def _inputs(B, n, r, seed):
    g = torch.Generator().manual_seed(seed)
    decay = torch.arange(r).add(1.0).rsqrt()
    c = (torch.randn((B, n, r), generator=g) * decay).to(torch.bfloat16)
    kr = torch.randn((B, n, 64), generator=g).to(torch.bfloat16)
    return c, kr


def _weights(H, r, seed):
    g = torch.Generator().manual_seed(seed)
    wk = (torch.randn((H, 128, r), generator=g) / math.sqrt(512)).to(torch.bfloat16)
    wv = (torch.randn((H, 128, r), generator=g) / math.sqrt(512)).to(torch.bfloat16)
    return wk, wv


@pytest.mark.parametrize("width", [512, 256, 128, 64])
def test_mla_decode_parity(width):
    B, r, H = 3, 512, 16
    lens = np.array([300, 65, 1])
    c_ = _mla_cache(B, 320, [width])
    c, kr = _inputs(B, 300, r, width)
    c_.append(0, c.cuda(), kr.cuda(), n_per_seq=torch.tensor(lens, dtype=torch.int32, device="cuda"))
    ex = c_.export(0)
    for b in range(B):   # truncate on write: the first `width` coordinates, bit for bit
        assert torch.equal(ex["c"][b, :lens[b]].cpu(), c[b, :lens[b], :width])
        assert torch.equal(ex["k_r"][b, :lens[b]].cpu(), kr[b, :lens[b]])
    wk, wv = _weights(H, r, 7)
    g = torch.Generator().manual_seed(11)
    qn = torch.randn((B, H, 128), generator=g).to(torch.bfloat16)
    qp = torch.randn((B, H, 64), generator=g).to(torch.bfloat16)
    sigma = 1.0 / math.sqrt(128 + 64)
    ref = oatt.mla_decode_unabsorbed(f32(qn), f32(qp), f32(c), f32(kr), f32(wk), f32(wv), width,
                                     lens, sigma)
    for ns in (0, 1, 4):
        out = c_.decode_mla(0, qn.cuda(), qp.cuda(), wk.cuda(), wv.cuda(), sigma, n_splits=ns)
        assert_close(f32(out), ref, what=f"mla d={width} splits={ns}")


def test_mla_depth_sharing_and_batch_over_64():
    # 70 sequences: the absorb / up-projection loop over 64-row blocks
    B, r, H = 70, 512, 16
    c_ = _mla_cache(B, 128, [256, 0])
    c, kr = _inputs(B, 100, r, 3)
    c_.append(0, c.cuda(), kr.cuda())
    wk, wv = _weights(H, r, 9)
    qn = torch.randn((B, H, 128)).to(torch.bfloat16)
    qp = torch.randn((B, H, 64)).to(torch.bfloat16)
    sigma = 1.0 / math.sqrt(192)
    a = c_.decode_mla(0, qn.cuda(), qp.cuda(), wk.cuda(), wv.cuda(), sigma, n_splits=2)
    b = c_.decode_mla(1, qn.cuda(), qp.cuda(), wk.cuda(), wv.cuda(), sigma, n_splits=2)
    assert torch.equal(a, b)
    sel = [0, 63, 64, 69]
    ref = oatt.mla_decode_unabsorbed(f32(qn[sel]), f32(qp[sel]), f32(c[sel]), f32(kr[sel]), f32(wk),
                                     f32(wv), 256, [100] * 4, sigma)
    assert_close(f32(a[sel]), ref, what="mla B=70")


@pytest.mark.parametrize("width", [512, 64])
def test_mla_fewer_heads_empty_sequence_many_splits(width):
    """H < 16 (padded head rows of the tensor-core operands), a sequence with
    no positions (its output is 0), a 1-position sequence, and more splits
    than tiles (empty splits merge away)."""
    B, r, H = 3, 512, 5
    lens = np.array([0, 1, 200])
    c_ = _mla_cache(B, 256, [width], H=H, max_splits=16)
    c, kr = _inputs(B, 200, r, 40 + width)
    c_.append(0, c.cuda(), kr.cuda(), n_per_seq=torch.tensor(lens, dtype=torch.int32, device="cuda"))
    wk, wv = _weights(H, r, 13)
    g = torch.Generator().manual_seed(17)
    qn = torch.randn((B, H, 128), generator=g).to(torch.bfloat16)
    qp = torch.randn((B, H, 64), generator=g).to(torch.bfloat16)
    sigma = 1.0 / math.sqrt(128 + 64)
    sel = [1, 2]
    ref = oatt.mla_decode_unabsorbed(f32(qn[sel]), f32(qp[sel]), f32(c[sel]), f32(kr[sel]), f32(wk),
                                     f32(wv), width, lens[sel], sigma)
    for ns in (0, 7, 16):
        out = c_.decode_mla(0, qn.cuda(), qp.cuda(), wk.cuda(), wv.cuda(), sigma, n_splits=ns)
        assert torch.isfinite(out).all()
        assert (out[0] == 0).all()
        assert_close(f32(out[sel]), ref, what=f"mla H=5 d={width} splits={ns}")
    assert c_.device_error() == 0
