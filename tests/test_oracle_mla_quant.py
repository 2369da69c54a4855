"""Pins for the quantised MLA anchor state (oracle/cache.py
mla_anchor_state): the kept latent and the positional key of each position
are each one quantised vector (Appendix C.2 truncation composed with the
quantisers of Appendix C.3).  Checked against the scalar quantisers of
test_oracle_quant, round trips within half a step, and the absorbed decode
with the scales factored out of both products against the unabsorbed oracle
decode on the dequantised cache."""
import numpy as np
import pytest

from oracle import attention, cache
from test_oracle_quant import _brute_group, _brute_symmetric

F32 = np.float32
CASES = [("symmetric", 8), ("symmetric", 4), ("symmetric", 2), ("grouped", 8), ("grouped", 4)]


def _inputs(seed, B=2, T=5, r=16, dR=4):
    rng = np.random.default_rng(seed)
    decay = 1.0 / np.sqrt(np.arange(r) + 1.0)
    c = (rng.standard_normal((B, T, r)) * decay).astype(F32)
    kr = rng.standard_normal((B, T, dR)).astype(F32)
    return c, kr


@pytest.mark.parametrize("scheme,bits", CASES)
def test_state_matches_scalar_quantisers(scheme, bits):
    c, kr = _inputs(bits)
    width, lens = 8, [5, 3]
    st = cache.mla_anchor_state(c, kr, lens, width, bits, scheme)
    for b in range(2):
        for t in range(5):
            for name, row in (("c", c[b, t, :width]), ("kr", kr[b, t])):
                if scheme == "symmetric":
                    codes, sc = _brute_symmetric(list(row), bits)
                    assert st[name + "_codes"][b, t].tolist() == codes
                    assert float(st[name + "_scale"][b, t]) == sc
                    want = [float(k) * sc for k in codes]
                else:
                    codes, sc, z = _brute_group(list(row), bits)
                    assert st[name + "_codes"][b, t].tolist() == codes
                    assert st[name + "_scale"][b, t] == sc and st[name + "_zero"][b, t] == z
                    want = [float(k) * float(sc) + float(z) for k in codes]
                got = st[name + "_hat"][b, t]
                assert got.tolist() == (want if t < lens[b] else [0.0] * len(want))
    # only the first `width` latent coordinates are stored
    c2 = c.copy()
    c2[..., width:] = 123.0
    st2 = cache.mla_anchor_state(c2, kr, lens, width, bits, scheme)
    assert np.array_equal(st2["c_hat"], st["c_hat"])


@pytest.mark.parametrize("scheme,bits", CASES)
def test_round_trip_within_half_a_step(scheme, bits):
    c, kr = _inputs(20 + bits, B=3, T=40, r=64, dR=16)
    st = cache.mla_anchor_state(c, kr, [40, 40, 40], 32, bits, scheme)
    for name, x in (("c", c[:, :, :32]), ("kr", kr)):
        s = st[name + "_scale"].astype(np.float64)
        err = np.abs(st[name + "_hat"] - x).max(-1)
        assert (err <= 0.5 * s + 1e-6 * np.abs(x).max()).all()


@pytest.mark.parametrize("scheme,bits", CASES)
def test_absorbed_with_factored_scales_equals_unabsorbed(scheme, bits):
    # the form a kernel can use: codes in both products, each position's
    # scales (and zeros) applied to its score and to its value weight
    rng = np.random.default_rng(7 + bits)
    B, T, H, Dn, dR, r, width = 2, 9, 3, 6, 4, 16, 8
    c, kr = _inputs(bits, B, T, r, dR)
    q_nope = rng.standard_normal((B, H, Dn))
    q_pe = rng.standard_normal((B, H, dR))
    w_uk = rng.standard_normal((H, Dn, r)) / 4
    w_uv = rng.standard_normal((H, Dn, r)) / 4
    lens, sigma = [9, 4], 0.3
    st = cache.mla_anchor_state(c, kr, lens, width, bits, scheme)
    ref = attention.mla_decode_unabsorbed(q_nope, q_pe, st["c_hat"], st["kr_hat"], w_uk, w_uv,
                                          width, lens, sigma)
    got = np.zeros_like(ref)
    for b in range(B):
        n = lens[b]
        cc = st["c_codes"][b, :n].astype(np.float64)
        rc = st["kr_codes"][b, :n].astype(np.float64)
        sc, sr = st["c_scale"][b, :n].astype(np.float64), st["kr_scale"][b, :n].astype(np.float64)
        zc = st["c_zero"][b, :n].astype(np.float64) if scheme == "grouped" else np.zeros(n)
        zr = st["kr_zero"][b, :n].astype(np.float64) if scheme == "grouped" else np.zeros(n)
        for h in range(H):
            q_lat = w_uk[h, :, :width].T @ q_nope[b, h]
            s = sigma * (sc * (cc @ q_lat) + zc * q_lat.sum() + sr * (rc @ q_pe[b, h]) + zr * q_pe[b, h].sum())
            p = np.exp(s - s.max())
            o_lat = ((p * sc) @ cc + (p * zc).sum()) / p.sum()
            got[b, h] = w_uv[h, :, :width] @ o_lat
    np.testing.assert_allclose(got, ref, rtol=1e-10, atol=1e-12)


def test_full_precision_stores_the_inputs():
    c, kr = _inputs(3)
    st = cache.mla_anchor_state(c, kr, [5, 2], 8, 16)
    assert np.array_equal(st["c_hat"][0], c[0, :, :8].astype(np.float64))
    assert (st["kr_hat"][1, 2:] == 0).all()
