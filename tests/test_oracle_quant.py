"""Pins for oracle/quant.py against closed forms, hand-worked cases and
brute force (no GPU).  Each test names the mistake it would catch."""
import numpy as np
import pytest

from oracle import quant

F32 = np.float32


def test_worked_example_two_bits():
    # 4 values spanning 3 steps: scale = 3/3 = 1, zero = 0, codes = values.
    c, s, z = quant.quantise_groups(np.array([0.0, 1.0, 2.0, 3.0], F32), 2)
    assert c.tolist() == [0, 1, 2, 3] and s == F32(1) and z == F32(0)
    # a wrong level count (2^b instead of 2^b - 1) would give scale 0.75


def test_zero_point_is_min_and_codes_unsigned():
    x = np.array([-3.0, -1.0, 1.0, 3.0], F32)
    c, s, z = quant.quantise_groups(x, 2)
    assert z == F32(-3.0) and s == F32(2.0)
    assert c.tolist() == [0, 1, 2, 3]


def test_round_half_to_even():
    # ratio values 0.5, 1.5, 2.5 -> 0, 2, 2 under half-to-even (floor or
    # half-up rounding would differ)
    x = np.array([0.0, 0.5, 1.5, 2.5, 3.0], F32)
    c, s, _ = quant.quantise_groups(x, 2)
    assert s == F32(1.0)
    assert c.tolist() == [0, 0, 2, 2, 3]


def test_constant_group():
    x = np.full(32, 0.375, F32)
    c, s, z = quant.quantise_groups(x, 4)
    assert s == F32(0) and (c == 0).all() and z == F32(0.375)
    xh = quant.dequantise_per_token(c, s[None], z[None], 32)
    assert (xh == 0.375).all()


@pytest.mark.parametrize("bits", [2, 4, 8])
def test_extremes_and_roundtrip(bits):
    rng = np.random.default_rng(bits)
    x = (rng.standard_normal((257, 64)) * rng.lognormal(0, 1, (257, 1))).astype(F32)
    c, s, z = quant.quantise_groups(x, bits)
    lev = (1 << bits) - 1
    assert c.dtype == np.uint8 and c.max() <= lev
    rows = np.arange(x.shape[0])
    assert (c[rows, x.argmin(1)] == 0).all()
    assert (c[rows, x.argmax(1)] == lev).all()
    xh = c.astype(np.float64) * s[:, None] + z[:, None]
    slack = 8 * np.finfo(np.float32).eps * np.abs(x).max(1)
    err = np.abs(xh - x).max(1)
    assert (err <= 0.5 * s.astype(np.float64) + slack).all()


def _brute_group(vals, bits):
    # scalar loop, one float32 op at a time
    lev = F32((1 << bits) - 1)
    mn = F32(min(vals)); mx = F32(max(vals))
    sc = F32(F32(mx - mn) / lev)
    out = []
    for v in vals:
        if sc == 0:
            out.append(0)
            continue
        r = F32(F32(F32(v) - mn) / sc)
        out.append(int(min(max(np.rint(r), 0), lev)))
    return out, sc, mn


def test_per_token_matches_brute_force():
    rng = np.random.default_rng(7)
    x = rng.standard_normal((3, 2, 5, 64)).astype(F32)
    c, s, z = quant.quantise_per_token(x, 4, 32)
    for idx in np.ndindex(3, 2, 5):
        for g in range(2):
            bc, bs, bz = _brute_group(list(x[idx][32 * g:32 * g + 32]), 4)
            assert list(c[idx][32 * g:32 * g + 32]) == bc
            assert s[idx][g] == bs and z[idx][g] == bz


def test_per_channel_matches_brute_force_and_keeps_residual():
    rng = np.random.default_rng(11)
    T, D, g = 77, 8, 32          # two full groups + 13 residual positions
    x = rng.standard_normal((T, D)).astype(F32)
    c, s, z, r = quant.quantise_per_channel(x, 8, g)
    assert c.shape == (64, D) and s.shape == (2, D) and r.shape == (13, D)
    assert (r == x[64:]).all()
    for G in range(2):
        for ch in range(D):
            bc, bs, bz = _brute_group(list(x[G * g:(G + 1) * g, ch]), 8)
            assert list(c[G * g:(G + 1) * g, ch]) == bc
            assert s[G, ch] == bs and z[G, ch] == bz
    xh = quant.dequantise_per_channel(c, s, z, g, r)
    assert xh.shape == x.shape and (xh[64:] == x[64:]).all()


def test_symmetric_two_bits_has_three_levels():
    # Appendix C.3: q = 2^(b-1) - 1; at two bits the codes are {-1, 0, 1}
    rng = np.random.default_rng(3)
    x = rng.standard_normal((100, 128)).astype(F32)
    c, s = quant.quantise_symmetric(x, 2)
    assert set(np.unique(c).tolist()) == {-1, 0, 1}
    c4, s4 = quant.quantise_symmetric(x, 4)
    assert c4.min() >= -7 and c4.max() <= 7
    # the element of largest magnitude maps to +-q exactly
    i = np.abs(x).argmax(1)
    assert (np.abs(c4[np.arange(100), i]) == 7).all()
    err = np.abs(quant.dequantise_symmetric(c4, s4) - x).max(1)
    assert (err <= 0.5 * s4 + 1e-6).all()


def test_round_bf16_matches_torch():
    # the bit-pattern rounding against torch's own float32 -> bfloat16
    # conversion (round to nearest even), on random values, exact ties with
    # an even and an odd kept bit, subnormals and large magnitudes
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(5)
    u = rng.integers(0, 0x7F000000, 20000, dtype=np.uint64).astype(np.uint32)
    ties = (rng.integers(0, 0x7F00, 2000, dtype=np.uint64).astype(np.uint32) << 16) | 0x8000
    sub = rng.integers(1, 0x007FFFFF, 2000, dtype=np.uint64).astype(np.uint32)
    bits = np.concatenate([u, ties, sub])
    x = np.concatenate([bits, bits | 0x80000000]).view(F32)
    ref = torch.from_numpy(x.copy()).to(torch.bfloat16).float().numpy()
    got = quant.round_bf16(x)
    assert (got.view(np.uint32) == ref.view(np.uint32)).all()


def _round_binary(v, p):
    """Nearest binary floating-point value with p significant bits to the
    exact rational v (ties to even), as a Fraction; normal range only."""
    from fractions import Fraction
    if v == 0:
        return Fraction(0)
    sign = -1 if v < 0 else 1
    a = abs(v)
    e = 0
    while a >= 2:
        a /= 2
        e += 1
    while a < 1:
        a *= 2
        e -= 1
    m = a * (1 << (p - 1))                  # in [2^(p-1), 2^p)
    n = round(m)                            # Fraction.__round__: ties to even
    return sign * Fraction(n, 1 << (p - 1)) * (Fraction(2) ** e)


def _brute_symmetric(vals, bits):
    # exact rationals, each binary32 step rounded to 24 bits, the scale to 8
    from fractions import Fraction
    q = (1 << (bits - 1)) - 1
    xs = [Fraction(float(F32(v))) for v in vals]
    amax = max(abs(x) for x in xs)
    if amax == 0:
        return [0] * len(xs), 0.0
    s = _round_binary(_round_binary(amax / q, 24), 8)
    codes = [int(max(-q, min(q, round(_round_binary(x / s, 24))))) for x in xs]
    return codes, float(s)


@pytest.mark.parametrize("bits", [2, 4, 8])
def test_symmetric_brute_force(bits):
    rng = np.random.default_rng(40 + bits)
    for trial in range(40):
        n = int(rng.integers(1, 9))
        x = (rng.standard_normal(n) * 2.0 ** rng.integers(-6, 6)).astype(F32)
        if trial % 5 == 0:
            x = np.round(x * 4) / 4           # dyadic values: exact ties occur
        c, s = quant.quantise_symmetric(x, bits)
        bc, bs = _brute_symmetric(x, bits)
        assert c.tolist() == bc and float(s) == bs, (x, c, s, bc, bs)


def test_symmetric_worked_examples():
    # b = 2 (q = 1): max|x| = 1 gives s = 1, codes rint(x)
    c, s = quant.quantise_symmetric(np.array([1.0, -0.4, 0.6, 0.2], F32), 2)
    assert float(s) == 1.0 and c.tolist() == [1, 0, 1, 0]
    # b = 4 (q = 7), s = 1: rint is half to even (-3.5 -> -4, 2.5 -> 2)
    c, s = quant.quantise_symmetric(np.array([7.0, -3.5, 2.5, 0.49], F32), 4)
    assert float(s) == 1.0 and c.tolist() == [7, -4, 2, 0]
    # b = 4, max|x| = 1: 1/7 stored in bf16 is 0.142578125 (8 significant
    # bits, rounded down), and 0.5 / 0.142578125 = 3.507 -> 4; with the
    # unrounded float32 scale the same element would give 3
    c, s = quant.quantise_symmetric(np.array([1.0, 0.5], F32), 4)
    assert float(s) == 0.142578125 and c.tolist() == [7, 4]
    # a zero vector stores scale 0 and codes 0
    c, s = quant.quantise_symmetric(np.zeros(128, F32), 8)
    assert float(s) == 0.0 and (c == 0).all()


def test_symmetric_anchor_state():
    from oracle import cache as ocache
    rng = np.random.default_rng(9)
    k = rng.standard_normal((2, 3, 10, 128)).astype(F32)
    v = rng.standard_normal((2, 3, 10, 128)).astype(F32)
    lens = [10, 4]
    st = ocache.anchor_state(k, v, lens, 4, scheme="symmetric")
    assert st["k_codes"].dtype == np.int8 and st["k_scale"].shape == (2, 3, 10)
    for b, n in enumerate(lens):
        for x, name in ((k, "k"), (v, "v")):
            err = np.abs(st[name + "_hat"][b, :, :n] - x[b, :, :n]).max(-1)
            assert (err <= 0.5 * st[name + "_scale"][b, :, :n] + 1e-6).all()
            assert (st[name + "_hat"][b, :, n:] == 0).all()


# ---- dequantisers: pinned against scalar loops over (position, channel) ----
# A group index taken as i % n_groups instead of i // g (np.tile for
# np.repeat), a scale/zero swap or a per-channel group indexed by channel
# instead of by position fails these: every group gets its own scale and zero.

@pytest.mark.parametrize("group", [32, 64])
def test_dequantise_per_token_matches_scalar_loop(group):
    rng = np.random.default_rng(100 + group)
    D = 128
    n_g = D // group
    codes = rng.integers(0, 16, (2, 3, D), dtype=np.uint8)
    scale = rng.uniform(0.1, 2.0, (2, 3, n_g)).astype(F32)
    zero = rng.uniform(-3.0, 3.0, (2, 3, n_g)).astype(F32)
    got = quant.dequantise_per_token(codes, scale, zero, group)
    assert got.shape == (2, 3, D) and got.dtype == np.float64
    for idx in np.ndindex(2, 3):
        for i in range(D):
            want = float(codes[idx][i]) * float(scale[idx][i // group]) + float(zero[idx][i // group])
            assert got[idx][i] == want, (idx, i)


@pytest.mark.parametrize("bits,group", [(8, 64), (4, 32), (4, 64), (2, 32)])
def test_per_token_roundtrip_through_dequantiser(bits, group):
    # |x - dequant(quant(x))| <= scale/2 of the element's own group (plus
    # binary32 slack), through the two library functions
    rng = np.random.default_rng(bits * 1000 + group)
    x = (rng.standard_normal((4, 2, 9, 128)) * rng.lognormal(0, 1, (1, 1, 1, 128))).astype(F32)
    c, s, z = quant.quantise_per_token(x, bits, group)
    xh = quant.dequantise_per_token(c, s, z, group)
    slack = 8 * np.finfo(np.float32).eps * np.abs(x).max()
    for i in range(128):
        bound = 0.5 * s[..., i // group].astype(np.float64) + slack
        assert (np.abs(xh[..., i] - x[..., i]) <= bound).all(), i


def test_dequantise_per_channel_matches_scalar_loop():
    rng = np.random.default_rng(12)
    g, nG, D, R = 32, 3, 8, 5
    codes = rng.integers(0, 256, (2, nG * g, D), dtype=np.uint8)
    scale = rng.uniform(0.1, 2.0, (2, nG, D)).astype(F32)
    zero = rng.uniform(-3.0, 3.0, (2, nG, D)).astype(F32)
    resid = rng.standard_normal((2, R, D)).astype(F32)
    got = quant.dequantise_per_channel(codes, scale, zero, g, resid)
    assert got.shape == (2, nG * g + R, D)
    for h in range(2):
        for t in range(nG * g):
            for ch in range(D):
                want = float(codes[h, t, ch]) * float(scale[h, t // g, ch]) + float(zero[h, t // g, ch])
                assert got[h, t, ch] == want, (h, t, ch)
        for t in range(R):
            assert (got[h, nG * g + t] == resid[h, t].astype(np.float64)).all()


@pytest.mark.parametrize("bits", [8, 4])
def test_per_channel_roundtrip_through_dequantiser(bits):
    rng = np.random.default_rng(60 + bits)
    g, T, D = 32, 100, 16          # three full groups + 4 residual positions
    x = (rng.standard_normal((T, D)) * rng.lognormal(0, 1, (1, D))).astype(F32)
    c, s, z, r = quant.quantise_per_channel(x, bits, g)
    xh = quant.dequantise_per_channel(c, s, z, g, r)
    slack = 8 * np.finfo(np.float32).eps * np.abs(x).max()
    for t in range(96):
        bound = 0.5 * s[t // g].astype(np.float64) + slack
        assert (np.abs(xh[t] - x[t]) <= bound).all(), t
    assert (xh[96:] == x[96:]).all()


@pytest.mark.parametrize("bits,group", [(8, 64), (4, 32)])
def test_grouped_per_token_anchor_state_matches_brute_force(bits, group):
    # the anchor state the grouped per-token workloads use, element by
    # element from the scalar quantiser of _brute_group: codes, scales,
    # zeros and x_hat = code * scale + zero, zeros past each length
    from oracle import cache as ocache
    rng = np.random.default_rng(bits + group)
    B, H, T, D = 2, 2, 6, 128
    k = rng.standard_normal((B, H, T, D)).astype(F32)
    v = (rng.standard_normal((B, H, T, D)) * 3.0).astype(F32)
    lens = [6, 3]
    st = ocache.anchor_state(k, v, lens, bits, group)
    for name, x in (("k", k), ("v", v)):
        for b in range(B):
            for h in range(H):
                for t in range(T):
                    for gi in range(D // group):
                        bc, bs, bz = _brute_group(list(x[b, h, t, gi * group:(gi + 1) * group]), bits)
                        assert list(st[name + "_codes"][b, h, t, gi * group:(gi + 1) * group]) == bc
                        assert st[name + "_scale"][b, h, t, gi] == bs
                        assert st[name + "_zero"][b, h, t, gi] == bz
                        for i in range(group):
                            want = float(bc[i]) * float(bs) + float(bz) if t < lens[b] else 0.0
                            assert st[name + "_hat"][b, h, t, gi * group + i] == want
