"""Shared helpers of the GPU parity tests.

The GPU side goes through the C ABI (``paper_2609_37988_gb300.cache``); the
expected side is computed by ``oracle/`` from the very input tensors the GPU
received (copied to the host).  Nothing the GPU computes is fed back to the
oracle.
"""
from __future__ import annotations

import os

import numpy as np
import torch

from oracle import attention as oatt
from oracle import cache as ocache
from oracle import quant as oquant

# spec tolerance for float outputs against the fp64 oracle
MAX_ABS = 2e-3
REL_L2 = 1e-3


def assert_close(got, ref, max_abs=MAX_ABS, rel_l2=REL_L2, what=""):
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    assert got.shape == ref.shape, (got.shape, ref.shape)
    assert np.isfinite(got).all(), f"{what}: non-finite output"
    err = np.abs(got - ref).max() if got.size else 0.0
    den = np.linalg.norm(ref)
    rel = np.linalg.norm(got - ref) / den if den > 0 else np.linalg.norm(got)
    log = os.environ.get("KVK_PARITY_LOG")
    if log:  # optional record of every comparison's errors (one line each)
        with open(log, "a") as f:
            f.write(f"{what}\t{err:.3e}\t{rel:.3e}\n")
    assert err <= max_abs and rel <= rel_l2, f"{what}: max-abs {err:.3e}, rel-L2 {rel:.3e}"
    return err, rel


def layers_from(w):
    from paper_2609_37988_gb300.cache import Layer
    return [Layer(**a) for a in w.layers]


def f32(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy()


def to_bhtd(x_bthd: np.ndarray) -> np.ndarray:
    """[B, T, H, D] append layout -> [B, H, T, D] oracle layout."""
    return np.ascontiguousarray(np.transpose(x_bthd, (0, 2, 1, 3)))


def oracle_state(k_bthd, v_bthd, lens, cfg):
    """Oracle anchor state from the appended inputs.  Per-channel keys are
    buffered in bf16 by the cache, so fp32 key inputs are rounded to bf16
    first (bf16 inputs are unchanged)."""
    k = to_bhtd(k_bthd)
    if cfg["bits"] != 16 and cfg.get("scheme", "grouped") == "symmetric":
        return ocache.anchor_state(k, to_bhtd(v_bthd), lens, cfg["bits"], scheme="symmetric")
    if cfg["bits"] != 16 and cfg["key_axis"] == "channel":
        k = torch.from_numpy(k).to(torch.bfloat16).float().numpy()
    if cfg["bits"] == 16:
        # bf16 storage of (possibly fp32) inputs
        k = torch.from_numpy(k).to(torch.bfloat16).float().numpy()
        v = torch.from_numpy(to_bhtd(v_bthd)).to(torch.bfloat16).float().numpy()
        return ocache.anchor_state(k, v, lens, 16)
    return ocache.anchor_state(k, to_bhtd(v_bthd), lens, cfg["bits"], cfg["group"], cfg["key_axis"])


def check_codes(exp: dict, st: dict, lens, cfg):
    """Exported GPU state equals the oracle's bit for bit on valid positions."""
    B = len(lens)
    for b in range(B):
        n = int(lens[b])
        if cfg["bits"] == 16:
            k = exp["k"][b, :, :n].float().cpu().numpy()
            np.testing.assert_array_equal(k, st["k_hat"][b, :, :n].astype(np.float32))
            continue
        if cfg.get("scheme", "grouped") == "symmetric":
            for x in ("k", "v"):
                np.testing.assert_array_equal(exp[x + "_codes"][b, :, :n].cpu().numpy(),
                                              st[x + "_codes"][b, :, :n])
                np.testing.assert_array_equal(exp[x + "_scale"][b, :, :n].cpu().numpy(),
                                              st[x + "_scale"][b, :, :n])
            continue
        g = cfg["group"]
        np.testing.assert_array_equal(exp["v_codes"][b, :, :n].cpu().numpy(), st["v_codes"][b, :, :n])
        np.testing.assert_array_equal(exp["v_scale"][b, :, :n].cpu().numpy(), st["v_scale"][b, :, :n])
        np.testing.assert_array_equal(exp["v_zero"][b, :, :n].cpu().numpy(), st["v_zero"][b, :, :n])
        if cfg["key_axis"] == "token":
            np.testing.assert_array_equal(exp["k_codes"][b, :, :n].cpu().numpy(), st["k_codes"][b, :, :n])
            np.testing.assert_array_equal(exp["k_scale"][b, :, :n].cpu().numpy(), st["k_scale"][b, :, :n])
            np.testing.assert_array_equal(exp["k_zero"][b, :, :n].cpu().numpy(), st["k_zero"][b, :, :n])
        else:
            nq = (n // g) * g
            np.testing.assert_array_equal(exp["k_codes"][b, :, :nq].cpu().numpy(), st["k_codes"][b])
            np.testing.assert_array_equal(exp["k_scale"][b, :, : n // g].cpu().numpy(), st["k_scale"][b])
            np.testing.assert_array_equal(exp["k_zero"][b, :, : n // g].cpu().numpy(), st["k_zero"][b])
            res = exp["k_residual"][b].float().cpu().numpy()
            for p in range(nq, n):
                np.testing.assert_array_equal(res[:, p % g], st["k_residual"][b][:, p - nq])


def gqa_expected(q, st, lens, sigma, kept=None):
    return oatt.gqa_decode(f32(q), st["k_hat"], st["v_hat"], lens, sigma, kept)
