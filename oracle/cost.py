"""Oracle cost accounting (test infrastructure; see ``oracle/__init__.py``).

* eq. (cost): an inherit action costs 0 bits per token; a cache-producing
  action ``(d, b)`` costs ``(d + d_R) * b``.  For a non-MLA backbone
  ``d = 2 n_kv d_h`` and ``d_R = 0``.
* eq. (compression): ``rho = C0 / sum_l c(a_l)`` with
  ``C0 = L * 2 n_kv d_h * 16`` (the bf16 GQA cache).
* eq. (action space): ``|A| = |D| |B| + 1`` with ``B = {2,4,8,16}`` and
  ``D = {r/8, r/4, r/2, r}``.
* eq. (range): ``rho_min = C0 / (L max_a c)``; ``rho_max = C0 / min_a c``
  with depth (a single anchor) and ``C0 / (L min_a c)`` without.
* Tab. realized_bits: bits per element including quantisation metadata and
  a full-precision residual window.
"""
from __future__ import annotations

import math

BITS = (2, 4, 8, 16)


def c0_bits(L: int, n_kv: int, d_h: int) -> int:
    """C0 of eq. (compression): the uncompressed bf16 GQA plan cost."""
    return L * 2 * n_kv * d_h * 16


def action_cost(action, n_kv: int, d_h: int, mla: bool, d_r: int = 64) -> int:
    """eq. (cost) for one action.

    ``action`` is ``"inherit"`` or a tuple ``(d, b)``; for a non-MLA backbone
    ``d`` is ignored (the layer's width is ``2 n_kv d_h``, no positional key).
    """
    if action == "inherit":
        return 0
    d, b = action
    if not mla:
        return 2 * n_kv * d_h * b
    return (d + d_r) * b


def compression(plan, L: int, n_kv: int, d_h: int, mla: bool, d_r: int = 64) -> float:
    """eq. (compression) for a plan (list of actions, one per layer)."""
    if len(plan) != L:
        raise ValueError("plan length must equal L")
    if plan[0] == "inherit":
        raise ValueError("layer 1 must own a cache")
    total = sum(action_cost(a, n_kv, d_h, mla, d_r) for a in plan)
    return c0_bits(L, n_kv, d_h) / total


def action_space(r: int, bits=BITS, depth=True, rank=True, precision=True):
    """Actions of eq. (action space) restricted to the enabled axes."""
    widths = [r // 8, r // 4, r // 2, r] if rank else [r]
    bs = list(bits) if precision else [16]
    acts = [(d, b) for d in widths for b in bs]
    if depth:
        acts = ["inherit"] + acts
    return acts


def rho_range(L, n_kv, d_h, r, mla, depth, rank, precision, d_r=64):
    """eq. (range): ``(rho_min, rho_max)`` over the enabled axes."""
    acts = [a for a in action_space(r, depth=depth, rank=rank, precision=precision)
            if a != "inherit"]
    costs = [action_cost(a, n_kv, d_h, mla, d_r) for a in acts]
    C0 = c0_bits(L, n_kv, d_h)
    rmin = C0 / (L * max(costs))
    rmax = C0 / min(costs) if depth else C0 / (L * min(costs))
    return rmin, rmax


def plan_count_log10(L: int, n_actions: int) -> float:
    """log10 of the number of plans ``|A|^L`` (Tab. ranges, "Plans")."""
    return L * math.log10(n_actions)


def bits_per_element_symmetric(b: int, row: int = 128, scale_bits: int = 16) -> float:
    """Paper's quantiser: one bf16 scale per ``row``-element token-head row."""
    return b + scale_bits / row


def bits_per_element_grouped(b: int, g: int, meta_bits: int = 32,
                             window: int = 0, context: int = 1,
                             window_bits: int = 16) -> float:
    """Grouped asymmetric quantiser with ``meta_bits`` of scale+zero per group
    of ``g`` and a full-precision window of ``window`` of ``context`` tokens."""
    quant = b + meta_bits / g
    frac = window / context
    return quant * (1.0 - frac) + window_bits * frac


def bytes_per_row_grouped(d_h: int, b: int, g: int, meta_bytes_per_group: int = 8) -> int:
    """Stored bytes of one quantised (token, head) row: codes + fp32 scale and
    zero per group (the layout the library stores)."""
    return d_h * b // 8 + (d_h // g) * meta_bytes_per_group
