"""Byte accounting for one decode step (host-side arithmetic only).

Two models:

* :func:`paper_read_budget` -- the paper's three-term per-token read budget (Eq. 2):
  attended rows, the index scan and admitted rows, in bytes per cached token.
* :func:`step_bytes` -- the algorithmic HBM bytes the decode step of this library must move, which the
  roofline is quoted against: the width-r score read of every cached row, plus every distinct attended row
  once (the union over heads of the selected sets), plus, in two-tier mode, the trigger's second scan of the
  archive (score columns + eta) and the fired rows not already gathered. Workspace traffic (candidate lists,
  bitmaps, split partials) is overhead and is not counted.
"""
from __future__ import annotations

D_LATENT, D_ROPE = 512, 64
ROW_DIMS = D_LATENT + D_ROPE


def paper_read_budget(rho: float, r_sk: int, f: float, index_bytes: int = 2, row_bytes: int = 2) -> float:
    """Eq. 2 in bytes/token: rho*576 attended dims + (1-rho)(64 + r_sk + 1) index dims + f*576 admitted dims.

    Attended and admitted dims are cache rows (``row_bytes`` per dim); index dims are ``index_bytes`` each.
    """
    return (rho * ROW_DIMS * row_bytes + (1.0 - rho) * (D_ROPE + r_sk + 1) * index_bytes
            + f * ROW_DIMS * row_bytes)


def row_bytes(dtype: str) -> int:
    return ROW_DIMS * (2 if dtype == "bf16" else 4)


def score_bytes_per_row(r: int, dtype: str) -> int:
    """Bytes of one cached row the scoring pass reads: the 64 RoPE columns, or the bf16 width-r digest."""
    if r == D_ROPE:
        return D_ROPE * (2 if dtype == "bf16" else 4)
    return 2 * r


def step_bytes(N: int, B: int, r: int, dtype: str, union_rows: int, trigger: bool = False,
               fired_new_rows: int = 0, r_sk: int = 0) -> int:
    """Algorithmic bytes of one decode step over B sequences of N cached rows.

    union_rows: total distinct rows gathered by tier-1 attention, summed over the batch.
    fired_new_rows: total fired rows not already in the tier-1 union, summed over the batch.
    r_sk: the trigger scan also reads each row's bf16 content sketch (2 r_sk bytes).
    """
    total = B * N * score_bytes_per_row(r, dtype) + union_rows * row_bytes(dtype)
    if trigger:
        total += B * N * (score_bytes_per_row(r, dtype) + 4 + 2 * r_sk) + fired_new_rows * row_bytes(dtype)
    return int(total)


def expected_union_fraction(N: int, H: int, k: int, window: int, n_sink: int = 0) -> float:
    """|U|/N for iid per-head selections: archive rows kept by at least one head, plus window and sinks."""
    A = max(0, N - window - n_sink)
    if A == 0:
        return min(1.0, (window + n_sink) / max(N, 1))
    p_none = (1.0 - k / A) ** H
    return ((1.0 - p_none) * A + window + n_sink) / N
