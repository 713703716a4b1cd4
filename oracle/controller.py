"""DLFP controller restated from the paper — TEST INFRASTRUCTURE ONLY.

§3.1 Eq. 2: after a guarded cycle with observed latency L_hat, the next
prefill cap is c_{t+1} = clamp(floor_128(c_t * T / L_hat), c_min, c_max).
§3.1 (activation/reset): the cap applies only when at least one request is
decoding and a prefill shares the cycle; with no decoder active the cap resets
to c_initial and an isolated prefill is not capped.
§3.1 (parameters): T = 80 ms, c_initial = 3072, c_min = 1024, c_max = 6144,
128-token quantum.

Reading where the paper is silent: floor_128(x) = 128 * floor(x / 128),
applied before the clamp, and the multiplier acts on the cap c_t (not on the
tokens actually prefilled), as Eq. 2 is written.
"""
from __future__ import annotations

import math

PAPER_T_MS = 80.0
PAPER_C_INIT = 3072
PAPER_C_MIN = 1024
PAPER_C_MAX = 6144
PAPER_QUANTUM = 128


def floor_q(x: float, quantum: int = PAPER_QUANTUM) -> int:
    """floor_128 of Eq. 2: the largest multiple of the quantum not above x."""
    return quantum * math.floor(x / quantum)


def eq2_next_cap(c_t: int, target: float, observed: float,
                 c_min: int = PAPER_C_MIN, c_max: int = PAPER_C_MAX,
                 quantum: int = PAPER_QUANTUM) -> int:
    """Eq. 2 exactly as printed: clamp(floor_128(c_t * T / L_hat), c_min, c_max)."""
    if observed <= 0:
        raise ValueError("observed latency must be positive")
    return min(max(floor_q(c_t * target / observed, quantum), c_min), c_max)


def cycle(c_t: int, n_decoding: int, prefill_pending: bool, observed: float | None,
          target: float = PAPER_T_MS, c_init: int = PAPER_C_INIT,
          c_min: int = PAPER_C_MIN, c_max: int = PAPER_C_MAX):
    """One scheduling cycle of the §3.1 policy.

    Returns (cap_applied_this_cycle or None for "uncapped", next c).  A cycle
    is guarded when a decoder is active and a prefill shares it; only a
    guarded cycle's observation updates the cap.  No decoder: reset to c_init.
    """
    if n_decoding == 0:
        return None, c_init
    if not prefill_pending:
        return None, c_t
    cap = c_t
    if observed is None:
        return cap, c_t
    return cap, eq2_next_cap(c_t, target, observed, c_min, c_max)
