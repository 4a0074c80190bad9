"""Acceptance statistics and the speedup model of the paper's evaluation
metrics (Sec. 5.1): average acceptance length tau, the per-position acceptance
rate n-alpha of chain drafts, the expected tokens per verification omega, and
the speedup ratio of Eq. 9.

Host arithmetic on the accepted lengths the step reports (msd_accept_compact /
msd_step write one per request and step); no model computation happens here.
"""
from __future__ import annotations

from typing import Iterable, Sequence


def tau(accept_lengths: Iterable[int]) -> float:
    """Average acceptance length: tokens emitted per drafting-verification
    cycle, i.e. the accepted drafts a plus the token the target adds."""
    a = list(accept_lengths)
    if not a:
        raise ValueError("no steps")
    return sum(x + 1 for x in a) / len(a)


def n_alpha(accept_lengths: Iterable[int], depth: int) -> list:
    """Acceptance rate of the n-th drafted token of a chain draft, n = 1..depth.

    With one draft token per depth, the n-th token is checked by the target
    only when the first n-1 were accepted, so n-alpha = #(a >= n) / #(a >= n-1)
    over the steps (None where no step reached position n)."""
    a = list(accept_lengths)
    out = []
    for n in range(1, depth + 1):
        reached = sum(1 for x in a if x >= n - 1)
        out.append(sum(1 for x in a if x >= n) / reached if reached else None)
    return out


def omega(gamma: int, alpha: float) -> float:
    """Expected tokens per verification step for speculative length gamma and
    acceptance rate alpha: (1 - alpha^(gamma+1)) / (1 - alpha), i.e. the sum
    of alpha^i for i = 0..gamma (gamma + 1 at alpha = 1)."""
    if not 0.0 <= alpha <= 1.0:
        raise ValueError("alpha must lie in [0, 1]")
    if alpha == 1.0:
        return float(gamma + 1)
    return (1.0 - alpha ** (gamma + 1)) / (1.0 - alpha)


def speedup_ratio(n_out: int, t_p: float, t_prof: float, t_cycle: float,
                  tokens_per_cycle: float) -> float:
    """Eq. 9: (N T_p + T_profiling) / (N t_cycle / tokens_per_cycle + T_profiling).

    t_cycle is the time of one drafting-verification cycle (gamma T_q +
    T_v(gamma) in the paper's notation); tokens_per_cycle is omega(gamma,
    alpha), or the measured tau."""
    if tokens_per_cycle <= 0:
        raise ValueError("tokens_per_cycle must be positive")
    return (n_out * t_p + t_prof) / (n_out * t_cycle / tokens_per_cycle + t_prof)


def acceptance_rate(accept_lengths: Iterable[int], gamma: int) -> float | None:
    """Acceptance rate alpha: accepted draft tokens over the draft tokens the
    target checked. A chain of gamma drafts is checked up to its first
    rejection: a accepted, plus the rejected one when a < gamma."""
    a = list(accept_lengths)
    checked = sum(x + (1 if x < gamma else 0) for x in a)
    return sum(a) / checked if checked else None
