"""Cost-model arithmetic of the paper (test infrastructure).

Section 3 states the usefulness condition of speculation: (C_d + C_v) / A must be
smaller than the cost of producing A tokens with the target model alone.
Appendix A.7 (Table 4) applies it as a draft-cost oracle: with measured iteration
time T0 and draft-side cost share rho_d, removing a fraction r of the draft cost
gives T(r) = T0 (1 - r rho_d), predicted throughput A / T(r), and the accepted
length needed to reach a competitor of throughput X is X * T(r).
"""
from __future__ import annotations

from typing import Dict, List, Sequence


def iteration_time(T0: float, rho_d: float, r: float) -> float:
    """T(r) = T0 (1 - r rho_d)  (Appendix A.7)."""
    return T0 * (1.0 - r * rho_d)


def predicted_tokens_per_s(A: float, T0: float, rho_d: float, r: float) -> float:
    """Throughput after removing a fraction r of the draft cost, acceptance held fixed."""
    return A / iteration_time(T0, rho_d, r)


def break_even_accept(t_draft: float, t_verify: float, t_target_step: float) -> float:
    """Accepted tokens per round at which (C_d + C_v)/A equals the target-only cost per token (Section 3)."""
    return (t_draft + t_verify) / t_target_step


def draft_cost_table(A: float, T0: float, rho_d: float, competitors: Dict[str, float],
                     reductions: Sequence[float] = (0.0, 0.25, 0.5, 0.75, 0.9, 1.0)) -> List[dict]:
    """Rows of the draft-cost oracle: r, predicted tok/s, and needed A per competitor."""
    rows = []
    for r in reductions:
        T = iteration_time(T0, rho_d, r)
        row = {"r": r, "tok_s": A / T}
        for name, tput in competitors.items():
            row["need_" + name] = tput * T
        rows.append(row)
    return rows
