"""Pins of the acceptance rule and the round bookkeeping (Section 3, steps 4-5; Appendix A.1).

Brute force over a 3-token vocabulary against a definition written a different way
(prefix-of-sequence equality), plus the budget stop rule.
"""
import itertools

import numpy as np

import oracle
from oracle import accept_length


def _naive_accept(draft, verify):
    # the accepted prefix is the longest k with (d_1..d_k) == (v_0..v_{k-1})
    best = 0
    for k in range(len(draft) + 1):
        if tuple(draft[:k]) == tuple(verify[:k]):
            best = k
    return best


def test_accept_bruteforce_v3_d3():
    V, D = 3, 3
    count = 0
    for draft in itertools.product(range(V), repeat=D):
        for verify in itertools.product(range(V), repeat=D + 1):
            assert accept_length(draft, verify) == _naive_accept(draft, verify)
            count += 1
    assert count == 27 * 81


def test_accept_edges():
    assert accept_length([], [5]) == 0
    assert accept_length([1, 2, 3], [1, 2, 3, 9]) == 3
    assert accept_length([1, 2, 3], [0, 2, 3, 9]) == 0
    assert accept_length([1, 2, 3], [1, 0, 3, 9]) == 1
    # a later match after a mismatch is never accepted
    assert accept_length([7, 8, 9, 10], [7, 1, 9, 10, 11]) == 1


def test_budget_stop_truncates_last_round(tiny):
    """Generation stops only at the budget; the last round is cut to max_new tokens."""
    m, prompt = tiny["model"], tiny["prompt"][:24]
    D = 4
    for max_new in (1, 2, 5, 6, 7, 11):
        forced = [D] * 64  # every round emits D+1 tokens
        out, rounds = oracle.spec_generate(m, prompt, max_new, D, forced_n=forced)
        assert len(out) == max_new
        assert sum(len(r["emitted"]) for r in rounds) == max_new - 1
        for r in rounds[:-1]:
            assert len(r["emitted"]) == r["n"] + 1


def test_round_emits_accepted_plus_bonus(tiny):
    """A round appends d_1..d_n and the verifier's v_n: A = n + 1 tokens."""
    m, prompt = tiny["model"], tiny["prompt"][:32]
    out, rounds = oracle.spec_generate(m, prompt, 40, 8)
    for r in rounds[:-1]:
        n = r["n"]
        assert r["emitted"] == r["draft"][:n] + [r["verify"][n]]
        assert r["n"] == accept_length(r["draft"], r["verify"])
    Ls = [r["L"] for r in rounds]
    for a, b, r in zip(Ls, Ls[1:], rounds):
        assert b - a == r["n"] + 1
