"""Generic Dempster-Shafer evidence theory over a finite frame (Sec. 3.2).

Test infrastructure only: a brute-force enumeration of focal sets, written
from the set-theoretic definitions (Eqs. 2-7) without any knowledge of the
three-state closed forms in Sec. 4.2, so that it can pin them.

A mass function is a dict {frozenset: mass}.
"""
from __future__ import annotations

from itertools import product
from typing import Dict, FrozenSet, Hashable

Mass = Dict[FrozenSet[Hashable], float]


def check_axioms(m: Mass, tol: float = 1e-12) -> bool:
    """Eq. 2: m(empty) = 0, masses non-negative and summing to 1."""
    if m.get(frozenset(), 0.0) != 0.0:
        return False
    if any(v < -tol for v in m.values()):
        return False
    return abs(sum(m.values()) - 1.0) <= tol


def conflict(m1: Mass, m2: Mass) -> float:
    """Eq. 3: K = sum over B, C with B n C = empty of m1(B) m2(C)."""
    return sum(v1 * v2 for (B, v1), (C, v2) in product(m1.items(), m2.items())
               if not (B & C))


def combine(m1: Mass, m2: Mass) -> Mass:
    """Eq. 4: m(A) = sum_{B n C = A} m1(B) m2(C) / (1 - K) for A != empty."""
    K = conflict(m1, m2)
    out: Mass = {}
    for (B, v1), (C, v2) in product(m1.items(), m2.items()):
        A = B & C
        if A:
            out[A] = out.get(A, 0.0) + v1 * v2
    return {A: v / (1.0 - K) for A, v in out.items()}


def belief(m: Mass, A: FrozenSet[Hashable]) -> float:
    """Eq. 6: Bel(A) = sum_{B subset of A} m(B)."""
    return sum(v for B, v in m.items() if B and B <= A)


def plausibility(m: Mass, A: FrozenSet[Hashable]) -> float:
    """Eq. 7: Pl(A) = sum_{B n A != empty} m(B)."""
    return sum(v for B, v in m.items() if B & A)
