"""Token-budget helpers for progressive pruning schedules (host logic).

Sec. 5.1.2, Eq. 24: AvgTokens = (1/N) sum_i T_i over the N LLM layers, where
T_i is the number of visual tokens layer i sees.  With pruning after layers
P = (p_1 < p_2 < ...), layers 1..p_1 see all N_V tokens, layers p_1+1..p_2
see the first stage's budget, and so on.
"""
from __future__ import annotations

from fractions import Fraction
from typing import Sequence


def tokens_per_layer(n_layers: int, n_visual: int, prune_after: Sequence[int],
                     keep: Sequence[int]):
    """T_i for i = 1..n_layers (Eq. 24's summands)."""
    if len(prune_after) != len(keep):
        raise ValueError("one budget per pruning layer")
    if list(prune_after) != sorted(prune_after) or (prune_after and
                                                    not 0 < prune_after[0] <= prune_after[-1] < n_layers):
        raise ValueError("pruning layers must be increasing and inside the model")
    out = []
    for i in range(1, n_layers + 1):
        t = n_visual
        for p, k in zip(prune_after, keep):
            if i > p:
                t = k
        out.append(t)
    return out


def avg_tokens(n_layers: int, n_visual: int, prune_after: Sequence[int],
               keep: Sequence[int]) -> Fraction:
    """Eq. 24, exactly (as a fraction)."""
    return Fraction(sum(tokens_per_layer(n_layers, n_visual, prune_after, keep)), n_layers)
