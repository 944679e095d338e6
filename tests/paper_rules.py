"""The hierarchical visibility mask built literally from the paper's index sets.

Independent of the oracle: it never looks at per-token roles.  It takes a
dialogue recipe, forms the sets I_sys, B_i, N_i, Q_curr of Sec. 3.1 (Eq. 1)
and applies the three rules of Sec. 3.2 one after another to an explicit
L x L additive matrix:

1. Basic causal rule (Eq. 3), applied to every pair: M[p, q] = -inf for q > p.
2. Historical body removal (Eq. 4): for every position p after the last Nexus
   token of segment i, M[p, q] = -inf for q in B_i.  A segment with no Nexus
   token is treated as ending at its last body token.
3. Bidirectional Nexus visibility (Eq. 5): M[a, b] = 0 for a in N_i,
   b in N_j, for all segments i, j (``causal_segments`` keeps only j <= i).
"""
from __future__ import annotations

import numpy as np


def index_sets(d):
    t = 0
    sys_idx = list(range(t, t + d.sys_len))
    t += d.sys_len
    bodies, nexus = [], []
    for b, k in d.segments:
        bodies.append(list(range(t, t + b)))
        t += b
        nexus.append(list(range(t, t + k)))
        t += k
    curr = list(range(t, t + d.curr_len))
    return sys_idx, bodies, nexus, curr


def rule_mask(d, causal_segments: bool = False) -> np.ndarray:
    L = d.length
    M = np.zeros((L, L))
    # Rule 1 (Eq. 3): causal everywhere.
    M[np.triu_indices(L, k=1)] = -np.inf
    _, bodies, nexus, _ = index_sets(d)
    # Rule 2 (Eq. 4): body of segment i hidden after max(N_i).
    for Bi, Ni in zip(bodies, nexus):
        end = max(Ni) if Ni else (max(Bi) if Bi else None)
        if end is None:
            continue
        for p in range(end + 1, L):
            for q in Bi:
                M[p, q] = -np.inf
    # Rule 3 (Eq. 5): Nexus tokens see each other, within and across segments.
    for i, Ni in enumerate(nexus):
        for j, Nj in enumerate(nexus):
            if causal_segments and j > i:
                continue
            for a in Ni:
                for b in Nj:
                    M[a, b] = 0.0
    return M


def retained_positions(d) -> list:
    """Positions of I_sys, every N_i and Q_curr in S_aug, in order (the
    effective context of App. C)."""
    s, _, nexus, c = index_sets(d)
    out = list(s)
    for Ni in nexus:
        out.extend(Ni)
    out.extend(c)
    return out
