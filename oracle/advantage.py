"""Oracle for TreePO's tree-based advantage (Sec. 2.3, Eq. tree_ae).

TEST INFRASTRUCTURE ONLY: imported by ``tests/`` and ``bench.py``'s CPU legs,
never by the product library.

The definition, written out in fp64 with plain loops. Trajectory i ends at
leaf node l_i with reward R_i. Its sub-groups are those of its predecessors
at depths 0 .. J_i - 1 (the root query, then each segment node above the
leaf; Eq. groups and the worked figure of Sec. 2.3): G_x = every trajectory
whose path passes through x. Then

    A_{i,j} = R_i - mean_{G_j} R                  (sub-group advantage)
    A_i     = (1 / |J_i|) sum_j A_{i,j}           (mean pooling)
    adv_i   = A_i / std(A)                        (global normalisation)

Readings where the equation is garbled or silent: std is the population
standard deviation of A over every accepted trajectory of the batch (the
"global variance normalisation" of REINFORCE++ named beside the equation); a
query whose rewards all agree (std(R) = 0, the equation's side condition) is
rejected -- its trajectories get 0 and stay out of the std; adv is 0 when
std(A) = 0; a leaf that is itself a root has no sub-group and is rejected.

Pinned by ``tests/test_oracle_rollout.py``: a hand-computed 8-leaf binary
tree (the shape of the paper's figure), the flat tree where it reduces to
GRPO's R - mean(R) (Eq. advantage_calculation), and the invariances of the
definition (shifting or scaling the rewards, relabelling node ids).
"""
from __future__ import annotations

import math
from typing import Dict, List, Sequence, Tuple

import numpy as np


def tree_advantage(parent: Sequence[int], leaves: Sequence[int], rewards: Sequence[float]
                   ) -> Tuple[np.ndarray, Dict[str, float]]:
    """parent[x] = parent node of x (-1 for a root); returns (adv [n] fp64,
    {"accepted", "mean", "std"})."""
    n = len(leaves)
    R = [float(r) for r in rewards]
    groups: List[List[int]] = []          # strict ancestors of each leaf
    for lf in leaves:
        chain, x = [], parent[lf]
        while x != -1:
            chain.append(x)
            x = parent[x]
        groups.append(chain)
    members: Dict[int, List[int]] = {}
    for i, chain in enumerate(groups):
        for x in chain:
            members.setdefault(x, []).append(i)
    root = [chain[-1] if chain else leaves[i] for i, chain in enumerate(groups)]
    by_root: Dict[int, List[float]] = {}
    for i in range(n):
        by_root.setdefault(root[i], []).append(R[i])
    A = np.zeros(n, dtype=np.float64)
    accepted = []
    for i in range(n):
        rs = by_root[root[i]]
        if not groups[i] or min(rs) == max(rs):
            continue
        total = 0.0
        for x in groups[i]:
            total += R[i] - sum(R[k] for k in members[x]) / len(members[x])
        A[i] = total / len(groups[i])
        accepted.append(i)
    if not accepted:
        return np.zeros(n), {"accepted": 0, "mean": 0.0, "std": 0.0}
    mean = sum(A[i] for i in accepted) / len(accepted)
    std = math.sqrt(sum((A[i] - mean) ** 2 for i in accepted) / len(accepted))
    adv = np.zeros(n, dtype=np.float64)
    if std > 0.0:
        for i in accepted:
            adv[i] = A[i] / std
    return adv, {"accepted": len(accepted), "mean": mean, "std": std}
