"""Plain CPU oracle of the route-aware heuristic pipeline scheduler (arXiv 2508.06024, Eq. 9-11).

TEST INFRASTRUCTURE.  Only the tests may import this module.  It shares no
code with the library's scheduler and never calls it.

The paper's scheduler places each task t_i (computational complexity C(t_i),
communication cost Comm(t_i)) on the End or on the Cloud:

* Eq. 10 - priority P(t_i) = C(t_i) / (Comm(t_i) + eps); a high priority
  favours local (End) execution.
* Eq. 11 - Location(t_i) = End if Load_end + C(t_i) <= T_end and
  P(t_i) >= beta, else Cloud.
* Eq. 9  - the heuristic's objective, sum_i alpha * ExecTime(t_i) +
  (1 - alpha) * Comm(t_i).

Readings where the paper is silent (each one is listed in the design notes):

* The greedy visits the tasks in decreasing priority, ties to the lower task
  index, and keeps going after a task that goes to the Cloud.
* Load_end starts at the given current end load and grows by C(t_i) for every
  task placed on the End; Load_cloud grows the same way for Cloud tasks and is
  reported only (Eq. 11 does not consult it).
* ExecTime(t_i) = C(t_i) / rate of the chosen side; Comm(t_i) is paid only by
  tasks placed on the Cloud (a task run on the End transmits nothing).
* Route-aware tasks: one task per expert that received rows; C = FLOPs of
  the expert's FFN on its rows, Comm = bytes shipped to the Cloud and back
  (the encoded rows, r values each, or the full rows when there is no codec;
  plus the d-wide output rows).

Everything is written with Python floats (IEEE double) in the order stated.
"""
from __future__ import annotations

from typing import Dict, List, Sequence

END = 0
CLOUD = 1


def priority(cost: Sequence[float], comm: Sequence[float], eps: float) -> List[float]:
    """Eq. 10: P(t_i) = C(t_i) / (Comm(t_i) + eps)."""
    return [float(c) / (float(m) + eps) for c, m in zip(cost, comm)]


def visit_order(P: Sequence[float]) -> List[int]:
    """Decreasing priority, ties to the lower index."""
    return sorted(range(len(P)), key=lambda i: (-P[i], i))


def schedule(cost, comm, load_end, load_cloud, T_end, beta, eps) -> Dict[str, object]:
    """Eq. 11 applied greedily in priority order; returns location[i] (END or
    CLOUD), the visit order and both final loads."""
    P = priority(cost, comm, eps)
    order = visit_order(P)
    location = [CLOUD] * len(P)
    le, lc = float(load_end), float(load_cloud)
    for i in order:
        c = float(cost[i])
        if le + c <= T_end and P[i] >= beta:
            location[i] = END
            le = le + c
        else:
            location[i] = CLOUD
            lc = lc + c
    return {"location": location, "order": order, "load_end": le, "load_cloud": lc, "priority": P}


def objective(cost, comm, location, rate_end, rate_cloud, alpha) -> float:
    """Eq. 9: sum_i alpha * ExecTime(t_i) + (1 - alpha) * Comm(t_i), with
    ExecTime = C / (rate of the chosen side) and Comm paid on the Cloud only."""
    total = 0.0
    for c, m, loc in zip(cost, comm, location):
        exec_time = float(c) / (rate_end if loc == END else rate_cloud)
        paid = float(m) if loc == CLOUD else 0.0
        total = total + (alpha * exec_time + (1.0 - alpha) * paid)
    return total


def expert_tasks(counts, d, d_ff, swiglu, r, elem_bytes):
    """Route-aware tasks from the routing histogram: one per expert with rows.

    C_e = 2 * rows * d * d_ff * (3 projections for SwiGLU, 2 for GELU);
    Comm_e = rows * (width_in + d) * elem_bytes, width_in = r (encoded rows)
    or d when there is no codec.  Returns (expert ids, C, Comm)."""
    proj = 3 if swiglu else 2
    w_in = r if r > 0 else d
    ids, C, M = [], [], []
    for e, n in enumerate(counts):
        n = int(n)
        if n > 0:
            ids.append(e)
            C.append(2.0 * n * d * d_ff * proj)
            M.append(float(n * (w_in + d) * elem_bytes))
    return ids, C, M
