"""Route-aware heuristic pipeline scheduler (Eq. 9-11): the oracle against
hand-worked cases and special cases, planted mistakes that the pins must
catch, and the library's C-ABI implementation against the oracle.  Host code
only: everything here runs on the CPU."""
import json
import math
import os
import random

import pytest

from oracle import scheduler_oracle as so
from paper_2508_06024_gb300 import build as B
from paper_2508_06024_gb300 import ec2moe as C

GOLDEN = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "scheduler_examples.json")))
INF = float("inf")


# ---------------------------------------------------------------- pins of the oracle
def pin_worked_example(impl=so):
    g = GOLDEN["greedy"]
    out = impl.schedule(g["cost"], g["comm"], g["load_end"], g["load_cloud"], g["T_end"], g["beta"], g["eps"])
    assert out["priority"] == g["priority"]
    assert out["order"] == g["order"]
    assert out["location"] == g["location"]
    assert out["load_end"] == g["load_end_final"]
    assert out["load_cloud"] == g["load_cloud_final"]
    o = g["objective"]
    val = impl.objective(g["cost"], g["comm"], g["location"], o["rate_end"], o["rate_cloud"], o["alpha"])
    assert val == o["value"]


def pin_special_cases(impl=so):
    cost = [3.0, 1.0, 7.0, 2.0]
    comm = [1.0, 2.0, 0.5, 4.0]
    # beta = +inf: nothing is local; Load_end unchanged
    out = impl.schedule(cost, comm, 2.0, 0.0, 100.0, INF, 1e-9)
    assert out["location"] == [so.CLOUD] * 4 and out["load_end"] == 2.0 and out["load_cloud"] == sum(cost)
    # unbounded end and beta = 0: everything is local
    out = impl.schedule(cost, comm, 0.0, 0.0, INF, 0.0, 1e-9)
    assert out["location"] == [so.END] * 4 and out["load_end"] == sum(cost)
    # end already over its threshold: nothing fits
    out = impl.schedule(cost, comm, 11.0, 0.0, 10.0, 0.0, 1e-9)
    assert out["location"] == [so.CLOUD] * 4
    # a task too big for the end does not stop later, smaller tasks
    out = impl.schedule([9.0, 1.0, 1.0], [0.1, 1.0, 2.0], 0.0, 0.0, 5.0, 0.0, 0.0)
    assert out["order"] == [0, 1, 2] and out["location"] == [so.CLOUD, so.END, so.END]
    # equal priorities: the lower index is visited first and takes the room
    out = impl.schedule([2.0, 2.0], [1.0, 1.0], 0.0, 0.0, 3.0, 0.0, 0.0)
    assert out["order"] == [0, 1] and out["location"] == [so.END, so.CLOUD]
    # both bounds are inclusive: load + C == T_end and P == beta stay local
    out = impl.schedule([4.0], [2.0], 6.0, 0.0, 10.0, 2.0, 0.0)
    assert out["location"] == [so.END]
    # eps keeps a free-to-ship task finite: P = C / eps
    out = impl.schedule([1.0, 1.0], [0.0, 1.0], 0.0, 0.0, INF, 2.0, 0.25)
    assert out["priority"] == [4.0, 0.8] and out["location"] == [so.END, so.CLOUD]
    # objective: alpha = 1 is pure execution time, alpha = 0 the Cloud's communication
    loc = [so.END, so.CLOUD, so.CLOUD, so.END]
    assert impl.objective(cost, comm, loc, 2.0, 8.0, 1.0) == 3.0 / 2 + 1.0 / 8 + 7.0 / 8 + 2.0 / 2
    assert impl.objective(cost, comm, loc, 2.0, 8.0, 0.0) == 2.0 + 0.5


def pin_expert_tasks(impl=so):
    g = GOLDEN["expert_tasks"]
    ids, cost, comm = impl.expert_tasks(g["counts"], g["d"], g["d_ff"], False, g["r"], g["elem_bytes"])
    assert (ids, cost, comm) == (g["gelu"]["ids"], g["gelu"]["cost"], g["gelu"]["comm"])
    ids, cost, comm = impl.expert_tasks(g["counts"], g["d"], g["d_ff"], True, 0, g["elem_bytes"])
    sw = g["swiglu_no_codec"]
    assert (ids, cost, comm) == (sw["ids"], sw["cost"], sw["comm"])


PINS = [pin_worked_example, pin_special_cases, pin_expert_tasks]


@pytest.mark.parametrize("pin", PINS, ids=lambda f: f.__name__)
def test_oracle_pins(pin):
    pin()


# ---------------------------------------------------------------- planted mistakes
class _Mutant:
    """The oracle with one function replaced."""

    def __init__(self, **over):
        self.__dict__.update({k: getattr(so, k) for k in ("END", "CLOUD", "priority", "visit_order", "objective",
                                                          "expert_tasks")})
        self.__dict__.update(over)

    def schedule(self, cost, comm, load_end, load_cloud, T_end, beta, eps):
        if "schedule_impl" in self.__dict__:
            return self.schedule_impl(self, cost, comm, load_end, load_cloud, T_end, beta, eps)
        P = self.priority(cost, comm, eps)
        order = self.visit_order(P)
        location = [so.CLOUD] * len(P)
        le, lc = float(load_end), float(load_cloud)
        for i in order:
            c = float(cost[i])
            if le + c <= T_end and P[i] >= beta:
                location[i] = so.END
                le += c
            else:
                lc += c
        return {"location": location, "order": order, "load_end": le, "load_cloud": lc, "priority": P}


def _sched_strict(self, cost, comm, load_end, load_cloud, T_end, beta, eps):
    P = so.priority(cost, comm, eps)
    order = so.visit_order(P)
    loc = [so.CLOUD] * len(P)
    le, lc = float(load_end), float(load_cloud)
    for i in order:
        if le + cost[i] < T_end and P[i] > beta:
            loc[i] = so.END
            le += cost[i]
        else:
            lc += cost[i]
    return {"location": loc, "order": order, "load_end": le, "load_cloud": lc, "priority": P}


def _sched_no_load(self, cost, comm, load_end, load_cloud, T_end, beta, eps):
    P = so.priority(cost, comm, eps)
    order = so.visit_order(P)
    loc = [so.CLOUD] * len(P)
    for i in order:
        if load_end + cost[i] <= T_end and P[i] >= beta:
            loc[i] = so.END
    le = load_end + sum(c for c, l in zip(cost, loc) if l == so.END)
    lc = load_cloud + sum(c for c, l in zip(cost, loc) if l == so.CLOUD)
    return {"location": loc, "order": order, "load_end": le, "load_cloud": lc, "priority": P}


def _sched_stop_at_cloud(self, cost, comm, load_end, load_cloud, T_end, beta, eps):
    P = so.priority(cost, comm, eps)
    order = so.visit_order(P)
    loc = [so.CLOUD] * len(P)
    le, lc, stopped = float(load_end), float(load_cloud), False
    for i in order:
        if not stopped and le + cost[i] <= T_end and P[i] >= beta:
            loc[i] = so.END
            le += cost[i]
        else:
            stopped = True
            lc += cost[i]
    return {"location": loc, "order": order, "load_end": le, "load_cloud": lc, "priority": P}


MUTANTS = {
    "priority_ignores_eps": dict(priority=lambda cost, comm, eps: [c / m if m else math.inf for c, m in zip(cost, comm)]),
    "priority_inverted": dict(priority=lambda cost, comm, eps: [(m + eps) / c if c else math.inf for c, m in zip(cost, comm)]),
    "ascending_order": dict(visit_order=lambda P: sorted(range(len(P)), key=lambda i: (P[i], i))),
    "ties_to_higher_index": dict(visit_order=lambda P: sorted(range(len(P)), key=lambda i: (-P[i], -i))),
    "index_order": dict(visit_order=lambda P: list(range(len(P)))),
    "strict_bounds": dict(schedule_impl=_sched_strict),
    "end_load_not_accumulated": dict(schedule_impl=_sched_no_load),
    "greedy_stops_at_first_cloud": dict(schedule_impl=_sched_stop_at_cloud),
    "objective_charges_end_comm": dict(objective=lambda cost, comm, loc, re, rc, a: sum(
        a * c / (re if l == so.END else rc) + (1 - a) * m for c, m, l in zip(cost, comm, loc))),
    "objective_one_rate": dict(objective=lambda cost, comm, loc, re, rc, a: sum(
        a * c / re + (1 - a) * (m if l == so.CLOUD else 0.0) for c, m, l in zip(cost, comm, loc))),
    "tasks_count_swiglu_as_two": dict(expert_tasks=lambda counts, d, dff, sw, r, eb: so.expert_tasks(
        counts, d, dff, False, r, eb)),
    "tasks_ignore_output_rows": dict(expert_tasks=lambda counts, d, dff, sw, r, eb: (
        lambda t: (t[0], t[1], [m * (r if r else d) / ((r if r else d) + d) for m in t[2]]))(
        so.expert_tasks(counts, d, dff, sw, r, eb))),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_catch_planted_mistake(name):
    m = _Mutant(**MUTANTS[name])
    caught = 0
    for pin in PINS:
        try:
            pin(m)
        except (AssertionError, ZeroDivisionError):
            caught += 1
    assert caught >= 1, f"mutant {name} passes every pin"


# ---------------------------------------------------------------- library against the oracle
@pytest.fixture(scope="module")
def lib():
    B.build()
    return C.load()


def _random_case(rng, n):
    cost = [rng.choice([0.0, rng.uniform(0, 10), float(rng.randint(0, 6))]) for _ in range(n)]
    comm = [rng.choice([0.0, rng.uniform(0, 5), float(rng.randint(0, 3))]) for _ in range(n)]
    eps = rng.choice([1e-9, 0.5, 1.0])
    return cost, comm, eps


def test_library_matches_oracle_worked_example(lib):
    g = GOLDEN["greedy"]
    loc, order, le, lc = C.ec2moe_schedule(g["cost"], g["comm"], g["load_end"], g["load_cloud"], g["T_end"],
                                           g["beta"], g["eps"])
    assert loc == g["location"] and order == g["order"]
    assert le == g["load_end_final"] and lc == g["load_cloud_final"]
    o = g["objective"]
    assert C.ec2moe_schedule_objective(g["cost"], g["comm"], loc, o["rate_end"], o["rate_cloud"], o["alpha"]) == o["value"]


@pytest.mark.parametrize("seed", range(40))
def test_library_matches_oracle_random(lib, seed):
    rng = random.Random(seed)
    n = rng.choice([0, 1, 2, 5, 17, 64, 300])
    cost, comm, eps = _random_case(rng, n)
    load_end = rng.choice([0.0, rng.uniform(0, 20)])
    T_end = rng.choice([INF, rng.uniform(0, 60), 0.0])
    beta = rng.choice([0.0, rng.uniform(0, 5), INF, -INF])
    ref = so.schedule(cost, comm, load_end, 3.0, T_end, beta, eps)
    loc, order, le, lc = C.ec2moe_schedule(cost, comm, load_end, 3.0, T_end, beta, eps)
    assert loc == ref["location"] and order == ref["order"]
    assert le == ref["load_end"] and lc == ref["load_cloud"]
    a = rng.uniform(0, 1)
    got = C.ec2moe_schedule_objective(cost, comm, loc, 1.5, 6.0, a)
    want = so.objective(cost, comm, loc, 1.5, 6.0, a)
    assert math.isclose(got, want, rel_tol=1e-12, abs_tol=1e-300)


def test_library_expert_tasks(lib):
    g = GOLDEN["expert_tasks"]
    d = C.make_desc(T=8, d=g["d"], E=3, d_ff=g["d_ff"], k=1, act=C.GELU, dtype=C.BF16, r=g["r"])
    assert C.ec2moe_expert_tasks(d, g["counts"]) == (g["gelu"]["ids"], g["gelu"]["cost"], g["gelu"]["comm"])
    d = C.make_desc(T=8, d=g["d"], E=3, d_ff=g["d_ff"], k=1, act=C.SWIGLU, dtype=C.BF16, r=0)
    sw = g["swiglu_no_codec"]
    assert C.ec2moe_expert_tasks(d, g["counts"]) == (sw["ids"], sw["cost"], sw["comm"])
    rng = random.Random(7)
    counts = [rng.choice([0, rng.randint(1, 5000)]) for _ in range(64)]
    d = C.make_desc(T=16384, d=2048, E=64, d_ff=1408, k=6, act=C.SWIGLU, dtype=C.BF16, r=256)
    assert C.ec2moe_expert_tasks(d, counts) == tuple(so.expert_tasks(counts, 2048, 1408, True, 256, 2))


def test_library_rejects_bad_inputs(lib):
    with pytest.raises(C.Ec2moeError):
        C.ec2moe_schedule([1.0], [-1.0])
    with pytest.raises(C.Ec2moeError):
        C.ec2moe_schedule([float("nan")], [1.0])
    with pytest.raises(C.Ec2moeError):
        C.ec2moe_schedule([1.0], [0.0], eps=0.0)      # Comm + eps = 0
    with pytest.raises(C.Ec2moeError):
        C.ec2moe_schedule_objective([1.0], [1.0], [2], 1.0, 1.0, 0.5)
    with pytest.raises(C.Ec2moeError):
        C.ec2moe_schedule_objective([1.0], [1.0], [0], 0.0, 1.0, 0.5)
    d = C.make_desc(T=8, d=4, E=2, d_ff=8, k=1)
    with pytest.raises(C.Ec2moeError):
        C.ec2moe_expert_tasks(d, [1, -1])
