"""Pins of oracle/mem_model.py (memory accounting, Alg. 2, Eq. 3) to values
fixed outside the model: Table 5's printed figures, a plan worked by hand on
the Table 5 node (tests/golden/alg2_worked.json), and invariants that any
correct greedy plan satisfies.  A mutation check then plants plausible
mistakes in a copy of the model and requires each to fail a pin."""
import json
import math
import os
import sys
import types

import numpy as np
import pytest

import oracle.mem_model as MM

GOLD = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
MB = 10 ** 6
GB = 10 ** 9


def _load(name):
    with open(os.path.join(GOLD, name)) as f:
        return json.load(f)


def table5_engines(mm, state):
    t = _load("table5_colocation.json")
    return [mm.Engine(state=state, ctx=m["cuda_graph_mb"] * MB, weights=round(m["weights_gb"] * 100) * 10 ** 7,
                      virtual_kv=round(m["virtual_kv_gb"] * 100) * 10 ** 7) for m in t["models"]], t


def worked_engines(mm):
    w = _load("alg2_worked.json")
    eng = []
    for e in w["engines"]:
        eng.append(mm.Engine(state=e["state"], ctx=e["ctx_mb"] * MB, weights=e["weights_mb"] * MB, kv=e["kv_mb"] * MB,
                             virtual_kv=e["virtual_kv_mb"] * MB, t_weights=e.get("t_weights", 0.0),
                             t_ctx=e.get("t_ctx", 0.0), t_swap=e.get("t_swap", 0.0), t_regen=e.get("t_regen", 0.0)))
    return eng, w


# ------------------------------------------------------------------ pins ---

def pin_table5_overcommit(mm):
    """Table 5 / §IV-C: about 122 GB of virtual KV on a 40 GB GPU is a 3.05x
    footprint, 205% overcommitment, 67.2% less HBM than reserving it all."""
    eng, t = table5_engines(mm, mm.SLEEPING)
    p = t["printed"]
    v = mm.virtual_kv(eng)
    total = t["gpu_gb"] * GB
    assert round(v / GB) == p["total_virtual_kv_gb_approx"]
    assert round(v / total, 2) == p["effective_footprint_x"]
    assert round(100 * (v / total - 1)) == p["overcommit_percent"]
    assert round(100 * (1 - total / v), 1) == p["hbm_reduction_percent"]


def pin_table5_contexts(mm):
    """Sleeping models keep only their contexts on the GPU: 194-286 MB each,
    about 1.15 GB for the five (the paper's GB here is 1024 MB)."""
    eng, t = table5_engines(mm, mm.SLEEPING)
    p = t["printed"]
    per = [mm.m_ctx(e) for e in eng]
    assert min(per) == p["context_mb_min"] * MB and max(per) == p["context_mb_max"] * MB
    res = mm.m_res(eng, 0)
    assert round(res / MB / 1024, 2) == p["context_total_gb_approx"]
    # a model that is Running also holds its weights
    run, _ = table5_engines(mm, mm.IDLE)
    assert mm.m_res(run, 0) - res == sum(e.weights for e in run)
    # only an Active engine's KV is in use; a stale figure elsewhere is not counted
    stale = [mm.Engine(state=st, ctx=MB, weights=2 * MB, kv=3 * GB) for st in (mm.IDLE, mm.SLEEPING, mm.COLD)]
    assert mm.m_kv(stale, 5) == 5
    stale.append(mm.Engine(state=mm.ACTIVE, kv=3 * GB))
    assert mm.m_kv(stale) == 3 * GB
    cold, _ = table5_engines(mm, mm.COLD)
    assert mm.m_res(cold, 7) == 7 and mm.virtual_kv(cold) == 0


def pin_table5_feasibility(mm):
    """All five Running need 54.67 GB of weights plus contexts: unsafe on 40 GB
    (negative headroom); all Sleeping leave 40 GB - 1.175 GB - M_other."""
    run, _ = table5_engines(mm, mm.IDLE)
    assert not mm.is_safe(run, 40 * GB, 0)
    assert mm.headroom(run, 40 * GB, 0) == 40 * GB - 54_670 * MB - 1175 * MB
    slp, _ = table5_engines(mm, mm.SLEEPING)
    assert mm.headroom(slp, 40 * GB, 500 * MB, extra=2 * GB) == 40 * GB - 1175 * MB - 500 * MB - 2 * GB
    assert mm.is_safe(slp, 40 * GB, 500 * MB)


def pin_worked_account(mm):
    eng, w = worked_engines(mm)
    a = w["account"]
    assert mm.m_res(eng, w["m_other_mb"] * MB) == a["m_res_mb"] * MB
    assert mm.m_kv(eng) == a["m_kv_mb"] * MB
    assert mm.headroom(eng, w["m_total_mb"] * MB, w["m_other_mb"] * MB) == a["headroom_mb"] * MB
    assert mm.virtual_kv(eng) == a["virtual_kv_mb"] * MB


def pin_worked_plans(mm):
    eng, w = worked_engines(mm)
    for c in w["cases"]:
        ok, plan, intr, cost, h = mm.admission(eng, w["m_total_mb"] * MB, w["m_other_mb"] * MB, 0,
                                               c["demand_mb"] * MB, c["host_swap_mb"] * MB, w["c_int"])
        assert ok == c["ok"], c
        assert [list(p) for p in plan] == c["plan"], c
        assert intr == c["interrupt"], c
        assert math.isclose(cost, c["c_deg"], abs_tol=1e-12), c
        if "headroom_after_mb" in c:
            after = mm.apply_plan(eng, plan)
            assert mm.headroom(after, w["m_total_mb"] * MB, w["m_other_mb"] * MB) == c["headroom_after_mb"] * MB


def random_engines(mm, rng, n):
    states = [mm.IDLE, mm.SLEEPING, mm.SLEEP_PENDING, mm.ACTIVE, mm.COLD]
    out = []
    for _ in range(n):
        st = states[int(rng.integers(0, 5))]
        out.append(mm.Engine(state=st, ctx=int(rng.integers(0, 4)) * 100 * MB,
                             weights=int(rng.integers(0, 30)) * 500 * MB,
                             kv=int(rng.integers(0, 20)) * 400 * MB if st == mm.ACTIVE else 0,
                             virtual_kv=int(rng.integers(0, 40)) * GB, t_weights=float(rng.random()),
                             t_ctx=float(rng.random()), t_swap=float(rng.random()), t_regen=float(rng.random())))
    return out


def _frees_nothing(mm, e):
    """Every action open to a warm engine in state e.state frees zero bytes."""
    if e.state == mm.IDLE:
        return e.weights == 0
    if e.state == mm.SLEEPING:
        return e.ctx == 0
    if e.state == mm.SLEEP_PENDING:
        return e.weights == 0 and e.ctx == 0
    return e.kv == 0


def pin_plan_invariants(mm):
    """Any plan: levels never decrease; it stops as soon as R is met (dropping
    its last step leaves less than R); interrupt iff a Preempt or Abort is in
    it; failure only when every engine with something to free was used; the
    node's headroom after the plan grows by exactly the freed bytes;
    C_deg adds c_int exactly when interrupted; Preempts never exceed the
    host swap space."""
    rng = np.random.default_rng(7)
    level = {mm.SLEEP: 1, mm.EVICT: 2, mm.STOP: 3, mm.PREEMPT: 4, mm.ABORT: 4}
    for trial in range(400):
        eng = random_engines(mm, rng, int(rng.integers(0, 7)))
        R = int(rng.integers(0, 60)) * 500 * MB
        swap = int(rng.integers(0, 20)) * 400 * MB
        ok, plan, intr, freed = mm.coordinate(R, eng, swap)
        lv = [level[a] for _, a in plan]
        assert lv == sorted(lv)
        assert ok == (freed >= R)
        if plan:
            last = plan[-1][0]
            h0 = mm.headroom(eng, 10 ** 12, 0)
            h1 = mm.headroom(mm.apply_plan(eng, plan), 10 ** 12, 0)
            assert h1 - h0 == freed
            before = mm.apply_plan(eng, plan[:-1])
            assert mm.headroom(before, 10 ** 12, 0) - h0 < R
            assert freed > 0 and last >= 0
        else:
            assert freed == 0
        assert intr == any(a in (mm.PREEMPT, mm.ABORT) for _, a in plan)
        assert sum(eng[i].kv for i, a in plan if a == mm.PREEMPT) <= swap
        if not ok:
            used = {i for i, _ in plan}
            for i, e in enumerate(eng):
                if mm.is_warm(e) and i not in used:
                    assert _frees_nothing(mm, e), (trial, i)
        c0 = mm.degradation_cost(eng, plan, False, 0.0)
        assert mm.degradation_cost(eng, plan, intr, 3.5) == pytest.approx(c0 + (3.5 if intr else 0.0))
        if R == 0:
            assert plan == [] and ok


def pin_degradation_is_least_disruptive_first(mm):
    """With one engine per state and room for everything, the plan walks the
    five levels in the paper's order (the Active one gets Preempt with swap
    space, Abort without)."""
    eng = [mm.Engine(state=mm.ACTIVE, kv=5 * GB, t_swap=1, t_regen=9),
           mm.Engine(state=mm.SLEEP_PENDING, ctx=GB, weights=3 * GB, t_weights=2, t_ctx=3),
           mm.Engine(state=mm.SLEEPING, ctx=GB, weights=8 * GB, t_ctx=4),
           mm.Engine(state=mm.IDLE, ctx=GB, weights=2 * GB, t_weights=5)]
    ok, plan, intr, freed = mm.coordinate(11 * GB, eng, host_swap=5 * GB)
    assert ok and intr and freed == 2 * GB + GB + 4 * GB + 5 * GB
    assert plan == [(3, mm.SLEEP), (2, mm.EVICT), (1, mm.STOP), (0, mm.PREEMPT)]
    assert mm.degradation_cost(eng, plan, intr, 10.0) == 5 + 4 + 5 + 1 + 10.0
    ok, plan, _, _ = mm.coordinate(11 * GB, eng, host_swap=0)
    assert plan[-1] == (0, mm.ABORT) and mm.degradation_cost(eng, plan, True, 0.0) == 5 + 4 + 5 + 9
    ok, plan, intr, _ = mm.coordinate(2 * GB, eng)
    assert plan == [(3, mm.SLEEP)] and not intr


PINS = [pin_table5_overcommit, pin_table5_contexts, pin_table5_feasibility, pin_worked_account, pin_worked_plans,
        pin_plan_invariants, pin_degradation_is_least_disruptive_first]


@pytest.mark.parametrize("pin", PINS, ids=lambda f: f.__name__)
def test_mem_model_pin(pin):
    pin(MM)


# ------------------------------------------------------------- mutation ---

MUTANTS = {
    "weights counted while sleeping": ("on_gpu = e.state in (IDLE, SLEEP_PENDING, ACTIVE)",
                                       "on_gpu = e.state in (IDLE, SLEEPING, SLEEP_PENDING, ACTIVE)"),
    "weights never counted": ("return e.ctx + (e.weights if on_gpu else 0)", "return e.ctx"),
    "M_other dropped": ("    total = m_other\n", "    total = 0\n"),
    "KV of idle engines counted": ("        if e.state == ACTIVE:\n            total += e.kv",
                                   "        if is_warm(e):\n            total += e.kv"),
    "headroom sign": ("return m_total - m_res(engines, m_other) - m_kv(engines, extra)",
                      "return m_total - m_res(engines, m_other) + m_kv(engines, extra)"),
    "cold engines warm": ("return e.state in (IDLE, SLEEPING, SLEEP_PENDING, ACTIVE)",
                          "return e.state in (IDLE, SLEEPING, SLEEP_PENDING, ACTIVE, COLD)"),
    "priority sleeping first": ("PRIORITY = {IDLE: 0, SLEEPING: 1,", "PRIORITY = {IDLE: 1, SLEEPING: 0,"),
    "active before pending": ("SLEEP_PENDING: 2, ACTIVE: 3}", "SLEEP_PENDING: 3, ACTIVE: 2}"),
    "no early stop": ("        if freed >= R:\n            break\n", ""),
    "stop one step late": ("        if freed >= R:\n            break\n", "        if freed > R:\n            break\n"),
    "interrupt never set": ("            interrupt = True\n", "            interrupt = False\n"),
    "c_int dropped": ("    if interrupt:\n        c += c_int", "    if interrupt:\n        c += 0.0"),
    "preempt ignores swap": ("if swap_in_use(engines, plan) + e.kv <= host_swap:", "if True:"),
    "stop frees weights only": ("    if action == STOP:\n        return e.weights + e.ctx",
                                "    if action == STOP:\n        return e.weights"),
    "evict frees weights": ("    if action == EVICT:\n        return e.ctx", "    if action == EVICT:\n        return e.weights"),
    "abort charged as swap": ("    return e.t_regen", "    return e.t_swap"),
    "R not net of headroom": ("coordinate(demand - h, engines, host_swap)", "coordinate(demand, engines, host_swap)"),
}


def _mutant(old, new):
    src = open(MM.__file__).read()
    assert src.count(old) == 1, old
    mod = types.ModuleType("mem_model_mutant")
    sys.modules["mem_model_mutant"] = mod  # dataclasses look their module up
    try:
        exec(compile(src.replace(old, new), "mem_model_mutant", "exec"), mod.__dict__)
    finally:
        del sys.modules["mem_model_mutant"]
    return mod


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_is_caught(name):
    old, new = MUTANTS[name]
    mod = _mutant(old, new)
    failed = []
    for pin in PINS:
        try:
            pin(mod)
        except (AssertionError, Exception):
            failed.append(pin.__name__)
    assert failed, f"mutant '{name}' passes every pin"
