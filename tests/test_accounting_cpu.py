"""The library's memory accounting, admission check and degradation planner
(kv_memory_account, kv_admission_check, kv_degradation_plan: §III-C, Alg. 2,
Eq. 3) against oracle/mem_model.py, through the C ABI.  Host code only."""
import json
import os

import numpy as np
import pytest

import oracle.mem_model as MM
from paper_2606_12950_gb300 import kvpool as K

GOLD = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
MB, GB = 10 ** 6, 10 ** 9
STATE = {MM.IDLE: K.KV_ENGINE_IDLE, MM.SLEEPING: K.KV_ENGINE_SLEEPING, MM.SLEEP_PENDING: K.KV_ENGINE_SLEEP_PENDING,
         MM.ACTIVE: K.KV_ENGINE_ACTIVE, MM.COLD: K.KV_ENGINE_COLD}
ACTION = {K.KV_ACT_SLEEP: MM.SLEEP, K.KV_ACT_EVICT: MM.EVICT, K.KV_ACT_STOP: MM.STOP, K.KV_ACT_PREEMPT: MM.PREEMPT,
          K.KV_ACT_ABORT: MM.ABORT}


def to_abi(e):
    return {"state": STATE[e.state], "ctx_bytes": e.ctx, "weight_bytes": e.weights, "kv_bytes": e.kv,
            "virtual_kv_bytes": e.virtual_kv, "weight_reload_s": e.t_weights, "ctx_rebuild_s": e.t_ctx,
            "kv_swap_in_s": e.t_swap, "kv_regen_s": e.t_regen}


def random_node(rng):
    states = [MM.IDLE, MM.SLEEPING, MM.SLEEP_PENDING, MM.ACTIVE, MM.COLD]
    eng = []
    for _ in range(int(rng.integers(0, 9))):
        st = states[int(rng.integers(0, 5))]
        eng.append(MM.Engine(state=st, ctx=int(rng.integers(0, 300)) * MB, weights=int(rng.integers(0, 30000)) * MB,
                             kv=int(rng.integers(0, 20000)) * MB if st == MM.ACTIVE else int(rng.integers(0, 2)) * MB,
                             virtual_kv=int(rng.integers(0, 40000)) * MB, t_weights=float(rng.random() * 3),
                             t_ctx=float(rng.random() * 3), t_swap=float(rng.random()), t_regen=float(rng.random() * 9)))
    return eng


def test_table5_through_the_library():
    t = json.load(open(os.path.join(GOLD, "table5_colocation.json")))
    eng = [{"state": K.KV_ENGINE_SLEEPING, "ctx_bytes": m["cuda_graph_mb"] * MB,
            "weight_bytes": round(m["weights_gb"] * 100) * 10 ** 7,
            "virtual_kv_bytes": round(m["virtual_kv_gb"] * 100) * 10 ** 7} for m in t["models"]]
    a = K.kv_memory_account(eng, t["gpu_gb"] * GB, 0)
    assert a["m_kv_virtual"] == 122_010 * MB
    assert round(a["overcommit"], 2) == t["printed"]["effective_footprint_x"]
    assert round(100 * (1 - 1 / a["overcommit"]), 1) == t["printed"]["hbm_reduction_percent"]
    assert a["m_res"] == 1175 * MB and a["safe"]


def test_worked_example_through_the_library():
    w = json.load(open(os.path.join(GOLD, "alg2_worked.json")))
    eng = [{"state": STATE[e["state"]], "ctx_bytes": e["ctx_mb"] * MB, "weight_bytes": e["weights_mb"] * MB,
            "kv_bytes": e["kv_mb"] * MB, "virtual_kv_bytes": e["virtual_kv_mb"] * MB,
            "weight_reload_s": e.get("t_weights", 0.0), "ctx_rebuild_s": e.get("t_ctx", 0.0),
            "kv_swap_in_s": e.get("t_swap", 0.0), "kv_regen_s": e.get("t_regen", 0.0)} for e in w["engines"]]
    for c in w["cases"]:
        r = K.kv_admission_check(eng, w["m_total_mb"] * MB, w["m_other_mb"] * MB, 0, c["demand_mb"] * MB,
                                 c["host_swap_mb"] * MB, w["c_int"])
        assert r["ok"] == c["ok"] and r["interrupt"] == c["interrupt"], c
        assert [[s["engine"], ACTION[s["action"]]] for s in r["steps"]] == c["plan"], c
        assert r["c_deg"] == pytest.approx(c["c_deg"], abs=1e-12)
        assert r["headroom"] == w["account"]["headroom_mb"] * MB


def test_account_matches_the_model_on_random_nodes():
    rng = np.random.default_rng(11)
    for _ in range(300):
        eng = random_node(rng)
        m_total = int(rng.integers(1, 200)) * GB
        m_other = int(rng.integers(0, 3000)) * MB
        extra = int(rng.integers(0, 2)) * int(rng.integers(0, 5000)) * MB
        a = K.kv_memory_account([to_abi(e) for e in eng], m_total, m_other, extra)
        assert a["m_res"] == MM.m_res(eng, m_other)
        assert a["m_kv"] == MM.m_kv(eng, extra)
        assert a["m_kv_virtual"] == MM.virtual_kv(eng)
        assert a["headroom"] == MM.headroom(eng, m_total, m_other, extra)
        assert a["safe"] == MM.is_safe(eng, m_total, m_other, extra)
        assert a["overcommit"] == MM.virtual_kv(eng) / m_total


def test_plans_match_the_model_on_random_nodes():
    rng = np.random.default_rng(12)
    fails = 0
    for _ in range(500):
        eng = random_node(rng)
        R = int(rng.integers(0, 80000)) * MB
        swap = int(rng.integers(0, 30000)) * MB
        c_int = float(rng.random() * 10)
        ok, plan, intr, freed = MM.coordinate(R, eng, swap)
        r = K.kv_degradation_plan([to_abi(e) for e in eng], R, swap, c_int)
        fails += not ok
        assert r["ok"] == ok and r["interrupt"] == intr and r["freed"] == freed
        assert [(s["engine"], ACTION[s["action"]]) for s in r["steps"]] == plan
        assert [s["freed_bytes"] for s in r["steps"]] == [MM.estimate_freed_memory(eng[i], a) for i, a in plan]
        assert [s["cost_s"] for s in r["steps"]] == [MM.restoration_cost(eng[i], a) for i, a in plan]
        assert r["c_deg"] == pytest.approx(MM.degradation_cost(eng, plan, intr, c_int), rel=1e-14, abs=1e-14)
    assert 50 < fails < 450  # both outcomes exercised


def test_admission_matches_the_model_on_random_nodes():
    rng = np.random.default_rng(13)
    for _ in range(300):
        eng = random_node(rng)
        m_total, m_other = int(rng.integers(1, 120)) * GB, int(rng.integers(0, 2000)) * MB
        demand, swap, c_int = int(rng.integers(0, 60000)) * MB, int(rng.integers(0, 20000)) * MB, 4.0
        ok, plan, intr, cost, h = MM.admission(eng, m_total, m_other, 0, demand, swap, c_int)
        r = K.kv_admission_check([to_abi(e) for e in eng], m_total, m_other, 0, demand, swap, c_int)
        assert (r["ok"], r["interrupt"], r["headroom"]) == (ok, intr, h)
        assert [(s["engine"], ACTION[s["action"]]) for s in r["steps"]] == plan
        assert r["c_deg"] == pytest.approx(cost, rel=1e-14, abs=1e-14)


def test_argument_validation():
    L = K.lib()
    bad = [{"state": 7}]
    with pytest.raises(K.KVError):
        K.kv_memory_account(bad, GB, 0)
    with pytest.raises(K.KVError):
        K.kv_degradation_plan(bad, GB)
    with pytest.raises(K.KVError):
        K.kv_admission_check([], GB, 0, 0, 1 << 63)  # demand beyond int64
    assert L.kv_memory_account(None, 0, GB, 0, 0, None) == K.KV_ERR_INVALID_ARG
    a = K.kv_memory_account([], 0, 0)
    assert a["overcommit"] == 0.0 and a["safe"] and a["headroom"] == 0
    r = K.kv_degradation_plan([], 0)
    assert r["ok"] and r["steps"] == [] and r["c_deg"] == 0.0
    assert not K.kv_degradation_plan([], 1)["ok"]
