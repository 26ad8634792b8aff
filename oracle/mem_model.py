"""Reference model of the node runtime's memory accounting and of
minimum-impact memory coordination (TEST INFRASTRUCTURE ONLY: tests, the
smoke check and the benchmark's CPU baseline use it; the library never does).

What it follows:
  * §III-C, explicit memory accounting: M_res = sum over warm models (Running
    or Sleeping) of M_ctx^k, plus M_other; memory is safe while
    M_kv + M_res <= M_total; the KV admission headroom is
    R_kv^head = M_total - M_res - M_kv; a stage whose extra KV demand does not
    fit the headroom is rejected or triggers the coordination below.
  * §III-C, the five degradation levels in ascending disruption: idle Running
    -> Sleeping; evict Sleeping; stop pending sleep transitions; swap out the
    KV of Active models; abort Active executions.
  * Alg. 2: sort the resident engines by priority (Idle, Sleeping, Active);
    walk them, stopping once the freed memory reaches R; each gets its best
    action; Preempt/Abort raise the interrupt flag; failure if the walk ends
    short of R.
  * Eq. 3: C_deg = sum of c(e, a) over the plan + 1[I_active] * c_int.

Readings where the paper leaves a choice open (each also listed with the
design notes): a warm model's M_ctx^k is its kept context plus its weights
while they are on the GPU; a pending sleep is ordered between Sleeping and
Active (level 3) and stopping it shuts the engine down, freeing weights and
context; Preempt is chosen for an Active engine while its KV fits the host
swap space the plan so far has left, Abort otherwise, both freeing the KV;
an engine whose action would free nothing is passed over; ties keep the
caller's order.

Everything is integer bytes and plain floats, evaluated one engine at a time.
"""
from __future__ import annotations

from dataclasses import dataclass

IDLE, SLEEPING, SLEEP_PENDING, ACTIVE, COLD = "idle", "sleeping", "sleep_pending", "active", "cold"
SLEEP, EVICT, STOP, PREEMPT, ABORT = "sleep", "evict", "stop", "preempt", "abort"

# priority of Alg. 2's sort, in the order of the five degradation levels
PRIORITY = {IDLE: 0, SLEEPING: 1, SLEEP_PENDING: 2, ACTIVE: 3}


@dataclass
class Engine:
    state: str
    ctx: int = 0          # kept runtime context (CUDA graphs etc.), bytes
    weights: int = 0      # weight bytes
    kv: int = 0           # KV of executing stages, bytes (Active only)
    virtual_kv: int = 0   # virtual KV address space, bytes
    t_weights: float = 0.0  # restore the weights
    t_ctx: float = 0.0      # rebuild the context
    t_swap: float = 0.0     # swap the KV back in
    t_regen: float = 0.0    # regenerate the KV


def is_warm(e: Engine) -> bool:
    """Warm = Running (idle, active or about to sleep) or Sleeping."""
    return e.state in (IDLE, SLEEPING, SLEEP_PENDING, ACTIVE)


def m_ctx(e: Engine) -> int:
    """Persistent footprint of one warm model."""
    if not is_warm(e):
        return 0
    on_gpu = e.state in (IDLE, SLEEP_PENDING, ACTIVE)
    return e.ctx + (e.weights if on_gpu else 0)


def m_res(engines, m_other: int) -> int:
    total = m_other
    for e in engines:
        if is_warm(e):
            total += m_ctx(e)
    return total


def m_kv(engines, extra: int = 0) -> int:
    total = extra
    for e in engines:
        if e.state == ACTIVE:
            total += e.kv
    return total


def virtual_kv(engines) -> int:
    return sum(e.virtual_kv for e in engines if is_warm(e))


def headroom(engines, m_total: int, m_other: int, extra: int = 0) -> int:
    """R_kv^head = M_total - M_res - M_kv."""
    return m_total - m_res(engines, m_other) - m_kv(engines, extra)


def is_safe(engines, m_total: int, m_other: int, extra: int = 0) -> bool:
    return m_kv(engines, extra) + m_res(engines, m_other) <= m_total


def sort_by_priority(engines):
    """Indices of the resident engines, Idle first, Active last (stable)."""
    idx = [i for i, e in enumerate(engines) if e.state in PRIORITY]
    return sorted(idx, key=lambda i: PRIORITY[engines[i].state])


def swap_in_use(engines, plan) -> int:
    return sum(engines[i].kv for i, a in plan if a == PREEMPT)


def determine_best_action(engines, i: int, plan, host_swap: int):
    """The least disruptive action engine i's state allows, given the plan so far."""
    e = engines[i]
    if e.state == IDLE:
        return SLEEP
    if e.state == SLEEPING:
        return EVICT
    if e.state == SLEEP_PENDING:
        return STOP
    # Active: swap the KV out if the host still has room for it
    if swap_in_use(engines, plan) + e.kv <= host_swap:
        return PREEMPT
    return ABORT


def estimate_freed_memory(e: Engine, action: str) -> int:
    if action == SLEEP:
        return e.weights
    if action == EVICT:
        return e.ctx
    if action == STOP:
        return e.weights + e.ctx
    return e.kv  # PREEMPT or ABORT


def restoration_cost(e: Engine, action: str) -> float:
    """c(e, a)."""
    if action == SLEEP:
        return e.t_weights
    if action == EVICT:
        return e.t_ctx
    if action == STOP:
        return e.t_weights + e.t_ctx
    if action == PREEMPT:
        return e.t_swap
    return e.t_regen


def coordinate(R: int, engines, host_swap: int = 0):
    """Alg. 2.  Returns (ok, plan, I_active, freed); plan = [(index, action)]."""
    freed = 0
    plan = []
    interrupt = False
    for i in sort_by_priority(engines):
        if freed >= R:
            break
        action = determine_best_action(engines, i, plan, host_swap)
        gain = estimate_freed_memory(engines[i], action)
        if gain == 0:
            continue
        if action in (PREEMPT, ABORT):
            interrupt = True
        freed += gain
        plan.append((i, action))
    return freed >= R, plan, interrupt, freed


def degradation_cost(engines, plan, interrupt: bool, c_int: float) -> float:
    """Eq. 3."""
    c = 0.0
    for i, a in plan:
        c += restoration_cost(engines[i], a)
    if interrupt:
        c += c_int
    return c


def admission(engines, m_total: int, m_other: int, extra: int, demand: int, host_swap: int, c_int: float):
    """Admission of a stage needing `demand` more KV bytes.
    Returns (ok, plan, I_active, C_deg, headroom)."""
    h = headroom(engines, m_total, m_other, extra)
    if demand <= h:
        return True, [], False, 0.0, h
    ok, plan, interrupt, _ = coordinate(demand - h, engines, host_swap)
    return ok, plan, interrupt, degradation_cost(engines, plan, interrupt, c_int), h


def apply_plan(engines, plan):
    """The engines after the plan has run (state transitions of each action)."""
    out = [Engine(**vars(e)) for e in engines]
    for i, a in plan:
        e = out[i]
        if a == SLEEP:
            e.state = SLEEPING
        elif a in (EVICT, STOP):
            e.state = COLD
        else:  # the KV left the GPU; the engine stays Running
            e.kv = 0
    return out
