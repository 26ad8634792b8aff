// accounting.cpp -- explicit memory accounting of a multi-model node, its
// KV admission headroom, and minimum-impact memory coordination (§III-C;
// Alg. 2; Eq. 3).  Host code only.
#include <algorithm>
#include <cstdint>
#include <vector>

#include "kvpool.h"

namespace {

bool valid_state(int32_t st) { return st >= KV_ENGINE_IDLE && st <= KV_ENGINE_COLD; }

bool weights_on_gpu(int32_t st)
{
    return st == KV_ENGINE_IDLE || st == KV_ENGINE_SLEEP_PENDING || st == KV_ENGINE_ACTIVE;
}

bool warm(int32_t st) { return st != KV_ENGINE_COLD; }

// M_ctx^k: the context a warm model keeps, plus its weights while resident
uint64_t footprint(const kv_engine &e)
{
    if (!warm(e.state)) return 0;
    return e.ctx_bytes + (weights_on_gpu(e.state) ? e.weight_bytes : 0);
}

// degradation level of the least disruptive action for a state (1..4; 0 = none)
int level(int32_t st)
{
    switch (st) {
    case KV_ENGINE_IDLE: return 1;
    case KV_ENGINE_SLEEPING: return 2;
    case KV_ENGINE_SLEEP_PENDING: return 3;
    case KV_ENGINE_ACTIVE: return 4;
    default: return 0;
    }
}

bool args_ok(const kv_engine *engines, int n)
{
    if (n < 0 || (n > 0 && !engines)) return false;
    for (int i = 0; i < n; ++i)
        if (!valid_state(engines[i].state)) return false;
    return true;
}

struct Plan {
    std::vector<kv_plan_step> steps;
    uint64_t freed = 0;
    int interrupt = 0;
    double c_deg = 0.0;
};

// Alg. 2: greedy walk over the engines in level order until R is met
Plan plan_for(const kv_engine *engines, int n, uint64_t required, uint64_t host_swap_bytes, double c_int)
{
    std::vector<int> order;
    for (int i = 0; i < n; ++i)
        if (level(engines[i].state) > 0) order.push_back(i);
    std::stable_sort(order.begin(), order.end(),
                     [&](int a, int b) { return level(engines[a].state) < level(engines[b].state); });
    Plan p;
    uint64_t swap_left = host_swap_bytes;
    double cost = 0.0;
    for (int i : order) {
        if (p.freed >= required) break;
        const kv_engine &e = engines[i];
        kv_plan_step st{};
        st.engine = i;
        switch (e.state) {
        case KV_ENGINE_IDLE:
            st.action = KV_ACT_SLEEP;
            st.freed_bytes = e.weight_bytes;
            st.cost_s = e.weight_reload_s;
            break;
        case KV_ENGINE_SLEEPING:
            st.action = KV_ACT_EVICT;
            st.freed_bytes = e.ctx_bytes;
            st.cost_s = e.ctx_rebuild_s;
            break;
        case KV_ENGINE_SLEEP_PENDING:
            st.action = KV_ACT_STOP;
            st.freed_bytes = e.weight_bytes + e.ctx_bytes;
            st.cost_s = e.weight_reload_s + e.ctx_rebuild_s;
            break;
        default:  // ACTIVE: swap the KV out while the host has room, else abort
            st.freed_bytes = e.kv_bytes;
            if (e.kv_bytes <= swap_left) {
                st.action = KV_ACT_PREEMPT;
                st.cost_s = e.kv_swap_in_s;
                swap_left -= e.kv_bytes;
            } else {
                st.action = KV_ACT_ABORT;
                st.cost_s = e.kv_regen_s;
            }
            break;
        }
        if (st.freed_bytes == 0) continue;  // nothing to gain from disturbing it
        if (st.action == KV_ACT_PREEMPT || st.action == KV_ACT_ABORT) p.interrupt = 1;
        p.freed += st.freed_bytes;
        cost += st.cost_s;
        p.steps.push_back(st);
    }
    p.c_deg = cost + (p.interrupt ? c_int : 0.0);  // Eq. 3
    return p;
}

void emit(const Plan &p, kv_plan_step *steps, int max_steps, int *n_steps, int *interrupt, double *c_deg)
{
    const int k = (int)p.steps.size();
    for (int i = 0; i < std::min(k, max_steps); ++i) steps[i] = p.steps[(size_t)i];
    *n_steps = k;
    *interrupt = p.interrupt;
    *c_deg = p.c_deg;
}

}  // namespace

extern "C" {

int kv_memory_account(const kv_engine *engines, int n, uint64_t m_total, uint64_t m_other, uint64_t extra_kv_bytes,
                      kv_account *out)
{
    if (!out || !args_ok(engines, n)) return KV_ERR_INVALID_ARG;
    uint64_t res = m_other, kv = extra_kv_bytes, virt = 0;
    for (int i = 0; i < n; ++i) {
        const kv_engine &e = engines[i];
        res += footprint(e);
        if (e.state == KV_ENGINE_ACTIVE) kv += e.kv_bytes;
        if (warm(e.state)) virt += e.virtual_kv_bytes;
    }
    out->m_res = res;
    out->m_kv = kv;
    out->m_kv_virtual = virt;
    out->headroom = (int64_t)m_total - (int64_t)res - (int64_t)kv;
    out->safe = kv + res <= m_total;
    out->reserved = 0;
    out->overcommit = m_total ? (double)virt / (double)m_total : 0.0;
    return KV_OK;
}

int kv_degradation_plan(const kv_engine *engines, int n, uint64_t required, uint64_t host_swap_bytes, double c_int,
                        kv_plan_step *steps, int max_steps, int *n_steps, int *interrupt, double *c_deg,
                        uint64_t *freed)
{
    if (!n_steps || !interrupt || !c_deg || max_steps < 0 || (max_steps > 0 && !steps) || !args_ok(engines, n))
        return KV_ERR_INVALID_ARG;
    const Plan p = plan_for(engines, n, required, host_swap_bytes, c_int);
    emit(p, steps, max_steps, n_steps, interrupt, c_deg);
    if (freed) *freed = p.freed;
    return p.freed >= required ? KV_OK : KV_ERR_OUT_OF_BLOCKS;
}

int kv_admission_check(const kv_engine *engines, int n, uint64_t m_total, uint64_t m_other, uint64_t extra_kv_bytes,
                       uint64_t demand, uint64_t host_swap_bytes, double c_int, kv_plan_step *steps, int max_steps,
                       int *n_steps, int *interrupt, double *c_deg, int64_t *headroom)
{
    if (!n_steps || !interrupt || !c_deg || !headroom || max_steps < 0 || (max_steps > 0 && !steps) ||
        demand > (uint64_t)INT64_MAX || m_total > (uint64_t)INT64_MAX)
        return KV_ERR_INVALID_ARG;
    kv_account acc;
    const int rc = kv_memory_account(engines, n, m_total, m_other, extra_kv_bytes, &acc);
    if (rc) return rc;
    *headroom = acc.headroom;
    if (acc.headroom >= 0 && demand <= (uint64_t)acc.headroom) {
        *n_steps = 0;
        *interrupt = 0;
        *c_deg = 0.0;
        return KV_OK;
    }
    const uint64_t required = (uint64_t)((int64_t)demand - acc.headroom);  // R = demand - R_kv^head > 0
    const Plan p = plan_for(engines, n, required, host_swap_bytes, c_int);
    emit(p, steps, max_steps, n_steps, interrupt, c_deg);
    return p.freed >= required ? KV_OK : KV_ERR_OUT_OF_BLOCKS;
}

}  // extern "C"
