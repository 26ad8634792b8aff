// vmm.cpp -- VMM-backed elastic KV pool (§III-C, "spatial multiplexing with
// virtual-memory KV cache").
//
// The pool's address range is reserved as virtual memory and may exceed the
// physical memory the KV is allowed (overcommitment, Table 5); physical
// chunks are mapped when the allocator needs their superpages and unmapped
// again by kv_pool_trim, so several colocated pools can each reserve their
// worst case while only the blocks in use occupy HBM.  A chunk that cannot
// be mapped (out of device memory, the pool's physical limit or a shared
// budget) rejects the allocation (KV_ERR_OUT_OF_BLOCKS) instead of failing
// later.  Every unmapped chunk is backed by one shared guard allocation, so a
// table entry naming an unallocated block reads harmless memory instead of
// faulting, as with a fixed pool.
#include <algorithm>
#include <atomic>
#include <mutex>
#include <numeric>

#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include "pool_internal.h"

struct kv_budget {
    uint64_t limit = 0;
    std::atomic<uint64_t> used{0};
    std::atomic<int> pools{0};
};

namespace {

struct Driver {
    PFN_cuMemAddressReserve_v10020 reserve = nullptr;
    PFN_cuMemAddressFree_v10020 addr_free = nullptr;
    PFN_cuMemCreate_v10020 create = nullptr;
    PFN_cuMemRelease_v10020 release = nullptr;
    PFN_cuMemMap_v10020 map = nullptr;
    PFN_cuMemUnmap_v10020 unmap = nullptr;
    PFN_cuMemSetAccess_v10020 set_access = nullptr;
    PFN_cuMemGetAllocationGranularity_v10020 granularity = nullptr;
    bool ok = false;
};

template <class F>
bool entry(const char *name, F &fn)
{
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion(name, &p, 10020, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
        return false;
    fn = reinterpret_cast<F>(p);
    return true;
}

const Driver &driver()
{
    static Driver d;
    static std::once_flag once;
    std::call_once(once, [] {
        d.ok = entry("cuMemAddressReserve", d.reserve) && entry("cuMemAddressFree", d.addr_free) &&
               entry("cuMemCreate", d.create) && entry("cuMemRelease", d.release) && entry("cuMemMap", d.map) &&
               entry("cuMemUnmap", d.unmap) && entry("cuMemSetAccess", d.set_access) &&
               entry("cuMemGetAllocationGranularity", d.granularity);
    });
    return d;
}

CUmemAllocationProp device_prop(int device)
{
    CUmemAllocationProp prop = {};
    prop.type = CU_MEM_ALLOCATION_TYPE_PINNED;
    prop.location.type = CU_MEM_LOCATION_TYPE_DEVICE;
    prop.location.id = device;
    return prop;
}

// per-pool CUDA backend state: the guard allocation mapped at unmapped chunks
struct CudaBacking {
    CUmemGenericAllocationHandle guard = 0;
    bool guard_ok = false;
};

CUdeviceptr chunk_va(const kv_pool *p, int64_t c)
{
    return (CUdeviceptr)((uintptr_t)p->desc.device_base + (uint64_t)c * p->vmm.chunk_bytes);
}

bool set_rw(const kv_pool *p, CUdeviceptr va, size_t bytes)
{
    CUmemAccessDesc acc = {};
    acc.location.type = CU_MEM_LOCATION_TYPE_DEVICE;
    acc.location.id = p->device;
    acc.flags = CU_MEM_ACCESS_FLAGS_PROT_READWRITE;
    return driver().set_access(va, bytes, &acc, 1) == CUDA_SUCCESS;
}

bool budget_take(kv_budget *b, uint64_t bytes)
{
    if (!b) return true;
    uint64_t cur = b->used.load();
    do {
        if (cur + bytes > b->limit) return false;
    } while (!b->used.compare_exchange_weak(cur, cur + bytes));
    return true;
}

void budget_give(kv_budget *b, uint64_t bytes)
{
    if (b) b->used.fetch_sub(bytes);
}

uint64_t gcd64(uint64_t a, uint64_t b) { return b ? gcd64(b, a % b) : a; }

}  // namespace

// The guard handle of a CUDA-backed pool lives in vmm.ctx.
int kvp_vmm_map_chunk(kv_pool *p)
{
    kv_vmm_state &v = p->vmm;
    if (v.unmapped_order.empty()) return KV_ERR_OUT_OF_BLOCKS;
    if (v.physical_limit && v.mapped_bytes + v.chunk_bytes > v.physical_limit) return KV_ERR_OUT_OF_BLOCKS;
    if (!budget_take(v.budget, v.chunk_bytes)) return KV_ERR_OUT_OF_BLOCKS;
    const int32_t c = v.unmapped_order.back();
    const uint64_t off = (uint64_t)c * v.chunk_bytes;
    if (v.map_fn) {
        if (v.map_fn(v.ctx, off, v.chunk_bytes) != 0) {
            budget_give(v.budget, v.chunk_bytes);
            return KV_ERR_OUT_OF_BLOCKS;
        }
    } else {
        const Driver &d = driver();
        CudaBacking *cb = static_cast<CudaBacking *>(v.ctx);
        CUmemAllocationProp prop = device_prop(p->device);
        CUmemGenericAllocationHandle h = 0;
        if (d.create(&h, v.chunk_bytes, &prop, 0) != CUDA_SUCCESS) {  // out of device memory
            budget_give(v.budget, v.chunk_bytes);
            return KV_ERR_OUT_OF_BLOCKS;
        }
        const CUdeviceptr va = chunk_va(p, c);
        bool ok = d.unmap(va, v.chunk_bytes) == CUDA_SUCCESS;  // the guard
        ok = ok && d.map(va, v.chunk_bytes, 0, h, 0) == CUDA_SUCCESS && set_rw(p, va, v.chunk_bytes);
        if (!ok) {
            // put the guard back so the range stays backed
            d.unmap(va, v.chunk_bytes);
            if (cb && cb->guard_ok && d.map(va, v.chunk_bytes, 0, cb->guard, 0) == CUDA_SUCCESS)
                set_rw(p, va, v.chunk_bytes);
            d.release(h);
            budget_give(v.budget, v.chunk_bytes);
            return KV_ERR_CUDA;
        }
        v.handle[(size_t)c] = (uint64_t)h;
    }
    v.unmapped_order.pop_back();
    v.mapped[(size_t)c] = 1;
    v.mapped_bytes += v.chunk_bytes;
    // its superpages become free capacity, popping in ascending order or, with
    // a shuffle seed, in a seeded order
    const int32_t spc = v.supers_per_chunk;
    std::vector<int32_t> sps((size_t)spc);
    for (int32_t i = 0; i < spc; ++i) sps[(size_t)i] = c * spc + i;
    if (p->desc.shuffle_seed) {
        for (int32_t i = spc - 1; i > 0; --i) {
            uint64_t z = (p->shuffle_state += 0x9E3779B97F4A7C15ull);
            z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
            z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
            z ^= z >> 31;
            std::swap(sps[(size_t)i], sps[(size_t)(z % (uint64_t)(i + 1))]);
        }
    }
    for (auto it = sps.rbegin(); it != sps.rend(); ++it) p->super_free.push_back(*it);
    v.free_supers[(size_t)c] = spc;
    return KV_OK;
}

int kvp_vmm_unmap_chunk(kv_pool *p, int64_t c)
{
    kv_vmm_state &v = p->vmm;
    const uint64_t off = (uint64_t)c * v.chunk_bytes;
    if (v.map_fn) {
        if (v.unmap_fn(v.ctx, off, v.chunk_bytes) != 0) return KV_ERR_CUDA;
    } else {
        const Driver &d = driver();
        CudaBacking *cb = static_cast<CudaBacking *>(v.ctx);
        const CUdeviceptr va = chunk_va(p, c);
        if (d.unmap(va, v.chunk_bytes) != CUDA_SUCCESS) return KV_ERR_CUDA;
        d.release((CUmemGenericAllocationHandle)v.handle[(size_t)c]);
        v.handle[(size_t)c] = 0;
        if (!cb || !cb->guard_ok || d.map(va, v.chunk_bytes, 0, cb->guard, 0) != CUDA_SUCCESS ||
            !set_rw(p, va, v.chunk_bytes))
            return KV_ERR_CUDA;
    }
    v.mapped[(size_t)c] = 0;
    v.free_supers[(size_t)c] = 0;
    v.mapped_bytes -= v.chunk_bytes;
    budget_give(v.budget, v.chunk_bytes);
    v.unmapped_order.push_back((int32_t)c);
    return KV_OK;
}

void kvp_vmm_release_all(kv_pool *p)
{
    kv_vmm_state &v = p->vmm;
    if (v.map_fn) {
        for (int64_t c = 0; c < v.n_chunks; ++c)
            if (v.mapped[(size_t)c]) {
                v.unmap_fn(v.ctx, (uint64_t)c * v.chunk_bytes, v.chunk_bytes);
                budget_give(v.budget, v.chunk_bytes);
            }
    } else {
        const Driver &d = driver();
        CudaBacking *cb = static_cast<CudaBacking *>(v.ctx);
        cudaDeviceSynchronize();  // no kernel may still read the range
        for (int64_t c = 0; c < v.n_chunks; ++c) {
            d.unmap(chunk_va(p, c), v.chunk_bytes);
            if (v.mapped[(size_t)c]) {
                d.release((CUmemGenericAllocationHandle)v.handle[(size_t)c]);
                budget_give(v.budget, v.chunk_bytes);
            }
        }
        if (cb && cb->guard_ok) d.release(cb->guard);
        if (v.owns_va) d.addr_free((CUdeviceptr)(uintptr_t)p->desc.device_base, v.va_bytes);
        delete cb;
        v.ctx = nullptr;
    }
    if (v.budget) v.budget->pools.fetch_sub(1);
    v.mapped_bytes = 0;
}

extern "C" {

int kv_budget_create(uint64_t limit_bytes, kv_budget **out)
{
    if (!out) return KV_ERR_INVALID_ARG;
    kv_budget *b = new kv_budget();
    b->limit = limit_bytes;
    *out = b;
    return KV_OK;
}

int kv_budget_destroy(kv_budget *b)
{
    if (!b || b->pools.load() != 0) return KV_ERR_INVALID_ARG;
    delete b;
    return KV_OK;
}

int kv_budget_used(const kv_budget *b, uint64_t *used)
{
    if (!b || !used) return KV_ERR_INVALID_ARG;
    *used = b->used.load();
    return KV_OK;
}

int kv_pool_create_vmm(const kv_pool_desc *desc, const kv_vmm_desc *vmm, kv_pool **out_pool)
{
    if (!desc || !vmm || !out_pool) return KV_ERR_INVALID_ARG;
    *out_pool = nullptr;
    if ((!vmm->map_fn) != (!vmm->unmap_fn)) return KV_ERR_INVALID_ARG;
    const bool cuda_backend = vmm->map_fn == nullptr;
    if (cuda_backend && desc->device_base) return KV_ERR_INVALID_ARG;  // the library reserves the range
    if (!cuda_backend && (!desc->device_base || vmm->chunk_bytes == 0)) return KV_ERR_INVALID_ARG;

    // geometry first (page, superpage), from the same rules as a fixed pool
    kv_pool_desc d = *desc;
    uint64_t chunk = vmm->chunk_bytes;
    const Driver *drv = nullptr;
    int device = vmm->device;
    if (cuda_backend) {
        drv = &driver();
        if (!drv->ok) return KV_ERR_CUDA;
        if (cudaSetDevice(device) != cudaSuccess || cudaFree(nullptr) != cudaSuccess) return KV_ERR_CUDA;
        CUmemAllocationProp prop = device_prop(device);
        size_t g = 0;
        if (drv->granularity(&g, &prop, CU_MEM_ALLOC_GRANULARITY_MINIMUM) != CUDA_SUCCESS || g == 0)
            return KV_ERR_CUDA;
        if (!chunk) chunk = g;
        if (chunk % g) return KV_ERR_INVALID_ARG;
        d.device_base = reinterpret_cast<void *>(uintptr_t(1) << 40);  // placeholder for validation
    }
    kv_pool *p = nullptr;
    int rc = kv_pool_create(&d, &p);
    if (rc) return rc;
    const uint64_t super_bytes = (uint64_t)p->super_pages * p->page_bytes;
    // a chunk holds whole superpages
    chunk = chunk / gcd64(chunk, super_bytes) * super_bytes;
    const int64_t supers = p->n_pages / p->super_pages;
    const int32_t spc = (int32_t)(chunk / super_bytes);
    const int64_t n_chunks = supers / spc;
    if (n_chunks < 1 || (vmm->physical_limit && vmm->physical_limit < chunk)) {
        kv_pool_destroy(p);
        return KV_ERR_INVALID_ARG;
    }
    // the pool covers whole chunks only
    p->n_pages = n_chunks * spc * p->super_pages;
    p->refcnt.assign((size_t)p->n_pages, 0);
    p->owner.assign((size_t)p->n_pages, (int8_t)-1);
    p->tally.assign((size_t)p->n_pages, 0);
    p->super_free.clear();
    kv_vmm_state &v = p->vmm;
    v.active = true;
    v.chunk_bytes = chunk;
    v.supers_per_chunk = spc;
    v.n_chunks = n_chunks;
    v.mapped.assign((size_t)n_chunks, 0);
    v.handle.assign((size_t)n_chunks, 0);
    v.free_supers.assign((size_t)n_chunks, 0);
    v.physical_limit = vmm->physical_limit;
    v.map_fn = vmm->map_fn;
    v.unmap_fn = vmm->unmap_fn;
    v.ctx = vmm->ctx;
    p->shuffle_state = desc->shuffle_seed;
    // chunks are mapped lowest first, or in a seeded order
    std::vector<int32_t> order((size_t)n_chunks);
    std::iota(order.begin(), order.end(), 0);
    if (desc->shuffle_seed) {
        for (int64_t i = n_chunks - 1; i > 0; --i) {
            uint64_t z = (p->shuffle_state += 0x9E3779B97F4A7C15ull);
            z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
            z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
            z ^= z >> 31;
            std::swap(order[(size_t)i], order[(size_t)(z % (uint64_t)(i + 1))]);
        }
    }
    v.unmapped_order.assign(order.rbegin(), order.rend());

    if (cuda_backend) {
        p->device = device;
        v.va_bytes = (uint64_t)n_chunks * chunk;
        CUdeviceptr va = 0;
        if (drv->reserve(&va, v.va_bytes, chunk, 0, 0) != CUDA_SUCCESS) {
            v.active = false;
            kv_pool_destroy(p);
            return KV_ERR_CUDA;
        }
        v.owns_va = true;
        p->desc.device_base = reinterpret_cast<void *>((uintptr_t)va);
        auto *cb = new CudaBacking();
        v.ctx = cb;
        CUmemAllocationProp prop = device_prop(device);
        bool ok = drv->create(&cb->guard, chunk, &prop, 0) == CUDA_SUCCESS;
        cb->guard_ok = ok;
        for (int64_t c = 0; ok && c < n_chunks; ++c) ok = drv->map(chunk_va(p, c), chunk, 0, cb->guard, 0) == CUDA_SUCCESS;
        ok = ok && set_rw(p, va, v.va_bytes);
        if (!ok) {
            kv_pool_destroy(p);  // unmaps what was mapped, frees the range
            return KV_ERR_CUDA;
        }
        cudaMemset(reinterpret_cast<void *>((uintptr_t)va), 0, chunk);  // guard reads as zeros
    }
    v.budget = vmm->budget;  // attached last: a failed creation never touched it
    if (v.budget) v.budget->pools.fetch_add(1);
    *out_pool = p;
    return KV_OK;
}

int kv_pool_get_base(const kv_pool *p, void **base)
{
    if (!p || !base) return KV_ERR_INVALID_ARG;
    *base = p->desc.device_base;
    return KV_OK;
}

}  // extern "C"
