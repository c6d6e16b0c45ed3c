// Device side of the persistent tile scheduler shared by both kernels.
//
// Work items are handed out in a fixed global order by an atomic ticket.  Every
// dependency of an item (the previous fused stage of its tile, the tile that
// last used its scratch slot, or all group-1 tiles of its frame) consists of
// items with smaller tickets, and a CTA only takes a ticket while it runs, so
// the smallest unfinished ticket can always make progress.  Waits are bounded
// by a wall-clock limit: when it runs out the kernel records
// MAFAT_DEV_TIMEOUT, raises the abort word and every later wait returns at
// once, so the launch always ends.
#pragma once
#include "../../include/mafat.h"
#include "kernels.h"

namespace mafat_dev {

__device__ __forceinline__ uint64_t globaltimer_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ uint32_t ld_acquire_u32(const uint32_t* p) {
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ void red_release_add(uint32_t* p, uint32_t v) {
    asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ void fence_proxy_async_global() {
    asm volatile("fence.proxy.async.global;" ::: "memory");
}

__device__ __forceinline__ void record_status(uint32_t* ctr, uint32_t code) {
    atomicCAS(&ctr[MAFAT_CTR_STATUS], 0u, code);
    atomicExch(&ctr[MAFAT_CTR_ABORT], 1u);
}

__device__ __forceinline__ bool aborted(const uint32_t* ctr) {
    return *(volatile const uint32_t*)&ctr[MAFAT_CTR_ABORT] != 0u;
}

// Wait until ctr[idx] >= target (acquire), bounded by timeout_ns.
__device__ __forceinline__ void wait_counter(uint32_t* ctr, int idx, int target, int64_t timeout_ns) {
    if (idx < 0) return;
    const uint32_t* p = ctr + idx;
    if (ld_acquire_u32(p) >= (uint32_t)target) return;
    uint64_t t0 = globaltimer_ns();
    uint32_t ns = 32;
    while (true) {
        if (ld_acquire_u32(p) >= (uint32_t)target) return;
        if (aborted(ctr)) return;
        if ((int64_t)(globaltimer_ns() - t0) > timeout_ns) {
            record_status(ctr, MAFAT_DEV_TIMEOUT);
            return;
        }
        __nanosleep(ns);
        if (ns < 128) ns <<= 1;  // a short cap: a completion is seen within ~0.1 us
    }
}

__device__ __forceinline__ uint32_t ld_relaxed_u32(const uint32_t* p) {
    uint32_t v;
    asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// Wait for every entry of a task's dependency list (halo reuse: the tasks of the previous
// layer around it).  The counters are read together, eight at a time (independent relaxed
// loads, one round trip), and only those still short are polled; a fence then gives the
// reads acquire order.  Out of line: only halo-reuse plans call it, and its unrolled polls
// would otherwise sit in every plan's producer code (measured on GB300, with the generic
// gather also out of line: 608x608 110.1 -> 109.4 us per frame).
static __device__ __noinline__ void wait_dep_list(uint32_t* ctr, const MafatDepDev* deps, int first, int count,
                                                  int64_t timeout_ns) {
    for (int d0 = 0; d0 < count; d0 += 8) {
        const int n = min(8, count - d0);
        MafatDepDev e[8];
        uint32_t v[8];
#pragma unroll
        for (int i = 0; i < 8; ++i)
            if (i < n) e[i] = deps[first + d0 + i];
#pragma unroll
        for (int i = 0; i < 8; ++i)
            if (i < n) v[i] = ld_relaxed_u32(ctr + e[i].ctr);
#pragma unroll
        for (int i = 0; i < 8; ++i)
            if (i < n && v[i] < (uint32_t)e[i].target) wait_counter(ctr, e[i].ctr, e[i].target, timeout_ns);
    }
    asm volatile("fence.acq_rel.gpu;" ::: "memory");
}

// Wait for both dependencies of an item; afterwards the data they published is
// visible to this thread's generic and async-proxy (TMA) reads.
__device__ __forceinline__ void wait_item_deps(uint32_t* ctr, const MafatItemDev& it, int64_t timeout_ns) {
    wait_counter(ctr, it.dep0, it.dep0_target, timeout_ns);
    wait_counter(ctr, it.dep1, it.dep1_target, timeout_ns);
    fence_proxy_async_global();
}

// Publish completion of an item (call once, after all of its stores are
// ordered before this thread by a CTA-level barrier).
// A release at gpu scope orders every write this thread has observed before it,
// including the other threads' writes ordered before it by a CTA barrier or an
// mbarrier (releases are cumulative), so no separate fence is needed.
__device__ __forceinline__ void publish_counters(uint32_t* ctr, int done_ctr, int extra_ctr) {
    red_release_add(ctr + done_ctr, 1u);
    if (extra_ctr >= 0) red_release_add(ctr + extra_ctr, 1u);
}

__device__ __forceinline__ void publish_item(uint32_t* ctr, const MafatItemDev& it, int done_ctr) {
    if (it.flags & 1) return;  // test hook: never published
    publish_counters(ctr, done_ctr, it.extra_ctr);
}

__device__ __forceinline__ uint32_t smid() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%smid;" : "=r"(r));
    return r;
}

// Trace record of an item: {ticket taken, deps satisfied, accumulator ready, published, SM}.
__device__ __forceinline__ void trace_put(unsigned long long* tr, int ticket, int field, uint64_t v) {
    if (tr) tr[(size_t)ticket * MAFAT_TRACE_WORDS + field] = v;
}

// Called by every thread of a CTA after its last use of the counters: the last
// CTA of the launch to get here zeroes the counter block (all but the status
// word) for the next run on the same stream.
__device__ __forceinline__ void finish_cta(uint32_t* ctr, int n_ctr) {
    __shared__ int s_last;
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        const uint32_t done = atomicAdd(&ctr[MAFAT_CTR_EXIT], 1u);
        s_last = (done == gridDim.x - 1) ? 1 : 0;
        __threadfence();
    }
    __syncthreads();
    if (!s_last) return;
    // the next launch on the stream starts after this one has completed, so these stores
    // need no fence of their own
    for (int i = threadIdx.x; i < n_ctr; i += blockDim.x)
        if (i != MAFAT_CTR_STATUS) ctr[i] = 0u;
}

}  // namespace mafat_dev
