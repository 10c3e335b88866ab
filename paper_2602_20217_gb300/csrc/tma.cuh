// Asynchronous-copy helpers shared by the streaming kernels: mbarriers, 2-D
// TMA loads, programmatic dependent launch, and bounded waits.  Every wait
// here gives up after a time limit instead of spinning forever; the caller
// records the failure in the device status word and returns.
#pragma once

#include <cuda.h>
#include <stdint.h>

#include "common.cuh"

namespace ks {

constexpr uint64_t kWaitLimitNs = 2000000000ull;  // 2 s: only a broken copy or peer waits this long

KS_DEV uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

KS_DEV void mbar_init(uint64_t* bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
KS_DEV void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
                 : "memory");
}
KS_DEV void mbar_arrive(uint64_t* bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
// 2-D tiled TMA load of the box at (x, y) of `map` (a tensor map in kernel
// parameter or global memory) into shared memory; completes on `bar`.
KS_DEV void tma_2d(void* dst, const CUtensorMap* map, int x, int y, uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], "
        "[%4];" ::"r"(smem_u32(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar))
        : "memory");
}
KS_DEV void tma_3d(void* dst, const CUtensorMap* map, int x, int y, int z, uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], "
        "[%5];" ::"r"(smem_u32(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(smem_u32(bar))
        : "memory");
}
KS_DEV void grid_dependency_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
KS_DEV void grid_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
KS_DEV uint64_t global_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
    return t;
}
// Wait for the mbarrier phase with the given parity; false after limit_ns.
KS_DEV bool mbar_wait(uint64_t* bar, uint32_t parity, uint64_t limit_ns) {
    const uint32_t b = smem_u32(bar);
    uint64_t t0 = 0;
    for (uint32_t i = 0;; ++i) {
        uint32_t ok;
        asm volatile(
            "{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
            : "=r"(ok)
            : "r"(b), "r"(parity)
            : "memory");
        if (ok) return true;
        if (i == 0) t0 = global_ns();
        else if ((i & 63) == 0 && global_ns() - t0 > limit_ns) return false;
    }
}
// Barrier of the four consumer warps (named barrier 1) that also ORs a flag.
KS_DEV bool consumers_or(bool v) {
    uint32_t r;
    asm volatile(
        "{ .reg .pred p, q; setp.ne.u32 p, %1, 0; bar.red.or.pred q, 1, 128, p; selp.u32 %0, 1, 0, q; }"
        : "=r"(r)
        : "r"((uint32_t)v)
        : "memory");
    return r != 0;
}
KS_DEV void consumers_sync() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

KS_DEV int ld_acquire(const int* p) {
    int v;
    asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
// Wait until *p >= target (another CTA of the same grid raises it); false
// after limit_ns.
KS_DEV bool wait_at_least(const int* p, int target, uint64_t limit_ns) {
    if (ld_acquire(p) >= target) return true;
    const uint64_t t0 = global_ns();
    for (;;) {
        __nanosleep(64);
        if (ld_acquire(p) >= target) return true;
        if (global_ns() - t0 > limit_ns) return false;
    }
}
// Order this thread's earlier generic-proxy writes/reads before its later
// asynchronous-proxy (TMA) operations on global memory.
KS_DEV void fence_proxy_async_global() { asm volatile("fence.proxy.async.global;" ::: "memory"); }

}  // namespace ks
