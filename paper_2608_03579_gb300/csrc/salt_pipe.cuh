// Inline-PTX wrappers of the warp-specialised pipelines (sm_100 family):
// mbarrier arrivals with the semantics each hand-off needs, TMA tile loads
// completing on an mbarrier by byte count, named barriers, proxy fences and
// programmatic dependent launch.
#pragma once

#include <cuda.h>
#include <stdint.h>

namespace salt {

// arrive on the mbarrier once all of this thread's earlier cp.async copies have landed
__device__ __forceinline__ void cp_async_arrive_noinc(uint32_t bar)
{
    asm volatile("cp.async.mbarrier.arrive.noinc.shared::cta.b64 [%0];\n" ::"r"(bar) : "memory");
}
// Relaxed arrive: orders nothing by itself, so it does not wait for this
// thread's global stores.  Used where what the barrier guards is already
// ordered: shared-memory values consumed into registers before the arrive,
// tensor-memory loads completed by tcgen05.wait::ld.
__device__ __forceinline__ void mbar_arrive_relaxed(uint32_t bar)
{
    asm volatile("mbarrier.arrive.relaxed.cta.shared::cta.b64 _, [%0];\n" ::"r"(bar) : "memory");
}
// Arrive with release semantics (CTA scope): shared-memory writes that
// happen before it are visible to a thread whose wait sees the phase complete.
__device__ __forceinline__ void mbar_arrive_release(uint32_t bar)
{
    asm volatile("mbarrier.arrive.release.cta.shared::cta.b64 _, [%0];\n" ::"r"(bar) : "memory");
}
// arrive on the mbarrier, adding `bytes` to the transaction count its phase waits for
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n" ::"r"(bar), "r"(bytes) : "memory");
}
// 2-D TMA tile load (coordinates in elements, x first) completing on bar by bytes
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap *map, int x, int y, uint32_t bar)
{
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];\n" ::"r"(dst),
        "l"(map), "r"(x), "r"(y), "r"(bar)
        : "memory");
}
// barrier among the first n threads of the CTA (n a multiple of 32), id 1..15
__device__ __forceinline__ void named_sync(int id, int n) { asm volatile("bar.sync %0, %1;\n" ::"r"(id), "r"(n) : "memory"); }
// named barrier that also ANDs a predicate over its n threads: every thread
// gets true only if all of them passed true
__device__ __forceinline__ bool named_sync_and(int id, int n, bool v)
{
    uint32_t r;
    asm volatile("{\n .reg .pred p, q;\n setp.ne.u32 q, %1, 0;\n bar.red.and.pred p, %2, %3, q;\n selp.u32 %0, 1, 0, p;\n}\n"
                 : "=r"(r)
                 : "r"((uint32_t)v), "r"(id), "r"(n)
                 : "memory");
    return r != 0;
}
// order global data this thread observed through the generic proxy before
// async-proxy (TMA) reads of it
__device__ __forceinline__ void fence_proxy_async_global() { asm volatile("fence.proxy.async.global;\n" ::: "memory"); }

__device__ __forceinline__ void pdl_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;\n" ::); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;\n" ::: "memory"); }

}  // namespace salt
