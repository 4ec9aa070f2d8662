// Inline-PTX wrappers for the sm_100-family (sm_103a) tensor-core path:
// mbarriers, tensor memory (TMEM) allocation and loads, tcgen05.mma with
// shared-memory matrix descriptors, and the proxy fences between them.
#pragma once

#include <stdint.h>

namespace salt {

// ---------------------------------------------------------------- mbarrier
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;\n" ::"r"(bar), "r"(count));
}
// make barrier initialisation visible to the async proxy and the cluster
__device__ __forceinline__ void mbar_fence_init() { asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory"); }

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// Bounded wait for the phase of the given parity: gives up after a fixed
// number of polls (each try_wait suspends for a bounded time) and returns
// false, so a lost arrival can never hang the GPU.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity)
{
    for (int i = 0; i < (1 << 20); ++i)
        if (mbar_try_wait(bar, parity)) return true;
    return false;
}

// ---------------------------------------------------------------- TMEM
// Allocate ncols (power of two, >= 32) tensor-memory columns; one whole warp
// executes it; the TMEM address lands in shared memory at dst.
__device__ __forceinline__ void tmem_alloc(uint32_t dst, uint32_t ncols)
{
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(dst), "r"(ncols));
}
__device__ __forceinline__ void tmem_relinquish()
{
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n" ::);
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols)
{
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(taddr), "r"(ncols));
}
// 32 lanes x 16 columns of 32-bit values: thread i of the warp gets lane
// (warp's lane quarter base + i), columns [col, col + 16)
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16])
{
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];\n"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory"); }

// ordering of tcgen05 operations around thread synchronisation
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory"); }
// generic-proxy shared-memory writes (cp.async, st.shared) -> visible to the async proxy (tcgen05.mma)
__device__ __forceinline__ void fence_async_smem() { asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory"); }

// ---------------------------------------------------------------- UMMA
// Shared-memory matrix descriptor of a K-major operand in the 128-byte
// swizzle layout: rows of 128 bytes (64 bf16 of K), 8-row atoms of 1024
// bytes (stride byte offset), the 16-byte chunk index XORed with the row
// index within the atom.  The tile base must be 1024-byte aligned; moving
// along K by 16 elements adds 32 bytes to the start address.
__device__ __forceinline__ uint64_t sdesc_kmajor_sw128(uint32_t saddr)
{
    return (uint64_t)((saddr & 0x3FFFFu) >> 4)      // start address >> 4, bits [0, 14)
           | ((uint64_t)1 << 16)                     // leading byte offset (unused for this layout)
           | ((uint64_t)(1024 >> 4) << 32)           // stride byte offset: 8 rows x 128 B
           | ((uint64_t)1 << 46)                     // descriptor version of the sm_100 family
           | ((uint64_t)2 << 61);                    // layout: 128-byte swizzle
}

// Shared-memory matrix descriptor of an MN-major operand in the 128-byte
// swizzle layout: rows of 128 bytes hold 64 consecutive MN elements of one K
// index, 8-row (8 K) atoms of 1024 bytes, the same address-based swizzle as
// above.  Used with an MN extent of one atom (64), so only the stride between
// 8-deep K groups (1024 bytes) is ever applied; both offset fields carry it.
// Moving along K by 16 adds 2048 bytes to the start address.
__device__ __forceinline__ uint64_t sdesc_mnmajor_sw128(uint32_t saddr)
{
    return (uint64_t)((saddr & 0x3FFFFu) >> 4)      // start address >> 4
           | ((uint64_t)(1024 >> 4) << 16)           // leading byte offset
           | ((uint64_t)(1024 >> 4) << 32)           // stride byte offset
           | ((uint64_t)1 << 46)                     // descriptor version of the sm_100 family
           | ((uint64_t)2 << 61);                    // layout: 128-byte swizzle
}

// Instruction descriptor of kind::f16: bf16 x bf16 -> fp32, both operands
// K-major, D of M x N.
__host__ __device__ constexpr uint32_t idesc_bf16_f32(int M, int N)
{
    return (1u << 4)                     // D format: f32
           | (1u << 7)                   // A format: bf16
           | (1u << 10)                  // B format: bf16
           | ((uint32_t)(N >> 3) << 17)  // N / 8
           | ((uint32_t)(M >> 4) << 24); // M / 16
}

// The same with B MN-major (bit 16: B transposed).
__host__ __device__ constexpr uint32_t idesc_bf16_f32_bmn(int M, int N) { return idesc_bf16_f32(M, N) | (1u << 16); }

// D[tmem] (+)= A * B^T for one K=16 step, issued by a single thread.
__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                          uint32_t accumulate)
{
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(
            d_tmem),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate));
}
// arrive on the mbarrier once every tcgen05 operation issued so far by this thread has completed
__device__ __forceinline__ void umma_commit(uint32_t bar)
{
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(bar)
                 : "memory");
}

}  // namespace salt
