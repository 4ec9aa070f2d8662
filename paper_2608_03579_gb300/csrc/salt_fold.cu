// Fold of a scaled centroid into a base weight (Section "Multi-Tenant
// Serving": a much-used centroid, already scaled, may be merged into the
// base weights when a node starts; its requests then apply residuals only).
//
//     W[Mdim][Ndim] += scale * P^T Q,   P = [rc][Mdim], Q = [rc][Ndim]
//
// with P and Q the pinned centroid factors as stored (row-major, the long
// dimension contiguous): for W[d_in][d_out], P = At_c and Q = B_c; for
// W[d_out][d_in], P = B_c and Q = At_c.  K = rc <= 64: a rank-rc update of a
// large matrix, bound by reading and writing W once.
//
// Items are (128-row tile of W, 64 columns); each CTA (two per SM) takes a
// contiguous range of them, so it mostly stays on one row tile.  Per row tile the CTA
// transposes P's 128 columns into a K-major 128-byte-swizzled tile (the
// UMMA A operand, K padded to a multiple of 16 with zeros); per item the Q
// columns (MN-major, as they lie in memory) and the W tile stream through a
// cp.async ring.  One thread issues D[128 x 64] = P_tile^T Q_chunk into one
// of two tensor-memory accumulators, the next item's MMAs before this
// item's epilogue; the epilogue (one W row a thread, half of the columns a
// warp) adds scale * D to W in fp32, rounds once to bf16 and writes the
// tile back in shared memory, from where all threads store it coalesced.
#include "salt_async.cuh"
#include "salt_internal.cuh"
#include "salt_tcgen05.cuh"

namespace salt {
namespace {

constexpr int FOLD_THREADS = 256;
constexpr int FOLD_TM = 128;                          // W rows per tile (UMMA M)
constexpr int FOLD_NC = 64;                           // W columns per item (UMMA N)
constexpr int FOLD_STAGES = 3;
constexpr int FOLD_CTAS_PER_SM = 2;                   // one CTA's epilogue overlaps the other's copies
constexpr int FOLD_Q_BYTES = 64 * 128;                // [K <= 64][64 columns], MN-major
constexpr int FOLD_W_BYTES = FOLD_TM * 128;           // [128 rows][64 columns], swizzled rows
constexpr int FOLD_STAGE_BYTES = FOLD_Q_BYTES + FOLD_W_BYTES;
constexpr int FOLD_A_BYTES = FOLD_TM * 128;           // [128 rows][K <= 64], K-major
constexpr int FOLD_SMEM = 1024 + 2 * FOLD_A_BYTES + FOLD_STAGES * FOLD_STAGE_BYTES;
static_assert(FOLD_CTAS_PER_SM * (FOLD_SMEM + 1024) <= 228 * 1024, "two fold CTAs must fit one SM");
static_assert(SALT_MAX_CENTROID_RANK <= 64, "K of the fold is one 128-byte row");

struct FoldParams {
    const uint16_t *P;  // [rc][Mdim]
    const uint16_t *Q;  // [rc][Ndim]
    uint16_t *W;        // [Mdim][Ndim]
    int32_t Mdim, Ndim, rc;
    float scale;
    uint32_t *err;
};

__global__ void __launch_bounds__(FOLD_THREADS, FOLD_CTAS_PER_SM) salt_fold_kernel(const __grid_constant__ FoldParams p)
{
    extern __shared__ __align__(128) uint8_t smem_raw[];
    uint8_t *base = smem_raw + ((1024 - (smem_u32(smem_raw) & 1023)) & 1023);
    const uint32_t a32 = smem_u32(base);                        // two A tiles
    const uint32_t st32 = a32 + 2 * FOLD_A_BYTES;               // the ring
    __shared__ uint64_t mma_bar[2];
    __shared__ uint32_t tmem_slot;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int Mdim = p.Mdim, Ndim = p.Ndim, rc = p.rc;
    const int n_ct = (Ndim + FOLD_NC - 1) / FOLD_NC;
    const int64_t items = (int64_t)((Mdim + FOLD_TM - 1) / FOLD_TM) * n_ct;
    const int64_t i0 = items * blockIdx.x / gridDim.x, i1 = items * (blockIdx.x + 1) / gridDim.x;
    if (i0 >= i1) return;  // the same for every thread of the CTA
    const int n_my = (int)(i1 - i0);
    const int kpad = (rc + 15) & ~15;

    if (warp == 0) {
        tmem_alloc(smem_u32(&tmem_slot), 128);  // two 64-column accumulators
        tmem_relinquish();
    }
    if (tid == 0) {
        mbar_init(smem_u32(&mma_bar[0]), 1);
        mbar_init(smem_u32(&mma_bar[1]), 1);
        mbar_fence_init();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;

    auto stage = [&](int j) { return st32 + (uint32_t)(j % FOLD_STAGES) * FOLD_STAGE_BYTES; };
    // Q columns and W tile of item i0 + j into its stage (rows >= rc and
    // columns >= Ndim of Q, rows >= Mdim and columns >= Ndim of W zero-filled)
    auto load_item = [&](int j) {
        const int64_t it = i0 + j;
        const int m0 = (int)(it / n_ct) * FOLD_TM, n0 = (int)(it % n_ct) * FOLD_NC;
        const uint32_t sq = stage(j), sw = sq + FOLD_Q_BYTES;
        for (int idx = tid; idx < kpad * 8; idx += FOLD_THREADS) {
            const int k = idx >> 3, c = idx & 7, n = n0 + c * 8;
            const bool ok = k < rc && n < Ndim;
            cp_async16(sq + swz128(k, c), ok ? p.Q + (int64_t)k * Ndim + n : p.Q, ok);
        }
        for (int idx = tid; idx < FOLD_TM * 8; idx += FOLD_THREADS) {
            const int r = idx >> 3, c = idx & 7, m = m0 + r, n = n0 + c * 8;
            const bool ok = m < Mdim && n < Ndim;
            cp_async16(sw + swz128(r, c), ok ? p.W + (int64_t)m * Ndim + n : p.W, ok);
        }
    };
    // P^T of row tile rt into A tile `buf`: element (m, k) at row m, K column k
    // (16-byte chunk k / 8 swizzled by m % 8); K columns in [rc, kpad) zero
    auto build_a = [&](int rt, int buf) {
        uint8_t *A = base + buf * FOLD_A_BYTES;
        const int m0 = rt * FOLD_TM;
        for (int idx = tid; idx < kpad * (FOLD_TM / 8); idx += FOLD_THREADS) {
            const int k = idx / (FOLD_TM / 8), c8 = idx - k * (FOLD_TM / 8), m = m0 + c8 * 8;
            uint4 v = make_uint4(0u, 0u, 0u, 0u);
            if (k < rc && m < Mdim) v = *reinterpret_cast<const uint4 *>(p.P + (int64_t)k * Mdim + m);
            const uint16_t *h = reinterpret_cast<const uint16_t *>(&v);
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                const int r = c8 * 8 + e;
                *reinterpret_cast<uint16_t *>(A + r * 128 + ((((k >> 3) ^ (r & 7))) << 4) + (k & 7) * 2) = h[e];
            }
        }
        fence_async_smem();
    };
    const uint32_t idesc = idesc_bf16_f32_bmn(FOLD_TM, FOLD_NC);
    auto issue_mma = [&](int j, int buf) {  // thread 0
        tc_fence_after();
        const uint32_t a = a32 + buf * FOLD_A_BYTES, q = stage(j);
        for (int kk = 0; kk < kpad / 16; ++kk)
            umma_bf16(tmem + (uint32_t)(j & 1) * FOLD_NC, sdesc_kmajor_sw128(a + kk * 32),
                      sdesc_mnmajor_sw128(q + kk * 2048), idesc, kk > 0 ? 1u : 0u);
        umma_commit(smem_u32(&mma_bar[j & 1]));
    };

    // prefetch; one commit group per item slot keeps the group count in step
    for (int j = 0; j < FOLD_STAGES; ++j) {
        if (j < n_my) load_item(j);
        cp_async_commit();
    }
    int rt_cur = (int)(i0 / n_ct), abuf = 0;
    build_a(rt_cur, abuf);
    cp_async_wait_dyn(FOLD_STAGES - 1);  // item 0 landed
    fence_async_smem();
    __syncthreads();
    if (tid == 0) issue_mma(0, abuf);
    bool ok_all = true;

    for (int j = 0; j < n_my; ++j) {
        // the next item's MMAs first, so they overlap this item's epilogue
        if (j + 1 < n_my) {
            const int rt = (int)((i0 + j + 1) / n_ct);
            int nbuf = abuf;
            if (rt != rt_cur) {
                // the other A tile was last read by MMAs whose results were consumed already
                nbuf = abuf ^ 1;
                build_a(rt, nbuf);
            }
            cp_async_wait_dyn(FOLD_STAGES - 2);  // items <= j + 1 landed
            fence_async_smem();
            __syncthreads();
            if (tid == 0) issue_mma(j + 1, nbuf);
            rt_cur = rt;
            abuf = nbuf;
        }
        // epilogue of item j: one W row a thread, 32 of the 64 columns a warp
        if (!mbar_wait(smem_u32(&mma_bar[j & 1]), (uint32_t)(j >> 1) & 1u)) ok_all = false;
        tc_fence_after();
        const int q = warp & 3, h = warp >> 2, r = q * 32 + lane;
        const int64_t it = i0 + j;
        const int m0 = (int)(it / n_ct) * FOLD_TM, n0 = (int)(it % n_ct) * FOLD_NC;
        const uint32_t sw = stage(j) + FOLD_Q_BYTES;
        uint8_t *swp = base + (sw - a32);
#pragma unroll
        for (int half = 0; half < 2; ++half) {
            uint32_t d[16];
            tmem_ld16(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(j & 1) * FOLD_NC + h * 32 + half * 16, d);
            tmem_ld_wait();
            if (m0 + r < Mdim) {
#pragma unroll
                for (int pc = 0; pc < 2; ++pc) {
                    const int c = h * 4 + half * 2 + pc;
                    uint4 *w = reinterpret_cast<uint4 *>(swp + swz128(r, c));
                    uint4 v = *w;
                    const float *f = reinterpret_cast<const float *>(d) + pc * 8;
                    v.x = add_bf16x2(v.x, p.scale * f[0], p.scale * f[1]);
                    v.y = add_bf16x2(v.y, p.scale * f[2], p.scale * f[3]);
                    v.z = add_bf16x2(v.z, p.scale * f[4], p.scale * f[5]);
                    v.w = add_bf16x2(v.w, p.scale * f[6], p.scale * f[7]);
                    *w = v;
                }
            }
        }
        tc_fence_before();
        __syncthreads();
        for (int idx = tid; idx < FOLD_TM * 8; idx += FOLD_THREADS) {
            const int rr = idx >> 3, c = idx & 7, m = m0 + rr, n = n0 + c * 8;
            if (m < Mdim && n < Ndim)
                *reinterpret_cast<uint4 *>(p.W + (int64_t)m * Ndim + n) =
                    *reinterpret_cast<const uint4 *>(swp + swz128(rr, c));
        }
        __syncthreads();  // the stage is free again
        if (j + FOLD_STAGES < n_my) load_item(j + FOLD_STAGES);
        cp_async_commit();
    }
    cp_async_wait<0>();
    if (!ok_all) atomicOr(p.err, SALT_DEVERR_TIMEOUT);
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tmem, 128);
}

}  // namespace

cudaError_t launch_fold(const uint16_t *P, const uint16_t *Q, uint16_t *W, int Mdim, int Ndim, int rc, float scale,
                        uint32_t *err, cudaStream_t stream)
{
    static unsigned long long configured = 0;
    int dev = 0, n_sm = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    e = cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    const unsigned long long bit = 1ull << (dev & 63);
    if (!(configured & bit)) {
        e = cudaFuncSetAttribute(salt_fold_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, FOLD_SMEM);
        if (e != cudaSuccess) return e;
        configured |= bit;
    }
    FoldParams p{P, Q, W, Mdim, Ndim, rc, scale, err};
    const int64_t items = (int64_t)((Mdim + FOLD_TM - 1) / FOLD_TM) * ((Ndim + FOLD_NC - 1) / FOLD_NC);
    const int64_t slots = (int64_t)FOLD_CTAS_PER_SM * n_sm;
    const int grid = (int)(items < slots ? items : slots);
    if (grid <= 0) return cudaSuccess;
    salt_fold_kernel<<<grid, FOLD_THREADS, FOLD_SMEM, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace salt
