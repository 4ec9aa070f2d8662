// Base-weight GEMM fused with the SALT delta (Section "Multi-Tenant Serving":
// the served weight is W_final = W_base + gamma * Wbar + delta_i).  For one
// projection:
//
//     y[t, :] = x[t, :] W_base + s_c (x[t] A_c) B_c + s_u (x[t] a_u) b_u
//
// y is written, never read.  The low-rank part reuses the apply path's row
// blocks: a shrink-only launch of the apply kernel leaves every block's V_ext
// tile (scaled and masked as in the apply) in the segments workspace; this
// kernel then runs the GEMM over 128-token tiles in grouped order and, for
// every row block overlapping a tile, adds V_ext * Stack_B into the same
// tensor-memory accumulator: one more group of MMAs whose A operand holds the
// block's V rows at their tile rows and zeros elsewhere.  Tokens with no
// term are in no block and get x W_base alone.
//
// One persistent CTA per SM over the (M tile, N tile) pairs, 12 warps in
// fixed roles:
//   producers (warps 0-6): per 64-wide K chunk, the tile's x rows (gathered
//       through the grouped order, cp.async) and the W tile (TMA: either
//       layout lands in the layout its UMMA descriptor reads); then per
//       overlapping block its V rows and stacked B columns (cp.async);
//   MMA (warp 7): tcgen05.mma into one of two 128-column accumulators;
//   epilogue (warps 8-11): one token row a thread, fp32 -> bf16 (RNE), store.
#include <cuda_bf16.h>

#include <mutex>

#include "salt_async.cuh"
#include "salt_internal.cuh"
#include "salt_pipe.cuh"
#include "salt_tcgen05.cuh"

namespace salt {
namespace {

constexpr int BM = 128;                    // tokens per tile (the UMMA M)
constexpr int BN = 128;                    // output columns per tile
constexpr int BK = 64;                     // K chunk (128-byte rows)
constexpr int NST = 4;                     // K stages in flight
constexpr int X_BYTES = BM * 128;          // x rows of a chunk
constexpr int W_BYTES = BN * 128;          // W tile of a chunk (either layout)
constexpr int STAGE = X_BYTES + W_BYTES;
constexpr int DV_BYTES = 2 * BM * 128;     // delta A operand: V rows, K 0..63 and 64..127
constexpr int DB_BYTES = 2 * S_MAX * 128;  // delta B operand: stacked B rows, N 0..63 and 64..127
constexpr int BASE_THREADS = 384;
constexpr int PW = 7;                      // producer warps
constexpr int PT = 32 * PW;
constexpr int MW = 7;                      // the MMA warp
constexpr int EW0 = 8;                     // first epilogue warp
constexpr int BAR_P = 1;                   // named barrier of the producers

struct BaseInfo {
    uint64_t full[NST], empty[NST];
    uint64_t dfull, dempty;
    uint64_t accf[2], acce[2];
    const uint16_t *bsrc[S_MAX];  // stacked B rows of the current block
    int32_t prow[BM];             // x rows of the current tile (-1: past the batch)
    uint32_t tmem;
};
constexpr size_t BASE_SMEM = 1024 + NST * STAGE + DV_BYTES + DB_BYTES + (sizeof(BaseInfo) + 127) / 128 * 128;
static_assert(BASE_SMEM <= 227 * 1024, "shared memory exceeds the per-block limit");

__device__ __forceinline__ const uint16_t *res_b_row(const BaseParams &p, int e)
{
    const int slot = res_slot(e), rank = res_rank(e), k = res_k(e);
    const uint16_t *base = reinterpret_cast<const uint16_t *>(p.pool + (int64_t)slot * p.slot_stride +
                                                              SALT_BLOB_HEADER_BYTES) + (int64_t)rank * p.res_off;
    return base + (int64_t)rank * p.d_in + (int64_t)k * p.d_out;
}

// Row blocks overlapping grouped positions [m0, m0 + BM): [*b0, *b1).
__device__ __forceinline__ void blocks_of_tile(const BaseParams &p, int n_blk, int m0, int &b0, int &b1)
{
    // first block ending after m0 (blocks lie in grouped order)
    int lo = 0, hi = n_blk;
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        const int end = p.blk[BLK_INTS * mid + BLK_START] + p.blk[BLK_INTS * mid + BLK_LEN];
        if (end <= m0) lo = mid + 1; else hi = mid;
    }
    b0 = lo;
    b1 = lo;
    while (b1 < n_blk && p.blk[BLK_INTS * b1 + BLK_START] < m0 + BM) ++b1;
}

__global__ void __launch_bounds__(BASE_THREADS, 1) salt_base_kernel(const __grid_constant__ BaseParams p)
{
    extern __shared__ __align__(128) uint8_t smem_raw[];
    uint8_t *ring = smem_raw + ((1024 - (smem_u32(smem_raw) & 1023)) & 1023);
    uint8_t *dv = ring + NST * STAGE;
    uint8_t *db = dv + DV_BYTES;
    BaseInfo &info = *reinterpret_cast<BaseInfo *>(db + DB_BYTES);
    const uint32_t ring32 = smem_u32(ring), dv32 = smem_u32(dv), db32 = smem_u32(db);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int T = p.T, n_blk = min(p.counts[3], p.blk_cap);
    const int n_mt = (T + BM - 1) / BM, n_nt = (p.d_out + BN - 1) / BN;
    const int n_tiles = n_mt * n_nt;
    const int nk = (p.d_in + BK - 1) / BK;
    if (T <= 0) return;
    auto bar = [](const uint64_t &b) { return smem_u32(&b); };
    if (warp == MW) {
        tmem_alloc(smem_u32(&info.tmem), 256);
        tmem_relinquish();
    }
    if (tid == 0) {
        for (int i = 0; i < NST; ++i) {
            mbar_init(bar(info.full[i]), PT + 1);  // every producer's copies + the W tile's bytes
            mbar_init(bar(info.empty[i]), 1);
        }
        mbar_init(bar(info.dfull), PT);
        mbar_init(bar(info.dempty), 1);
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar(info.accf[i]), 1);
            mbar_init(bar(info.acce[i]), 4);
        }
        mbar_fence_init();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = info.tmem;
    bool ok_all = true;
    auto wait_bar = [&](const uint64_t &b, uint32_t parity) {
        if (!mbar_wait(smem_u32(&b), parity)) ok_all = false;
    };
    // tile t: M tile t % n_mt, N tile t / n_mt (the M tiles of one W column
    // block run side by side, so W is read from memory about once)
    if (warp < PW) {
        // ============================================================ producers
        uint32_t g = 0, dg = 0;  // K stages and delta stages issued
        for (int t = blockIdx.x; t < n_tiles; t += gridDim.x) {
            const int m0 = (t % n_mt) * BM, n0 = (t / n_mt) * BN;
            named_sync(BAR_P, PT);  // the previous tile's copies are out: the row table is free
            if (tid < BM) info.prow[tid] = m0 + tid < T ? p.perm[m0 + tid] : -1;
            named_sync(BAR_P, PT);
            for (int kc = 0; kc < nk; ++kc, ++g) {
                const uint32_t slot = g % NST;
                if (g >= NST) wait_bar(info.empty[slot], ((g / NST) - 1) & 1);
                const uint32_t xs = ring32 + slot * STAGE, ws = xs + X_BYTES;
                const int k0 = kc * BK;
                if (tid == 0) {
                    mbar_expect_tx(bar(info.full[slot]), W_BYTES);
                    if (p.w_layout == SALT_W_IN_OUT) {
                        // W[d_in][d_out]: two boxes of 64 K rows x 64 N columns (MN-major)
                        tma_load_2d(ws, &p.wmap, n0, k0, bar(info.full[slot]));
                        tma_load_2d(ws + 64 * 128, &p.wmap, n0 + 64, k0, bar(info.full[slot]));
                    } else {
                        // W[d_out][d_in]: one box of 128 N rows x 64 K (K-major)
                        tma_load_2d(ws, &p.wmap, k0, n0, bar(info.full[slot]));
                    }
                }
                for (int idx = tid; idx < BM * 8; idx += PT) {
                    const int r = idx >> 3, c = idx & 7;
                    const int row = info.prow[r];
                    const bool ok = row >= 0 && k0 + c * 8 < p.d_in;
                    cp_async16(xs + swz128(r, c), p.x + (ok ? (int64_t)row * p.d_in + k0 + c * 8 : 0), ok);
                }
                cp_async_arrive_noinc(bar(info.full[slot]));
            }
            // the delta of every row block overlapping the tile
            int b0, b1;
            blocks_of_tile(p, n_blk, m0, b0, b1);
            for (int b = b0; b < b1; ++b) {
                const int4 m0r = *reinterpret_cast<const int4 *>(p.blk + BLK_INTS * b);
                const int start = m0r.x, M = m0r.y, d = m0r.z, rc = m0r.w;
                const int S = rc + p.blk[BLK_INTS * b + BLK_NRES];
                const int S_pad = (S + 15) & ~15;
                if (S <= 0 || S > S_MAX) continue;  // flagged by the shrink
                // the delta area's previous block has been consumed by the MMAs
                if (dg > 0) wait_bar(info.dempty, (dg - 1) & 1);
                named_sync(BAR_P, PT);
                if (tid < S)
                    info.bsrc[tid] = tid < rc ? p.B + ((int64_t)d * p.rc_max + tid) * p.d_out
                                              : res_b_row(p, p.blk_res[(int64_t)b * S_MAX + (tid - rc)]);
                named_sync(BAR_P, PT);
                // V rows of the block at their tile rows (other rows zero), K-major halves
                const uint16_t *vt = p.vext + (int64_t)b * (TM * VEXT_COLS);
                for (int idx = tid; idx < BM * 16; idx += PT) {
                    const int r = idx >> 4, c = idx & 15;  // c: 16-byte piece of the row's 256 bytes
                    const int gp = m0 + r, i = gp - start;
                    const bool ok = i >= 0 && i < M && c * 8 < S_pad;
                    cp_async16(dv32 + (c >> 3) * (BM * 128) + swz128(r, c & 7), vt + (ok ? i * VEXT_COLS + c * 8 : 0), ok);
                }
                // stacked B rows, columns n0 .. n0 + 127 as two MN-major halves
                for (int idx = tid; idx < S_pad * 16; idx += PT) {
                    const int k = idx >> 4, c = idx & 15, col = n0 + c * 8;
                    const bool ok = k < S && col < p.d_out;
                    cp_async16(db32 + (c >> 3) * (S_MAX * 128) + swz128(k, c & 7), ok ? info.bsrc[k] + col : p.x, ok);
                }
                cp_async_arrive_noinc(bar(info.dfull));
                ++dg;
            }
        }
        cp_async_wait<0>();
    } else if (warp == MW) {
        // ============================================================ MMA issue
        if (lane == 0) {
            const uint32_t id_k = idesc_bf16_f32(BM, BN);          // W K-major (N = 128)
            const uint32_t id_mn = idesc_bf16_f32_bmn(BM, 64);     // W / stacked B MN-major, N = 64 per half
            uint32_t g = 0, dg = 0, lt = 0;
            for (int t = blockIdx.x; t < n_tiles; t += gridDim.x, ++lt) {
                const int m0 = (t % n_mt) * BM;
                const uint32_t buf = lt & 1, acc = tmem + buf * BN;
                if (lt >= 2) wait_bar(info.acce[buf], ((lt - 2) >> 1) & 1);
                tc_fence_after();
                for (int kc = 0; kc < nk; ++kc, ++g) {
                    const uint32_t slot = g % NST;
                    wait_bar(info.full[slot], (g / NST) & 1);
                    fence_async_smem();
                    tc_fence_after();
                    const uint32_t xs = ring32 + slot * STAGE, ws = xs + X_BYTES;
#pragma unroll
                    for (int kk = 0; kk < BK / 16; ++kk) {
                        const uint32_t a = (kc > 0 || kk > 0) ? 1u : 0u;
                        const uint64_t ad = sdesc_kmajor_sw128(xs + kk * 32);
                        if (p.w_layout == SALT_W_IN_OUT) {
                            umma_bf16(acc, ad, sdesc_mnmajor_sw128(ws + kk * 2048), id_mn, a);
                            umma_bf16(acc + 64, ad, sdesc_mnmajor_sw128(ws + 64 * 128 + kk * 2048), id_mn, a);
                        } else {
                            umma_bf16(acc, ad, sdesc_kmajor_sw128(ws + kk * 32), id_k, a);
                        }
                    }
                    umma_commit(bar(info.empty[slot]));
                }
                int b0, b1;
                blocks_of_tile(p, n_blk, m0, b0, b1);
                for (int b = b0; b < b1; ++b) {
                    const int rc = p.blk[BLK_INTS * b + BLK_RC];
                    const int S = rc + p.blk[BLK_INTS * b + BLK_NRES];
                    if (S <= 0 || S > S_MAX) continue;
                    const int S_pad = (S + 15) & ~15;
                    wait_bar(info.dfull, dg & 1);
                    fence_async_smem();
                    tc_fence_after();
                    for (int ks = 0; ks < (S_pad >> 4); ++ks) {
                        const uint64_t ad = sdesc_kmajor_sw128(dv32 + (ks >> 2) * (BM * 128) + (ks & 3) * 32);
                        umma_bf16(acc, ad, sdesc_mnmajor_sw128(db32 + ks * 2048), id_mn, 1u);
                        umma_bf16(acc + 64, ad, sdesc_mnmajor_sw128(db32 + S_MAX * 128 + ks * 2048), id_mn, 1u);
                    }
                    umma_commit(bar(info.dempty));
                    ++dg;
                }
                umma_commit(bar(info.accf[buf]));
            }
        }
        __syncwarp();
    } else {
        // ============================================================ epilogue
        const int q = warp & 3, row = q * 32 + lane;
        uint32_t lt = 0;
        for (int t = blockIdx.x; t < n_tiles; t += gridDim.x, ++lt) {
            const int m0 = (t % n_mt) * BM, n0 = (t / n_mt) * BN;
            const uint32_t buf = lt & 1;
            const int gp = m0 + row;
            const int tok = gp < T ? p.perm[gp] : -1;
            wait_bar(info.accf[buf], (lt >> 1) & 1);
            tc_fence_after();
            uint16_t *yr = tok >= 0 ? p.y + (int64_t)tok * p.d_out : nullptr;
#pragma unroll 1
            for (int c16 = 0; c16 < BN / 16; ++c16) {
                uint32_t v[16];
                tmem_ld16(tmem + ((uint32_t)(q * 32) << 16) + buf * BN + c16 * 16, v);
                tmem_ld_wait();
                const int col = n0 + c16 * 16;
                if (yr) {
                    uint32_t w[8];
#pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        const __nv_bfloat162 h =
                            __floats2bfloat162_rn(__uint_as_float(v[2 * i]), __uint_as_float(v[2 * i + 1]));
                        w[i] = *reinterpret_cast<const uint32_t *>(&h);
                    }
                    if (col < p.d_out) *reinterpret_cast<uint4 *>(yr + col) = make_uint4(w[0], w[1], w[2], w[3]);
                    if (col + 8 < p.d_out) *reinterpret_cast<uint4 *>(yr + col + 8) = make_uint4(w[4], w[5], w[6], w[7]);
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_relaxed(bar(info.acce[buf]));
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == MW) tmem_dealloc(tmem, 256);
    if (!ok_all) atomicOr(p.err, SALT_DEVERR_TIMEOUT);
}

int g_base_sms[64];

}  // namespace

cudaError_t base_prepare(int device)
{
    if (device < 0 || device >= 64) return cudaErrorInvalidDevice;
    cudaError_t e = cudaDeviceGetAttribute(&g_base_sms[device], cudaDevAttrMultiProcessorCount, device);
    if (e != cudaSuccess) return e;
    return cudaFuncSetAttribute(salt_base_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)BASE_SMEM);
}

cudaError_t launch_base(const BaseParams &p, cudaStream_t stream)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const int n_sm = (dev >= 0 && dev < 64 && g_base_sms[dev] > 0) ? g_base_sms[dev] : 1;
    const int n_tiles = ((p.T + BM - 1) / BM) * ((p.d_out + BN - 1) / BN);
    const int grid = n_tiles < n_sm ? n_tiles : n_sm;
    if (grid <= 0) return cudaSuccess;
    salt_base_kernel<<<grid, BASE_THREADS, BASE_SMEM, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace salt
