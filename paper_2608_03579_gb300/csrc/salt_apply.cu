// Fused centroid + residual apply (Section "Multi-Tenant Serving":
// W_final = W_base + gamma * Wbar + delta_i, evaluated in low-rank form).
//
// Work unit: one row block (<= TM tokens of one domain, <= umax user runs,
// from the segment builder) of one projection, handled by a cluster of
// CLUSTER CTAs.  The block's factors are concatenated into one stack of
// S = rc + sum_u r_u rows, [A_c | a_u1 | a_u2 | ...] - the paper's
// "centroid and residual concatenated into one standard adapter" identity,
// applied per block - so the whole block is one dense contraction:
//
//   shrink   V[M x S]   = X[M x d_in] * Stack_A^T     (CTA c: its d_in slice)
//   reduce   V          = sum over the cluster's partials (DSMEM), then
//            V_ext[t,s] = s_c V[t,s]         for s < rc
//                       = s_u(t) V[t,s]      for s in the token's own user's rows
//                       = 0                  otherwise
//   expand   Y[M x d_out] += V_ext * Stack_B  (CTA c: its d_out slice)
//
// x rows are gathered by the grouped order, y is read and written once, each
// factor row is read once per block.  Operands are staged by cp.async in
// 128-byte-row XOR-swizzled tiles (two stages) and multiplied with bf16
// mma.sync (fp32 accumulation); V_ext is rounded to bf16 for the expand.
// The clusters are persistent and stride over (projection, block) items.
// No global scratch: partial sums live in shared memory.
#include <cooperative_groups.h>
#include <cuda_bf16.h>

#include "salt_internal.cuh"

namespace cg = cooperative_groups;

namespace salt {
namespace {

constexpr int KC = 64;                        // K chunk in elements (128-byte rows)
constexpr int NC = 64;                        // N chunk of the expand
constexpr int NSTAGE = 2;
constexpr int TILE_BYTES = TM * 128;          // 128 rows x 128 B
constexpr int STAGE_BYTES = 2 * TILE_BYTES;   // (X, A) or (Y, B)
constexpr int STAGES_BYTES = NSTAGE * STAGE_BYTES;
constexpr int PW = SALT_MAX_CENTROID_RANK + SALT_MAX_RESIDUAL_RANK;  // compact partial width
constexpr int P_BYTES = TM * PW * 4;
constexpr int RED_ROWS = (TM + CLUSTER - 1) / CLUSTER;
constexpr int RED_BYTES = RED_ROWS * PW * 4;
constexpr int VEXT_ROW = S_MAX * 2;           // bytes per V_ext row
constexpr int VEXT_BYTES = TM * VEXT_ROW;
static_assert(P_BYTES + RED_BYTES <= STAGES_BYTES, "partials must fit in the stage area");
static_assert(S_MAX <= 128 && TM <= 128, "tile shapes");

struct Info {
    const uint16_t *srcA[S_MAX];  // stacked At rows (element 0 of the row for this layer)
    const uint16_t *srcB[S_MAX];  // stacked B rows
    int32_t row[TM];              // x / y row of the i-th token of the block
    int32_t ucol[TM];             // first stacked row of the token's user, -1: none
    int32_t urank[TM];
    float usu[TM];
    int32_t wsum[4];
};
constexpr int INFO_BYTES = (sizeof(Info) + 127) / 128 * 128;
constexpr size_t SMEM_BYTES = STAGES_BYTES + VEXT_BYTES + INFO_BYTES;

__device__ __forceinline__ uint32_t smem_u32(const void *p)
{
    return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ int swz128(int row, int chunk) { return row * 128 + ((chunk ^ (row & 7)) << 4); }
__device__ __forceinline__ int swz256(int row, int chunk) { return row * VEXT_ROW + ((chunk ^ (row & 7)) << 4); }

__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src, bool valid)
{
    int n = valid ? 16 : 0;  // 0: zero-fill, nothing read
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src), "r"(n));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N)); }

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2, uint32_t &r3)
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3) : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2, uint32_t &r3)
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3) : "r"(addr));
}
__device__ __forceinline__ void mma_bf16(float (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1)
{
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};\n"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ float bf16_to_f(uint16_t h) { return __uint_as_float(((uint32_t)h) << 16); }
__device__ __forceinline__ uint16_t f_to_bf16(float f)
{
    __nv_bfloat16 b = __float2bfloat16_rn(f);
    return *reinterpret_cast<uint16_t *>(&b);
}

__global__ void __launch_bounds__(APPLY_THREADS, 2) salt_apply_kernel(const __grid_constant__ ApplyParams p)
{
    extern __shared__ __align__(128) uint8_t smem[];
    uint8_t *stages = smem;
    float *P = reinterpret_cast<float *>(smem);
    float *RED = reinterpret_cast<float *>(smem + P_BYTES);
    uint8_t *vext = smem + STAGES_BYTES;
    Info &info = *reinterpret_cast<Info *>(smem + STAGES_BYTES + VEXT_BYTES);

    cg::cluster_group cluster = cg::this_cluster();
    const int crank = (int)cluster.block_rank();
    const int cid = blockIdx.x / CLUSTER;
    const int n_clusters = gridDim.x / CLUSTER;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int g = lane >> 2, q4 = lane & 3;
    const int n_blk = p.counts[3];
    const int n_items = n_blk * p.n_proj;

    for (int item = cid; item < n_items; item += n_clusters) {
        const int pi = item / n_blk, b = item - pi * n_blk;
        const ApplyProj &pr = p.proj[pi];
        const int start = p.blk[3 * b], M = p.blk[3 * b + 1], d = p.blk[3 * b + 2];
        const int rc = d >= 0 ? p.dom_rc[d] : 0;
        const float s_c = d >= 0 ? p.dom_sc[d] : 0.f;
        const int d_in = pr.d_in, d_out = pr.d_out;

        // ---------------- block setup: tokens, users, stacked factor rows
        int slot = -1, rank = 0, contrib = 0;
        float su = 0.f;
        if (tid < M) {
            info.row[tid] = p.perm[start + tid];
            int raw = p.sorted_slot[start + tid];
            if (raw >= 0) {
                const uint8_t *h = p.pool + (int64_t)raw * p.slot_stride;
                const salt_blob_header *hd = reinterpret_cast<const salt_blob_header *>(h);
                if (hd->magic == SALT_BLOB_MAGIC && hd->rank >= 1 && hd->rank <= p.r_max) {
                    slot = raw;
                    rank = hd->rank;
                    su = hd->s_u;
                } else {
                    atomicOr(p.err, SALT_DEVERR_SLOT_EMPTY);
                }
            }
            bool head = tid == 0 || raw != p.sorted_slot[start + tid - 1];
            contrib = (head && slot >= 0) ? rank : 0;
        }
        // inclusive scan of contrib over the first TM threads (warps 0..3)
        int incl = contrib;
        if (tid < TM) {
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                int y = __shfl_up_sync(0xffffffffu, incl, o);
                if (lane >= o) incl += y;
            }
            if (lane == 31) info.wsum[warp] = incl;
        }
        __syncthreads();
        int S;
        {
            int w0 = info.wsum[0], w1 = info.wsum[1], w2 = info.wsum[2], w3 = info.wsum[3];
            int before = warp == 0 ? 0 : warp == 1 ? w0 : warp == 2 ? w0 + w1 : w0 + w1 + w2;
            S = rc + w0 + w1 + w2 + w3;
            if (tid < M) {
                int uc = slot >= 0 ? rc + before + incl - rank : -1;
                info.ucol[tid] = uc;
                info.urank[tid] = slot >= 0 ? rank : 0;
                info.usu[tid] = su;
                if (contrib > 0 && uc + rank <= S_MAX) {
                    const uint16_t *base = reinterpret_cast<const uint16_t *>(
                        p.pool + (int64_t)slot * p.slot_stride + SALT_BLOB_HEADER_BYTES) + (int64_t)rank * pr.res_off;
                    for (int k = 0; k < rank; ++k) {
                        info.srcA[uc + k] = base + (int64_t)k * d_in;
                        info.srcB[uc + k] = base + (int64_t)rank * d_in + (int64_t)k * d_out;
                    }
                }
            }
            if (tid >= TM && tid - TM < rc) {
                int k = tid - TM;
                info.srcA[k] = pr.A + ((int64_t)d * p.rc_max + k) * d_in;
                info.srcB[k] = pr.B + ((int64_t)d * p.rc_max + k) * d_out;
            }
        }
        __syncthreads();
        // S is computed from the same memory by every CTA of the cluster, so
        // skipping is uniform and no cluster barrier is left unmatched.
        if (S > S_MAX || S == 0) {
            if (S > S_MAX && tid == 0 && crank == 0) atomicOr(p.err, SALT_DEVERR_RANK);
            __syncthreads();
            continue;
        }
        const int S_pad = (S + 15) & ~15;

        // ---------------- shrink: partial V over this CTA's d_in slice
        const int nk = (d_in + KC - 1) / KC;
        const int kc0 = crank * nk / CLUSTER, kc1 = (crank + 1) * nk / CLUSTER;
        const int m_tiles = (M + 15) >> 4;
        const int n_nt = S_pad >> 3;
        const int warps_n = n_nt > 8 ? 2 : 1;
        const int warps_m = 8 / warps_n;
        const int wn = warp % warps_n, wm = warp / warps_n;
        const int nt_lo = wn * 8, nt_hi = min(n_nt, nt_lo + 8);
        const int mt0 = wm, mt1 = wm + warps_m;
        const bool act0 = mt0 < m_tiles, act1 = (warps_m == 4) && mt1 < m_tiles;

        float acc[2][8][4];
#pragma unroll
        for (int i = 0; i < 2; ++i)
#pragma unroll
            for (int j = 0; j < 8; ++j)
#pragma unroll
                for (int e = 0; e < 4; ++e) acc[i][j][e] = 0.f;

        auto load_shrink = [&](int kc, int st) {
            uint8_t *xs = stages + st * STAGE_BYTES;
            uint8_t *as = xs + TILE_BYTES;
            const int k0 = kc * KC;
            for (int idx = tid; idx < M * 8; idx += APPLY_THREADS) {
                int r = idx >> 3, c = idx & 7, col = k0 + c * 8;
                bool ok = col < d_in;
                const uint16_t *src = pr.x + (int64_t)info.row[r] * d_in + (ok ? col : 0);
                cp_async16(smem_u32(xs + swz128(r, c)), src, ok);
            }
            for (int idx = tid; idx < S * 8; idx += APPLY_THREADS) {
                int r = idx >> 3, c = idx & 7, col = k0 + c * 8;
                bool ok = col < d_in;
                cp_async16(smem_u32(as + swz128(r, c)), info.srcA[r] + (ok ? col : 0), ok);
            }
        };

        if (kc0 < kc1) {
            load_shrink(kc0, 0);
            cp_async_commit();
            for (int kc = kc0; kc < kc1; ++kc) {
                const int st = (kc - kc0) & 1;
                if (kc + 1 < kc1) {
                    load_shrink(kc + 1, st ^ 1);
                    cp_async_commit();
                    cp_async_wait<1>();
                } else {
                    cp_async_wait<0>();
                }
                __syncthreads();
                const uint32_t xs = smem_u32(stages + st * STAGE_BYTES);
                const uint32_t as = xs + TILE_BYTES;
#pragma unroll
                for (int kk = 0; kk < KC / 16; ++kk) {
                    uint32_t a0[4], a1[4];
                    if (act0) {
                        int r = mt0 * 16 + (lane & 15);
                        ldsm_x4(xs + swz128(r, kk * 2 + (lane >> 4)), a0[0], a0[1], a0[2], a0[3]);
                    }
                    if (act1) {
                        int r = mt1 * 16 + (lane & 15);
                        ldsm_x4(xs + swz128(r, kk * 2 + (lane >> 4)), a1[0], a1[1], a1[2], a1[3]);
                    }
#pragma unroll
                    for (int np = 0; np < 4; ++np) {
                        const int nt = nt_lo + 2 * np;
                        if (nt < nt_hi && (act0 || act1)) {
                            int mi = lane >> 3;
                            int n = nt * 8 + (mi >> 1) * 8 + (lane & 7);
                            uint32_t b0, b1, b2, b3;
                            ldsm_x4(as + swz128(n, kk * 2 + (mi & 1)), b0, b1, b2, b3);
                            if (act0) {
                                mma_bf16(acc[0][2 * np], a0, b0, b1);
                                mma_bf16(acc[0][2 * np + 1], a0, b2, b3);
                            }
                            if (act1) {
                                mma_bf16(acc[1][2 * np], a1, b0, b1);
                                mma_bf16(acc[1][2 * np + 1], a1, b2, b3);
                            }
                        }
                    }
                }
                __syncthreads();
            }
        }

        // compact partials: the centroid columns and the token's own user columns
#pragma unroll
        for (int i = 0; i < 2; ++i) {
            const bool act = i == 0 ? act0 : act1;
            const int mt = i == 0 ? mt0 : mt1;
            if (!act) continue;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int nt = nt_lo + j;
                if (nt >= nt_hi) continue;
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int row = mt * 16 + g + (e >> 1) * 8;
                    const int col = nt * 8 + 2 * q4 + (e & 1);
                    if (row >= M) continue;
                    if (col < rc) {
                        P[row * PW + col] = acc[i][j][e];
                    } else {
                        const int uc = info.ucol[row];
                        if (uc >= 0 && col >= uc && col < uc + info.urank[row])
                            P[row * PW + rc + (col - uc)] = acc[i][j][e];
                    }
                }
            }
        }
        cluster.sync();

        // ---------------- reduce-scatter over the cluster, then all-gather V_ext
        const int r0 = crank * M / CLUSTER, r1 = (crank + 1) * M / CLUSTER;
        for (int idx = tid; idx < (r1 - r0) * PW; idx += APPLY_THREADS) {
            const int rr = idx / PW, col = idx - rr * PW, row = r0 + rr;
            if (col < rc + info.urank[row]) {
                float s = 0.f;
#pragma unroll
                for (int qq = 0; qq < CLUSTER; ++qq) {
                    const float *peer = cluster.map_shared_rank(P, qq);
                    s += peer[row * PW + col];
                }
                RED[rr * PW + col] = s;
            }
        }
        __syncthreads();
        const int nch = S_pad >> 3;
        for (int idx = tid; idx < (r1 - r0) * nch; idx += APPLY_THREADS) {
            const int rr = idx / nch, c = idx - rr * nch, row = r0 + rr;
            const int uc = info.ucol[row], ur = info.urank[row];
            const float us = info.usu[row];
            uint32_t w[4];
#pragma unroll
            for (int h = 0; h < 4; ++h) {
                uint16_t v2[2];
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                    const int col = c * 8 + 2 * h + e;
                    float v = 0.f;
                    if (col < rc) v = s_c * RED[rr * PW + col];
                    else if (uc >= 0 && col >= uc && col < uc + ur) v = us * RED[rr * PW + rc + (col - uc)];
                    v2[e] = f_to_bf16(v);
                }
                w[h] = (uint32_t)v2[0] | ((uint32_t)v2[1] << 16);
            }
            const uint4 val = make_uint4(w[0], w[1], w[2], w[3]);
            const int off = swz256(row, c);
#pragma unroll
            for (int qq = 0; qq < CLUSTER; ++qq) {
                uint8_t *peer = cluster.map_shared_rank(vext, qq);
                *reinterpret_cast<uint4 *>(peer + off) = val;
            }
        }
        cluster.sync();

        // ---------------- expand: y slice += V_ext * Stack_B
        const int nn = (d_out + NC - 1) / NC;
        const int nc0 = crank * nn / CLUSTER, nc1 = (crank + 1) * nn / CLUSTER;
        const int em = warp >> 1, en = warp & 1;
        const int emt0 = em, emt1 = em + 4;
        const bool eact0 = emt0 < m_tiles, eact1 = emt1 < m_tiles;

        auto load_expand = [&](int ncn, int st) {
            uint8_t *ys = stages + st * STAGE_BYTES;
            uint8_t *bs = ys + TILE_BYTES;
            const int n0 = ncn * NC;
            for (int idx = tid; idx < M * 8; idx += APPLY_THREADS) {
                int r = idx >> 3, c = idx & 7, col = n0 + c * 8;
                bool ok = col < d_out;
                const uint16_t *src = pr.y + (int64_t)info.row[r] * d_out + (ok ? col : 0);
                cp_async16(smem_u32(ys + swz128(r, c)), src, ok);
            }
            for (int idx = tid; idx < S_pad * 8; idx += APPLY_THREADS) {
                int r = idx >> 3, c = idx & 7, col = n0 + c * 8;
                bool ok = r < S && col < d_out;
                const uint16_t *src = ok ? info.srcB[r] + col : pr.y;
                cp_async16(smem_u32(bs + swz128(r, c)), src, ok);
            }
        };

        if (nc0 < nc1) {
            load_expand(nc0, 0);
            cp_async_commit();
            for (int ncn = nc0; ncn < nc1; ++ncn) {
                const int st = (ncn - nc0) & 1;
                if (ncn + 1 < nc1) {
                    load_expand(ncn + 1, st ^ 1);
                    cp_async_commit();
                    cp_async_wait<1>();
                } else {
                    cp_async_wait<0>();
                }
                __syncthreads();
                uint8_t *ys = stages + st * STAGE_BYTES;
                const uint32_t ys32 = smem_u32(ys);
                const uint32_t bs32 = ys32 + TILE_BYTES;
                const uint32_t vx32 = smem_u32(vext);
                float c2[2][4][4];
#pragma unroll
                for (int i = 0; i < 2; ++i)
#pragma unroll
                    for (int j = 0; j < 4; ++j)
#pragma unroll
                        for (int e = 0; e < 4; ++e) c2[i][j][e] = 0.f;
                for (int ks = 0; ks < (S_pad >> 4); ++ks) {
                    uint32_t a0[4], a1[4];
                    if (eact0) {
                        int r = emt0 * 16 + (lane & 15);
                        ldsm_x4(vx32 + swz256(r, ks * 2 + (lane >> 4)), a0[0], a0[1], a0[2], a0[3]);
                    }
                    if (eact1) {
                        int r = emt1 * 16 + (lane & 15);
                        ldsm_x4(vx32 + swz256(r, ks * 2 + (lane >> 4)), a1[0], a1[1], a1[2], a1[3]);
                    }
#pragma unroll
                    for (int np = 0; np < 2; ++np) {
                        const int nt = en * 4 + 2 * np;
                        if (eact0 || eact1) {
                            int mi = lane >> 3;
                            int kr = ks * 16 + (mi & 1) * 8 + (lane & 7);
                            uint32_t b0, b1, b2, b3;
                            ldsm_x4_t(bs32 + swz128(kr, nt + (mi >> 1)), b0, b1, b2, b3);
                            if (eact0) {
                                mma_bf16(c2[0][2 * np], a0, b0, b1);
                                mma_bf16(c2[0][2 * np + 1], a0, b2, b3);
                            }
                            if (eact1) {
                                mma_bf16(c2[1][2 * np], a1, b0, b1);
                                mma_bf16(c2[1][2 * np + 1], a1, b2, b3);
                            }
                        }
                    }
                }
                // epilogue: y_in (staged) + delta, one rounding, back into the staged tile
#pragma unroll
                for (int i = 0; i < 2; ++i) {
                    const bool act = i == 0 ? eact0 : eact1;
                    const int mt = i == 0 ? emt0 : emt1;
                    if (!act) continue;
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        const int nt = en * 4 + j;
#pragma unroll
                        for (int h = 0; h < 2; ++h) {
                            const int row = mt * 16 + g + h * 8;
                            if (row >= M) continue;
                            uint32_t *cell = reinterpret_cast<uint32_t *>(ys + swz128(row, nt) + q4 * 4);
                            uint32_t v = *cell;
                            float lo = bf16_to_f((uint16_t)(v & 0xffffu)) + c2[i][j][2 * h];
                            float hi = bf16_to_f((uint16_t)(v >> 16)) + c2[i][j][2 * h + 1];
                            *cell = (uint32_t)f_to_bf16(lo) | ((uint32_t)f_to_bf16(hi) << 16);
                        }
                    }
                }
                __syncthreads();
                const int n0 = ncn * NC;
                for (int idx = tid; idx < M * 8; idx += APPLY_THREADS) {
                    int r = idx >> 3, c = idx & 7, col = n0 + c * 8;
                    if (col < d_out) {
                        uint4 v = *reinterpret_cast<const uint4 *>(ys + swz128(r, c));
                        *reinterpret_cast<uint4 *>(pr.y + (int64_t)info.row[r] * d_out + col) = v;
                    }
                }
                __syncthreads();
            }
        }
    }
}

}  // namespace

size_t apply_smem_bytes() { return SMEM_BYTES; }

cudaError_t apply_prepare(int device, int *max_active_clusters)
{
    (void)device;
    cudaError_t e = cudaFuncSetAttribute(salt_apply_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)SMEM_BYTES);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = CLUSTER;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.gridDim = dim3(CLUSTER * 64, 1, 1);
    cfg.blockDim = dim3(APPLY_THREADS, 1, 1);
    cfg.dynamicSmemBytes = SMEM_BYTES;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    e = cudaOccupancyMaxActiveClusters(&n, salt_apply_kernel, &cfg);
    if (e != cudaSuccess) return e;
    *max_active_clusters = n > 0 ? n : 1;
    return cudaSuccess;
}

cudaError_t launch_apply(const ApplyParams &p, int n_clusters, cudaStream_t stream)
{
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = CLUSTER;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.gridDim = dim3(CLUSTER * n_clusters, 1, 1);
    cfg.blockDim = dim3(APPLY_THREADS, 1, 1);
    cfg.dynamicSmemBytes = SMEM_BYTES;
    cfg.stream = stream;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, salt_apply_kernel, p);
}

}  // namespace salt
