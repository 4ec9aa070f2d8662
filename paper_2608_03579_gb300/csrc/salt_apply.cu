// Fused centroid + residual apply (Section "Multi-Tenant Serving":
// W_final = W_base + gamma * Wbar + delta_i, evaluated in low-rank form).
//
// A row block (<= TM tokens of one domain, <= umax user runs, from the
// segment builder) concatenates its factors into one stack of
// S = rc + sum_u r_u rows, [A_c | a_u1 | a_u2 | ...] - the paper's
// "centroid and residual concatenated into one standard adapter" identity,
// applied per block - so each block is one dense contraction.  Two kernels:
//
//   shrink (one cluster of C CTAs per block and projection; CTA c takes
//           every C-th 64-wide chunk of d_in):
//       V^T[S x M] = Stack_A[S x d_in] * X[M x d_in]^T on the tensor cores
//       (tcgen05.mma, fp32 accumulator in tensor memory; the stack is the
//       128-row operand, the tokens the N = 16..128 operand), partial sums
//       reduced across the cluster through distributed shared memory, then
//       V_ext[t,s] = s_c V[t,s]    for s < rc (centroid rows)
//                  = s_u V[t,s]    for s in the token's own user's rows
//                  = 0             otherwise,
//       rounded to bf16 into the workspace tile of the block.
//   expand (persistent, one CTA per SM, launched as a programmatic
//           dependent of the shrink; items are (block, 64 output columns)):
//       Y[M x 64] += V_ext * Stack_B[:, cols] on the tensor cores
//       (tcgen05.mma, V_ext K-major and the B rows MN-major as they lie in
//       memory, fp32 accumulators double-buffered in tensor memory), the y
//       and B rows of the next items streaming through a shared-memory ring
//       meanwhile; the first items' rows are fetched before the dependency
//       wait, so their latency overlaps the shrink.  y is read once and
//       written once, rounded once (RNE).
//
// Operands are staged by cp.async in 128-byte-row, 128-byte-swizzled tiles
// (the layout the UMMA descriptors read).  Partial sums never leave the
// chip; the only scratch is the bf16 V tile per block.
#include <cooperative_groups.h>
#include <cuda_bf16.h>

#include <mutex>

#include "salt_internal.cuh"
#include "salt_tcgen05.cuh"

namespace cg = cooperative_groups;

namespace salt {
namespace {

constexpr int KC = 64;                         // K chunk of the shrink (128-byte rows)
constexpr int NC = 64;                         // output columns per expand CTA
constexpr int TILE_BYTES = TM * 128;           // 128 rows x 128 B
constexpr int STAGES_BYTES = 96 * 1024;        // shrink stage ring
constexpr int MAX_STAGES = 6;
constexpr int MAX_CLUSTER = 16;
constexpr int TMEM_COLS = 128;                 // D^T: up to 128 token columns
constexpr int PW = SALT_MAX_CENTROID_RANK + SALT_MAX_RESIDUAL_RANK;  // compact partial width
constexpr int P_BYTES = TM * PW * 4;
constexpr int RED_ROWS = TM / CLUSTER;         // rows each CTA reduces (clusters of >= CLUSTER CTAs)
constexpr int RED_BYTES = RED_ROWS * PW * 4;
constexpr int VT_ROW = VEXT_COLS * 2;          // bytes per V tile row
constexpr int VT_BYTES = TM * VT_ROW;
static_assert(P_BYTES + RED_BYTES <= STAGES_BYTES, "partials must fit in the stage area");
static_assert(S_MAX <= 128, "the factor stack is the 128-row UMMA operand");

struct ShrinkInfo {
    const uint16_t *srcA[S_MAX];  // stacked At rows (element 0 of the row for this layer)
    int32_t row[TM];              // x row of the i-th token of the block
    int32_t ucol[TM];             // first stacked row of the token's user, -1: none
    int32_t urank[TM];
    float usu[TM];
    int16_t rt0[S_MAX];           // residual stack row -> first token of its user run
    int16_t rt1[S_MAX];           //                    -> one past the last token
    int16_t rk[S_MAX];            //                    -> rank index within the user
    uint64_t bar[MAX_STAGES];     // per stage: the MMAs reading it have completed
    uint32_t tmem;                // tensor-memory base of D^T
};
constexpr size_t SHRINK_SMEM = 1024 + STAGES_BYTES + (sizeof(ShrinkInfo) + 127) / 128 * 128;

__device__ __forceinline__ uint32_t smem_u32(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ int swz128(int row, int chunk) { return row * 128 + ((chunk ^ (row & 7)) << 4); }
__device__ __forceinline__ int swz256(int row, int chunk) { return row * VT_ROW + ((chunk ^ (row & 7)) << 4); }

__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src, bool valid)
{
    int n = valid ? 16 : 0;  // 0: zero-fill, nothing read
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src), "r"(n));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory"); }
// wait until at most n groups are pending (n in [1, MAX_STAGES - 2])
__device__ __forceinline__ void cp_async_wait_dyn(int n)
{
    switch (n) {
    case 1: cp_async_wait<1>(); break;
    case 2: cp_async_wait<2>(); break;
    case 3: cp_async_wait<3>(); break;
    default: cp_async_wait<4>(); break;
    }
}

__device__ __forceinline__ void pdl_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;\n" ::); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;\n" ::: "memory"); }

__device__ __forceinline__ float bf16_to_f(uint16_t h) { return __uint_as_float(((uint32_t)h) << 16); }
__device__ __forceinline__ uint16_t f_to_bf16(float f)
{
    __nv_bfloat16 b = __float2bfloat16_rn(f);
    return *reinterpret_cast<uint16_t *>(&b);
}

// Residual row entry of a block's factor stack -> first element of that row.
__device__ __forceinline__ const uint16_t *residual_row(const ApplyParams &p, const ApplyProj &pr, int e, bool b_side)
{
    const int slot = e >> 8, rank = ((e >> 4) & 15) + 1, k = e & 15;
    const uint16_t *base = reinterpret_cast<const uint16_t *>(p.pool + (int64_t)slot * p.slot_stride +
                                                              SALT_BLOB_HEADER_BYTES) + (int64_t)rank * pr.res_off;
    return b_side ? base + (int64_t)rank * pr.d_in + (int64_t)k * pr.d_out : base + (int64_t)k * pr.d_in;
}

// ---------------------------------------------------------------------------- shrink
constexpr int MAX_PIECES = (TM * 8 + APPLY_THREADS - 1) / APPLY_THREADS;  // 16-byte pieces per thread and chunk

__global__ void __launch_bounds__(APPLY_THREADS, 2) salt_shrink_kernel(const __grid_constant__ ApplyParams p)
{
    extern __shared__ __align__(128) uint8_t smem_raw[];
    // 1024-byte aligned stage ring (the 128-byte swizzle atom of the UMMA operands)
    uint8_t *stages = smem_raw + ((1024 - (smem_u32(smem_raw) & 1023)) & 1023);
    float *P = reinterpret_cast<float *>(stages);
    float *RED = reinterpret_cast<float *>(stages + P_BYTES);
    ShrinkInfo &info = *reinterpret_cast<ShrinkInfo *>(stages + STAGES_BYTES);

    // Before the dependency wait this kernel reads only the segment tables
    // and the factors: the host launches it as a programmatic dependent only
    // when the previous kernel on the stream did not write those tables.
    cg::cluster_group cluster = cg::this_cluster();
    const int C = (int)cluster.num_blocks();
    const int crank = (int)cluster.block_rank();
    const int item = blockIdx.x / C;
    const int b = item / p.n_proj, pi = item - b * p.n_proj;
    const int n_blk = p.counts[3];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    // every CTA of a cluster takes the same exits, before any cluster barrier
    if (b >= n_blk || b >= p.blk_cap) {
        if (b < n_blk && tid == 0 && crank == 0 && pi == 0) atomicOr(p.err, SALT_DEVERR_RANK);
        pdl_wait();
        pdl_launch_dependents();
        return;
    }
    const ApplyProj &pr = p.proj[pi];
    const int4 m0 = *reinterpret_cast<const int4 *>(p.blk + BLK_INTS * b);
    const int4 m1 = *reinterpret_cast<const int4 *>(p.blk + BLK_INTS * b + 4);
    const int start = m0.x, M = m0.y, d = m0.z, rc = m0.w;
    const int S = rc + m1.x;
    const float s_c = __int_as_float(m1.y);
    if (S > S_MAX || S == 0) {
        if (S > S_MAX && tid == 0 && crank == 0) atomicOr(p.err, SALT_DEVERR_RANK);
        pdl_wait();
        pdl_launch_dependents();
        return;
    }
    const int d_in = pr.d_in;

    // ---- block setup from the segment tables
    if (tid < M) {
        const int t = tid;
        info.row[t] = p.perm[start + t];
        const int uo = p.tok_uoff[start + t];
        const int ur = p.tok_urank[start + t];
        info.ucol[t] = uo >= 0 ? rc + uo : -1;
        info.urank[t] = ur;
        info.usu[t] = p.tok_su[start + t];
        if (uo >= 0) {
            const bool head = t == 0 || p.tok_uoff[start + t - 1] != uo;
            const bool tail = t == M - 1 || p.tok_uoff[start + t + 1] != uo;
            for (int k = 0; k < ur; ++k) {
                const int s = rc + uo + k;
                if (s < S_MAX) {
                    if (head) {
                        info.rt0[s] = (int16_t)t;
                        info.rk[s] = (int16_t)k;
                    }
                    if (tail) info.rt1[s] = (int16_t)(t + 1);
                }
            }
        }
    }
    if (tid < S) {
        info.srcA[tid] = tid < rc ? pr.A + ((int64_t)d * p.rc_max + tid) * d_in
                                  : residual_row(p, pr, p.blk_res[(int64_t)b * S_MAX + (tid - rc)], false);
    }
    if (warp == 0) {
        tmem_alloc(smem_u32(&info.tmem), TMEM_COLS);
        tmem_relinquish();
    }
    if (tid == 0) {
        for (int s = 0; s < MAX_STAGES; ++s) mbar_init(smem_u32(&info.bar[s]), 1);
        mbar_fence_init();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = info.tmem;

    // ---- stage geometry: A = the factor stack (always 128 rows: the UMMA M
    // operand), X = the block's tokens rounded to the 16-row UMMA N step
    const int m_rows = ((M + 15) >> 4) << 4;
    const int stage_bytes = TILE_BYTES + m_rows * 128;
    const int nstage = min(MAX_STAGES, STAGES_BYTES / stage_bytes);
    const uint32_t ring = smem_u32(stages);
    const uint32_t idesc = idesc_bf16_f32(128, m_rows);

    // chunks are dealt round-robin over the cluster: at any moment the C CTAs
    // read adjacent pieces of every row
    const int nk = (d_in + KC - 1) / KC;
    const int n_my = nk > crank ? (nk - crank + C - 1) / C : 0;

    // each thread's 16-byte pieces of a chunk, resolved once
    // piece j of this thread is (row (tid + j*256) / 8, 16-byte chunk tid % 8),
    // the same for every j, so one column offset serves all pieces
    const int cb = (tid & 7) * 8;
    const uint16_t *a_src[MAX_PIECES];
    const uint16_t *x_src[MAX_PIECES];
#pragma unroll
    for (int j = 0; j < MAX_PIECES; ++j) {
        const int r = (tid + j * APPLY_THREADS) >> 3;
        a_src[j] = r < S ? info.srcA[r] + cb : nullptr;
        x_src[j] = r < M ? pr.x + (int64_t)info.row[r] * d_in + cb : nullptr;
    }
    auto load_a = [&](int i, int st) {
        const int k0 = (crank + i * C) * KC;
        const bool ok = k0 + cb < d_in;
        const uint32_t base = ring + st * stage_bytes;
#pragma unroll
        for (int j = 0; j < MAX_PIECES; ++j) {
            const int r = (tid + j * APPLY_THREADS) >> 3;
            if (r < S) cp_async16(base + swz128(r, tid & 7), a_src[j] + (ok ? k0 : 0), ok);
        }
    };
    auto load_x = [&](int i, int st) {
        const int k0 = (crank + i * C) * KC;
        const bool ok = k0 + cb < d_in;
        const uint32_t base = ring + st * stage_bytes + TILE_BYTES;
#pragma unroll
        for (int j = 0; j < MAX_PIECES; ++j) {
            const int r = (tid + j * APPLY_THREADS) >> 3;
            if (r < M) cp_async16(base + swz128(r, tid & 7), x_src[j] + (ok ? k0 : 0), ok);
        }
    };

    // ---- nstage-deep pipeline.  The factor rows of the first chunks are
    // requested before the dependency wait (no preceding kernel writes them),
    // x only after it; the first commit group carries those factor rows.
    bool ok_all = true;
    for (int s = 0; s < nstage - 1 && s < n_my; ++s) load_a(s, s);
    pdl_wait();
    // the expand may start once every CTA has passed the wait: anything it
    // reads before its own wait (y, B rows) is final by now
    pdl_launch_dependents();
    for (int s = 0; s < nstage - 1; ++s) {
        if (s < n_my) load_x(s, s);
        cp_async_commit();
    }
    for (int it = 0; it < n_my; ++it) {
        const int st = it % nstage;
        cp_async_wait_dyn(nstage - 2);
        fence_async_smem();
        __syncthreads();
        if (tid == 0) {
            tc_fence_after();
            const uint32_t sa = ring + st * stage_bytes, sx = sa + TILE_BYTES;
#pragma unroll
            for (int kk = 0; kk < KC / 16; ++kk)
                umma_bf16(tmem, sdesc_kmajor_sw128(sa + kk * 32), sdesc_kmajor_sw128(sx + kk * 32), idesc,
                          (it > 0 || kk > 0) ? 1u : 0u);
            umma_commit(smem_u32(&info.bar[st]));
        }
        const int nxt = it + nstage - 1;
        if (nxt < n_my) {
            // the stage of chunk nxt last held chunk it - 1: its MMAs must be done
            if (it >= 1 && !mbar_wait(smem_u32(&info.bar[(it - 1) % nstage]), ((it - 1) / nstage) & 1))
                ok_all = false;
            load_a(nxt, nxt % nstage);
            load_x(nxt, nxt % nstage);
        }
        cp_async_commit();
    }
    cp_async_wait<0>();
    if (n_my > 0 && !mbar_wait(smem_u32(&info.bar[(n_my - 1) % nstage]), ((n_my - 1) / nstage) & 1))
        ok_all = false;
    tc_fence_after();
    __syncthreads();  // the stage ring becomes the partial-sum area

    // ---- D^T (TMEM lanes = stack rows, columns = tokens) -> compact partials:
    // the centroid rows for every token, a user's rows for that user's tokens
    if (warp < 4) {
        const int s = warp * 32 + lane;
        int col = -1, t0 = 0, t1 = 0;
        if (s < rc) {
            col = s;
            t1 = M;
        } else if (s < S) {
            col = rc + info.rk[s];
            t0 = info.rt0[s];
            t1 = info.rt1[s];
        }
        for (int cg16 = 0; cg16 < (m_rows >> 4); ++cg16) {
            uint32_t v[16];
            if (n_my > 0) {
                tmem_ld16(tmem + ((uint32_t)(warp * 32) << 16) + cg16 * 16, v);
                tmem_ld_wait();
            } else {
#pragma unroll
                for (int e = 0; e < 16; ++e) v[e] = 0u;
            }
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                const int t = cg16 * 16 + e;
                if (col >= 0 && t >= t0 && t < t1) P[t * PW + col] = __uint_as_float(v[e]);
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tmem, TMEM_COLS);
    if (!ok_all) atomicOr(p.err, SALT_DEVERR_TIMEOUT);
    cluster.sync();

    // ---- reduce the rows this CTA owns over the cluster, scale, mask, store V_ext.
    // All peers' float4 pieces are requested before any is summed; the sum
    // runs in peer order, so the result does not depend on timing.
    const int S_pad = (S + 15) & ~15;
    const int r0 = crank * M / C, r1 = (crank + 1) * M / C;
    constexpr int PW4 = PW / 4;
    for (int idx = tid; idx < (r1 - r0) * PW4; idx += APPLY_THREADS) {
        const int rr = idx / PW4, c4 = idx - rr * PW4, row = r0 + rr;
        if (c4 * 4 < rc + info.urank[row]) {
            float4 v[MAX_CLUSTER];
#pragma unroll
            for (int qq = 0; qq < MAX_CLUSTER; ++qq)
                if (qq < C)
                    v[qq] = *reinterpret_cast<const float4 *>(cluster.map_shared_rank(P, qq) + row * PW + c4 * 4);
            float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
            for (int qq = 0; qq < MAX_CLUSTER; ++qq)
                if (qq < C) {
                    s.x += v[qq].x;
                    s.y += v[qq].y;
                    s.z += v[qq].z;
                    s.w += v[qq].w;
                }
            *reinterpret_cast<float4 *>(RED + rr * PW + c4 * 4) = s;
        }
    }
    __syncthreads();
    uint16_t *vt = p.vext + ((int64_t)pi * p.blk_cap + b) * (TM * VEXT_COLS);
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
        *reinterpret_cast<uint4 *>(vt + (int64_t)row * VEXT_COLS + c * 8) = make_uint4(w[0], w[1], w[2], w[3]);
    }
    cluster.sync();  // peers have read this CTA's partials
}

// ---------------------------------------------------------------------------- expand
// Persistent, one CTA per SM.  The items of a launch are (row block b,
// 64-column unit u) pairs in block-major order, u running over the columns
// of every projection of the group.  CTA i takes the items whose cost
// position (running sum of blk_weight, from the block records) falls in the
// i-th equal share of the total.  Per item, on the tensor cores:
//     D[128 x 64] = V_ext[128 x S] * Stack_B[S x 64]      (tcgen05.mma, fp32 in TMEM)
// with V_ext (K-major) resident in shared memory for the current
// (block, projection) and the stacked B rows (MN-major: the rows as they lie
// in memory) streamed with the item's y rows through an EX_STAGES-deep ring.
// The accumulator is double-buffered in TMEM: item j's MMAs run while the
// epilogue of item j-1 (TMEM -> registers, + staged y, one rounding, store)
// runs on all eight warps.
constexpr int EX_STAGES = 6;
constexpr int EX_STAGE_BYTES = 2 * TILE_BYTES;  // y rows | stacked B rows of one item
constexpr int EX_TMEM_COLS = 2 * NC;           // two 128 x 64 fp32 accumulators

struct ExpandInfo {
    const uint16_t *srcB[S_MAX];  // stacked B rows of the current (block, projection)
    int32_t row[TM];              // y row of the i-th token of the current block
    int32_t range[4];             // first item (block, unit), end item (block, unit)
    uint64_t bar[2];              // per accumulator: its MMAs have completed
    uint32_t tmem;
};
constexpr size_t EXPAND_SMEM = 1024 + EX_STAGES * EX_STAGE_BYTES + VT_BYTES + (sizeof(ExpandInfo) + 127) / 128 * 128;
static_assert(EXPAND_SMEM <= 227 * 1024, "expand shared memory exceeds the per-block limit");

__device__ __forceinline__ int64_t blk_wend(const int32_t *blk, int b) { return blk[(int64_t)BLK_INTS * b + BLK_WEND]; }

// First block b with nu * wend(b) > c, for 0 <= c < nu * wend(n_blk - 1).
// Whole warp; each step narrows the range 32-fold.
__device__ int find_block(const int32_t *blk, int n_blk, int64_t nu, int64_t c, int lane)
{
    int lo = 0, hi = n_blk;  // the answer lies in [lo, hi)
    while (hi - lo > 32) {
        const int step = (hi - lo + 31) >> 5;
        const int i = lo + lane * step;
        const bool past = i >= hi || nu * blk_wend(blk, i) > c;
        const unsigned m = __ballot_sync(0xffffffffu, past);
        const int f = m ? __ffs(m) - 1 : 32;
        const int nlo = f == 0 ? lo : lo + (f - 1) * step + 1;
        const int nhi = f == 32 ? hi : min(hi, lo + f * step + 1);
        lo = nlo;
        hi = nhi;
    }
    const int i = lo + lane;
    const bool past = i >= hi || nu * blk_wend(blk, i) > c;
    const unsigned m = __ballot_sync(0xffffffffu, past);
    return m ? lo + __ffs(m) - 1 : hi;
}

// First item whose cost start is >= c; (n_blk, 0) past the end.  Whole warp.
__device__ void item_at(const int32_t *blk, int n_blk, int nu, int64_t total, int64_t c, int lane, int &b, int &u)
{
    if (c >= total) {
        b = n_blk;
        u = 0;
        return;
    }
    b = find_block(blk, n_blk, nu, c, lane);
    const int64_t wend = blk_wend(blk, b), wbeg = b ? blk_wend(blk, b - 1) : 0;
    const int64_t w = wend - wbeg;
    const int64_t off = c - (int64_t)nu * wbeg;
    u = (int)((off + w - 1) / w);
    if (u >= nu) {
        ++b;
        u = 0;
    }
}

__global__ void __launch_bounds__(APPLY_THREADS, 1) salt_expand_kernel(const __grid_constant__ ApplyParams p)
{
    extern __shared__ __align__(128) uint8_t smem_raw[];
    // 1024-byte aligned ring (the 128-byte swizzle atom of the UMMA operands)
    uint8_t *ring = smem_raw + ((1024 - (smem_u32(smem_raw) & 1023)) & 1023);
    uint8_t *vs = ring + EX_STAGES * EX_STAGE_BYTES;  // V_ext: two K-major tiles (K 0..63, 64..127)
    ExpandInfo &info = *reinterpret_cast<ExpandInfo *>(vs + VT_BYTES);

    // The next apply's shrink reads only tables and factors before its own
    // dependency wait, so it may be scheduled as soon as this grid has started.
    pdl_launch_dependents();
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    // block records: written by the segment kernel, complete before the shrink began
    const int n_blk = min(p.counts[3], p.blk_cap);
    const int nu = p.n_unit_prefix[p.n_proj];
    if (n_blk <= 0 || nu <= 0) return;
    const int64_t total = (int64_t)nu * blk_wend(p.blk, n_blk - 1);
    if (warp < 2) {
        int b, u;
        item_at(p.blk, n_blk, nu, total, total * (blockIdx.x + warp) / gridDim.x, lane, b, u);
        if (lane == 0) {
            info.range[2 * warp] = b;
            info.range[2 * warp + 1] = u;
        }
    }
    if (warp == 2) {
        tmem_alloc(smem_u32(&info.tmem), EX_TMEM_COLS);
        tmem_relinquish();
    }
    if (tid == 0) {
        mbar_init(smem_u32(&info.bar[0]), 1);
        mbar_init(smem_u32(&info.bar[1]), 1);
        mbar_fence_init();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = info.tmem;
    int b = info.range[0], u = info.range[1];
    const int b_end = info.range[2], u_end = info.range[3];
    bool waited = false, ok_all = true;
    uint32_t n_done = 0;  // items of earlier runs (accumulator use count)
    const uint32_t ring32 = smem_u32(ring), vs32 = smem_u32(vs);
    const uint32_t idesc = idesc_bf16_f32_bmn(TM, NC);
    const int q = warp & 3, h = warp >> 2;  // epilogue: TMEM lane quarter, column half

    while (b < b_end || (b == b_end && u < u_end)) {
        // a run: consecutive items of one (block, projection)
        int pi = 0;
        while (pi + 1 < p.n_proj && p.n_unit_prefix[pi + 1] <= u) ++pi;
        const int u0 = u, cb = b;
        const int u_stop = min(p.n_unit_prefix[pi + 1], b == b_end ? u_end : nu);
        u = u_stop;
        if (u == nu) {
            ++b;
            u = 0;
        }
        const ApplyProj &pr = p.proj[pi];
        const int4 m0 = *reinterpret_cast<const int4 *>(p.blk + BLK_INTS * cb);
        const int4 m1 = *reinterpret_cast<const int4 *>(p.blk + BLK_INTS * cb + 4);
        const int start = m0.x, M = m0.y, d = m0.z, rc = m0.w;
        const int S = rc + m1.x;
        if (S > S_MAX || S == 0 || M <= 0) continue;  // the shrink flagged S > S_MAX
        const int S_pad = (S + 15) & ~15;
        const int d_out = pr.d_out;

        __syncthreads();  // the previous run is done with the ring, V and info
        if (tid < M) info.row[tid] = p.perm[start + tid];
        if (tid < S) {
            info.srcB[tid] = tid < rc ? pr.B + ((int64_t)d * p.rc_max + tid) * d_out
                                      : residual_row(p, pr, p.blk_res[(int64_t)cb * S_MAX + (tid - rc)], true);
        }
        __syncthreads();

        const int n = u_stop - u0;
        const int ubase = p.n_unit_prefix[pi];
        auto load_item = [&](int j) {
            const int n0 = (u0 + j - ubase) * NC;
            const uint32_t ys = ring32 + (j % EX_STAGES) * EX_STAGE_BYTES, bs = ys + TILE_BYTES;
            for (int idx = tid; idx < M * 8; idx += APPLY_THREADS) {
                const int r = idx >> 3, c = idx & 7, col = n0 + c * 8;
                const bool ok = col < d_out;
                cp_async16(ys + swz128(r, c), pr.y + (int64_t)info.row[r] * d_out + (ok ? col : 0), ok);
            }
            for (int idx = tid; idx < S_pad * 8; idx += APPLY_THREADS) {
                const int r = idx >> 3, c = idx & 7, col = n0 + c * 8;
                const bool ok = r < S && col < d_out;
                cp_async16(bs + swz128(r, c), ok ? info.srcB[r] + col : pr.y, ok);
            }
        };
        const uint16_t *vt = p.vext + ((int64_t)pi * p.blk_cap + cb) * (TM * VEXT_COLS);
        const int nch = S_pad >> 3;
        auto load_v = [&]() {
            for (int idx = tid; idx < M * nch; idx += APPLY_THREADS) {
                const int r = idx / nch, c = idx - r * nch;
                cp_async16(vs32 + (c >> 3) * TILE_BYTES + swz128(r, c & 7), vt + (int64_t)r * VEXT_COLS + c * 8, true);
            }
        };
        // commit groups: [V] P0 .. P(EX_STAGES-3) [V], then one per iteration
        const bool v_last = !waited;
        if (waited) {
            load_v();
            cp_async_commit();
        }
        for (int s = 0; s < EX_STAGES - 2; ++s) {
            if (s < n) load_item(s);
            cp_async_commit();
        }
        if (!waited) {
            // y and B rows above do not depend on the shrink; V does
            pdl_wait();
            waited = true;
            load_v();
            cp_async_commit();
        }

        for (int j = 0; j <= n; ++j) {
            if (j < n) {
                if (v_last && j == 0)
                    cp_async_wait<0>();
                else
                    cp_async_wait<EX_STAGES - 3>();
                fence_async_smem();
            }
            tc_fence_before();
            __syncthreads();  // item j is visible; the epilogue of item j-2 is over everywhere
            tc_fence_after();
            if (j < n && tid == 0) {
                const uint32_t cnt = n_done + j, buf = cnt & 1;
                const uint32_t sb = ring32 + (j % EX_STAGES) * EX_STAGE_BYTES + TILE_BYTES;
                for (int ks = 0; ks < (S_pad >> 4); ++ks)
                    umma_bf16(tmem + buf * NC, sdesc_kmajor_sw128(vs32 + (ks >> 2) * TILE_BYTES + (ks & 3) * 32),
                              sdesc_mnmajor_sw128(sb + ks * 2048), idesc, ks > 0 ? 1u : 0u);
                umma_commit(smem_u32(&info.bar[buf]));
            }
            // the stage of item j-2 is free: its MMAs and its epilogue are done
            if (j + EX_STAGES - 2 < n) load_item(j + EX_STAGES - 2);
            cp_async_commit();

            if (j >= 1) {
                const int jj = j - 1;
                const uint32_t cnt = n_done + jj, buf = cnt & 1;
                if (!mbar_wait(smem_u32(&info.bar[buf]), (cnt >> 1) & 1)) ok_all = false;
                tc_fence_after();
                uint32_t acc[32];
                const uint32_t ta = tmem + ((uint32_t)(q * 32) << 16) + buf * NC + h * 32;
                tmem_ld16(ta, *reinterpret_cast<uint32_t(*)[16]>(acc));
                tmem_ld16(ta + 16, *reinterpret_cast<uint32_t(*)[16]>(acc + 16));
                tmem_ld_wait();
                const int row = q * 32 + lane;
                if (row < M) {
                    const uint8_t *ysp = ring + (jj % EX_STAGES) * EX_STAGE_BYTES;
                    const int n0 = (u0 + jj - ubase) * NC + h * 32;
                    uint16_t *yg = pr.y + (int64_t)info.row[row] * d_out + n0;
#pragma unroll
                    for (int c = 0; c < 4; ++c) {
                        if (n0 + c * 8 < d_out) {
                            const uint4 v = *reinterpret_cast<const uint4 *>(ysp + swz128(row, h * 4 + c));
                            const uint32_t in[4] = {v.x, v.y, v.z, v.w};
                            uint32_t o[4];
#pragma unroll
                            for (int e = 0; e < 4; ++e) {
                                const float lo = bf16_to_f((uint16_t)(in[e] & 0xffffu)) + __uint_as_float(acc[c * 8 + 2 * e]);
                                const float hi = bf16_to_f((uint16_t)(in[e] >> 16)) + __uint_as_float(acc[c * 8 + 2 * e + 1]);
                                o[e] = (uint32_t)f_to_bf16(lo) | ((uint32_t)f_to_bf16(hi) << 16);
                            }
                            *reinterpret_cast<uint4 *>(yg + c * 8) = make_uint4(o[0], o[1], o[2], o[3]);
                        }
                    }
                }
            }
        }
        cp_async_wait<0>();
        n_done += n;
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 2) tmem_dealloc(tmem, EX_TMEM_COLS);
    if (!ok_all) atomicOr(p.err, SALT_DEVERR_TIMEOUT);
}

// Scratch of salt_lora_apply_static: V tiles for up to STATIC_APPLY_BLOCKS
// row blocks of one projection, in device memory that exists from module
// load to process exit (no allocation at run time).
__device__ __align__(256) uint16_t g_static_vext[STATIC_APPLY_BLOCKS * TM * VEXT_COLS];

}  // namespace

size_t apply_smem_bytes() { return SHRINK_SMEM; }

cudaError_t apply_static_workspace(uint16_t **out)
{
    // The host-side name of a __device__ array is not a device address:
    // resolve it once per device, with that device current.
    static std::mutex mu;
    static uint16_t *ptr[64] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(mu);
    if (!ptr[dev]) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_static_vext);
        if (e != cudaSuccess) return e;
        ptr[dev] = static_cast<uint16_t *>(p);
    }
    *out = ptr[dev];
    return cudaSuccess;
}

// SM count per device (the expand grid), filled by apply_prepare
static int g_sm_count[64];

cudaError_t apply_prepare(int device)
{
    if (device < 0 || device >= 64) return cudaErrorInvalidDevice;
    cudaError_t e = cudaDeviceGetAttribute(&g_sm_count[device], cudaDevAttrMultiProcessorCount, device);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(salt_shrink_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)SHRINK_SMEM);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(salt_shrink_kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(salt_expand_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)EXPAND_SMEM);
    return e;
}

cudaError_t launch_apply(const ApplyParams &p, int n_blk_bound, int cluster, bool shrink_pdl, cudaStream_t stream)
{
    if (n_blk_bound <= 0) return cudaSuccess;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = cluster;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.gridDim = dim3(cluster * p.n_proj * n_blk_bound, 1, 1);
    cfg.blockDim = dim3(APPLY_THREADS, 1, 1);
    cfg.dynamicSmemBytes = SHRINK_SMEM;
    cfg.stream = stream;
    cfg.attrs = attr;
    cfg.numAttrs = shrink_pdl ? 2 : 1;
    cudaError_t e = cudaLaunchKernelEx(&cfg, salt_shrink_kernel, p);
    if (e != cudaSuccess) return e;

    int dev = 0;
    e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const int n_sm = (dev >= 0 && dev < 64 && g_sm_count[dev] > 0) ? g_sm_count[dev] : 1;
    const int64_t items = (int64_t)p.n_unit_prefix[p.n_proj] * n_blk_bound;
    cudaLaunchConfig_t cfg2 = {};
    cudaLaunchAttribute attr2[1];
    attr2[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr2[0].val.programmaticStreamSerializationAllowed = 1;
    cfg2.gridDim = dim3((unsigned)(items < n_sm ? items : n_sm), 1, 1);
    cfg2.blockDim = dim3(APPLY_THREADS, 1, 1);
    cfg2.dynamicSmemBytes = EXPAND_SMEM;
    cfg2.stream = stream;
    cfg2.attrs = attr2;
    cfg2.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg2, salt_expand_kernel, p);
}

}  // namespace salt
