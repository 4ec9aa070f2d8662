// Fused centroid + residual apply (Section "Multi-Tenant Serving":
// W_final = W_base + gamma * Wbar + delta_i, evaluated in low-rank form).
//
// A row block (<= TM tokens of one domain, <= umax user runs, from the
// segment builder) concatenates its factors into one stack of
// S = rc + sum_u r_u rows, [A_c | a_u1 | a_u2 | ...] - the paper's long-tail
// identity (centroid and residual stacked into one ordinary adapter),
// applied per block - so each block is one dense contraction pair.
//
// One persistent kernel per apply, one CTA per SM, in two phases:
//
//   shrink units (row block b, projection, K-split s of KS): the unit's
//       contiguous range of 64-wide d_in chunks streams through a deep
//       shared-memory ring into the tensor cores,
//           V^T[S x M] (+)= Stack_A[S x chunk] * X[M x chunk]^T
//       (tcgen05.mma, fp32 accumulator in tensor memory; the stack is the
//       128-row operand, the tokens the N = 16..128 operand).  Each token
//       keeps the centroid columns and its own user's columns.  With KS = 1
//       the unit writes V_ext directly.  Otherwise every split stores an
//       fp32 partial, waits (bounded) until all splits of the block have,
//       and then reduces its own slice of the token rows over the splits in
//       split order (so the result does not depend on timing), writing
//           V_ext[t,s] = s_c V[t,s]    for s < rc (centroid rows; s_c is the
//                                      token's: the domain's scale times its gamma)
//                      = s_u V[t,s]    for s in the token's own user's rows
//                      = 0             otherwise
//       as bf16.  Each unit then counts its rows as written.
//   expand items (row block, 64 output columns), cost-balanced over CTAs:
//       Y[M x 64] += V_ext * Stack_B[:, cols] on the tensor cores (V_ext
//       K-major, the B rows MN-major as they lie in memory, four fp32
//       accumulators in tensor memory), the y and B rows of the next items
//       streaming through the ring meanwhile.  A run of items of one block
//       starts by prefetching its first items, then waits (bounded) until
//       every row of the block's V tile is written.  y is read once and
//       written once, rounded once.
//
// The arrival counters come in two halves chosen by the parity of a launch
// counter kept in device memory (the last CTA of a launch advances it); a
// launch zeroes the half the next launch uses, so graph replays of a launch
// stay correct.
//
// Operands are staged by cp.async in 128-byte-row, 128-byte-swizzled tiles
// (the layout the UMMA descriptors read).
#include <cuda_bf16.h>

#include <mutex>

#include "salt_async.cuh"
#include "salt_pipe.cuh"
#include "salt_internal.cuh"
#include "salt_tcgen05.cuh"

namespace salt {
namespace {

constexpr int KC = 64;                         // K chunk of the shrink (128-byte rows)
constexpr int NC = 64;                         // output columns per expand item
constexpr int TILE_BYTES = TM * 128;           // 128 rows x 128 B
constexpr int RING_BYTES = 216 * 1024;         // shared-memory ring of both phases
constexpr int A_MAX_STAGES = 8;
constexpr int B_MAX_STAGES = 10;               // expand: stages of (y rows | stacked B rows) per item
constexpr int PRODUCER_WARPS = 7;              // expand roles: producers, one MMA warp, epilogue warps
constexpr int PRODUCER_THREADS = 32 * PRODUCER_WARPS;
constexpr int EPI_WARPS = 4;
static_assert(PRODUCER_WARPS + 1 + EPI_WARPS == APPLY_THREADS / 32, "expand warp roles cover the CTA");
constexpr int TMEM_COLS = 512;                 // expand: N_ACC x 64 accumulator columns; shrink: D^T at DT_COL
constexpr int DT_COL = 256;                    // first column of the shrink accumulator (<= 128 tokens)
constexpr int N_ACC = 4;                       // expand accumulators in tensor memory
constexpr int KS_MAX = 16;
constexpr int VT_ROW = VEXT_COLS * 2;          // bytes per V tile row
constexpr int VT_BYTES = TM * VT_ROW;
// a deferred unit stages the sums of its slice (<= TM / 2 token rows: the
// block's non-empty splits are >= 2) in the V tile's region
static_assert((TM / 2) * SALT_MAX_TOKEN_RANK * 4 <= VT_BYTES, "deferred reduction staging exceeds the V tile");
static_assert(5 * 2 * TILE_BYTES + VT_BYTES <= RING_BYTES, "the expand ring must hold 5 full stages and the V tile");
static_assert(VT_BYTES <= RING_BYTES, "V staging exceeds the ring");
static_assert(S_MAX <= 128, "the factor stack is the 128-row UMMA operand");

struct FusedInfo {
    const uint16_t *src[S_MAX];  // shrink: stacked A rows of the current unit's block
    const uint16_t *esrc[S_MAX]; // expand: stacked B rows of the current run's block
    int32_t row[TM];             // shrink: x row of the i-th token of the unit's block
    int32_t erow[TM];            // expand: y row of the i-th token of the run's block
    int32_t ucol[TM];            // first stacked row of the token's user, -1: none
    int32_t urank[TM];
    float usu[TM];
    float usc[TM];               // the token's centroid scale
    int16_t rt0[S_MAX];          // residual stack row -> first token of its user run
    int16_t rt1[S_MAX];          //                    -> one past the last token
    int16_t rk[S_MAX];           //                    -> rank index within the user
    uint64_t bar[A_MAX_STAGES];  // shrink: per stage, its MMAs have completed
    // expand: full, empty per stage; acc full, acc empty; V full; run table published; item range published
    uint64_t bbar[2 * B_MAX_STAGES + 2 * N_ACC + 4];
    int32_t range[4];            // expand: first item (block, unit), end item (block, unit)
    uint32_t tmem;
    uint32_t epoch;
};
constexpr size_t FUSED_SMEM = 1024 + RING_BYTES + (sizeof(FusedInfo) + 127) / 128 * 128;
static_assert(FUSED_SMEM <= 227 * 1024, "shared memory exceeds the per-block limit");

__device__ __forceinline__ uint32_t ld_acquire(const uint32_t *p)
{
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];\n" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// Called by one thread after a CTA barrier: every write the CTA made before
// the barrier is visible GPU-wide before the counter moves.
__device__ __forceinline__ void signal_add(uint32_t *c)
{
    asm volatile("fence.acq_rel.gpu;\n" ::: "memory");
    atomicAdd(c, 1u);
}

// Bounded wait (about a quarter of a second) until the counter reads n.
__device__ bool wait_count(const uint32_t *c, uint32_t n)
{
    for (int i = 0; i < (1 << 22); ++i) {
        if (ld_acquire(c) == n) return true;
        __nanosleep(32);
    }
    return false;
}

// Residual row entry of a block's factor stack -> first element of that row.
__device__ __forceinline__ const uint16_t *residual_row(const ApplyParams &p, const ApplyProj &pr, int e, bool b_side)
{
    const int slot = res_slot(e), rank = res_rank(e), k = res_k(e);
    const uint16_t *base = reinterpret_cast<const uint16_t *>(p.pool + (int64_t)slot * p.slot_stride +
                                                              SALT_BLOB_HEADER_BYTES) + (int64_t)rank * pr.res_off;
    return b_side ? base + (int64_t)rank * pr.d_in + (int64_t)k * pr.d_out : base + (int64_t)k * pr.d_in;
}

// K-split s of KS over nk chunks: [nk * s / KS, nk * (s + 1) / KS)
// (s <= KS <= 16, so nk * s fits 32 bits for any d_in below 8e9)
__device__ __forceinline__ int split_lo(int nk, int s, int KS) { return nk * s / KS; }

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

// First expand item whose cost start is >= c; (n_blk, 0) past the end.  Whole warp.
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

// With no more (row block, projection) pairs than CTAs, each pair gets its
// own contiguous CTAs: one each, plus a share of the rest proportional to
// the pair's expand cost (its 64-column items times the block's weight), so
// that no CTA expands two pairs (a second run costs a table phase, a V wait
// and a refill of the ring: measured at 3-5 us, enough to make those CTAs
// the launch's tail).  The pair's items are split evenly over its CTAs.
// CTA g gets block *b and items [*u0, *u1) (absolute unit indices, u1 <= nu).
// Whole warp.
__device__ void pair_range(const ApplyParams &p, int n_blk, int nu, int g, int lane, int &b, int &u0, int &u1)
{
    const int G = gridDim.x, np = p.n_proj;
    const int n_bp = n_blk * np;
    const int64_t R = G - n_bp;  // CTAs beyond one per pair
    const int64_t total = (int64_t)nu * blk_wend(p.blk, n_blk - 1);
    // first CTA of pair j = (bb, pi): j + floor(C_j * R / total), C_j its cost prefix
    auto first_cta = [&](int bb, int pi) -> int64_t {
        if (bb >= n_blk) return G;
        const int64_t wbeg = bb ? blk_wend(p.blk, bb - 1) : 0;
        const int64_t w = blk_wend(p.blk, bb) - wbeg;
        const int64_t C = (int64_t)nu * wbeg + (int64_t)p.n_unit_prefix[pi] * w;
        return (int64_t)bb * np + pi + (total > 0 ? C * R / total : 0);
    };
    // the last block whose first pair starts at or before g
    int lo = 0, hi = n_blk;  // answer in [lo, hi)
    while (hi - lo > 1) {
        const int step = (hi - lo + 31) >> 5;
        const int i = lo + lane * step;
        const bool le = i < hi && first_cta(i, 0) <= g;
        const unsigned m = __ballot_sync(0xffffffffu, le);
        const int last = 31 - __clz(m);  // lane 0 always holds (first_cta(lo, 0) <= g)
        lo = lo + last * step;
        hi = min(hi, lo + step);
    }
    b = lo;
    int pi = 0;
    while (pi + 1 < np && first_cta(b, pi + 1) <= g) ++pi;
    const int64_t f0 = first_cta(b, pi);
    const int64_t f1 = pi + 1 < np ? first_cta(b, pi + 1) : first_cta(b + 1, 0);
    const int64_t c = f1 - f0, k = g - f0;
    const int base = p.n_unit_prefix[pi], U = p.n_unit_prefix[pi + 1] - base;
    u0 = base + (int)(k * U / c);
    u1 = base + (int)((k + 1) * U / c);
}

constexpr int MAX_PIECES = (TM * 8 + APPLY_THREADS - 1) / APPLY_THREADS;  // 16-byte pieces per thread and chunk
constexpr int N_QUADS = APPLY_THREADS / 128;  // full groups of 4 warps (one per TMEM lane quarter)
constexpr int EPI_WARP0 = PRODUCER_WARPS + 1;  // first epilogue warp
constexpr int EPI_THREADS = 32 * EPI_WARPS;
constexpr int ROLE_THREADS = 32 * EPI_WARP0;   // producers + the MMA warp
// named barriers (id 0 is __syncthreads)
constexpr int BAR_EPI = 2;                     // the epilogue warps
constexpr int BAR_ROLES = 3;                   // producers + the MMA warp
constexpr int BAR_ALL = 4;                     // every thread (the inline unit finish)

// The work of a shrink unit after its K loop, done by `nthr` threads
// (warps first_warp .. first_warp + nthr/32 - 1, a whole number of groups of
// four so that every TMEM lane quarter is read): with one split, V_ext
// straight from the accumulator; otherwise the fp32 partial, the wait for
// the other splits of the block, the reduction of this unit's slice of the
// token rows over the splits (in split order) and the V rows written.  Then
// the unit's rows are counted as written.  The shrink tables of the unit
// (info.usc / usu / ucol / urank / rt0 / rt1 / rk) must still hold; Ps is
// shared memory for the sums of the slice (its rows x PART_COLS floats).
struct UnitGeom {
    int unit, pair, s, b, pi, KS;
    int M, rc, S, m_rows, nk, c0;
};

__device__ __forceinline__ UnitGeom unit_geom(const ApplyParams &p, int unit, int KS)
{
    UnitGeom g;
    g.unit = unit;
    g.KS = KS;
    g.pair = unit / KS;
    g.s = unit - g.pair * KS;
    g.b = g.pair / p.n_proj;
    g.pi = g.pair - g.b * p.n_proj;
    const int4 m0 = *reinterpret_cast<const int4 *>(p.blk + BLK_INTS * g.b);
    const int4 m1 = *reinterpret_cast<const int4 *>(p.blk + BLK_INTS * g.b + 4);
    g.M = m0.y;
    g.rc = m0.w;
    g.S = g.rc + m1.x;
    g.m_rows = ((g.M + 15) >> 4) << 4;
    g.nk = (p.proj[g.pi].d_in + KC - 1) / KC;
    g.c0 = split_lo(g.nk, g.s, KS);
    return g;
}

__device__ void finish_split_unit(const ApplyParams &p, FusedInfo &info, const UnitGeom &g, uint32_t tmem,
                                  uint32_t epoch, int first_warp, int nthr, int bar_id, float *Ps, bool &ok_all)
{
    const int tid = threadIdx.x - 32 * first_warp, lane = threadIdx.x & 31;
    const int wrel = tid >> 5, q = (threadIdx.x >> 5) & 3, th = wrel >> 2, nth = nthr >> 7;
    const int M = g.M, rc = g.rc, S = g.S, KS = g.KS, nk = g.nk;
    const int n_pairs = SALT_MAX_GROUP * p.w.blk_cap;
    const int64_t pidx = (int64_t)g.pi * p.w.blk_cap + g.b;
    uint16_t *vt = p.w.vext + pidx * (TM * VEXT_COLS);
    const int S_pad = (S + 15) & ~15;
    const int nch = S_pad >> 3;
    const int n_ne = min(KS, nk);  // splits with at least one chunk

    // fp32 partial: token t's centroid columns, then its own user's columns
    const int sr = q * 32 + lane;
    int t0 = 0, t1 = 0, col = -1;  // tokens this stack row serves, its compact column
    if (sr < rc) {
        t1 = M;
        col = sr;
    } else if (sr < S) {
        t0 = info.rt0[sr];
        t1 = info.rt1[sr];
        col = rc + info.rk[sr];
    }
    float *P = p.w.part + (int64_t)g.unit * (TM * PART_COLS);
    for (int gg = th; gg < (g.m_rows >> 4); gg += nth) {
        uint32_t v[16];
        tmem_ld16(tmem + ((uint32_t)(q * 32) << 16) + DT_COL + gg * 16, v);
        tmem_ld_wait();
        if (col >= 0) {
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                const int t = gg * 16 + e;
                if (t < M && t >= t0 && t < t1) P[t * PART_COLS + col] = __uint_as_float(v[e]);
            }
        }
    }
    tc_fence_before();
    named_sync(bar_id, nthr);
    // every split of the block stores its partial, then each reduces its own
    // slice of the token rows over all splits, in split order
    if (tid == 0) {
        uint32_t *ctr = p.w.arrive + (epoch & 1) * n_pairs + pidx;
        signal_add(ctr);
        if (!wait_count(ctr, n_ne)) ok_all = false;
    }
    named_sync(bar_id, nthr);
    // the non-empty splits: all of them unless d_in has fewer chunks than splits
    uint32_t ne_mask = KS >= 32 ? ~0u : (1u << KS) - 1u;
    if (nk < KS) {
        ne_mask = 0;
        for (int s2 = 0; s2 < KS; ++s2)
            if (split_lo(nk, s2 + 1, KS) > split_lo(nk, s2, KS)) ne_mask |= 1u << s2;
    }
    const int si = nk >= KS ? g.s : g.c0;  // index among the non-empty splits
    const int r0 = M * si / n_ne, r1 = M * (si + 1) / n_ne;
    // sums of the slice's partial columns (centroid, then the token's own
    // user's), in split order, staged in shared memory, then scaled, masked
    // and written as bf16 V rows
    constexpr int PC4 = PART_COLS / 4;
    const int n_it = (r1 - r0) * PC4;
    // (row, 4 columns) items of the slice; with up to 8 splits a thread
    // takes two items at once, so all of its loads are in flight together
    constexpr int KS_PAIR = 8;
    for (int idx = tid; KS <= KS_PAIR && idx < n_it; idx += 2 * nthr) {
        float4 v[2][KS_PAIR];
        bool use[2];
        const float *src[2];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int it = idx + h * nthr, rr = it / PC4, c4 = it - rr * PC4, t = r0 + rr;
            use[h] = it < n_it && c4 * 4 < rc + info.urank[t];
            src[h] = p.w.part + ((int64_t)g.pair * KS * TM + t) * PART_COLS + c4 * 4;
#pragma unroll
            for (int s2 = 0; s2 < KS_PAIR; ++s2) {
                v[h][s2] = make_float4(0.f, 0.f, 0.f, 0.f);
                if (use[h] && ((ne_mask >> s2) & 1))
                    v[h][s2] = __ldcg(reinterpret_cast<const float4 *>(src[h] + (int64_t)s2 * (TM * PART_COLS)));
            }
        }
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            if (!use[h]) continue;
            float4 acc = v[h][0];
#pragma unroll
            for (int s2 = 1; s2 < KS_PAIR; ++s2) {
                acc.x += v[h][s2].x;
                acc.y += v[h][s2].y;
                acc.z += v[h][s2].z;
                acc.w += v[h][s2].w;
            }
            const int it = idx + h * nthr, rr = it / PC4, c4 = it - rr * PC4;
            *reinterpret_cast<float4 *>(Ps + rr * PART_COLS + c4 * 4) = acc;
        }
    }
    for (int idx = tid; KS > KS_PAIR && idx < n_it; idx += nthr) {
        const int rr = idx / PC4, c4 = idx - rr * PC4, t = r0 + rr;
        if (c4 * 4 >= rc + info.urank[t]) continue;
        float4 v[KS_MAX];
        const float *src = p.w.part + ((int64_t)g.pair * KS * TM + t) * PART_COLS + c4 * 4;
#pragma unroll
        for (int s2 = 0; s2 < KS_MAX; ++s2) {
            v[s2] = make_float4(0.f, 0.f, 0.f, 0.f);
            if ((ne_mask >> s2) & 1)
                v[s2] = __ldcg(reinterpret_cast<const float4 *>(src + (int64_t)s2 * (TM * PART_COLS)));
        }
        float4 acc = v[0];
#pragma unroll
        for (int s2 = 1; s2 < KS_MAX; ++s2) {
            acc.x += v[s2].x;
            acc.y += v[s2].y;
            acc.z += v[s2].z;
            acc.w += v[s2].w;
        }
        *reinterpret_cast<float4 *>(Ps + rr * PART_COLS + c4 * 4) = acc;
    }
    named_sync(bar_id, nthr);
    for (int idx = tid; idx < (r1 - r0) * nch; idx += nthr) {
        const int rr = idx / nch, ch = idx - rr * nch, t = r0 + rr;
        const int uc = info.ucol[t], ur = info.urank[t];
        const float us = info.usu[t], sc = info.usc[t];
        const float *ps = Ps + rr * PART_COLS;
        uint32_t w4[4];
#pragma unroll
        for (int hh = 0; hh < 4; ++hh) {
            uint16_t v2[2];
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                const int c = ch * 8 + 2 * hh + e;
                float val = 0.f;
                if (c < rc) val = sc * ps[c];
                else if (uc >= 0 && c >= uc && c < uc + ur) val = us * ps[rc + (c - uc)];
                v2[e] = f_to_bf16(val);
            }
            w4[hh] = (uint32_t)v2[0] | ((uint32_t)v2[1] << 16);
        }
        *reinterpret_cast<uint4 *>(vt + t * VEXT_COLS + ch * 8) = make_uint4(w4[0], w4[1], w4[2], w4[3]);
    }
    // the staging area becomes the V tile of a TMA load later
    fence_async_smem();
    // this unit's rows of the block's V tile are written
    named_sync(bar_id, nthr);
    if (tid == 0) signal_add(p.w.vdone + (epoch & 1) * n_pairs + pidx);
}

__global__ void __launch_bounds__(APPLY_THREADS, 1) salt_apply_kernel(const __grid_constant__ ApplyParams p)
{
    extern __shared__ __align__(128) uint8_t smem_raw[];
    // 1024-byte aligned ring (the 128-byte swizzle atom of the UMMA operands)
    uint8_t *ring = smem_raw + ((1024 - (smem_u32(smem_raw) & 1023)) & 1023);
    FusedInfo &info = *reinterpret_cast<FusedInfo *>(ring + RING_BYTES);
    const uint32_t ring32 = smem_u32(ring);
    uint16_t *Vs = reinterpret_cast<uint16_t *>(ring);  // shrink: V tile staging [TM][VEXT_COLS]

    // Before the dependency wait this kernel reads only the segment tables
    // and the factors: the host launches it as a programmatic dependent only
    // when the previous kernel on the stream did not write those tables.
    // The next kernel may be scheduled as soon as every CTA of this one runs.
    pdl_launch_dependents();
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int n_blk = min(p.counts[3], p.w.blk_cap);
    if (p.counts[3] > p.w.blk_cap && blockIdx.x == 0 && threadIdx.x == 0) atomicOr(p.err, SALT_DEVERR_RANK);
    const int nu = p.n_unit_prefix[p.n_proj];
    if (n_blk <= 0 || nu <= 0) return;  // the same for every CTA
    const int n_bp = n_blk * p.n_proj;
    int KS = max(1, min(KS_MAX, (int)gridDim.x / n_bp));
    if (KS > 1 && (int64_t)n_bp * KS > p.w.part_cap) KS = max(1, p.w.part_cap / n_bp);
    const int n_units = n_bp * KS;
    // With at most one unit per CTA the units go to the lowest CTA indices:
    // the CTAs of a launch start in index order as the previous launch's
    // CTAs leave their SMs, so the last ones to start (up to a few
    // microseconds late) are the ones without a shrink unit, and no block
    // waits for a late split.
    const int ua = n_units <= (int)gridDim.x ? min((int)blockIdx.x, n_units)
                                             : (int)((int64_t)n_units * blockIdx.x / gridDim.x);
    const int ub = n_units <= (int)gridDim.x ? min((int)blockIdx.x + 1, n_units)
                                             : (int)((int64_t)n_units * (blockIdx.x + 1) / gridDim.x);

    const uint32_t bb = smem_u32(&info.bbar[0]);
    auto full_bar = [&](int st) { return bb + 8u * st; };
    auto empty_bar = [&](int st) { return bb + 8u * (B_MAX_STAGES + st); };
    auto accf_bar = [&](int i) { return bb + 8u * (2 * B_MAX_STAGES + i); };
    auto acce_bar = [&](int i) { return bb + 8u * (2 * B_MAX_STAGES + N_ACC + i); };
    const uint32_t vfull_bar = bb + 8u * (2 * B_MAX_STAGES + 2 * N_ACC);
    const uint32_t tbl_bar = vfull_bar + 8u;    // a run's table is written (producers -> epilogue)
    const uint32_t range_bar = vfull_bar + 16u; // the CTA's item range is written
    const uint32_t stg_bar = vfull_bar + 24u;   // the epilogue no longer stages in the V tile region
    if (warp == 2) {
        tmem_alloc(smem_u32(&info.tmem), TMEM_COLS);
        tmem_relinquish();
    }
    if (tid == 0) {
        for (int i = 0; i < A_MAX_STAGES; ++i) mbar_init(smem_u32(&info.bar[i]), 1);
        // The expand's barriers are set up once; their phases run on across
        // runs: item g (counted over all runs of this CTA) uses slot
        // g % B_MAX_STAGES and accumulator g % N_ACC, the r-th run's V tile
        // and table the r-th phases of "V full" and "table".
        for (int st = 0; st < B_MAX_STAGES; ++st) {
            mbar_init(full_bar(st), PRODUCER_THREADS);
            mbar_init(empty_bar(st), 1 + EPI_WARPS);
        }
        for (int i = 0; i < N_ACC; ++i) {
            mbar_init(accf_bar(i), 1);
            mbar_init(acce_bar(i), EPI_WARPS);
        }
        mbar_init(vfull_bar, 1);
        mbar_init(tbl_bar, 1);
        mbar_init(range_bar, 1);
        mbar_init(stg_bar, 1);
        mbar_fence_init();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = info.tmem;
    bool ok_all = true, waited = false;
    // Once per CTA: wait for the previous kernel on the stream (x and y may be
    // its outputs), then read this launch's epoch; its parity selects the
    // half of the counters this launch uses.
    const int n_pairs = SALT_MAX_GROUP * p.w.blk_cap;
    // (No barrier here: the epoch is first used after the K loop, whose CTA
    // barriers publish it; the x loads need not wait for it.)
    auto dep_wait = [&]() {
        pdl_wait();
        waited = true;
        if (tid == 0) info.epoch = *reinterpret_cast<volatile uint32_t *>(p.w.seq);
    };

    // This CTA's share of the expand items: the first (e = 0) or end (e = 1)
    // item of its range, into info.range; one warp each.  With split
    // shrinks, searched by warps 0 and 1 when the shrink phase is over
    // (while the block's splits are reduced), so that the first shrink
    // unit's table phase does not wait for the search; with single splits,
    // during that table phase.
    bool have_range = false;
    auto find_range = [&](int e) {
        int b = n_blk, u = 0;  // no expand items when only the V tiles are wanted
        if (p.shrink_only) {
        } else if (n_bp <= (int)gridDim.x) {
            int u0, u1;
            pair_range(p, n_blk, nu, blockIdx.x, lane, b, u0, u1);
            u = e ? u1 : u0;
        } else {
            const int64_t total = (int64_t)nu * blk_wend(p.blk, n_blk - 1);
            item_at(p.blk, n_blk, nu, total, total * (blockIdx.x + e) / gridDim.x, lane, b, u);
        }
        if (lane == 0) {
            info.range[2 * e] = b;
            info.range[2 * e + 1] = u;
        }
    };

    // ================================================================ shrink units
    uint32_t a_phase = 0;  // parity of the next completion of each stage barrier
    // The CTA's last unit of a split shrink is finished by the epilogue warps
    // while the producers already stream the first expand items.
    bool deferred = false;
    UnitGeom dgeom{};
    for (int unit = ua; unit < ub; ++unit) {
        const UnitGeom g = unit_geom(p, unit, KS);
        const int b = g.b;
        const ApplyProj &pr = p.proj[g.pi];
        const int start = p.blk[BLK_INTS * b + BLK_START], d = p.blk[BLK_INTS * b + BLK_DOM];
        const int M = g.M, rc = g.rc, S = g.S;
        const int d_in = pr.d_in;
        const int nk = g.nk;
        const int c0 = g.c0, n_my = split_lo(nk, g.s + 1, KS) - c0;
        if (S > S_MAX || S == 0 || M <= 0 || n_my <= 0) {
            if (S > S_MAX && g.s == 0 && tid == 0) atomicOr(p.err, SALT_DEVERR_RANK);
            continue;
        }
        __syncthreads();  // the previous unit is done with info and the ring
        // the token and factor tables (threads 64..191); with single splits
        // (the expand follows each unit at once) warps 0 and 1 meanwhile
        // find the CTA's expand items
        if (KS == 1 && !have_range && warp < 2) {
            find_range(warp);
        } else if (tid >= 64 && tid < 64 + TM) {
            const int t = tid - 64;
            if (t < M) {
                info.row[t] = p.perm[start + t];
                const int uo = p.tok_uoff[start + t];
                const int ur = p.tok_urank[start + t];
                info.ucol[t] = uo >= 0 ? rc + uo : -1;
                info.urank[t] = ur;
                info.usu[t] = p.tok_su[start + t];
                info.usc[t] = p.tok_sc[start + t];
                if (uo >= 0) {
                    const bool head = t == 0 || p.tok_uoff[start + t - 1] != uo;
                    const bool tail = t == M - 1 || p.tok_uoff[start + t + 1] != uo;
                    for (int k = 0; k < ur; ++k) {
                        const int sr = rc + uo + k;
                        if (sr < S_MAX) {
                            if (head) {
                                info.rt0[sr] = (int16_t)t;
                                info.rk[sr] = (int16_t)k;
                            }
                            if (tail) info.rt1[sr] = (int16_t)(t + 1);
                        }
                    }
                }
            }
            if (t < S) {
                info.src[t] = t < rc ? pr.A + ((int64_t)d * p.rc_max + t) * d_in
                                     : residual_row(p, pr, p.blk_res[(int64_t)b * S_MAX + (t - rc)], false);
            }
        }
        have_range = have_range || KS == 1;
        __syncthreads();

        // stage geometry: A = the factor stack (the 128-row UMMA M operand; rows
        // >= S are never read back), X = the block's tokens rounded to the
        // 16-row UMMA N step
        const int m_rows = g.m_rows;
        const int stage_bytes = TILE_BYTES + m_rows * 128;
        const int nstage = min(A_MAX_STAGES, RING_BYTES / stage_bytes);
        const uint32_t idesc = idesc_bf16_f32(128, m_rows);
        // each thread's 16-byte pieces of a chunk: piece j is (row (tid + j*384) / 8,
        // 16-byte column tid % 8), so one column offset serves all pieces
        const int cb = (tid & 7) * 8;
        const uint16_t *a_src[MAX_PIECES];
        const uint16_t *x_src[MAX_PIECES];
#pragma unroll
        for (int j = 0; j < MAX_PIECES; ++j) {
            const int r = (tid + j * APPLY_THREADS) >> 3;
            a_src[j] = r < S ? info.src[r] + cb : nullptr;
            x_src[j] = r < M ? pr.x + (int64_t)info.row[r] * d_in + cb : nullptr;
        }
        auto load_a = [&](int i, int st) {
            const int k0 = (c0 + i) * KC;
            const bool ok = k0 + cb < d_in;
            const uint32_t base = ring32 + st * stage_bytes;
#pragma unroll
            for (int j = 0; j < MAX_PIECES; ++j) {
                const int r = (tid + j * APPLY_THREADS) >> 3;
                if (r < S) cp_async16(base + swz128(r, tid & 7), a_src[j] + (ok ? k0 : 0), ok);
            }
        };
        auto load_x = [&](int i, int st) {
            const int k0 = (c0 + i) * KC;
            const bool ok = k0 + cb < d_in;
            const uint32_t base = ring32 + st * stage_bytes + TILE_BYTES;
#pragma unroll
            for (int j = 0; j < MAX_PIECES; ++j) {
                const int r = (tid + j * APPLY_THREADS) >> 3;
                if (r < M) cp_async16(base + swz128(r, tid & 7), x_src[j] + (ok ? k0 : 0), ok);
            }
        };

        // nstage-deep pipeline; the factor rows of the first chunks are
        // requested before the dependency wait, x only after it; the first
        // commit group carries those factor rows
        for (int st = 0; st < nstage - 1 && st < n_my; ++st) load_a(st, st);
        if (!waited) dep_wait();
        for (int st = 0; st < nstage - 1; ++st) {
            if (st < n_my) load_x(st, st);
            cp_async_commit();
        }
        uint32_t pending = 0;  // stages with a commit not yet waited for
        for (int it = 0; it < n_my; ++it) {
            const int st = it % nstage;
            cp_async_wait_dyn(nstage - 2);
            fence_async_smem();
            __syncthreads();
            if (tid == 0) {
                tc_fence_after();
                const uint32_t sa = ring32 + st * stage_bytes, sx = sa + TILE_BYTES;
#pragma unroll
                for (int kk = 0; kk < KC / 16; ++kk)
                    umma_bf16(tmem + DT_COL, sdesc_kmajor_sw128(sa + kk * 32), sdesc_kmajor_sw128(sx + kk * 32), idesc,
                              (it > 0 || kk > 0) ? 1u : 0u);
                umma_commit(smem_u32(&info.bar[st]));
            }
            pending |= 1u << st;
            const int nxt = it + nstage - 1;
            if (nxt < n_my) {
                // the stage of chunk nxt last held chunk it - 1: its MMAs must be done
                if (it >= 1) {
                    const int ps = (it - 1) % nstage;
                    if (!mbar_wait(smem_u32(&info.bar[ps]), (a_phase >> ps) & 1)) ok_all = false;
                    a_phase ^= 1u << ps;
                    pending &= ~(1u << ps);
                }
                load_a(nxt, nxt % nstage);
                load_x(nxt, nxt % nstage);
            }
            cp_async_commit();
        }
        cp_async_wait<0>();
        // every commit is waited for exactly once, keeping the parities in step
        for (int st = 0; st < nstage; ++st)
            if ((pending >> st) & 1) {
                if (!mbar_wait(smem_u32(&info.bar[st]), (a_phase >> st) & 1)) ok_all = false;
                a_phase ^= 1u << st;
            }
        tc_fence_after();

        if (KS == 1) {
            // ---- V_ext straight from the accumulator (TMEM lanes = stack rows,
            // columns = tokens) into the staging tile.  Warp w of the first
            // N_QUADS groups of four reads lanes 32 (w % 4) .. + 31 and every
            // N_QUADS-th 16-token group.
            const int q = warp & 3, th = warp >> 2;
            const int sr = q * 32 + lane;
            int t0 = 0, t1 = 0;  // tokens this stack row serves
            if (sr < rc) {
                t1 = M;
            } else if (sr < S) {
                t0 = info.rt0[sr];
                t1 = info.rt1[sr];
            }
            const int S_pad = (S + 15) & ~15;
            const int64_t pidx = (int64_t)g.pi * p.w.blk_cap + b;
            uint16_t *vt = p.w.vext + pidx * (TM * VEXT_COLS);
            const int nch = S_pad >> 3;
            for (int gg = th; th < N_QUADS && gg < (m_rows >> 4); gg += N_QUADS) {
                uint32_t v[16];
                tmem_ld16(tmem + ((uint32_t)(q * 32) << 16) + DT_COL + gg * 16, v);
                tmem_ld_wait();
                if (sr < S_pad) {
#pragma unroll
                    for (int e = 0; e < 16; ++e) {
                        const int t = gg * 16 + e;
                        if (t < M) {
                            float val = 0.f;
                            if (sr < rc) val = info.usc[t] * __uint_as_float(v[e]);
                            else if (t >= t0 && t < t1) val = info.usu[t] * __uint_as_float(v[e]);
                            Vs[t * VEXT_COLS + sr] = f_to_bf16(val);
                        }
                    }
                }
            }
            tc_fence_before();
            __syncthreads();
            for (int idx = tid; idx < M * nch; idx += APPLY_THREADS) {
                const int r = idx / nch, c = idx - r * nch;
                *reinterpret_cast<uint4 *>(vt + r * VEXT_COLS + c * 8) =
                    *reinterpret_cast<const uint4 *>(Vs + r * VEXT_COLS + c * 8);
            }
            __syncthreads();
            if (tid == 0) signal_add(p.w.vdone + (info.epoch & 1) * n_pairs + pidx);
        } else if (unit + 1 < ub || min(KS, nk) < 2) {
            // a later unit of this CTA reuses the accumulator, or the slice
            // (the whole block when d_in has one chunk) would not fit the V
            // tile's region: finish now, all threads
            __syncthreads();  // info.epoch is published
            finish_split_unit(p, info, g, tmem, info.epoch, 0, APPLY_THREADS, BAR_ALL,
                              reinterpret_cast<float *>(ring), ok_all);
        } else {
            deferred = true;
            dgeom = g;
        }
    }
    if (!waited) dep_wait();
    tc_fence_before();
    __syncthreads();  // the shrink phase is over: the ring changes hands
    tc_fence_after();
    const uint32_t epoch = info.epoch;

    // ================================================================ expand items
    // Warp roles per run of items of one (block, projection):
    //   warps 0-6  producers: cp.async of each item's y rows and stacked B
    //              rows into a stage; each thread's copies complete on the
    //              stage's "full" barrier;
    //   warp 7     one thread waits for the block's V tile to be written,
    //              loads it (TMA), then issues the MMAs of an item into one
    //              of N_ACC accumulators and commits them to "acc full" and
    //              "empty";
    //   warps 8-11 first the deferred split unit (partial, reduction, V
    //              rows), then the epilogue: TMEM lanes 32 (w % 4) .. + 31
    //              (one token row a thread), the item's 64 columns: + staged
    //              y, one rounding, store; then "acc empty" and "empty".
    //              In a run that fits the ring the epilogue writes the
    //              results back into the stage and the producers, whose loads
    //              are all issued, store them.
    // The producers do not wait for V: y and B do not depend on it, so the
    // first items stream in while the splits are reduced.
    uint8_t *vs = ring + RING_BYTES - VT_BYTES;  // V_ext: two K-major tiles (K 0..63, 64..127)
    const uint32_t vs32 = smem_u32(vs);
    const uint32_t idesc_b = idesc_bf16_f32_bmn(TM, NC);
    if (warp < EPI_WARP0) {
        // the counters of the next launch start from zero (the previous
        // launch, which used them, is complete)
        const int nxt = ((epoch + 1) & 1) * n_pairs;
        for (int i = blockIdx.x * ROLE_THREADS + tid; i < n_pairs; i += gridDim.x * ROLE_THREADS) {
            p.w.arrive[nxt + i] = 0u;
            p.w.vdone[nxt + i] = 0u;
        }
        if (!have_range && warp < 2) find_range(warp);
        named_sync(BAR_ROLES, ROLE_THREADS);
        if (tid == 0) mbar_arrive_release(range_bar);
    } else {
        // the sums are staged in the V tile's region, unused until this
        // CTA's V rows (among others) are written
        if (deferred)
            finish_split_unit(p, info, dgeom, tmem, epoch, EPI_WARP0, EPI_THREADS, BAR_EPI,
                              reinterpret_cast<float *>(vs), ok_all);
        // the V tile region is free for the MMA warp's first V load (its
        // staging writes go before those TMA writes)
        fence_async_smem();
        named_sync(BAR_EPI, EPI_THREADS);
        if (tid == 32 * EPI_WARP0) mbar_arrive_release(stg_bar);
        if (!mbar_wait(range_bar, 0)) ok_all = false;
    }
    int b = info.range[0], u = info.range[1];
    const int b_end = info.range[2], u_end = info.range[3];
    uint32_t g0 = 0, runs = 0;  // items and runs of this CTA so far
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
        if (S > S_MAX || S == 0 || M <= 0) continue;  // flagged by the shrink phase
        const int S_pad = (S + 15) & ~15;
        const int d_out = pr.d_out;
        const int n = u_stop - u0;
        const int ubase = p.n_unit_prefix[pi];
        // stages sized to this block: y rows rounded to 16, then the stacked
        // B rows (both parts start on 2048-byte boundaries)
        const int m_rows = ((M + 15) >> 4) << 4;
        const int bst = (m_rows + S_pad) * 128;
        const int nbs = min(B_MAX_STAGES, (RING_BYTES - VT_BYTES) / bst);
        // a run whose items all fit the ring at once: the producers, idle
        // after its loads, store its results (see below)
        const bool pstore = n <= nbs;

        // The run's table: written by the producers and the MMA warp,
        // published to the epilogue warps through "table" (the previous run
        // is over in every role: the CTA barrier at the end of each run).
        if (warp < EPI_WARP0) {
            if (tid < M) info.erow[tid] = p.perm[start + tid];
            if (tid >= TM && tid - TM < S) {
                const int t = tid - TM;
                info.esrc[t] = t < rc ? pr.B + ((int64_t)d * p.rc_max + t) * d_out
                                      : residual_row(p, pr, p.blk_res[(int64_t)cb * S_MAX + (t - rc)], true);
            }
            named_sync(BAR_ROLES, ROLE_THREADS);
            if (tid == 0) mbar_arrive_release(tbl_bar);
        }

        if (warp < PRODUCER_WARPS) {
            auto load_item = [&](int j) {
                const int n0 = (u0 + j - ubase) * NC;
                const uint32_t ys = ring32 + (j % nbs) * bst, bs = ys + m_rows * 128;
                for (int idx = tid; idx < M * 8; idx += PRODUCER_THREADS) {
                    const int r = idx >> 3, c = idx & 7, col = n0 + c * 8;
                    const bool ok = col < d_out;
                    cp_async16(ys + swz128(r, c), pr.y + (int64_t)info.erow[r] * d_out + (ok ? col : 0), ok);
                }
                for (int idx = tid; idx < S_pad * 8; idx += PRODUCER_THREADS) {
                    const int r = idx >> 3, c = idx & 7, col = n0 + c * 8;
                    const bool ok = r < S && col < d_out;
                    cp_async16(bs + swz128(r, c), ok ? info.esrc[r] + col : pr.y, ok);
                }
                cp_async_commit();
                cp_async_arrive_noinc(full_bar((g0 + j) % B_MAX_STAGES));
            };
            const int npre = min(n, nbs);
            for (int j = 0; j < npre; ++j) load_item(j);
            for (int j = npre; j < n; ++j) {
                // the stage last held item j - nbs of this run
                const uint32_t gp = g0 + j - nbs;
                if (!mbar_wait(empty_bar(gp % B_MAX_STAGES), (gp / B_MAX_STAGES) & 1)) ok_all = false;
                load_item(j);
            }
            if (pstore) {
                // A run that fits the ring: every load is issued, so the
                // producers store the items' results (written back into their
                // stages by the epilogue warps) as each stage empties, 8
                // threads per 128-byte row piece, and the epilogue warps go on
                // to the next accumulator at once.
                for (int j = 0; j < n; ++j) {
                    const uint32_t gp = g0 + j;
                    if (!mbar_wait(empty_bar(gp % B_MAX_STAGES), (gp / B_MAX_STAGES) & 1)) ok_all = false;
                    const int n0 = (u0 + j - ubase) * NC;
                    const uint8_t *ysp = ring + (j % nbs) * bst;
                    for (int idx = tid; idx < M * 8; idx += PRODUCER_THREADS) {
                        const int r = idx >> 3, c = idx & 7, col = n0 + c * 8;
                        if (col < d_out)
                            *reinterpret_cast<uint4 *>(pr.y + (int64_t)info.erow[r] * d_out + col) =
                                *reinterpret_cast<const uint4 *>(ysp + swz128(r, c));
                    }
                }
            }
            cp_async_wait<0>();
        } else if (warp == PRODUCER_WARPS) {
            if (lane == 0) {
                // V: once every row of the block's tile is written, two TMA tile
                // loads (K 0..63 and 64..127, each straight into the K-major
                // 128-byte-swizzled layout) complete on "V full" by byte count.
                const int n_ne = min(KS, (pr.d_in + KC - 1) / KC);
                const int64_t pidx = (int64_t)pi * p.w.blk_cap + cb;
                // (the first run's load waits until the epilogue warps have
                // staged their deferred sums in the same region)
                if (runs == 0 && !mbar_wait(stg_bar, 0)) ok_all = false;
                if (!wait_count(p.w.vdone + (epoch & 1) * n_pairs + pidx, n_ne)) ok_all = false;
                fence_proxy_async_global();  // the tile was written through the generic proxy
                const int row0 = (int)(pidx * TM);
                mbar_expect_tx(vfull_bar, 2 * TILE_BYTES);
                tma_load_2d(vs32, &p.w.vmap, 0, row0, vfull_bar);
                tma_load_2d(vs32 + TILE_BYTES, &p.w.vmap, 64, row0, vfull_bar);
                if (!mbar_wait(vfull_bar, runs & 1)) ok_all = false;
                for (int j = 0; j < n; ++j) {
                    const uint32_t gi = g0 + j, slot = gi % B_MAX_STAGES, buf = gi % N_ACC;
                    if (!mbar_wait(full_bar(slot), (gi / B_MAX_STAGES) & 1)) ok_all = false;
                    if (gi >= N_ACC && !mbar_wait(acce_bar(buf), ((gi / N_ACC) - 1) & 1)) ok_all = false;
                    fence_async_smem();
                    tc_fence_after();
                    const uint32_t sb = ring32 + (j % nbs) * bst + m_rows * 128;
                    for (int ks = 0; ks < (S_pad >> 4); ++ks)
                        umma_bf16(tmem + buf * NC, sdesc_kmajor_sw128(vs32 + (ks >> 2) * TILE_BYTES + (ks & 3) * 32),
                                  sdesc_mnmajor_sw128(sb + ks * 2048), idesc_b, ks > 0 ? 1u : 0u);
                    umma_commit(accf_bar(buf));
                    umma_commit(empty_bar(slot));
                }
            }
            __syncwarp();
        } else {
            if (!mbar_wait(tbl_bar, runs & 1)) ok_all = false;
            const int q = warp & 3;
            const int row = q * 32 + lane;
            // the y rows this thread stores: 8 lanes per 128-byte row piece, 4 rows per store
            int32_t srow[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const int r = q * 32 + i * 4 + (lane >> 3);
                srow[i] = r < M ? info.erow[r] : -1;
            }
            for (int j = 0; j < n; ++j) {
                const uint32_t gi = g0 + j, slot = gi % B_MAX_STAGES, buf = gi % N_ACC;
                const int st = j % nbs;
                if (!mbar_wait(accf_bar(buf), (gi / N_ACC) & 1)) ok_all = false;
                tc_fence_after();
                uint32_t acc[64];
                const uint32_t ta = tmem + ((uint32_t)(q * 32) << 16) + buf * NC;
#pragma unroll
                for (int g = 0; g < 4; ++g) tmem_ld16(ta + 16 * g, *reinterpret_cast<uint32_t(*)[16]>(acc + 16 * g));
                tmem_ld_wait();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive_relaxed(acce_bar(buf));
                // the staged y rows of the item (its "full" phase has completed)
                if (!mbar_wait(full_bar(slot), (gi / B_MAX_STAGES) & 1)) ok_all = false;
                // y + delta, rounded once, back into the staged tile (this
                // thread's row) ...
                uint8_t *ysp = ring + st * bst;
                const int n0 = (u0 + j - ubase) * NC;
                if (row < M) {
                    // all loads first: the swizzled cells do not alias, but the
                    // compiler cannot tell, so interleaved stores would serialise
                    uint32_t yv[32];
#pragma unroll
                    for (int c = 0; c < 8; ++c) {
                        const uint4 v = *reinterpret_cast<const uint4 *>(ysp + swz128(row, c));
                        yv[4 * c] = v.x;
                        yv[4 * c + 1] = v.y;
                        yv[4 * c + 2] = v.z;
                        yv[4 * c + 3] = v.w;
                    }
#pragma unroll
                    for (int i = 0; i < 32; ++i)
                        yv[i] = add_bf16x2(yv[i], __uint_as_float(acc[2 * i]), __uint_as_float(acc[2 * i + 1]));
#pragma unroll
                    for (int c = 0; c < 8; ++c)
                        *reinterpret_cast<uint4 *>(ysp + swz128(row, c)) =
                            make_uint4(yv[4 * c], yv[4 * c + 1], yv[4 * c + 2], yv[4 * c + 3]);
                }
                __syncwarp();
                if (pstore) {
                    // the producers store the item once its stage is empty
                    if (lane == 0) mbar_arrive_release(empty_bar(slot));
                    continue;
                }
                // ... then the warp's 32 rows go out whole (all reads first)
                {
                    uint4 vv[8];
                    int64_t off[8];
#pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        const int r = q * 32 + i * 4 + (lane >> 3), c = lane & 7, col = n0 + c * 8;
                        const bool ok = srow[i] >= 0 && col < d_out;
                        vv[i] = ok ? *reinterpret_cast<const uint4 *>(ysp + swz128(r, c)) : make_uint4(0u, 0u, 0u, 0u);
                        off[i] = ok ? (int64_t)srow[i] * d_out + col : -1;
                    }
#pragma unroll
                    for (int i = 0; i < 8; ++i)
                        if (off[i] >= 0) *reinterpret_cast<uint4 *>(pr.y + off[i]) = vv[i];
                }
                __syncwarp();
                if (lane == 0) mbar_arrive_relaxed(empty_bar(slot));
            }
        }
        g0 += n;
        ++runs;
        // the run is over in every role: its MMAs have completed (the epilogue
        // saw each accumulator full), so the ring, the V tile and the run
        // table may take the next run's rows
        __syncthreads();
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 2) tmem_dealloc(tmem, TMEM_COLS);
    if (!ok_all) atomicOr(p.err, SALT_DEVERR_TIMEOUT);
    // the last CTA to finish advances the epoch (every CTA read it above)
    if (tid == 0) {
        __threadfence();
        const uint32_t done = atomicAdd(p.w.seq + 1, 1u);
        if (done == gridDim.x - 1) {
            atomicExch(p.w.seq + 1, 0u);
            __threadfence();
            atomicAdd(p.w.seq, 1u);
        }
    }
}

// Scratch of salt_lora_apply_static: V tiles, partial tiles, flags and the
// epoch for up to STATIC_APPLY_BLOCKS row blocks of one projection, in device
// memory that exists from module load to process exit (no allocation at run
// time).  Zero-initialised.
__device__ __align__(256) uint16_t g_static_vext[STATIC_APPLY_BLOCKS * TM * VEXT_COLS];
static_assert(sizeof(g_static_vext) == (size_t)1 * STATIC_APPLY_BLOCKS * TM * VEXT_COLS * 2,
              "the static V tiles are the extent the static tensor map encodes (one projection)");
__device__ __align__(256) float g_static_part[STATIC_PART_CAP * TM * PART_COLS];
__device__ __align__(256) uint32_t g_static_arrive[2 * SALT_MAX_GROUP * STATIC_APPLY_BLOCKS];
__device__ __align__(256) uint32_t g_static_vdone[2 * SALT_MAX_GROUP * STATIC_APPLY_BLOCKS];
__device__ __align__(256) uint32_t g_static_seq[2];

// SM count per device (the grid of the apply kernel), filled by apply_prepare
int g_sm_count[64];

// A device word nothing ever writes: the failure-path self-test waits on it.
__device__ uint32_t g_never_set;

// One thread waits for g_never_set to read 1 through the bounded wait the
// apply uses for other CTAs' results; it gives up and raises the timeout flag.
__global__ void salt_wait_selftest_kernel(uint32_t *err)
{
    if (threadIdx.x == 0 && blockIdx.x == 0 && !wait_count(&g_never_set, 1u)) atomicOr(err, SALT_DEVERR_TIMEOUT);
}

}  // namespace

size_t apply_smem_bytes() { return FUSED_SMEM; }

cudaError_t apply_static_workspace(ApplyWork *out)
{
    // The host-side name of a __device__ array is not a device address:
    // resolve them once per device, with that device current.
    static std::mutex mu;
    static ApplyWork ws[64] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(mu);
    if (!ws[dev].vext) {
        ApplyWork w = {};
        void *a = nullptr, *b = nullptr, *c = nullptr, *d = nullptr, *f = nullptr;
        if ((e = cudaGetSymbolAddress(&a, g_static_vext)) != cudaSuccess) return e;
        if ((e = cudaGetSymbolAddress(&b, g_static_part)) != cudaSuccess) return e;
        if ((e = cudaGetSymbolAddress(&c, g_static_arrive)) != cudaSuccess) return e;
        if ((e = cudaGetSymbolAddress(&d, g_static_vdone)) != cudaSuccess) return e;
        if ((e = cudaGetSymbolAddress(&f, g_static_seq)) != cudaSuccess) return e;
        w.vext = static_cast<uint16_t *>(a);
        w.blk_cap = STATIC_APPLY_BLOCKS;
        w.max_group = 1;  // one projection per call: the V array holds exactly these tiles
        w.part = static_cast<float *>(b);
        w.part_cap = STATIC_PART_CAP;
        w.arrive = static_cast<uint32_t *>(c);
        w.vdone = static_cast<uint32_t *>(d);
        w.seq = static_cast<uint32_t *>(f);
        if ((e = apply_encode_vmap(w)) != cudaSuccess) return e;
        ws[dev] = w;
    }
    *out = ws[dev];
    return cudaSuccess;
}

cudaError_t encode_base_map(CUtensorMap *out, const uint16_t *W, int d_in, int d_out, int layout)
{
    using Encode = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
    static Encode encode = nullptr;
    static std::mutex mu;
    {
        std::lock_guard<std::mutex> lock(mu);
        if (!encode) {
            void *fn = nullptr;
            cudaDriverEntryPointQueryResult q;
            cudaError_t e = cudaGetDriverEntryPoint("cuTensorMapEncodeTiled", &fn, cudaEnableDefault, &q);
            if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !fn) return e != cudaSuccess ? e : cudaErrorNotSupported;
            encode = reinterpret_cast<Encode>(fn);
        }
    }
    // IN_OUT: [d_in][d_out], inner dimension N, box 64 N x 64 K;
    // OUT_IN: [d_out][d_in], inner dimension K, box 64 K x 128 N
    const bool in_out = layout == SALT_W_IN_OUT;
    const cuuint64_t dims[2] = {(cuuint64_t)(in_out ? d_out : d_in), (cuuint64_t)(in_out ? d_in : d_out)};
    const cuuint64_t strides[1] = {(cuuint64_t)(in_out ? d_out : d_in) * 2};
    const cuuint32_t box[2] = {64, in_out ? 64u : 128u};
    const cuuint32_t es[2] = {1, 1};
    const CUresult r = encode(out, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<uint16_t *>(W), dims, strides, box, es,
                              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

cudaError_t apply_encode_vmap(ApplyWork &w)
{
    using Encode = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
    static Encode encode = nullptr;
    static std::mutex mu;
    {
        std::lock_guard<std::mutex> lock(mu);
        if (!encode) {
            void *fn = nullptr;
            cudaDriverEntryPointQueryResult q;
            cudaError_t e = cudaGetDriverEntryPoint("cuTensorMapEncodeTiled", &fn, cudaEnableDefault, &q);
            if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !fn) return e != cudaSuccess ? e : cudaErrorNotSupported;
            encode = reinterpret_cast<Encode>(fn);
        }
    }
    if (w.max_group < 1 || w.max_group > SALT_MAX_GROUP || w.blk_cap < 1) return cudaErrorInvalidValue;
    const cuuint64_t dims[2] = {(cuuint64_t)VEXT_COLS, (cuuint64_t)w.max_group * w.blk_cap * TM};
    const cuuint64_t strides[1] = {(cuuint64_t)VEXT_COLS * 2};
    const cuuint32_t box[2] = {64, (cuuint32_t)TM};
    const cuuint32_t es[2] = {1, 1};
    const CUresult r = encode(&w.vmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, w.vext, dims, strides, box, es,
                              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

cudaError_t apply_prepare(int device)
{
    if (device < 0 || device >= 64) return cudaErrorInvalidDevice;
    cudaError_t e = cudaDeviceGetAttribute(&g_sm_count[device], cudaDevAttrMultiProcessorCount, device);
    if (e != cudaSuccess) return e;
    return cudaFuncSetAttribute(salt_apply_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)FUSED_SMEM);
}

cudaError_t launch_wait_selftest(uint32_t *err, cudaStream_t stream)
{
    salt_wait_selftest_kernel<<<1, 32, 0, stream>>>(err);
    return cudaGetLastError();
}

cudaError_t launch_apply(const ApplyParams &p, bool pdl, cudaStream_t stream)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const int n_sm = (dev >= 0 && dev < 64 && g_sm_count[dev] > 0) ? g_sm_count[dev] : 1;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.gridDim = dim3(n_sm, 1, 1);
    cfg.blockDim = dim3(APPLY_THREADS, 1, 1);
    cfg.dynamicSmemBytes = FUSED_SMEM;
    cfg.stream = stream;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, salt_apply_kernel, p);
}

}  // namespace salt
