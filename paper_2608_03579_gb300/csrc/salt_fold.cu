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
// One launch folds one weight or a table of them (a fold plan: every
// adapted weight of a model when a node starts, with no gap between the
// weights).  Items are (weight, 128-row tile of W, 64 columns), numbered
// weight by weight; each CTA (one per SM) takes a contiguous range of them,
// so it mostly stays on one row tile.  The CTA is
// split into warp roles joined by mbarriers, so reads, tensor-core work,
// epilogue and write-back of different items overlap:
//   warp 0     TMA loads of the W tile (128 x 64, 128-byte swizzle) and of
//              the Q columns (MN-major, rows >= rc zero-filled by the copy)
//              into a ring of stages;
//   warp 1     tensor memory and the MMAs: D[128 x 64] = P_tile^T Q_chunk
//              into one of four accumulators;
//   warp 2     P^T of each row tile into a K-major swizzled A tile (two
//              buffers), an 8 x 8 register transpose per 16-byte chunk;
//   warps 3-6  the epilogue, one W row a thread: scale * D added to the W
//              tile in shared memory in fp32, rounded once to bf16, and the
//              tile written back by a TMA store; the stage is released once
//              the store has read it.
// Rows >= Mdim and columns >= Ndim are zero on load and clipped on store.
#include "salt_async.cuh"
#include "salt_internal.cuh"
#include "salt_pipe.cuh"
#include "salt_tcgen05.cuh"

#include <cstring>
#include <mutex>

namespace salt {
namespace {

constexpr int FOLD_THREADS = 224;
constexpr int FOLD_TM = 128;                          // W rows per tile (UMMA M)
constexpr int FOLD_NC = 64;                           // W columns per item (UMMA N)
constexpr int FOLD_STAGES = 7;
constexpr int FOLD_NACC = 4;                          // TMEM accumulators of FOLD_NC columns
constexpr int FOLD_W_BYTES = FOLD_TM * 128;           // [128 rows][64 columns], swizzled rows
constexpr int FOLD_Q_BYTES = 64 * 128;                // [K <= 64][64 columns], MN-major
constexpr int FOLD_STAGE_BYTES = FOLD_W_BYTES + FOLD_Q_BYTES;
constexpr int FOLD_A_BYTES = FOLD_TM * 128;           // [128 rows][K <= 64], K-major
constexpr int FOLD_SMEM = 1024 + 2 * FOLD_A_BYTES + FOLD_STAGES * FOLD_STAGE_BYTES;
constexpr int FOLD_EPI_WARP0 = 3;
constexpr int FOLD_EPI_THREADS = 128;
constexpr int FOLD_BAR_EPI = 1;                       // named barrier of the epilogue warps
static_assert(FOLD_SMEM <= 227 * 1024, "fold shared memory");
static_assert(FOLD_THREADS == 32 * FOLD_EPI_WARP0 + FOLD_EPI_THREADS, "warp roles");
static_assert(SALT_MAX_CENTROID_RANK <= 64, "K of the fold is one 128-byte row");

// One weight of a fold launch.  In a plan's device table the records lie
// back to back, so the two maps stay 64-byte aligned.
struct alignas(64) FoldMat {
    CUtensorMap wmap;   // W[Mdim][Ndim], box 64 x 128, 128-byte swizzle
    CUtensorMap qmap;   // Q[rc][Ndim], box 64 x kpad, 128-byte swizzle
    const uint16_t *P;  // [rc][Mdim]
    int64_t item0;      // the weight's first item in the launch
    int32_t Mdim, Ndim, rc, pad;
};

struct FoldParams {
    FoldMat one;           // the weight of a single-weight launch
    const FoldMat *mats;   // a plan's table in device memory, or null: `one`
    int32_t n_mats;
    int64_t items;         // items of all weights
    float scale;
    uint32_t *err;
};

// the weight that holds item `it` (item0 ascending, mats[0].item0 = 0)
__device__ __forceinline__ int fold_find(const FoldMat *M, int nm, int64_t it)
{
    int lo = 0, hi = nm - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (M[mid].item0 <= it) lo = mid;
        else hi = mid - 1;
    }
    return lo;
}
__device__ __forceinline__ void fold_advance(const FoldMat *M, int nm, int64_t it, int &mat)
{
    while (mat + 1 < nm && it >= M[mat + 1].item0) ++mat;
}
// a table map written by the host is read by the TMA unit through the
// tensor-map proxy
__device__ __forceinline__ void tensormap_acquire(const CUtensorMap *map)
{
    asm volatile("fence.proxy.tensormap::generic.acquire.gpu [%0], 128;\n" ::"l"(map) : "memory");
}

__device__ __forceinline__ void tma_store_2d(const CUtensorMap *map, uint32_t src, int x, int y)
{
    asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.tile.bulk_group [%0, {%1, %2}], [%3];\n" ::"l"(map), "r"(x),
                 "r"(y), "r"(src)
                 : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void bulk_wait_read() { asm volatile("cp.async.bulk.wait_group.read %0;\n" ::"n"(N) : "memory"); }
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;\n" ::: "memory"); }

// 8 x 8 transpose of 16-bit elements held as 8 rows of 4 words (element 2j
// in the low half of word j): three levels of off-diagonal block swaps
__device__ __forceinline__ void transpose8x8(uint32_t (&w)[8][4])
{
#pragma unroll
    for (int i = 0; i < 4; ++i) {  // 4 x 4 blocks: rows i, i + 4
        uint32_t t0 = w[i][2], t1 = w[i][3];
        w[i][2] = w[i + 4][0];
        w[i][3] = w[i + 4][1];
        w[i + 4][0] = t0;
        w[i + 4][1] = t1;
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) {  // 2 x 2 blocks: rows i, i + 2 within each half
        if (i & 2) continue;
#pragma unroll
        for (int j = 0; j < 4; j += 2) {
            uint32_t t = w[i][j + 1];
            w[i][j + 1] = w[i + 2][j];
            w[i + 2][j] = t;
        }
    }
#pragma unroll
    for (int i = 0; i < 8; i += 2) {  // single elements: rows i, i + 1
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const uint32_t x = w[i][j], y = w[i + 1][j];
            w[i][j] = __byte_perm(x, y, 0x5410);
            w[i + 1][j] = __byte_perm(x, y, 0x7632);
        }
    }
}

__global__ void __launch_bounds__(FOLD_THREADS, 1) salt_fold_kernel(const __grid_constant__ FoldParams p)
{
    extern __shared__ __align__(128) uint8_t smem_raw[];
    uint8_t *base = smem_raw + ((1024 - (smem_u32(smem_raw) & 1023)) & 1023);
    const uint32_t a32 = smem_u32(base);                        // two A tiles
    const uint32_t st32 = a32 + 2 * FOLD_A_BYTES;               // the ring: W tile, then Q tile, per stage
    __shared__ uint64_t full_bar[FOLD_STAGES], empty_bar[FOLD_STAGES];
    __shared__ uint64_t afull_bar[2], aempty_bar[2], tfull_bar[FOLD_NACC], tempty_bar[FOLD_NACC];
    __shared__ uint32_t tmem_slot;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const bool table = p.mats != nullptr;
    const FoldMat *M = table ? p.mats : &p.one;
    const int nm = table ? p.n_mats : 1;
    const int64_t items = p.items;
    const int64_t i0 = items * blockIdx.x / gridDim.x, i1 = items * (blockIdx.x + 1) / gridDim.x;
    if (i0 >= i1) return;  // the same for every thread of the CTA
    const int n_my = (int)(i1 - i0);

    if (warp == 1) {
        tmem_alloc(smem_u32(&tmem_slot), FOLD_NACC * FOLD_NC);
        tmem_relinquish();
    }
    if (tid == 0) {
        for (int s = 0; s < FOLD_STAGES; ++s) {
            mbar_init(smem_u32(&full_bar[s]), 1);
            mbar_init(smem_u32(&empty_bar[s]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_u32(&afull_bar[b]), 32);
            mbar_init(smem_u32(&aempty_bar[b]), 1);
        }
        for (int a = 0; a < FOLD_NACC; ++a) {
            mbar_init(smem_u32(&tfull_bar[a]), 1);
            mbar_init(smem_u32(&tempty_bar[a]), FOLD_EPI_THREADS);
        }
        mbar_fence_init();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;
    bool ok_all = true;
    // Launched with programmatic dependent launch: the set-up above overlaps
    // the tail of the previous kernel on the stream; every global access
    // below waits until that kernel has completed and its writes are visible
    // (a fold of the same weight may be the one before).
    pdl_launch_dependents();
    pdl_wait();

    if (warp == 0) {
        // ---------------------------------------------------------- TMA loads
        if (lane == 0) {
            int n_issued = 0, mat = fold_find(M, nm, i0), mat_seen = -1;
            for (int j = 0; j < n_my && ok_all; ++j) {
                const int s = j % FOLD_STAGES;
                if (j >= FOLD_STAGES && !mbar_wait(smem_u32(&empty_bar[s]), (uint32_t)(j / FOLD_STAGES - 1) & 1u)) {
                    ok_all = false;
                    break;
                }
                const int64_t it = i0 + j;
                fold_advance(M, nm, it, mat);
                const FoldMat &F = M[mat];
                if (table && mat != mat_seen) {
                    tensormap_acquire(&F.wmap);
                    tensormap_acquire(&F.qmap);
                    mat_seen = mat;
                }
                const int n_ct = (F.Ndim + FOLD_NC - 1) / FOLD_NC;
                const int64_t loc = it - F.item0;
                const int m0 = (int)(loc / n_ct) * FOLD_TM, n0 = (int)(loc % n_ct) * FOLD_NC;
                const uint32_t sw = st32 + (uint32_t)s * FOLD_STAGE_BYTES, bar = smem_u32(&full_bar[s]);
                mbar_expect_tx(bar, (uint32_t)FOLD_W_BYTES + (uint32_t)((F.rc + 15) & ~15) * 128u);
                tma_load_2d(sw, &F.wmap, n0, m0, bar);
                tma_load_2d(sw + FOLD_W_BYTES, &F.qmap, n0, 0, bar);
                n_issued = j + 1;
            }
            // every copy issued has landed before the CTA may exit
            for (int j = n_issued - FOLD_STAGES > 0 ? n_issued - FOLD_STAGES : 0; j < n_issued; ++j)
                if (!mbar_wait(smem_u32(&full_bar[j % FOLD_STAGES]), (uint32_t)(j / FOLD_STAGES) & 1u)) ok_all = false;
        }
    } else if (warp == 1) {
        // ---------------------------------------------------------- MMAs
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16_f32_bmn(FOLD_TM, FOLD_NC);
            int mat = fold_find(M, nm, i0), key_mat = -1, key_rt = -1, n_tiles = 0, abuf = 0;
            for (int j = 0; j < n_my && ok_all; ++j) {
                const int64_t it = i0 + j;
                fold_advance(M, nm, it, mat);
                const FoldMat &F = M[mat];
                const int n_ct = (F.Ndim + FOLD_NC - 1) / FOLD_NC;
                const int rt = (int)((it - F.item0) / n_ct);
                if (mat != key_mat || rt != key_rt) {  // a new (weight, row tile): its A tile
                    abuf = n_tiles & 1;
                    if (!mbar_wait(smem_u32(&afull_bar[abuf]), (uint32_t)(n_tiles >> 1) & 1u)) { ok_all = false; break; }
                    ++n_tiles;
                    key_mat = mat;
                    key_rt = rt;
                }
                const int s = j % FOLD_STAGES, acc = j % FOLD_NACC;
                if (!mbar_wait(smem_u32(&full_bar[s]), (uint32_t)(j / FOLD_STAGES) & 1u)) { ok_all = false; break; }
                if (j >= FOLD_NACC && !mbar_wait(smem_u32(&tempty_bar[acc]), (uint32_t)(j / FOLD_NACC - 1) & 1u)) {
                    ok_all = false;
                    break;
                }
                tc_fence_after();
                const uint32_t a = a32 + (uint32_t)abuf * FOLD_A_BYTES;
                const uint32_t q = st32 + (uint32_t)s * FOLD_STAGE_BYTES + FOLD_W_BYTES;
                const int kpad = (F.rc + 15) & ~15;
                for (int kk = 0; kk < kpad / 16; ++kk)
                    umma_bf16(tmem + (uint32_t)acc * FOLD_NC, sdesc_kmajor_sw128(a + kk * 32),
                              sdesc_mnmajor_sw128(q + kk * 2048), idesc, kk > 0 ? 1u : 0u);
                umma_commit(smem_u32(&tfull_bar[acc]));
                // the A tile is free once the last MMA of its row tile has completed
                const bool last_of_tile = j + 1 == n_my ||
                                          (mat + 1 < nm && it + 1 >= M[mat + 1].item0) ||
                                          (int)((it + 1 - F.item0) / n_ct) != rt;
                if (last_of_tile) umma_commit(smem_u32(&aempty_bar[abuf]));
            }
        }
    } else if (warp == 2) {
        // ---------------------------------------------------------- P^T tiles
        // the CTA's (weight, row tile) pairs in item order
        int64_t it = i0;
        int mat = fold_find(M, nm, i0);
        for (int t = 0; it < i1 && ok_all; ++t) {
            fold_advance(M, nm, it, mat);
            const FoldMat &F = M[mat];
            const int n_ct = (F.Ndim + FOLD_NC - 1) / FOLD_NC;
            const int rt = (int)((it - F.item0) / n_ct);
            const int Mdim = F.Mdim, rc = F.rc, kb_n = ((rc + 15) & ~15) / 8;
            const uint16_t *P = F.P;
            const int b = t & 1;
            if (t >= 2 && !mbar_wait(smem_u32(&aempty_bar[b]), (uint32_t)((t >> 1) - 1) & 1u)) {
                ok_all = false;
                break;
            }
            uint8_t *A = base + b * FOLD_A_BYTES;
            const int m0 = rt * FOLD_TM;
            // 8 x 8 blocks (k block kb, m block mb); a warp's lanes take
            // consecutive k blocks first, so the 16-byte stores of one m row
            // group fall into distinct swizzled chunks
            for (int idx = lane; idx < kb_n * (FOLD_TM / 8); idx += 32) {
                const int kb = idx % kb_n, mb = idx / kb_n, m = m0 + mb * 8;
                uint32_t w[8][4];
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    const int k = kb * 8 + i;
                    uint4 v = make_uint4(0u, 0u, 0u, 0u);
                    if (k < rc && m < Mdim) v = *reinterpret_cast<const uint4 *>(P + (int64_t)k * Mdim + m);
                    w[i][0] = v.x;
                    w[i][1] = v.y;
                    w[i][2] = v.z;
                    w[i][3] = v.w;
                }
                transpose8x8(w);
#pragma unroll
                for (int i = 0; i < 8; ++i) {  // row mb * 8 + i of the tile: K chunk kb
                    const int r = mb * 8 + i;
                    *reinterpret_cast<uint4 *>(A + swz128(r, kb)) = make_uint4(w[i][0], w[i][1], w[i][2], w[i][3]);
                }
            }
            // K columns [kpad, 64) are never read by the MMAs
            fence_async_smem();
            mbar_arrive_release(smem_u32(&afull_bar[b]));
            // the next row tile's first item
            const int64_t nxt = F.item0 + (int64_t)(rt + 1) * n_ct;
            it = nxt;
        }
    } else {
        // ---------------------------------------------------------- epilogue
        const int et = tid - 32 * FOLD_EPI_WARP0;
        const int q = warp & 3, r = q * 32 + lane;  // TMEM lane quarter of this warp
        const float scale = p.scale;
        int mat = fold_find(M, nm, i0), mat_seen = -1;
        for (int j = 0; j < n_my; ++j) {
            const int s = j % FOLD_STAGES, acc = j % FOLD_NACC;
            // the four warps decide together whether to go on, so none is
            // left at the barrier after another gave up
            bool ok = mbar_wait(smem_u32(&tfull_bar[acc]), (uint32_t)(j / FOLD_NACC) & 1u) &&
                      mbar_wait(smem_u32(&full_bar[s]), (uint32_t)(j / FOLD_STAGES) & 1u);
            ok = __all_sync(0xffffffffu, ok);
            if (ok) {
                tc_fence_after();
                uint32_t d[4][16];
#pragma unroll
                for (int h = 0; h < 4; ++h)
                    tmem_ld16(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)acc * FOLD_NC + h * 16, d[h]);
                tmem_ld_wait();
                tc_fence_before();
                mbar_arrive_relaxed(smem_u32(&tempty_bar[acc]));
                uint8_t *wt = base + 2 * FOLD_A_BYTES + s * FOLD_STAGE_BYTES;
#pragma unroll
                for (int c = 0; c < 8; ++c) {
                    uint4 *wp = reinterpret_cast<uint4 *>(wt + swz128(r, c));
                    uint4 v = *wp;
                    const float *f = reinterpret_cast<const float *>(d[c >> 1]) + (c & 1) * 8;
                    v.x = add_bf16x2(v.x, scale * f[0], scale * f[1]);
                    v.y = add_bf16x2(v.y, scale * f[2], scale * f[3]);
                    v.z = add_bf16x2(v.z, scale * f[4], scale * f[5]);
                    v.w = add_bf16x2(v.w, scale * f[6], scale * f[7]);
                    *wp = v;
                }
                fence_async_smem();
            }
            if (!named_sync_and(FOLD_BAR_EPI, FOLD_EPI_THREADS, ok)) {
                ok_all = false;
                break;
            }
            if (et == 0) {
                const int64_t it = i0 + j;
                fold_advance(M, nm, it, mat);
                const FoldMat &F = M[mat];
                if (table && mat != mat_seen) {
                    tensormap_acquire(&F.wmap);
                    mat_seen = mat;
                }
                const int n_ct = (F.Ndim + FOLD_NC - 1) / FOLD_NC;
                const int64_t loc = it - F.item0;
                tma_store_2d(&F.wmap, st32 + (uint32_t)s * FOLD_STAGE_BYTES, (int)(loc % n_ct) * FOLD_NC,
                             (int)(loc / n_ct) * FOLD_TM);
                bulk_commit();
                // the previous item's store has read its stage: hand it back
                bulk_wait_read<1>();
                if (j >= 1) mbar_arrive_release(smem_u32(&empty_bar[(j - 1) % FOLD_STAGES]));
            }
        }
        if (et == 0) bulk_wait_all();
    }
    if (!ok_all) atomicOr(p.err, SALT_DEVERR_TIMEOUT);
    tc_fence_before();
    __syncthreads();
    if (warp == 1) tmem_dealloc(tmem, FOLD_NACC * FOLD_NC);
}

using EncodeFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                              const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                              CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

// bf16 matrix [outer][inner] (row stride inner * 2 bytes), box of
// box_inner x box_outer elements, 128-byte swizzle, out-of-range elements zero
cudaError_t encode_rows_sw128(CUtensorMap *out, const void *ptr, int inner, int outer, int box_inner, int box_outer)
{
    static EncodeFn encode = nullptr;
    static std::mutex mu;
    {
        std::lock_guard<std::mutex> lock(mu);
        if (!encode) {
            void *fn = nullptr;
            cudaDriverEntryPointQueryResult q;
            cudaError_t e = cudaGetDriverEntryPoint("cuTensorMapEncodeTiled", &fn, cudaEnableDefault, &q);
            if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !fn) return e != cudaSuccess ? e : cudaErrorNotSupported;
            encode = reinterpret_cast<EncodeFn>(fn);
        }
    }
    const cuuint64_t dims[2] = {(cuuint64_t)inner, (cuuint64_t)outer};
    const cuuint64_t strides[1] = {(cuuint64_t)inner * 2};
    const cuuint32_t box[2] = {(cuuint32_t)box_inner, (cuuint32_t)box_outer};
    const cuuint32_t es[2] = {1, 1};
    const CUresult r = encode(out, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(ptr), dims, strides, box, es,
                              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

}  // namespace

static cudaError_t fold_configure(int *n_sm)
{
    static unsigned long long configured = 0;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    e = cudaDeviceGetAttribute(n_sm, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    const unsigned long long bit = 1ull << (dev & 63);
    if (!(configured & bit)) {
        e = cudaFuncSetAttribute(salt_fold_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, FOLD_SMEM);
        if (e != cudaSuccess) return e;
        configured |= bit;
    }
    return cudaSuccess;
}

static cudaError_t fold_launch(const FoldParams &p, int n_sm, cudaStream_t stream)
{
    const int grid = (int)(p.items < n_sm ? p.items : n_sm);
    if (grid <= 0) return cudaSuccess;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.gridDim = dim3(grid, 1, 1);
    cfg.blockDim = dim3(FOLD_THREADS, 1, 1);
    cfg.dynamicSmemBytes = FOLD_SMEM;
    cfg.stream = stream;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, salt_fold_kernel, p);
}

size_t fold_record_bytes() { return sizeof(FoldMat); }

cudaError_t fold_record(void *rec, const uint16_t *P, const uint16_t *Q, uint16_t *W, int Mdim, int Ndim, int rc,
                        int64_t item0, int64_t *n_items)
{
    if (rc < 1 || rc > 64 || Mdim < 1 || Ndim < 1 || (Mdim % 8) || (Ndim % 8)) return cudaErrorInvalidValue;
    FoldMat f{};
    cudaError_t e;
    if ((e = encode_rows_sw128(&f.wmap, W, Ndim, Mdim, FOLD_NC, FOLD_TM)) != cudaSuccess) return e;
    if ((e = encode_rows_sw128(&f.qmap, Q, Ndim, rc, FOLD_NC, (rc + 15) & ~15)) != cudaSuccess) return e;
    f.P = P;
    f.item0 = item0;
    f.Mdim = Mdim;
    f.Ndim = Ndim;
    f.rc = rc;
    *n_items = (int64_t)((Mdim + FOLD_TM - 1) / FOLD_TM) * ((Ndim + FOLD_NC - 1) / FOLD_NC);
    std::memcpy(rec, &f, sizeof f);
    return cudaSuccess;
}

cudaError_t launch_fold(const uint16_t *P, const uint16_t *Q, uint16_t *W, int Mdim, int Ndim, int rc, float scale,
                        uint32_t *err, cudaStream_t stream)
{
    int n_sm = 0;
    cudaError_t e = fold_configure(&n_sm);
    if (e != cudaSuccess) return e;
    FoldParams p{};
    int64_t n_items = 0;
    if ((e = fold_record(&p.one, P, Q, W, Mdim, Ndim, rc, 0, &n_items)) != cudaSuccess) return e;
    p.mats = nullptr;
    p.n_mats = 1;
    p.items = n_items;
    p.scale = scale;
    p.err = err;
    return fold_launch(p, n_sm, stream);
}

cudaError_t launch_fold_table(const void *table, int n, int64_t items, float scale, uint32_t *err, cudaStream_t stream)
{
    int n_sm = 0;
    cudaError_t e = fold_configure(&n_sm);
    if (e != cudaSuccess) return e;
    if (!table || n < 1) return cudaErrorInvalidValue;
    FoldParams p{};
    p.mats = static_cast<const FoldMat *>(table);
    p.n_mats = n;
    p.items = items;
    p.scale = scale;
    p.err = err;
    return fold_launch(p, n_sm, stream);
}

}  // namespace salt
