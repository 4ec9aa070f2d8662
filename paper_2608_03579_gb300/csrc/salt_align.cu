// The alignment regulariser of Phase 1 (Eq. 2) in factored form.
//
//     L_align = 1 - Tr(dW^T Wbar) / (||dW||_F ||Wbar||_F + eps),
//     dW = s A B (rank r),   Wbar = s_c A_c B_c (rank rc)
//
// Neither d_in x d_out matrix is formed.  With the stacked factors
// F_in = [At ; At_c] ([r + rc][d_in]) and F_out = [B ; B_c] ([r + rc][d_out])
// and their Gram matrices G = F F^T,
//     Tr(dW^T Wbar) = s s_c sum_{k < r, l >= r} G_in[k][l] G_out[k][l]
//     ||dW||_F^2    = s^2   sum_{k, l < r}      G_in[k][l] G_out[k][l]
//     ||Wbar||_F^2  = s_c^2 sum_{k, l >= r}     G_in[k][l] G_out[k][l]
// so the work is two Gram contractions per pair, each a pass over its
// factors: HBM-bound, (r + rc)(d_in + d_out) bf16 read once.
//
// align_gram_kernel: one CTA per unit (pair, side, K-split); the unit's
// 64-column chunks of F stream through a cp.async ring into a 128-byte-
// swizzled K-major tile that is both operands of tcgen05.mma
// (D[128 x S] += F_chunk F_chunk^T, fp32 in tensor memory); the unit writes
// its S x S partial, then counts itself done for its pair.  The unit that
// completes a pair (the last of its units to finish) combines it in the same
// launch: its 128 threads sum each side's partials over the splits in split
// order and form the three block sums of G_in o G_out, each thread over a
// fixed set of entries, then a fixed shuffle tree and the four warps in
// order, so the result does not depend on which unit finished last.  The
// sums are fp32: this GPU's fp64 rate is a small fraction of its fp32 rate
// (a dependent fp64 chain cost microseconds at the end of the launch), and
// the rounding error added is far below the Gram entries' own fp32
// accumulation error over d columns.
#include "salt_async.cuh"
#include "salt_internal.cuh"
#include "salt_tcgen05.cuh"

#include <algorithm>
#include <cstring>
#include <vector>

namespace salt {
namespace {

constexpr int ALIGN_THREADS = 128;
constexpr int ALIGN_STAGES = 4;
constexpr int ALIGN_STAGE_BYTES = 128 * 128;     // <= 128 stacked rows x 64 columns
constexpr int ALIGN_SMEM = 1024 + ALIGN_STAGES * ALIGN_STAGE_BYTES;
constexpr int ALIGN_MAX_PAIRS = 256;             // pairs per launch (the parameter block stays < 32 KB)
constexpr int ALIGN_PART = 128 * 128;            // floats per unit partial (row pitch S)
constexpr int KS_CAP = 16;                       // K-splits of one side at most
static_assert(SALT_MAX_ALIGN_RANK <= 128, "a stack is the 128-row UMMA operand");

struct AlignSide {
    const uint16_t *top;  // [r][len]: the task update's factor
    const uint16_t *bot;  // [rc][len]: the centroid's factor
    int32_t len;
    int32_t ks;           // K-splits of this side
};
struct AlignPairP {
    AlignSide side[2];    // 0: d_in (A factors), 1: d_out (B factors)
    int32_t r, rc;
    float s, s_c;
};
struct AlignParams {
    AlignPairP pair[ALIGN_MAX_PAIRS];
    int32_t n_pairs;
    int32_t unit_start[2 * ALIGN_MAX_PAIRS + 1];  // first unit of (pair, side), then the total
    float *part;                                  // [units][ALIGN_PART]
    uint32_t *done;                               // [pairs]: units finished (zeroed)
    float *loss;
    float *cosine;                                // may be null
    float eps;
    uint32_t *err;                                // set when a bounded wait gave up
};
static_assert(sizeof(AlignParams) <= 32000, "kernel parameter block too large");

__global__ void __launch_bounds__(ALIGN_THREADS) align_gram_kernel(const __grid_constant__ AlignParams p)
{
    extern __shared__ __align__(128) uint8_t smem_raw[];
    uint8_t *ring = smem_raw + ((1024 - (smem_u32(smem_raw) & 1023)) & 1023);
    const uint32_t ring32 = smem_u32(ring);
    __shared__ uint64_t bar[ALIGN_STAGES];
    __shared__ uint32_t tmem_slot;

    const int unit = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    // the (pair, side) of this unit: the last ps with unit_start[ps] <= unit
    int ps = 0, hi = 2 * p.n_pairs;
    while (hi - ps > 1) {
        const int mid = (ps + hi) >> 1;
        if (p.unit_start[mid] <= unit) ps = mid;
        else hi = mid;
    }
    const AlignPairP &pr = p.pair[ps >> 1];
    const AlignSide &sd = pr.side[ps & 1];
    const int split = unit - p.unit_start[ps];
    const int r = pr.r, S = pr.r + pr.rc, n_pad = (S + 15) & ~15, len = sd.len;
    const int nk = (len + 63) / 64;
    const int c0 = (int)((int64_t)nk * split / sd.ks), n_my = (int)((int64_t)nk * (split + 1) / sd.ks) - c0;

    if (warp == 0) {
        tmem_alloc(smem_u32(&tmem_slot), 128);
        tmem_relinquish();
    }
    if (tid == 0) {
        for (int i = 0; i < ALIGN_STAGES; ++i) mbar_init(smem_u32(&bar[i]), 1);
        mbar_fence_init();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;

    // chunk i of this unit into stage st: rows < S, 16-byte pieces (columns
    // past len zero-filled); rows >= S are never loaded and only reach
    // accumulator rows and columns >= S, which are not read
    auto load = [&](int i, int st) {
        const int k0 = (c0 + i) * 64;
        const uint32_t dst = ring32 + st * ALIGN_STAGE_BYTES;
        for (int idx = tid; idx < S * 8; idx += ALIGN_THREADS) {
            const int row = idx >> 3, c = idx & 7, col = k0 + c * 8;
            const uint16_t *src = row < r ? sd.top + (int64_t)row * len : sd.bot + (int64_t)(row - r) * len;
            const bool ok = col < len;
            cp_async16(dst + swz128(row, c), ok ? src + col : src, ok);
        }
    };
    const uint32_t idesc = idesc_bf16_f32(128, n_pad);
    bool ok_all = true;
    uint32_t phase = 0, pending = 0;
    for (int st = 0; st < ALIGN_STAGES - 1; ++st) {
        if (st < n_my) load(st, st);
        cp_async_commit();
    }
    for (int it = 0; it < n_my; ++it) {
        const int st = it % ALIGN_STAGES;
        cp_async_wait_dyn(ALIGN_STAGES - 2);
        fence_async_smem();
        __syncthreads();
        if (tid == 0) {
            tc_fence_after();
            const uint32_t a = ring32 + st * ALIGN_STAGE_BYTES;
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
                umma_bf16(tmem, sdesc_kmajor_sw128(a + kk * 32), sdesc_kmajor_sw128(a + kk * 32), idesc,
                          (it > 0 || kk > 0) ? 1u : 0u);
            umma_commit(smem_u32(&bar[st]));
        }
        pending |= 1u << st;
        const int nxt = it + ALIGN_STAGES - 1;
        if (nxt < n_my) {
            // the stage of chunk nxt last held chunk it - 1: its MMAs must be done
            if (it >= 1) {
                const int pst = (it - 1) % ALIGN_STAGES;
                if (!mbar_wait(smem_u32(&bar[pst]), (phase >> pst) & 1)) ok_all = false;
                phase ^= 1u << pst;
                pending &= ~(1u << pst);
            }
            load(nxt, nxt % ALIGN_STAGES);
        }
        cp_async_commit();
    }
    cp_async_wait<0>();
    for (int st = 0; st < ALIGN_STAGES; ++st)
        if ((pending >> st) & 1) {
            if (!mbar_wait(smem_u32(&bar[st]), (phase >> st) & 1)) ok_all = false;
            phase ^= 1u << st;
        }
    tc_fence_after();

    // D rows (tensor-memory lanes) = stack rows, columns = stack rows.  D
    // is symmetric: thread `row` writes D's row as column `row`, so a
    // warp's stores of one column are contiguous.
    float *out = p.part + (int64_t)unit * ALIGN_PART;
    const int row = warp * 32 + lane;
    for (int g = 0; g < n_pad / 16; ++g) {
        uint32_t v[16];
        tmem_ld16(tmem + ((uint32_t)(warp * 32) << 16) + g * 16, v);
        tmem_ld_wait();
        if (row < S) {
#pragma unroll
            for (int e = 0; e < 16; ++e)
                if (g * 16 + e < S) __stcg(out + (g * 16 + e) * S + row, __uint_as_float(v[e]));
        }
    }
    if (!ok_all) atomicOr(p.err, SALT_DEVERR_TIMEOUT);
    __threadfence();
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tmem, 128);

    // ------------------------------------------------ the pair's combine
    __shared__ int last;
    __shared__ float red[3][ALIGN_THREADS / 32];
    const int pi = ps >> 1;
    const AlignPairP &pq = p.pair[pi];
    const int u_in = p.unit_start[2 * pi], u_out = p.unit_start[2 * pi + 1];
    const int ks_in = pq.side[0].ks, ks_out = pq.side[1].ks;
    if (tid == 0) {
        last = atomicAdd(p.done + pi, 1u) == (uint32_t)(ks_in + ks_out) - 1u;
        __threadfence();
    }
    __syncthreads();
    if (!last) return;
    // every partial of the pair is written.  Thread t takes the float4 of
    // entries t, t + 128, ... (the partials' pitch of 16384 floats keeps the
    // last float4 in bounds; entries past S * S are skipped); up to four
    // splits of a side are loaded together before they are added.
    const int SS = S * S, n4 = (SS + 3) / 4;
    const float4 *pin = reinterpret_cast<const float4 *>(p.part + (int64_t)u_in * ALIGN_PART);
    const float4 *pout = reinterpret_cast<const float4 *>(p.part + (int64_t)u_out * ALIGN_PART);
    constexpr int U4 = ALIGN_PART / 4;
    float num = 0.f, na = 0.f, nc = 0.f;
    for (int b4 = tid; b4 < n4; b4 += ALIGN_THREADS) {
        float gi[4] = {0.f, 0.f, 0.f, 0.f}, go[4] = {0.f, 0.f, 0.f, 0.f};
        auto add_side = [&](const float4 *base, int ks, float (&acc)[4]) {
            for (int k0 = 0; k0 < ks; k0 += 4) {
                float4 x[4];
#pragma unroll
                for (int k = 0; k < 4; ++k)
                    x[k] = k0 + k < ks ? __ldcg(base + (int64_t)(k0 + k) * U4 + b4) : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    acc[0] += x[k].x;
                    acc[1] += x[k].y;
                    acc[2] += x[k].z;
                    acc[3] += x[k].w;
                }
            }
        };
        add_side(pin, ks_in, gi);
        add_side(pout, ks_out, go);
        const int idx0 = b4 * 4;
        int i = idx0 / S, j = idx0 - i * S;
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            // the lower cross block mirrors the upper one
            if (idx0 + e < SS && !(i >= r && j < r)) {
                const float prod = gi[e] * go[e];
                if (i < r && j < r) na += prod;
                else if (i >= r) nc += prod;
                else num += prod;
            }
            if (++j == S) {
                j = 0;
                ++i;
            }
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        num += __shfl_xor_sync(0xffffffffu, num, o);
        na += __shfl_xor_sync(0xffffffffu, na, o);
        nc += __shfl_xor_sync(0xffffffffu, nc, o);
    }
    if (lane == 0) {
        red[0][warp] = num;
        red[1][warp] = na;
        red[2][warp] = nc;
    }
    __syncthreads();
    if (tid == 0) {
        float snum = 0.f, sna = 0.f, snc = 0.f;
        for (int w = 0; w < ALIGN_THREADS / 32; ++w) {
            snum += red[0][w];
            sna += red[1][w];
            snc += red[2][w];
        }
        const float tr = pq.s * pq.s_c * snum;
        const float n_dw = fabsf(pq.s) * sqrtf(fmaxf(sna, 0.f));
        const float n_wb = fabsf(pq.s_c) * sqrtf(fmaxf(snc, 0.f));
        float cosv = tr / (n_dw * n_wb + p.eps);
        if (*reinterpret_cast<volatile uint32_t *>(p.err) != 0u) cosv = __int_as_float(0x7fc00000);
        p.loss[pi] = 1.f - cosv;
        if (p.cosine) p.cosine[pi] = cosv;
    }
}

bool aligned16(const void *q) { return (reinterpret_cast<uintptr_t>(q) & 15u) == 0; }

}  // namespace

salt_status align_loss_run(int32_t n, const salt_align_pair *pairs, float eps, float *loss, float *cosine,
                           cudaStream_t stream)
{
    if (n < 0 || (n > 0 && (!pairs || !loss))) return SALT_ERR_INVALID_ARG;
    for (int i = 0; i < n; ++i) {
        const salt_align_pair &q = pairs[i];
        if (!q.At || !q.B || !q.At_c || !q.B_c) return SALT_ERR_INVALID_ARG;
        if (q.r < 1 || q.rc < 1 || q.r + q.rc > SALT_MAX_ALIGN_RANK) return SALT_ERR_RANK;
        if (q.d_in <= 0 || q.d_out <= 0 || (q.d_in % 8) || (q.d_out % 8)) return SALT_ERR_INVALID_ARG;
        if (!aligned16(q.At) || !aligned16(q.B) || !aligned16(q.At_c) || !aligned16(q.B_c)) return SALT_ERR_ALIGN;
    }
    if (n == 0) return SALT_OK;
    int dev = 0, n_sm = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
        cudaGetLastError();
        return SALT_ERR_CUDA;
    }
    static unsigned long long configured = 0;
    const unsigned long long bit = 1ull << (dev & 63);
    if (!(configured & bit)) {
        if (cudaFuncSetAttribute(align_gram_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, ALIGN_SMEM) !=
            cudaSuccess) {
            cudaGetLastError();
            return SALT_ERR_CUDA;
        }
        configured |= bit;
    }
    for (int first = 0; first < n; first += ALIGN_MAX_PAIRS) {
        const int m = std::min(ALIGN_MAX_PAIRS, n - first);
        AlignParams p;
        std::memset(&p, 0, sizeof p);
        p.n_pairs = m;
        p.eps = eps;
        p.loss = loss + first;
        p.cosine = cosine ? cosine + first : nullptr;
        // K-splits: at most 64 chunks (4096 columns) a unit, then more
        // splits (up to KS_CAP) while the launch has fewer than three units per SM
        int nk[2 * ALIGN_MAX_PAIRS], ks[2 * ALIGN_MAX_PAIRS];
        int64_t units = 0;
        for (int i = 0; i < m; ++i) {
            const salt_align_pair &q = pairs[first + i];
            nk[2 * i] = (q.d_in + 63) / 64;
            nk[2 * i + 1] = (q.d_out + 63) / 64;
            for (int sd = 0; sd < 2; ++sd) {
                ks[2 * i + sd] = std::min(KS_CAP, (nk[2 * i + sd] + 63) / 64);
                units += ks[2 * i + sd];
            }
        }
        const int64_t target = 3LL * n_sm;
        if (units < target) {
            const int64_t f = (target + units - 1) / units;
            units = 0;
            for (int k = 0; k < 2 * m; ++k) {
                ks[k] = (int)std::min<int64_t>(nk[k], std::min<int64_t>(KS_CAP, (int64_t)ks[k] * f));
                units += ks[k];
            }
        }
        int u = 0;
        for (int i = 0; i < m; ++i) {
            const salt_align_pair &q = pairs[first + i];
            AlignPairP &d = p.pair[i];
            d.r = q.r;
            d.rc = q.rc;
            d.s = q.s;
            d.s_c = q.s_c;
            d.side[0] = AlignSide{static_cast<const uint16_t *>(q.At), static_cast<const uint16_t *>(q.At_c), q.d_in,
                                  ks[2 * i]};
            d.side[1] = AlignSide{static_cast<const uint16_t *>(q.B), static_cast<const uint16_t *>(q.B_c), q.d_out,
                                  ks[2 * i + 1]};
            p.unit_start[2 * i] = u;
            u += ks[2 * i];
            p.unit_start[2 * i + 1] = u;
            u += ks[2 * i + 1];
        }
        p.unit_start[2 * m] = u;
        // scratch: the error word and the pairs' counters (zeroed), then
        // the partials
        const size_t head = 256 + (size_t)ALIGN_MAX_PAIRS * 4;
        void *ws = nullptr;
        const size_t bytes = head + (size_t)u * ALIGN_PART * sizeof(float);
        if (cudaMallocAsync(&ws, bytes, stream) != cudaSuccess) {
            cudaGetLastError();
            return SALT_ERR_OOM;
        }
        uint8_t *w8 = static_cast<uint8_t *>(ws);
        p.err = reinterpret_cast<uint32_t *>(w8);
        p.done = reinterpret_cast<uint32_t *>(w8 + 256);
        p.part = reinterpret_cast<float *>(w8 + head);
        cudaError_t e = cudaMemsetAsync(ws, 0, head, stream);
        if (e == cudaSuccess) {
            align_gram_kernel<<<u, ALIGN_THREADS, ALIGN_SMEM, stream>>>(p);
            e = cudaGetLastError();
        }
        cudaError_t f = cudaFreeAsync(ws, stream);
        if (e != cudaSuccess || f != cudaSuccess) {
            cudaGetLastError();
            return SALT_ERR_CUDA;
        }
    }
    return SALT_OK;
}

}  // namespace salt
