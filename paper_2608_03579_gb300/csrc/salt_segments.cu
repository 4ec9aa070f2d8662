// Segment builder: groups a heterogeneous batch for the apply kernel.
//
// Section "Multi-Tenant Serving" groups requests by their (centroid, gamma)
// pair, and the residuals are batched heterogeneously (SGMV, Section
// "Multi-Tenant LoRA Serving").  One CTA of 1024 threads:
//   1. validates every (domain, gamma bin, slot) id into the device error
//      word (an invalid id is treated as -1, never dereferenced; a token
//      without a centroid has no bin),
//   2. sorts the keys (domain + 1, bin + 1, slot + 1, token) with a bitonic
//      network in shared memory; keys are unique, so the order is the
//      stable order of (domain, bin, slot) with ties in token order and -1
//      first,
//   3. writes perm / sorted_slot and the maximal (domain, bin) and user runs
//      (two passes over per-thread chunks with a block-wide scan),
//   4. cuts row blocks for the apply kernel: within a domain (over all of
//      its bins), user runs are grouped umax at a time and each group is
//      split evenly into ceil(len / TM) blocks of at most TM tokens.  gamma
//      enters as each token's centroid scale s_c(domain) * gamma[bin], so the
//      bins of one centroid share its blocks and factor reads.  The leading
//      (-1, -1) run (tokens with neither term) gets no block, so those rows
//      are never touched.
// No global scratch is used: the per-group table lives in the shared memory
// the keys occupied.
#include "salt_internal.cuh"

namespace salt {
namespace {

// key = (domain + 1) << 47 | (bin + 1) << 42 | (slot + 1) << 21 | token
constexpr int KEY_TOK_BITS = 21;
constexpr int KEY_SLOT_BITS = 21;
constexpr int KEY_GB_BITS = 5;
constexpr int KEY_CENT_SHIFT = KEY_TOK_BITS + KEY_SLOT_BITS;
constexpr uint64_t KEY_TOK_MASK = (1ull << KEY_TOK_BITS) - 1;
constexpr uint64_t KEY_SLOT_MASK = (1ull << KEY_SLOT_BITS) - 1;
constexpr uint64_t KEY_GB_MASK = (1ull << KEY_GB_BITS) - 1;
static_assert(SALT_MAX_GAMMA_BINS + 1 <= (1 << KEY_GB_BITS), "gamma bins must fit the key");

__device__ __forceinline__ int key_dom(uint64_t k) { return (int)(k >> (KEY_CENT_SHIFT + KEY_GB_BITS)) - 1; }
__device__ __forceinline__ int key_gb(uint64_t k) { return (int)((k >> KEY_CENT_SHIFT) & KEY_GB_MASK) - 1; }
__device__ __forceinline__ uint64_t key_cent(uint64_t k) { return k >> KEY_CENT_SHIFT; }
__device__ __forceinline__ int key_slot(uint64_t k) { return (int)((k >> KEY_TOK_BITS) & KEY_SLOT_MASK) - 1; }
__device__ __forceinline__ int key_tok(uint64_t k) { return (int)(k & KEY_TOK_MASK); }
__device__ __forceinline__ uint64_t key_pair(uint64_t k) { return k >> KEY_TOK_BITS; }

// Exclusive scan of one int per thread over the whole block; *total gets the sum.
__device__ int block_exclusive_scan(int v, int *total, int *warp_sums)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int nwarps = blockDim.x >> 5;
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) warp_sums[warp] = x;
    __syncthreads();
    if (warp == 0) {
        int w = lane < nwarps ? warp_sums[lane] : 0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            int y = __shfl_up_sync(0xffffffffu, w, o);
            if (lane >= o) w += y;
        }
        warp_sums[lane] = w;  // inclusive
    }
    __syncthreads();
    int before = (warp ? warp_sums[warp - 1] : 0) + x - v;
    *total = warp_sums[nwarps - 1];
    __syncthreads();
    return before;
}

// Largest index i in [lo, hi) with a[i] <= v (a non-decreasing, a[lo] <= v).
__device__ __forceinline__ int upper_index(const int32_t *a, int lo, int hi, int v)
{
    while (hi - lo > 1) {
        int mid = (lo + hi) >> 1;
        if (a[mid] <= v) lo = mid; else hi = mid;
    }
    return lo;
}

// Ascending bitonic sort of n (a power of two) keys in shared memory; the
// whole block calls it.
__device__ void bitonic_sort(uint64_t *keys, int n)
{
    for (int k = 2; k <= n; k <<= 1) {
        for (int j = k >> 1; j > 0; j >>= 1) {
            for (int i = threadIdx.x; i < n; i += blockDim.x) {
                int ixj = i ^ j;
                if (ixj > i) {
                    uint64_t a = keys[i], b = keys[ixj];
                    bool up = (i & k) == 0;
                    if ((a > b) == up) {
                        keys[i] = b;
                        keys[ixj] = a;
                    }
                }
            }
            __syncthreads();
        }
    }
}

__global__ void __launch_bounds__(SEG_THREADS, 1) seg_build_kernel(SegParams p)
{
    extern __shared__ __align__(16) uint64_t keys[];
    __shared__ int warp_sums[32];
    const int T = p.T;
    const int tid = threadIdx.x, nth = blockDim.x;

    if (T == 0) {
        if (tid == 0) {
            p.s.dseg_ptr[0] = 0;
            p.s.useg_ptr[0] = 0;
            p.s.counts[0] = p.s.counts[1] = p.s.counts[2] = p.s.counts[3] = 0;
        }
        return;
    }
    int P2 = 1;
    while (P2 < T) P2 <<= 1;

    // 1. validate and build keys
    uint32_t errbits = 0;
    const int32_t *dom_ids = p.s.ids, *slot_ids = p.s.ids + p.max_tokens, *gb_ids = p.s.ids + 2 * p.max_tokens;
    for (int i = tid; i < P2; i += nth) {
        uint64_t key = ~0ull;
        if (i < T) {
            int d = dom_ids[i], s = slot_ids[i], gb = -1;
            if (d < -1 || d >= p.n_domains) {
                errbits |= SALT_DEVERR_DOMAIN_RANGE;
                d = -1;
            } else if (d >= 0 && p.dom_rc[d] <= 0) {
                errbits |= SALT_DEVERR_DOMAIN_NOT_PINNED;
                d = -1;
            }
            if (p.has_gbin && d >= 0) {
                gb = gb_ids[i];
                if (gb < -1 || gb >= p.n_gamma) {
                    errbits |= SALT_DEVERR_GAMMA_RANGE;
                    gb = -1;
                }
            }
            if (s < -1 || s >= p.n_slots) {
                errbits |= SALT_DEVERR_SLOT_RANGE;
                s = -1;
            } else if (s >= 0) {
                const uint8_t *h = p.pool + (int64_t)s * p.slot_stride;
                uint64_t magic = *reinterpret_cast<const uint64_t *>(h);
                int rank = *reinterpret_cast<const int32_t *>(h + 12);
                if (magic != SALT_BLOB_MAGIC) {
                    errbits |= SALT_DEVERR_SLOT_EMPTY;
                    s = -1;
                } else if (rank < 1 || rank > p.r_max) {
                    errbits |= SALT_DEVERR_RANK;
                    s = -1;
                }
            }
            key = ((uint64_t)(d + 1) << (KEY_CENT_SHIFT + KEY_GB_BITS)) | ((uint64_t)(gb + 1) << KEY_CENT_SHIFT) |
                  ((uint64_t)(s + 1) << KEY_TOK_BITS) | (uint64_t)i;
        }
        keys[i] = key;
    }
    if (errbits) atomicOr(p.err, errbits);
    __syncthreads();

    // 2. bitonic sort, ascending
    bitonic_sort(keys, P2);

    // 3. runs: count heads per contiguous chunk, scan, then write
    const int E = (T + nth - 1) / nth;
    const int lo = min(T, tid * E), hi = min(T, lo + E);
    int nd = 0, nu = 0;
    for (int i = lo; i < hi; ++i) {
        uint64_t k = keys[i];
        bool dh = i == 0 || key_cent(k) != key_cent(keys[i - 1]);
        bool uh = i == 0 || key_pair(k) != key_pair(keys[i - 1]);
        nd += dh;
        nu += uh;
    }
    int n_dseg, n_useg;
    int od = block_exclusive_scan(nd, &n_dseg, warp_sums);
    int ou = block_exclusive_scan(nu, &n_useg, warp_sums);
    for (int i = lo; i < hi; ++i) {
        uint64_t k = keys[i];
        int d = key_dom(k), gb = key_gb(k), s = key_slot(k);
        p.s.perm[i] = key_tok(k);
        p.s.aperm[i] = key_tok(k);
        p.s.sorted_slot[i] = s;
        p.s.tok_sc[i] = d >= 0 ? p.dom_sc[d] * (gb >= 0 ? p.gamma[gb] : 1.f) : 0.f;
        bool dh = i == 0 || key_cent(k) != key_cent(keys[i - 1]);
        bool uh = i == 0 || key_pair(k) != key_pair(keys[i - 1]);
        if (dh) {
            p.s.dseg_ptr[od] = i;
            p.s.dseg_dom[od] = d;
            p.s.dseg_gbin[od] = gb;
            ++od;
        }
        if (uh) {
            p.s.useg_ptr[ou] = i;
            p.s.useg_dom[ou] = d;
            p.s.useg_gbin[ou] = gb;
            p.s.useg_slot[ou] = s;
            ++ou;
        }
    }
    if (tid == 0) {
        p.s.dseg_ptr[n_dseg] = T;
        p.s.useg_ptr[n_useg] = T;
    }
    const bool skip0 = key_dom(keys[0]) == -1 && key_slot(keys[0]) == -1;
    // The runs the row blocks are cut from: the grouped order's, unless the
    // batch has gamma bins (below).
    const int32_t *dptr = p.s.dseg_ptr, *ddom = p.s.dseg_dom, *uptr = p.s.useg_ptr, *udom = p.s.useg_dom;
    int n_dr = n_dseg, n_ur = n_useg;
    if (p.has_gbin) {
        // 3'. The apply order: the same keys re-sorted by (domain, slot, bin,
        //     token), so that a user's tokens in several bins form one run
        //     and take one set of residual rows in a block (gamma is applied
        //     per token).  Writes aperm and, in this order, sorted_slot,
        //     tok_sc and the domain and (domain, slot) runs.
        __syncthreads();  // every thread is done with the grouped order
        for (int i = tid; i < P2; i += nth) {
            const uint64_t k = keys[i];
            if (k != ~0ull)
                keys[i] = (key_cent(k) >> KEY_GB_BITS) << (KEY_CENT_SHIFT + KEY_GB_BITS) |
                          (uint64_t)(key_slot(k) + 1) << (KEY_TOK_BITS + KEY_GB_BITS) |
                          (uint64_t)(key_gb(k) + 1) << KEY_TOK_BITS | (uint64_t)key_tok(k);
        }
        __syncthreads();
        bitonic_sort(keys, P2);
        // fields of an apply-order key: domain + 1 | slot + 1 | bin + 1 | token
        auto a_dom = [](uint64_t k) { return (int)(k >> (KEY_CENT_SHIFT + KEY_GB_BITS)) - 1; };
        auto a_slot = [](uint64_t k) { return (int)((k >> (KEY_TOK_BITS + KEY_GB_BITS)) & KEY_SLOT_MASK) - 1; };
        auto a_gb = [](uint64_t k) { return (int)((k >> KEY_TOK_BITS) & KEY_GB_MASK) - 1; };
        auto a_user = [](uint64_t k) { return k >> (KEY_TOK_BITS + KEY_GB_BITS); };
        int ad = 0, au = 0;
        for (int i = lo; i < hi; ++i) {
            const uint64_t k = keys[i];
            ad += i == 0 || a_dom(k) != a_dom(keys[i - 1]);
            au += i == 0 || a_user(k) != a_user(keys[i - 1]);
        }
        int oad = block_exclusive_scan(ad, &n_dr, warp_sums);
        int oau = block_exclusive_scan(au, &n_ur, warp_sums);
        for (int i = lo; i < hi; ++i) {
            const uint64_t k = keys[i];
            const int d = a_dom(k), gb = a_gb(k), sl = a_slot(k);
            p.s.aperm[i] = key_tok(k);
            p.s.sorted_slot[i] = sl;
            p.s.tok_sc[i] = d >= 0 ? p.dom_sc[d] * (gb >= 0 ? p.gamma[gb] : 1.f) : 0.f;
            if (i == 0 || a_dom(k) != a_dom(keys[i - 1])) {
                p.s.a_dptr[oad] = i;
                p.s.a_ddom[oad] = d;
                ++oad;
            }
            if (i == 0 || a_user(k) != a_user(keys[i - 1])) {
                p.s.a_uptr[oau] = i;
                p.s.a_udom[oau] = d;
                ++oau;
            }
        }
        if (tid == 0) {
            p.s.a_dptr[n_dr] = T;
            p.s.a_uptr[n_ur] = T;
        }
        dptr = p.s.a_dptr;
        ddom = p.s.a_ddom;
        uptr = p.s.a_uptr;
        udom = p.s.a_udom;
    }
    __syncthreads();  // keys are dead from here; run arrays are visible block-wide

    // 4a. group heads over user runs; a group stays within one domain (the
    //     (domain, bin) runs of a domain are consecutive)
    int32_t *grp_first = reinterpret_cast<int32_t *>(keys);  // [n_groups]
    const int Eu = (n_ur + nth - 1) / nth;
    const int ulo = min(n_ur, tid * Eu), uhi = min(n_ur, ulo + Eu);
    auto group_head = [&](int j) -> bool {
        if (j == 0) return true;
        if (skip0 && j == 1) return true;
        int start = uptr[j];
        int dr = upper_index(dptr, 0, n_dr, start);
        const int d = ddom[dr];
        while (dr > 0 && ddom[dr - 1] == d) --dr;  // at most SALT_MAX_GAMMA_BINS steps
        int dstart = dptr[dr];
        if (dstart == start) return true;  // first user run of a domain
        int first = upper_index(uptr, 0, n_ur, dstart);
        int idx = j - first - ((skip0 && dr == 0) ? 1 : 0);
        return idx % p.umax == 0;
    };
    int ng = 0;
    for (int j = ulo; j < uhi; ++j) ng += group_head(j);
    int n_groups;
    int og = block_exclusive_scan(ng, &n_groups, warp_sums);
    for (int j = ulo; j < uhi; ++j)
        if (group_head(j)) grp_first[og++] = j;
    __syncthreads();

    // 4b. blocks per group
    const int Eg = (n_groups + nth - 1) / nth;
    const int glo = min(n_groups, tid * Eg), ghi = min(n_groups, glo + Eg);
    auto group_range = [&](int g, int *start, int *len) {
        int a = uptr[grp_first[g]];
        int b = g + 1 < n_groups ? uptr[grp_first[g + 1]] : T;
        *start = a;
        *len = (g == 0 && skip0) ? 0 : b - a;
    };
    int nb = 0;
    for (int g = glo; g < ghi; ++g) {
        int a, len;
        group_range(g, &a, &len);
        nb += (len + TM - 1) / TM;
    }
    int n_blk;
    int ob = block_exclusive_scan(nb, &n_blk, warp_sums);
    for (int g = glo; g < ghi; ++g) {
        int a, len;
        group_range(g, &a, &len);
        int q = (len + TM - 1) / TM;
        int d = udom[grp_first[g]];
        const float sc = d >= 0 ? p.dom_sc[d] : 0.f;
        for (int b = 0; b < q; ++b) {
            int s0 = a + (int)(((int64_t)b * len) / q);
            int s1 = a + (int)(((int64_t)(b + 1) * len) / q);
            int32_t *rec = p.s.blk + (int64_t)BLK_INTS * ob;
            rec[BLK_START] = s0;
            rec[BLK_LEN] = s1 - s0;
            rec[BLK_DOM] = d;
            rec[BLK_RC] = d >= 0 ? p.dom_rc[d] : 0;
            rec[BLK_SC] = __float_as_int(sc);
            ++ob;
        }
    }
    if (tid == 0) {
        p.s.counts[0] = T;
        p.s.counts[1] = n_dseg;
        p.s.counts[2] = n_useg;
        p.s.counts[3] = n_blk;
    }
    __syncthreads();

    // 5. per-block factor stacks: the residual rows of block b are the rows
    //    of its user runs in order (res_code(slot, rank, k)); each token
    //    records where its own user's rows start.  One warp per block.
    const int lane = tid & 31, warp = tid >> 5, nwarp = nth >> 5;
    for (int b = warp; b < n_blk; b += nwarp) {
        const int s0 = p.s.blk[BLK_INTS * b + BLK_START], M = p.s.blk[BLK_INTS * b + BLK_LEN];
        int carry = 0;
        for (int base = 0; base < M; base += 32) {
            const int i = base + lane;
            int slot = -1, rank = 0, contrib = 0;
            float su = 0.f;
            if (i < M) {
                slot = p.s.sorted_slot[s0 + i];
                if (slot >= 0) {
                    const salt_blob_header *h =
                        reinterpret_cast<const salt_blob_header *>(p.pool + (int64_t)slot * p.slot_stride);
                    rank = h->rank;
                    su = h->s_u;
                }
                bool head = i == 0 || slot != p.s.sorted_slot[s0 + i - 1];
                contrib = (head && slot >= 0) ? rank : 0;
            }
            int incl = contrib;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                int y = __shfl_up_sync(0xffffffffu, incl, o);
                if (lane >= o) incl += y;
            }
            const int total = __shfl_sync(0xffffffffu, incl, 31);
            if (i < M) {
                const int off = carry + incl - rank;
                p.s.tok_uoff[s0 + i] = slot >= 0 ? off : -1;
                p.s.tok_urank[s0 + i] = rank;
                p.s.tok_su[s0 + i] = su;
                if (contrib > 0)
                    for (int k = 0; k < rank; ++k)
                        if (off + k < S_MAX)
                            p.s.blk_res[(int64_t)b * S_MAX + off + k] = res_code(slot, rank, k);
            }
            carry += total;
        }
        if (lane == 0) p.s.blk[BLK_INTS * b + BLK_NRES] = carry;
    }
    __syncthreads();

    // 6. running sum of the expand cost weights over blocks
    const int Eb = (n_blk + nth - 1) / nth;
    const int blo = min(n_blk, tid * Eb), bhi = min(n_blk, blo + Eb);
    auto weight = [&](int b) {
        const int32_t *rec = p.s.blk + (int64_t)BLK_INTS * b;
        return blk_weight(rec[BLK_LEN], rec[BLK_RC] + rec[BLK_NRES]);
    };
    int wsum = 0;
    for (int b = blo; b < bhi; ++b) wsum += weight(b);
    int w_total;
    int wo = block_exclusive_scan(wsum, &w_total, warp_sums);
    for (int b = blo; b < bhi; ++b) {
        wo += weight(b);
        p.s.blk[(int64_t)BLK_INTS * b + BLK_WEND] = wo;
    }
}

}  // namespace

cudaError_t launch_segments(const SegParams &p, cudaStream_t stream)
{
    int P2 = 1;
    while (P2 < p.T) P2 <<= 1;
    size_t smem = (size_t)P2 * sizeof(uint64_t);
    if (smem < 16) smem = 16;
    // the attribute is per device; set it once for each device used
    static unsigned long long configured = 0;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const unsigned long long bit = 1ull << (dev & 63);
    if (!(configured & bit)) {
        e = cudaFuncSetAttribute(seg_build_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)(SALT_MAX_TOKENS * sizeof(uint64_t)));
        if (e != cudaSuccess) return e;
        configured |= bit;
    }
    seg_build_kernel<<<1, SEG_THREADS, smem, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace salt
