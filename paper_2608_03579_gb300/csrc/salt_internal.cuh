// Internal definitions shared by the runtime (salt_runtime.cu) and the
// kernels (salt_segments.cu, salt_apply.cu).  Not part of the public ABI.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "salt.h"

namespace salt {

// Row blocks handed to the apply kernel hold at most TM tokens of one
// domain (of any gamma bins: gamma scales each token's centroid columns of
// V) and at most `umax` user runs, chosen so that the concatenated
// factor stack [A_c | a_u1 | a_u2 | ...] of a block never exceeds S_MAX
// rows: rc_max + umax * r_max <= S_MAX.
constexpr int TM = 128;
constexpr int S_MAX = 128;
constexpr int APPLY_THREADS = 384;  // 12 warps: in the expand 7 producers, 1 MMA, 4 epilogue
constexpr int SEG_THREADS = 1024;

constexpr int VEXT_COLS = S_MAX;    // row pitch (elements) of a block's V tile in the workspace

// Row-block record (BLK_INTS int32 per block, 32 bytes, read as two int4):
// first grouped token, token count, domain (-1: none), centroid rank of the
// domain, residual rows of the factor stack, centroid scale s_c (float bits),
// and the running sum over blocks 0..b of the expand cost weight
// blk_weight(M, S) (the expand splits its items over CTAs by this weight).
constexpr int BLK_INTS = 8;
constexpr int BLK_START = 0, BLK_LEN = 1, BLK_DOM = 2, BLK_RC = 3, BLK_NRES = 4, BLK_SC = 5, BLK_WEND = 6;

// Cost of one 64-column expand item of a block in 128-byte rows moved: y
// read and written (2 M), the stacked B rows (S), plus a fixed share for the
// per-item handoffs between the expand's warp roles (an item was measured to
// take about 1 us whatever its size, so the fixed share dominates).
__host__ __device__ constexpr int blk_weight(int M, int S) { return 2 * M + S + 384; }

// Device arrays of one segments object.
struct SegDev {
    int32_t *ids;          // [3 * max_tokens]: domain ids, slot ids, then gamma bins
    int32_t *perm;         // [max_tokens] token index in grouped order
    int32_t *sorted_slot;  // [max_tokens] validated slot of the i-th grouped token (-1: none)
    int32_t *dseg_ptr;     // [max_tokens + 1] runs of equal (domain, gamma bin)
    int32_t *dseg_dom;     // [max_tokens]
    int32_t *dseg_gbin;    // [max_tokens]
    int32_t *useg_ptr;     // [max_tokens + 1] runs of equal (domain, gamma bin, slot)
    int32_t *useg_dom;     // [max_tokens]
    int32_t *useg_gbin;    // [max_tokens]
    int32_t *useg_slot;    // [max_tokens]
    int32_t *blk;          // [BLK_INTS * max_tokens], see BLK_* below
    int32_t *counts;       // [4]: n_tokens, domain runs, user runs, row blocks
    // per grouped token: first stacked row of its user among the block's
    // residual rows (-1: no residual), the user's rank and scale s_u
    int32_t *tok_uoff;     // [max_tokens]
    int32_t *tok_urank;    // [max_tokens]
    float *tok_su;         // [max_tokens]
    // per grouped token: its centroid scale s_c(domain) * gamma[bin] (0: no centroid)
    float *tok_sc;         // [max_tokens]
    // per row block: residual rows of the factor stack, res_code(slot, rank, k)
    int32_t *blk_res;      // [max_tokens * S_MAX]
    // The apply order: the tokens stably sorted by (domain, slot), gamma bin
    // after the slot.  Row blocks, blk_res and the per-token tables above
    // (sorted_slot, tok_*) index this order.  Without gamma bins it is the
    // grouped order (perm); with them a user's tokens in several bins are
    // one run here, so they share one set of residual rows in a block.
    int32_t *aperm;        // [max_tokens] token index in apply order
    int32_t *a_dptr;       // [max_tokens + 1] domain runs of the apply order (gamma builds)
    int32_t *a_ddom;       // [max_tokens]
    int32_t *a_uptr;       // [max_tokens + 1] (domain, slot) runs of the apply order (gamma builds)
    int32_t *a_udom;       // [max_tokens]
};

// Code of one residual row of a factor stack: row k of the rank-`rank`
// residual in slot `slot` (slot < 2^17, 1 <= rank <= 128, k < rank).
__host__ __device__ constexpr int32_t res_code(int slot, int rank, int k) { return (slot << 14) | ((rank - 1) << 7) | k; }
__host__ __device__ constexpr int res_slot(int32_t e) { return e >> 14; }
__host__ __device__ constexpr int res_rank(int32_t e) { return ((e >> 7) & 127) + 1; }
__host__ __device__ constexpr int res_k(int32_t e) { return e & 127; }
static_assert(SALT_MAX_RESIDUAL_RANK <= 128, "a residual row code holds ranks up to 128");

// Scratch of the apply path, owned by a segments object (one apply at a
// time uses it; applies on different streams are serialised).
//   vext:   one V tile (bf16 [TM][VEXT_COLS]) per (projection of a group,
//           row block), written by the shrink phase, read by the expand
//           phase of the same launch;
//   part:   fp32 partial V tiles ([TM][PART_COLS]) of the K-split shrink units;
//   arrive: [2][pairs], per (projection, row block): split partials stored;
//   vdone:  [2][pairs], per (projection, row block): V row slices written;
//           a launch uses the half of its epoch's parity and zeroes the
//           other half for the next launch;
//   seq:    [0] launch counter (the epoch), [1] CTAs of the running launch
//           that have finished.
struct ApplyWork {
    // TMA map of vext as a 2-D bf16 tensor [rows][VEXT_COLS], box 64 x TM,
    // 128-byte swizzle (the K-major UMMA layout of a V tile half)
    alignas(64) CUtensorMap vmap;
    uint16_t *vext;        // [max_group * blk_cap * TM * VEXT_COLS]
    int32_t blk_cap;
    int32_t max_group;     // projections per launch the V tiles are sized for (vmap covers exactly these)
    float *part;           // [part_cap * TM * PART_COLS]
    int32_t part_cap;
    uint32_t *arrive;      // [2 * SALT_MAX_GROUP * blk_cap]
    uint32_t *vdone;       // [2 * SALT_MAX_GROUP * blk_cap]
    uint32_t *seq;         // [2]
};
constexpr int PART_COLS = SALT_MAX_TOKEN_RANK;  // centroid | own residual, per token
static_assert(PART_COLS % 4 == 0, "partial rows are read as float4");
constexpr int PART_CAP = 512;  // partial tiles per segments object (20 MiB)

struct SegParams {
    SegDev s;
    int32_t T;
    int32_t max_tokens;
    int32_t n_domains;
    int32_t n_slots;
    int32_t r_max;
    int32_t umax;
    const int32_t *dom_rc;   // [n_domains] pinned rank, 0 = not pinned
    const float *dom_sc;     // [n_domains] centroid scale
    int32_t has_gbin;        // ids hold gamma bins
    int32_t n_gamma;         // gamma bins of this build
    float gamma[SALT_MAX_GAMMA_BINS];
    const uint8_t *pool;     // slot pool base
    int64_t slot_stride;     // bytes per slot
    uint32_t *err;           // device error word
};

// One projection of a (grouped) apply launch.
struct ApplyProj {
    const uint16_t *x;   // [T][d_in]
    uint16_t *y;         // [T][d_out]
    const uint16_t *A;   // centroid arena of this layer: [n_domains][rc_max][d_in]
    const uint16_t *B;   // [n_domains][rc_max][d_out]
    int64_t res_off;     // sum over earlier layers of (d_in + d_out), in elements
    int32_t d_in;
    int32_t d_out;
};


struct ApplyParams {
    ApplyProj proj[SALT_MAX_GROUP];
    int32_t n_proj;
    int32_t n_unit_prefix[SALT_MAX_GROUP + 1];  // expand: 64-column units of projections before p
    const int32_t *perm;
    const int32_t *blk;
    const int32_t *counts;
    const int32_t *tok_uoff;
    const int32_t *tok_urank;
    const float *tok_su;
    const float *tok_sc;
    const int32_t *blk_res;
    int32_t rc_max;
    int32_t min_nk;      // fewest 64-wide d_in chunks over the group's projections (caps the K splits)
    int32_t shrink_only; // write the V tiles of the row blocks and stop (the base-weight kernel expands)
    const uint8_t *pool;
    int64_t slot_stride;
    ApplyWork w;
    uint32_t *err;
};

// One projection of the base-weight GEMM fused with the SALT delta
// (salt_lora_apply_with_base).
struct BaseParams {
    // W_base as a 2-D bf16 TMA map, 128-byte swizzle: for SALT_W_IN_OUT the
    // tensor [d_in][d_out] with box 64 (N) x 64 (K); for SALT_W_OUT_IN the
    // tensor [d_out][d_in] with box 64 (K) x 128 (N)
    alignas(64) CUtensorMap wmap;
    const uint16_t *x;       // [T][d_in]
    uint16_t *y;             // [T][d_out], written
    const int32_t *perm;     // grouped position -> token
    const int32_t *blk;      // row blocks of the segments object
    const int32_t *counts;
    const int32_t *blk_res;
    const uint16_t *vext;    // the blocks' V_ext tiles (projection 0 of the workspace)
    const uint16_t *B;       // centroid arena of this layer: [n_domains][rc_max][d_out]
    const uint8_t *pool;
    int64_t slot_stride;
    int64_t res_off;         // sum over earlier layers of (d_in + d_out), in elements
    int32_t T, d_in, d_out, rc_max, w_layout, blk_cap;
    uint32_t *err;
};
cudaError_t base_prepare(int device);
cudaError_t launch_base(const BaseParams &p, cudaStream_t stream);
// The base weight as the TMA map the fused kernel reads (host).
cudaError_t encode_base_map(CUtensorMap *out, const uint16_t *W, int d_in, int d_out, int layout);

// Encode w.vmap over the max_group * blk_cap V tiles of w.vext (host; once
// per workspace).
cudaError_t apply_encode_vmap(ApplyWork &w);

// Kernel launchers (defined next to the kernels).
cudaError_t launch_segments(const SegParams &p, cudaStream_t stream);
cudaError_t apply_prepare(int device);
// One persistent CTA per SM: the shrink units (row block, projection,
// K-split) first, then the expand items (row block, 64 output columns).
// With pdl the launch is a programmatic dependent of the previous kernel on
// the stream (only when that kernel did not write the segment tables).
cudaError_t launch_apply(const ApplyParams &p, bool pdl, cudaStream_t stream);
size_t apply_smem_bytes();
// W[Mdim][Ndim] += scale * P^T Q for P = [rc][Mdim], Q = [rc][Ndim] (bf16,
// rows contiguous, rc <= 64): the centroid fold; a timed-out wait sets
// SALT_DEVERR_TIMEOUT in *err.
cudaError_t launch_fold(const uint16_t *P, const uint16_t *Q, uint16_t *W, int Mdim, int Ndim, int rc, float scale,
                        uint32_t *err, cudaStream_t stream);
// A fold plan's table: one record of fold_record_bytes() per weight (the
// weight's TMA maps, P, its first item in the launch), written on the host
// and copied to device memory; *n_items gets the weight's item count.
size_t fold_record_bytes();
cudaError_t fold_record(void *rec, const uint16_t *P, const uint16_t *Q, uint16_t *W, int Mdim, int Ndim, int rc,
                        int64_t item0, int64_t *n_items);
// Every weight of a device table of n records (items in all) in one launch.
cudaError_t launch_fold_table(const void *table, int n, int64_t items, float scale, uint32_t *err, cudaStream_t stream);
// salt_align_loss on the current device.
salt_status align_loss_run(int32_t n, const salt_align_pair *pairs, float eps, float *loss, float *cosine,
                           cudaStream_t stream);
// One thread waits, with the apply's bounded cross-CTA wait, on a device word
// nothing sets; raises SALT_DEVERR_TIMEOUT in *err when it gives up.
cudaError_t launch_wait_selftest(uint32_t *err, cudaStream_t stream);

// Row blocks and partial tiles the allocation-free apply
// (salt_lora_apply_static) can use from its static device scratch.
constexpr int STATIC_APPLY_BLOCKS = 64;
// A single-layer apply splits a row block's shrink at most (SMs / blocks)
// ways, so up to 256 SMs the static partial tiles never bind and the static
// apply makes the same split as salt_lora_apply.
constexpr int STATIC_PART_CAP = 256;
// The static scratch on the current device (addresses resolved once per
// device with cudaGetSymbolAddress); blk_cap = STATIC_APPLY_BLOCKS.
cudaError_t apply_static_workspace(ApplyWork *out);

}  // namespace salt
