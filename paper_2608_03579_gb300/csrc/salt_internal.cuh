// Internal definitions shared by the runtime (salt_runtime.cu) and the
// kernels (salt_segments.cu, salt_apply.cu).  Not part of the public ABI.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "salt.h"

namespace salt {

// Row blocks handed to the apply kernel hold at most TM tokens of one
// domain and at most `umax` user runs, chosen so that the concatenated
// factor stack [A_c | a_u1 | a_u2 | ...] of a block never exceeds S_MAX
// rows: rc_max + umax * r_max <= S_MAX.
constexpr int TM = 128;
constexpr int S_MAX = 128;
constexpr int CLUSTER = 8;          // CTAs per row block (split of d_in and d_out)
constexpr int APPLY_THREADS = 256;
constexpr int SEG_THREADS = 1024;

// Device arrays of one segments object.
struct SegDev {
    int32_t *ids;          // [2 * max_tokens]: domain ids, then slot ids
    int32_t *perm;         // [max_tokens] token index in grouped order
    int32_t *sorted_slot;  // [max_tokens] validated slot of the i-th grouped token (-1: none)
    int32_t *dseg_ptr;     // [max_tokens + 1]
    int32_t *dseg_dom;     // [max_tokens]
    int32_t *useg_ptr;     // [max_tokens + 1]
    int32_t *useg_dom;     // [max_tokens]
    int32_t *useg_slot;    // [max_tokens]
    int32_t *blk;          // [3 * max_tokens] (start, length, domain)
    int32_t *counts;       // [4]: n_tokens, domain runs, user runs, row blocks
};

struct SegParams {
    SegDev s;
    int32_t T;
    int32_t max_tokens;
    int32_t n_domains;
    int32_t n_slots;
    int32_t r_max;
    int32_t umax;
    const int32_t *dom_rc;   // [n_domains] pinned rank, 0 = not pinned
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
    const int32_t *perm;
    const int32_t *sorted_slot;
    const int32_t *blk;
    const int32_t *counts;
    const int32_t *dom_rc;
    const float *dom_sc;
    int32_t rc_max;
    const uint8_t *pool;
    int64_t slot_stride;
    int32_t r_max;
    uint32_t *err;
};

// Kernel launchers (defined next to the kernels).
cudaError_t launch_segments(const SegParams &p, cudaStream_t stream);
cudaError_t apply_prepare(int device, int *max_active_clusters);
cudaError_t launch_apply(const ApplyParams &p, int n_clusters, cudaStream_t stream);
size_t apply_smem_bytes();

}  // namespace salt
