/*
 * salt.h - C ABI of the SALT serving hot path on GB300 (sm_103a).
 *
 * SALT ("Pin Once, Swap Light", Section "Multi-Tenant Serving") serves a
 * request with W_final = W_base + gamma * Wbar + delta_i: a high-rank domain
 * centroid Wbar = A_c B_c stays pinned in device memory, an ultra-low-rank
 * (r <= 2) user residual delta_i = a_u b_u is swapped in on demand
 * (Section "The Centroid-Residual Decomposition").  This library evaluates
 * the LoRA part of that composition for every token of a heterogeneous
 * batch, in place:
 *
 *     y[t, :] += s_c(d) * (x[t, :] A_c(d)) B_c(d) + s_u(u) * (x[t, :] a_u(u)) b_u(u)
 *
 * where d is the token's domain (centroid) id and u its residual slot id,
 * y already holds x W_base, and an id of -1 drops its term.  s_c carries
 * gamma (and any LoRA alpha/r the caller folds in); s_u the residual's.
 *
 * Conventions
 *  - Math is in row vectors.  A factor is stored transposed: At[k][i] with
 *    i over d_in (PEFT's lora_A.weight); B[k][j] with j over d_out
 *    (PEFT's lora_B.weight transposed).  All factors and activations are
 *    bf16, row-major, passed as raw bit patterns (uint16).
 *  - A "layer" is one adapted weight matrix (one projection of one
 *    transformer layer); the context's layer table lists their shapes.
 *  - Streams are cudaStream_t values passed as void*; NULL is the legacy
 *    default stream.  Device pointers are CUDA device addresses of the
 *    context's device; host pointers are ordinary host addresses.
 *  - Every call returns a salt_status; no C++ exception crosses this ABI.
 *    On failure salt_last_error(ctx) holds a one-line message.  A context
 *    is not thread-safe: serialise calls on one context.
 *  - Calls marked "asynchronous" enqueue work and return without waiting
 *    for the device; their device-side faults in the ids are reported by
 *    salt_get_device_error.
 */
#ifndef SALT_H
#define SALT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define SALT_ABI_VERSION 1

/* Library limits. */
#define SALT_MAX_TOKENS 16384        /* tokens per segments build */
#define SALT_MAX_CENTROID_RANK 64    /* rc_max */
#define SALT_MAX_RESIDUAL_RANK 80    /* r_max: up to a rank-64 centroid concatenated with a rank-16 residual */
#define SALT_MAX_TOKEN_RANK 80       /* rc_max + r_max (a token's centroid plus residual rank) */
#define SALT_MAX_GROUP 8             /* projections per grouped apply */
#define SALT_MAX_GAMMA_BINS 16       /* gamma bins of one segments build */
#define SALT_MAX_ALIGN_RANK 128      /* r + rc of one alignment pair */
#define SALT_BLOB_HEADER_BYTES 256
#define SALT_BLOB_MAGIC 0x3153455254414C53ULL /* "SALTRES1" little-endian */

typedef void *salt_stream_t;
typedef struct salt_ctx salt_ctx;
typedef struct salt_segments salt_segments;

typedef enum salt_status {
    SALT_OK = 0,
    SALT_ERR_INVALID_ARG = 1,        /* NULL pointer, bad size, bad config */
    SALT_ERR_OOM = 2,                /* device or pinned-host allocation failed */
    SALT_ERR_NOT_PINNED_HOST = 3,    /* residual blob is not page-locked host memory */
    SALT_ERR_DOMAIN_NOT_PINNED = 4,  /* a token names a domain with no pinned centroid */
    SALT_ERR_SLOT_RANGE = 5,         /* slot id outside [-1, n_slots) */
    SALT_ERR_RANK = 6,               /* rank above the context's limit, or zero */
    SALT_ERR_LAYER_RANGE = 7,        /* layer index outside the layer table */
    SALT_ERR_ALIGN = 8,              /* x / y not 16-byte aligned */
    SALT_ERR_BAD_BLOB = 9,           /* wrong magic, version, layer count or layout hash */
    SALT_ERR_DEVICE_IDS = 10,        /* device-side id check failed (see salt_get_device_error) */
    SALT_ERR_TIMEOUT = 11,           /* reserved: a bounded device wait gave up */
    SALT_ERR_CUDA = 12,              /* a CUDA runtime call failed */
    SALT_ERR_SLOT_EMPTY = 13,        /* a token names a slot that was never loaded */
    SALT_ERR_TOO_MANY_TOKENS = 14,   /* n_tokens above the context's max_tokens */
    SALT_ERR_DOMAIN_RANGE = 15,      /* domain id outside [-1, n_domains) */
    SALT_ERR_STALE_SEGMENTS = 16,    /* a slot the segments read was reloaded after the build */
    SALT_ERR_NOT_BUILT = 17,         /* segments object was never built */
    SALT_ERR_GAMMA_RANGE = 18        /* gamma bin outside [-1, n_gamma) */
} salt_status;

/* Bits of the device error word (salt_get_device_error). */
#define SALT_DEVERR_DOMAIN_RANGE 0x1u
#define SALT_DEVERR_DOMAIN_NOT_PINNED 0x2u
#define SALT_DEVERR_SLOT_RANGE 0x4u
#define SALT_DEVERR_SLOT_EMPTY 0x8u
#define SALT_DEVERR_RANK 0x10u
#define SALT_DEVERR_TIMEOUT 0x20u        /* a bounded in-kernel wait gave up (results of that call invalid) */
#define SALT_DEVERR_GAMMA_RANGE 0x40u

/*
 * Context configuration.  d_in / d_out are host arrays of n_layers entries,
 * each a positive multiple of 8 (16-byte rows).  rc_max <=
 * SALT_MAX_CENTROID_RANK, 1 <= r_max <= SALT_MAX_RESIDUAL_RANK,
 * rc_max + r_max <= SALT_MAX_TOKEN_RANK, 1 <= max_tokens <= SALT_MAX_TOKENS,
 * n_domains < 2^17 - 1, n_slots < 2^17.
 */
typedef struct salt_config {
    int32_t n_layers;
    const int32_t *d_in;
    const int32_t *d_out;
    int32_t n_domains;   /* centroid table size */
    int32_t rc_max;      /* largest centroid rank to be pinned */
    int32_t n_slots;     /* residual slot pool size */
    int32_t r_max;       /* largest residual rank a slot holds */
    int32_t max_tokens;  /* largest batch a segments object accepts */
    int32_t device;      /* CUDA device ordinal */
} salt_config;

/*
 * Residual blob: the unit swapped host -> device (Section "Multi-Tenant
 * Serving": only the residual is swapped; its size is the paper's "Swap"
 * column).  A 256-byte header followed by, for each layer l in table order,
 * At_u[rank][d_in_l] then B_u[rank][d_out_l] (bf16).  payload_bytes =
 * rank * sum_l (d_in_l + d_out_l) * 2.  layout_hash is FNV-1a 64 over the
 * (d_in, d_out) pairs as little-endian int32, so a blob built for another
 * layer table is rejected.
 */
typedef struct salt_blob_header {
    uint64_t magic;          /* SALT_BLOB_MAGIC */
    uint32_t version;        /* 1 */
    int32_t rank;            /* 1 .. SALT_MAX_RESIDUAL_RANK (and <= r_max of the loading context) */
    int32_t n_layers;
    float s_u;               /* residual scale */
    uint64_t payload_bytes;
    uint64_t layout_hash;
    uint8_t reserved[SALT_BLOB_HEADER_BYTES - 40];
} salt_blob_header;

int32_t salt_abi_version(void);
const char *salt_status_string(salt_status s);

/*
 * Create a context on config->device: allocates the centroid arena
 * (n_domains * rc_max * sum(d_in + d_out) bf16), the zeroed residual slot
 * pool (n_slots slots of header + r_max * sum(d_in + d_out) bf16) and the
 * device error word.  The context owns all of it until salt_ctx_destroy.
 * On failure *out is NULL.  Synchronous.
 */
salt_status salt_ctx_create(const salt_config *config, salt_ctx **out);

/* Synchronise the device and free everything the context owns.  Segments
 * objects of the context must be destroyed first.  NULL is a no-op. */
void salt_ctx_destroy(salt_ctx *ctx);

/* Last error message of the context ("" when none).  Owned by the context. */
const char *salt_last_error(const salt_ctx *ctx);

/* Sizes and launch shape the context chose (diagnostics; no device work). */
typedef struct salt_ctx_info {
    int64_t arena_bytes;        /* centroid arena, device */
    int64_t pool_bytes;         /* residual slot pool, device */
    int64_t slot_stride;        /* bytes per slot */
    int32_t apply_ctas;         /* CTAs of one apply launch (one per SM) */
    int32_t k_splits_max;       /* most d_in splits of one row block's shrink */
    int32_t apply_smem_bytes;   /* dynamic shared memory per apply CTA */
    int32_t block_tokens;       /* max tokens per row block */
    int32_t block_users;        /* max user runs per row block */
    int32_t reserved;
} salt_ctx_info;
salt_status salt_ctx_get_info(const salt_ctx *ctx, salt_ctx_info *info);

/*
 * Pin domain `domain`'s centroid (Section "Multi-Tenant Serving": the
 * centroid is loaded once and stays resident).  At_c holds, for each layer
 * in table order, [rc][d_in_l]; B_c holds, for each layer, [rc][d_out_l]
 * (bf16).  Either may be host or device memory.  s_c is the centroid scale
 * (gamma, with any alpha/r folded in).  1 <= rc <= rc_max.  Re-pinning a
 * domain replaces it.  Synchronous: waits for the device to go idle first,
 * so no apply in flight reads a half-written centroid.  Setup call, not for
 * the per-step path.
 */
salt_status salt_centroid_pin(salt_ctx *ctx, int32_t domain, int32_t rc,
                              const void *At_c, const void *B_c, float s_c);

/* Blob size (header + payload) for a rank-`rank` residual over the layer
 * table of `config`; -1 on an invalid argument.  Host only. */
int64_t salt_residual_blob_bytes(const salt_config *config, int32_t rank);

/*
 * Write a blob: header plus At_u (for each layer [rank][d_in_l]) and B_u
 * (for each layer [rank][d_out_l]), both host arrays of bf16.  blob must
 * hold salt_residual_blob_bytes(config, rank) bytes (pinned host memory if
 * it is to be swapped with salt_residual_load).  Host only, synchronous.
 */
salt_status salt_residual_blob_pack(const salt_config *config, int32_t rank, float s_u,
                                    const void *At_u, const void *B_u,
                                    void *blob, int64_t blob_bytes);

/*
 * The long-tail form of a request (Section "Multi-Tenant Serving": for rare
 * tasks the scaled centroid and the residual are stacked ahead of time into
 * one ordinary adapter - rank 17 in the paper's example - served like any
 * other adapter of a mixed batch): write a blob of rank rc + rank whose
 * factors are, per layer,
 *     At = [At_c ; At_u]           ([rc + rank][d_in_l])
 *     B  = [(s_c / s) B_c ; B_u]   ([rc + rank][d_out_l])
 * with blob scale s = s_u (s = 1 and B_u scaled by 0 when s_u == 0), so
 * that s (x At^T) B = s_c (x A_c) B_c + s_u (x a_u) b_u.  At_c / B_c are
 * host arrays in salt_centroid_pin's layout (rank rc), At_u / B_u in
 * salt_residual_blob_pack's (rank `rank`); s_c is the centroid's scale
 * with gamma applied.  The A rows are copied bit for bit; a scaled B row is
 * rounded once to bf16 (round to nearest even) and copied bit for bit when
 * s_c == s.  rc + rank <= SALT_MAX_RESIDUAL_RANK; the blob loads into a
 * context whose r_max is at least that and is applied with domain id -1.
 * Host only, synchronous.
 */
salt_status salt_residual_blob_concat(const salt_config *config, int32_t rc, const void *At_c,
                                      const void *B_c, float s_c, int32_t rank, const void *At_u,
                                      const void *B_u, float s_u, void *blob, int64_t blob_bytes);

/*
 * Fuse a scaled centroid into a base weight (Section "Multi-Tenant
 * Serving": a much-used centroid, already scaled, may be merged into the
 * base weights when a node starts, after which its requests swap and apply
 * only residuals: build their segments with domain id -1).  For layer `layer` and pinned
 * domain `domain`:
 *     W += gamma * s_c(domain) * A_c B_c
 * in place, each element accumulated in fp32 and rounded once to bf16
 * (round to nearest even).  W is device bf16, 16-byte aligned, in one of
 *     SALT_W_IN_OUT: W[d_in][d_out]  (y = x W, this library's convention)
 *     SALT_W_OUT_IN: W[d_out][d_in]  (y = x W^T, a linear layer's weight)
 * gamma = -g undoes a fold by g up to the two roundings.  One tcgen05
 * kernel; asynchronous on `stream`, after earlier work on it.  The
 * centroid must not be re-pinned while the fold runs.
 */
#define SALT_W_IN_OUT 0
#define SALT_W_OUT_IN 1
salt_status salt_centroid_fold(salt_ctx *ctx, int32_t domain, int32_t layer, float gamma, void *W,
                               int32_t layout, salt_stream_t stream);

/*
 * A fold plan: salt_centroid_fold over many weights in ONE launch (the
 * same Section: when a node starts, a centroid is merged into every weight
 * it adapts).  layers[i] and W[i] (i < n) name weight i as in
 * salt_centroid_fold, all in `layout`; a layer may appear more than once
 * with different weights, but no two weights may overlap in memory
 * (SALT_ERR_INVALID_ARG).  The plan keeps the weights' addresses and the
 * domain's pinned factors in device memory: the weights must stay allocated,
 * and the centroid pinned, while the plan lives.  Host-side checks and one
 * synchronous table upload; destroy the plan before its context.
 */
typedef struct salt_fold_plan salt_fold_plan;
salt_status salt_fold_plan_create(salt_ctx *ctx, int32_t domain, int32_t n, const int32_t *layers,
                                  void *const *W, int32_t layout, salt_fold_plan **out);
/*
 * W_i += gamma * s_c(domain) * A_c(layer_i) B_c(layer_i) for every weight
 * of the plan, each element rounded once as in salt_centroid_fold (the
 * results are bit-identical to n salt_centroid_fold calls).  One kernel,
 * asynchronous on `stream`.  SALT_ERR_RANK when the domain was re-pinned
 * with another rank after the plan was made.
 */
salt_status salt_fold_plan_run(salt_fold_plan *plan, float gamma, salt_stream_t stream);
void salt_fold_plan_destroy(salt_fold_plan *plan);

/*
 * Page-locked host memory for residual blobs, backed by transparent huge
 * pages where the kernel offers them (anonymous mapping rounded up to the
 * huge-page size, madvise(MADV_HUGEPAGE), every page touched, a request to
 * collapse what still has base pages (MADV_COLLAPSE, where the kernel has
 * it), then cudaHostRegister).  The host-to-device copies of a swap translate host
 * addresses page by page; with the base pages of an ordinary pinned
 * allocation (64 KiB on Arm servers) sustained swapping was measured to
 * stall for 30-100 ms every few hundred copies, with huge pages not at all.
 * (The paper has no counterpart; this is a deployment convenience for the
 * host side of the residual cache.)  Returns NULL on failure; the memory
 * is zeroed.  Release with salt_host_free (not free or cudaFreeHost).
 */
void *salt_host_alloc(int64_t bytes);
void salt_host_free(void *ptr);

/*
 * Swap a residual into slot `slot` (Section "Multi-Tenant Serving": only
 * the ultra-low-rank residual moves host -> device).  host_blob must be
 * page-locked host memory holding a valid blob (checked on the host:
 * magic, version, rank <= r_max, layer count, layout hash).  Asynchronous
 * on side_stream: the copy first waits for every apply already enqueued
 * that reads a segments object referring to `slot`, then one
 * cudaMemcpyAsync moves the whole blob, then the slot's ready event is
 * recorded.  The caller keeps host_blob unchanged until side_stream has
 * passed the copy.  Segments objects built before this call that refer to
 * `slot` become stale (apply on them returns SALT_ERR_STALE_SEGMENTS until
 * they are rebuilt).
 */
salt_status salt_residual_load(salt_ctx *ctx, int32_t slot, const void *host_blob,
                               salt_stream_t side_stream);

/*
 * salt_residual_load for n residuals at once (the per-step swap of a
 * serving engine, Section "Multi-Tenant Serving").  slots[n] (distinct) and
 * host_blobs[n] are host arrays; every blob is checked as in
 * salt_residual_load before anything is enqueued (an error leaves every
 * slot as it was).  On side_stream: one wait for the applies enqueued so
 * far on every segments object that refers to any of the slots, then one
 * cudaMemcpyAsync per blob, each followed by its slot's ready event.  The
 * result is that of n salt_residual_load calls in order; the host-side cost
 * is one hazard wait instead of n.  n == 0 does nothing.
 */
salt_status salt_residual_load_batch(salt_ctx *ctx, int32_t n, const int32_t *slots, const void *const *host_blobs,
                                     salt_stream_t side_stream);

/* Allocate a segments object able to hold max_tokens tokens of this
 * context (device metadata plus a pinned id staging area).  Synchronous. */
salt_status salt_segments_create(salt_ctx *ctx, salt_segments **out);

/* Wait for every use of the segments object and free it.  NULL is a no-op. */
void salt_segments_destroy(salt_segments *seg);

/*
 * Group a batch (Section "Multi-Tenant Serving": requests are grouped by
 * their centroid; residuals are batched heterogeneously, as with SGMV in
 * Section "Multi-Tenant LoRA Serving").  domain_ids and slot_ids are
 * int32[n_tokens], -1 meaning "no term"; 0 <= n_tokens <= max_tokens.
 *
 * If the ids are host memory they are validated here (range, pinned
 * domain, loaded slot) and errors return at once; the set of slots they
 * name is recorded so that swaps and applies wait only on what they must.
 * If they are device memory they are validated by the kernel into the
 * device error word, and every slot counts as referenced.
 *
 * Output (device, owned by seg): tokens stably sorted by (domain, slot),
 * -1 first, ties in token order; domain runs; user runs; and row blocks
 * for the apply kernels.  Asynchronous on `stream`; waits for the swaps
 * of the slots it reads.  Rebuilding a segments object waits for every
 * apply enqueued on it.
 */
salt_status salt_build_segments(salt_ctx *ctx, salt_segments *seg,
                                 const int32_t *domain_ids, const int32_t *slot_ids,
                                 int32_t n_tokens, salt_stream_t stream);

/*
 * salt_build_segments with gamma bins (Section "Multi-Tenant Serving":
 * gamma takes one of a small fixed set of values (bins) and the frontend groups
 * requests by their (centroid, gamma) pair).  gamma_bins is int32[n_tokens]
 * in the same kind of memory as the other ids; each entry is -1 (no gamma:
 * the pinned s_c as is) or a bin in [0, n_gamma), and gamma[0..n_gamma)
 * (host floats, 0 <= n_gamma <= SALT_MAX_GAMMA_BINS, read during the call)
 * are the bins' values.  A token with domain d and bin g has the centroid
 * scale s_c(d) * gamma[g]; a token without a centroid ignores its bin.
 * Tokens are sorted stably by (domain, bin, slot), -1 first; domain runs
 * become runs of equal (domain, bin) and user runs runs of equal (domain,
 * bin, slot) (their bins: salt_segments_export_gamma).  The row blocks of
 * the apply kernels are cut from the same tokens ordered by (domain, slot)
 * instead (gamma multiplies each token's centroid term), so a user whose
 * tokens fall in several bins takes one set of residual rows in a block;
 * the blocks salt_segments_export reports index that order, which spans the
 * same positions as the grouped order for every domain.  A bin outside the
 * range is SALT_ERR_GAMMA_RANGE for host ids, SALT_DEVERR_GAMMA_RANGE (and
 * bin -1) for device ids.  Otherwise as salt_build_segments, which is this
 * call with every bin -1.
 */
salt_status salt_build_segments_gamma(salt_ctx *ctx, salt_segments *seg, const int32_t *domain_ids,
                                      const int32_t *gamma_bins, const int32_t *slot_ids,
                                      int32_t n_tokens, int32_t n_gamma, const float *gamma,
                                      salt_stream_t stream);

/* The gamma bins of the last build's domain runs and user runs (-1: none),
 * in the order of salt_segments_export's dseg_* and useg_* arrays.  Either
 * pointer may be NULL.  Synchronous. */
salt_status salt_segments_export_gamma(salt_ctx *ctx, const salt_segments *seg, int32_t *dseg_gbin,
                                       int32_t *useg_gbin);

/*
 * Copy the segment metadata to host buffers (synchronous; for tests and
 * diagnostics).  counts[0..3] = n_tokens, domain runs, user runs, row
 * blocks.  Each array pointer may be NULL; sizes: perm[n_tokens],
 * dseg_ptr[runs + 1], dseg_dom[runs], useg_ptr[runs + 1], useg_dom[runs],
 * useg_slot[runs], blocks[3 * blocks] as (start, length, domain) triples.
 * Buffers of max_tokens + 1 entries (3 * max_tokens for blocks) always
 * suffice.
 */
salt_status salt_segments_export(salt_ctx *ctx, const salt_segments *seg, int32_t *counts,
                                 int32_t *perm, int32_t *dseg_ptr, int32_t *dseg_dom,
                                 int32_t *useg_ptr, int32_t *useg_dom, int32_t *useg_slot,
                                 int32_t *blocks);

/*
 * Apply centroid + residual LoRA to one layer (Section "Multi-Tenant
 * Serving", W_final): for every token t of the batch seg was built from,
 * y[t, :] += s_c (x[t] A_c) B_c + s_u (x[t] a_u) b_u, accumulated in fp32
 * and rounded once to bf16 (round to nearest even).  x is device
 * bf16[n_tokens][d_in_layer], y device bf16[n_tokens][d_out_layer], both
 * 16-byte aligned, rows contiguous; y is read and written in place and
 * must not overlap x.  Tokens whose ids are both -1 are not touched.
 * Asynchronous on `stream`.
 */
salt_status salt_lora_apply(salt_ctx *ctx, const salt_segments *seg, int32_t layer,
                            const void *x, void *y, salt_stream_t stream);

/*
 * The same for n (1..SALT_MAX_GROUP) layers that share the batch, in one
 * launch: layers[i], x[i], y[i] as in salt_lora_apply.  Use it for
 * projections that read the same step's activations (q/k/v, gate/up).
 * The y buffers must not overlap one another or any x.
 */
salt_status salt_lora_apply_grouped(salt_ctx *ctx, const salt_segments *seg, int32_t n,
                                    const int32_t *layers, const void *const *x,
                                    void *const *y, salt_stream_t stream);

/*
 * The projection with its base weight (Section "Multi-Tenant Serving": the
 * served weight is W_final = W_base + gamma * Wbar + delta_i): for every
 * token t of the batch seg was built from,
 *     y[t, :] = x[t] W_base + s_c (x[t] A_c) B_c + s_u (x[t] a_u) b_u,
 * accumulated in fp32 and rounded once to bf16 (round to nearest even); y
 * is written, never read (tokens with both ids -1 get x[t] W_base).  W is
 * device bf16 in one of the layouts of salt_centroid_fold
 * (SALT_W_IN_OUT: W[d_in][d_out]; SALT_W_OUT_IN: W[d_out][d_in]); x, W and
 * y are 16-byte aligned, y does not overlap x or W.  Two launches on
 * `stream`: the apply kernel writing the row blocks' V tiles into the
 * segments workspace, then one tcgen05 kernel that runs the GEMM over
 * 128-token tiles in grouped order and adds each overlapping row block's
 * V * [B_c; b_u] into the same accumulator.  Asynchronous; the workspace
 * is shared with salt_lora_apply on the same segments object (stream
 * order keeps them apart).
 */
salt_status salt_lora_apply_with_base(salt_ctx *ctx, const salt_segments *seg, int32_t layer,
                                      const void *x, const void *W, int32_t layout, void *y,
                                      salt_stream_t stream);

/*
 * salt_lora_apply for callers that cannot allocate device memory when they
 * apply - for example a serving engine whose device memory is planned up
 * front and that forbids allocations once serving starts, or code that
 * runs where cudaMalloc is not allowed.  (The paper has no counterpart;
 * this is a deployment convenience of the library.)
 *
 * Same arguments, result and ordering as salt_lora_apply, for one layer.
 * The apply's scratch - the intermediate V tiles, the partial sums of the
 * split shrink, the per-block ready flags and a launch counter, about
 * 12 MiB - lives in static device arrays of this library (held by every
 * device that loads the library until the process exits, zero when it
 * loads) instead of the segments object's workspace; the call itself
 * allocates nothing.  Limit: the batch may need at most 64 row blocks
 * (blocks hold <= 128 tokens of one domain); a larger batch returns
 * SALT_ERR_TOO_MANY_TOKENS before any device work.  The host judges this
 * from the ids of the build: for host ids it counts the blocks each domain
 * can need (ceil(tokens / 128) + ceil(user runs / block_users), see
 * salt_ctx_get_info); device ids cannot be read on the host, so it uses the
 * bound that holds for any ids, n_tokens / 128 + n_tokens / block_users +
 * n_domains + 3, which refuses some batches that would fit (with rank-64
 * centroids and rank-2 residuals, block_users = 32, from about 1,400 tokens
 * with 8 domains).  The first call on a
 * device looks up the arrays' device addresses (cudaGetSymbolAddress);
 * make that first call before any stream capture.  Every call shares the
 * one set of arrays: calls that may overlap on the GPU (on different
 * streams, or from different contexts or threads) race on them and must be
 * serialised by the caller.
 */
salt_status salt_lora_apply_static(salt_ctx *ctx, const salt_segments *seg, int32_t layer,
                                   const void *x, void *y, salt_stream_t stream);

/*
 * Applies on activations that live in host memory (Section "Multi-Tenant
 * Serving": the same W_final apply, for an engine whose activations of a
 * step arrive from and return to the host).  A pipe owns n_stages device
 * staging areas of stage_bytes each (0: room for the SALT_MAX_GROUP
 * largest layers of the table at max_tokens tokens), one host-to-device and
 * one device-to-host copy stream, and the events that order them.
 * salt_host_pipe_create allocates all of it (synchronous); 2 <= n_stages
 * <= 8 (0: 3).  The pipe belongs to ctx and must be destroyed before it.
 */
typedef struct salt_host_pipe salt_host_pipe;
salt_status salt_host_pipe_create(salt_ctx *ctx, int32_t n_stages, int64_t stage_bytes, salt_host_pipe **out);

/* Wait for everything the pipe enqueued, then free it.  NULL is a no-op. */
void salt_host_pipe_destroy(salt_host_pipe *pipe);

/*
 * salt_lora_apply_grouped on host activations: x_host[i]
 * ([n_tokens][d_in] bf16) and y_host[i] ([n_tokens][d_out] bf16, updated in
 * place) are page-locked host buffers (SALT_ERR_NOT_PINNED_HOST otherwise),
 * 16-byte aligned.  The call takes the pipe's next staging area, and
 * enqueues: on the pipe's H2D stream, once the area's previous results
 * have been copied out, one cudaMemcpyAsync per x and per y buffer; on
 * `stream`, after those copies, the grouped apply on the staged copies; on
 * the pipe's D2H stream, after the apply, one cudaMemcpyAsync per y back
 * into y_host[i].  So with consecutive calls the copies in of call k + 1
 * and the copies out of call k - 1 overlap the apply of call k.  The
 * buffers' contents must stay unchanged (x, y) and unread (y) until the
 * results are out: salt_host_pipe_wait.  The group's buffers must fit one
 * staging area (SALT_ERR_INVALID_ARG otherwise).  Asynchronous.
 */
salt_status salt_lora_apply_host(salt_host_pipe *pipe, const salt_segments *seg, int32_t n,
                                 const int32_t *layers, const void *const *x_host, void *const *y_host,
                                 salt_stream_t stream);

/* Make `stream` wait (asynchronously) until every result the pipe has
 * enqueued so far is back in host memory. */
salt_status salt_host_pipe_wait(salt_host_pipe *pipe, salt_stream_t stream);

/*
 * The alignment regulariser of Phase 1 (Eq. 2), for n pairs of a task
 * update and a centroid:
 *     L_align = 1 - Tr(dW^T Wbar) / (||dW||_F ||Wbar||_F + eps),
 *     dW = s A B (rank r),  Wbar = s_c A_c B_c (rank rc),
 * evaluated without forming either d_in x d_out matrix: with the stacked
 * factors F_in = [At ; At_c] ([r + rc][d_in]) and F_out = [B ; B_c], the
 * trace and both squared norms are sums over blocks of G_in o G_out, where
 * G = F F^T are (r + rc)^2 Gram matrices contracted on the tensor cores
 * (bf16 operands, fp32 accumulation) and combined in fp32 in a fixed
 * order (the result does not depend on timing).  The paper's
 * eps is 1e-8.  pairs is a host array; its factor pointers are device bf16
 * arrays, rows contiguous, 16-byte aligned; 1 <= r, 1 <= rc,
 * r + rc <= SALT_MAX_ALIGN_RANK, d_in and d_out positive multiples of 8.
 * loss and cosine (the quotient; may be NULL) are device float[n].
 * Scratch comes from the stream-ordered allocator of the current device.
 * Asynchronous on `stream`.  Not on the serving path: the regulariser of
 * centroid training, offered for checking or monitoring alignment.
 */
typedef struct salt_align_pair {
    const void *At;     /* [r][d_in]   task update's A, transposed */
    const void *B;      /* [r][d_out]  task update's B */
    const void *At_c;   /* [rc][d_in]  centroid's A, transposed */
    const void *B_c;    /* [rc][d_out] centroid's B */
    int32_t r, rc, d_in, d_out;
    float s, s_c;       /* scales of dW and Wbar */
} salt_align_pair;
salt_status salt_align_loss(int32_t n, const salt_align_pair *pairs, float eps, float *loss,
                            float *cosine, salt_stream_t stream);

/*
 * Self-test of the failure path.  Enqueues on `stream` one thread that
 * waits, with the same bounded wait the apply uses for results of other
 * CTAs (the V rows of a row block), on a device word nothing ever sets.  The
 * wait gives up after its limit (a fraction of a second), raises
 * SALT_DEVERR_TIMEOUT in the device error word and returns; the context and
 * the GPU stay usable.  Read the flag with salt_get_device_error.  (The
 * paper has no counterpart; it demonstrates that a lost result produces an
 * error status instead of a hang.)
 */
salt_status salt_selftest_wait_timeout(salt_ctx *ctx, salt_stream_t stream);

/*
 * Guard-band check (a diagnostic; the paper has no counterpart).  The
 * library's device buffers that kernels write or gather from - the centroid
 * arenas, the residual slot pool and, for a segments object, its V tiles and
 * split partials - sit between two 4 KiB bands of a fixed byte pattern.
 * This call waits for the device, reads the bands back and sets *damaged to
 * the number of bands that changed (0 when no store or copy ran past a
 * buffer).  seg may be NULL (context buffers only).  Synchronous.
 */
salt_status salt_guard_check(salt_ctx *ctx, const salt_segments *seg, int32_t *damaged);

/*
 * Synchronise `stream`, then read and clear the device error word.
 * *flags gets the SALT_DEVERR_* bits raised since the last call.  Returns
 * SALT_ERR_DEVICE_IDS if any bit was set, else SALT_OK.
 */
salt_status salt_get_device_error(salt_ctx *ctx, salt_stream_t stream, uint32_t *flags);

#ifdef __cplusplus
}
#endif

#endif /* SALT_H */
