// Host runtime behind the C ABI of include/salt.h.
//
// Owns the device state of SALT serving (Section "Multi-Tenant Serving"):
// the centroid arena (pinned once), the fixed residual slot pool filled by
// host -> device swaps on a side stream, and segments objects.  Ordering
// between swaps and applies is kept with events only; no call here waits
// for the device except the setup calls (create, pin, destroy) and the
// diagnostic ones (export, device error).
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <new>
#include <set>
#include <string>
#include <vector>
#include <algorithm>
#include <functional>
#include <map>
#include <mutex>

#include <sys/mman.h>

#include <nvtx3/nvToolsExt.h>

#include "salt_internal.cuh"

using namespace salt;

struct salt_ctx {
    int device = 0;
    int n_layers = 0;
    std::vector<int32_t> d_in, d_out;
    std::vector<int64_t> a_off, b_off, res_off;  // elements
    int64_t sum_din = 0, sum_dout = 0;
    int n_domains = 0, rc_max = 0, n_slots = 0, r_max = 0, max_tokens = 0;
    int umax = 1;
    uint64_t layout_hash = 0;

    uint16_t *arenaA = nullptr, *arenaB = nullptr;
    size_t arenaA_bytes = 0, arenaB_bytes = 0, pool_bytes = 0;
    int32_t *dom_rc_dev = nullptr;
    float *dom_sc_dev = nullptr;
    std::vector<int32_t> dom_rc;
    std::vector<float> dom_sc;

    uint8_t *pool = nullptr;
    int64_t slot_stride = 0;
    std::vector<int32_t> slot_rank;        // 0 = never loaded
    std::vector<uint64_t> slot_seq;        // loads issued
    std::vector<cudaEvent_t> slot_ready;
    std::vector<uint64_t> slot_waited_seq;
    std::vector<cudaStream_t> slot_waited_stream;

    uint32_t *err_dev = nullptr;
    std::set<salt_segments *> segs;
    std::string last_error;
};

struct salt_segments {
    salt_ctx *ctx = nullptr;
    SegDev d{};
    int32_t *staging[2] = {nullptr, nullptr};  // pinned host [2 * max_tokens]
    cudaEvent_t staging_ev[2] = {nullptr, nullptr};
    bool staging_used[2] = {false, false};
    int staging_next = 0;
    bool built = false;
    bool stale = false;
    bool tables_fresh = false;                 // built, and no apply launched since
    bool device_ids = false;
    int T = 0;
    int n_blk_bound = 0;                       // launch bound on the row blocks of the last build
    ApplyWork work{};                          // V tiles of the apply path
    std::vector<uint8_t> refs;                 // slots named by the last build (host ids)
    cudaStream_t build_stream = nullptr;
    std::vector<cudaStream_t> use_streams;     // build stream + apply streams since the build
    cudaEvent_t built_ev = nullptr;
    cudaEvent_t tmp_ev = nullptr;
};

// Staging and copy streams of applies on host activations.
struct salt_host_pipe {
    salt_ctx *ctx = nullptr;
    int n_stages = 0;
    int64_t stage_bytes = 0;
    std::vector<uint8_t *> stage;              // device staging areas
    cudaStream_t h2d = nullptr, d2h = nullptr;
    std::vector<cudaEvent_t> in_ready;         // staged copies in (H2D stream)
    std::vector<cudaEvent_t> applied;          // apply done (caller's stream)
    std::vector<cudaEvent_t> out_done;         // results copied out (D2H stream)
    std::vector<uint8_t> used;
    int next = 0;
    int last = -1;
};

namespace {

// A named NVTX range around a library call on the host (what a timeline
// tool shows next to the kernels the call enqueues); free when no tool is
// attached.
struct NvtxRange {
    explicit NvtxRange(const char *name) { nvtxRangePushA(name); }
    ~NvtxRange() { nvtxRangePop(); }
    NvtxRange(const NvtxRange &) = delete;
    NvtxRange &operator=(const NvtxRange &) = delete;
};

salt_status fail(salt_ctx *ctx, salt_status s, const char *fmt, ...)
{
    if (ctx) {
        char buf[512];
        va_list ap;
        va_start(ap, fmt);
        vsnprintf(buf, sizeof buf, fmt, ap);
        va_end(ap);
        ctx->last_error = buf;
    }
    return s;
}

#define CUDA_OR_FAIL(ctx, call)                                                                    \
    do {                                                                                           \
        cudaError_t e_ = (call);                                                                   \
        if (e_ != cudaSuccess)                                                                     \
            return fail((ctx), SALT_ERR_CUDA, "%s failed: %s", #call, cudaGetErrorString(e_));     \
    } while (0)

// Guard bands: the device buffers the kernels write or gather from (the
// centroid arena, the slot pool, the V tiles and the split partials) are
// allocated with GUARD_BYTES of a fixed byte pattern before and after
// them; salt_guard_check reads the bands back, so a store or a copy that
// runs past one of these buffers is detected (the pool's are also the
// bounds of every swap).
constexpr size_t GUARD_BYTES = 4096;
constexpr unsigned char GUARD_BYTE = 0xA5;

struct Guarded {
    void *usable;
    size_t bytes;
};

cudaError_t guarded_malloc(void **usable, size_t bytes)
{
    *usable = nullptr;
    uint8_t *base = nullptr;
    cudaError_t e = cudaMalloc(&base, bytes + 2 * GUARD_BYTES);
    if (e != cudaSuccess) return e;
    if ((e = cudaMemset(base, GUARD_BYTE, GUARD_BYTES)) != cudaSuccess ||
        (e = cudaMemset(base + GUARD_BYTES + bytes, GUARD_BYTE, GUARD_BYTES)) != cudaSuccess) {
        cudaFree(base);
        return e;
    }
    *usable = base + GUARD_BYTES;
    return cudaSuccess;
}

void guarded_free(void *usable)
{
    if (usable) cudaFree(static_cast<uint8_t *>(usable) - GUARD_BYTES);
}

// Number of the two bands of the buffer that no longer hold the pattern
// (synchronous); -1 if they cannot be read.
int guard_damage(const Guarded &g)
{
    if (!g.usable) return 0;
    std::vector<unsigned char> h(2 * GUARD_BYTES);
    const uint8_t *u = static_cast<const uint8_t *>(g.usable);
    if (cudaMemcpy(h.data(), u - GUARD_BYTES, GUARD_BYTES, cudaMemcpyDeviceToHost) != cudaSuccess ||
        cudaMemcpy(h.data() + GUARD_BYTES, u + g.bytes, GUARD_BYTES, cudaMemcpyDeviceToHost) != cudaSuccess) {
        cudaGetLastError();
        return -1;
    }
    int bad = 0;
    for (int side = 0; side < 2; ++side)
        for (size_t i = 0; i < GUARD_BYTES; ++i)
            if (h[side * GUARD_BYTES + i] != GUARD_BYTE) {
                ++bad;
                break;
            }
    return bad;
}

uint64_t fnv1a_layout(int n, const int32_t *din, const int32_t *dout)
{
    uint64_t h = 1469598103934665603ull;
    auto mix = [&](int32_t v) {
        uint32_t u = (uint32_t)v;
        for (int b = 0; b < 4; ++b) {
            h ^= (u >> (8 * b)) & 0xffu;
            h *= 1099511628211ull;
        }
    };
    for (int l = 0; l < n; ++l) {
        mix(din[l]);
        mix(dout[l]);
    }
    return h;
}

salt_status check_config(const salt_config *c)
{
    if (!c || c->n_layers < 1 || !c->d_in || !c->d_out) return SALT_ERR_INVALID_ARG;
    for (int l = 0; l < c->n_layers; ++l) {
        if (c->d_in[l] <= 0 || c->d_out[l] <= 0 || (c->d_in[l] % 8) || (c->d_out[l] % 8))
            return SALT_ERR_INVALID_ARG;
    }
    // the segment key holds domain + 1 in 17 bits; a residual row code holds the slot in 17
    if (c->n_domains < 0 || c->n_domains >= (1 << 17) - 1) return SALT_ERR_INVALID_ARG;
    if (c->n_slots < 0 || c->n_slots >= (1 << 17)) return SALT_ERR_INVALID_ARG;
    if (c->rc_max < 0 || c->rc_max > SALT_MAX_CENTROID_RANK) return SALT_ERR_RANK;
    if (c->r_max < 1 || c->r_max > SALT_MAX_RESIDUAL_RANK) return SALT_ERR_RANK;
    if (c->rc_max + c->r_max > SALT_MAX_TOKEN_RANK) return SALT_ERR_RANK;
    if (c->max_tokens < 1 || c->max_tokens > SALT_MAX_TOKENS) return SALT_ERR_TOO_MANY_TOKENS;
    return SALT_OK;
}

int64_t payload_elems(const salt_config *c, int rank)
{
    int64_t s = 0;
    for (int l = 0; l < c->n_layers; ++l) s += (int64_t)c->d_in[l] + c->d_out[l];
    return s * rank;
}

bool set_device(salt_ctx *ctx)
{
    int cur = -1;
    if (cudaGetDevice(&cur) != cudaSuccess) return false;
    if (cur == ctx->device) return true;
    return cudaSetDevice(ctx->device) == cudaSuccess;
}

bool is_device_pointer(const void *p)
{
    cudaPointerAttributes a;
    if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged;
}

void add_stream(std::vector<cudaStream_t> &v, cudaStream_t s)
{
    for (cudaStream_t x : v)
        if (x == s) return;
    v.push_back(s);
}

// Row blocks of a T-token batch, whatever the ids: blocks <= T/TM + groups
// and groups <= user runs / umax + domains (+ 1 for the skipped run).
int block_bound_loose(const salt_ctx *ctx, int T)
{
    int64_t b = (int64_t)T / TM + (int64_t)T / ctx->umax + ctx->n_domains + 3;
    return (int)(b < T ? (b > 0 ? b : 1) : (T > 0 ? T : 1));
}

// Tighter bound from validated host ids: a domain with n tokens (those
// with a term) in u user runs (runs of equal gamma bin and slot) yields at
// most ceil(n / TM) + ceil(u / umax) blocks.  Only sizes the launch grid;
// the block list itself comes from the segment kernel, and CTAs past its
// count exit at once.
int block_bound_host(const salt_ctx *ctx, const int32_t *dom, const int32_t *gbin, const int32_t *slot, int T)
{
    std::vector<uint64_t> keys;
    keys.reserve(T);
    for (int t = 0; t < T; ++t) {
        if (dom[t] < 0 && slot[t] < 0) continue;
        const uint32_t g = (gbin && dom[t] >= 0) ? (uint32_t)(gbin[t] + 1) : 0u;
        keys.push_back(((uint64_t)(uint32_t)(dom[t] + 1) << 32) | (g << 20) | (uint32_t)(slot[t] + 1));
    }
    std::sort(keys.begin(), keys.end());
    int64_t bound = 0;
    size_t i = 0;
    while (i < keys.size()) {
        uint32_t d = (uint32_t)(keys[i] >> 32);
        int64_t n = 0, u = 0;
        uint64_t prev = ~0ull;
        while (i < keys.size() && (uint32_t)(keys[i] >> 32) == d) {
            if (keys[i] != prev) ++u;
            prev = keys[i];
            ++n;
            ++i;
        }
        bound += (n + TM - 1) / TM + (u + ctx->umax - 1) / ctx->umax;
    }
    int cap = block_bound_loose(ctx, ctx->max_tokens);
    return (int)(bound < cap ? bound : cap);
}

// Make `stream` wait for all work enqueued so far on the streams that used seg.
cudaError_t wait_for_uses(salt_segments *seg, cudaStream_t stream)
{
    for (cudaStream_t s : seg->use_streams) {
        if (s == stream) continue;
        cudaError_t e = cudaEventRecord(seg->tmp_ev, s);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(stream, seg->tmp_ev, 0);
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

// Huge-page size of the kernel's transparent huge pages (2 MiB when unknown).
int64_t thp_bytes()
{
    int64_t v = 0;
    if (FILE *f = std::fopen("/sys/kernel/mm/transparent_hugepage/hpage_pmd_size", "r")) {
        long long x = 0;
        if (std::fscanf(f, "%lld", &x) == 1) v = x;
        std::fclose(f);
    }
    return v > 0 ? v : (int64_t)2 << 20;
}

std::mutex g_host_mu;
std::map<void *, size_t> g_host_maps;  // salt_host_alloc regions and their mapped sizes

// Whether [p, p + bytes) lies in one salt_host_alloc region (page-locked by
// this library: no driver query needed).
bool in_host_region(const void *p, uint64_t bytes)
{
    std::lock_guard<std::mutex> lock(g_host_mu);
    auto it = g_host_maps.upper_bound(const_cast<void *>(p));
    if (it == g_host_maps.begin()) return false;
    --it;
    const uintptr_t a = reinterpret_cast<uintptr_t>(it->first), q = reinterpret_cast<uintptr_t>(p);
    return q >= a && q + bytes <= a + it->second;
}

// Checks of one residual blob for a load into `slot`; *rank and *bytes get
// its rank and its size (header and payload).
salt_status check_blob(salt_ctx *ctx, int32_t slot, const void *host_blob, int32_t *rank, uint64_t *bytes)
{
    if (slot < 0 || slot >= ctx->n_slots) return fail(ctx, SALT_ERR_SLOT_RANGE, "slot %d outside [0, %d)", slot, ctx->n_slots);
    if (!host_blob) return fail(ctx, SALT_ERR_INVALID_ARG, "null blob");
    auto pinned_by_driver = [&]() -> salt_status {
        cudaPointerAttributes attr;
        if (cudaPointerGetAttributes(&attr, host_blob) != cudaSuccess) {
            cudaGetLastError();
            return fail(ctx, SALT_ERR_NOT_PINNED_HOST, "blob pointer is not registered with CUDA");
        }
        if (attr.type != cudaMemoryTypeHost)
            return fail(ctx, SALT_ERR_NOT_PINNED_HOST, "blob is not page-locked host memory (type %d)", (int)attr.type);
        return SALT_OK;
    };
    // the header is read on the host only once it is known to be host memory
    const bool in_region = in_host_region(host_blob, SALT_BLOB_HEADER_BYTES);
    if (!in_region) {
        salt_status st = pinned_by_driver();
        if (st != SALT_OK) return st;
    }
    salt_blob_header h;
    std::memcpy(&h, host_blob, sizeof h);
    if (h.magic != SALT_BLOB_MAGIC || h.version != 1) return fail(ctx, SALT_ERR_BAD_BLOB, "bad blob magic or version");
    if (h.n_layers != ctx->n_layers || h.layout_hash != ctx->layout_hash)
        return fail(ctx, SALT_ERR_BAD_BLOB, "blob was built for another layer table");
    if (h.rank < 1 || h.rank > ctx->r_max) return fail(ctx, SALT_ERR_RANK, "blob rank %d outside [1, %d]", h.rank, ctx->r_max);
    uint64_t pay = (uint64_t)(ctx->sum_din + ctx->sum_dout) * (uint64_t)h.rank * 2;
    if (h.payload_bytes != pay) return fail(ctx, SALT_ERR_BAD_BLOB, "blob payload size mismatch");
    if (in_region && !in_host_region(host_blob, SALT_BLOB_HEADER_BYTES + pay)) {
        salt_status st = pinned_by_driver();  // the blob runs past the region
        if (st != SALT_OK) return st;
    }
    *rank = h.rank;
    *bytes = SALT_BLOB_HEADER_BYTES + pay;
    return SALT_OK;
}

// The loads of n checked blobs on `side`: readers first (every segments
// object that names one of the slots waits for its uses, once), then one
// copy and one ready event per slot.
salt_status enqueue_loads(salt_ctx *ctx, int32_t n, const int32_t *slots, const void *const *blobs, const int32_t *ranks,
                          const uint64_t *bytes, cudaStream_t side)
{
    for (salt_segments *seg : ctx->segs) {
        if (!seg->built) continue;
        bool names = seg->device_ids;
        for (int32_t i = 0; i < n && !names; ++i) names = seg->refs[slots[i]] != 0;
        if (!names) continue;
        seg->stale = true;
        CUDA_OR_FAIL(ctx, wait_for_uses(seg, side));
    }
    for (int32_t i = 0; i < n; ++i) {
        const int32_t slot = slots[i];
        uint8_t *dst = ctx->pool + (int64_t)slot * ctx->slot_stride;
        CUDA_OR_FAIL(ctx, cudaMemcpyAsync(dst, blobs[i], bytes[i], cudaMemcpyHostToDevice, side));
        CUDA_OR_FAIL(ctx, cudaEventRecord(ctx->slot_ready[slot], side));
        ctx->slot_rank[slot] = ranks[i];
        ctx->slot_seq[slot] += 1;
    }
    return SALT_OK;
}
}  // namespace

extern "C" {

void *salt_host_alloc(int64_t bytes)
{
    if (bytes <= 0) return nullptr;
    const int64_t hp = thp_bytes();
    const size_t size = (size_t)((bytes + hp - 1) / hp * hp);
    void *p = mmap(nullptr, size, PROT_READ | PROT_WRITE, MAP_PRIVATE | MAP_ANONYMOUS, -1, 0);
    if (p == MAP_FAILED) return nullptr;
#ifdef MADV_HUGEPAGE
    madvise(p, size, MADV_HUGEPAGE);  // advice only: base pages if refused
#endif
    std::memset(p, 0, size);  // fault every page in before it is registered
    // Where the faults got base pages (no free huge page at the time),
    // ask the kernel to collapse the range into huge pages now (Linux 6.1
    // and later; refused or ignored elsewhere, which leaves base pages).
    constexpr int kMadvCollapse = 25;
    madvise(p, size, kMadvCollapse);
    if (cudaHostRegister(p, size, cudaHostRegisterDefault) != cudaSuccess) {
        cudaGetLastError();
        munmap(p, size);
        return nullptr;
    }
    std::lock_guard<std::mutex> lock(g_host_mu);
    g_host_maps[p] = size;
    return p;
}

void salt_host_free(void *ptr)
{
    if (!ptr) return;
    size_t size = 0;
    {
        std::lock_guard<std::mutex> lock(g_host_mu);
        auto it = g_host_maps.find(ptr);
        if (it == g_host_maps.end()) return;
        size = it->second;
        g_host_maps.erase(it);
    }
    cudaHostUnregister(ptr);
    munmap(ptr, size);
}

int32_t salt_abi_version(void) { return SALT_ABI_VERSION; }

const char *salt_status_string(salt_status s)
{
    switch (s) {
    case SALT_OK: return "ok";
    case SALT_ERR_INVALID_ARG: return "invalid argument";
    case SALT_ERR_OOM: return "out of memory";
    case SALT_ERR_NOT_PINNED_HOST: return "host buffer is not page-locked";
    case SALT_ERR_DOMAIN_NOT_PINNED: return "domain has no pinned centroid";
    case SALT_ERR_SLOT_RANGE: return "slot id out of range";
    case SALT_ERR_RANK: return "rank out of range";
    case SALT_ERR_LAYER_RANGE: return "layer index out of range";
    case SALT_ERR_ALIGN: return "pointer not 16-byte aligned";
    case SALT_ERR_BAD_BLOB: return "invalid residual blob";
    case SALT_ERR_DEVICE_IDS: return "device-side id check failed";
    case SALT_ERR_TIMEOUT: return "device wait timed out";
    case SALT_ERR_CUDA: return "CUDA error";
    case SALT_ERR_SLOT_EMPTY: return "slot was never loaded";
    case SALT_ERR_TOO_MANY_TOKENS: return "too many tokens";
    case SALT_ERR_DOMAIN_RANGE: return "domain id out of range";
    case SALT_ERR_STALE_SEGMENTS: return "segments refer to a slot reloaded after the build";
    case SALT_ERR_NOT_BUILT: return "segments object not built";
    case SALT_ERR_GAMMA_RANGE: return "gamma bin out of range";
    }
    return "unknown status";
}

const char *salt_last_error(const salt_ctx *ctx) { return ctx ? ctx->last_error.c_str() : "null context"; }

salt_status salt_ctx_get_info(const salt_ctx *ctx, salt_ctx_info *info)
{
    if (!ctx || !info) return SALT_ERR_INVALID_ARG;
    std::memset(info, 0, sizeof *info);
    info->arena_bytes = (int64_t)ctx->n_domains * ctx->rc_max * (ctx->sum_din + ctx->sum_dout) * 2;
    info->pool_bytes = ctx->slot_stride * (int64_t)ctx->n_slots;
    info->slot_stride = ctx->slot_stride;
    int dev_sms = 0;
    if (cudaDeviceGetAttribute(&dev_sms, cudaDevAttrMultiProcessorCount, ctx->device) != cudaSuccess) {
        cudaGetLastError();
        dev_sms = 0;
    }
    info->apply_ctas = dev_sms;
    info->k_splits_max = 16;
    info->apply_smem_bytes = (int32_t)apply_smem_bytes();
    info->block_tokens = TM;
    info->block_users = ctx->umax;
    return SALT_OK;
}

salt_status salt_ctx_create(const salt_config *config, salt_ctx **out)
{
    if (!out) return SALT_ERR_INVALID_ARG;
    *out = nullptr;
    salt_status st = check_config(config);
    if (st != SALT_OK) return st;
    salt_ctx *ctx = new (std::nothrow) salt_ctx;
    if (!ctx) return SALT_ERR_OOM;
    ctx->device = config->device;
    if (cudaSetDevice(ctx->device) != cudaSuccess) {
        cudaGetLastError();
        delete ctx;
        return SALT_ERR_CUDA;
    }
    ctx->n_layers = config->n_layers;
    ctx->d_in.assign(config->d_in, config->d_in + config->n_layers);
    ctx->d_out.assign(config->d_out, config->d_out + config->n_layers);
    ctx->n_domains = config->n_domains;
    ctx->rc_max = config->rc_max;
    ctx->n_slots = config->n_slots;
    ctx->r_max = config->r_max;
    ctx->max_tokens = config->max_tokens;
    ctx->umax = (S_MAX - ctx->rc_max) / ctx->r_max;
    ctx->layout_hash = fnv1a_layout(ctx->n_layers, config->d_in, config->d_out);
    int64_t a = 0, b = 0, r = 0;
    for (int l = 0; l < ctx->n_layers; ++l) {
        ctx->a_off.push_back(a);
        ctx->b_off.push_back(b);
        ctx->res_off.push_back(r);
        a += (int64_t)ctx->n_domains * ctx->rc_max * ctx->d_in[l];
        b += (int64_t)ctx->n_domains * ctx->rc_max * ctx->d_out[l];
        r += (int64_t)ctx->d_in[l] + ctx->d_out[l];
        ctx->sum_din += ctx->d_in[l];
        ctx->sum_dout += ctx->d_out[l];
    }
    auto cleanup_fail = [&](salt_status s) {
        salt_ctx_destroy(ctx);
        return s;
    };
    ctx->arenaA_bytes = (size_t)a * 2;
    ctx->arenaB_bytes = (size_t)b * 2;
    if (a > 0 && guarded_malloc(reinterpret_cast<void **>(&ctx->arenaA), ctx->arenaA_bytes) != cudaSuccess)
        return cleanup_fail(SALT_ERR_OOM);
    if (b > 0 && guarded_malloc(reinterpret_cast<void **>(&ctx->arenaB), ctx->arenaB_bytes) != cudaSuccess)
        return cleanup_fail(SALT_ERR_OOM);
    // rows of a domain beyond its pinned rank stay zero
    if (a > 0 && cudaMemset(ctx->arenaA, 0, (size_t)a * 2) != cudaSuccess) return cleanup_fail(SALT_ERR_CUDA);
    if (b > 0 && cudaMemset(ctx->arenaB, 0, (size_t)b * 2) != cudaSuccess) return cleanup_fail(SALT_ERR_CUDA);
    int nd = ctx->n_domains > 0 ? ctx->n_domains : 1;
    if (cudaMalloc(&ctx->dom_rc_dev, sizeof(int32_t) * nd) != cudaSuccess) return cleanup_fail(SALT_ERR_OOM);
    if (cudaMalloc(&ctx->dom_sc_dev, sizeof(float) * nd) != cudaSuccess) return cleanup_fail(SALT_ERR_OOM);
    if (cudaMemset(ctx->dom_rc_dev, 0, sizeof(int32_t) * nd) != cudaSuccess) return cleanup_fail(SALT_ERR_CUDA);
    if (cudaMemset(ctx->dom_sc_dev, 0, sizeof(float) * nd) != cudaSuccess) return cleanup_fail(SALT_ERR_CUDA);
    ctx->dom_rc.assign(nd, 0);
    ctx->dom_sc.assign(nd, 0.f);
    ctx->slot_stride = (SALT_BLOB_HEADER_BYTES + payload_elems(config, ctx->r_max) * 2 + 255) / 256 * 256;
    int ns = ctx->n_slots > 0 ? ctx->n_slots : 1;
    ctx->pool_bytes = (size_t)ctx->slot_stride * ns;
    if (guarded_malloc(reinterpret_cast<void **>(&ctx->pool), ctx->pool_bytes) != cudaSuccess)
        return cleanup_fail(SALT_ERR_OOM);
    if (cudaMemset(ctx->pool, 0, (size_t)ctx->slot_stride * ns) != cudaSuccess) return cleanup_fail(SALT_ERR_CUDA);
    ctx->slot_rank.assign(ns, 0);
    ctx->slot_seq.assign(ns, 0);
    ctx->slot_waited_seq.assign(ns, 0);
    ctx->slot_waited_stream.assign(ns, nullptr);
    ctx->slot_ready.assign(ns, nullptr);
    for (int s = 0; s < ns; ++s)
        if (cudaEventCreateWithFlags(&ctx->slot_ready[s], cudaEventDisableTiming) != cudaSuccess)
            return cleanup_fail(SALT_ERR_CUDA);
    if (cudaMalloc(&ctx->err_dev, sizeof(uint32_t)) != cudaSuccess) return cleanup_fail(SALT_ERR_OOM);
    if (cudaMemset(ctx->err_dev, 0, sizeof(uint32_t)) != cudaSuccess) return cleanup_fail(SALT_ERR_CUDA);
    if (apply_prepare(ctx->device) != cudaSuccess || base_prepare(ctx->device) != cudaSuccess) {
        cudaGetLastError();
        return cleanup_fail(SALT_ERR_CUDA);
    }
    if (cudaDeviceSynchronize() != cudaSuccess) return cleanup_fail(SALT_ERR_CUDA);
    *out = ctx;
    return SALT_OK;
}

void salt_ctx_destroy(salt_ctx *ctx)
{
    if (!ctx) return;
    set_device(ctx);
    cudaDeviceSynchronize();
    guarded_free(ctx->arenaA);
    guarded_free(ctx->arenaB);
    cudaFree(ctx->dom_rc_dev);
    cudaFree(ctx->dom_sc_dev);
    guarded_free(ctx->pool);
    cudaFree(ctx->err_dev);
    for (cudaEvent_t e : ctx->slot_ready)
        if (e) cudaEventDestroy(e);
    cudaGetLastError();
    delete ctx;
}

salt_status salt_centroid_pin(salt_ctx *ctx, int32_t domain, int32_t rc, const void *At_c, const void *B_c,
                              float s_c)
{
    NvtxRange nvtx_range("salt_centroid_pin");
    if (!ctx) return SALT_ERR_INVALID_ARG;
    if (domain < 0 || domain >= ctx->n_domains)
        return fail(ctx, SALT_ERR_DOMAIN_RANGE, "domain %d outside [0, %d)", domain, ctx->n_domains);
    if (rc < 1 || rc > ctx->rc_max) return fail(ctx, SALT_ERR_RANK, "centroid rank %d outside [1, %d]", rc, ctx->rc_max);
    if (!At_c || !B_c) return fail(ctx, SALT_ERR_INVALID_ARG, "null factor pointer");
    if (!set_device(ctx)) return fail(ctx, SALT_ERR_CUDA, "cannot select device %d", ctx->device);
    CUDA_OR_FAIL(ctx, cudaDeviceSynchronize());
    const uint16_t *A = static_cast<const uint16_t *>(At_c);
    const uint16_t *B = static_cast<const uint16_t *>(B_c);
    int64_t oa = 0, ob = 0;
    for (int l = 0; l < ctx->n_layers; ++l) {
        int64_t na = (int64_t)rc * ctx->d_in[l], nb = (int64_t)rc * ctx->d_out[l];
        uint16_t *da = ctx->arenaA + ctx->a_off[l] + (int64_t)domain * ctx->rc_max * ctx->d_in[l];
        uint16_t *db = ctx->arenaB + ctx->b_off[l] + (int64_t)domain * ctx->rc_max * ctx->d_out[l];
        CUDA_OR_FAIL(ctx, cudaMemcpy(da, A + oa, (size_t)na * 2, cudaMemcpyDefault));
        CUDA_OR_FAIL(ctx, cudaMemcpy(db, B + ob, (size_t)nb * 2, cudaMemcpyDefault));
        oa += na;
        ob += nb;
    }
    CUDA_OR_FAIL(ctx, cudaMemcpy(ctx->dom_rc_dev + domain, &rc, sizeof rc, cudaMemcpyHostToDevice));
    CUDA_OR_FAIL(ctx, cudaMemcpy(ctx->dom_sc_dev + domain, &s_c, sizeof s_c, cudaMemcpyHostToDevice));
    ctx->dom_rc[domain] = rc;
    ctx->dom_sc[domain] = s_c;
    return SALT_OK;
}

int64_t salt_residual_blob_bytes(const salt_config *config, int32_t rank)
{
    if (!config || config->n_layers < 1 || !config->d_in || !config->d_out || rank < 1) return -1;
    for (int l = 0; l < config->n_layers; ++l)
        if (config->d_in[l] <= 0 || config->d_out[l] <= 0) return -1;
    return SALT_BLOB_HEADER_BYTES + payload_elems(config, rank) * 2;
}

salt_status salt_residual_blob_pack(const salt_config *config, int32_t rank, float s_u, const void *At_u,
                                    const void *B_u, void *blob, int64_t blob_bytes)
{
    int64_t need = salt_residual_blob_bytes(config, rank);
    if (need < 0 || !At_u || !B_u || !blob) return SALT_ERR_INVALID_ARG;
    if (rank > SALT_MAX_RESIDUAL_RANK) return SALT_ERR_RANK;
    if (blob_bytes < need) return SALT_ERR_INVALID_ARG;
    salt_blob_header h;
    std::memset(&h, 0, sizeof h);
    h.magic = SALT_BLOB_MAGIC;
    h.version = 1;
    h.rank = rank;
    h.n_layers = config->n_layers;
    h.s_u = s_u;
    h.payload_bytes = (uint64_t)payload_elems(config, rank) * 2;
    h.layout_hash = fnv1a_layout(config->n_layers, config->d_in, config->d_out);
    uint8_t *out = static_cast<uint8_t *>(blob);
    std::memcpy(out, &h, sizeof h);
    uint16_t *pay = reinterpret_cast<uint16_t *>(out + SALT_BLOB_HEADER_BYTES);
    const uint16_t *A = static_cast<const uint16_t *>(At_u);
    const uint16_t *B = static_cast<const uint16_t *>(B_u);
    int64_t oa = 0, ob = 0, op = 0;
    for (int l = 0; l < config->n_layers; ++l) {
        int64_t na = (int64_t)rank * config->d_in[l], nb = (int64_t)rank * config->d_out[l];
        std::memcpy(pay + op, A + oa, (size_t)na * 2);
        std::memcpy(pay + op + na, B + ob, (size_t)nb * 2);
        oa += na;
        ob += nb;
        op += na + nb;
    }
    return SALT_OK;
}

salt_status salt_centroid_fold(salt_ctx *ctx, int32_t domain, int32_t layer, float gamma, void *W, int32_t layout,
                               salt_stream_t stream)
{
    NvtxRange nvtx_range("salt_centroid_fold");
    if (!ctx) return SALT_ERR_INVALID_ARG;
    if (domain < 0 || domain >= ctx->n_domains)
        return fail(ctx, SALT_ERR_DOMAIN_RANGE, "domain %d outside [0, %d)", domain, ctx->n_domains);
    if (ctx->dom_rc[domain] == 0) return fail(ctx, SALT_ERR_DOMAIN_NOT_PINNED, "domain %d has no pinned centroid", domain);
    if (layer < 0 || layer >= ctx->n_layers)
        return fail(ctx, SALT_ERR_LAYER_RANGE, "layer %d outside [0, %d)", layer, ctx->n_layers);
    if (layout != SALT_W_IN_OUT && layout != SALT_W_OUT_IN) return fail(ctx, SALT_ERR_INVALID_ARG, "unknown layout %d", layout);
    if (!W) return fail(ctx, SALT_ERR_INVALID_ARG, "null weight");
    if (reinterpret_cast<uintptr_t>(W) & 15u) return fail(ctx, SALT_ERR_ALIGN, "weight not 16-byte aligned");
    if (!set_device(ctx)) return fail(ctx, SALT_ERR_CUDA, "cannot select device %d", ctx->device);
    const int din = ctx->d_in[layer], dout = ctx->d_out[layer], rc = ctx->dom_rc[domain];
    const uint16_t *A = ctx->arenaA + ctx->a_off[layer] + (int64_t)domain * ctx->rc_max * din;
    const uint16_t *B = ctx->arenaB + ctx->b_off[layer] + (int64_t)domain * ctx->rc_max * dout;
    const float scale = gamma * ctx->dom_sc[domain];
    uint16_t *w = static_cast<uint16_t *>(W);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (layout == SALT_W_IN_OUT) CUDA_OR_FAIL(ctx, launch_fold(A, B, w, din, dout, rc, scale, ctx->err_dev, st));
    else CUDA_OR_FAIL(ctx, launch_fold(B, A, w, dout, din, rc, scale, ctx->err_dev, st));
    return SALT_OK;
}

struct salt_fold_plan {
    salt_ctx *ctx = nullptr;
    int32_t domain = 0, rc = 0, n = 0;
    int64_t items = 0;
    void *table = nullptr;  // device: n fold records
};

salt_status salt_fold_plan_create(salt_ctx *ctx, int32_t domain, int32_t n, const int32_t *layers, void *const *W,
                                  int32_t layout, salt_fold_plan **out)
{
    if (!ctx || !out) return SALT_ERR_INVALID_ARG;
    *out = nullptr;
    if (domain < 0 || domain >= ctx->n_domains)
        return fail(ctx, SALT_ERR_DOMAIN_RANGE, "domain %d outside [0, %d)", domain, ctx->n_domains);
    if (ctx->dom_rc[domain] == 0) return fail(ctx, SALT_ERR_DOMAIN_NOT_PINNED, "domain %d has no pinned centroid", domain);
    if (n < 1 || !layers || !W) return fail(ctx, SALT_ERR_INVALID_ARG, "a fold plan needs n >= 1 layers and weights");
    if (layout != SALT_W_IN_OUT && layout != SALT_W_OUT_IN) return fail(ctx, SALT_ERR_INVALID_ARG, "unknown layout %d", layout);
    std::vector<std::pair<uintptr_t, uintptr_t>> spans;
    for (int i = 0; i < n; ++i) {
        const int l = layers[i];
        if (l < 0 || l >= ctx->n_layers) return fail(ctx, SALT_ERR_LAYER_RANGE, "layer %d outside [0, %d)", l, ctx->n_layers);
        if (!W[i]) return fail(ctx, SALT_ERR_INVALID_ARG, "null weight %d", i);
        if (reinterpret_cast<uintptr_t>(W[i]) & 15u) return fail(ctx, SALT_ERR_ALIGN, "weight %d not 16-byte aligned", i);
        const uintptr_t a = reinterpret_cast<uintptr_t>(W[i]);
        spans.push_back({a, a + (uintptr_t)ctx->d_in[l] * ctx->d_out[l] * 2});
    }
    // the weights are updated in place by one launch: none may overlap another
    std::sort(spans.begin(), spans.end());
    for (size_t i = 1; i < spans.size(); ++i)
        if (spans[i].first < spans[i - 1].second) return fail(ctx, SALT_ERR_INVALID_ARG, "weights of a fold plan overlap");
    if (!set_device(ctx)) return fail(ctx, SALT_ERR_CUDA, "cannot select device %d", ctx->device);
    const int rc = ctx->dom_rc[domain];
    const size_t rb = fold_record_bytes();
    std::vector<uint8_t> host((size_t)n * rb);
    int64_t items = 0;
    for (int i = 0; i < n; ++i) {
        const int l = layers[i];
        const int din = ctx->d_in[l], dout = ctx->d_out[l];
        const uint16_t *A = ctx->arenaA + ctx->a_off[l] + (int64_t)domain * ctx->rc_max * din;
        const uint16_t *B = ctx->arenaB + ctx->b_off[l] + (int64_t)domain * ctx->rc_max * dout;
        uint16_t *w = static_cast<uint16_t *>(W[i]);
        int64_t k = 0;
        const cudaError_t e = layout == SALT_W_IN_OUT ? fold_record(host.data() + i * rb, A, B, w, din, dout, rc, items, &k)
                                                      : fold_record(host.data() + i * rb, B, A, w, dout, din, rc, items, &k);
        if (e != cudaSuccess) return fail(ctx, SALT_ERR_CUDA, "fold record %d: %s", i, cudaGetErrorString(e));
        items += k;
    }
    salt_fold_plan *pl = new (std::nothrow) salt_fold_plan;
    if (!pl) return fail(ctx, SALT_ERR_OOM, "fold plan allocation failed");
    if (cudaMalloc(&pl->table, host.size()) != cudaSuccess) {
        delete pl;
        return fail(ctx, SALT_ERR_OOM, "fold plan table allocation failed");
    }
    if (cudaMemcpy(pl->table, host.data(), host.size(), cudaMemcpyHostToDevice) != cudaSuccess) {
        cudaFree(pl->table);
        delete pl;
        return fail(ctx, SALT_ERR_CUDA, "fold plan table copy failed");
    }
    pl->ctx = ctx;
    pl->domain = domain;
    pl->rc = rc;
    pl->n = n;
    pl->items = items;
    *out = pl;
    return SALT_OK;
}

salt_status salt_fold_plan_run(salt_fold_plan *plan, float gamma, salt_stream_t stream)
{
    NvtxRange nvtx_range("salt_fold_plan_run");
    if (!plan || !plan->ctx) return SALT_ERR_INVALID_ARG;
    salt_ctx *ctx = plan->ctx;
    if (ctx->dom_rc[plan->domain] != plan->rc)
        return fail(ctx, SALT_ERR_RANK, "domain %d was re-pinned with rank %d after the plan was made (rank %d)", plan->domain,
                    ctx->dom_rc[plan->domain], plan->rc);
    if (!set_device(ctx)) return fail(ctx, SALT_ERR_CUDA, "cannot select device %d", ctx->device);
    const float scale = gamma * ctx->dom_sc[plan->domain];
    CUDA_OR_FAIL(ctx, launch_fold_table(plan->table, plan->n, plan->items, scale, ctx->err_dev,
                                        static_cast<cudaStream_t>(stream)));
    return SALT_OK;
}

void salt_fold_plan_destroy(salt_fold_plan *plan)
{
    if (!plan) return;
    if (plan->ctx) set_device(plan->ctx);
    if (plan->table) cudaFree(plan->table);
    delete plan;
}

salt_status salt_align_loss(int32_t n, const salt_align_pair *pairs, float eps, float *loss, float *cosine,
                            salt_stream_t stream)
{
    NvtxRange nvtx_range("salt_align_loss");
    return align_loss_run(n, pairs, eps, loss, cosine, static_cast<cudaStream_t>(stream));
}

// float -> bf16, round to nearest even (NaN kept quiet)
static uint16_t host_f32_to_bf16(float f)
{
    uint32_t u;
    std::memcpy(&u, &f, sizeof u);
    if ((u & 0x7fffffffu) > 0x7f800000u) return (uint16_t)((u >> 16) | 0x40u);
    u += 0x7fffu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

static float host_bf16_to_f32(uint16_t h)
{
    uint32_t u = (uint32_t)h << 16;
    float f;
    std::memcpy(&f, &u, sizeof f);
    return f;
}

salt_status salt_residual_blob_concat(const salt_config *config, int32_t rc, const void *At_c, const void *B_c,
                                      float s_c, int32_t rank, const void *At_u, const void *B_u, float s_u,
                                      void *blob, int64_t blob_bytes)
{
    if (rc < 1 || rank < 1) return SALT_ERR_RANK;
    const int32_t R = rc + rank;
    int64_t need = salt_residual_blob_bytes(config, R);
    if (need < 0 || !At_c || !B_c || !At_u || !B_u || !blob) return SALT_ERR_INVALID_ARG;
    if (R > SALT_MAX_RESIDUAL_RANK) return SALT_ERR_RANK;
    if (blob_bytes < need) return SALT_ERR_INVALID_ARG;
    const float s = s_u != 0.f ? s_u : 1.f;
    const float fc = s_c / s, fu = s_u != 0.f ? 1.f : 0.f;
    salt_blob_header h;
    std::memset(&h, 0, sizeof h);
    h.magic = SALT_BLOB_MAGIC;
    h.version = 1;
    h.rank = R;
    h.n_layers = config->n_layers;
    h.s_u = s;
    h.payload_bytes = (uint64_t)payload_elems(config, R) * 2;
    h.layout_hash = fnv1a_layout(config->n_layers, config->d_in, config->d_out);
    uint8_t *out = static_cast<uint8_t *>(blob);
    std::memcpy(out, &h, sizeof h);
    uint16_t *pay = reinterpret_cast<uint16_t *>(out + SALT_BLOB_HEADER_BYTES);
    const uint16_t *Ac = static_cast<const uint16_t *>(At_c), *Bc = static_cast<const uint16_t *>(B_c);
    const uint16_t *Au = static_cast<const uint16_t *>(At_u), *Bu = static_cast<const uint16_t *>(B_u);
    auto scaled = [](const uint16_t *src, int64_t n, float f, uint16_t *dst) {
        if (f == 1.f) {
            std::memcpy(dst, src, (size_t)n * 2);
            return;
        }
        for (int64_t i = 0; i < n; ++i) dst[i] = host_f32_to_bf16(f * host_bf16_to_f32(src[i]));
    };
    int64_t oc_a = 0, oc_b = 0, ou_a = 0, ou_b = 0, op = 0;
    for (int l = 0; l < config->n_layers; ++l) {
        const int64_t di = config->d_in[l], dout = config->d_out[l];
        std::memcpy(pay + op, Ac + oc_a, (size_t)(rc * di) * 2);
        std::memcpy(pay + op + rc * di, Au + ou_a, (size_t)(rank * di) * 2);
        op += R * di;
        scaled(Bc + oc_b, rc * dout, fc, pay + op);
        scaled(Bu + ou_b, rank * dout, fu, pay + op + rc * dout);
        op += R * dout;
        oc_a += rc * di;
        ou_a += rank * di;
        oc_b += rc * dout;
        ou_b += rank * dout;
    }
    return SALT_OK;
}

salt_status salt_residual_load(salt_ctx *ctx, int32_t slot, const void *host_blob, salt_stream_t side_stream)
{
    NvtxRange nvtx_range("salt_residual_load");
    if (!ctx) return SALT_ERR_INVALID_ARG;
    int32_t rank = 0;
    uint64_t bytes = 0;
    salt_status st = check_blob(ctx, slot, host_blob, &rank, &bytes);
    if (st != SALT_OK) return st;
    if (!set_device(ctx)) return fail(ctx, SALT_ERR_CUDA, "cannot select device %d", ctx->device);
    return enqueue_loads(ctx, 1, &slot, &host_blob, &rank, &bytes, static_cast<cudaStream_t>(side_stream));
}

salt_status salt_residual_load_batch(salt_ctx *ctx, int32_t n, const int32_t *slots, const void *const *host_blobs,
                                     salt_stream_t side_stream)
{
    NvtxRange nvtx_range("salt_residual_load_batch");
    if (!ctx) return SALT_ERR_INVALID_ARG;
    if (n < 0 || (n > 0 && (!slots || !host_blobs))) return fail(ctx, SALT_ERR_INVALID_ARG, "bad batch of %d loads", n);
    if (n == 0) return SALT_OK;
    std::vector<int32_t> ranks(n);
    std::vector<uint64_t> bytes(n);
    for (int32_t i = 0; i < n; ++i) {
        salt_status st = check_blob(ctx, slots[i], host_blobs[i], &ranks[i], &bytes[i]);
        if (st != SALT_OK) return st;
    }
    if (!set_device(ctx)) return fail(ctx, SALT_ERR_CUDA, "cannot select device %d", ctx->device);
    return enqueue_loads(ctx, n, slots, host_blobs, ranks.data(), bytes.data(), static_cast<cudaStream_t>(side_stream));
}

salt_status salt_segments_create(salt_ctx *ctx, salt_segments **out)
{
    if (!ctx || !out) return SALT_ERR_INVALID_ARG;
    *out = nullptr;
    if (!set_device(ctx)) return fail(ctx, SALT_ERR_CUDA, "cannot select device %d", ctx->device);
    salt_segments *seg = new (std::nothrow) salt_segments;
    if (!seg) return SALT_ERR_OOM;
    seg->ctx = ctx;
    const int n = ctx->max_tokens;
    auto alloc = [&](int32_t **p, size_t count) { return cudaMalloc(p, count * sizeof(int32_t)) == cudaSuccess; };
    bool ok = alloc(&seg->d.ids, 3 * (size_t)n) && alloc(&seg->d.perm, n) && alloc(&seg->d.sorted_slot, n) &&
              alloc(&seg->d.dseg_ptr, n + 1) && alloc(&seg->d.dseg_dom, n) && alloc(&seg->d.dseg_gbin, n) &&
              alloc(&seg->d.useg_ptr, n + 1) && alloc(&seg->d.useg_dom, n) && alloc(&seg->d.useg_gbin, n) &&
              alloc(&seg->d.useg_slot, n) &&
              alloc(&seg->d.blk, (size_t)BLK_INTS * n) && alloc(&seg->d.counts, 4) && alloc(&seg->d.tok_uoff, n) &&
              alloc(&seg->d.tok_urank, n) && alloc(reinterpret_cast<int32_t **>(&seg->d.tok_su), n) &&
              alloc(reinterpret_cast<int32_t **>(&seg->d.tok_sc), n) &&
              alloc(&seg->d.blk_res, (size_t)n * S_MAX) && alloc(&seg->d.aperm, n) && alloc(&seg->d.a_dptr, n + 1) &&
              alloc(&seg->d.a_ddom, n) && alloc(&seg->d.a_uptr, n + 1) && alloc(&seg->d.a_udom, n);
    seg->work.blk_cap = block_bound_loose(ctx, n);
    seg->work.max_group = SALT_MAX_GROUP;
    seg->work.part_cap = PART_CAP;
    const size_t n_pairs = (size_t)SALT_MAX_GROUP * seg->work.blk_cap;
    ok = ok && guarded_malloc(reinterpret_cast<void **>(&seg->work.vext), n_pairs * TM * VEXT_COLS * 2) == cudaSuccess &&
         guarded_malloc(reinterpret_cast<void **>(&seg->work.part), (size_t)PART_CAP * TM * PART_COLS * sizeof(float)) ==
             cudaSuccess &&
         cudaMalloc(&seg->work.arrive, 2 * n_pairs * sizeof(uint32_t)) == cudaSuccess &&
         cudaMalloc(&seg->work.vdone, 2 * n_pairs * sizeof(uint32_t)) == cudaSuccess &&
         cudaMalloc(&seg->work.seq, 2 * sizeof(uint32_t)) == cudaSuccess &&
         cudaMemset(seg->work.arrive, 0, 2 * n_pairs * sizeof(uint32_t)) == cudaSuccess &&
         cudaMemset(seg->work.vdone, 0, 2 * n_pairs * sizeof(uint32_t)) == cudaSuccess &&
         cudaMemset(seg->work.seq, 0, 2 * sizeof(uint32_t)) == cudaSuccess &&
         apply_encode_vmap(seg->work) == cudaSuccess;
    for (int i = 0; ok && i < 2; ++i) {
        ok = cudaHostAlloc(&seg->staging[i], 3 * (size_t)n * sizeof(int32_t), cudaHostAllocDefault) == cudaSuccess &&
             cudaEventCreateWithFlags(&seg->staging_ev[i], cudaEventDisableTiming) == cudaSuccess;
    }
    ok = ok && cudaEventCreateWithFlags(&seg->built_ev, cudaEventDisableTiming) == cudaSuccess &&
         cudaEventCreateWithFlags(&seg->tmp_ev, cudaEventDisableTiming) == cudaSuccess;
    ok = ok && cudaMemset(seg->d.counts, 0, 4 * sizeof(int32_t)) == cudaSuccess;
    if (!ok) {
        cudaGetLastError();
        ctx->segs.insert(seg);
        salt_segments_destroy(seg);
        return fail(ctx, SALT_ERR_OOM, "segments allocation failed");
    }
    seg->refs.assign(ctx->n_slots > 0 ? ctx->n_slots : 1, 0);
    ctx->segs.insert(seg);
    *out = seg;
    return SALT_OK;
}

void salt_segments_destroy(salt_segments *seg)
{
    if (!seg) return;
    salt_ctx *ctx = seg->ctx;
    if (ctx) set_device(ctx);
    for (cudaStream_t s : seg->use_streams) cudaStreamSynchronize(s);
    for (int i = 0; i < 2; ++i)
        if (seg->staging_ev[i]) cudaEventSynchronize(seg->staging_ev[i]);
    int32_t *arrs[] = {seg->d.ids, seg->d.perm, seg->d.sorted_slot, seg->d.dseg_ptr, seg->d.dseg_dom,
                       seg->d.dseg_gbin, seg->d.useg_ptr, seg->d.useg_dom, seg->d.useg_gbin,
                       seg->d.useg_slot, seg->d.blk, seg->d.counts,
                       seg->d.tok_uoff, seg->d.tok_urank, reinterpret_cast<int32_t *>(seg->d.tok_su),
                       reinterpret_cast<int32_t *>(seg->d.tok_sc),
                       seg->d.blk_res, seg->d.aperm, seg->d.a_dptr, seg->d.a_ddom, seg->d.a_uptr, seg->d.a_udom};
    for (int32_t *p : arrs) cudaFree(p);
    guarded_free(seg->work.vext);
    guarded_free(seg->work.part);
    cudaFree(seg->work.arrive);
    cudaFree(seg->work.vdone);
    cudaFree(seg->work.seq);
    for (int i = 0; i < 2; ++i) {
        if (seg->staging[i]) cudaFreeHost(seg->staging[i]);
        if (seg->staging_ev[i]) cudaEventDestroy(seg->staging_ev[i]);
    }
    if (seg->built_ev) cudaEventDestroy(seg->built_ev);
    if (seg->tmp_ev) cudaEventDestroy(seg->tmp_ev);
    cudaGetLastError();
    if (ctx) ctx->segs.erase(seg);
    delete seg;
}

salt_status salt_build_segments(salt_ctx *ctx, salt_segments *seg, const int32_t *domain_ids,
                                const int32_t *slot_ids, int32_t n_tokens, salt_stream_t stream)
{
    return salt_build_segments_gamma(ctx, seg, domain_ids, nullptr, slot_ids, n_tokens, 0, nullptr, stream);
}

salt_status salt_build_segments_gamma(salt_ctx *ctx, salt_segments *seg, const int32_t *domain_ids,
                                      const int32_t *gamma_bins, const int32_t *slot_ids, int32_t n_tokens,
                                      int32_t n_gamma, const float *gamma, salt_stream_t stream_)
{
    NvtxRange nvtx_range("salt_build_segments");
    if (!ctx || !seg || seg->ctx != ctx) return SALT_ERR_INVALID_ARG;
    if (n_tokens < 0) return fail(ctx, SALT_ERR_INVALID_ARG, "negative token count");
    if (n_tokens > ctx->max_tokens)
        return fail(ctx, SALT_ERR_TOO_MANY_TOKENS, "%d tokens > max_tokens %d", n_tokens, ctx->max_tokens);
    if (n_tokens > 0 && (!domain_ids || !slot_ids)) return fail(ctx, SALT_ERR_INVALID_ARG, "null id array");
    if (n_gamma < 0 || n_gamma > SALT_MAX_GAMMA_BINS)
        return fail(ctx, SALT_ERR_INVALID_ARG, "%d gamma bins outside [0, %d]", n_gamma, SALT_MAX_GAMMA_BINS);
    if (n_gamma > 0 && !gamma) return fail(ctx, SALT_ERR_INVALID_ARG, "null gamma table");
    if (!set_device(ctx)) return fail(ctx, SALT_ERR_CUDA, "cannot select device %d", ctx->device);
    cudaStream_t stream = static_cast<cudaStream_t>(stream_);
    const int T = n_tokens;
    const bool has_gbin = gamma_bins != nullptr;
    bool dev_ids = T > 0 && is_device_pointer(domain_ids);
    if (T > 0 && (dev_ids != is_device_pointer(slot_ids) || (has_gbin && dev_ids != is_device_pointer(gamma_bins))))
        return fail(ctx, SALT_ERR_INVALID_ARG, "the id arrays must all be host or all be device memory");

    std::vector<uint8_t> refs;
    if (!dev_ids) {
        refs.assign(seg->refs.size(), 0);
        for (int t = 0; t < T; ++t) {
            int d = domain_ids[t], s = slot_ids[t];
            if (d < -1 || d >= ctx->n_domains)
                return fail(ctx, SALT_ERR_DOMAIN_RANGE, "token %d: domain %d outside [-1, %d)", t, d, ctx->n_domains);
            if (d >= 0 && ctx->dom_rc[d] == 0)
                return fail(ctx, SALT_ERR_DOMAIN_NOT_PINNED, "token %d: domain %d has no pinned centroid", t, d);
            if (s < -1 || s >= ctx->n_slots)
                return fail(ctx, SALT_ERR_SLOT_RANGE, "token %d: slot %d outside [-1, %d)", t, s, ctx->n_slots);
            if (s >= 0) {
                if (ctx->slot_rank[s] == 0)
                    return fail(ctx, SALT_ERR_SLOT_EMPTY, "token %d: slot %d was never loaded", t, s);
                refs[s] = 1;
            }
            if (has_gbin && d >= 0 && (gamma_bins[t] < -1 || gamma_bins[t] >= n_gamma))
                return fail(ctx, SALT_ERR_GAMMA_RANGE, "token %d: gamma bin %d outside [-1, %d)", t, gamma_bins[t],
                            n_gamma);
        }
    }
    // The device buffers of seg may still be read by earlier uses on other streams.
    CUDA_OR_FAIL(ctx, wait_for_uses(seg, stream));
    // Swaps of the slots this batch reads must land first.
    for (int s = 0; s < ctx->n_slots; ++s) {
        if (!(dev_ids ? true : refs[s])) continue;
        if (ctx->slot_seq[s] == 0) continue;
        if (ctx->slot_waited_seq[s] == ctx->slot_seq[s] && ctx->slot_waited_stream[s] == stream) continue;
        CUDA_OR_FAIL(ctx, cudaStreamWaitEvent(stream, ctx->slot_ready[s], 0));
        ctx->slot_waited_seq[s] = ctx->slot_seq[s];
        ctx->slot_waited_stream[s] = stream;
    }
    if (T > 0) {
        const int32_t *src[3] = {domain_ids, slot_ids, gamma_bins};
        const int n_arr = has_gbin ? 3 : 2;
        if (dev_ids) {
            for (int a = 0; a < n_arr; ++a)
                CUDA_OR_FAIL(ctx, cudaMemcpyAsync(seg->d.ids + (size_t)a * ctx->max_tokens, src[a], (size_t)T * 4,
                                                  cudaMemcpyDeviceToDevice, stream));
        } else {
            int k = seg->staging_next;
            seg->staging_next ^= 1;
            if (seg->staging_used[k]) CUDA_OR_FAIL(ctx, cudaEventSynchronize(seg->staging_ev[k]));
            int32_t *h = seg->staging[k];
            for (int a = 0; a < n_arr; ++a) {
                std::memcpy(h + (size_t)a * ctx->max_tokens, src[a], (size_t)T * 4);
                CUDA_OR_FAIL(ctx, cudaMemcpyAsync(seg->d.ids + (size_t)a * ctx->max_tokens,
                                                  h + (size_t)a * ctx->max_tokens, (size_t)T * 4,
                                                  cudaMemcpyHostToDevice, stream));
            }
            CUDA_OR_FAIL(ctx, cudaEventRecord(seg->staging_ev[k], stream));
            seg->staging_used[k] = true;
        }
    }
    SegParams p;
    p.s = seg->d;
    p.T = T;
    p.max_tokens = ctx->max_tokens;
    p.n_domains = ctx->n_domains;
    p.n_slots = ctx->n_slots;
    p.r_max = ctx->r_max;
    p.umax = ctx->umax;
    p.dom_rc = ctx->dom_rc_dev;
    p.dom_sc = ctx->dom_sc_dev;
    p.has_gbin = has_gbin ? 1 : 0;
    p.n_gamma = n_gamma;
    for (int g = 0; g < SALT_MAX_GAMMA_BINS; ++g) p.gamma[g] = g < n_gamma ? gamma[g] : 1.f;
    p.pool = ctx->pool;
    p.slot_stride = ctx->slot_stride;
    p.err = ctx->err_dev;
    CUDA_OR_FAIL(ctx, launch_segments(p, stream));
    CUDA_OR_FAIL(ctx, cudaEventRecord(seg->built_ev, stream));

    seg->built = true;
    seg->tables_fresh = true;
    seg->stale = false;
    seg->device_ids = dev_ids;
    seg->T = T;
    if (dev_ids) std::fill(seg->refs.begin(), seg->refs.end(), 1);
    else seg->refs.swap(refs);
    if (T == 0) seg->n_blk_bound = 0;
    else if (dev_ids) seg->n_blk_bound = std::min(block_bound_loose(ctx, T), seg->work.blk_cap);
    else seg->n_blk_bound = std::min(block_bound_host(ctx, domain_ids, gamma_bins, slot_ids, T), seg->work.blk_cap);
    seg->build_stream = stream;
    seg->use_streams.clear();
    seg->use_streams.push_back(stream);
    return SALT_OK;
}

salt_status salt_segments_export(salt_ctx *ctx, const salt_segments *seg, int32_t *counts, int32_t *perm,
                                 int32_t *dseg_ptr, int32_t *dseg_dom, int32_t *useg_ptr, int32_t *useg_dom,
                                 int32_t *useg_slot, int32_t *blocks)
{
    if (!ctx || !seg || seg->ctx != ctx || !counts) return SALT_ERR_INVALID_ARG;
    if (!seg->built) return fail(ctx, SALT_ERR_NOT_BUILT, "segments object was never built");
    if (!set_device(ctx)) return fail(ctx, SALT_ERR_CUDA, "cannot select device %d", ctx->device);
    CUDA_OR_FAIL(ctx, cudaEventSynchronize(seg->built_ev));
    CUDA_OR_FAIL(ctx, cudaMemcpy(counts, seg->d.counts, 4 * sizeof(int32_t), cudaMemcpyDeviceToHost));
    const int T = counts[0], nd = counts[1], nu = counts[2], nb = counts[3];
    auto cp = [&](int32_t *dst, const int32_t *src, int n) -> cudaError_t {
        if (!dst || n <= 0) return cudaSuccess;
        return cudaMemcpy(dst, src, (size_t)n * sizeof(int32_t), cudaMemcpyDeviceToHost);
    };
    CUDA_OR_FAIL(ctx, cp(perm, seg->d.perm, T));
    CUDA_OR_FAIL(ctx, cp(dseg_ptr, seg->d.dseg_ptr, nd + 1));
    CUDA_OR_FAIL(ctx, cp(dseg_dom, seg->d.dseg_dom, nd));
    CUDA_OR_FAIL(ctx, cp(useg_ptr, seg->d.useg_ptr, nu + 1));
    CUDA_OR_FAIL(ctx, cp(useg_dom, seg->d.useg_dom, nu));
    CUDA_OR_FAIL(ctx, cp(useg_slot, seg->d.useg_slot, nu));
    if (blocks && nb > 0) {
        std::vector<int32_t> rec((size_t)BLK_INTS * nb);
        CUDA_OR_FAIL(ctx, cp(rec.data(), seg->d.blk, BLK_INTS * nb));
        for (int b = 0; b < nb; ++b) {
            blocks[3 * b + 0] = rec[(size_t)BLK_INTS * b + BLK_START];
            blocks[3 * b + 1] = rec[(size_t)BLK_INTS * b + BLK_LEN];
            blocks[3 * b + 2] = rec[(size_t)BLK_INTS * b + BLK_DOM];
        }
    }
    return SALT_OK;
}

salt_status salt_segments_export_gamma(salt_ctx *ctx, const salt_segments *seg, int32_t *dseg_gbin,
                                       int32_t *useg_gbin)
{
    if (!ctx || !seg || seg->ctx != ctx) return SALT_ERR_INVALID_ARG;
    if (!seg->built) return fail(ctx, SALT_ERR_NOT_BUILT, "segments object was never built");
    if (!set_device(ctx)) return fail(ctx, SALT_ERR_CUDA, "cannot select device %d", ctx->device);
    CUDA_OR_FAIL(ctx, cudaEventSynchronize(seg->built_ev));
    int32_t counts[4];
    CUDA_OR_FAIL(ctx, cudaMemcpy(counts, seg->d.counts, sizeof counts, cudaMemcpyDeviceToHost));
    if (dseg_gbin && counts[1] > 0)
        CUDA_OR_FAIL(ctx, cudaMemcpy(dseg_gbin, seg->d.dseg_gbin, (size_t)counts[1] * 4, cudaMemcpyDeviceToHost));
    if (useg_gbin && counts[2] > 0)
        CUDA_OR_FAIL(ctx, cudaMemcpy(useg_gbin, seg->d.useg_gbin, (size_t)counts[2] * 4, cudaMemcpyDeviceToHost));
    return SALT_OK;
}

}  // extern "C"

namespace {
// The grouped apply; with shrink_only the launch only writes the row blocks'
// V tiles into the segments workspace (y is not touched and may be null).
salt_status apply_grouped(salt_ctx *ctx, const salt_segments *seg_, int32_t n, const int32_t *layers,
                          const void *const *x, void *const *y, salt_stream_t stream_, bool shrink_only)
{
    NvtxRange nvtx_range("salt_lora_apply");
    if (!ctx || !seg_ || seg_->ctx != ctx) return SALT_ERR_INVALID_ARG;
    salt_segments *seg = const_cast<salt_segments *>(seg_);
    if (n < 1 || n > SALT_MAX_GROUP || !layers || !x || !y)
        return fail(ctx, SALT_ERR_INVALID_ARG, "group size %d outside [1, %d] or null arrays", n, SALT_MAX_GROUP);
    if (!seg->built) return fail(ctx, SALT_ERR_NOT_BUILT, "segments object was never built");
    if (seg->stale) return fail(ctx, SALT_ERR_STALE_SEGMENTS, "a slot named by the segments was reloaded; rebuild");
    ApplyParams p;
    std::memset(&p, 0, sizeof p);
    for (int i = 0; i < n; ++i) {
        int l = layers[i];
        if (l < 0 || l >= ctx->n_layers)
            return fail(ctx, SALT_ERR_LAYER_RANGE, "layer %d outside [0, %d)", l, ctx->n_layers);
        if (seg->T > 0 && (!x[i] || (!y[i] && !shrink_only))) return fail(ctx, SALT_ERR_INVALID_ARG, "null x or y");
        if ((reinterpret_cast<uintptr_t>(x[i]) | reinterpret_cast<uintptr_t>(y[i])) & 15)
            return fail(ctx, SALT_ERR_ALIGN, "x / y of group entry %d not 16-byte aligned", i);
        ApplyProj &pr = p.proj[i];
        pr.x = static_cast<const uint16_t *>(x[i]);
        pr.y = static_cast<uint16_t *>(y[i]);
        pr.A = ctx->arenaA ? ctx->arenaA + ctx->a_off[l] : nullptr;
        pr.B = ctx->arenaB ? ctx->arenaB + ctx->b_off[l] : nullptr;
        pr.res_off = ctx->res_off[l];
        pr.d_in = ctx->d_in[l];
        pr.d_out = ctx->d_out[l];
    }
    if (seg->T == 0) return SALT_OK;
    if (!set_device(ctx)) return fail(ctx, SALT_ERR_CUDA, "cannot select device %d", ctx->device);
    cudaStream_t stream = static_cast<cudaStream_t>(stream_);
    // The segments object's V workspace is shared by its applies: applies on
    // different streams are serialised (no-op for the usual single stream).
    if (seg->use_streams.size() > 1 || (seg->use_streams.size() == 1 && seg->use_streams[0] != stream))
        CUDA_OR_FAIL(ctx, wait_for_uses(seg, stream));
    add_stream(seg->use_streams, stream);
    p.n_proj = n;
    int units = 0;
    for (int i = 0; i < n; ++i) {
        p.n_unit_prefix[i] = units;
        units += (p.proj[i].d_out + 63) / 64;
    }
    p.n_unit_prefix[n] = units;
    p.min_nk = 1 << 30;
    for (int i = 0; i < n; ++i) p.min_nk = std::min(p.min_nk, (p.proj[i].d_in + 63) / 64);
    p.perm = seg->d.aperm;
    p.blk = seg->d.blk;
    p.counts = seg->d.counts;
    p.tok_uoff = seg->d.tok_uoff;
    p.tok_urank = seg->d.tok_urank;
    p.tok_su = seg->d.tok_su;
    p.tok_sc = seg->d.tok_sc;
    p.blk_res = seg->d.blk_res;
    p.rc_max = ctx->rc_max;
    p.pool = ctx->pool;
    p.slot_stride = ctx->slot_stride;
    p.w = seg->work;
    p.err = ctx->err_dev;
    p.shrink_only = shrink_only ? 1 : 0;
    // The first apply after a build waits for the segment kernel in full;
    // later ones overlap their table reads with the previous kernel.
    CUDA_OR_FAIL(ctx, launch_apply(p, !seg->tables_fresh, stream));
    seg->tables_fresh = false;
    return SALT_OK;
}
}  // namespace

extern "C" {

salt_status salt_lora_apply_grouped(salt_ctx *ctx, const salt_segments *seg, int32_t n, const int32_t *layers,
                                    const void *const *x, void *const *y, salt_stream_t stream)
{
    return apply_grouped(ctx, seg, n, layers, x, y, stream, false);
}

salt_status salt_lora_apply_with_base(salt_ctx *ctx, const salt_segments *seg_, int32_t layer, const void *x,
                                      const void *W, int32_t layout, void *y, salt_stream_t stream_)
{
    NvtxRange nvtx_range("salt_lora_apply_with_base");
    if (!ctx || !seg_ || seg_->ctx != ctx) return SALT_ERR_INVALID_ARG;
    salt_segments *seg = const_cast<salt_segments *>(seg_);
    if (layer < 0 || layer >= ctx->n_layers)
        return fail(ctx, SALT_ERR_LAYER_RANGE, "layer %d outside [0, %d)", layer, ctx->n_layers);
    if (layout != SALT_W_IN_OUT && layout != SALT_W_OUT_IN) return fail(ctx, SALT_ERR_INVALID_ARG, "unknown layout %d", layout);
    if (!seg->built) return fail(ctx, SALT_ERR_NOT_BUILT, "segments object was never built");
    if (seg->stale) return fail(ctx, SALT_ERR_STALE_SEGMENTS, "a slot named by the segments was reloaded; rebuild");
    if (seg->T > 0 && (!x || !W || !y)) return fail(ctx, SALT_ERR_INVALID_ARG, "null x, W or y");
    if ((reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(y) | reinterpret_cast<uintptr_t>(W)) & 15)
        return fail(ctx, SALT_ERR_ALIGN, "x, W or y not 16-byte aligned");
    if (seg->T == 0) return SALT_OK;
    // 1. the row blocks' V tiles (shrink only)
    const void *xs[1] = {x};
    void *ys[1] = {nullptr};
    salt_status st = apply_grouped(ctx, seg, 1, &layer, xs, ys, stream_, true);
    if (st != SALT_OK) return st;
    // 2. the base GEMM with the delta of every overlapping row block
    BaseParams bp;
    std::memset(&bp, 0, sizeof bp);
    const int din = ctx->d_in[layer], dout = ctx->d_out[layer];
    CUDA_OR_FAIL(ctx, encode_base_map(&bp.wmap, static_cast<const uint16_t *>(W), din, dout, layout));
    bp.x = static_cast<const uint16_t *>(x);
    bp.y = static_cast<uint16_t *>(y);
    bp.perm = seg->d.aperm;
    bp.blk = seg->d.blk;
    bp.counts = seg->d.counts;
    bp.blk_res = seg->d.blk_res;
    bp.vext = seg->work.vext;
    bp.B = ctx->arenaB ? ctx->arenaB + ctx->b_off[layer] : nullptr;
    bp.pool = ctx->pool;
    bp.slot_stride = ctx->slot_stride;
    bp.res_off = ctx->res_off[layer];
    bp.T = seg->T;
    bp.d_in = din;
    bp.d_out = dout;
    bp.rc_max = ctx->rc_max;
    bp.w_layout = layout;
    bp.blk_cap = seg->work.blk_cap;
    bp.err = ctx->err_dev;
    CUDA_OR_FAIL(ctx, launch_base(bp, static_cast<cudaStream_t>(stream_)));
    return SALT_OK;
}

salt_status salt_lora_apply(salt_ctx *ctx, const salt_segments *seg, int32_t layer, const void *x, void *y,
                            salt_stream_t stream)
{
    const void *xs[1] = {x};
    void *ys[1] = {y};
    return salt_lora_apply_grouped(ctx, seg, 1, &layer, xs, ys, stream);
}

// Allocation-free variant of salt_lora_apply: the V tiles between the two
// kernels live in a static device array of this library instead of the
// segments object's workspace.  See include/salt.h for the contract.
salt_status salt_lora_apply_static(salt_ctx *ctx, const salt_segments *seg_, int32_t layer, const void *x, void *y,
                                   salt_stream_t stream_)
{
    if (!ctx || !seg_ || seg_->ctx != ctx) return SALT_ERR_INVALID_ARG;
    salt_segments *seg = const_cast<salt_segments *>(seg_);
    if (!seg->built) return fail(ctx, SALT_ERR_NOT_BUILT, "segments object was never built");
    if (seg->stale) return fail(ctx, SALT_ERR_STALE_SEGMENTS, "a slot named by the segments was reloaded; rebuild");
    if (layer < 0 || layer >= ctx->n_layers)
        return fail(ctx, SALT_ERR_LAYER_RANGE, "layer %d outside [0, %d)", layer, ctx->n_layers);
    if (seg->T > 0 && (!x || !y)) return fail(ctx, SALT_ERR_INVALID_ARG, "null x or y");
    if ((reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(y)) & 15)
        return fail(ctx, SALT_ERR_ALIGN, "x / y not 16-byte aligned");
    if (seg->n_blk_bound > STATIC_APPLY_BLOCKS)
        return fail(ctx, SALT_ERR_TOO_MANY_TOKENS,
                    "batch may need %d row blocks; the static scratch of salt_lora_apply_static holds %d",
                    seg->n_blk_bound, STATIC_APPLY_BLOCKS);
    if (seg->T == 0) return SALT_OK;
    if (!set_device(ctx)) return fail(ctx, SALT_ERR_CUDA, "cannot select device %d", ctx->device);
    ApplyWork scratch;
    CUDA_OR_FAIL(ctx, apply_static_workspace(&scratch));
    cudaStream_t stream = static_cast<cudaStream_t>(stream_);
    if (seg->use_streams.size() > 1 || (seg->use_streams.size() == 1 && seg->use_streams[0] != stream))
        CUDA_OR_FAIL(ctx, wait_for_uses(seg, stream));
    add_stream(seg->use_streams, stream);
    ApplyParams p;
    std::memset(&p, 0, sizeof p);
    ApplyProj &pr = p.proj[0];
    pr.x = static_cast<const uint16_t *>(x);
    pr.y = static_cast<uint16_t *>(y);
    pr.A = ctx->arenaA ? ctx->arenaA + ctx->a_off[layer] : nullptr;
    pr.B = ctx->arenaB ? ctx->arenaB + ctx->b_off[layer] : nullptr;
    pr.res_off = ctx->res_off[layer];
    pr.d_in = ctx->d_in[layer];
    pr.d_out = ctx->d_out[layer];
    p.n_proj = 1;
    p.n_unit_prefix[0] = 0;
    p.n_unit_prefix[1] = (pr.d_out + 63) / 64;
    p.min_nk = (pr.d_in + 63) / 64;
    p.perm = seg->d.aperm;
    p.blk = seg->d.blk;
    p.counts = seg->d.counts;
    p.tok_uoff = seg->d.tok_uoff;
    p.tok_urank = seg->d.tok_urank;
    p.tok_su = seg->d.tok_su;
    p.tok_sc = seg->d.tok_sc;
    p.blk_res = seg->d.blk_res;
    p.rc_max = ctx->rc_max;
    p.pool = ctx->pool;
    p.slot_stride = ctx->slot_stride;
    p.w = scratch;
    p.err = ctx->err_dev;
    CUDA_OR_FAIL(ctx, launch_apply(p, !seg->tables_fresh, stream));
    seg->tables_fresh = false;
    return SALT_OK;
}

salt_status salt_host_pipe_create(salt_ctx *ctx, int32_t n_stages, int64_t stage_bytes, salt_host_pipe **out)
{
    if (!ctx || !out) return SALT_ERR_INVALID_ARG;
    *out = nullptr;
    if (n_stages == 0) n_stages = 3;
    if (n_stages < 2 || n_stages > 8) return fail(ctx, SALT_ERR_INVALID_ARG, "%d stages outside [2, 8]", n_stages);
    if (stage_bytes < 0) return fail(ctx, SALT_ERR_INVALID_ARG, "negative stage size");
    if (!set_device(ctx)) return fail(ctx, SALT_ERR_CUDA, "cannot select device %d", ctx->device);
    if (stage_bytes == 0) {
        // the SALT_MAX_GROUP largest layers of the table, x and y, at max_tokens
        std::vector<int64_t> per;
        for (int l = 0; l < ctx->n_layers; ++l) {
            const int64_t a = ((int64_t)ctx->max_tokens * ctx->d_in[l] * 2 + 255) / 256 * 256;
            const int64_t b = ((int64_t)ctx->max_tokens * ctx->d_out[l] * 2 + 255) / 256 * 256;
            per.push_back(a + b);
        }
        std::sort(per.begin(), per.end(), std::greater<int64_t>());
        for (size_t i = 0; i < per.size() && i < (size_t)SALT_MAX_GROUP; ++i) stage_bytes += per[i];
    }
    salt_host_pipe *pp = new (std::nothrow) salt_host_pipe;
    if (!pp) return SALT_ERR_OOM;
    pp->ctx = ctx;
    pp->n_stages = n_stages;
    pp->stage_bytes = (stage_bytes + 255) / 256 * 256;
    pp->stage.assign(n_stages, nullptr);
    pp->in_ready.assign(n_stages, nullptr);
    pp->applied.assign(n_stages, nullptr);
    pp->out_done.assign(n_stages, nullptr);
    pp->used.assign(n_stages, 0);
    bool ok = cudaStreamCreateWithFlags(&pp->h2d, cudaStreamNonBlocking) == cudaSuccess &&
              cudaStreamCreateWithFlags(&pp->d2h, cudaStreamNonBlocking) == cudaSuccess;
    for (int k = 0; ok && k < n_stages; ++k) {
        ok = cudaMalloc(&pp->stage[k], (size_t)pp->stage_bytes) == cudaSuccess &&
             cudaEventCreateWithFlags(&pp->in_ready[k], cudaEventDisableTiming) == cudaSuccess &&
             cudaEventCreateWithFlags(&pp->applied[k], cudaEventDisableTiming) == cudaSuccess &&
             cudaEventCreateWithFlags(&pp->out_done[k], cudaEventDisableTiming) == cudaSuccess;
    }
    if (!ok) {
        cudaGetLastError();
        salt_host_pipe_destroy(pp);
        return fail(ctx, SALT_ERR_OOM, "host pipe allocation failed (%d stages of %lld bytes)", n_stages,
                    (long long)pp->stage_bytes);
    }
    *out = pp;
    return SALT_OK;
}

void salt_host_pipe_destroy(salt_host_pipe *pipe)
{
    if (!pipe) return;
    if (pipe->ctx) set_device(pipe->ctx);
    if (pipe->h2d) cudaStreamSynchronize(pipe->h2d);
    if (pipe->d2h) cudaStreamSynchronize(pipe->d2h);
    for (int k = 0; k < pipe->n_stages; ++k) {
        if (pipe->out_done[k]) cudaEventSynchronize(pipe->out_done[k]);
        cudaFree(pipe->stage[k]);
        for (cudaEvent_t e : {pipe->in_ready[k], pipe->applied[k], pipe->out_done[k]})
            if (e) cudaEventDestroy(e);
    }
    if (pipe->h2d) cudaStreamDestroy(pipe->h2d);
    if (pipe->d2h) cudaStreamDestroy(pipe->d2h);
    cudaGetLastError();
    delete pipe;
}

salt_status salt_lora_apply_host(salt_host_pipe *pipe, const salt_segments *seg, int32_t n, const int32_t *layers,
                                 const void *const *x_host, void *const *y_host, salt_stream_t stream_)
{
    NvtxRange nvtx_range("salt_lora_apply_host");
    if (!pipe || !pipe->ctx) return SALT_ERR_INVALID_ARG;
    salt_ctx *ctx = pipe->ctx;
    if (!seg || seg->ctx != ctx) return fail(ctx, SALT_ERR_INVALID_ARG, "segments of another context");
    if (n < 1 || n > SALT_MAX_GROUP || !layers || !x_host || !y_host)
        return fail(ctx, SALT_ERR_INVALID_ARG, "group size %d outside [1, %d] or null arrays", n, SALT_MAX_GROUP);
    if (!seg->built) return fail(ctx, SALT_ERR_NOT_BUILT, "segments object was never built");
    if (seg->stale) return fail(ctx, SALT_ERR_STALE_SEGMENTS, "a slot named by the segments was reloaded; rebuild");
    if (!set_device(ctx)) return fail(ctx, SALT_ERR_CUDA, "cannot select device %d", ctx->device);
    const int64_t T = seg->T;
    int64_t off = 0;
    int64_t xo[SALT_MAX_GROUP], yo[SALT_MAX_GROUP], xb[SALT_MAX_GROUP], yb[SALT_MAX_GROUP];
    for (int i = 0; i < n; ++i) {
        const int l = layers[i];
        if (l < 0 || l >= ctx->n_layers)
            return fail(ctx, SALT_ERR_LAYER_RANGE, "layer %d outside [0, %d)", l, ctx->n_layers);
        if (T > 0) {
            if (!x_host[i] || !y_host[i]) return fail(ctx, SALT_ERR_INVALID_ARG, "null x or y");
            if ((reinterpret_cast<uintptr_t>(x_host[i]) | reinterpret_cast<uintptr_t>(y_host[i])) & 15)
                return fail(ctx, SALT_ERR_ALIGN, "x / y of group entry %d not 16-byte aligned", i);
            for (const void *h : {static_cast<const void *>(x_host[i]), static_cast<const void *>(y_host[i])}) {
                cudaPointerAttributes a;
                if (cudaPointerGetAttributes(&a, h) != cudaSuccess || a.type != cudaMemoryTypeHost) {
                    cudaGetLastError();
                    return fail(ctx, SALT_ERR_NOT_PINNED_HOST, "x / y of group entry %d is not page-locked host memory",
                                i);
                }
            }
        }
        xb[i] = T * ctx->d_in[l] * 2;
        yb[i] = T * ctx->d_out[l] * 2;
        xo[i] = off;
        off += (xb[i] + 255) / 256 * 256;
        yo[i] = off;
        off += (yb[i] + 255) / 256 * 256;
    }
    if (off > pipe->stage_bytes)
        return fail(ctx, SALT_ERR_INVALID_ARG, "the group's activations (%lld bytes) exceed a staging area (%lld)",
                    (long long)off, (long long)pipe->stage_bytes);
    if (T == 0) return SALT_OK;
    cudaStream_t stream = static_cast<cudaStream_t>(stream_);
    const int k = pipe->next;
    uint8_t *base = pipe->stage[k];
    // copies in, once the area's previous results are out
    if (pipe->used[k]) CUDA_OR_FAIL(ctx, cudaStreamWaitEvent(pipe->h2d, pipe->out_done[k], 0));
    const void *xs[SALT_MAX_GROUP];
    void *ys[SALT_MAX_GROUP];
    for (int i = 0; i < n; ++i) {
        xs[i] = base + xo[i];
        ys[i] = base + yo[i];
        CUDA_OR_FAIL(ctx, cudaMemcpyAsync(base + xo[i], x_host[i], (size_t)xb[i], cudaMemcpyHostToDevice, pipe->h2d));
        CUDA_OR_FAIL(ctx, cudaMemcpyAsync(base + yo[i], y_host[i], (size_t)yb[i], cudaMemcpyHostToDevice, pipe->h2d));
    }
    CUDA_OR_FAIL(ctx, cudaEventRecord(pipe->in_ready[k], pipe->h2d));
    // the apply on the staged copies
    CUDA_OR_FAIL(ctx, cudaStreamWaitEvent(stream, pipe->in_ready[k], 0));
    salt_status st = salt_lora_apply_grouped(ctx, seg, n, layers, xs, ys, stream_);
    if (st != SALT_OK) return st;
    CUDA_OR_FAIL(ctx, cudaEventRecord(pipe->applied[k], stream));
    // copies out
    CUDA_OR_FAIL(ctx, cudaStreamWaitEvent(pipe->d2h, pipe->applied[k], 0));
    for (int i = 0; i < n; ++i)
        CUDA_OR_FAIL(ctx, cudaMemcpyAsync(y_host[i], base + yo[i], (size_t)yb[i], cudaMemcpyDeviceToHost, pipe->d2h));
    CUDA_OR_FAIL(ctx, cudaEventRecord(pipe->out_done[k], pipe->d2h));
    pipe->used[k] = 1;
    pipe->last = k;
    pipe->next = (k + 1) % pipe->n_stages;
    return SALT_OK;
}

salt_status salt_host_pipe_wait(salt_host_pipe *pipe, salt_stream_t stream)
{
    if (!pipe || !pipe->ctx) return SALT_ERR_INVALID_ARG;
    salt_ctx *ctx = pipe->ctx;
    if (!set_device(ctx)) return fail(ctx, SALT_ERR_CUDA, "cannot select device %d", ctx->device);
    if (pipe->last >= 0)
        CUDA_OR_FAIL(ctx, cudaStreamWaitEvent(static_cast<cudaStream_t>(stream), pipe->out_done[pipe->last], 0));
    return SALT_OK;
}

salt_status salt_guard_check(salt_ctx *ctx, const salt_segments *seg, int32_t *damaged)
{
    if (!ctx || !damaged) return SALT_ERR_INVALID_ARG;
    if (seg && seg->ctx != ctx) return fail(ctx, SALT_ERR_INVALID_ARG, "segments of another context");
    if (!set_device(ctx)) return fail(ctx, SALT_ERR_CUDA, "cannot select device %d", ctx->device);
    CUDA_OR_FAIL(ctx, cudaDeviceSynchronize());
    std::vector<Guarded> bufs = {{ctx->arenaA, ctx->arenaA_bytes}, {ctx->arenaB, ctx->arenaB_bytes},
                                 {ctx->pool, ctx->pool_bytes}};
    if (seg) {
        const size_t n_pairs = (size_t)SALT_MAX_GROUP * seg->work.blk_cap;
        bufs.push_back({seg->work.vext, n_pairs * TM * VEXT_COLS * 2});
        bufs.push_back({seg->work.part, (size_t)PART_CAP * TM * PART_COLS * sizeof(float)});
    }
    int bad = 0;
    for (const Guarded &g : bufs) {
        const int d = guard_damage(g);
        if (d < 0) return fail(ctx, SALT_ERR_CUDA, "guard bands could not be read");
        bad += d;
    }
    *damaged = bad;
    return SALT_OK;
}

salt_status salt_selftest_wait_timeout(salt_ctx *ctx, salt_stream_t stream)
{
    if (!ctx) return SALT_ERR_INVALID_ARG;
    if (!set_device(ctx)) return fail(ctx, SALT_ERR_CUDA, "cannot select device %d", ctx->device);
    CUDA_OR_FAIL(ctx, launch_wait_selftest(ctx->err_dev, static_cast<cudaStream_t>(stream)));
    return SALT_OK;
}

salt_status salt_get_device_error(salt_ctx *ctx, salt_stream_t stream, uint32_t *flags)
{
    if (!ctx || !flags) return SALT_ERR_INVALID_ARG;
    if (!set_device(ctx)) return fail(ctx, SALT_ERR_CUDA, "cannot select device %d", ctx->device);
    CUDA_OR_FAIL(ctx, cudaStreamSynchronize(static_cast<cudaStream_t>(stream)));
    uint32_t v = 0;
    CUDA_OR_FAIL(ctx, cudaMemcpy(&v, ctx->err_dev, sizeof v, cudaMemcpyDeviceToHost));
    CUDA_OR_FAIL(ctx, cudaMemset(ctx->err_dev, 0, sizeof v));
    *flags = v;
    if (v) return fail(ctx, SALT_ERR_DEVICE_IDS, "device id check raised flags 0x%x", v);
    return SALT_OK;
}

}  // extern "C"
