// Host side of the C ABI declared in include/dsm.h: argument checking, the
// arena layout, the tile table, the per-launch scalars and the order of
// Algorithm 1 (arXiv 2411.17866).  Allocates no device memory.

#include "dsm.h"

#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <new>
#include <string>
#include <vector>

#include <cuda_runtime.h>

#include "dsm_internal.h"

using namespace dsm;

namespace {

thread_local std::string g_last_error;

int fail(int code, const char* fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    g_last_error = buf;
    return code;
}

int cuda_fail(cudaError_t e, const char* what) {
    return fail(DSM_ECUDA, "%s: %s (%s)", what, cudaGetErrorString(e), cudaGetErrorName(e));
}

constexpr uint64_t kAlign = 256;
constexpr uint64_t kGuardBytes = 256;       // guard region after every arena buffer
constexpr unsigned char kGuardByte = 0xA5;  // its fill pattern
constexpr uint64_t kStrideAlign = 64;  // elements; keeps every worker slice 256-byte aligned
constexpr uint64_t kMaxD = 1ull << 40;

uint64_t round_up(uint64_t v, uint64_t a) { return (v + a - 1) / a * a; }

// SplitMix64 (Steele, Lea, Flood, OOPSLA 2014) on the host: keys of the
// synthetic generators.  key(seed, stream, idx) is output 1 + stream*2^40 + idx
// of the generator seeded with `seed`.
uint64_t sm64_finalise(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

uint64_t draw_key(uint64_t seed, uint64_t stream, uint64_t idx) {
    const uint64_t j = 1ull + (stream << 40) + idx;
    return sm64_finalise(seed + j * 0x9E3779B97F4A7C15ull);
}

// The key of the same family for a layout that starts at element first_element (even) of a larger
// model: element e of the layout takes output (first_element + e)/2 + 1 = e/2 + 1 + first_element/2
// of the family, and output j of a generator seeded with `key` is the finaliser of key + j * gamma,
// so moving the key by (first_element/2) * gamma moves every output index by first_element/2.
uint64_t shard_key(uint64_t key, uint64_t first_element) {
    return key + (first_element >> 1) * 0x9E3779B97F4A7C15ull;
}

bool finite(float v) { return std::isfinite(v); }

// The arena: every region starts on a 256-byte boundary.
struct ArenaLayout {
    uint64_t d = 0, d_stride = 0;
    uint32_t num_tensors = 0, num_tiles = 0;
    uint64_t off_tensors = 0, off_tiles = 0, off_x = 0, off_m = 0, off_gv = 0, off_X = 0, off_om = 0, off_ov = 0,
             off_grad = 0, off_partials = 0, off_stats = 0, total = 0;
    size_t grad_esize = 4;
    std::vector<uint64_t> guards;  // offsets of the guard regions
};

int check_layout_and_hp(const dsm_layout* layout, uint32_t n, const dsm_hparams* hp, ArenaLayout* al) {
    if (!layout || !hp) return fail(DSM_EINVAL, "layout and hparams must not be NULL");
    if (n == 0) return fail(DSM_EINVAL, "n (workers) must be >= 1");
    if (n > kMaxWorkers) return fail(DSM_ERANGE, "n = %u exceeds the maximum of %u workers", n, kMaxWorkers);
    if (hp->base != DSM_BASE_ADAMW && hp->base != DSM_BASE_SGDM)
        return fail(DSM_EINVAL, "base optimizer %d unknown", hp->base);
    if (!(finite(hp->lr) && hp->lr > 0.f)) return fail(DSM_EINVAL, "lr (gamma) must be finite and > 0");
    if (hp->base == DSM_BASE_ADAMW) {
        if (!(hp->b1 >= 0.f && hp->b1 < 1.f) || !(hp->b2 >= 0.f && hp->b2 < 1.f))
            return fail(DSM_EINVAL, "AdamW betas must lie in [0, 1)");
        if (!(finite(hp->eps) && hp->eps > 0.f)) return fail(DSM_EINVAL, "AdamW eps must be finite and > 0");
        if (!(finite(hp->wd) && hp->wd >= 0.f)) return fail(DSM_EINVAL, "AdamW wd must be finite and >= 0");
    } else {
        if (!(hp->mu >= 0.f && hp->mu < 1.f)) return fail(DSM_EINVAL, "SGD momentum mu must lie in [0, 1)");
    }
    if (!(hp->g_b1 >= 0.f && hp->g_b1 <= 1.f) || !(hp->g_b2 >= 0.f && hp->g_b2 <= 1.f))
        return fail(DSM_EINVAL, "global betas must lie in [0, 1]");
    if (!(finite(hp->g_eta) && hp->g_eta >= 0.f)) return fail(DSM_EINVAL, "global eta must be finite and >= 0");
    if (!(finite(hp->g_wd) && hp->g_wd >= 0.f)) return fail(DSM_EINVAL, "global lambda must be finite and >= 0");
    if (hp->sign_mode != DSM_SIGN && hp->sign_mode != DSM_RSIGN_ZERO && hp->sign_mode != DSM_RSIGN_PM)
        return fail(DSM_EINVAL, "sign mode %d unknown", hp->sign_mode);
    if (hp->global_mode < DSM_GLOBAL_SIGN_MOMENTUM || hp->global_mode > DSM_GLOBAL_ADAMW)
        return fail(DSM_EINVAL, "global mode %d unknown", hp->global_mode);
    if (hp->global_mode != DSM_GLOBAL_SIGN_MOMENTUM && hp->sign_mode != DSM_SIGN)
        return fail(DSM_EINVAL, "the randomized sign applies to the sign-momentum global step only");
    if (hp->global_mode == DSM_GLOBAL_ADAMW) {
        if (!(hp->g_b1 < 1.f) || !(hp->g_b2 < 1.f)) return fail(DSM_EINVAL, "global AdamW betas must lie in [0, 1)");
        if (!(finite(hp->g_eps) && hp->g_eps > 0.f)) return fail(DSM_EINVAL, "global AdamW eps must be finite and > 0");
    }
    if (hp->sign_mode != DSM_SIGN && !(finite(hp->rsign_B) && hp->rsign_B > 0.f))
        return fail(DSM_EINVAL, "randomized sign needs a finite bound B > 0");
    if (hp->grad_dtype != DSM_F32 && hp->grad_dtype != DSM_BF16)
        return fail(DSM_EINVAL, "gradient dtype %d unknown", hp->grad_dtype);
    if (hp->flags & ~(DSM_FLAG_FUSED_ROUND | DSM_FLAG_RESET_LOCAL_STATE))
        return fail(DSM_EINVAL, "unknown bits in hparams.flags");

    uint64_t d = 0, tiles = 0;
    const int rc = check_tensor_list(layout, &d, &tiles);
    if (rc != DSM_OK) return rc;
    if (tiles * n >= (1ull << 32)) return fail(DSM_ERANGE, "too many tiles (%llu) for n = %u", (unsigned long long)tiles, n);

    ArenaLayout a;
    a.d = d;
    a.d_stride = round_up(d, kStrideAlign);
    a.num_tensors = layout->count;
    a.num_tiles = static_cast<uint32_t>(tiles);
    a.grad_esize = hp->grad_dtype == DSM_BF16 ? 2 : 4;
    uint64_t off = 0;
    auto take = [&](uint64_t bytes) {  // a buffer, then its guard region
        const uint64_t o = off;
        off = round_up(off + bytes, kAlign);
        a.guards.push_back(off);
        off += kGuardBytes;
        return o;
    };
    a.off_tensors = take(uint64_t(a.num_tensors) * sizeof(TensorDesc));
    a.off_tiles = take(uint64_t(a.num_tiles) * sizeof(TileDesc));
    a.off_x = take(a.d_stride * 4);
    a.off_m = take(a.d_stride * 4);
    a.off_gv = hp->global_mode == DSM_GLOBAL_ADAMW ? take(a.d_stride * 4) : 0;
    a.off_X = take(uint64_t(n) * a.d_stride * 4);
    a.off_om = take(uint64_t(n) * a.d_stride * 4);
    a.off_ov = hp->base == DSM_BASE_ADAMW ? take(uint64_t(n) * a.d_stride * 4) : 0;
    a.off_grad = take(uint64_t(n) * a.d_stride * a.grad_esize);
    a.off_partials = take(uint64_t(a.num_tiles) * sizeof(StatPartial));
    a.off_stats = take(uint64_t(a.num_tensors) * sizeof(TensorStats));
    a.total = off;
    *al = a;
    return DSM_OK;
}

// Makes the handle's device current for the duration of a call.
struct DeviceGuard {
    int prev = -1;
    cudaError_t err = cudaSuccess;
    explicit DeviceGuard(int dev) {
        err = cudaGetDevice(&prev);
        if (err == cudaSuccess && prev != dev) err = cudaSetDevice(dev);
        else if (err == cudaSuccess) prev = -1;
    }
    ~DeviceGuard() {
        if (prev >= 0) cudaSetDevice(prev);
    }
};

}  // namespace

void dsm::set_last_error_message(const char* msg) { g_last_error = msg; }

int dsm::check_tensor_list(const dsm_layout* layout, uint64_t* d_out, uint64_t* tiles_out) {
    if (!layout || layout->count == 0 || !layout->tensors) return fail(DSM_EINVAL, "layout has no tensors");
    uint64_t d = 0, tiles = 0;
    for (uint32_t i = 0; i < layout->count; ++i) {
        const dsm_tensor& t = layout->tensors[i];
        if (t.kind > DSM_KIND_LN_B) return fail(DSM_EINVAL, "tensor %u: kind %u unknown", i, t.kind);
        if (!finite(t.grad_scale)) return fail(DSM_EINVAL, "tensor %u: grad_scale not finite", i);
        if (t.reserved != 0) return fail(DSM_EINVAL, "tensor %u: reserved must be 0", i);
        if (t.numel > kMaxD) return fail(DSM_ERANGE, "tensor %u: numel too large", i);
        d += t.numel;
        tiles += (t.numel + kTile - 1) / kTile;
        if (d > kMaxD) return fail(DSM_ERANGE, "model larger than 2^40 elements");
    }
    if (d == 0) return fail(DSM_EINVAL, "the model has no elements (every tensor has numel 0)");
    if (layout->first_element % 4 != 0 || layout->first_element >= (1ull << 60))
        return fail(DSM_EINVAL, "first_element must be a multiple of 4 below 2^60");
    *d_out = d;
    *tiles_out = tiles;
    return DSM_OK;
}

struct dsm_handle {
    int device = 0;
    uint32_t n = 0, tau = 0;
    dsm_hparams hp{};
    ArenaLayout al;
    char* arena = nullptr;
    Problem prob{};
    LaunchShape shape{};
    std::vector<TensorDesc> tensors;
    std::vector<TileDesc> tiles;
    uint64_t t = 0;        // completed global steps
    uint32_t k = 0;        // local steps done in this round
    float gamma = 0.f;     // gamma_t of this round
    double b1_pow = 1.0;   // beta1^j and beta2^j for the last local step count j
    double b2_pow = 1.0;
    double gb1_pow = 1.0;  // global AdamW: beta1^t and beta2^t after t global steps
    double gb2_pow = 1.0;
    // fused round (DSM_FLAG_FUSED_ROUND)
    bool fused = false;           // flag set and a fused kernel exists for this problem
    bool lazy_reset = false;      // flag set: the replicas' reset is deferred (fused kernel or not)
    bool replicas_stale = false;  // the replicas' reset to x is pending
    bool last_pending = false;    // the round's last local step waits for the global step
    // DSM_FLAG_RESET_LOCAL_STATE
    bool reset_local = false;     // every round restarts the base optimizer
    bool states_zero = false;     // the base-optimizer states are zero; their zeroing in memory is pending
    AdamScalars pending_a{};
    SgdmScalars pending_sa{};
    uint64_t j = 0;        // AdamW step count of the last local step (restarts each round with the reset flag)
    uint64_t first_element = 0;  // the layout's first element within a larger model (a parameter shard)
    uint32_t first_worker = 0;   // worker 0's index in a larger set of workers (synthetic gradients)
    // local steps with host gradients (dsm_local_step_host_grads): chunk c covers tiles
    // [chunk_tile[c], chunk_tile[c+1]); ev_copied[c] marks its gradients in the arena
    std::vector<uint32_t> chunk_tile;
    std::vector<cudaEvent_t> ev_copied;
    cudaEvent_t ev_entry = nullptr;  // the caller's stream at entry (every earlier reader or writer)
    ~dsm_handle() {
        for (cudaEvent_t e : ev_copied) cudaEventDestroy(e);
        if (ev_entry) cudaEventDestroy(ev_entry);
    }
};

namespace {

cudaStream_t S(dsm_stream_t s) { return reinterpret_cast<cudaStream_t>(s); }

float* buffer_ptr(dsm_handle* h, int which, uint32_t worker) {
    const uint64_t ws = uint64_t(worker) * h->al.d_stride;
    switch (which) {
        case DSM_BUF_X: return h->prob.x;
        case DSM_BUF_M: return h->prob.m;
        case DSM_BUF_REPLICA: return h->prob.X + ws;
        case DSM_BUF_OPT_M: return h->prob.opt_m + ws;
        case DSM_BUF_OPT_V: return h->prob.opt_v ? h->prob.opt_v + ws : nullptr;
        case DSM_BUF_GLOBAL_V: return h->prob.gv;
        default: return nullptr;
    }
}

// Resolves (which, worker) to a device address and element size.
int resolve_buffer(dsm_handle* h, int which, uint32_t worker, uint64_t offset, uint64_t count, char** ptr,
                   size_t* esize) {
    if (which < DSM_BUF_X || which > DSM_BUF_GLOBAL_V) return fail(DSM_EINVAL, "buffer %d unknown", which);
    const bool per_worker = which >= DSM_BUF_REPLICA && which <= DSM_BUF_GRAD;
    if (per_worker && worker >= h->n) return fail(DSM_ERANGE, "worker %u >= n = %u", worker, h->n);
    if (offset > h->al.d || count > h->al.d - offset)
        return fail(DSM_ERANGE, "elements [%llu, %llu) outside the model of %llu", (unsigned long long)offset,
                    (unsigned long long)(offset + count), (unsigned long long)h->al.d);
    if (which == DSM_BUF_GRAD) {
        *esize = h->al.grad_esize;
        *ptr = static_cast<char*>(h->prob.grad) + (uint64_t(worker) * h->al.d_stride + offset) * *esize;
        return DSM_OK;
    }
    float* b = buffer_ptr(h, which, per_worker ? worker : 0);
    if (!b) return fail(DSM_EINVAL, "buffer %d does not exist for this base optimizer", which);
    *esize = 4;
    *ptr = reinterpret_cast<char*>(b + offset);
    return DSM_OK;
}

cudaMemcpyKind copy_kind(int other_is_device, bool to_device) {
    if (other_is_device) return cudaMemcpyDeviceToDevice;
    return to_device ? cudaMemcpyHostToDevice : cudaMemcpyDeviceToHost;
}

// Scalars of the next local step (count j + 1) and the beta powers that step
// reaches; the handle is updated only once the step is launched or deferred.
void next_local_scalars(const dsm_handle* h, AdamScalars* a, SgdmScalars* sa, double* nb1, double* nb2) {
    *a = AdamScalars{};
    *sa = SgdmScalars{};
    *nb1 = h->b1_pow;
    *nb2 = h->b2_pow;
    if (h->hp.base == DSM_BASE_ADAMW) {
        *nb1 = h->b1_pow * double(h->hp.b1);
        *nb2 = h->b2_pow * double(h->hp.b2);
        a->b1 = h->hp.b1;
        a->omb1 = float(1.0 - double(h->hp.b1));
        a->b2 = h->hp.b2;
        a->omb2 = float(1.0 - double(h->hp.b2));
        a->bc1 = float(1.0 - *nb1);
        a->bc2 = float(1.0 - *nb2);
        a->lr = h->gamma;
        a->eps = h->hp.eps;
    } else {
        sa->mu = h->hp.mu;
        sa->lr = h->gamma;
    }
}

// The local step on the tiles of problem q (the whole model, or a chunk of it).
cudaError_t launch_local_on(const dsm_handle* h, const Problem& q, const AdamScalars& a, const SgdmScalars& sa,
                            cudaStream_t s) {
    const bool from_x = h->replicas_stale, zero_state = h->states_zero;
    return h->hp.base == DSM_BASE_ADAMW ? launch_local_adamw(q, h->shape, a, from_x, zero_state, s)
                                        : launch_local_sgdm(q, h->shape, sa, from_x, zero_state, s);
}

cudaError_t launch_local(dsm_handle* h, const AdamScalars& a, const SgdmScalars& sa, cudaStream_t s) {
    cudaError_t err = launch_local_on(h, h->prob, a, sa, s);
    if (err == cudaSuccess) h->replicas_stale = h->states_zero = false;
    return err;
}

// Records a local step as done: deferred to the global step (fused round, last step) or launched.
void count_local_step(dsm_handle* h, bool deferred, const AdamScalars& a, const SgdmScalars& sa, double nb1,
                      double nb2) {
    if (deferred) {
        h->pending_a = a;
        h->pending_sa = sa;
        h->last_pending = true;
    }
    h->b1_pow = nb1;
    h->b2_pow = nb2;
    h->j += 1;
    h->k += 1;
}

// Chunks of whole tiles for dsm_local_step_host_grads: about kChunkBytes of gradients (all
// workers) each, at most kMaxChunks, and their events (created on first use).
constexpr uint64_t kChunkBytes = 64ull << 20;
constexpr uint32_t kMaxChunks = 64;

int prepare_chunks(dsm_handle* h) {
    if (!h->chunk_tile.empty()) return DSM_OK;
    const uint64_t grad_bytes = uint64_t(h->n) * h->al.d * h->al.grad_esize;
    uint64_t chunk_bytes = kChunkBytes;
    if (const char* env = std::getenv("DSM_HOST_GRAD_CHUNK_BYTES")) {  // a different chunk size (tests, tuning)
        const unsigned long long v = std::strtoull(env, nullptr, 10);
        if (v > 0) chunk_bytes = v;
    }
    uint64_t c = (grad_bytes + chunk_bytes - 1) / chunk_bytes;
    c = c < 1 ? 1 : (c > kMaxChunks ? kMaxChunks : c);
    if (c > h->al.num_tiles) c = h->al.num_tiles;
    std::vector<cudaEvent_t> ev(c, nullptr);
    cudaError_t err = cudaSuccess;
    for (uint64_t i = 0; i < c && err == cudaSuccess; ++i) err = cudaEventCreateWithFlags(&ev[i], cudaEventDisableTiming);
    cudaEvent_t entry = nullptr;
    if (err == cudaSuccess) err = cudaEventCreateWithFlags(&entry, cudaEventDisableTiming);
    if (err != cudaSuccess) {
        for (cudaEvent_t e : ev)
            if (e) cudaEventDestroy(e);
        return cuda_fail(err, "create the events of the host-gradient chunks");
    }
    h->ev_copied = std::move(ev);
    h->ev_entry = entry;
    h->chunk_tile.resize(c + 1);
    for (uint64_t i = 0; i <= c; ++i) h->chunk_tile[i] = static_cast<uint32_t>(uint64_t(h->al.num_tiles) * i / c);
    return DSM_OK;
}

// Runs a deferred last local step unfused (before its inputs or outputs are touched).
int materialize_pending(dsm_handle* h, cudaStream_t s) {
    if (!h->last_pending) return DSM_OK;
    cudaError_t err = launch_local(h, h->pending_a, h->pending_sa, s);
    if (err != cudaSuccess) return cuda_fail(err, "launch the deferred local step");
    h->last_pending = false;
    return DSM_OK;
}

// Writes x into every replica (the reset the fused round left pending).
int materialize_replicas(dsm_handle* h, cudaStream_t s) {
    if (!h->replicas_stale) return DSM_OK;
    cudaError_t err = launch_init(h->prob, h->shape, 0, 0, s);
    if (err != cudaSuccess) return cuda_fail(err, "reset the replicas");
    h->replicas_stale = false;
    return DSM_OK;
}

// Zeroes the base-optimizer states in memory (the restart DSM_FLAG_RESET_LOCAL_STATE left pending).
int materialize_states(dsm_handle* h, cudaStream_t s) {
    if (!h->states_zero) return DSM_OK;
    const size_t bytes = size_t(h->n) * h->al.d_stride * 4;
    cudaError_t err = cudaMemsetAsync(h->prob.opt_m, 0, bytes, s);
    if (err == cudaSuccess && h->prob.opt_v) err = cudaMemsetAsync(h->prob.opt_v, 0, bytes, s);
    if (err != cudaSuccess) return cuda_fail(err, "zero the base-optimizer states");
    h->states_zero = false;
    return DSM_OK;
}

// After a global step: the restart of the base optimizer (if the flag asks for it) becomes pending,
// and AdamW's step count starts again at 1.
void begin_next_round_states(dsm_handle* h) {
    if (!h->reset_local) return;
    h->states_zero = true;
    h->b1_pow = h->b2_pow = 1.0;
    h->j = 0;
}

}  // namespace

extern "C" {

size_t dsm_state_bytes(const dsm_layout* layout, uint32_t n, const dsm_hparams* hp) {
    ArenaLayout al;
    if (check_layout_and_hp(layout, n, hp, &al) != DSM_OK) return 0;
    return static_cast<size_t>(al.total);
}

int dsm_create(const dsm_layout* layout, uint32_t n, uint32_t tau, const dsm_hparams* hp, void* dev_arena,
               size_t arena_bytes, const float* x0, int x0_is_device, dsm_stream_t stream, dsm_handle** out) {
    if (!out) return fail(DSM_EINVAL, "out must not be NULL");
    *out = nullptr;
    ArenaLayout al;
    int rc = check_layout_and_hp(layout, n, hp, &al);
    if (rc != DSM_OK) return rc;
    if (tau == 0) return fail(DSM_EINVAL, "tau (local steps per round) must be >= 1");
    if (!dev_arena) return fail(DSM_EINVAL, "arena must not be NULL");
    if (reinterpret_cast<uintptr_t>(dev_arena) % kAlign != 0)
        return fail(DSM_EALIGN, "arena %p is not 256-byte aligned", dev_arena);
    if (arena_bytes < al.total)
        return fail(DSM_ENOMEM, "arena holds %zu bytes, the problem needs %llu", arena_bytes,
                    (unsigned long long)al.total);

    cudaPointerAttributes attr;
    cudaError_t err = cudaPointerGetAttributes(&attr, dev_arena);
    if (err != cudaSuccess) {
        cudaGetLastError();
        return cuda_fail(err, "cudaPointerGetAttributes(arena)");
    }
    if (attr.type != cudaMemoryTypeDevice && attr.type != cudaMemoryTypeManaged)
        return fail(DSM_EALIGN, "arena %p is not device memory", dev_arena);

    // DSM_INJECT_HOST_ALLOC_FAILURE=1 makes this allocation fail (host-side fault injection for tests)
    const char* inject = std::getenv("DSM_INJECT_HOST_ALLOC_FAILURE");
    dsm_handle* h = (inject && inject[0] == '1') ? nullptr : new (std::nothrow) dsm_handle();
    if (!h) return fail(DSM_ENOMEM, "out of host memory for the handle");
    h->device = attr.device;
    h->n = n;
    h->tau = tau;
    h->hp = *hp;
    h->al = al;
    h->arena = static_cast<char*>(dev_arena);
    h->gamma = hp->lr;
    h->reset_local = (hp->flags & DSM_FLAG_RESET_LOCAL_STATE) != 0;
    h->first_element = layout->first_element;

    // tensor and tile tables
    h->tensors.resize(al.num_tensors);
    h->tiles.reserve(al.num_tiles);
    uint64_t off = 0;
    for (uint32_t i = 0; i < al.num_tensors; ++i) {
        const dsm_tensor& t = layout->tensors[i];
        TensorDesc& td = h->tensors[i];
        td.off = off;
        td.numel = t.numel;
        td.scale = t.grad_scale;
        td.scale2 = 0.1f * t.grad_scale;
        td.lam_local = t.wd ? hp->wd : 0.0f;
        td.lam_global = t.wd ? hp->g_wd : 0.0f;
        td.kind = t.kind;
        td.tile_begin = static_cast<uint32_t>(h->tiles.size());
        for (uint64_t o = 0; o < t.numel; o += kTile) {
            TileDesc tl;
            tl.start = off + o;
            tl.len = static_cast<uint32_t>(t.numel - o < kTile ? t.numel - o : kTile);
            tl.tensor = i;
            h->tiles.push_back(tl);
        }
        td.tile_end = static_cast<uint32_t>(h->tiles.size());
        td.pad = 0;
        off += t.numel;
    }

    char* A = h->arena;
    Problem& p = h->prob;
    p.tensors = reinterpret_cast<const TensorDesc*>(A + al.off_tensors);
    p.tiles = reinterpret_cast<const TileDesc*>(A + al.off_tiles);
    p.num_tensors = al.num_tensors;
    p.num_tiles = al.num_tiles;
    p.n = n;
    p.d_stride = al.d_stride;
    p.x = reinterpret_cast<float*>(A + al.off_x);
    p.m = reinterpret_cast<float*>(A + al.off_m);
    p.gv = hp->global_mode == DSM_GLOBAL_ADAMW ? reinterpret_cast<float*>(A + al.off_gv) : nullptr;
    p.global_mode = hp->global_mode;
    p.X = reinterpret_cast<float*>(A + al.off_X);
    p.opt_m = reinterpret_cast<float*>(A + al.off_om);
    p.opt_v = hp->base == DSM_BASE_ADAMW ? reinterpret_cast<float*>(A + al.off_ov) : nullptr;
    p.grad = A + al.off_grad;
    p.grad_bf16 = hp->grad_dtype == DSM_BF16;
    p.partials = reinterpret_cast<StatPartial*>(A + al.off_partials);
    p.stats = reinterpret_cast<TensorStats*>(A + al.off_stats);

    DeviceGuard guard(h->device);
    if (guard.err != cudaSuccess) {
        delete h;
        return cuda_fail(guard.err, "cudaSetDevice");
    }
    cudaStream_t s = S(stream);
    auto bail = [&](cudaError_t e, const char* what) {
        delete h;
        return cuda_fail(e, what);
    };
    if ((err = query_launch_shape(p, &h->shape)) != cudaSuccess) return bail(err, "occupancy query");
    h->fused = (hp->flags & DSM_FLAG_FUSED_ROUND) && fused_round_available(p);
    h->lazy_reset = (hp->flags & DSM_FLAG_FUSED_ROUND) != 0;
    // The tables are copied from the handle's own vectors, which outlive the copies.
    if ((err = cudaMemcpyAsync(A + al.off_tensors, h->tensors.data(), h->tensors.size() * sizeof(TensorDesc),
                               cudaMemcpyHostToDevice, s)) != cudaSuccess)
        return bail(err, "copy tensor table");
    if ((err = cudaMemcpyAsync(A + al.off_tiles, h->tiles.data(), h->tiles.size() * sizeof(TileDesc),
                               cudaMemcpyHostToDevice, s)) != cudaSuccess)
        return bail(err, "copy tile table");
    // m_0 = 0, base-optimizer states = 0, gradients = 0, statistics = 0
    const uint64_t zero_from = al.off_m;
    if ((err = cudaMemsetAsync(A + zero_from, 0, al.total - zero_from, s)) != cudaSuccess)
        return bail(err, "zero the state");
    for (uint64_t g : al.guards)
        if ((err = cudaMemsetAsync(A + g, kGuardByte, kGuardBytes, s)) != cudaSuccess) return bail(err, "fill guards");
    if (x0) {
        if ((err = cudaMemcpyAsync(p.x, x0, al.d * 4, x0_is_device ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice,
                                   s)) != cudaSuccess)
            return bail(err, "copy x0");
    }
    if ((err = launch_init(p, h->shape, shard_key(draw_key(hp->seed, 2, 0), h->first_element), x0 ? 0 : 1, s)) !=
        cudaSuccess)
        return bail(err, "launch init");
    *out = h;
    return DSM_OK;
}

int dsm_set_gamma(dsm_handle* h, float gamma) {
    if (!h) return fail(DSM_EINVAL, "handle is NULL");
    if (!(finite(gamma) && gamma > 0.f)) return fail(DSM_EINVAL, "gamma must be finite and > 0");
    if (h->k != 0) return fail(DSM_ESTATE, "gamma can change only between rounds (%u local steps done)", h->k);
    h->gamma = gamma;
    return DSM_OK;
}

int dsm_fill_synthetic_grads(dsm_handle* h, uint64_t step, dsm_stream_t stream) {
    if (!h) return fail(DSM_EINVAL, "handle is NULL");
    GradKeys k;
    k.step = shard_key(draw_key(h->hp.seed, 0, step), h->first_element);
    for (uint32_t i = 0; i < kMaxWorkers; ++i)
        k.worker[i] = i < h->n ? shard_key(draw_key(h->hp.seed, 1, uint64_t(h->first_worker) + i), h->first_element) : 0;
    DeviceGuard guard(h->device);
    if (guard.err != cudaSuccess) return cuda_fail(guard.err, "cudaSetDevice");
    int rc = materialize_pending(h, S(stream));
    if (rc != DSM_OK) return rc;
    cudaError_t err = launch_grad_fill(h->prob, h->shape, k, S(stream));
    if (err != cudaSuccess) return cuda_fail(err, "launch grad fill");
    return DSM_OK;
}

int dsm_set_first_worker(dsm_handle* h, uint32_t first_worker) {
    if (!h) return fail(DSM_EINVAL, "handle is NULL");
    if (uint64_t(first_worker) + h->n > (uint64_t(1) << 32))
        return fail(DSM_ERANGE, "workers %u .. %u + %u exceed 2^32", first_worker, first_worker, h->n);
    h->first_worker = first_worker;
    return DSM_OK;
}

int dsm_grad_ptr(dsm_handle* h, uint32_t worker, void** dev_ptr) {
    if (!h || !dev_ptr) return fail(DSM_EINVAL, "NULL argument");
    if (worker >= h->n) return fail(DSM_ERANGE, "worker %u >= n = %u", worker, h->n);
    *dev_ptr = static_cast<char*>(h->prob.grad) + uint64_t(worker) * h->al.d_stride * h->al.grad_esize;
    return DSM_OK;
}

int dsm_replica_ptr(dsm_handle* h, uint32_t worker, dsm_stream_t stream, const float** dev_ptr) {
    if (!h || !dev_ptr) return fail(DSM_EINVAL, "NULL argument");
    if (worker >= h->n) return fail(DSM_ERANGE, "worker %u >= n = %u", worker, h->n);
    DeviceGuard guard(h->device);
    if (guard.err != cudaSuccess) return cuda_fail(guard.err, "cudaSetDevice");
    int rc = materialize_pending(h, S(stream));
    if (rc != DSM_OK) return rc;
    *dev_ptr = h->replicas_stale ? h->prob.x : h->prob.X + uint64_t(worker) * h->al.d_stride;
    return DSM_OK;
}

int dsm_load_grads(dsm_handle* h, const void* src, int src_is_device, dsm_stream_t stream) {
    if (!h || !src) return fail(DSM_EINVAL, "NULL argument");
    DeviceGuard guard(h->device);
    if (guard.err != cudaSuccess) return cuda_fail(guard.err, "cudaSetDevice");
    int rc = materialize_pending(h, S(stream));
    if (rc != DSM_OK) return rc;
    const size_t es = h->al.grad_esize;
    const cudaMemcpyKind kind = src_is_device ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice;
    cudaError_t err;
    if (h->al.d_stride == h->al.d)  // the workers' slices are contiguous: one linear copy
        err = cudaMemcpyAsync(h->prob.grad, src, h->al.d * es * h->n, kind, S(stream));
    else
        err = cudaMemcpy2DAsync(h->prob.grad, h->al.d_stride * es, src, h->al.d * es, h->al.d * es, h->n, kind,
                                S(stream));
    if (err != cudaSuccess) return cuda_fail(err, "copy gradients");
    return DSM_OK;
}

int dsm_local_step(dsm_handle* h, dsm_stream_t stream) {
    if (!h) return fail(DSM_EINVAL, "handle is NULL");
    if (h->k >= h->tau)
        return fail(DSM_ESTATE, "all %u local steps of round %llu are done; call dsm_global_step", h->tau,
                    (unsigned long long)h->t);
    DeviceGuard guard(h->device);
    if (guard.err != cudaSuccess) return cuda_fail(guard.err, "cudaSetDevice");
    // step count j = t*tau + k + 1; beta^j by successive float64 products
    AdamScalars a;
    SgdmScalars sa;
    double nb1, nb2;
    next_local_scalars(h, &a, &sa, &nb1, &nb2);
    const bool defer = h->fused && h->k + 1 == h->tau;  // the last step runs inside dsm_global_step
    if (!defer) {
        cudaError_t err = launch_local(h, a, sa, S(stream));
        if (err != cudaSuccess) return cuda_fail(err, "launch local step");  // the handle is unchanged
    }
    count_local_step(h, defer, a, sa, nb1, nb2);
    return DSM_OK;
}

int dsm_local_step_host_grads(dsm_handle* h, const void* src, dsm_stream_t stream, dsm_stream_t copy_stream) {
    if (!h || !src) return fail(DSM_EINVAL, "NULL argument");
    if (h->k >= h->tau)
        return fail(DSM_ESTATE, "all %u local steps of round %llu are done; call dsm_global_step", h->tau,
                    (unsigned long long)h->t);
    DeviceGuard guard(h->device);
    if (guard.err != cudaSuccess) return cuda_fail(guard.err, "cudaSetDevice");
    cudaStream_t s = S(stream), cs = S(copy_stream);
    int rc = prepare_chunks(h);
    if (rc != DSM_OK) return rc;
    AdamScalars a;
    SgdmScalars sa;
    double nb1, nb2;
    next_local_scalars(h, &a, &sa, &nb1, &nb2);
    const bool defer = h->fused && h->k + 1 == h->tau;  // the update runs inside dsm_global_step
    const size_t es = h->al.grad_esize;
    char* grad = static_cast<char*>(h->prob.grad);
    const char* host = static_cast<const char*>(src);
    // the copies follow everything already enqueued on the caller's stream (earlier readers and
    // writers of the gradient buffers)
    cudaError_t err = cudaEventRecord(h->ev_entry, s);
    if (err == cudaSuccess) err = cudaStreamWaitEvent(cs, h->ev_entry, 0);
    if (err != cudaSuccess) return cuda_fail(err, "order the gradient copies after the stream");
    const uint32_t chunks = static_cast<uint32_t>(h->ev_copied.size());
    for (uint32_t c = 0; c < chunks; ++c) {
        const uint32_t t0 = h->chunk_tile[c], t1 = h->chunk_tile[c + 1];
        const uint64_t e0 = h->tiles[t0].start, e1 = h->tiles[t1 - 1].start + h->tiles[t1 - 1].len;
        err = cudaMemcpy2DAsync(grad + e0 * es, h->al.d_stride * es, host + e0 * es, h->al.d * es, (e1 - e0) * es,
                                h->n, cudaMemcpyHostToDevice, cs);
        if (err == cudaSuccess) err = cudaEventRecord(h->ev_copied[c], cs);
        if (err == cudaSuccess) err = cudaStreamWaitEvent(s, h->ev_copied[c], 0);
        if (err != cudaSuccess) return cuda_fail(err, "copy a chunk of gradients");
        if (!defer) {
            Problem q = h->prob;
            q.tiles = h->prob.tiles + t0;
            q.num_tiles = t1 - t0;
            err = launch_local_on(h, q, a, sa, s);
            if (err != cudaSuccess) return cuda_fail(err, "launch the local step on a chunk");
        }
    }
    if (!defer) h->replicas_stale = h->states_zero = false;
    count_local_step(h, defer, a, sa, nb1, nb2);
    return DSM_OK;
}

int dsm_global_step(dsm_handle* h, dsm_stream_t stream, dsm_tensor_stats* stats, uint32_t stats_count) {
    if (!h) return fail(DSM_EINVAL, "handle is NULL");
    if (h->k != h->tau)
        return fail(DSM_ESTATE, "global step needs %u local steps in this round, %u done", h->tau, h->k);
    if (stats && stats_count < h->al.num_tensors)
        return fail(DSM_EINVAL, "stats holds %u entries, the layout has %u tensors", stats_count, h->al.num_tensors);
    DeviceGuard guard(h->device);
    if (guard.err != cudaSuccess) return cuda_fail(guard.err, "cudaSetDevice");
    GlobalScalars g{};
    g.b1 = h->hp.g_b1;
    g.b2 = h->hp.g_b2;
    g.c1 = float((1.0 - double(h->hp.g_b1)) / double(h->gamma));
    g.c2 = float((1.0 - double(h->hp.g_b2)) / double(h->gamma));
    g.eta_gamma = float(double(h->hp.g_eta) * double(h->gamma));
    g.inv_gamma = float(1.0 / double(h->gamma));
    // global AdamW at step count t+1: beta^(t+1) by successive float64 products
    const double ngb1 = h->gb1_pow * double(h->hp.g_b1);
    const double ngb2 = h->gb2_pow * double(h->hp.g_b2);
    g.omb1 = float(1.0 - double(h->hp.g_b1));
    g.omb2 = float(1.0 - double(h->hp.g_b2));
    g.bc1 = float(1.0 - ngb1);
    g.bc2 = float(1.0 - ngb2);
    g.eps = h->hp.g_eps;
    g.eta = h->hp.g_eta;
    g.B = h->hp.rsign_B;
    g.n_f = float(h->n);
    g.sign_mode = h->hp.sign_mode;
    g.mode = h->hp.global_mode;
    g.philox_k0 = static_cast<uint32_t>(h->hp.seed & 0xFFFFFFFFull);
    g.philox_k1 = static_cast<uint32_t>(h->t & 0xFFFFFFFFull);
    g.philox_q0 = h->first_element >> 2;
    cudaStream_t s = S(stream);
    cudaError_t err;
    uint32_t grid = 0;  // CTAs of the global-step launch (the statistics reduction needs it)
    if (h->last_pending) {  // fused round: last local step + global step, reset left pending
        const int opts = (h->replicas_stale ? kFusedFromX : 0) | (h->states_zero ? kFusedZeroState : 0) |
                         (h->reset_local ? kFusedDropState : 0);
        err = launch_fused_last_global(h->prob, h->shape, h->pending_a, h->pending_sa, g, opts, s, &grid);
        if (err != cudaSuccess) return cuda_fail(err, "launch fused last local step and global step");
        h->last_pending = false;
        h->replicas_stale = true;
        h->states_zero = false;  // (set again below when the round restarts the base optimizer)
    } else {
        int rc = materialize_replicas(h, s);
        if (rc != DSM_OK) return rc;
        g.skip_reset = h->lazy_reset ? 1 : 0;  // more than 8 workers: only the reset is deferred
        err = launch_global(h->prob, h->shape, g, s, &grid);
        if (err != cudaSuccess) return cuda_fail(err, "launch global step");
        if (h->lazy_reset) h->replicas_stale = true;
    }
    err = launch_stats(h->prob, grid, s);
    if (err != cudaSuccess) return cuda_fail(err, "launch statistics");
    h->t += 1;
    h->k = 0;
    h->gb1_pow = ngb1;
    h->gb2_pow = ngb2;
    begin_next_round_states(h);
    if (stats) {
        err = cudaMemcpyAsync(stats, h->prob.stats, size_t(h->al.num_tensors) * sizeof(TensorStats),
                              cudaMemcpyDeviceToHost, s);
        if (err != cudaSuccess) return cuda_fail(err, "copy statistics");
        err = cudaStreamSynchronize(s);
        if (err != cudaSuccess) return cuda_fail(err, "synchronise after the global step");
    }
    return DSM_OK;
}

int dsm_stats_ptr(dsm_handle* h, const dsm_tensor_stats** dev_ptr) {
    if (!h || !dev_ptr) return fail(DSM_EINVAL, "NULL argument");
    *dev_ptr = reinterpret_cast<const dsm_tensor_stats*>(h->prob.stats);
    return DSM_OK;
}

int dsm_read_params(dsm_handle* h, int which, uint32_t worker, void* dst, uint64_t offset, uint64_t count,
                    int dst_is_device, dsm_stream_t stream) {
    if (!h || (!dst && count)) return fail(DSM_EINVAL, "NULL argument");
    char* src;
    size_t es;
    int rc = resolve_buffer(h, which, worker, offset, count, &src, &es);
    if (rc != DSM_OK) return rc;
    if (count == 0) return DSM_OK;
    DeviceGuard guard(h->device);
    if (guard.err != cudaSuccess) return cuda_fail(guard.err, "cudaSetDevice");
    if (which >= DSM_BUF_REPLICA && which <= DSM_BUF_OPT_V) {
        rc = materialize_pending(h, S(stream));
        if (rc != DSM_OK) return rc;
    }
    if (which == DSM_BUF_REPLICA && h->replicas_stale) src = reinterpret_cast<char*>(h->prob.x + offset);
    cudaError_t err;
    if ((which == DSM_BUF_OPT_M || which == DSM_BUF_OPT_V) && h->states_zero) {  // restart pending: zeros
        if (dst_is_device) {
            err = cudaMemsetAsync(dst, 0, count * es, S(stream));
            if (err != cudaSuccess) return cuda_fail(err, "read buffer");
            return DSM_OK;
        }
        if ((err = cudaStreamSynchronize(S(stream))) != cudaSuccess) return cuda_fail(err, "synchronise before read");
        std::memset(dst, 0, count * es);
        return DSM_OK;
    }
    const cudaMemcpyKind kind = copy_kind(dst_is_device, false);
    err = cudaMemcpyAsync(dst, src, count * es, kind, S(stream));
    if (err != cudaSuccess) return cuda_fail(err, "read buffer");
    if (!dst_is_device && (err = cudaStreamSynchronize(S(stream))) != cudaSuccess)
        return cuda_fail(err, "synchronise after read");
    return DSM_OK;
}

int dsm_write_params(dsm_handle* h, int which, uint32_t worker, const void* src, uint64_t offset, uint64_t count,
                     int src_is_device, dsm_stream_t stream) {
    if (!h || (!src && count)) return fail(DSM_EINVAL, "NULL argument");
    char* dst;
    size_t es;
    int rc = resolve_buffer(h, which, worker, offset, count, &dst, &es);
    if (rc != DSM_OK) return rc;
    if (count == 0) return DSM_OK;
    DeviceGuard guard(h->device);
    if (guard.err != cudaSuccess) return cuda_fail(guard.err, "cudaSetDevice");
    if ((rc = materialize_pending(h, S(stream))) != DSM_OK) return rc;
    if ((rc = materialize_replicas(h, S(stream))) != DSM_OK) return rc;
    if ((which == DSM_BUF_OPT_M || which == DSM_BUF_OPT_V) && (rc = materialize_states(h, S(stream))) != DSM_OK)
        return rc;
    const cudaMemcpyKind kind = copy_kind(src_is_device, true);
    cudaError_t err = cudaMemcpyAsync(dst, src, count * es, kind, S(stream));
    if (err != cudaSuccess) return cuda_fail(err, "write buffer");
    if (!src_is_device && (err = cudaStreamSynchronize(S(stream))) != cudaSuccess)
        return cuda_fail(err, "synchronise after write");
    return DSM_OK;
}

int dsm_cosine_gamma(float peak, float final_ratio, uint64_t warmup_steps, uint64_t total_steps, uint64_t step,
                     float* gamma) {
    if (!gamma) return fail(DSM_EINVAL, "gamma must not be NULL");
    if (!(finite(peak) && peak > 0.f)) return fail(DSM_EINVAL, "peak must be finite and > 0");
    if (!(final_ratio >= 0.f && final_ratio <= 1.f)) return fail(DSM_EINVAL, "final_ratio must lie in [0, 1]");
    if (total_steps == 0 || warmup_steps > total_steps)
        return fail(DSM_EINVAL, "need 0 < total_steps and warmup_steps <= total_steps");
    const double P = peak, F = double(final_ratio) * double(peak);
    double g;
    if (step < warmup_steps) {
        g = P * double(step + 1) / double(warmup_steps);
    } else if (step >= total_steps) {
        g = F;
    } else {
        const double r = double(step - warmup_steps) / double(total_steps - warmup_steps);
        g = F + 0.5 * (1.0 + std::cos(M_PI * r)) * (P - F);
    }
    *gamma = float(g);
    return DSM_OK;
}

int dsm_set_round(dsm_handle* h, uint64_t round) {
    if (!h) return fail(DSM_EINVAL, "handle is NULL");
    if (h->k != 0) return fail(DSM_ESTATE, "the round counter can change only between rounds");
    h->t = round;
    h->j = h->reset_local ? 0 : round * h->tau;
    double p1 = 1.0, p2 = 1.0;
    for (uint64_t i = 0; i < h->j; ++i) {
        p1 *= double(h->hp.b1);
        p2 *= double(h->hp.b2);
    }
    h->b1_pow = p1;
    h->b2_pow = p2;
    double q1 = 1.0, q2 = 1.0;
    for (uint64_t i = 0; i < round; ++i) {
        q1 *= double(h->hp.g_b1);
        q2 *= double(h->hp.g_b2);
    }
    h->gb1_pow = q1;
    h->gb2_pow = q2;
    return DSM_OK;
}

int dsm_end_round(dsm_handle* h, const float* x_next, int x_is_device, dsm_stream_t stream) {
    if (!h || !x_next) return fail(DSM_EINVAL, "NULL argument");
    if (h->k != h->tau)
        return fail(DSM_ESTATE, "ending round %llu needs its %u local steps, %u done", (unsigned long long)h->t,
                    h->tau, h->k);
    DeviceGuard guard(h->device);
    if (guard.err != cudaSuccess) return cuda_fail(guard.err, "cudaSetDevice");
    cudaStream_t s = S(stream);
    int rc = materialize_pending(h, s);  // the workers' last base-optimizer step
    if (rc != DSM_OK) return rc;
    cudaError_t err = cudaMemcpyAsync(h->prob.x, x_next, size_t(h->al.d) * 4, copy_kind(x_is_device, true), s);
    if (err != cudaSuccess) return cuda_fail(err, "write the next global model");
    h->replicas_stale = true;  // every worker restarts from x
    h->t += 1;
    h->k = 0;
    h->gb1_pow *= double(h->hp.g_b1);
    h->gb2_pow *= double(h->hp.g_b2);
    begin_next_round_states(h);
    if (!x_is_device && (err = cudaStreamSynchronize(s)) != cudaSuccess)
        return cuda_fail(err, "synchronise after writing the global model");
    return DSM_OK;
}

int dsm_check_guards(dsm_handle* h, dsm_stream_t stream, uint32_t* bad_regions) {
    if (!h || !bad_regions) return fail(DSM_EINVAL, "NULL argument");
    DeviceGuard guard(h->device);
    if (guard.err != cudaSuccess) return cuda_fail(guard.err, "cudaSetDevice");
    std::vector<unsigned char> buf(h->al.guards.size() * kGuardBytes);
    cudaStream_t s = S(stream);
    cudaError_t err;
    for (size_t i = 0; i < h->al.guards.size(); ++i)
        if ((err = cudaMemcpyAsync(buf.data() + i * kGuardBytes, h->arena + h->al.guards[i], kGuardBytes,
                                   cudaMemcpyDeviceToHost, s)) != cudaSuccess)
            return cuda_fail(err, "read guards");
    if ((err = cudaStreamSynchronize(s)) != cudaSuccess) return cuda_fail(err, "synchronise after reading guards");
    uint32_t bad = 0;
    for (size_t i = 0; i < h->al.guards.size(); ++i) {
        for (uint64_t b = 0; b < kGuardBytes; ++b)
            if (buf[i * kGuardBytes + b] != kGuardByte) {
                ++bad;
                break;
            }
    }
    *bad_regions = bad;
    return DSM_OK;
}

int dsm_get_info(const dsm_handle* h, dsm_info* out) {
    if (!h || !out) return fail(DSM_EINVAL, "NULL argument");
    out->d = h->al.d;
    out->d_stride = h->al.d_stride;
    out->n = h->n;
    out->tau = h->tau;
    out->num_tensors = h->al.num_tensors;
    out->num_tiles = h->al.num_tiles;
    out->round = h->t;
    out->local_steps = h->k;
    out->gamma = h->gamma;
    return DSM_OK;
}

int dsm_destroy(dsm_handle* h) {
    if (!h) return DSM_OK;
    DeviceGuard guard(h->device);  // the handle's events belong to its device
    delete h;
    return DSM_OK;
}

const char* dsm_last_error(void) { return g_last_error.c_str(); }

}  // extern "C"
