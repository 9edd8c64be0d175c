// dsm_global_step_noalloc: the global step of dsm_global_step() on buffers
// the caller already owns, for callers that cannot allocate device memory
// (a host framework that owns all of HBM through its own pool and forbids
// outside allocations, or a latency-critical loop that must not block or
// synchronise in cudaMalloc/cudaFree).  The tile table and the per-tile
// statistics, which dsm_create() keeps in the caller's arena, live here in
// one static device array instead; this file allocates nothing.

#include <cstdio>
#include <string>

#include "dsm.h"
#include "dsm_internal.h"

namespace dsm {
namespace {

constexpr uint64_t align256(uint64_t v) { return (v + 255) / 256 * 256; }

constexpr uint32_t kNaMaxTensors = DSM_NOALLOC_MAX_TENSORS;
constexpr uint32_t kNaMaxTiles = DSM_NOALLOC_MAX_TILES;
// Regions of the scratch array (byte offsets).
constexpr uint64_t kOffLayout = 0;  // copy of the caller's dsm_tensor list
constexpr uint64_t kOffTensors = align256(kOffLayout + sizeof(dsm_tensor) * kNaMaxTensors);
constexpr uint64_t kOffTiles = align256(kOffTensors + sizeof(TensorDesc) * kNaMaxTensors);
constexpr uint64_t kOffPartials = align256(kOffTiles + sizeof(TileDesc) * uint64_t(kNaMaxTiles));
constexpr uint64_t kOffStats = align256(kOffPartials + sizeof(StatPartial) * uint64_t(kNaMaxTiles));
constexpr uint64_t kScratchBytes = align256(kOffStats + sizeof(TensorStats) * kNaMaxTensors);
static_assert(kScratchBytes == DSM_NOALLOC_SCRATCH_BYTES, "scratch size in dsm.h is out of date");

// The scratch array: shared by every call on a device, kept until the process exits.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kScratchBytes];

// One CTA: tensor offsets and tile ranges by a prefix sum over the tensor list.
__global__ void __launch_bounds__(kThreads) k_noalloc_tensor_table(unsigned char* scratch, uint32_t count,
                                                                   float lam_global) {
    const dsm_tensor* in = reinterpret_cast<const dsm_tensor*>(scratch + kOffLayout);
    TensorDesc* out = reinterpret_cast<TensorDesc*>(scratch + kOffTensors);
    __shared__ unsigned long long s_el[kThreads], s_ti[kThreads];
    const uint32_t per = (count + kThreads - 1) / kThreads;
    const uint32_t b = threadIdx.x * per, e = min(b + per, count);
    unsigned long long el = 0, ti = 0;
    for (uint32_t i = b; i < e; ++i) {
        el += in[i].numel;
        ti += (in[i].numel + kTile - 1) / kTile;
    }
    s_el[threadIdx.x] = el;
    s_ti[threadIdx.x] = ti;
    __syncthreads();
    if (threadIdx.x == 0) {  // exclusive scan of the 256 chunk sums
        unsigned long long a = 0, c = 0;
        for (uint32_t k = 0; k < kThreads; ++k) {
            const unsigned long long va = s_el[k], vc = s_ti[k];
            s_el[k] = a;
            s_ti[k] = c;
            a += va;
            c += vc;
        }
    }
    __syncthreads();
    el = s_el[threadIdx.x];
    ti = s_ti[threadIdx.x];
    for (uint32_t i = b; i < e; ++i) {
        TensorDesc t;
        t.off = el;
        t.numel = in[i].numel;
        t.scale = in[i].grad_scale;
        t.scale2 = 0.0f;
        t.lam_local = 0.0f;
        t.lam_global = in[i].wd ? lam_global : 0.0f;
        t.kind = in[i].kind;
        t.tile_begin = static_cast<uint32_t>(ti);
        ti += (in[i].numel + kTile - 1) / kTile;
        t.tile_end = static_cast<uint32_t>(ti);
        t.pad = 0;
        out[i] = t;
        el += in[i].numel;
    }
}

// Tile table: tile ti belongs to the last tensor whose tile_begin <= ti.
__global__ void __launch_bounds__(kThreads) k_noalloc_tile_table(unsigned char* scratch, uint32_t count,
                                                                 uint32_t num_tiles) {
    const TensorDesc* t = reinterpret_cast<const TensorDesc*>(scratch + kOffTensors);
    TileDesc* tiles = reinterpret_cast<TileDesc*>(scratch + kOffTiles);
    for (uint32_t ti = blockIdx.x * blockDim.x + threadIdx.x; ti < num_tiles; ti += gridDim.x * blockDim.x) {
        uint32_t lo = 0, hi = count;  // first tensor with tile_begin > ti
        while (lo < hi) {
            const uint32_t mid = (lo + hi) / 2;
            if (t[mid].tile_begin <= ti) lo = mid + 1;
            else hi = mid;
        }
        const TensorDesc& T = t[lo - 1];
        const uint64_t o = uint64_t(ti - T.tile_begin) * kTile;
        TileDesc d;
        d.start = T.off + o;
        d.len = static_cast<uint32_t>(T.numel - o < kTile ? T.numel - o : kTile);
        d.tensor = lo - 1;
        tiles[ti] = d;
    }
}

}  // namespace
}  // namespace dsm

using namespace dsm;

namespace {

// Failures are reported through dsm_last_error(), like every other call.
int na_fail(int code, const char* msg) {
    char buf[512];
    snprintf(buf, sizeof buf, "dsm_global_step_noalloc: %s", msg);
    set_last_error_message(buf);
    return code;
}

int na_cuda(cudaError_t e, const char* what) {
    char buf[512];
    snprintf(buf, sizeof buf, "dsm_global_step_noalloc: %s: %s", what, cudaGetErrorString(e));
    set_last_error_message(buf);
    return DSM_ECUDA;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// DSM_OK if p is device (or managed) memory of device `dev`; the name goes into the message otherwise.
int check_device_buffer(const void* p, int dev, const char* name) {
    cudaPointerAttributes attr;
    const cudaError_t err = cudaPointerGetAttributes(&attr, p);
    if (err != cudaSuccess) {
        cudaGetLastError();
        char what[96];
        snprintf(what, sizeof what, "cudaPointerGetAttributes(%s)", name);
        return na_cuda(err, what);
    }
    if ((attr.type != cudaMemoryTypeDevice && attr.type != cudaMemoryTypeManaged) || attr.device != dev) {
        char msg[128];
        snprintf(msg, sizeof msg, "%s is not device memory of the current device", name);
        return na_fail(DSM_EINVAL, msg);
    }
    return DSM_OK;
}

}  // namespace

extern "C" int dsm_global_step_noalloc(const dsm_layout* layout, uint32_t n, const dsm_hparams* hp, float gamma,
                                       uint64_t round, float* x, float* m, float* replicas,
                                       uint64_t replica_stride, dsm_tensor_stats* stats, int stats_is_device,
                                       dsm_stream_t stream) {
    if (!layout || !hp || !x || !m || !replicas) return na_fail(DSM_EINVAL, "NULL argument");
    // the tensor list passes the same checks as in dsm_create()
    uint64_t d = 0, tiles = 0;
    if (const int rc = check_tensor_list(layout, &d, &tiles); rc != DSM_OK) {
        const std::string why = dsm_last_error();
        return na_fail(rc, why.c_str());
    }
    if (layout->count > kNaMaxTensors) return na_fail(DSM_ERANGE, "more than DSM_NOALLOC_MAX_TENSORS (4096) tensors");
    if (n == 0 || n > kMaxWorkers) return na_fail(n == 0 ? DSM_EINVAL : DSM_ERANGE, "n must lie in [1, 64]");
    if (!(gamma > 0.f && gamma < 3.0e38f)) return na_fail(DSM_EINVAL, "gamma must be finite and > 0");
    if (!(hp->g_b1 >= 0.f && hp->g_b1 <= 1.f) || !(hp->g_b2 >= 0.f && hp->g_b2 <= 1.f))
        return na_fail(DSM_EINVAL, "global betas must lie in [0, 1]");
    if (!(hp->g_eta >= 0.f && hp->g_eta < 3.0e38f) || !(hp->g_wd >= 0.f && hp->g_wd < 3.0e38f))
        return na_fail(DSM_EINVAL, "global eta and lambda must be finite and >= 0");
    if (hp->sign_mode < DSM_SIGN || hp->sign_mode > DSM_RSIGN_PM) return na_fail(DSM_EINVAL, "sign mode unknown");
    if (hp->global_mode < DSM_GLOBAL_SIGN_MOMENTUM || hp->global_mode > DSM_GLOBAL_LOOKAHEAD)
        return na_fail(DSM_EINVAL, "global step must be DSM_GLOBAL_SIGN_MOMENTUM, _SLOWMO, _SIGNED_SLOWMO or "
                                   "_LOOKAHEAD here (global AdamW needs a second-moment buffer)");
    if (hp->global_mode != DSM_GLOBAL_SIGN_MOMENTUM && hp->sign_mode != DSM_SIGN)
        return na_fail(DSM_EINVAL, "the randomized signs apply to the sign-momentum global step only");
    if (hp->sign_mode != DSM_SIGN && !(hp->rsign_B > 0.f && hp->rsign_B < 3.0e38f))
        return na_fail(DSM_EINVAL, "randomized sign needs a finite bound B > 0");
    if (tiles > kNaMaxTiles)
        return na_fail(DSM_ERANGE, "layout needs more than DSM_NOALLOC_MAX_TILES (524288) tiles of 1024 elements");
    if (replica_stride < d || replica_stride % 8 != 0)
        return na_fail(DSM_EINVAL, "replica_stride must be >= d and a multiple of 8");
    if (!aligned16(x) || !aligned16(m) || !aligned16(replicas))
        return na_fail(DSM_EALIGN, "x, m and replicas must be 16-byte aligned");

    int dev = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err != cudaSuccess) return na_cuda(err, "cudaGetDevice");
    if (int rc = check_device_buffer(x, dev, "x"); rc != DSM_OK) return rc;
    if (int rc = check_device_buffer(m, dev, "m"); rc != DSM_OK) return rc;
    if (int rc = check_device_buffer(replicas, dev, "replicas"); rc != DSM_OK) return rc;
    if (stats && stats_is_device)
        if (int rc = check_device_buffer(stats, dev, "stats"); rc != DSM_OK) return rc;

    // The scratch array's device address on the current device, looked up by every call (a lookup,
    // no allocation), so that it is never stale: not after cudaDeviceReset, and not in another
    // context.  The first call on a device may load the library's device code there.
    void* scratch_v = nullptr;
    err = cudaGetSymbolAddress(&scratch_v, g_noalloc_scratch);
    if (err != cudaSuccess) return na_cuda(err, "cudaGetSymbolAddress(scratch)");
    unsigned char* scratch = static_cast<unsigned char*>(scratch_v);
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);

    // Tensor and tile tables, rebuilt in the scratch array by every call.
    err = cudaMemcpyAsync(scratch + kOffLayout, layout->tensors, sizeof(dsm_tensor) * layout->count,
                          cudaMemcpyHostToDevice, s);
    if (err != cudaSuccess) return na_cuda(err, "copy the tensor list");
    k_noalloc_tensor_table<<<1, kThreads, 0, s>>>(scratch, layout->count, hp->g_wd);
    if ((err = cudaGetLastError()) != cudaSuccess) return na_cuda(err, "launch tensor table");
    const uint32_t num_tiles = static_cast<uint32_t>(tiles);
    const uint32_t tb = (num_tiles + kThreads - 1) / kThreads;
    k_noalloc_tile_table<<<tb < 1024 ? tb : 1024, kThreads, 0, s>>>(scratch, layout->count, num_tiles);
    if ((err = cudaGetLastError()) != cudaSuccess) return na_cuda(err, "launch tile table");

    Problem p{};
    p.tensors = reinterpret_cast<const TensorDesc*>(scratch + kOffTensors);
    p.tiles = reinterpret_cast<const TileDesc*>(scratch + kOffTiles);
    p.num_tensors = layout->count;
    p.num_tiles = num_tiles;
    p.n = n;
    p.d_stride = replica_stride;
    p.x = x;
    p.m = m;
    p.X = replicas;
    p.partials = reinterpret_cast<StatPartial*>(scratch + kOffPartials);
    p.stats = reinterpret_cast<TensorStats*>(scratch + kOffStats);

    p.global_mode = hp->global_mode;
    LaunchShape ls;
    if ((err = query_launch_shape(p, &ls)) != cudaSuccess) return na_cuda(err, "occupancy query");
    GlobalScalars g{};
    g.b1 = hp->g_b1;
    g.b2 = hp->g_b2;
    g.c1 = float((1.0 - double(hp->g_b1)) / double(gamma));
    g.c2 = float((1.0 - double(hp->g_b2)) / double(gamma));
    g.eta_gamma = float(double(hp->g_eta) * double(gamma));
    g.inv_gamma = float(1.0 / double(gamma));
    g.eta = hp->g_eta;
    g.mode = hp->global_mode;
    g.B = hp->rsign_B;
    g.n_f = float(n);
    g.sign_mode = hp->sign_mode;
    g.philox_k0 = static_cast<uint32_t>(hp->seed & 0xFFFFFFFFull);
    g.philox_k1 = static_cast<uint32_t>(round & 0xFFFFFFFFull);
    g.philox_q0 = layout->first_element >> 2;
    uint32_t grid = 0;
    if ((err = launch_global(p, ls, g, s, &grid)) != cudaSuccess) return na_cuda(err, "launch global step");
    if ((err = launch_stats(p, grid, s)) != cudaSuccess) return na_cuda(err, "launch statistics");
    if (stats) {
        err = cudaMemcpyAsync(stats, p.stats, sizeof(TensorStats) * layout->count,
                              stats_is_device ? cudaMemcpyDeviceToDevice : cudaMemcpyDeviceToHost, s);
        if (err != cudaSuccess) return na_cuda(err, "copy statistics");
        if (!stats_is_device && (err = cudaStreamSynchronize(s)) != cudaSuccess)
            return na_cuda(err, "synchronise after the global step");
    }
    return DSM_OK;
}
