// The local steps of one global round (arXiv 2411.17866, Eq. (local-steps)):
// K2, one AdamW step, and K3, one SGD-momentum step (Appendix A), on every
// worker's replica.  Persistent grid-stride kernels over (worker, tile)
// items of 4 elements per thread, double-buffered in registers (see
// dsm_kernels.cu for the common design).

#include <algorithm>

#include "dsm_device.cuh"

namespace dsm {
namespace {

// Where a local-step work item (worker w, tile) lives.  Items are worker-major
// (all tiles of worker 0, then worker 1, ...), or tile-major when the step
// starts every worker from the global x (the workers of one tile then run
// together and read that tile of x once from HBM).
struct LocalItem {
    uint64_t base;   // w * d_stride + tile start
    uint64_t start;  // tile start (offset in x)
    uint32_t len;
    float lam;
    bool vec;
};

// A CTA's walk over the items: the (worker, tile) position of its current item, advanced by the grid
// stride with one precomputed quotient and remainder instead of a division per item (the division by
// the runtime tile count cost 0.4-0.7% of the local step on GPT-2 M and XL).
template <bool kTileMajor>
struct ItemWalk {
    uint32_t w, ti;        // position of the current item
    uint32_t dq, dr;       // the stride as whole rows (tiles, or workers) and a remainder
    __device__ __forceinline__ ItemWalk(const Problem& p, uint32_t item, uint32_t stride) {
        const uint32_t row = kTileMajor ? p.n : p.num_tiles;  // items per row of the order
        const uint32_t q = item / row, r = item - q * row;
        if (kTileMajor) { ti = q; w = r; } else { w = q; ti = r; }
        dq = stride / row;
        dr = stride - dq * row;
    }
    __device__ __forceinline__ void advance(const Problem& p) {
        if (kTileMajor) {
            ti += dq;
            w += dr;
            if (w >= p.n) { w -= p.n; ++ti; }
        } else {
            w += dq;
            ti += dr;
            if (ti >= p.num_tiles) { ti -= p.num_tiles; ++w; }
        }
    }
};

__device__ __forceinline__ LocalItem local_item(const Problem& p, uint32_t w, uint32_t ti, uint32_t e0,
                                                bool local_lam) {
    const TileDesc td = p.tiles[ti];
    LocalItem it;
    it.base = w * p.d_stride + td.start;
    it.start = td.start;
    it.len = td.len;
    it.lam = local_lam ? p.tensors[td.tensor].lam_local : 0.f;
    it.vec = vector_ok(td, e0);
    return it;
}

// K2: one AdamW local step on every worker (work item = (worker, tile)),
// double-buffered in registers.  kFromGlobal: every worker starts from the
// global x (the replicas' reset is still pending).  kZeroState: the moments
// are zero (the round restarts the base optimizer) and are not read.
template <bool kBf16, bool kFromGlobal, bool kZeroState>
__global__ void __launch_bounds__(kThreads) k_local_adamw(Problem p, AdamScalars a) {
    const uint32_t items = p.num_tiles * p.n;
    const uint32_t e0 = threadIdx.x * kElemsPerThread;
    uint32_t item = blockIdx.x;
    if (item >= items) return;
    ItemWalk<kFromGlobal> walk(p, item, gridDim.x);
    LocalItem nx = local_item(p, walk.w, walk.ti, e0, true);
    float x[4], m[4] = {0.f, 0.f, 0.f, 0.f}, v[4] = {0.f, 0.f, 0.f, 0.f}, g[4];
    if (nx.vec) {
        load4(kFromGlobal ? p.x + nx.start + e0 : p.X + nx.base + e0, x);
        if (!kZeroState) {
            load4(p.opt_m + nx.base + e0, m);
            load4(p.opt_v + nx.base + e0, v);
        }
        load4_grad<kBf16>(p.grad, nx.base + e0, g);
    }
    for (; item < items; item += gridDim.x) {
        const LocalItem cur = nx;
        float cx[4], cm[4], cv[4], cg[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) { cx[j] = x[j]; cm[j] = m[j]; cv[j] = v[j]; cg[j] = g[j]; }
        const uint32_t next = item + gridDim.x;
        if (next < items) {  // issue the next item's loads before computing this one
            walk.advance(p);
            nx = local_item(p, walk.w, walk.ti, e0, true);
            if (nx.vec) {
                load4(kFromGlobal ? p.x + nx.start + e0 : p.X + nx.base + e0, x);
                if (!kZeroState) {
                    load4(p.opt_m + nx.base + e0, m);
                    load4(p.opt_v + nx.base + e0, v);
                }
                load4_grad<kBf16>(p.grad, nx.base + e0, g);
            }
        }
        if (cur.vec) {
#pragma unroll
            for (int j = 0; j < 4; ++j) adamw_elem(cx[j], cm[j], cv[j], cg[j], a, cur.lam);
            store4(p.X + cur.base + e0, cx);
            store4(p.opt_m + cur.base + e0, cm);
            store4(p.opt_v + cur.base + e0, cv);
        } else {
            const uint32_t e1 = min(e0 + kElemsPerThread, cur.len);
            for (uint32_t e = e0; e < e1; ++e) {
                const uint64_t i = cur.base + e;
                float xs = kFromGlobal ? p.x[cur.start + e] : p.X[i];
                float ms = kZeroState ? 0.f : p.opt_m[i], vs = kZeroState ? 0.f : p.opt_v[i];
                adamw_elem(xs, ms, vs, load_grad1(p.grad, kBf16, i), a, cur.lam);
                p.X[i] = xs; p.opt_m[i] = ms; p.opt_v[i] = vs;
            }
        }
    }
}

// K3: one SGD-momentum local step on every worker, double-buffered.
// kFromGlobal, kZeroState: as for K2 (the buffer is zero and not read).
template <bool kBf16, bool kFromGlobal, bool kZeroState>
__global__ void __launch_bounds__(kThreads) k_local_sgdm(Problem p, SgdmScalars a) {
    const uint32_t items = p.num_tiles * p.n;
    const uint32_t e0 = threadIdx.x * kElemsPerThread;
    uint32_t item = blockIdx.x;
    if (item >= items) return;
    ItemWalk<kFromGlobal> walk(p, item, gridDim.x);
    LocalItem nx = local_item(p, walk.w, walk.ti, e0, false);
    float x[4], b[4] = {0.f, 0.f, 0.f, 0.f}, g[4];
    if (nx.vec) {
        load4(kFromGlobal ? p.x + nx.start + e0 : p.X + nx.base + e0, x);
        if (!kZeroState) load4(p.opt_m + nx.base + e0, b);
        load4_grad<kBf16>(p.grad, nx.base + e0, g);
    }
    for (; item < items; item += gridDim.x) {
        const LocalItem cur = nx;
        float cx[4], cb[4], cg[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) { cx[j] = x[j]; cb[j] = b[j]; cg[j] = g[j]; }
        const uint32_t next = item + gridDim.x;
        if (next < items) {
            walk.advance(p);
            nx = local_item(p, walk.w, walk.ti, e0, false);
            if (nx.vec) {
                load4(kFromGlobal ? p.x + nx.start + e0 : p.X + nx.base + e0, x);
                if (!kZeroState) load4(p.opt_m + nx.base + e0, b);
                load4_grad<kBf16>(p.grad, nx.base + e0, g);
            }
        }
        if (cur.vec) {
#pragma unroll
            for (int j = 0; j < 4; ++j) sgdm_elem(cx[j], cb[j], cg[j], a);
            store4(p.X + cur.base + e0, cx);
            store4(p.opt_m + cur.base + e0, cb);
        } else {
            const uint32_t e1 = min(e0 + kElemsPerThread, cur.len);
            for (uint32_t e = e0; e < e1; ++e) {
                const uint64_t i = cur.base + e;
                float xs = kFromGlobal ? p.x[cur.start + e] : p.X[i], bs = kZeroState ? 0.f : p.opt_m[i];
                sgdm_elem(xs, bs, load_grad1(p.grad, kBf16, i), a);
                p.X[i] = xs; p.opt_m[i] = bs;
            }
        }
    }
}

}  // namespace

cudaError_t query_local_shape(const Problem& p, LaunchShape* out) {
    const int sms = out->sms;
    // The AdamW step fits 4 CTAs per SM.  With fp32 gradients it streams better with 3 (GB300, GPT-2 S,
    // n = 4: 1.00 of the copy bandwidth with 3, 0.95 with 4); with bf16 gradients 4 are better
    // (GPT-2 M, n = 8: 0.97 with 4, 0.90 with 3; GPT-2 XL, n = 4: 0.96 with 4, 0.87 with 3).
    const int kAdamwCtasPerSm = p.grad_bf16 ? 4 : 3;
    out->grid_adamw = std::min(p.grad_bf16 ? grid_for(k_local_adamw<true, false, false>, sms)
                                           : grid_for(k_local_adamw<false, false, false>, sms), kAdamwCtasPerSm * sms);
    // The SGD-momentum step fits 6 CTAs per SM, but 4 stream better (GB300, GPT-2 L layout, n = 8:
    // 0.96 of the copy bandwidth with 4, 0.91 with 6, 0.91 with 3), as many as the AdamW step holds.
    constexpr int kSgdmCtasPerSm = 4;
    out->grid_sgdm = std::min(p.grad_bf16 ? grid_for(k_local_sgdm<true, false, false>, sms)
                                          : grid_for(k_local_sgdm<false, false, false>, sms), kSgdmCtasPerSm * sms);
    {  // the from-x variants (first local step after a lazy reset)
        out->grid_adamw_from_x = std::min(p.grad_bf16 ? grid_for(k_local_adamw<true, true, false>, sms)
                                                      : grid_for(k_local_adamw<false, true, false>, sms),
                                          kAdamwCtasPerSm * sms);
        out->grid_sgdm_from_x = std::min(p.grad_bf16 ? grid_for(k_local_sgdm<true, true, false>, sms)
                                                     : grid_for(k_local_sgdm<false, true, false>, sms),
                                         kSgdmCtasPerSm * sms);
    }
    return cudaGetLastError();
}

// The kernel instantiation for (gradient type, from x, zero state).
using AdamwKernel = void (*)(Problem, AdamScalars);
using SgdmKernel = void (*)(Problem, SgdmScalars);

static AdamwKernel adamw_kernel_for(bool bf16, bool from_x, bool zero_state) {
    if (bf16) {
        if (from_x) return zero_state ? k_local_adamw<true, true, true> : k_local_adamw<true, true, false>;
        return zero_state ? k_local_adamw<true, false, true> : k_local_adamw<true, false, false>;
    }
    if (from_x) return zero_state ? k_local_adamw<false, true, true> : k_local_adamw<false, true, false>;
    return zero_state ? k_local_adamw<false, false, true> : k_local_adamw<false, false, false>;
}

static SgdmKernel sgdm_kernel_for(bool bf16, bool from_x, bool zero_state) {
    if (bf16) {
        if (from_x) return zero_state ? k_local_sgdm<true, true, true> : k_local_sgdm<true, true, false>;
        return zero_state ? k_local_sgdm<true, false, true> : k_local_sgdm<true, false, false>;
    }
    if (from_x) return zero_state ? k_local_sgdm<false, true, true> : k_local_sgdm<false, true, false>;
    return zero_state ? k_local_sgdm<false, false, true> : k_local_sgdm<false, false, false>;
}

cudaError_t launch_local_adamw(const Problem& p, const LaunchShape& ls, const AdamScalars& a, bool from_x,
                               bool zero_state, cudaStream_t s) {
    const uint64_t items = static_cast<uint64_t>(p.num_tiles) * p.n;
    // the zero-state variants read less and use the grids of the state-reading ones
    const int grid = clamp_grid(from_x ? ls.grid_adamw_from_x : ls.grid_adamw, items);
    if (grid == 0) return cudaSuccess;
    adamw_kernel_for(p.grad_bf16, from_x, zero_state)<<<grid, kThreads, 0, s>>>(p, a);
    return cudaGetLastError();
}

cudaError_t launch_local_sgdm(const Problem& p, const LaunchShape& ls, const SgdmScalars& a, bool from_x,
                              bool zero_state, cudaStream_t s) {
    const uint64_t items = static_cast<uint64_t>(p.num_tiles) * p.n;
    const int grid = clamp_grid(from_x ? ls.grid_sgdm_from_x : ls.grid_sgdm, items);
    if (grid == 0) return cudaSuccess;
    sgdm_kernel_for(p.grad_bf16, from_x, zero_state)<<<grid, kThreads, 0, s>>>(p, a);
    return cudaGetLastError();
}

}  // namespace dsm
