// The fused round's kernel (DSM_FLAG_FUSED_ROUND): the last local step of a
// round inside the global step (arXiv 2411.17866, Algorithm 1).  The kernel
// template lives here; dsm_fused_sign.cu, dsm_fused_variants.cu and
// dsm_fused_adamw.cu instantiate it for the three global-step families in
// parallel translation units, and dsm_fused.cu holds the host side.
#pragma once

#include "dsm_device.cuh"

namespace dsm {

using FusedKernel = void (*)(Problem, AdamScalars, SgdmScalars, GlobalScalars, int);
// The instantiation for p's worker count and gradient type (nullptr for n > 8), per global-step family.
FusedKernel fused_kernel_sign(const Problem& p, bool adamw);      // Algorithm 1
FusedKernel fused_kernel_variants(const Problem& p, bool adamw);  // SlowMo, signed SlowMo, Lookahead
FusedKernel fused_kernel_adamw(const Problem& p, bool adamw);     // global AdamW

namespace {


// K6: the round's last local step fused with the sign-momentum global step.
// One thread owns 4 elements of every worker: it runs the base optimizer's
// last step on each worker (writing the worker's optimizer state, but not
// its new replica, which only feeds the average), then the global step of
// Algorithm 1 on those elements.  The replicas are not reset: the next
// round's first local step starts every worker from x.  opts (kFused* bits):
// kFusedFromX, the replicas' reset from the previous round is still pending
// (tau = 1); kFusedZeroState, the base-optimizer states are zero and not read
// (the round restarts the base optimizer and tau = 1); kFusedDropState, the
// new states are not written (the round restarts the base optimizer).
// kGlobal: the global step, kGlobalSign (Algorithm 1's), kGlobalRuntime
// (g.mode: SlowMo, signed SlowMo or Lookahead, which keep x and m), or
// kGlobalAdamW (the global AdamW step, which also keeps the second moment v).
// A CTA walks its tiles worker by worker; each thread keeps the next
// kFusedDepth (tile, worker) items in flight with cp.async into its own
// shared-memory slots: x_i, m_i (v_i) and g_i per item, and x, m with a tile's
// first worker into a set of slots for the tile.
// Items in flight per thread: 2, or 3 for AdamW with more than 4 workers,
// whose registers already limit the resident CTAs (measured on GB300: depth 2
// gives 0.92 / 1.00 of the copy bandwidth on GPT-2 S (AdamW, n = 4) / L
// (SGD-momentum, n = 8), depth 3 gives 0.85 on GPT-2 M (AdamW, n = 8) where
// depth 2 gives 0.79).  Staging x and m once per tile instead of in every
// item's slots (59 instead of 72 KB per CTA for GPT-2 M) raised GPT-2 M to
// 0.87; four items in flight in the same 72 KB gave 0.86.  The x/m slots of
// tile q are set q % S: two sets (by tile parity), or one for AdamW with more
// than 4 workers (50 instead of 59 KB per CTA: GPT-2 M 0.88 against 0.87,
// where one set for n = 4 gave 0.93 / 0.94 against 0.94 / 0.95 on GPT-2 XL / S).
constexpr int kGlobalSign = 0, kGlobalRuntime = 1, kGlobalAdamW = 2;
__host__ __device__ constexpr int fused_depth(bool adamw, int nw) { return (adamw && nw > 4) ? 3 : 2; }
// Sets of x/m slots S.  A tile's set is refilled with the first item of the
// tile S tiles later, issued when the item `depth` places before that one is
// consumed; that item comes after the tile's own first item (which takes x
// and m into registers) only if depth <= S * nw.
__host__ __device__ constexpr int fused_glob_sets(bool adamw, int nw) { return (adamw && nw > 4) ? 1 : 2; }
// Staging per thread: for every item in flight the worker's x_i, m_i (and v_i
// for AdamW) in 16-byte slots and its gradient in an 8- or 16-byte slot; for
// each set, x and m (and the global v) of a tile.
__host__ __device__ constexpr int fused_states(bool adamw) { return adamw ? 3 : 2; }
__host__ __device__ constexpr int fused_globals(int global) { return global == kGlobalAdamW ? 3 : 2; }
__host__ __device__ constexpr size_t fused_smem(bool adamw, bool bf16, int nw, int global) {
    return (size_t(fused_depth(adamw, nw)) * (fused_states(adamw) * 16 + (bf16 ? 8 : 16)) +
            size_t(fused_glob_sets(adamw, nw)) * fused_globals(global) * 16) * kThreads;
}

template <bool kAdamW, bool kBf16, int NW, int kGlobal>
__global__ void __launch_bounds__(kThreads) k_fused_last_global(Problem p, AdamScalars a, SgdmScalars sa,
                                                                GlobalScalars g, int opts) {
    constexpr int kFusedDepth = fused_depth(kAdamW, NW);
    constexpr int kStates = fused_states(kAdamW), kGlobals = fused_globals(kGlobal);
    constexpr int kGradBytes = kBf16 ? 8 : 16;
    constexpr int kGlobSets = fused_glob_sets(kAdamW, NW);
    static_assert(kFusedDepth <= kGlobSets * NW, "a tile's x/m slots are refilled only after its first item");
    const bool from_global = opts & kFusedFromX, zero_state = opts & kFusedZeroState,
               keep_state = !(opts & kFusedDropState);
    // [kFusedDepth][kStates][kThreads] float4 | [kFusedDepth][kThreads] gradients | [kGlobSets][kGlobals][kThreads] float4
    extern __shared__ float4 fsm[];
    char* const grad_base = reinterpret_cast<char*>(fsm + size_t(kFusedDepth) * kStates * kThreads);
    float4* const glob_base = reinterpret_cast<float4*>(grad_base + size_t(kFusedDepth) * kThreads * kGradBytes);
    const uint32_t e0 = threadIdx.x * kElemsPerThread;
    auto state_slot = [&](uint32_t it, int s) -> float4* {
        return fsm + (size_t(it % kFusedDepth) * kStates + s) * kThreads + threadIdx.x;
    };
    auto grad_slot = [&](uint32_t it) -> void* {
        return grad_base + (size_t(it % kFusedDepth) * kThreads + threadIdx.x) * kGradBytes;
    };
    auto glob_slot = [&](uint32_t q, int s) -> float4* {
        return glob_base + (size_t(q % kGlobSets) * kGlobals + s) * kThreads + threadIdx.x;
    };
    // Issue item `it` (tile number it / NW of this CTA, worker it % NW); always commits one group.
    auto issue = [&](uint32_t it) {
        const uint32_t q = it / NW, w = it - q * NW;
        const uint64_t ti = blockIdx.x + uint64_t(q) * gridDim.x;
        if (ti < p.num_tiles) {
            const TileDesc t = p.tiles[ti];
            if (vector_ok(t, e0)) {
                const uint64_t gi = t.start + e0;
                const uint64_t o = w * p.d_stride + gi;
                if (!from_global) cp_async16(state_slot(it, 0), p.X + o);
                if (!zero_state) {
                    cp_async16(state_slot(it, 1), p.opt_m + o);
                    if (kAdamW) cp_async16(state_slot(it, 2), p.opt_v + o);
                }
                if (kBf16) cp_async8(grad_slot(it), reinterpret_cast<const __nv_bfloat16*>(p.grad) + o);
                else cp_async16(grad_slot(it), reinterpret_cast<const float*>(p.grad) + o);
                if (w == 0) {
                    cp_async16(glob_slot(q, 0), p.x + gi);
                    cp_async16(glob_slot(q, 1), p.m + gi);
                    if (kGlobal == kGlobalAdamW) cp_async16(glob_slot(q, 2), p.gv + gi);
                }
            }
        }
        cp_async_commit();
    };
    auto take = [&](const float4* src, float (&v)[4]) {
        const float4 t = *src;
        v[0] = t.x; v[1] = t.y; v[2] = t.z; v[3] = t.w;
    };
    uint32_t next_issue = 0;
    for (int k = 0; k < kFusedDepth; ++k) issue(next_issue++);
    ThreadStats st;
    uint32_t it = 0;
    for (uint32_t ti = blockIdx.x; ti < p.num_tiles; ti += gridDim.x) {
        const TileDesc td = p.tiles[ti];
        const TensorDesc& T = p.tensors[td.tensor];
        const float lam_l = kAdamW ? T.lam_local : 0.f, lam_g = T.lam_global;
        const uint64_t gi = td.start + e0;
        if (vector_ok(td, e0)) {
            float x[4], m[4], gv[4] = {0.f, 0.f, 0.f, 0.f}, dif[NW][4];
#pragma unroll
            for (int w = 0; w < NW; ++w, ++it) {
                cp_async_wait<kFusedDepth - 1>();  // item `it` has landed
                float xi[4], mi[4], vi[4], gr[4];
                if (w == 0) {
                    const uint32_t q = it / NW;
                    take(glob_slot(q, 0), x);
                    take(glob_slot(q, 1), m);
                    if (kGlobal == kGlobalAdamW) take(glob_slot(q, 2), gv);
                }
                if (from_global) {
#pragma unroll
                    for (int j = 0; j < 4; ++j) xi[j] = x[j];
                } else {
                    take(state_slot(it, 0), xi);
                }
                if (zero_state) {
#pragma unroll
                    for (int j = 0; j < 4; ++j) mi[j] = vi[j] = 0.f;
                } else {
                    take(state_slot(it, 1), mi);
                    if (kAdamW) take(state_slot(it, 2), vi);
                }
                if (kBf16) {
                    const uint2 raw = *reinterpret_cast<const uint2*>(grad_slot(it));
                    gr[0] = __uint_as_float(raw.x << 16);
                    gr[1] = __uint_as_float(raw.x & 0xFFFF0000u);
                    gr[2] = __uint_as_float(raw.y << 16);
                    gr[3] = __uint_as_float(raw.y & 0xFFFF0000u);
                } else {
                    take(reinterpret_cast<const float4*>(grad_slot(it)), gr);
                }
                const uint64_t o = w * p.d_stride + gi;
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    if (kAdamW) adamw_elem(xi[j], mi[j], vi[j], gr[j], a, lam_l);
                    else sgdm_elem(xi[j], mi[j], gr[j], sa);
                    dif[w][j] = __fsub_rn(x[j], xi[j]);
                }
                if (keep_state) {
                    store4(p.opt_m + o, mi);
                    if (kAdamW) store4(p.opt_v + o, vi);
                }
                // refill the slot just read; the arithmetic above consumed its values, so the
                // shared-memory reads are complete before the asynchronous copy can overwrite them
                issue(next_issue++);
            }
            float ru[4] = {0.f, 0.f, 0.f, 0.f};
            if (kGlobal == kGlobalSign && g.sign_mode != 0) {
                const uint4 b = philox_block((gi >> 2) + g.philox_q0, g.philox_k0, g.philox_k1);
                ru[0] = philox_unit(b.x); ru[1] = philox_unit(b.y); ru[2] = philox_unit(b.z); ru[3] = philox_unit(b.w);
            }
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                float d[NW];
#pragma unroll
                for (int w = 0; w < NW; ++w) d[w] = dif[w][j];
                if (kGlobal == kGlobalRuntime) {
                    global_elem_rt<NW>(x[j], m[j], d, g, lam_g, ru[j], st);
                } else if (kGlobal == kGlobalAdamW) {
                    global_elem<NW, 4>(x[j], m[j], gv[j], d, NW, g, lam_g, ru[j], st);
                } else {
                    float unused = 0.f;
                    global_elem<NW, 0>(x[j], m[j], unused, d, NW, g, lam_g, ru[j], st);
                }
            }
            store4(p.x + gi, x);
            store4(p.m + gi, m);
            if (kGlobal == kGlobalAdamW) store4(p.gv + gi, gv);
        } else {
            // this thread issued no copies for the tile; keep the group count in step
#pragma unroll
            for (int w = 0; w < NW; ++w, ++it) issue(next_issue++);
            const uint32_t e1 = min(e0 + kElemsPerThread, td.len);
            for (uint32_t e = e0; e < e1; ++e) {
                const uint64_t gj = td.start + e;
                float x = p.x[gj], m = p.m[gj], d[NW];
#pragma unroll
                for (int w = 0; w < NW; ++w) {
                    const uint64_t o = w * p.d_stride + gj;
                    float xi = from_global ? x : p.X[o], mi = zero_state ? 0.f : p.opt_m[o];
                    if (kAdamW) {
                        float vi = zero_state ? 0.f : p.opt_v[o];
                        adamw_elem(xi, mi, vi, load_grad1(p.grad, kBf16, o), a, lam_l);
                        if (keep_state) p.opt_v[o] = vi;
                    } else {
                        sgdm_elem(xi, mi, load_grad1(p.grad, kBf16, o), sa);
                    }
                    if (keep_state) p.opt_m[o] = mi;
                    d[w] = __fsub_rn(x, xi);
                }
                float r = 0.f;
                if (kGlobal == kGlobalSign && g.sign_mode != 0)
                    r = philox_unit(word_of(philox_block((gj >> 2) + g.philox_q0, g.philox_k0, g.philox_k1), gj & 3));
                if (kGlobal == kGlobalRuntime) {
                    global_elem_rt<NW>(x, m, d, g, lam_g, r, st);
                } else if (kGlobal == kGlobalAdamW) {
                    float v = p.gv[gj];
                    global_elem<NW, 4>(x, m, v, d, NW, g, lam_g, r, st);
                    p.gv[gj] = v;
                } else {
                    float unused = 0.f;
                    global_elem<NW, 0>(x, m, unused, d, NW, g, lam_g, r, st);
                }
                p.x[gj] = x;
                p.m[gj] = m;
            }
        }
        const uint32_t next = ti + gridDim.x;
        if (next >= p.num_tiles || p.tiles[next].tensor != td.tensor) {  // uniform across the CTA
            reduce_stats(st, p.partials + ti);  // a CTA's last tile of this tensor (as in K4)
            st = ThreadStats();
        }
    }
    cp_async_wait<0>();  // the groups issued past the last tile are empty; nothing is left in flight
}

template <bool kAdamW, bool kBf16, int kGlobal>
FusedKernel fused_kernel_n(uint32_t n) {
    switch (n) {
        case 1: return k_fused_last_global<kAdamW, kBf16, 1, kGlobal>;
        case 2: return k_fused_last_global<kAdamW, kBf16, 2, kGlobal>;
        case 3: return k_fused_last_global<kAdamW, kBf16, 3, kGlobal>;
        case 4: return k_fused_last_global<kAdamW, kBf16, 4, kGlobal>;
        case 5: return k_fused_last_global<kAdamW, kBf16, 5, kGlobal>;
        case 6: return k_fused_last_global<kAdamW, kBf16, 6, kGlobal>;
        case 7: return k_fused_last_global<kAdamW, kBf16, 7, kGlobal>;
        case 8: return k_fused_last_global<kAdamW, kBf16, 8, kGlobal>;
        default: return nullptr;
    }
}

template <int kGlobal>
FusedKernel fused_kernel_v(const Problem& p, bool adamw) {
    if (adamw) return p.grad_bf16 ? fused_kernel_n<true, true, kGlobal>(p.n) : fused_kernel_n<true, false, kGlobal>(p.n);
    return p.grad_bf16 ? fused_kernel_n<false, true, kGlobal>(p.n) : fused_kernel_n<false, false, kGlobal>(p.n);
}

}  // namespace
}  // namespace dsm
