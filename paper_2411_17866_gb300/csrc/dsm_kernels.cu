// CUDA kernels (sm_103a) for one global round of distributed sign momentum
// with local steps (arXiv 2411.17866, Algorithm 1): initialisation, the
// synthetic gradients (K1), the global step (K4) and its statistics (K5).
// The local steps are in dsm_local.cu, the fused round in dsm_fused.cuh.
//
// Every kernel is a persistent, grid-stride loop over work items: tiles of
// at most kTile = 1024 elements that lie inside one tensor (for the local
// steps, a tile of one worker).  A CTA of 256 threads takes one item at a
// time; each thread owns 4 consecutive elements and moves them with one
// 16-byte load or store per fp32 stream (8 bytes per bf16 stream), so every
// warp instruction covers 512 contiguous bytes.  (K1 instead runs 64-thread
// CTAs whose threads own four such groups of a tile.)  The local and global
// steps double-buffer in registers: a thread issues the loads of its next
// item before it computes the current one, so the HBM requests of one item
// are in flight during the arithmetic of the previous one.  The work is streaming and
// elementwise, bound by HBM bandwidth; nothing is a contraction, and no tensor
// core is used.
//
// All method arithmetic uses the explicit round-to-nearest intrinsics
// (__fadd_rn, __fmul_rn, __fdiv_rn, __fsqrt_rn, ...), which the compiler
// never contracts into FMAs, so each result is the fp32 value of the
// paper's expression evaluated one operation at a time.

#include <algorithm>
#include <type_traits>

#include "dsm_device.cuh"

namespace dsm {
namespace {

// ---------------------------------------------------------------------------
// Kernels
// ---------------------------------------------------------------------------

// Initial state: x (hash init by tensor kind, or as already copied) and every replica = x.
__global__ void __launch_bounds__(kThreads) k_init(Problem p, uint64_t key_init, int from_hash) {
    for (uint32_t ti = blockIdx.x; ti < p.num_tiles; ti += gridDim.x) {
        const TileDesc td = p.tiles[ti];
        const uint32_t kind = p.tensors[td.tensor].kind;
        const uint32_t e0 = threadIdx.x * kElemsPerThread;
        const uint32_t e1 = min(e0 + kElemsPerThread, td.len);
        for (uint32_t e = e0; e < e1; ++e) {
            const uint64_t gi = td.start + e;
            float v;
            if (from_hash) {
                if (kind == 0) {
                    const float u = hash_uniform(key_init, gi);
                    v = __fmul_rn(0.02f, __fsub_rn(__fmul_rn(2.0f, u), 1.0f));
                } else {
                    v = (kind == 2) ? 1.0f : 0.0f;
                }
                p.x[gi] = v;
            } else {
                v = p.x[gi];
            }
            for (uint32_t w = 0; w < p.n; ++w) p.X[w * p.d_stride + gi] = v;
        }
    }
}

// K1: synthetic gradients of one local step for every worker.  Bound by the
// integer work of the hash (one 64-bit SplitMix64 output per two elements
// and per draw family), not by its write stream.  A CTA of kFillThreads
// threads fills one tile; a thread owns kFillGroups groups of 4 elements
// (group q at 4*thread + q*4*kFillThreads), so it carries 2*kFillGroups
// independent hash chains per family, and every warp store covers 512
// contiguous bytes of fp32 (256 of bf16).
constexpr uint32_t kFillThreads = 64;
constexpr uint32_t kFillGroups = kTile / (4 * kFillThreads);  // 4

// Output j of any family is finalise(key + j*gamma); the j*gamma of a
// group (j = e/2 + 1 and e/2 + 2 for its even first element e) is shared by
// the step family and every worker family.
template <bool kBf16, bool kPrescaled, int kGroups, uint32_t kGroupStride>
__device__ __forceinline__ void grad_fill_groups(const Problem& p, const GradKeys& k, uint64_t gi0, float s,
                                                 float s2) {
    uint64_t jg0[kGroups], jg1[kGroups];
    float a[kGroups][4];
#pragma unroll
    for (int q = 0; q < kGroups; ++q) {
        const uint64_t gi = gi0 + q * kGroupStride;
        jg0[q] = ((gi >> 1) + 1) * kGoldenGamma;
        jg1[q] = jg0[q] + kGoldenGamma;
        const uint64_t h0 = sm64_finalise(k.step + jg0[q]), h1 = sm64_finalise(k.step + jg1[q]);
        if (kPrescaled) {
            a[q][0] = __fmul_rn(s, centred_even(h0)); a[q][1] = __fmul_rn(s, centred_odd(h0));
            a[q][2] = __fmul_rn(s, centred_even(h1)); a[q][3] = __fmul_rn(s, centred_odd(h1));
        } else {
            a[q][0] = step_term(s, draw_even(h0)); a[q][1] = step_term(s, draw_odd(h0));
            a[q][2] = step_term(s, draw_even(h1)); a[q][3] = step_term(s, draw_odd(h1));
        }
    }
    using Elem = typename std::conditional<kBf16, __nv_bfloat16, float>::type;
    Elem* out = reinterpret_cast<Elem*>(p.grad) + gi0;
    for (uint32_t w = 0; w < p.n; ++w, out += p.d_stride) {
#pragma unroll
        for (int q = 0; q < kGroups; ++q) {
            const uint64_t q0 = sm64_finalise(k.worker[w] + jg0[q]), q1 = sm64_finalise(k.worker[w] + jg1[q]);
            float g[4];
            if (kPrescaled) {
                g[0] = __fadd_rn(a[q][0], __fmul_rn(s2, centred_even(q0)));
                g[1] = __fadd_rn(a[q][1], __fmul_rn(s2, centred_odd(q0)));
                g[2] = __fadd_rn(a[q][2], __fmul_rn(s2, centred_even(q1)));
                g[3] = __fadd_rn(a[q][3], __fmul_rn(s2, centred_odd(q1)));
            } else {
                g[0] = grad_value(a[q][0], s2, draw_even(q0)); g[1] = grad_value(a[q][1], s2, draw_odd(q0));
                g[2] = grad_value(a[q][2], s2, draw_even(q1)); g[3] = grad_value(a[q][3], s2, draw_odd(q1));
            }
            if (kBf16) store4_bf16(reinterpret_cast<__nv_bfloat16*>(out) + q * kGroupStride, g);
            else store4(reinterpret_cast<float*>(out) + q * kGroupStride, g);
        }
    }
}

// Element-by-element fill (tile starts that are not 4-aligned, ragged tails).
template <bool kBf16>
__device__ __forceinline__ void grad_fill_elem(const Problem& p, const GradKeys& k, uint64_t gi, float s, float s2) {
    const float a = step_term(s, hash_uniform(k.step, gi));
    for (uint32_t w = 0; w < p.n; ++w) {
        const float g = grad_value(a, s2, hash_uniform(k.worker[w], gi));
        const uint64_t o = w * p.d_stride + gi;
        if (kBf16) reinterpret_cast<__nv_bfloat16*>(p.grad)[o] = __float2bfloat16_rn(g);
        else reinterpret_cast<float*>(p.grad)[o] = g;
    }
}

template <bool kBf16>
__global__ void __launch_bounds__(kFillThreads) k_grad_fill(Problem p, GradKeys k) {
    constexpr uint32_t kStride = 4 * kFillThreads;  // elements between a thread's groups
    for (uint32_t ti = blockIdx.x; ti < p.num_tiles; ti += gridDim.x) {
        const TileDesc td = p.tiles[ti];
        const TensorDesc& T = p.tensors[td.tensor];
        const float s = T.scale, s2 = T.scale2;
        // one multiplication per draw where both scales allow it (see centred_even)
        const bool pre = fabsf(s) >= kMinPrescaled && fabsf(s2) >= kMinPrescaled;
        const float sp = __fmul_rn(s, kTwoPowM24), sp2 = __fmul_rn(s2, kTwoPowM24);
        const bool aligned = (td.start & 3u) == 0;
        if (aligned && td.len == kTile) {  // a full tile (uniform across the CTA)
            const uint64_t gi0 = td.start + threadIdx.x * 4;
            if (pre) grad_fill_groups<kBf16, true, kFillGroups, kStride>(p, k, gi0, sp, sp2);
            else grad_fill_groups<kBf16, false, kFillGroups, kStride>(p, k, gi0, s, s2);
            continue;
        }
        for (uint32_t e0 = threadIdx.x * 4; e0 < td.len; e0 += kStride) {  // a ragged tile, group by group
            if (aligned && e0 + 4 <= td.len) {
                if (pre) grad_fill_groups<kBf16, true, 1, kStride>(p, k, td.start + e0, sp, sp2);
                else grad_fill_groups<kBf16, false, 1, kStride>(p, k, td.start + e0, s, s2);
            } else {
                const uint32_t e1 = min(e0 + 4u, td.len);
                for (uint32_t e = e0; e < e1; ++e) grad_fill_elem<kBf16>(p, k, td.start + e, s, s2);
            }
        }
    }
}

// Global step on one element, any number of workers, reading each replica
// once for the average and once more for the statistics.
template <int MODE>
__device__ __forceinline__ void global_elem_generic(const Problem& p, const GlobalScalars& g, float lam,
                                                    uint64_t gi, ThreadStats& st) {
    float x = p.x[gi], m = p.m[gi], v = MODE == 4 ? p.gv[gi] : 0.f;
    const float x0 = x;
    float r = 0.f;
    if (MODE == 0 && g.sign_mode != 0)
        r = philox_unit(word_of(philox_block((gi >> 2) + g.philox_q0, g.philox_k0, g.philox_k1), gi & 3));
    float acc = 0.f;
    for (uint32_t i = 0; i < p.n; ++i) acc = __fadd_rn(acc, __fsub_rn(x0, p.X[i * p.d_stride + gi]));
    const float D = __fdiv_rn(acc, g.n_f);
    float u, s;
    global_update<MODE>(D, x, m, v, g, lam, r, u, s);
    const int sD = sgn(D);
    float dr = 0.f;
    bool unan = true;
    for (uint32_t i = 0; i < p.n; ++i) {
        const float di = __fsub_rn(x0, p.X[i * p.d_stride + gi]);
        const float ei = __fsub_rn(di, D);
        dr = __fadd_rn(dr, __fmul_rn(ei, ei));
        unan = unan && (sgn(di) == sD);
    }
    csum_add(st.dsq, __fmul_rn(D, D));
    csum_add(st.drift, dr);
    st.zero += (s == 0.f);
    st.flips += (sgn(u) != sD);
    st.unanimous += unan;
    st.clamped += (MODE == 0 && g.sign_mode != 0 && fabsf(u) > g.B);
    p.x[gi] = x;
    p.m[gi] = m;
    if (MODE == 4) p.gv[gi] = v;
    if (!g.skip_reset)
        for (uint32_t i = 0; i < p.n; ++i) p.X[i * p.d_stride + gi] = x;
}

// Global step on a thread's 4 aligned elements for any number of workers:
// 16-byte accesses, the replicas read once for the average and once more
// (from L2) for the statistics, then overwritten by the reset.
template <int MODE>
__device__ __forceinline__ void global_vec_generic(const Problem& p, const GlobalScalars& g, float lam,
                                                   uint64_t gi, ThreadStats& st) {
    float x[4], m[4], v[4] = {0.f, 0.f, 0.f, 0.f}, acc[4] = {0.f, 0.f, 0.f, 0.f};
    load4(p.x + gi, x);
    load4(p.m + gi, m);
    if (MODE == 4) load4(p.gv + gi, v);
    // pass 1: the average; the loads of up to kGenChunk workers are issued before their additions,
    // which stay in worker order (kept in L2 for pass 2)
    constexpr uint32_t kGenChunk = 8;
    for (uint32_t i0 = 0; i0 < p.n; i0 += kGenChunk) {
        float4 r[kGenChunk];
#pragma unroll
        for (uint32_t c = 0; c < kGenChunk; ++c)
            if (i0 + c < p.n) r[c] = *reinterpret_cast<const float4*>(p.X + (i0 + c) * p.d_stride + gi);
#pragma unroll
        for (uint32_t c = 0; c < kGenChunk; ++c) {
            if (i0 + c < p.n) {
                acc[0] = __fadd_rn(acc[0], __fsub_rn(x[0], r[c].x));
                acc[1] = __fadd_rn(acc[1], __fsub_rn(x[1], r[c].y));
                acc[2] = __fadd_rn(acc[2], __fsub_rn(x[2], r[c].z));
                acc[3] = __fadd_rn(acc[3], __fsub_rn(x[3], r[c].w));
            }
        }
    }
    float ru[4] = {0.f, 0.f, 0.f, 0.f};
    if (MODE == 0 && g.sign_mode != 0) {
        const uint4 b = philox_block((gi >> 2) + g.philox_q0, g.philox_k0, g.philox_k1);
        ru[0] = philox_unit(b.x); ru[1] = philox_unit(b.y); ru[2] = philox_unit(b.z); ru[3] = philox_unit(b.w);
    }
    float D[4], xn[4], dr[4] = {0.f, 0.f, 0.f, 0.f};
    int sD[4];
    bool unan[4] = {true, true, true, true};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        D[j] = __fdiv_rn(acc[j], g.n_f);
        sD[j] = sgn(D[j]);
        xn[j] = x[j];
        float u, s;
        global_update<MODE>(D[j], xn[j], m[j], v[j], g, lam, ru[j], u, s);
        st.zero += (s == 0.f);
        st.flips += (sgn(u) != sD[j]);
        st.clamped += (MODE == 0 && g.sign_mode != 0 && fabsf(u) > g.B);
        csum_add(st.dsq, __fmul_rn(D[j], D[j]));
    }
    // pass 2: the statistics and the reset, again kGenChunk workers' loads at a time
    for (uint32_t i0 = 0; i0 < p.n; i0 += kGenChunk) {
        float4 r[kGenChunk];
#pragma unroll
        for (uint32_t c = 0; c < kGenChunk; ++c)
            if (i0 + c < p.n) r[c] = __ldcs(reinterpret_cast<const float4*>(p.X + (i0 + c) * p.d_stride + gi));
#pragma unroll
        for (uint32_t c = 0; c < kGenChunk; ++c) {
            if (i0 + c < p.n) {
                const float rr[4] = {r[c].x, r[c].y, r[c].z, r[c].w};
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const float di = __fsub_rn(x[j], rr[j]);
                    const float ei = __fsub_rn(di, D[j]);
                    dr[j] = __fadd_rn(dr[j], __fmul_rn(ei, ei));
                    unan[j] = unan[j] && (sgn(di) == sD[j]);
                }
                if (!g.skip_reset) store4(p.X + (i0 + c) * p.d_stride + gi, xn);
            }
        }
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        csum_add(st.drift, dr[j]);
        st.unanimous += unan[j];
    }
    store4(p.x + gi, xn);
    store4(p.m + gi, m);
    if (MODE == 4) store4(p.gv + gi, v);
}

// K4: the fused global step (average over the replicas, sign-momentum update,
// momentum update, reset of every replica unless g.skip_reset) with statistics.
// NW > 0: exactly NW replicas, held in registers and double-buffered.
// NW == 0: any n, one element at a time.
// Statistics: a CTA keeps per-thread sums while its successive tiles belong
// to one tensor and reduces them only when the tensor changes (or at its last
// tile), writing the segment's partial at the segment's last tile.  With a
// grid of G CTAs, tile t is a CTA's last tile of its tensor exactly when
// t + G lies beyond the tensor, so the partials of a tensor are its last
// min(G, tiles) tiles, which K5 sums.
template <int NW, int MODE>
__global__ void __launch_bounds__(kThreads) k_global(Problem p, GlobalScalars g) {
    const uint32_t e0 = threadIdx.x * kElemsPerThread;
    constexpr int W = NW > 0 ? NW : 1;
    uint32_t ti = blockIdx.x;
    if (ti >= p.num_tiles) return;
    TileDesc nt = p.tiles[ti];
    bool nvec = NW > 0 && vector_ok(nt, e0);
    float x[4], m[4], v[4] = {0.f, 0.f, 0.f, 0.f}, r[W][4];
    ThreadStats st;
    if (nvec) {
        load4(p.x + nt.start + e0, x);
        load4(p.m + nt.start + e0, m);
        if (MODE == 4) load4(p.gv + nt.start + e0, v);
#pragma unroll
        for (int i = 0; i < W; ++i) load4(p.X + i * p.d_stride + nt.start + e0, r[i]);
    }
    for (; ti < p.num_tiles; ti += gridDim.x) {
        const TileDesc td = nt;
        const bool vec = nvec;
        float cx[4], cm[4], cv[4], cr[W][4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            cx[j] = x[j];
            cm[j] = m[j];
            cv[j] = v[j];
#pragma unroll
            for (int i = 0; i < W; ++i) cr[i][j] = r[i][j];
        }
        const uint32_t next = ti + gridDim.x;
        if (next < p.num_tiles) {
            nt = p.tiles[next];
            nvec = NW > 0 && vector_ok(nt, e0);
            if (nvec) {
                load4(p.x + nt.start + e0, x);
                load4(p.m + nt.start + e0, m);
                if (MODE == 4) load4(p.gv + nt.start + e0, v);
#pragma unroll
                for (int i = 0; i < W; ++i) load4(p.X + i * p.d_stride + nt.start + e0, r[i]);
            }
        }
        const float lam = p.tensors[td.tensor].lam_global;
        if (vec) {
            const uint64_t gi = td.start + e0;  // a multiple of 4: the four words of one Philox block
            float ru[4] = {0.f, 0.f, 0.f, 0.f};
            if (MODE == 0 && g.sign_mode != 0) {
                const uint4 b = philox_block((gi >> 2) + g.philox_q0, g.philox_k0, g.philox_k1);
                ru[0] = philox_unit(b.x); ru[1] = philox_unit(b.y); ru[2] = philox_unit(b.z); ru[3] = philox_unit(b.w);
            }
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                float dif[W];
#pragma unroll
                for (int i = 0; i < W; ++i) dif[i] = __fsub_rn(cx[j], cr[i][j]);
                global_elem<W, MODE>(cx[j], cm[j], cv[j], dif, W, g, lam, ru[j], st);
            }
            store4(p.x + gi, cx);
            store4(p.m + gi, cm);
            if (MODE == 4) store4(p.gv + gi, cv);
            if (!g.skip_reset) {
#pragma unroll
                for (int i = 0; i < W; ++i) store4(p.X + i * p.d_stride + gi, cx);
            }
        } else if (NW == 0 && vector_ok(td, e0)) {
            global_vec_generic<MODE>(p, g, lam, td.start + e0, st);
        } else {
            const uint32_t e1 = min(e0 + kElemsPerThread, td.len);
            for (uint32_t e = e0; e < e1; ++e) global_elem_generic<MODE>(p, g, lam, td.start + e, st);
        }
        if (next >= p.num_tiles || nt.tensor != td.tensor) {  // uniform across the CTA
            reduce_stats(st, p.partials + ti);
            st = ThreadStats();
        }
    }
}

// K5: per-tensor statistics from the tile partials, in a fixed order: a
// tensor's partials are its last min(G, tiles) tiles for a producing grid of
// G CTAs (see K4).
__global__ void __launch_bounds__(kThreads) k_stats(Problem p, uint32_t producer_grid) {
    const uint32_t T = blockIdx.x;
    const TensorDesc td = p.tensors[T];
    double a = 0.0, b = 0.0;
    unsigned long long c0 = 0, c1 = 0, c2 = 0, c3 = 0;
    const uint32_t first =
        td.tile_end - td.tile_begin > producer_grid ? td.tile_end - producer_grid : td.tile_begin;
    // each thread sums partials first + tid, first + tid + 256, ...; the loads of up to 4 of them are
    // issued before their additions (a tensor has at most producer_grid partials)
    for (uint32_t t0 = first + threadIdx.x; t0 < td.tile_end; t0 += 4 * kThreads) {
        StatPartial q[4];
#pragma unroll
        for (int u = 0; u < 4; ++u)
            if (t0 + u * kThreads < td.tile_end) q[u] = p.partials[t0 + u * kThreads];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            if (t0 + u * kThreads < td.tile_end) {
                a += q[u].delta_sq; b += q[u].drift;
                c0 += q[u].zero_sign; c1 += q[u].flips; c2 += q[u].unanimous; c3 += q[u].clamped;
            }
        }
    }
    // the lanes of each warp by shuffles in a fixed pattern, then the warps in order
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
        a += __shfl_down_sync(0xffffffffu, a, off);
        b += __shfl_down_sync(0xffffffffu, b, off);
        c0 += __shfl_down_sync(0xffffffffu, c0, off);
        c1 += __shfl_down_sync(0xffffffffu, c1, off);
        c2 += __shfl_down_sync(0xffffffffu, c2, off);
        c3 += __shfl_down_sync(0xffffffffu, c3, off);
    }
    __shared__ double s_d[kThreads / 32][2];
    __shared__ unsigned long long s_c[kThreads / 32][4];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) {
        s_d[warp][0] = a; s_d[warp][1] = b;
        s_c[warp][0] = c0; s_c[warp][1] = c1; s_c[warp][2] = c2; s_c[warp][3] = c3;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        TensorStats o;
        o.delta_sq = 0.0; o.drift = 0.0;
        o.zero_sign = o.flips = o.unanimous = o.clamped = 0;
        for (int w = 0; w < kThreads / 32; ++w) {
            o.delta_sq += s_d[w][0]; o.drift += s_d[w][1];
            o.zero_sign += s_c[w][0]; o.flips += s_c[w][1]; o.unanimous += s_c[w][2]; o.clamped += s_c[w][3];
        }
        p.stats[T] = o;
    }
}

using GlobalKernel = void (*)(Problem, GlobalScalars);

template <int MODE>
GlobalKernel global_kernel_mode(uint32_t n) {
    switch (n) {
        case 1: return k_global<1, MODE>;
        case 2: return k_global<2, MODE>;
        case 3: return k_global<3, MODE>;
        case 4: return k_global<4, MODE>;
        case 5: return k_global<5, MODE>;
        case 6: return k_global<6, MODE>;
        case 7: return k_global<7, MODE>;
        case 8: return k_global<8, MODE>;
        default: return k_global<0, MODE>;
    }
}

GlobalKernel global_kernel_for(uint32_t n, int mode) {
    switch (mode) {
        case 1: return global_kernel_mode<1>(n);
        case 2: return global_kernel_mode<2>(n);
        case 3: return global_kernel_mode<3>(n);
        case 4: return global_kernel_mode<4>(n);
        default: return global_kernel_mode<0>(n);
    }
}

}  // namespace

cudaError_t query_launch_shape(const Problem& p, LaunchShape* out) {
    int dev = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err != cudaSuccess) return err;
    int sms = 0;
    err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (err != cudaSuccess) return err;
    out->sms = sms;
    out->grid_init = grid_for(k_init, sms);
    out->grid_grad = p.grad_bf16 ? grid_for(k_grad_fill<true>, sms, 0, kFillThreads)
                                 : grid_for(k_grad_fill<false>, sms, 0, kFillThreads);
    cudaError_t e = query_local_shape(p, out);
    if (e != cudaSuccess) return e;
    if (fused_round_available(p) && (e = query_fused_shape(p, out)) != cudaSuccess) return e;
    out->grid_global = grid_for(global_kernel_for(p.n, p.global_mode), sms);
    return cudaGetLastError();
}

cudaError_t launch_init(const Problem& p, const LaunchShape& ls, uint64_t key_init, int from_hash, cudaStream_t s) {
    const int grid = clamp_grid(ls.grid_init, p.num_tiles);
    if (grid == 0) return cudaSuccess;
    k_init<<<grid, kThreads, 0, s>>>(p, key_init, from_hash);
    return cudaGetLastError();
}

cudaError_t launch_grad_fill(const Problem& p, const LaunchShape& ls, const GradKeys& k, cudaStream_t s) {
    const int grid = clamp_grid(ls.grid_grad, p.num_tiles);
    if (grid == 0) return cudaSuccess;
    if (p.grad_bf16) k_grad_fill<true><<<grid, kFillThreads, 0, s>>>(p, k);
    else k_grad_fill<false><<<grid, kFillThreads, 0, s>>>(p, k);
    return cudaGetLastError();
}

cudaError_t launch_global(const Problem& p, const LaunchShape& ls, const GlobalScalars& g, cudaStream_t s,
                          uint32_t* grid_used) {
    const int grid = clamp_grid(ls.grid_global, p.num_tiles);
    *grid_used = static_cast<uint32_t>(grid);
    if (grid == 0) return cudaSuccess;
    global_kernel_for(p.n, p.global_mode)<<<grid, kThreads, 0, s>>>(p, g);
    return cudaGetLastError();
}

cudaError_t launch_stats(const Problem& p, uint32_t producer_grid, cudaStream_t s) {
    if (p.num_tensors == 0) return cudaSuccess;
    k_stats<<<p.num_tensors, kThreads, 0, s>>>(p, producer_grid);
    return cudaGetLastError();
}

}  // namespace dsm
