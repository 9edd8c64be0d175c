// CUDA kernels (sm_103a) for one global round of distributed sign momentum
// with local steps (arXiv 2411.17866, Algorithm 1).
//
// Every kernel is a persistent, grid-stride loop over work items: tiles of
// at most kTile = 1024 elements that lie inside one tensor (for the local
// steps, a tile of one worker).  A CTA of 256 threads takes one item at a
// time; each thread owns 4 consecutive elements and moves them with one
// 16-byte load or store per fp32 stream (8 bytes per bf16 stream), so every
// warp instruction covers 512 contiguous bytes.  The local and global steps
// double-buffer in registers: a thread issues the loads of its next item
// before it computes the current one, so the HBM requests of one item are in
// flight during the arithmetic of the previous one.  The work is streaming and
// elementwise, bound by HBM bandwidth; nothing is a contraction, and no tensor
// core is used.
//
// All method arithmetic uses the explicit round-to-nearest intrinsics
// (__fadd_rn, __fmul_rn, __fdiv_rn, __fsqrt_rn, ...), which the compiler
// never contracts into FMAs, so each result is the fp32 value of the
// paper's expression evaluated one operation at a time.

#include <cuda_bf16.h>

#include "dsm_internal.h"

namespace dsm {
namespace {

// ---------------------------------------------------------------------------
// Counter-based generators
// ---------------------------------------------------------------------------

// SplitMix64 (Steele, Lea, Flood, OOPSLA 2014): output j of a generator
// seeded with `state` is the state advanced j times by the golden-ratio
// increment, passed through Stafford's variant-13 finaliser.
constexpr uint64_t kGoldenGamma = 0x9E3779B97F4A7C15ull;
constexpr float kTwoPowM24 = 5.9604644775390625e-08f;  // 2^-24

__device__ __forceinline__ uint64_t sm64_finalise(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

__device__ __forceinline__ uint64_t sm64_output(uint64_t key, uint64_t j) {
    return sm64_finalise(key + j * kGoldenGamma);
}

// The two 24-bit draws of one output: bits 63..40 (even element) and
// 39..16 (odd element), each times 2^-24 (exact in fp32).
__device__ __forceinline__ float draw_even(uint64_t h) {
    return __fmul_rn(__uint2float_rn(static_cast<uint32_t>(h >> 40)), kTwoPowM24);
}
__device__ __forceinline__ float draw_odd(uint64_t h) {
    return __fmul_rn(__uint2float_rn(static_cast<uint32_t>(h >> 16) & 0xFFFFFFu), kTwoPowM24);
}

// u of element e: output floor(e/2)+1 of SplitMix64(key), field by parity.
__device__ __forceinline__ float hash_uniform(uint64_t key, uint64_t e) {
    const uint64_t h = sm64_output(key, (e >> 1) + 1);
    return (e & 1) ? draw_odd(h) : draw_even(h);
}

// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC 2011): ten rounds of the
// two-multiplier S-box with a Weyl key schedule.
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint32_t k0, uint32_t k1) {
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        if (r) {
            k0 += 0x9E3779B9u;
            k1 += 0xBB67AE85u;
        }
        const uint32_t hi0 = __umulhi(0xD2511F53u, c.x), lo0 = 0xD2511F53u * c.x;
        const uint32_t hi1 = __umulhi(0xCD9E8D57u, c.z), lo1 = 0xCD9E8D57u * c.z;
        c = make_uint4(hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0);
    }
    return c;
}

__device__ __forceinline__ uint4 philox_block(uint64_t q, uint32_t k0, uint32_t k1) {
    return philox4x32_10(make_uint4(static_cast<uint32_t>(q), static_cast<uint32_t>(q >> 32), 0u, 0u), k0, k1);
}

__device__ __forceinline__ uint32_t word_of(const uint4& b, uint32_t i) {
    return i == 0 ? b.x : (i == 1 ? b.y : (i == 2 ? b.z : b.w));
}

// r = (word >> 8) * 2^-24, exact in fp32.
__device__ __forceinline__ float philox_unit(uint32_t w) {
    return __fmul_rn(__uint2float_rn(w >> 8), kTwoPowM24);
}

// ---------------------------------------------------------------------------
// 16-byte streaming memory access (4 elements per thread)
// ---------------------------------------------------------------------------

__device__ __forceinline__ void load4(const float* p, float (&v)[4]) {
    const float4 a = __ldcs(reinterpret_cast<const float4*>(p));
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
}

__device__ __forceinline__ void store4(float* p, const float (&v)[4]) {
    __stcs(reinterpret_cast<float4*>(p), make_float4(v[0], v[1], v[2], v[3]));
}

// bf16 -> fp32 is exact: the bf16 bits are the top half of the fp32 encoding.
__device__ __forceinline__ void load4_bf16(const __nv_bfloat16* p, float (&v)[4]) {
    const uint2 raw = __ldcs(reinterpret_cast<const uint2*>(p));
    v[0] = __uint_as_float(raw.x << 16);
    v[1] = __uint_as_float(raw.x & 0xFFFF0000u);
    v[2] = __uint_as_float(raw.y << 16);
    v[3] = __uint_as_float(raw.y & 0xFFFF0000u);
}

__device__ __forceinline__ void store4_bf16(__nv_bfloat16* p, const float (&v)[4]) {
    uint32_t h[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) h[i] = __bfloat16_as_ushort(__float2bfloat16_rn(v[i]));
    __stcs(reinterpret_cast<uint2*>(p), make_uint2(h[0] | (h[1] << 16), h[2] | (h[3] << 16)));
}

template <bool kBf16>
__device__ __forceinline__ void load4_grad(const void* g, uint64_t i, float (&v)[4]) {
    if (kBf16) load4_bf16(reinterpret_cast<const __nv_bfloat16*>(g) + i, v);
    else load4(reinterpret_cast<const float*>(g) + i, v);
}

__device__ __forceinline__ float load_grad1(const void* g, int bf16, uint64_t i) {
    if (bf16) return __bfloat162float(reinterpret_cast<const __nv_bfloat16*>(g)[i]);
    return reinterpret_cast<const float*>(g)[i];
}

// A thread's 4 elements take the vector path when the tile start is
// 4-element aligned (every fp32 stream 16-byte aligned, every bf16 stream
// 8-byte aligned) and all 4 lie in the tile; otherwise the thread handles
// its elements one at a time.
__device__ __forceinline__ bool vector_ok(const TileDesc& td, uint32_t e0) {
    return (td.start & 3u) == 0 && e0 + kElemsPerThread <= td.len;
}

// ---------------------------------------------------------------------------
// Per-element arithmetic of the method
// ---------------------------------------------------------------------------

// Synthetic gradient: s*(u_step - 1/2) + s2*(u_worker - 1/2), left to right.
__device__ __forceinline__ float step_term(float s, float u) { return __fmul_rn(s, __fsub_rn(u, 0.5f)); }
__device__ __forceinline__ float grad_value(float a, float s2, float u2) {
    return __fadd_rn(a, __fmul_rn(s2, __fsub_rn(u2, 0.5f)));
}

// AdamW (Appendix A): m <- b1 m + (1-b1) g; v <- b2 v + (1-b2) g*g;
// x <- x - lr (mhat/(sqrt(vhat)+eps) + lam x), mhat = m/bc1, vhat = v/bc2.
__device__ __forceinline__ void adamw_elem(float& x, float& m, float& v, float g, const AdamScalars& a, float lam) {
    m = __fadd_rn(__fmul_rn(a.b1, m), __fmul_rn(a.omb1, g));
    v = __fadd_rn(__fmul_rn(a.b2, v), __fmul_rn(a.omb2, __fmul_rn(g, g)));
    const float mhat = __fdiv_rn(m, a.bc1);
    const float vhat = __fdiv_rn(v, a.bc2);
    const float den = __fadd_rn(__fsqrt_rn(vhat), a.eps);
    const float upd = __fadd_rn(__fdiv_rn(mhat, den), __fmul_rn(lam, x));
    x = __fsub_rn(x, __fmul_rn(a.lr, upd));
}

// Polyak momentum (Appendix A): buf <- mu buf + g; x <- x - lr buf.
__device__ __forceinline__ void sgdm_elem(float& x, float& b, float g, const SgdmScalars& a) {
    b = __fadd_rn(__fmul_rn(a.mu, b), g);
    x = __fsub_rn(x, __fmul_rn(a.lr, b));
}

__device__ __forceinline__ int sgn(float v) { return (v > 0.f) - (v < 0.f); }

// Applied sign S(u): deterministic sign, or the randomized sign of
// Eq. (rand-sign-2) (mode 1) / Eq. (rand-sign-1) (mode 2) with uniform r.
__device__ __forceinline__ float applied_sign(float u, const GlobalScalars& g, float r) {
    const float s = static_cast<float>(sgn(u));
    if (g.sign_mode == 0) return s;
    const float p = fminf(__fdiv_rn(fabsf(u), g.B), 1.0f);
    if (g.sign_mode == 1) return r < p ? s : 0.0f;
    const float q = __fadd_rn(0.5f, __fmul_rn(0.5f, p));
    return r < q ? s : -s;
}

// Compensated fp32 sum (hi + lo): each addition keeps its rounding error
// (Knuth's TwoSum, six fp32 operations), so long sums stay accurate to about
// 2^-44 relative without using the fp64 pipe.
struct CSum {
    float hi = 0.f, lo = 0.f;
};

__device__ __forceinline__ void csum_add(CSum& s, float v) {
    const float t = __fadd_rn(s.hi, v);
    const float bp = __fsub_rn(t, s.hi);
    const float err = __fadd_rn(__fsub_rn(s.hi, __fsub_rn(t, bp)), __fsub_rn(v, bp));
    s.lo = __fadd_rn(s.lo, err);
    s.hi = t;
}

__device__ __forceinline__ void csum_merge(CSum& a, const CSum& b) {
    csum_add(a, b.hi);
    a.lo = __fadd_rn(a.lo, b.lo);
}

struct ThreadStats {
    CSum dsq, drift;
    uint32_t zero = 0, flips = 0, unanimous = 0, clamped = 0;
};

// Global-step update of one element from Delta (mode = DSM_GLOBAL_*); returns u
// and the sign entering the statistics, and updates x, m (and v for AdamW).
template <int MODE>
__device__ __forceinline__ void global_update(float D, float& x, float& m, float& v, const GlobalScalars& g,
                                              float lam, float r, float& u, float& s) {
    if (MODE == 0) {         // Algorithm 1: Eqs. (ut-update), (model-update), (mom-update)
        u = __fadd_rn(__fmul_rn(g.b1, m), __fmul_rn(g.c1, D));
        s = applied_sign(u, g, r);
        const float xn = __fsub_rn(x, __fmul_rn(g.eta_gamma, __fadd_rn(s, __fmul_rn(lam, x))));
        m = __fadd_rn(__fmul_rn(g.b2, m), __fmul_rn(g.c2, D));
        x = xn;
    } else if (MODE == 1) {  // SlowMo: u <- b u + (1/gamma) Delta; x <- x - alpha gamma u
        u = __fadd_rn(__fmul_rn(g.b1, m), __fmul_rn(g.inv_gamma, D));
        s = static_cast<float>(sgn(u));
        x = __fsub_rn(x, __fmul_rn(g.eta_gamma, u));
        m = u;
    } else if (MODE == 2) {  // signed SlowMo: the pseudo-gradient's sign enters u
        const float sd = static_cast<float>(sgn(D));
        u = __fadd_rn(__fmul_rn(g.b1, m), __fmul_rn(g.c1, sd));
        s = sd;
        x = __fsub_rn(x, __fmul_rn(g.eta_gamma, u));
        m = __fadd_rn(__fmul_rn(g.b2, m), __fmul_rn(g.c2, D));
    } else if (MODE == 3) {  // Lookahead: Algorithm 1 with x' = x - eta gamma u
        u = __fadd_rn(__fmul_rn(g.b1, m), __fmul_rn(g.c1, D));
        s = static_cast<float>(sgn(u));
        x = __fsub_rn(x, __fmul_rn(g.eta_gamma, u));
        m = __fadd_rn(__fmul_rn(g.b2, m), __fmul_rn(g.c2, D));
    } else {                 // global AdamW on the pseudo-gradient Delta/gamma
        const float gg = __fmul_rn(g.inv_gamma, D);
        m = __fadd_rn(__fmul_rn(g.b1, m), __fmul_rn(g.omb1, gg));
        v = __fadd_rn(__fmul_rn(g.b2, v), __fmul_rn(g.omb2, __fmul_rn(gg, gg)));
        const float mhat = __fdiv_rn(m, g.bc1);
        const float vhat = __fdiv_rn(v, g.bc2);
        const float den = __fadd_rn(__fsqrt_rn(vhat), g.eps);
        x = __fsub_rn(x, __fmul_rn(g.eta, __fadd_rn(__fdiv_rn(mhat, den), __fmul_rn(lam, x))));
        u = m;
        s = static_cast<float>(sgn(u));
    }
}

// Global step on one element given x, m (v) and the worker differences d_i = x - x_i:
// Delta = (sum_i d_i)/n, then the mode's update.  Accumulates the element's statistics.
template <int NW, int MODE>
__device__ __forceinline__ void global_elem(float& x, float& m, float& v, const float (&dif)[NW], int nw,
                                            const GlobalScalars& g, float lam, float r, ThreadStats& st) {
    float acc = 0.f;
#pragma unroll
    for (int i = 0; i < NW; ++i)
        if (i < nw) acc = __fadd_rn(acc, dif[i]);
    const float D = __fdiv_rn(acc, g.n_f);
    float u, s;
    global_update<MODE>(D, x, m, v, g, lam, r, u, s);
    // statistics
    const int sD = sgn(D);
    csum_add(st.dsq, __fmul_rn(D, D));
    bool unan = true;
    float dr = 0.f;
#pragma unroll
    for (int i = 0; i < NW; ++i) {
        if (i < nw) {
            const float e = __fsub_rn(dif[i], D);
            dr = __fadd_rn(dr, __fmul_rn(e, e));
            unan = unan && (sgn(dif[i]) == sD);
        }
    }
    csum_add(st.drift, dr);
    st.zero += (s == 0.f);
    st.flips += (sgn(u) != sD);
    st.unanimous += unan;
    st.clamped += (MODE == 0 && g.sign_mode != 0 && fabsf(u) > g.B);
}

// Fixed-order CTA reduction of the per-thread statistics into one partial:
// compensated fp32 across the lanes of a warp, fp64 across the warps.
__device__ __forceinline__ void reduce_stats(const ThreadStats& st, StatPartial* out) {
    __shared__ double s_d[kThreads / 32][2];
    __shared__ uint32_t s_c[kThreads / 32][4];
    CSum a = st.dsq, b = st.drift;
    uint32_t c0 = st.zero, c1 = st.flips, c2 = st.unanimous, c3 = st.clamped;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
        CSum oa, ob;
        oa.hi = __shfl_down_sync(0xffffffffu, a.hi, off);
        oa.lo = __shfl_down_sync(0xffffffffu, a.lo, off);
        ob.hi = __shfl_down_sync(0xffffffffu, b.hi, off);
        ob.lo = __shfl_down_sync(0xffffffffu, b.lo, off);
        csum_merge(a, oa);
        csum_merge(b, ob);
        c0 += __shfl_down_sync(0xffffffffu, c0, off);
        c1 += __shfl_down_sync(0xffffffffu, c1, off);
        c2 += __shfl_down_sync(0xffffffffu, c2, off);
        c3 += __shfl_down_sync(0xffffffffu, c3, off);
    }
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) {
        s_d[warp][0] = static_cast<double>(a.hi) + static_cast<double>(a.lo);
        s_d[warp][1] = static_cast<double>(b.hi) + static_cast<double>(b.lo);
        s_c[warp][0] = c0; s_c[warp][1] = c1; s_c[warp][2] = c2; s_c[warp][3] = c3;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        StatPartial p;
        p.delta_sq = 0.0; p.drift = 0.0;
        p.zero_sign = p.flips = p.unanimous = p.clamped = 0;
        for (int w = 0; w < kThreads / 32; ++w) {
            p.delta_sq += s_d[w][0]; p.drift += s_d[w][1];
            p.zero_sign += s_c[w][0]; p.flips += s_c[w][1]; p.unanimous += s_c[w][2]; p.clamped += s_c[w][3];
        }
        *out = p;
    }
    __syncthreads();  // the shared arrays are reused by the next reduction
}

__device__ __forceinline__ void zero_partial(StatPartial* out) {
    if (threadIdx.x == 0) {
        StatPartial p;
        p.delta_sq = 0.0; p.drift = 0.0;
        p.zero_sign = p.flips = p.unanimous = p.clamped = 0;
        *out = p;
    }
}

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
// and per draw family), not by its write stream.
template <bool kBf16>
__global__ void __launch_bounds__(kThreads) k_grad_fill(Problem p, GradKeys k) {
    const uint32_t e0 = threadIdx.x * kElemsPerThread;
    for (uint32_t ti = blockIdx.x; ti < p.num_tiles; ti += gridDim.x) {
        const TileDesc td = p.tiles[ti];
        const TensorDesc& T = p.tensors[td.tensor];
        const float s = T.scale, s2 = T.scale2;
        if (vector_ok(td, e0)) {
            const uint64_t gi = td.start + e0;  // even: elements gi..gi+3 use outputs gi/2+1, gi/2+2
            // output j of any family is finalise(key + j*gamma): j*gamma is shared by all families
            const uint64_t jg0 = ((gi >> 1) + 1) * kGoldenGamma, jg1 = jg0 + kGoldenGamma;
            const uint64_t h0 = sm64_finalise(k.step + jg0), h1 = sm64_finalise(k.step + jg1);
            const float a[4] = {step_term(s, draw_even(h0)), step_term(s, draw_odd(h0)),
                                step_term(s, draw_even(h1)), step_term(s, draw_odd(h1))};
            for (uint32_t w = 0; w < p.n; ++w) {
                const uint64_t q0 = sm64_finalise(k.worker[w] + jg0), q1 = sm64_finalise(k.worker[w] + jg1);
                const float g[4] = {grad_value(a[0], s2, draw_even(q0)), grad_value(a[1], s2, draw_odd(q0)),
                                    grad_value(a[2], s2, draw_even(q1)), grad_value(a[3], s2, draw_odd(q1))};
                const uint64_t o = w * p.d_stride + gi;
                if (kBf16) store4_bf16(reinterpret_cast<__nv_bfloat16*>(p.grad) + o, g);
                else store4(reinterpret_cast<float*>(p.grad) + o, g);
            }
        } else {
            const uint32_t e1 = min(e0 + kElemsPerThread, td.len);
            for (uint32_t e = e0; e < e1; ++e) {
                const uint64_t gi = td.start + e;
                const float a = step_term(s, hash_uniform(k.step, gi));
                for (uint32_t w = 0; w < p.n; ++w) {
                    const float g = grad_value(a, s2, hash_uniform(k.worker[w], gi));
                    const uint64_t o = w * p.d_stride + gi;
                    if (kBf16) reinterpret_cast<__nv_bfloat16*>(p.grad)[o] = __float2bfloat16_rn(g);
                    else reinterpret_cast<float*>(p.grad)[o] = g;
                }
            }
        }
    }
}

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

template <bool kTileMajor>
__device__ __forceinline__ LocalItem local_item(const Problem& p, uint32_t item, uint32_t e0, bool local_lam) {
    uint32_t w, ti;
    if (kTileMajor) {
        ti = item / p.n;
        w = item - ti * p.n;
    } else {
        w = item / p.num_tiles;
        ti = item - w * p.num_tiles;
    }
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
// global x (the replicas' reset is still pending).
template <bool kBf16, bool kFromGlobal>
__global__ void __launch_bounds__(kThreads) k_local_adamw(Problem p, AdamScalars a) {
    const uint32_t items = p.num_tiles * p.n;
    const uint32_t e0 = threadIdx.x * kElemsPerThread;
    uint32_t item = blockIdx.x;
    if (item >= items) return;
    LocalItem nx = local_item<kFromGlobal>(p, item, e0, true);
    float x[4], m[4], v[4], g[4];
    if (nx.vec) {
        load4(kFromGlobal ? p.x + nx.start + e0 : p.X + nx.base + e0, x);
        load4(p.opt_m + nx.base + e0, m);
        load4(p.opt_v + nx.base + e0, v);
        load4_grad<kBf16>(p.grad, nx.base + e0, g);
    }
    for (; item < items; item += gridDim.x) {
        const LocalItem cur = nx;
        float cx[4], cm[4], cv[4], cg[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) { cx[j] = x[j]; cm[j] = m[j]; cv[j] = v[j]; cg[j] = g[j]; }
        const uint32_t next = item + gridDim.x;
        if (next < items) {  // issue the next item's loads before computing this one
            nx = local_item<kFromGlobal>(p, next, e0, true);
            if (nx.vec) {
                load4(kFromGlobal ? p.x + nx.start + e0 : p.X + nx.base + e0, x);
                load4(p.opt_m + nx.base + e0, m);
                load4(p.opt_v + nx.base + e0, v);
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
                float xs = kFromGlobal ? p.x[cur.start + e] : p.X[i], ms = p.opt_m[i], vs = p.opt_v[i];
                adamw_elem(xs, ms, vs, load_grad1(p.grad, kBf16, i), a, cur.lam);
                p.X[i] = xs; p.opt_m[i] = ms; p.opt_v[i] = vs;
            }
        }
    }
}

// K3: one SGD-momentum local step on every worker, double-buffered.
template <bool kBf16, bool kFromGlobal>
__global__ void __launch_bounds__(kThreads) k_local_sgdm(Problem p, SgdmScalars a) {
    const uint32_t items = p.num_tiles * p.n;
    const uint32_t e0 = threadIdx.x * kElemsPerThread;
    uint32_t item = blockIdx.x;
    if (item >= items) return;
    LocalItem nx = local_item<kFromGlobal>(p, item, e0, false);
    float x[4], b[4], g[4];
    if (nx.vec) {
        load4(kFromGlobal ? p.x + nx.start + e0 : p.X + nx.base + e0, x);
        load4(p.opt_m + nx.base + e0, b);
        load4_grad<kBf16>(p.grad, nx.base + e0, g);
    }
    for (; item < items; item += gridDim.x) {
        const LocalItem cur = nx;
        float cx[4], cb[4], cg[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) { cx[j] = x[j]; cb[j] = b[j]; cg[j] = g[j]; }
        const uint32_t next = item + gridDim.x;
        if (next < items) {
            nx = local_item<kFromGlobal>(p, next, e0, false);
            if (nx.vec) {
                load4(kFromGlobal ? p.x + nx.start + e0 : p.X + nx.base + e0, x);
                load4(p.opt_m + nx.base + e0, b);
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
                float xs = kFromGlobal ? p.x[cur.start + e] : p.X[i], bs = p.opt_m[i];
                sgdm_elem(xs, bs, load_grad1(p.grad, kBf16, i), a);
                p.X[i] = xs; p.opt_m[i] = bs;
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
        r = philox_unit(word_of(philox_block(gi >> 2, g.philox_k0, g.philox_k1), gi & 3));
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
        const uint4 b = philox_block(gi >> 2, g.philox_k0, g.philox_k1);
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
                store4(p.X + (i0 + c) * p.d_stride + gi, xn);
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
// momentum update, reset of every replica) with statistics.
// NW > 0: exactly NW replicas, held in registers and double-buffered.
// NW == 0: any n, one element at a time.
// Statistics: a CTA keeps per-thread sums while its successive tiles belong
// to one tensor and reduces them only when the tensor changes (or at its last
// tile), writing the segment's partial at the segment's last tile and zeros
// at its other tiles; the per-tensor sum over tiles is then unchanged.
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
                const uint4 b = philox_block(gi >> 2, g.philox_k0, g.philox_k1);
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
#pragma unroll
            for (int i = 0; i < W; ++i) store4(p.X + i * p.d_stride + gi, cx);
        } else if (NW == 0 && vector_ok(td, e0)) {
            global_vec_generic<MODE>(p, g, lam, td.start + e0, st);
        } else {
            const uint32_t e1 = min(e0 + kElemsPerThread, td.len);
            for (uint32_t e = e0; e < e1; ++e) global_elem_generic<MODE>(p, g, lam, td.start + e, st);
        }
        if (next >= p.num_tiles || nt.tensor != td.tensor) {  // uniform across the CTA
            reduce_stats(st, p.partials + ti);
            st = ThreadStats();
        } else {
            zero_partial(p.partials + ti);
        }
    }
}

// Per-thread asynchronous global -> shared copies (cp.async): the copy holds
// no register while in flight, and a thread waits only for its own groups.
__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(static_cast<uint32_t>(__cvta_generic_to_shared(smem))),
                 "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async8(void* smem, const void* gmem) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 8;" ::"r"(static_cast<uint32_t>(__cvta_generic_to_shared(smem))),
                 "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

// K6: the round's last local step fused with the sign-momentum global step.
// One thread owns 4 elements of every worker: it runs the base optimizer's
// last step on each worker (writing the worker's optimizer state, but not
// its new replica, which only feeds the average), then the global step of
// Algorithm 1 on those elements.  The replicas are not reset: the next
// round's first local step starts every worker from x.  from_global: the
// replicas' reset from the previous round is still pending (tau = 1).
// A CTA walks its tiles worker by worker; each thread keeps the next
// kFusedDepth (tile, worker) items in flight with cp.async into its own
// shared-memory slots (x_i, m_i, v_i, g_i, and x, m with a tile's first worker).
// Items in flight per thread: 2, or 3 for AdamW with more than 4 workers,
// whose registers already limit the resident CTAs (measured on GB300: depth 2
// gives 0.92 / 1.00 of the copy bandwidth on GPT-2 S (AdamW, n = 4) / L
// (SGD-momentum, n = 8), depth 3 gives 0.85 on GPT-2 M (AdamW, n = 8) where
// depth 2 gives 0.79).
constexpr int kFusedStreams = 6;
__host__ __device__ constexpr int fused_depth(bool adamw, int nw) { return (adamw && nw > 4) ? 3 : 2; }
__host__ __device__ constexpr size_t fused_smem(int depth) { return size_t(depth) * kFusedStreams * kThreads * sizeof(float4); }

template <bool kAdamW, bool kBf16, int NW>
__global__ void __launch_bounds__(kThreads) k_fused_last_global(Problem p, AdamScalars a, SgdmScalars sa,
                                                                GlobalScalars g, int from_global) {
    constexpr int kFusedDepth = fused_depth(kAdamW, NW);
    extern __shared__ float4 fsm[];  // [kFusedDepth][kFusedStreams][kThreads]
    const uint32_t e0 = threadIdx.x * kElemsPerThread;
    auto slot = [&](int it, int stream) -> float4* {
        return fsm + (size_t(it % kFusedDepth) * kFusedStreams + stream) * kThreads + threadIdx.x;
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
                if (!from_global) cp_async16(slot(it, 0), p.X + o);
                cp_async16(slot(it, 1), p.opt_m + o);
                if (kAdamW) cp_async16(slot(it, 2), p.opt_v + o);
                if (kBf16) cp_async8(slot(it, 3), reinterpret_cast<const __nv_bfloat16*>(p.grad) + o);
                else cp_async16(slot(it, 3), reinterpret_cast<const float*>(p.grad) + o);
                if (w == 0) {
                    cp_async16(slot(it, 4), p.x + gi);
                    cp_async16(slot(it, 5), p.m + gi);
                }
            }
        }
        cp_async_commit();
    };
    auto take = [&](int it, int stream, float (&v)[4]) {
        const float4 t = *slot(it, stream);
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
            float x[4], m[4], dif[NW][4];
#pragma unroll
            for (int w = 0; w < NW; ++w, ++it) {
                cp_async_wait<kFusedDepth - 1>();  // item `it` has landed
                float xi[4], mi[4], vi[4], gr[4];
                if (w == 0) {
                    take(it, 4, x);
                    take(it, 5, m);
                }
                if (from_global) {
#pragma unroll
                    for (int j = 0; j < 4; ++j) xi[j] = x[j];
                } else {
                    take(it, 0, xi);
                }
                take(it, 1, mi);
                if (kAdamW) take(it, 2, vi);
                if (kBf16) {
                    const uint2 raw = *reinterpret_cast<const uint2*>(slot(it, 3));
                    gr[0] = __uint_as_float(raw.x << 16);
                    gr[1] = __uint_as_float(raw.x & 0xFFFF0000u);
                    gr[2] = __uint_as_float(raw.y << 16);
                    gr[3] = __uint_as_float(raw.y & 0xFFFF0000u);
                } else {
                    take(it, 3, gr);
                }
                const uint64_t o = w * p.d_stride + gi;
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    if (kAdamW) adamw_elem(xi[j], mi[j], vi[j], gr[j], a, lam_l);
                    else sgdm_elem(xi[j], mi[j], gr[j], sa);
                    dif[w][j] = __fsub_rn(x[j], xi[j]);
                }
                store4(p.opt_m + o, mi);
                if (kAdamW) store4(p.opt_v + o, vi);
                // refill the slot just read; the arithmetic above consumed its values, so the
                // shared-memory reads are complete before the asynchronous copy can overwrite them
                issue(next_issue++);
            }
            float ru[4] = {0.f, 0.f, 0.f, 0.f};
            if (g.sign_mode != 0) {
                const uint4 b = philox_block(gi >> 2, g.philox_k0, g.philox_k1);
                ru[0] = philox_unit(b.x); ru[1] = philox_unit(b.y); ru[2] = philox_unit(b.z); ru[3] = philox_unit(b.w);
            }
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                float d[NW];
#pragma unroll
                for (int w = 0; w < NW; ++w) d[w] = dif[w][j];
                float unused = 0.f;
                global_elem<NW, 0>(x[j], m[j], unused, d, NW, g, lam_g, ru[j], st);
            }
            store4(p.x + gi, x);
            store4(p.m + gi, m);
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
                    float xi = from_global ? x : p.X[o], mi = p.opt_m[o];
                    if (kAdamW) {
                        float vi = p.opt_v[o];
                        adamw_elem(xi, mi, vi, load_grad1(p.grad, kBf16, o), a, lam_l);
                        p.opt_v[o] = vi;
                    } else {
                        sgdm_elem(xi, mi, load_grad1(p.grad, kBf16, o), sa);
                    }
                    p.opt_m[o] = mi;
                    d[w] = __fsub_rn(x, xi);
                }
                float r = 0.f;
                if (g.sign_mode != 0) r = philox_unit(word_of(philox_block(gj >> 2, g.philox_k0, g.philox_k1), gj & 3));
                float unused = 0.f;
                global_elem<NW, 0>(x, m, unused, d, NW, g, lam_g, r, st);
                p.x[gj] = x;
                p.m[gj] = m;
            }
        }
        const uint32_t next = ti + gridDim.x;
        if (next >= p.num_tiles || p.tiles[next].tensor != td.tensor) {  // uniform across the CTA
            reduce_stats(st, p.partials + ti);
            st = ThreadStats();
        } else {
            zero_partial(p.partials + ti);
        }
    }
    cp_async_wait<0>();  // the groups issued past the last tile are empty; nothing is left in flight
}

// K5: per-tensor statistics from the tile partials, in a fixed order.
__global__ void __launch_bounds__(kThreads) k_stats(Problem p) {
    const uint32_t T = blockIdx.x;
    const TensorDesc td = p.tensors[T];
    double a = 0.0, b = 0.0;
    unsigned long long c0 = 0, c1 = 0, c2 = 0, c3 = 0;
    for (uint32_t t = td.tile_begin + threadIdx.x; t < td.tile_end; t += blockDim.x) {
        const StatPartial q = p.partials[t];
        a += q.delta_sq; b += q.drift;
        c0 += q.zero_sign; c1 += q.flips; c2 += q.unanimous; c3 += q.clamped;
    }
    __shared__ double s_d[kThreads][2];
    __shared__ unsigned long long s_c[kThreads][4];
    s_d[threadIdx.x][0] = a; s_d[threadIdx.x][1] = b;
    s_c[threadIdx.x][0] = c0; s_c[threadIdx.x][1] = c1; s_c[threadIdx.x][2] = c2; s_c[threadIdx.x][3] = c3;
    __syncthreads();
    for (uint32_t off = kThreads / 2; off > 0; off >>= 1) {
        if (threadIdx.x < off) {
            s_d[threadIdx.x][0] += s_d[threadIdx.x + off][0];
            s_d[threadIdx.x][1] += s_d[threadIdx.x + off][1];
#pragma unroll
            for (int k = 0; k < 4; ++k) s_c[threadIdx.x][k] += s_c[threadIdx.x + off][k];
        }
        __syncthreads();
    }
    if (threadIdx.x == 0) {
        TensorStats o;
        o.delta_sq = s_d[0][0]; o.drift = s_d[0][1];
        o.zero_sign = s_c[0][0]; o.flips = s_c[0][1]; o.unanimous = s_c[0][2]; o.clamped = s_c[0][3];
        p.stats[T] = o;
    }
}

template <typename K>
int grid_for(K kernel, int sms, size_t smem = 0) {
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, kThreads, smem) != cudaSuccess || per_sm < 1)
        per_sm = 1;
    return sms * per_sm;
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

using FusedKernel = void (*)(Problem, AdamScalars, SgdmScalars, GlobalScalars, int);

template <bool kAdamW, bool kBf16>
FusedKernel fused_kernel_n(uint32_t n) {
    switch (n) {
        case 1: return k_fused_last_global<kAdamW, kBf16, 1>;
        case 2: return k_fused_last_global<kAdamW, kBf16, 2>;
        case 3: return k_fused_last_global<kAdamW, kBf16, 3>;
        case 4: return k_fused_last_global<kAdamW, kBf16, 4>;
        case 5: return k_fused_last_global<kAdamW, kBf16, 5>;
        case 6: return k_fused_last_global<kAdamW, kBf16, 6>;
        case 7: return k_fused_last_global<kAdamW, kBf16, 7>;
        case 8: return k_fused_last_global<kAdamW, kBf16, 8>;
        default: return nullptr;
    }
}

FusedKernel fused_kernel_for(const Problem& p, bool adamw) {
    if (adamw) return p.grad_bf16 ? fused_kernel_n<true, true>(p.n) : fused_kernel_n<true, false>(p.n);
    return p.grad_bf16 ? fused_kernel_n<false, true>(p.n) : fused_kernel_n<false, false>(p.n);
}

size_t fused_smem_for(const Problem& p, bool adamw) { return fused_smem(fused_depth(adamw, int(p.n))); }

}  // namespace

bool fused_round_available(const Problem& p) {
    return p.global_mode == 0 && p.n >= 1 && p.n <= kMaxUnrolledWorkers;
}

cudaError_t query_launch_shape(const Problem& p, LaunchShape* out) {
    int dev = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err != cudaSuccess) return err;
    int sms = 0;
    err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (err != cudaSuccess) return err;
    out->sms = sms;
    out->grid_init = grid_for(k_init, sms);
    out->grid_grad = p.grad_bf16 ? grid_for(k_grad_fill<true>, sms) : grid_for(k_grad_fill<false>, sms);
    out->grid_adamw = p.grad_bf16 ? grid_for(k_local_adamw<true, false>, sms) : grid_for(k_local_adamw<false, false>, sms);
    out->grid_sgdm = p.grad_bf16 ? grid_for(k_local_sgdm<true, false>, sms) : grid_for(k_local_sgdm<false, false>, sms);
    if (fused_round_available(p)) {
        const FusedKernel fk = fused_kernel_for(p, p.opt_v != nullptr);
        const size_t smem = fused_smem_for(p, p.opt_v != nullptr);
        cudaError_t e = cudaFuncSetAttribute(fk, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
        if (e != cudaSuccess) return e;
        out->grid_fused = grid_for(fk, sms, smem);
        out->grid_adamw_from_x = p.grad_bf16 ? grid_for(k_local_adamw<true, true>, sms) : grid_for(k_local_adamw<false, true>, sms);
        out->grid_sgdm_from_x = p.grad_bf16 ? grid_for(k_local_sgdm<true, true>, sms) : grid_for(k_local_sgdm<false, true>, sms);
    }
    out->grid_global = grid_for(global_kernel_for(p.n, p.global_mode), sms);
    return cudaGetLastError();
}

static int clamp_grid(int grid, uint64_t items) {
    if (items == 0) return 0;
    return static_cast<int>(items < static_cast<uint64_t>(grid) ? items : static_cast<uint64_t>(grid));
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
    if (p.grad_bf16) k_grad_fill<true><<<grid, kThreads, 0, s>>>(p, k);
    else k_grad_fill<false><<<grid, kThreads, 0, s>>>(p, k);
    return cudaGetLastError();
}

cudaError_t launch_local_adamw(const Problem& p, const LaunchShape& ls, const AdamScalars& a, bool from_x,
                               cudaStream_t s) {
    const uint64_t items = static_cast<uint64_t>(p.num_tiles) * p.n;
    const int grid = clamp_grid(from_x ? ls.grid_adamw_from_x : ls.grid_adamw, items);
    if (grid == 0) return cudaSuccess;
    if (from_x) {
        if (p.grad_bf16) k_local_adamw<true, true><<<grid, kThreads, 0, s>>>(p, a);
        else k_local_adamw<false, true><<<grid, kThreads, 0, s>>>(p, a);
    } else {
        if (p.grad_bf16) k_local_adamw<true, false><<<grid, kThreads, 0, s>>>(p, a);
        else k_local_adamw<false, false><<<grid, kThreads, 0, s>>>(p, a);
    }
    return cudaGetLastError();
}

cudaError_t launch_local_sgdm(const Problem& p, const LaunchShape& ls, const SgdmScalars& a, bool from_x,
                              cudaStream_t s) {
    const uint64_t items = static_cast<uint64_t>(p.num_tiles) * p.n;
    const int grid = clamp_grid(from_x ? ls.grid_sgdm_from_x : ls.grid_sgdm, items);
    if (grid == 0) return cudaSuccess;
    if (from_x) {
        if (p.grad_bf16) k_local_sgdm<true, true><<<grid, kThreads, 0, s>>>(p, a);
        else k_local_sgdm<false, true><<<grid, kThreads, 0, s>>>(p, a);
    } else {
        if (p.grad_bf16) k_local_sgdm<true, false><<<grid, kThreads, 0, s>>>(p, a);
        else k_local_sgdm<false, false><<<grid, kThreads, 0, s>>>(p, a);
    }
    return cudaGetLastError();
}

cudaError_t launch_fused_last_global(const Problem& p, const LaunchShape& ls, const AdamScalars& a,
                                     const SgdmScalars& sa, const GlobalScalars& g, bool from_x, cudaStream_t s) {
    if (!fused_round_available(p)) return cudaErrorInvalidValue;
    const int grid = clamp_grid(ls.grid_fused, p.num_tiles);
    if (grid == 0) return cudaSuccess;
    fused_kernel_for(p, p.opt_v != nullptr)<<<grid, kThreads, fused_smem_for(p, p.opt_v != nullptr), s>>>(
        p, a, sa, g, from_x ? 1 : 0);
    return cudaGetLastError();
}

cudaError_t launch_global(const Problem& p, const LaunchShape& ls, const GlobalScalars& g, cudaStream_t s) {
    const int grid = clamp_grid(ls.grid_global, p.num_tiles);
    if (grid == 0) return cudaSuccess;
    global_kernel_for(p.n, p.global_mode)<<<grid, kThreads, 0, s>>>(p, g);
    return cudaGetLastError();
}

cudaError_t launch_stats(const Problem& p, cudaStream_t s) {
    if (p.num_tensors == 0) return cudaSuccess;
    k_stats<<<p.num_tensors, kThreads, 0, s>>>(p);
    return cudaGetLastError();
}

}  // namespace dsm
