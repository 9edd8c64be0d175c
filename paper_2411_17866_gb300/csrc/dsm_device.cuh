// Device helpers shared by the CUDA translation units of the library: the
// counter-based generators, 16-byte memory access, the per-element arithmetic
// of the method, the statistics accumulators and reductions, cp.async.
// Everything here is inline device code (or host-side launch helpers).
#pragma once

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

// fp32 -> bf16 rounds to nearest even, two values per conversion (the first in the low half).
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<const uint32_t*>(&h);
}

__device__ __forceinline__ void store4_bf16(__nv_bfloat16* p, const float (&v)[4]) {
    __stcs(reinterpret_cast<uint2*>(p), make_uint2(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3])));
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

// The same products with one multiplication per draw.  u - 1/2 equals
// (h24 - 2^23) * 2^-24 exactly, and for |s| >= 2^-102 so is s * 2^-24
// (a normal number), so s*(u - 1/2) and (s*2^-24)*(h24 - 2^23) are the same
// real number and round to the same float.  `sp` is s*2^-24; the draw
// enters as the signed integer h24 - 2^23, which converts exactly.
constexpr float kMinPrescaled = 1.9721522630525295e-31f;  // 2^-102
__device__ __forceinline__ float centred_even(uint64_t h) {
    return __int2float_rn(static_cast<int32_t>(static_cast<uint32_t>(h >> 40)) - 0x800000);
}
__device__ __forceinline__ float centred_odd(uint64_t h) {
    return __int2float_rn(static_cast<int32_t>(static_cast<uint32_t>(h >> 16) & 0xFFFFFFu) - 0x800000);
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

// global_elem with the global step chosen at run time among Algorithm 1 and
// the variants that keep only x and m (SlowMo, signed SlowMo, Lookahead).
template <int NW>
__device__ __forceinline__ void global_elem_rt(float& x, float& m, const float (&dif)[NW], const GlobalScalars& g,
                                               float lam, float r, ThreadStats& st) {
    float unused = 0.f;
    switch (g.mode) {
        case 1: global_elem<NW, 1>(x, m, unused, dif, NW, g, lam, r, st); break;
        case 2: global_elem<NW, 2>(x, m, unused, dif, NW, g, lam, r, st); break;
        case 3: global_elem<NW, 3>(x, m, unused, dif, NW, g, lam, r, st); break;
        default: global_elem<NW, 0>(x, m, unused, dif, NW, g, lam, r, st); break;
    }
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

// Persistent grid: every SM times the CTAs of `kernel` that fit on one SM.
template <typename K>
int grid_for(K kernel, int sms, size_t smem = 0, int threads = kThreads) {
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, threads, smem) != cudaSuccess || per_sm < 1)
        per_sm = 1;
    return sms * per_sm;
}

inline int clamp_grid(int grid, uint64_t items) {
    if (items == 0) return 0;
    return static_cast<int>(items < static_cast<uint64_t>(grid) ? items : static_cast<uint64_t>(grid));
}

}  // namespace
}  // namespace dsm
