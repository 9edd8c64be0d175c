// C++ CPU oracle for one global round of distributed sign momentum with
// local steps (arXiv 2411.17866, Algorithm 1).
//
// TEST INFRASTRUCTURE.  Only the tests, __graft_entry__.smoke() and the
// CPU-baseline / reference arms of bench.py may load this library
// (through oracle/cxx_oracle.py).  It shares no code, header or table with
// the CUDA library, and neither side includes or links the other.
//
// What it computes, element by element, in the paper's order:
//   * the synthetic gradients standing in for the backward pass of
//     Eq. (dist-opt)'s local losses (a SplitMix64 draw per element);
//   * the local steps, Eq. (local-steps), with the base optimizers of
//     Appendix A: AdamW (Algorithm "AdamW") and Polyak's momentum
//     (Algorithm "Polyak"; plain SGD, Eq. (base-sgd), at mu = 0);
//   * the global step of Algorithm 1: the all-reduce average
//     Delta = (1/n) sum_i (x - x_i) summed over i = 0..n-1, Eqs. (ut-update),
//     (model-update), (mom-update), with the deterministic sign or the
//     randomized signs of Sec. 4.1, Eqs. (rand-sign-2) and (rand-sign-1),
//     driven by Philox4x32-10; then every replica is reset to the new x;
//   * the ablations' global steps (Sec. 5): SlowMo (Appendix A, Algorithm
//     "SlowMo"), signed SlowMo, Lookahead, and the global AdamW step
//     (Appendix, Algorithm "global AdamW");
//   * the per-tensor statistics of each global step, in double, summed in
//     element order.
//
// Precision: fp32, one rounding per operation, no contraction (build with
// -ffp-contract=off and without -ffast-math): this is the same evaluation
// as the numpy oracle (oracle/dsm_oracle.py), which it must equal bit for
// bit.  Derived scalars are computed in double from the fp32
// hyper-parameters and rounded once to fp32.
//
// Every step is elementwise, so a run covers any subset of element indices;
// elements are independent, and OpenMP splits them over threads without
// changing any result (the statistics are summed afterwards, in element
// order, on one thread).
//
// Parity pins: tests/test_cxx_oracle.py checks this oracle against the exact
// d = 8 worked examples (tests/golden/worked_example_d8.json,
// stats_example_d8.json), the published known-answer vectors of SplitMix64
// and Philox4x32-10 (tests/golden/known_answers.json), and the numpy oracle,
// bit for bit, over the workloads' configurations.

#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <vector>

#ifdef _OPENMP
#include <omp.h>
#endif

namespace {

// ---------------------------------------------------------------------------
// Counter-based generators, each from its published definition
// ---------------------------------------------------------------------------

// SplitMix64 (Steele, Lea, Flood, OOPSLA 2014): output j of the generator
// seeded with `state` is state + j * golden gamma, through Stafford's
// variant-13 finaliser.
const uint64_t kGolden = 0x9E3779B97F4A7C15ull;

uint64_t mix64(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

uint64_t sm64(uint64_t state, uint64_t j) { return mix64(state + j * kGolden); }

// Key of the draw family (seed, stream, idx): output 1 + stream * 2^40 + idx of SplitMix64(seed).
// Streams: 0 the step term of the gradient, 1 the worker term, 2 the initial model.
uint64_t family_key(uint64_t seed, uint64_t stream, uint64_t idx) { return sm64(seed, 1 + (stream << 40) + idx); }

// u of element e in [0, 1): output floor(e/2) + 1 of SplitMix64(key), bits 63..40 for even e and
// 39..16 for odd e, times 2^-24 (exact in fp32).
float uniform24(uint64_t key, uint64_t e) {
    const uint64_t h = sm64(key, (e >> 1) + 1);
    const uint64_t b = (e & 1) ? (h >> 16) & 0xFFFFFFull : (h >> 40) & 0xFFFFFFull;
    return static_cast<float>(b) * 5.9604644775390625e-08f;
}

// Round a float to the nearest bfloat16 (ties to even); the result as a float.
float bf16_round(float v) {
    uint32_t b;
    std::memcpy(&b, &v, 4);
    uint32_t r;
    if (std::isnan(v)) {
        r = (b | 0x00400000u) & 0xFFFF0000u;
    } else {
        const uint64_t w = static_cast<uint64_t>(b) + 0x7FFFu + ((b >> 16) & 1u);
        r = static_cast<uint32_t>((w >> 16) << 16);
    }
    float out;
    std::memcpy(&out, &r, 4);
    return out;
}

// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC 2011): ten rounds of the
// two-multiplier S-box, the key bumped by the Weyl constants between rounds.
void philox(const uint32_t in[4], const uint32_t key[2], uint32_t out[4]) {
    uint32_t c0 = in[0], c1 = in[1], c2 = in[2], c3 = in[3], k0 = key[0], k1 = key[1];
    for (int r = 0; r < 10; ++r) {
        if (r > 0) {
            k0 += 0x9E3779B9u;
            k1 += 0xBB67AE85u;
        }
        const uint64_t p0 = static_cast<uint64_t>(0xD2511F53u) * c0;
        const uint64_t p1 = static_cast<uint64_t>(0xCD9E8D57u) * c2;
        const uint32_t n0 = static_cast<uint32_t>(p1 >> 32) ^ c1 ^ k0;
        const uint32_t n1 = static_cast<uint32_t>(p1);
        const uint32_t n2 = static_cast<uint32_t>(p0 >> 32) ^ c3 ^ k1;
        const uint32_t n3 = static_cast<uint32_t>(p0);
        c0 = n0; c1 = n1; c2 = n2; c3 = n3;
    }
    out[0] = c0; out[1] = c1; out[2] = c2; out[3] = c3;
}

// r_e of round t: key (seed mod 2^32, t mod 2^32), counter (floor(e/4) low, high, 0, 0), word e mod 4,
// top 24 bits times 2^-24.
float philox_uniform(uint64_t seed, uint64_t t, uint64_t e) {
    const uint64_t q = e >> 2;
    const uint32_t ctr[4] = {static_cast<uint32_t>(q), static_cast<uint32_t>(q >> 32), 0u, 0u};
    const uint32_t key[2] = {static_cast<uint32_t>(seed), static_cast<uint32_t>(t)};
    uint32_t w[4];
    philox(ctr, key, w);
    return static_cast<float>(w[e & 3] >> 8) * 5.9604644775390625e-08f;
}

// Threads of an element loop: the problem's setting, else OpenMP's default.
int loop_threads(int requested) {
#ifdef _OPENMP
    return requested > 0 ? requested : omp_get_max_threads();
#else
    (void)requested;
    return 1;
#endif
}

// sign(v) = (v > 0) - (v < 0): 0 at +-0 and at NaN.
float sgn(float v) { return static_cast<float>(v > 0.0f) - static_cast<float>(v < 0.0f); }

float f32(double v) { return static_cast<float>(v); }

// beta^j in double, by j successive products of the fp32 beta.
double beta_power(float beta, uint64_t j) {
    double p = 1.0;
    for (uint64_t i = 0; i < j; ++i) p *= static_cast<double>(beta);
    return p;
}

}  // namespace

extern "C" {

struct dsmo_tensor {
    uint64_t numel;
    float grad_scale;
    uint32_t kind;  // 0 weight, 1 bias, 2 LayerNorm weight, 3 LayerNorm bias
    uint32_t wd;    // nonzero: decoupled weight decay applies
};

struct dsmo_hparams {
    int32_t base;        // 0 AdamW, 1 Polyak momentum
    float lr, b1, b2, eps, wd, mu;
    float g_b1, g_b2, g_eta, g_wd;
    int32_t sign_mode;   // 0 sign, 1 Eq. (rand-sign-2), 2 Eq. (rand-sign-1)
    float rsign_B;
    int32_t grad_dtype;  // 0 fp32, 1 bf16
    uint32_t flags;      // bit 1 (value 2): the base optimizer restarts every round
    uint64_t seed;
    int32_t global_mode; // 0 Algorithm 1, 1 SlowMo, 2 signed SlowMo, 3 Lookahead, 4 global AdamW
    float g_eps;
};

struct dsmo_stats {
    double delta_sq, drift;
    uint64_t zero_sign, flips, unanimous, clamped;
};

// A problem over a subset of elements: per element its tensor, gradient scales, kind and decay flag.
struct dsmo_problem {
    uint32_t n, num_tensors;
    dsmo_hparams hp;
    uint64_t count;
    std::vector<uint64_t> elem;  // index in the larger model (first_element + logical index)
    std::vector<uint32_t> tensor;
    std::vector<float> scale, scale2;
    std::vector<uint32_t> kind, wd;
    int threads;
};

// The problem over elements elems[0..count) (logical indices into the packed tensor list; each must lie
// inside the model).  first_element: the layout's first element within a larger model of which it is a
// contiguous part (a parameter shard); the generators and the Philox counter take element e as element
// first_element + e of that model (0 for a whole model).  threads <= 0: OpenMP's default.  Returns NULL
// if an element lies outside the model.
dsmo_problem* dsmo_create(const dsmo_tensor* tensors, uint32_t num_tensors, uint32_t n, const dsmo_hparams* hp,
                          const int64_t* elems, uint64_t count, uint64_t first_element, int threads) {
    std::vector<uint64_t> starts(num_tensors + 1, 0);
    for (uint32_t T = 0; T < num_tensors; ++T) starts[T + 1] = starts[T] + tensors[T].numel;
    dsmo_problem* p = new dsmo_problem();
    p->n = n;
    p->num_tensors = num_tensors;
    p->hp = *hp;
    p->count = count;
    p->threads = threads;
    p->elem.resize(count);
    p->tensor.resize(count);
    p->scale.resize(count);
    p->scale2.resize(count);
    p->kind.resize(count);
    p->wd.resize(count);
    for (uint64_t k = 0; k < count; ++k) {
        const int64_t e = elems[k];
        if (e < 0 || static_cast<uint64_t>(e) >= starts[num_tensors]) {
            delete p;
            return nullptr;
        }
        // the tensor holding e: the last one whose start is <= e (empty tensors hold nothing)
        const uint32_t T = static_cast<uint32_t>(
            std::upper_bound(starts.begin(), starts.end(), static_cast<uint64_t>(e)) - starts.begin() - 1);
        p->elem[k] = first_element + static_cast<uint64_t>(e);  // its index in the larger model
        p->tensor[k] = T;
        p->scale[k] = tensors[T].grad_scale;
        p->scale2[k] = 0.1f * tensors[T].grad_scale;
        p->kind[k] = tensors[T].kind;
        p->wd[k] = tensors[T].wd != 0;
    }
    return p;
}

void dsmo_destroy(dsmo_problem* p) { delete p; }

// The initial model x_{0,0} (the paper gives none): weights 0.02 * (2u - 1) with u from stream 2,
// LayerNorm weights 1, biases and LayerNorm biases 0.
void dsmo_init_x0(const dsmo_problem* p, float* x) {
    const uint64_t key = family_key(p->hp.seed, 2, 0);
    for (uint64_t k = 0; k < p->count; ++k) {
        const float u = uniform24(key, p->elem[k]);
        float v = 0.0f;
        if (p->kind[k] == 0) v = 0.02f * (2.0f * u - 1.0f);
        else if (p->kind[k] == 2) v = 1.0f;
        x[k] = v;
    }
}

// Synthetic gradient of worker i at local step `step` on the problem's elements:
// g = s * (u(seed, 0, step) - 1/2) + fp32(0.1 s) * (u(seed, 1, i) - 1/2), left to right, then rounded to
// bfloat16 for bf16 gradients.
void dsmo_synthetic_grad(const dsmo_problem* p, uint64_t step, uint32_t worker, float* g) {
    const uint64_t ks = family_key(p->hp.seed, 0, step), kw = family_key(p->hp.seed, 1, worker);
    for (uint64_t k = 0; k < p->count; ++k) {
        const float a = p->scale[k] * (uniform24(ks, p->elem[k]) - 0.5f);
        const float b = p->scale2[k] * (uniform24(kw, p->elem[k]) - 0.5f);
        const float v = a + b;
        g[k] = p->hp.grad_dtype == 1 ? bf16_round(v) : v;
    }
}

// Local step k of the round on every worker (Eq. (local-steps)): X, opt_m, opt_v are [n][count].
// grads: [n][count] fp32 values (bf16 values widened), or NULL for the synthetic gradients of local step
// index `step`.  j: AdamW's step count (>= 1).  gamma: the round's learning rate.
void dsmo_local_step(const dsmo_problem* p, float* X, float* opt_m, float* opt_v, const float* grads,
                     uint64_t step, uint64_t j, float gamma) {
    const dsmo_hparams& h = p->hp;
    const uint64_t cnt = p->count;
    const uint32_t n = p->n;
    // AdamW's scalars: 1 - beta, bias corrections 1 - beta^j, in double, rounded once
    const float b1 = h.b1, b2 = h.b2, omb1 = f32(1.0 - h.b1), omb2 = f32(1.0 - h.b2);
    const float bc1 = f32(1.0 - beta_power(h.b1, j)), bc2 = f32(1.0 - beta_power(h.b2, j));
    const float lr = gamma, eps = h.eps, wd = h.wd, mu = h.mu;
    const uint64_t ks = family_key(h.seed, 0, step);
    std::vector<uint64_t> kw(n);
    for (uint32_t i = 0; i < n; ++i) kw[i] = family_key(h.seed, 1, i);
    const int nt = loop_threads(p->threads);
    (void)nt;  // unused when built without OpenMP
#pragma omp parallel for schedule(static) num_threads(nt)
    for (int64_t kk = 0; kk < static_cast<int64_t>(cnt); ++kk) {
        const uint64_t k = static_cast<uint64_t>(kk);
        const uint64_t e = p->elem[k];
        const float a = grads ? 0.0f : p->scale[k] * (uniform24(ks, e) - 0.5f);
        const float lam = p->wd[k] ? wd : 0.0f;
        for (uint32_t i = 0; i < n; ++i) {
            const uint64_t o = static_cast<uint64_t>(i) * cnt + k;
            float g;
            if (grads) {
                g = grads[o];
            } else {
                const float v = a + p->scale2[k] * (uniform24(kw[i], e) - 0.5f);
                g = h.grad_dtype == 1 ? bf16_round(v) : v;
            }
            float x = X[o];
            if (h.base == 0) {  // AdamW (Appendix A)
                float m = opt_m[o], v = opt_v[o];
                m = b1 * m + omb1 * g;
                v = b2 * v + omb2 * (g * g);
                const float mhat = m / bc1;
                const float vhat = v / bc2;
                x = x - lr * (mhat / (std::sqrt(vhat) + eps) + lam * x);
                opt_m[o] = m;
                opt_v[o] = v;
            } else {            // Polyak momentum (Appendix A)
                float b = opt_m[o];
                b = mu * b + g;
                x = x - lr * b;
                opt_m[o] = b;
            }
            X[o] = x;
        }
    }
}

// The global step of round t and the reset of every replica (Algorithm 1), or an ablation's global step
// (hp.global_mode).  x, m, gv (global AdamW's second moment; may be NULL otherwise) are [count]; X is
// [n][count].  stats: NULL or num_tensors entries.  delta, u, sg: NULL or [count] outputs of the
// average, the signed vector and the applied sign.  r: NULL (Philox4x32-10 of round t) or [count]
// uniforms for the randomized sign; lam: NULL (hp.g_wd where the tensor decays) or [count] decays.
void dsmo_global_step(const dsmo_problem* p, float* x, float* m, float* gv, float* X, float gamma, uint64_t t,
                      dsmo_stats* stats, float* delta_out, float* u_out, float* sg_out, const float* r_in,
                      const float* lam_in) {
    const dsmo_hparams& h = p->hp;
    const uint64_t cnt = p->count;
    const uint32_t n = p->n;
    const int mode = h.global_mode;
    const int sign_mode = mode == 0 ? h.sign_mode : 0;
    const float c1 = f32((1.0 - h.g_b1) / gamma), c2 = f32((1.0 - h.g_b2) / gamma);
    const float eg = f32(static_cast<double>(h.g_eta) * gamma);
    const float inv_g = f32(1.0 / gamma);
    const float B = h.rsign_B;
    const float gomb1 = f32(1.0 - h.g_b1), gomb2 = f32(1.0 - h.g_b2);
    const float gbc1 = f32(1.0 - beta_power(h.g_b1, t + 1)), gbc2 = f32(1.0 - beta_power(h.g_b2, t + 1));
    // per-element terms of the statistics, summed in element order afterwards
    std::vector<double> dsq(stats ? cnt : 0), drift(stats ? cnt : 0);
    std::vector<uint8_t> zero(stats ? cnt : 0), flip(stats ? cnt : 0), unan(stats ? cnt : 0), clamp(stats ? cnt : 0);
    const int nt = loop_threads(p->threads);
    (void)nt;  // unused when built without OpenMP
#pragma omp parallel for schedule(static) num_threads(nt)
    for (int64_t kk = 0; kk < static_cast<int64_t>(cnt); ++kk) {
        const uint64_t k = static_cast<uint64_t>(kk);
        const float xv = x[k], mv = m[k];
        const float lam = lam_in ? lam_in[k] : (p->wd[k] ? h.g_wd : 0.0f);
        // the all-reduce average of the worker differences, summed in worker order
        float acc = 0.0f;
        for (uint32_t i = 0; i < n; ++i) acc = acc + (xv - X[static_cast<uint64_t>(i) * cnt + k]);
        const float D = acc / static_cast<float>(n);
        float u, s, x_new, m_new;
        if (mode == 0) {         // Algorithm 1: Eqs. (ut-update), (model-update), (mom-update)
            u = h.g_b1 * mv + c1 * D;
            s = sgn(u);
            if (sign_mode != 0) {  // Sec. 4.1: p = min(|u|/B, 1) (NaN stays NaN), then Eq. (rand-sign-2) or (1)
                const float r = r_in ? r_in[k] : philox_uniform(h.seed, t, p->elem[k]);
                const float a = std::fabs(u) / B;
                const float pr = std::isnan(a) ? a : (a < 1.0f ? a : 1.0f);
                if (sign_mode == 1) s = r < pr ? s : 0.0f;
                else s = r < 0.5f + 0.5f * pr ? s : -s;
            }
            x_new = xv - eg * (s + lam * xv);
            m_new = h.g_b2 * mv + c2 * D;
        } else if (mode == 1) {  // SlowMo: u <- beta u + (1/gamma) Delta, x' = x - alpha gamma u
            u = h.g_b1 * mv + inv_g * D;
            s = sgn(u);
            x_new = xv - eg * u;
            m_new = u;
        } else if (mode == 2) {  // signed SlowMo: the sign of the average enters u
            const float sd = sgn(D);
            u = h.g_b1 * mv + c1 * sd;
            s = sd;
            x_new = xv - eg * u;
            m_new = h.g_b2 * mv + c2 * D;
        } else if (mode == 3) {  // Lookahead: Algorithm 1 with x' = x - eta gamma u
            u = h.g_b1 * mv + c1 * D;
            s = sgn(u);
            x_new = xv - eg * u;
            m_new = h.g_b2 * mv + c2 * D;
        } else {                 // global AdamW on the pseudo-gradient Delta / gamma
            const float g = inv_g * D;
            m_new = h.g_b1 * mv + gomb1 * g;
            const float v_new = h.g_b2 * gv[k] + gomb2 * (g * g);
            const float mhat = m_new / gbc1;
            const float vhat = v_new / gbc2;
            x_new = xv - h.g_eta * (mhat / (std::sqrt(vhat) + h.g_eps) + lam * xv);
            gv[k] = v_new;
            u = m_new;
            s = sgn(u);
        }
        if (stats) {
            const double Dd = static_cast<double>(D);
            const float sD = sgn(D);
            dsq[k] = Dd * Dd;
            double dr = 0.0;
            bool all = true;
            for (uint32_t i = 0; i < n; ++i) {
                const float di = xv - X[static_cast<uint64_t>(i) * cnt + k];
                const double ei = static_cast<double>(di) - Dd;
                dr += ei * ei;
                all = all && (sgn(di) == sD);
            }
            drift[k] = dr;
            zero[k] = s == 0.0f;
            flip[k] = sgn(u) != sD;
            unan[k] = all;
            clamp[k] = sign_mode != 0 && std::fabs(u) > B;
        }
        if (delta_out) delta_out[k] = D;
        if (u_out) u_out[k] = u;
        if (sg_out) sg_out[k] = s;
        x[k] = x_new;
        m[k] = m_new;
        for (uint32_t i = 0; i < n; ++i) X[static_cast<uint64_t>(i) * cnt + k] = x_new;  // synchronise
    }
    if (stats) {
        for (uint32_t T = 0; T < p->num_tensors; ++T) stats[T] = dsmo_stats{0.0, 0.0, 0, 0, 0, 0};
        for (uint64_t k = 0; k < cnt; ++k) {  // element order
            dsmo_stats& st = stats[p->tensor[k]];
            st.delta_sq += dsq[k];
            st.drift += drift[k];
            st.zero_sign += zero[k];
            st.flips += flip[k];
            st.unanimous += unan[k];
            st.clamped += clamp[k];
        }
    }
}

// The generators on their own, for the known-answer pins.
uint64_t dsmo_splitmix64_output(uint64_t state, uint64_t j) { return sm64(state, j); }
void dsmo_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]) { philox(ctr, key, out); }
float dsmo_philox_uniform(uint64_t seed, uint64_t t, uint64_t e) { return philox_uniform(seed, t, e); }
float dsmo_uniform24(uint64_t seed, uint64_t stream, uint64_t idx, uint64_t e) {
    return uniform24(family_key(seed, stream, idx), e);
}
float dsmo_bf16_round(float v) { return bf16_round(v); }
int dsmo_max_threads(void) { return loop_threads(0); }

}  // extern "C"
