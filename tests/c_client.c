/* A client of the C ABI in plain C99, with no Python and no torch: it
 * allocates the arena with cudaMalloc, runs rounds of Algorithm 1
 * (synthetic gradients, tau local steps, global step with statistics)
 * through include/dsm.h, and prints the per-tensor statistics and the
 * global model x as fp32 bit patterns.  tests/test_c_client.py builds it
 * and compares its output with the CPU oracle.
 *
 * usage: c_client adamw|sgdm <rounds>
 *   adamw: AdamW base, deterministic sign, fused round, n = 3, tau = 2
 *   sgdm:  SGD-momentum base, randomized sign (Eq. (rand-sign-2), B = 1e-2),
 *          unfused, n = 4, tau = 3
 */
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <cuda_runtime.h>

#include "dsm.h"

static int fail(const char* what, int rc) {
    fprintf(stderr, "%s failed: %d (%s)\n", what, rc, dsm_last_error());
    return 1;
}

int main(int argc, char** argv) {
    const dsm_tensor tensors[3] = {
        {5000, 1e-2f, DSM_KIND_WEIGHT, 1, 0},
        {77, 1e-3f, DSM_KIND_BIAS, 1, 0},
        {2048, 1e-3f, DSM_KIND_LN_W, 1, 0},
    };
    const uint32_t count = 3;
    const dsm_layout layout = {tensors, count, 0};  /* a whole model: first_element 0 */
    dsm_hparams hp;
    uint32_t n, tau;
    int rounds;
    if (argc != 3 || (strcmp(argv[1], "adamw") != 0 && strcmp(argv[1], "sgdm") != 0)) {
        fprintf(stderr, "usage: %s adamw|sgdm <rounds>\n", argv[0]);
        return 2;
    }
    rounds = atoi(argv[2]);
    memset(&hp, 0, sizeof hp);
    hp.b1 = 0.9f;
    hp.b2 = 0.95f;
    hp.eps = 1e-8f;
    hp.wd = 0.1f;
    hp.mu = 0.9f;
    hp.g_b1 = 0.9f;
    hp.g_b2 = 0.99f;
    hp.g_eta = 1e-3f;
    hp.g_wd = 0.1f;
    hp.rsign_B = 1e-2f;
    hp.grad_dtype = DSM_F32;
    hp.seed = 0;
    hp.global_mode = DSM_GLOBAL_SIGN_MOMENTUM;
    hp.g_eps = 1e-8f;
    if (strcmp(argv[1], "adamw") == 0) {
        hp.base = DSM_BASE_ADAMW;
        hp.lr = 6e-4f;
        hp.sign_mode = DSM_SIGN;
        hp.flags = DSM_FLAG_FUSED_ROUND;
        n = 3;
        tau = 2;
    } else {
        hp.base = DSM_BASE_SGDM;
        hp.lr = 1e-2f;
        hp.sign_mode = DSM_RSIGN_ZERO;
        hp.flags = 0;
        n = 4;
        tau = 3;
    }

    const size_t bytes = dsm_state_bytes(&layout, n, &hp);
    if (bytes == 0) return fail("dsm_state_bytes", DSM_EINVAL);
    void* arena = NULL;
    if (cudaMalloc(&arena, bytes) != cudaSuccess) return fail("cudaMalloc", DSM_ECUDA);
    cudaStream_t stream;
    if (cudaStreamCreate(&stream) != cudaSuccess) return fail("cudaStreamCreate", DSM_ECUDA);
    dsm_handle* h = NULL;
    int rc = dsm_create(&layout, n, tau, &hp, arena, bytes, NULL, 0, stream, &h);
    if (rc != DSM_OK) return fail("dsm_create", rc);

    dsm_tensor_stats stats[3];
    for (int t = 0; t < rounds; ++t) {
        for (uint32_t k = 0; k < tau; ++k) {
            if ((rc = dsm_fill_synthetic_grads(h, (uint64_t)t * tau + k, stream)) != DSM_OK)
                return fail("dsm_fill_synthetic_grads", rc);
            if ((rc = dsm_local_step(h, stream)) != DSM_OK) return fail("dsm_local_step", rc);
        }
        if ((rc = dsm_global_step(h, stream, stats, count)) != DSM_OK) return fail("dsm_global_step", rc);
    }

    dsm_info info;
    if ((rc = dsm_get_info(h, &info)) != DSM_OK) return fail("dsm_get_info", rc);
    float* x = (float*)malloc(info.d * sizeof(float));
    if (!x) return fail("malloc", DSM_ENOMEM);
    if ((rc = dsm_read_params(h, DSM_BUF_X, 0, x, 0, info.d, 0, stream)) != DSM_OK)
        return fail("dsm_read_params", rc);
    printf("d %llu round %llu\n", (unsigned long long)info.d, (unsigned long long)info.round);
    for (uint32_t i = 0; i < count; ++i)
        printf("stats %u %.17g %.17g %llu %llu %llu %llu\n", i, stats[i].delta_sq, stats[i].drift,
               (unsigned long long)stats[i].zero_sign, (unsigned long long)stats[i].flips,
               (unsigned long long)stats[i].unanimous, (unsigned long long)stats[i].clamped);
    for (uint64_t e = 0; e < info.d; ++e) {
        uint32_t bits;
        memcpy(&bits, &x[e], sizeof bits);
        printf("%08x\n", bits);
    }
    free(x);
    dsm_destroy(h);
    cudaStreamDestroy(stream);
    cudaFree(arena);
    return 0;
}
