/*
 * abi_parity.c -- a plain C caller of libspire: builds small seeded inputs,
 * runs spire_verify_attention and spire_draft_sparse_attention through the C
 * ABI (device buffers from the CUDA runtime, the default stream), and checks
 * the results against the fp64 oracle compiled into this test program (whole
 * tensor: relative L2 <= 1e-3 and max |diff| <= 1e-2).  Prints "ok" and exits
 * 0 on success.  Test code: it links the oracle, the library does not.
 */
#include <math.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <cuda_runtime_api.h>

#include "spire.h"

/* the oracle's entry points (oracle/spire_oracle.c) */
int64_t oracle_verify(const uint16_t *q, const uint16_t *k_cache, const uint16_t *v_cache,
                      const int32_t *block_table, const int32_t *ctx_lens, int32_t B, int32_t k,
                      int32_t Hq, int32_t Hkv, int32_t D, int32_t page_size, int32_t max_pages,
                      int32_t num_pages, double scale, const uint8_t *unit_mask, double *out,
                      int32_t n_threads);
int64_t oracle_draft_ring(const uint16_t *q, const uint16_t *kv, const int32_t *ctx_lens,
                          int32_t B, int32_t Hq, int32_t Hkv, int32_t D, int32_t n_sink,
                          int32_t window, double scale, const uint8_t *unit_mask, double *out,
                          int32_t n_threads);

static uint64_t rng_state = 0x9e3779b97f4a7c15ull;

/* a uniform value in [-1, 1) from a 64-bit linear congruential step */
static double uniform(void)
{
    rng_state = rng_state * 6364136223846793005ull + 1442695040888963407ull;
    return (double)(rng_state >> 11) * (2.0 / 9007199254740992.0) - 1.0;
}

/* bf16 bits of a float (round to nearest even; inputs here are finite) */
static uint16_t to_bf16(float f)
{
    uint32_t u;
    memcpy(&u, &f, 4);
    u += 0x7fffu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

static void fill_bf16(uint16_t *a, size_t n, double amp)
{
    for (size_t i = 0; i < n; ++i)
        a[i] = to_bf16((float)(amp * uniform()));
}

#define CHECK_CUDA(x)                                                            \
    do {                                                                         \
        cudaError_t e_ = (x);                                                    \
        if (e_ != cudaSuccess) {                                                 \
            fprintf(stderr, "%s: %s\n", #x, cudaGetErrorString(e_));            \
            return 1;                                                            \
        }                                                                        \
    } while (0)

#define CHECK_SPIRE(x)                                                           \
    do {                                                                         \
        spire_status s_ = (x);                                                   \
        if (s_ != SPIRE_OK) {                                                    \
            fprintf(stderr, "%s: %s\n", #x, spire_status_string(s_));           \
            return 1;                                                            \
        }                                                                        \
    } while (0)

static int compare(const char *what, const float *got, const double *ref, size_t n)
{
    double num = 0.0, den = 0.0, mx = 0.0;
    for (size_t i = 0; i < n; ++i) {
        const double d = (double)got[i] - ref[i];
        if (!(fabs(d) <= 1e30)) {
            fprintf(stderr, "%s: non-finite output at %zu\n", what, i);
            return 1;
        }
        num += d * d;
        den += ref[i] * ref[i];
        if (fabs(d) > mx) mx = fabs(d);
    }
    const double rel = sqrt(num / (den > 0.0 ? den : 1.0));
    printf("%s: rel-L2 %.3e, max-abs %.3e over %zu values\n", what, rel, mx, n);
    return (rel <= 1e-3 && mx <= 1e-2) ? 0 : 1;
}

static int run_verify(void)
{
    enum { B = 3, K = 4, HQ = 8, HKV = 2, D = 64, PAGE = 64, MAXP = 5 };
    const int32_t ctx[B] = {70, 300, 5};
    const int num_pages = 2 * B * MAXP;
    const size_t nq = (size_t)B * (K + 1) * HQ * D;
    const size_t nkv = (size_t)num_pages * HKV * PAGE * D;
    uint16_t *q = malloc(nq * 2), *kc = malloc(nkv * 2), *vc = malloc(nkv * 2);
    int32_t bt[B * MAXP];
    float *out = malloc(nq * 4);
    double *ref = malloc(nq * sizeof(double));
    if (!q || !kc || !vc || !out || !ref) return 1;
    fill_bf16(q, nq, 0.125);
    fill_bf16(kc, nkv, 1.0);
    fill_bf16(vc, nkv, 1.0);
    /* pages in a scattered order: sequence b, page t -> 2 (t B + b) + 1 */
    for (int b = 0; b < B; ++b)
        for (int t = 0; t < MAXP; ++t)
            bt[b * MAXP + t] = 2 * (t * B + b) + 1;

    spire_attn_desc desc = {B, HQ, HKV, D, PAGE, MAXP, num_pages, 1.0f};
    const size_t ws_bytes = spire_verify_workspace_bytes(&desc, K);
    if (!ws_bytes) return 1;
    void *dq, *dk, *dv, *dbt, *dctx, *dout, *dws;
    CHECK_CUDA(cudaMalloc(&dq, nq * 2));
    CHECK_CUDA(cudaMalloc(&dk, nkv * 2));
    CHECK_CUDA(cudaMalloc(&dv, nkv * 2));
    CHECK_CUDA(cudaMalloc(&dbt, sizeof bt));
    CHECK_CUDA(cudaMalloc(&dctx, sizeof ctx));
    CHECK_CUDA(cudaMalloc(&dout, nq * 4));
    CHECK_CUDA(cudaMalloc(&dws, ws_bytes));
    CHECK_CUDA(cudaMemcpy(dq, q, nq * 2, cudaMemcpyHostToDevice));
    CHECK_CUDA(cudaMemcpy(dk, kc, nkv * 2, cudaMemcpyHostToDevice));
    CHECK_CUDA(cudaMemcpy(dv, vc, nkv * 2, cudaMemcpyHostToDevice));
    CHECK_CUDA(cudaMemcpy(dbt, bt, sizeof bt, cudaMemcpyHostToDevice));
    CHECK_CUDA(cudaMemcpy(dctx, ctx, sizeof ctx, cudaMemcpyHostToDevice));
    CHECK_SPIRE(spire_verify_attention(dq, dk, dv, (const int32_t *)dbt, (const int32_t *)dctx,
                                       K, &desc, (float *)dout, dws, ws_bytes, NULL));
    int32_t code = -1;
    CHECK_SPIRE(spire_get_device_error(dws, &code, NULL));
    if (code != 0) {
        fprintf(stderr, "verify: device error %d\n", code);
        return 1;
    }
    CHECK_CUDA(cudaMemcpy(out, dout, nq * 4, cudaMemcpyDeviceToHost));
    if (oracle_verify(q, kc, vc, bt, ctx, B, K, HQ, HKV, D, PAGE, MAXP, num_pages, 1.0, NULL,
                      ref, 4) != 0)
        return 1;
    const int rc = compare("verify", out, ref, nq);
    cudaFree(dq); cudaFree(dk); cudaFree(dv); cudaFree(dbt); cudaFree(dctx);
    cudaFree(dout); cudaFree(dws);
    free(q); free(kc); free(vc); free(out); free(ref);
    return rc;
}

static int run_draft(void)
{
    enum { B = 3, HQ = 4, HKV = 1, D = 128, NS = 4, W = 128 };
    const int32_t t[B] = {3, 100, 700};
    const size_t nq = (size_t)B * HQ * D;
    const size_t nkv = (size_t)B * 2 * HKV * (NS + W) * D;
    uint16_t *q = malloc(nq * 2), *kv = malloc(nkv * 2);
    float *out = malloc(nq * 4);
    double *ref = malloc(nq * sizeof(double));
    if (!q || !kv || !out || !ref) return 1;
    fill_bf16(q, nq, 0.09);
    fill_bf16(kv, nkv, 1.0);

    spire_attn_desc desc = {B, HQ, HKV, D, 64, 0, 0, 1.0f};
    const size_t ws_bytes = spire_draft_workspace_bytes(&desc, NS, W);
    if (!ws_bytes) return 1;
    void *dq, *dkv, *dt, *dout, *dws;
    CHECK_CUDA(cudaMalloc(&dq, nq * 2));
    CHECK_CUDA(cudaMalloc(&dkv, nkv * 2));
    CHECK_CUDA(cudaMalloc(&dt, sizeof t));
    CHECK_CUDA(cudaMalloc(&dout, nq * 4));
    CHECK_CUDA(cudaMalloc(&dws, ws_bytes));
    CHECK_CUDA(cudaMemcpy(dq, q, nq * 2, cudaMemcpyHostToDevice));
    CHECK_CUDA(cudaMemcpy(dkv, kv, nkv * 2, cudaMemcpyHostToDevice));
    CHECK_CUDA(cudaMemcpy(dt, t, sizeof t, cudaMemcpyHostToDevice));
    CHECK_SPIRE(spire_draft_sparse_attention(dq, dkv, (const int32_t *)dt, NS, W, &desc,
                                             (float *)dout, dws, ws_bytes, NULL));
    int32_t code = -1;
    CHECK_SPIRE(spire_get_device_error(dws, &code, NULL));
    if (code != 0) {
        fprintf(stderr, "draft: device error %d\n", code);
        return 1;
    }
    CHECK_CUDA(cudaMemcpy(out, dout, nq * 4, cudaMemcpyDeviceToHost));
    if (oracle_draft_ring(q, kv, t, B, HQ, HKV, D, NS, W, 1.0, NULL, ref, 4) != 0)
        return 1;
    const int rc = compare("draft", out, ref, nq);
    cudaFree(dq); cudaFree(dkv); cudaFree(dt); cudaFree(dout); cudaFree(dws);
    free(q); free(kv); free(out); free(ref);
    return rc;
}

int main(void)
{
    if (run_verify() || run_draft()) return 1;
    printf("ok\n");
    return 0;
}
