/*
 * abi_client.c -- a plain C client of libbarycache.so, with no Python in between.
 *
 *   abi_client host     host-only calls (weights, footprints, schedules, errors): no GPU
 *   abi_client hostcost host time of bc_forecast calls on small caches of 1-64 layers
 *                       (launch included; the GPU work is tiny), and per tensor of
 *                       forecasts and pushes over 4096 and 65,536 tensors, one JSON line per
 *                       size
 *   abi_client device   one cache on the current GPU: allocate with cudaMalloc, push three
 *                       full-step features, forecast, read back, and compare every element
 *                       with the fp64 oracle (liboracle, linked for the check only); then
 *                       the probe drift of the two newest slots against the oracle's
 *   abi_client manylayers 2048 ragged tensors: pushes and a forecast of one launch each
 *                       through the device layer tables (oracle on every element, a planted
 *                       NaN), then the same history as slot images through bc_cache_push_flat
 *                       and bc_forecast_flat, bit for bit the per-layer forecast
 *
 * Exit status 0 on success; a failing check prints what failed and exits 1.
 */
#define _POSIX_C_SOURCE 199309L
#include <math.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>
#include <time.h>

#include "barycache.h"

/* The oracle's C entry points (test infrastructure). */
int oracle_paper_weights(const double *s, int m, double t, double delta, double lambda, double C,
                         double eta, double *W);
void oracle_combine(int dtype, const void *const *F, int m, const double *W, int64_t n,
                    double *out, double *bound);
void oracle_drift(int dtype, const void *cur, const void *prev, int64_t n, double *out);

/* The few CUDA runtime calls the device check needs, declared here so that the client
 * compiles with a plain C compiler against libcudart. */
typedef int cudaError_t;
extern cudaError_t cudaMalloc(void **p, size_t n);
extern cudaError_t cudaFree(void *p);
extern cudaError_t cudaMemcpy(void *dst, const void *src, size_t n, int kind);
extern cudaError_t cudaDeviceSynchronize(void);
#define H2D 1
#define D2H 2

static int failures = 0;
#define CHECK(cond, ...)                                                     \
    do {                                                                     \
        if (!(cond)) {                                                       \
            fprintf(stderr, "FAILED %s:%d: ", __FILE__, __LINE__);          \
            fprintf(stderr, __VA_ARGS__);                                    \
            fprintf(stderr, "\n");                                           \
            ++failures;                                                      \
        }                                                                    \
    } while (0)

static int host_checks(void) {
    bc_params p;
    bc_params_default(&p);
    CHECK(p.mode == BC_MODE_PAPER && p.clip_C == 10.0, "defaults");

    /* Exact mode: one step past three equispaced nodes is (3, -3, 1). */
    double nodes[3] = {940.0, 960.0, 980.0}, c[3];
    p.mode = BC_MODE_EXACT;
    CHECK(bc_solve(nodes, 3, 920.0, &p, c) == BC_OK, "bc_solve exact");
    CHECK(fabs(c[0] - 3) < 1e-12 && fabs(c[1] + 3) < 1e-12 && fabs(c[2] - 1) < 1e-12,
          "exact weights %g %g %g", c[0], c[1], c[2]);

    /* Paper mode against the oracle's independent implementation. */
    bc_params_default(&p);
    double w_ref[3];
    CHECK(bc_solve(nodes, 3, 920.0, &p, c) == BC_OK, "bc_solve paper");
    oracle_paper_weights(nodes, 3, 920.0, 0.95, 0.0, 10.0, 1e-12, w_ref);
    for (int j = 0; j < 3; ++j) CHECK(fabs(c[j] - w_ref[j]) < 1e-12, "paper weight %d", j);

    /* Footprint of the 60-layer video cache at K = 3 and the equal-spaced schedule. */
    int64_t numels[60], bytes = 0;
    for (int l = 0; l < 60; ++l) numels[l] = (int64_t)118800 * 3072;
    CHECK(bc_cache_bytes_for(numels, 60, 3, BC_DTYPE_BF16, &bytes) == BC_OK &&
              bytes == 131383296000LL, "footprint %lld", (long long)bytes);
    uint8_t full[50];
    int n_full = 0;
    CHECK(bc_schedule_equal(50, 4, 2, full) == BC_OK, "schedule");
    for (int i = 0; i < 50; ++i) n_full += full[i];
    CHECK(n_full == 14, "full steps %d", n_full);

    /* Errors come back as codes with a message. */
    double dup[2] = {0.5, 0.5};
    p.mode = BC_MODE_EXACT;
    CHECK(bc_solve(dup, 2, 0.4, &p, c) == BC_ERR_DUPLICATE_NODE && bc_last_error()[0] != 0,
          "duplicate nodes");
    CHECK(bc_cache_bytes(NULL, &bytes) == BC_ERR_BAD_HANDLE, "null handle");
    CHECK(strcmp(bc_status_string(BC_OK), "ok") == 0, "status string");
    return failures;
}

/* bf16 bit pattern of a float (round to nearest even), for the test data. */
static uint16_t to_bf16(float f) {
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    u += 0x7FFFu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

static int device_checks(void) {
    const int64_t n = 3 * 8192 * 16 + 77;   /* several tiles and a ragged tail */
    const double times[3] = {0.9, 0.85, 0.8};
    const double t_new = 0.75;
    uint16_t *host[3];
    void *dev_in = NULL, *dev_out = NULL;
    bc_handle h = NULL;
    for (int k = 0; k < 3; ++k) {
        host[k] = (uint16_t *)malloc(n * sizeof(uint16_t));
        for (int64_t e = 0; e < n; ++e) {
            const double a = sin(0.001 * e), b = cos(0.0007 * e), q = 0.3 * sin(0.0003 * e);
            host[k][e] = to_bf16((float)(a + b * times[k] + q * times[k] * times[k]));
        }
    }
    CHECK(bc_cache_create(&n, 1, 3, BC_DTYPE_BF16, NULL, &h) == BC_OK, "create: %s",
          bc_last_error());
    CHECK(cudaMalloc(&dev_in, n * 2) == 0 && cudaMalloc(&dev_out, n * 2) == 0, "cudaMalloc");
    for (int k = 0; k < 3 && !failures; ++k) {
        CHECK(cudaMemcpy(dev_in, host[k], n * 2, H2D) == 0, "upload");
        const void *ptrs[1] = {dev_in};
        CHECK(bc_cache_push(h, ptrs, times[k], NULL) == BC_OK, "push: %s", bc_last_error());
        cudaDeviceSynchronize();
    }
    void *outs[1] = {dev_out};
    CHECK(bc_forecast(h, t_new, outs, BC_DTYPE_BF16, NULL) == BC_OK, "forecast: %s",
          bc_last_error());
    CHECK(bc_cache_check(h) == BC_OK, "device status");
    uint16_t *got = (uint16_t *)malloc(n * 2);
    CHECK(cudaMemcpy(got, dev_out, n * 2, D2H) == 0, "download");

    double nodes[3] = {times[2], times[1], times[0]}, W[3];
    oracle_paper_weights(nodes, 3, t_new, 0.95, 0.0, 10.0, 1e-12, W);
    const void *F[3] = {host[2], host[1], host[0]};
    double *ref = (double *)malloc(n * sizeof(double)), *bound = (double *)malloc(n * sizeof(double));
    oracle_combine(1, F, 3, W, n, ref, bound);
    int64_t bad = 0;
    for (int64_t e = 0; e < n; ++e) {
        uint32_t u = (uint32_t)got[e] << 16;
        float g;
        memcpy(&g, &u, sizeof g);
        if (!(fabs((double)g - ref[e]) <= ldexp(1.0, -8) * bound[e])) ++bad;
    }
    CHECK(bad == 0, "%lld of %lld elements outside 2^-8 * sum |W||F|", (long long)bad,
          (long long)n);
    /* probe drift between the two newest slots (device) and the same arrays (oracle) */
    void *s0[1], *s1[1];
    double *dev_drift = NULL, drift[3], ref_drift[3];
    CHECK(bc_cache_slot_ptrs(h, 0, s0) == BC_OK && bc_cache_slot_ptrs(h, 1, s1) == BC_OK,
          "slot pointers");
    CHECK(cudaMalloc((void **)&dev_drift, sizeof drift) == 0, "cudaMalloc drift");
    CHECK(bc_probe_drift(h, s0[0], s1[0], n, BC_DTYPE_BF16, dev_drift, NULL) == BC_OK,
          "probe drift: %s", bc_last_error());
    CHECK(cudaMemcpy(drift, dev_drift, sizeof drift, D2H) == 0, "download drift");
    CHECK(bc_cache_check(h) == BC_OK, "device status after the drift");
    oracle_drift(1, host[2], host[1], n, ref_drift);
    for (int i = 0; i < 3; ++i)
        CHECK(fabs(drift[i] - ref_drift[i]) <= 2e-6 * fabs(ref_drift[i]),
              "drift[%d] = %.17g, oracle %.17g", i, drift[i], ref_drift[i]);
    cudaFree(dev_drift);
    bc_stats st;
    CHECK(bc_cache_stats(h, &st) == BC_OK && st.forecasts == 1 && st.pushes == 3, "stats");
    bc_cache_destroy(h);
    cudaFree(dev_in);
    cudaFree(dev_out);
    for (int k = 0; k < 3; ++k) free(host[k]);
    free(got);
    free(ref);
    free(bound);
    return failures;
}

/* A blockwise-style cache of 2048 ragged bf16 tensors: pushes and the forecast each run as
 * one launch (the layer tables travel through the handle's device copies), every element of
 * every tensor matches the oracle, and a NaN planted in one stored value comes out as NaN. */
/* The same history pushed as slot images (bc_cache_push_flat) into a second cache and
 * forecast into one slot-shaped output (bc_forecast_flat): one launch each and no layer
 * table, bit for bit the per-layer forecast `want` (laid out at `offs`). */
static int flat_slot_checks(const int64_t *numels, int L, const int64_t *offs,
                            uint16_t *const *host, const double *times, double t_new,
                            const uint16_t *want) {
    int failures = 0;
    bc_handle h = NULL;
    int64_t *lay = (int64_t *)malloc((size_t)(L + 1) * sizeof(int64_t));
    CHECK(bc_cache_create(numels, L, 3, BC_DTYPE_BF16, NULL, &h) == BC_OK, "create: %s",
          bc_last_error());
    CHECK(bc_cache_layout(h, lay) == BC_OK, "layout");
    if (failures) return failures;
    const size_t slot_bytes = (size_t)lay[L];
    uint16_t *img = (uint16_t *)calloc(slot_bytes / 2, sizeof(uint16_t));
    uint16_t *flat = (uint16_t *)malloc(slot_bytes);
    void *dev_img = NULL, *dev_flat = NULL;
    CHECK(cudaMalloc(&dev_img, slot_bytes) == 0 && cudaMalloc(&dev_flat, slot_bytes) == 0,
          "cudaMalloc");
    bc_stats st0, st1;
    CHECK(bc_cache_stats(h, &st0) == BC_OK, "stats");
    for (int k = 0; k < 3 && !failures; ++k) {
        for (int l = 0; l < L; ++l)
            memcpy(img + lay[l] / 2, host[k] + offs[l], (size_t)numels[l] * 2);
        CHECK(cudaMemcpy(dev_img, img, slot_bytes, H2D) == 0, "upload");
        CHECK(bc_cache_push_flat(h, dev_img, times[k], NULL) == BC_OK, "push_flat: %s",
              bc_last_error());
        cudaDeviceSynchronize();
    }
    CHECK(bc_forecast_flat(h, t_new, dev_flat, NULL) == BC_OK, "forecast_flat: %s",
          bc_last_error());
    CHECK(bc_cache_check(h) == BC_OK, "device status");
    CHECK(bc_cache_stats(h, &st1) == BC_OK, "stats");
    CHECK(st1.kernel_launches - st0.kernel_launches == 4, "%lld launches for 3 flat pushes "
          "and a flat forecast", (long long)(st1.kernel_launches - st0.kernel_launches));
    CHECK(st1.table_uploads == st0.table_uploads, "the flat calls uploaded a layer table");
    CHECK(cudaMemcpy(flat, dev_flat, slot_bytes, D2H) == 0, "download");
    int64_t diff = 0;
    for (int l = 0; l < L && !failures; ++l)
        for (int64_t e = 0; e < numels[l]; ++e)
            if (flat[lay[l] / 2 + e] != want[offs[l] + e]) ++diff;
    CHECK(diff == 0, "%lld flat elements differ from the per-layer forecast", (long long)diff);
    bc_cache_destroy(h);
    cudaFree(dev_img);
    cudaFree(dev_flat);
    free(img);
    free(flat);
    free(lay);
    return failures;
}

static int many_layer_checks(void) {
    enum { L = 2048 };
    const double times[3] = {0.9, 0.85, 0.8};
    const double t_new = 0.75;
    static int64_t numels[L], offs[L + 1];
    int64_t total = 0;
    for (int l = 0; l < L; ++l) {
        numels[l] = (l * 37) % 900 + 1 + (l % 9 == 0 ? 8192 : 0);
        offs[l] = total;
        total += (numels[l] + 7) / 8 * 8;       /* 16-byte aligned tensors in one buffer */
    }
    offs[L] = total;
    uint16_t *host[3];
    for (int k = 0; k < 3; ++k) {
        host[k] = (uint16_t *)calloc((size_t)total, sizeof(uint16_t));
        for (int l = 0; l < L; ++l)
            for (int64_t e = 0; e < numels[l]; ++e) {
                const double a = sin(0.01 * e + l), b = cos(0.003 * e - l);
                host[k][offs[l] + e] = to_bf16((float)(a + b * times[k]));
            }
    }
    const int64_t nan_layer = 777, nan_elem = 3;
    host[1][offs[nan_layer] + nan_elem] = 0x7FC0;          /* NaN in the middle node */
    void *dev_in = NULL, *dev_out = NULL;
    bc_handle h = NULL;
    CHECK(bc_cache_create(numels, L, 3, BC_DTYPE_BF16, NULL, &h) == BC_OK, "create: %s",
          bc_last_error());
    CHECK(cudaMalloc(&dev_in, (size_t)total * 2) == 0 && cudaMalloc(&dev_out, (size_t)total * 2) == 0,
          "cudaMalloc");
    static const void *src[L];
    static void *outs[L];
    for (int l = 0; l < L; ++l) {
        src[l] = (const char *)dev_in + offs[l] * 2;
        outs[l] = (char *)dev_out + offs[l] * 2;
    }
    bc_stats st0, st1;
    CHECK(bc_cache_stats(h, &st0) == BC_OK, "stats");
    for (int k = 0; k < 3 && !failures; ++k) {
        CHECK(cudaMemcpy(dev_in, host[k], (size_t)total * 2, H2D) == 0, "upload");
        CHECK(bc_cache_push(h, src, times[k], NULL) == BC_OK, "push: %s", bc_last_error());
        cudaDeviceSynchronize();
    }
    CHECK(bc_forecast(h, t_new, outs, BC_DTYPE_BF16, NULL) == BC_OK, "forecast: %s",
          bc_last_error());
    CHECK(bc_cache_check(h) == BC_OK, "device status");
    CHECK(bc_cache_stats(h, &st1) == BC_OK, "stats");
    CHECK(st1.kernel_launches - st0.kernel_launches == 4, "%lld launches for 3 pushes and a "
          "forecast of %d tensors", (long long)(st1.kernel_launches - st0.kernel_launches), L);
    CHECK(st1.table_uploads - st0.table_uploads == 2, "%lld table uploads (one per table)",
          (long long)(st1.table_uploads - st0.table_uploads));
    uint16_t *got = (uint16_t *)malloc((size_t)total * 2);
    CHECK(cudaMemcpy(got, dev_out, (size_t)total * 2, D2H) == 0, "download");
    double nodes[3] = {times[2], times[1], times[0]}, W[3];
    oracle_paper_weights(nodes, 3, t_new, 0.95, 0.0, 10.0, 1e-12, W);
    double *ref = (double *)malloc((size_t)total * sizeof(double));
    double *bound = (double *)malloc((size_t)total * sizeof(double));
    int64_t bad = 0;
    for (int l = 0; l < L; ++l) {
        const void *F[3] = {host[2] + offs[l], host[1] + offs[l], host[0] + offs[l]};
        oracle_combine(1, F, 3, W, numels[l], ref, bound);
        for (int64_t e = 0; e < numels[l]; ++e) {
            uint32_t u = (uint32_t)got[offs[l] + e] << 16;
            float g;
            memcpy(&g, &u, sizeof g);
            if (isnan(ref[e])) {
                if (!isnan(g)) ++bad;
            } else if (!(fabs((double)g - ref[e]) <= ldexp(1.0, -8) * bound[e])) {
                ++bad;
            }
        }
        if (l == nan_layer) {
            uint32_t u = (uint32_t)got[offs[l] + nan_elem] << 16;
            float g;
            memcpy(&g, &u, sizeof g);
            CHECK(isnan(ref[nan_elem]) && isnan(g), "the planted NaN did not propagate");
        }
    }
    CHECK(bad == 0, "%lld elements off the oracle", (long long)bad);
    if (!failures) failures += flat_slot_checks(numels, L, offs, host, times, t_new, got);
    bc_cache_destroy(h);
    cudaFree(dev_in);
    cudaFree(dev_out);
    for (int k = 0; k < 3; ++k) free(host[k]);
    free(got);
    free(ref);
    free(bound);
    return failures;
}

static double now_s(void) {
    struct timespec ts;
    clock_gettime(CLOCK_MONOTONIC, &ts);
    return (double)ts.tv_sec + 1e-9 * (double)ts.tv_nsec;
}

/* Host cost of one forecast call through the ABI (memo hit, table build, launch), on
 * caches of 1, 4, 16 and 64 layers of 4096 bf16 elements, and of one memo lookup; then the
 * host cost per tensor of forecasts and pushes over 4096 and 65,536 such tensors (device
 * layer tables, reused each call). */
static int host_cost(void) {
    enum { kMaxLayers = 65536, kCalls = 500, kElems = 4096 };
    static const int sizes[] = {1, 4, 16, 64, 4096, 65536};
    void *src = NULL, *out = NULL;
    CHECK(cudaMalloc(&src, kElems * 2) == 0 && cudaMalloc(&out, (size_t)kMaxLayers * kElems * 2) == 0,
          "cudaMalloc");
    int64_t *numels = (int64_t *)malloc(sizeof(int64_t) * kMaxLayers);
    const void **ptrs = (const void **)malloc(sizeof(void *) * kMaxLayers);
    void **outs = (void **)malloc(sizeof(void *) * kMaxLayers);
    for (size_t si = 0; si < sizeof sizes / sizeof sizes[0] && !failures; ++si) {
        const int L = sizes[si];
        for (int l = 0; l < L; ++l) {
            numels[l] = kElems;
            ptrs[l] = src;
            outs[l] = (char *)out + (size_t)l * kElems * 2;
        }
        bc_handle h = NULL;
        CHECK(bc_cache_create(numels, L, 3, BC_DTYPE_BF16, NULL, &h) == BC_OK, "create");
        if (failures) break;
        double t = 0.9;
        for (int k = 0; k < 3; ++k, t -= 0.05)
            CHECK(bc_cache_push(h, ptrs, t, NULL) == BC_OK, "push");
        const int calls = L > 64 ? 50 : kCalls;
        for (int i = 0; i < 20; ++i) bc_forecast(h, 0.75, outs, BC_DTYPE_BF16, NULL);
        cudaDeviceSynchronize();
        const double t0 = now_s();
        for (int i = 0; i < calls; ++i)
            CHECK(bc_forecast(h, 0.75, outs, BC_DTYPE_BF16, NULL) == BC_OK, "forecast");
        const double t1 = now_s();
        cudaDeviceSynchronize();
        const double t2 = now_s();
        double c[BC_MAX_K];
        int m = 0;
        const double t3 = now_s();
        for (int i = 0; i < calls; ++i) bc_coefficients(h, 0.75, c, &m);
        const double t4 = now_s();
        const double t5 = now_s();
        for (int i = 0; i < calls; ++i, t -= 1e-4)
            CHECK(bc_cache_push(h, ptrs, t, NULL) == BC_OK, "push");
        const double t6 = now_s();
        cudaDeviceSynchronize();
        CHECK(bc_cache_check(h) == BC_OK, "device status");
        printf("{\"layers\": %d, \"host_us_per_forecast\": %.2f, \"device_us_per_forecast\": %.2f, "
               "\"memo_lookup_us\": %.3f, \"host_us_per_push\": %.2f, "
               "\"host_ns_per_tensor_forecast\": %.2f, \"host_ns_per_tensor_push\": %.2f}\n",
               L, 1e6 * (t1 - t0) / calls, 1e6 * (t2 - t0) / calls, 1e6 * (t4 - t3) / calls,
               1e6 * (t6 - t5) / calls, 1e9 * (t1 - t0) / calls / L,
               1e9 * (t6 - t5) / calls / L);
        bc_cache_destroy(h);
    }
    free(numels);
    free(ptrs);
    free(outs);
    cudaFree(src);
    cudaFree(out);
    return failures;
}

int main(int argc, char **argv) {
    if (argc < 2) return 2;
    int rc = 0;
    if (strcmp(argv[1], "host") == 0) rc = host_checks();
    else if (strcmp(argv[1], "device") == 0) rc = device_checks();
    else if (strcmp(argv[1], "hostcost") == 0) rc = host_cost();
    else if (strcmp(argv[1], "manylayers") == 0) rc = many_layer_checks();
    else return 2;
    printf("%s checks: %s\n", argv[1], rc ? "FAILED" : "ok");
    return rc ? 1 : 0;
}
