/*
 * A plain C consumer of the FadeMem C ABI (include/fademem.h): it allocates
 * device memory with the CUDA runtime, drives one fp32 memory through
 * insert / consolidate / attend / attend_ext, and checks every result against
 * the fp64 CPU oracle (oracle/fademem_oracle.c, linked in as test
 * infrastructure): entry tables bit-exact after every consolidate, attention
 * within 1e-5 relative (max-norm).  Exit status 0 on success.
 *
 * Inputs are a fixed-seed stream of a 64-bit linear congruential generator,
 * uniform in [-1, 1); the same fp32 values go to both sides.
 */
#include <math.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <cuda_runtime_api.h>

#include "fademem.h"

typedef struct oracle_memory oracle_memory;
oracle_memory *oracle_create(int M, double beta, int anchor, int op, long long elems);
void oracle_destroy(oracle_memory *m);
int oracle_insert(oracle_memory *m, const double *K_t, const double *V_t);
int oracle_count(const oracle_memory *m);
void oracle_entries(const oracle_memory *m, int *slot, long long *first, long long *span, double *mu);
int oracle_attend(const oracle_memory *m, int tokens, int H, int D, const double *Q, long long Lq, double scale,
                  double *out);
int oracle_attend_ext(const oracle_memory *m, int tokens, int H, int D, const double *Kcur, const double *Vcur,
                      long long ncur, const double *Q, long long Lq, double scale, double *out);

enum { M = 5, H = 2, D = 64, N = 16, F = 3, SEGMENTS = 7, LQ = 40, NCUR = 24 };

static uint64_t g_state = 0x9E3779B97F4A7C15ull;
static float next_uniform(void) {
    g_state = g_state * 6364136223846793005ull + 1442695040888963407ull;
    return (float)((double)(g_state >> 11) * (1.0 / 9007199254740992.0) * 2.0 - 1.0);
}

#define CUDA_OK(x)                                                             \
    do {                                                                       \
        cudaError_t e_ = (x);                                                  \
        if (e_ != cudaSuccess) {                                               \
            fprintf(stderr, "CUDA error %s at line %d\n", cudaGetErrorString(e_), __LINE__); \
            return 2;                                                          \
        }                                                                      \
    } while (0)
#define FM_OK(x)                                                               \
    do {                                                                       \
        fademem_status s_ = (x);                                               \
        if (s_ != FADEMEM_OK) {                                                \
            fprintf(stderr, "fademem status %d at line %d: %s\n", (int)s_, __LINE__, fademem_last_error()); \
            return 3;                                                          \
        }                                                                      \
    } while (0)

static double max_rel_err(const float *got, const double *ref, size_t n) {
    double err = 0.0, mag = 1e-30;
    for (size_t i = 0; i < n; ++i) {
        err = fmax(err, fabs((double)got[i] - ref[i]));
        mag = fmax(mag, fabs(ref[i]));
    }
    return err / mag;
}

int main(void) {
    const size_t frame_elems = (size_t)N * H * D;
    fademem_config cfg;
    memset(&cfg, 0, sizeof(cfg));
    cfg.budget = M;
    cfg.heads = H;
    cfg.head_dim = D;
    cfg.tokens_per_frame = N;
    cfg.num_layers = 1;
    cfg.beta = 0.3;
    cfg.anchor = 1;
    cfg.merge_op = FADEMEM_MERGE_WEIGHTED;
    cfg.dtype = FADEMEM_F32;
    const size_t ws_bytes = fademem_workspace_bytes(&cfg);
    if (ws_bytes == 0) { fprintf(stderr, "workspace size 0\n"); return 4; }
    void *ws = NULL, *dK = NULL, *dV = NULL, *dQ = NULL, *dOut = NULL, *dKc = NULL, *dVc = NULL;
    CUDA_OK(cudaMalloc(&ws, ws_bytes));
    CUDA_OK(cudaMalloc(&dK, F * frame_elems * sizeof(float)));
    CUDA_OK(cudaMalloc(&dV, F * frame_elems * sizeof(float)));
    CUDA_OK(cudaMalloc(&dQ, (size_t)LQ * H * D * sizeof(float)));
    CUDA_OK(cudaMalloc(&dOut, (size_t)LQ * H * D * sizeof(float)));
    CUDA_OK(cudaMalloc(&dKc, (size_t)NCUR * H * D * sizeof(float)));
    CUDA_OK(cudaMalloc(&dVc, (size_t)NCUR * H * D * sizeof(float)));
    fademem_t h = NULL;
    FM_OK(fademem_create(&cfg, ws, ws_bytes, &h));
    oracle_memory *ora = oracle_create(M, cfg.beta, cfg.anchor, 0, (long long)frame_elems);
    if (!ora) { fprintf(stderr, "oracle_create failed\n"); return 4; }

    float *K = malloc(F * frame_elems * sizeof(float)), *V = malloc(F * frame_elems * sizeof(float));
    double *Kd = malloc(frame_elems * sizeof(double)), *Vd = malloc(frame_elems * sizeof(double));
    int failures = 0;
    for (int seg = 0; seg < SEGMENTS; ++seg) {
        for (size_t i = 0; i < F * frame_elems; ++i) { K[i] = next_uniform(); V[i] = next_uniform(); }
        CUDA_OK(cudaMemcpy(dK, K, F * frame_elems * sizeof(float), cudaMemcpyHostToDevice));
        CUDA_OK(cudaMemcpy(dV, V, F * frame_elems * sizeof(float), cudaMemcpyHostToDevice));
        FM_OK(fademem_insert(h, 0, dK, dV, F));
        FM_OK(fademem_consolidate(h, NULL));
        for (int f = 0; f < F; ++f) {
            for (size_t i = 0; i < frame_elems; ++i) { Kd[i] = K[f * frame_elems + i]; Vd[i] = V[f * frame_elems + i]; }
            oracle_insert(ora, Kd, Vd);
        }
        int count = 0, slot[M + 1];
        int64_t first[M + 1], span[M + 1], mu2[M + 1];
        FM_OK(fademem_get_entries(h, NULL, M + 1, &count, slot, first, span, mu2));
        int oslot[M + 1];
        long long ofirst[M + 1], ospan[M + 1];
        double omu[M + 1];
        oracle_entries(ora, oslot, ofirst, ospan, omu);
        if (count != oracle_count(ora)) { fprintf(stderr, "segment %d: count %d vs %d\n", seg, count, oracle_count(ora)); ++failures; continue; }
        for (int i = 0; i < count; ++i)
            if (slot[i] != oslot[i] || first[i] != ofirst[i] || span[i] != ospan[i] || mu2[i] != (int64_t)llround(2 * omu[i])) {
                fprintf(stderr, "segment %d entry %d differs\n", seg, i);
                ++failures;
            }
    }
    /* Attention over the memory, then over the memory and a current chunk. */
    float *Q = malloc((size_t)LQ * H * D * sizeof(float)), *out = malloc((size_t)LQ * H * D * sizeof(float));
    double *Qd = malloc((size_t)LQ * H * D * sizeof(double)), *ref = malloc((size_t)LQ * H * D * sizeof(double));
    float *Kc = malloc((size_t)NCUR * H * D * sizeof(float)), *Vc = malloc((size_t)NCUR * H * D * sizeof(float));
    double *Kcd = malloc((size_t)NCUR * H * D * sizeof(double)), *Vcd = malloc((size_t)NCUR * H * D * sizeof(double));
    for (size_t i = 0; i < (size_t)LQ * H * D; ++i) { Q[i] = 3.0f * next_uniform(); Qd[i] = Q[i]; }
    for (size_t i = 0; i < (size_t)NCUR * H * D; ++i) { Kc[i] = next_uniform(); Vc[i] = next_uniform(); Kcd[i] = Kc[i]; Vcd[i] = Vc[i]; }
    CUDA_OK(cudaMemcpy(dQ, Q, (size_t)LQ * H * D * sizeof(float), cudaMemcpyHostToDevice));
    CUDA_OK(cudaMemcpy(dKc, Kc, (size_t)NCUR * H * D * sizeof(float), cudaMemcpyHostToDevice));
    CUDA_OK(cudaMemcpy(dVc, Vc, (size_t)NCUR * H * D * sizeof(float), cudaMemcpyHostToDevice));
    const double scale = 1.0 / sqrt((double)D);
    FM_OK(fademem_attend(h, 0, dQ, dOut, LQ, NULL));
    CUDA_OK(cudaMemcpy(out, dOut, (size_t)LQ * H * D * sizeof(float), cudaMemcpyDeviceToHost));
    oracle_attend(ora, N, H, D, Qd, LQ, scale, ref);
    const double e1 = max_rel_err(out, ref, (size_t)LQ * H * D);
    FM_OK(fademem_attend_ext(h, 0, dQ, dKc, dVc, NCUR, dOut, LQ, NULL));
    CUDA_OK(cudaMemcpy(out, dOut, (size_t)LQ * H * D * sizeof(float), cudaMemcpyDeviceToHost));
    oracle_attend_ext(ora, N, H, D, Kcd, Vcd, NCUR, Qd, LQ, scale, ref);
    const double e2 = max_rel_err(out, ref, (size_t)LQ * H * D);
    uint32_t word = 0;
    FM_OK(fademem_get_device_status(h, NULL, &word));
    if (!(e1 <= 1e-5)) { fprintf(stderr, "attention error %.3e\n", e1); ++failures; }
    if (!(e2 <= 1e-5)) { fprintf(stderr, "attention + chunk error %.3e\n", e2); ++failures; }
    printf("c-abi consumer: %d segments, entries checked, attention rel err %.2e, with chunk %.2e, %s\n", SEGMENTS,
           e1, e2, failures ? "FAILED" : "ok");
    fademem_destroy(h);
    oracle_destroy(ora);
    cudaFree(ws); cudaFree(dK); cudaFree(dV); cudaFree(dQ); cudaFree(dOut); cudaFree(dKc); cudaFree(dVc);
    free(K); free(V); free(Kd); free(Vd); free(Q); free(out); free(Qd); free(ref); free(Kc); free(Vc); free(Kcd); free(Vcd);
    return failures ? 1 : 0;
}
