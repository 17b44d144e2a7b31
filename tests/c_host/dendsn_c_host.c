/*
 * Plain C99 host program driving libdendsn through include/dendsn.h only: reads a layer's
 * config and inputs from binary files, allocates device memory with the CUDA runtime,
 * runs dendsn_forward and dendsn_backward, and writes spikes, V^s, grad_x and the
 * parameter gradients back to files. Used by tests/test_c_host.py.
 *
 *   dendsn_c_host <dir>    reads <dir>/cfg.txt, x.bin, alpha.bin, xi.bin, zeta.bin,
 *                          kappa.bin, gs.bin; writes spikes.bin, v.bin, gx.bin, galpha.bin,
 *                          gxi.bin, gzeta.bin, gkappa.bin
 * cfg.txt: "T B N K G C inner psi reset" (float32 x, mexican hat = 1, hard reset = 0).
 */
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <cuda_runtime_api.h>

#include "dendsn.h"

static int fail(const char *what, const char *detail)
{
    fprintf(stderr, "dendsn_c_host: %s: %s\n", what, detail);
    return 1;
}

static void *read_file(const char *dir, const char *name, size_t bytes)
{
    char path[4096];
    snprintf(path, sizeof path, "%s/%s", dir, name);
    FILE *f = fopen(path, "rb");
    if (!f)
        return NULL;
    void *buf = malloc(bytes ? bytes : 1);
    size_t got = fread(buf, 1, bytes, f);
    fclose(f);
    if (got != bytes) {
        free(buf);
        return NULL;
    }
    return buf;
}

static int write_file(const char *dir, const char *name, const void *buf, size_t bytes)
{
    char path[4096];
    snprintf(path, sizeof path, "%s/%s", dir, name);
    FILE *f = fopen(path, "wb");
    if (!f)
        return 1;
    size_t put = fwrite(buf, 1, bytes, f);
    fclose(f);
    return put != bytes;
}

/* Copies a host file's contents to a fresh device buffer. */
static void *upload(const char *dir, const char *name, size_t bytes, int *err)
{
    void *h = read_file(dir, name, bytes), *d = NULL;
    if (!h || cudaMalloc(&d, bytes ? bytes : 16) != cudaSuccess ||
        cudaMemcpy(d, h, bytes, cudaMemcpyHostToDevice) != cudaSuccess) {
        fprintf(stderr, "dendsn_c_host: cannot upload %s\n", name);
        *err = 1;
    }
    free(h);
    return d;
}

static int download(const char *dir, const char *name, const void *d, size_t bytes)
{
    void *h = malloc(bytes ? bytes : 1);
    int bad = cudaMemcpy(h, d, bytes, cudaMemcpyDeviceToHost) != cudaSuccess ||
              write_file(dir, name, h, bytes);
    free(h);
    return bad;
}

int main(int argc, char **argv)
{
    if (argc != 2)
        return fail("usage", "dendsn_c_host <dir>");
    const char *dir = argv[1];
    char path[4096];
    snprintf(path, sizeof path, "%s/cfg.txt", dir);
    FILE *f = fopen(path, "r");
    if (!f)
        return fail("cannot open", path);
    dendsn_config cfg;
    memset(&cfg, 0, sizeof cfg);
    int n = fscanf(f, "%d %d %d %d %d %d %d %d %d", &cfg.T, &cfg.B, &cfg.N, &cfg.K, &cfg.G,
                   &cfg.C, &cfg.inner, &cfg.psi, &cfg.reset);
    fclose(f);
    if (n != 9)
        return fail("bad config file", path);
    cfg.x_dtype = DENDSN_F32;
    cfg.surrogate = DENDSN_SG_ATAN;
    cfg.theta = 1.0f;
    cfg.beta = 0.5f;
    cfg.layout = DENDSN_LAYOUT_KINNER;

    size_t saved_bytes = 0, scratch_bytes = 0;
    dendsn_status st = dendsn_workspace_size(&cfg, &saved_bytes, &scratch_bytes);
    if (st != DENDSN_OK)
        return fail("dendsn_workspace_size", dendsn_last_error());

    const size_t ns = (size_t)cfg.T * cfg.B * cfg.N;
    const size_t Kb = (size_t)(cfg.K / cfg.G);
    const size_t xb = ns * cfg.K * sizeof(float), sb = ns * sizeof(float);
    const size_t pk = (size_t)cfg.C * cfg.K * sizeof(float), pb = (size_t)cfg.C * Kb * sizeof(float);
    int err = 0;
    void *x = upload(dir, "x.bin", xb, &err);
    float *alpha = upload(dir, "alpha.bin", pk, &err), *xi = upload(dir, "xi.bin", pk, &err);
    float *zeta = upload(dir, "zeta.bin", pb, &err), *kappa = upload(dir, "kappa.bin", pb, &err);
    void *gs = upload(dir, "gs.bin", sb, &err);
    if (err)
        return 1;
    void *spikes = NULL, *gx = NULL, *saved = NULL, *scratch = NULL;
    float *v = NULL, *ga = NULL, *gxi = NULL, *gz = NULL, *gk = NULL;
    if (cudaMalloc(&spikes, sb) || cudaMalloc((void **)&v, sb) || cudaMalloc(&gx, xb) ||
        cudaMalloc((void **)&ga, pk) || cudaMalloc((void **)&gxi, pk) ||
        cudaMalloc((void **)&gz, pb) || cudaMalloc((void **)&gk, pb) ||
        cudaMalloc(&scratch, scratch_bytes ? scratch_bytes : 16) ||
        (saved_bytes && cudaMalloc(&saved, saved_bytes)))
        return fail("cudaMalloc", "failed");

    cudaStream_t stream;
    if (cudaStreamCreate(&stream) != cudaSuccess)
        return fail("cudaStreamCreate", "failed");
    st = dendsn_forward(&cfg, x, alpha, xi, zeta, kappa, NULL, spikes, v, saved, stream);
    if (st != DENDSN_OK)
        return fail("dendsn_forward", dendsn_last_error());
    st = dendsn_backward(&cfg, x, alpha, xi, zeta, kappa, NULL, gs, NULL, saved, gx, ga, gxi,
                         gz, gk, scratch, stream);
    if (st != DENDSN_OK)
        return fail("dendsn_backward", dendsn_last_error());
    if (cudaStreamSynchronize(stream) != cudaSuccess)
        return fail("cudaStreamSynchronize", "failed");

    if (download(dir, "spikes.bin", spikes, sb) || download(dir, "v.bin", v, sb) ||
        download(dir, "gx.bin", gx, xb) || download(dir, "galpha.bin", ga, pk) ||
        download(dir, "gxi.bin", gxi, pk) || download(dir, "gzeta.bin", gz, pb) ||
        download(dir, "gkappa.bin", gk, pb))
        return fail("download", "failed");
    printf("ok %s launches=%llu\n", dendsn_status_string(DENDSN_OK),
           (unsigned long long)dendsn_launch_count());
    cudaFree(x); cudaFree(alpha); cudaFree(xi); cudaFree(zeta); cudaFree(kappa); cudaFree(gs);
    cudaFree(spikes); cudaFree(v); cudaFree(gx); cudaFree(ga); cudaFree(gxi); cudaFree(gz);
    cudaFree(gk); cudaFree(scratch);
    if (saved)
        cudaFree(saved);
    cudaStreamDestroy(stream);
    return 0;
}
