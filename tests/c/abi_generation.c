/* One cached-Picard generation through the C ABI alone (no Python, no torch):
 * device buffers from cudaMalloc, the synthetic mixture denoiser of the same
 * library, host x_init in and host x_T out.
 *
 *   abi_generation <dir>
 * reads  <dir>/sizes.txt   "T window batch K c h w tol cache_thresh std"
 *        <dir>/alphas.bin  fp64 [T+1]      <dir>/x0.bin  fp32 [batch][D]
 *        <dir>/mu.bin      fp32 [K][D]
 * writes <dir>/xT.bin      fp32 [batch][D] and prints "nfe <n> iters <k> hits <h>". */
#include <stdio.h>
#include <stdlib.h>

#include <cuda_runtime.h>

#include "paraanya.h"

static void* read_all(const char* dir, const char* name, size_t bytes) {
  char path[4096];
  snprintf(path, sizeof path, "%s/%s", dir, name);
  FILE* f = fopen(path, "rb");
  if (!f) { fprintf(stderr, "cannot open %s\n", path); exit(2); }
  void* p = malloc(bytes);
  if (fread(p, 1, bytes, f) != bytes) { fprintf(stderr, "short read %s\n", path); exit(2); }
  fclose(f);
  return p;
}

#define CHECK_PA(call)                                                          \
  do {                                                                          \
    pa_status st_ = (call);                                                     \
    if (st_ < 0) {                                                              \
      fprintf(stderr, "%s -> %s: %s\n", #call, pa_status_string(st_), pa_last_error()); \
      return 1;                                                                 \
    }                                                                           \
  } while (0)
#define CHECK_CUDA(call)                                                        \
  do {                                                                          \
    cudaError_t e_ = (call);                                                    \
    if (e_ != cudaSuccess) { fprintf(stderr, "%s -> %s\n", #call, cudaGetErrorString(e_)); return 1; } \
  } while (0)

int main(int argc, char** argv) {
  if (argc != 2) { fprintf(stderr, "usage: %s <dir>\n", argv[0]); return 2; }
  const char* dir = argv[1];
  char path[4096];
  snprintf(path, sizeof path, "%s/sizes.txt", dir);
  FILE* f = fopen(path, "r");
  if (!f) { fprintf(stderr, "cannot open %s\n", path); return 2; }
  int T, window, batch, K;
  long long c, h, w;
  double tol, thr, sd;
  if (fscanf(f, "%d %d %d %d %lld %lld %lld %lf %lf %lf", &T, &window, &batch, &K, &c, &h, &w, &tol, &thr, &sd) != 10) {
    fprintf(stderr, "bad sizes.txt\n");
    return 2;
  }
  fclose(f);
  const int64_t shape[3] = {c, h, w};
  const int64_t D = c * h * w;
  double* alphas = (double*)read_all(dir, "alphas.bin", sizeof(double) * (size_t)(T + 1));
  float* x0 = (float*)read_all(dir, "x0.bin", sizeof(float) * (size_t)(batch * D));
  float* mu = (float*)read_all(dir, "mu.bin", sizeof(float) * (size_t)(K * D));

  const int P = window < T ? window : T;
  const int max_rows = batch * P;
  size_t ws_bytes = pa_workspace_bytes(T, window, D, batch);
  size_t gws_bytes = pa_gmm_workspace_bytes(K, D, max_rows, T);
  if (!ws_bytes || !gws_bytes) { fprintf(stderr, "unsupported sizes\n"); return 1; }
  void *ws, *gws, *mu_dev, *eps_dev;
  CHECK_CUDA(cudaMalloc(&ws, ws_bytes));
  CHECK_CUDA(cudaMalloc(&gws, gws_bytes));
  CHECK_CUDA(cudaMalloc(&mu_dev, sizeof(float) * (size_t)(K * D)));
  CHECK_CUDA(cudaMalloc(&eps_dev, sizeof(float) * (size_t)max_rows * (size_t)D));
  CHECK_CUDA(cudaMemcpy(mu_dev, mu, sizeof(float) * (size_t)(K * D), cudaMemcpyHostToDevice));

  pa_solver* s = NULL;
  pa_gmm* g = NULL;
  CHECK_PA(pa_create(&s, T, window, shape, 3, alphas, tol, thr, batch, ws, ws_bytes, NULL));
  CHECK_PA(pa_gmm_create(&g, K, D, (const float*)mu_dev, sd, alphas, T, max_rows, gws, gws_bytes, NULL));
  CHECK_PA(pa_init(s, x0));  /* host pointer */
  for (;;) {
    int n_miss = 0;
    const float* batch_x = NULL;
    const int32_t* miss_bt = NULL;
    pa_status st = pa_step(s, &n_miss, &batch_x, &miss_bt);
    if (st == PA_DONE) break;
    CHECK_PA(st);
    CHECK_PA(pa_gmm_eps(g, batch_x, miss_bt, pa_n_miss_dev(s), (float*)eps_dev));
    CHECK_PA(pa_submit_eps(s, (const float*)eps_dev));
  }
  float* xT = (float*)malloc(sizeof(float) * (size_t)(batch * D));
  CHECK_PA(pa_result(s, xT));  /* host pointer */
  pa_stats_t stats;
  CHECK_PA(pa_stats(s, &stats));
  snprintf(path, sizeof path, "%s/xT.bin", dir);
  f = fopen(path, "wb");
  if (!f || fwrite(xT, sizeof(float), (size_t)(batch * D), f) != (size_t)(batch * D)) {
    fprintf(stderr, "cannot write %s\n", path);
    return 1;
  }
  fclose(f);
  printf("nfe %lld iters %lld hits %lld\n", (long long)stats.nfe, (long long)stats.iters, (long long)stats.hits);
  pa_gmm_destroy(g);
  pa_destroy(s);
  cudaFree(eps_dev);
  cudaFree(mu_dev);
  cudaFree(gws);
  cudaFree(ws);
  free(xT); free(mu); free(x0); free(alphas);
  return 0;
}
