/* One cached-Picard generation through the C ABI alone (no Python, no torch):
 * device buffers from cudaMalloc, the synthetic mixture denoiser of the same
 * library, host x_init in and host x_T out.
 *
 *   abi_generation <dir> [loop]
 * With "loop" the generation runs as the device-driven loop: four iterations
 * (the library's pa_step_async, pa_gmm_eps and pa_submit_eps) captured once
 * as the body of a conditional WHILE node (pa_loop_capture_begin/_end) on a
 * stream of this program, then pa_loop_launch with the host x_init and
 * pa_poll_result into the host x_T: no host round trip inside the generation.
 * reads  <dir>/sizes.txt   "T window batch K c h w tol cache_thresh std"
 *        <dir>/alphas.bin  fp64 [T+1]      <dir>/x0.bin  fp32 [batch][D]
 *        <dir>/mu.bin      fp32 [K][D]
 * writes <dir>/xT.bin      fp32 [batch][D] and prints "nfe <n> iters <k> hits <h>". */
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

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
  if (argc != 2 && !(argc == 3 && strcmp(argv[2], "loop") == 0)) {
    fprintf(stderr, "usage: %s <dir> [loop]\n", argv[0]);
    return 2;
  }
  const char* dir = argv[1];
  const int loop = argc == 3;
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
  cudaStream_t stream = NULL;  /* a capture needs a stream other than the legacy default one */
  if (loop) CHECK_CUDA(cudaStreamCreateWithFlags(&stream, cudaStreamNonBlocking));
  CHECK_PA(pa_create(&s, T, window, shape, 3, alphas, tol, thr, batch, ws, ws_bytes, stream));
  CHECK_PA(pa_gmm_create(&g, K, D, (const float*)mu_dev, sd, alphas, T, max_rows, gws, gws_bytes, stream));
  float* xT = (float*)malloc(sizeof(float) * (size_t)(batch * D));
  if (!loop) {
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
    CHECK_PA(pa_result(s, xT));  /* host pointer */
  } else {
    const float* batch_x = NULL;
    const int32_t* miss_bt = NULL;
    const int32_t* n_miss_dev = NULL;
    CHECK_PA(pa_init(s, x0));
    /* one eager iteration: launch-time set-up happens outside the capture */
    CHECK_PA(pa_step_async(s, &batch_x, &miss_bt, &n_miss_dev));
    CHECK_PA(pa_gmm_eps(g, batch_x, miss_bt, n_miss_dev, (float*)eps_dev));
    CHECK_PA(pa_submit_eps(s, (const float*)eps_dev));
    CHECK_PA(pa_init(s, x0));
    CHECK_PA(pa_loop_capture_begin(s));
    for (int k = 0; k < 4; ++k) {
      CHECK_PA(pa_step_async(s, &batch_x, &miss_bt, &n_miss_dev));
      CHECK_PA(pa_gmm_eps(g, batch_x, miss_bt, n_miss_dev, (float*)eps_dev));
      CHECK_PA(pa_submit_eps(s, (const float*)eps_dev));
    }
    CHECK_PA(pa_loop_capture_end(s));
    for (int rep = 0; rep < 2; ++rep) {  /* the graph is reusable: run the generation twice */
      int n_active = -1;
      CHECK_PA(pa_loop_launch(s, x0));  /* host x_init */
      pa_status st = pa_poll_result(s, xT, &n_active);  /* host x_T */
      CHECK_PA(st);
      if (st != PA_DONE || n_active != 0) { fprintf(stderr, "the loop ended with %d active\n", n_active); return 1; }
    }
  }
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
  if (stream) cudaStreamDestroy(stream);
  cudaFree(eps_dev);
  cudaFree(mu_dev);
  cudaFree(gws);
  cudaFree(ws);
  free(xT); free(mu); free(x0); free(alphas);
  return 0;
}
