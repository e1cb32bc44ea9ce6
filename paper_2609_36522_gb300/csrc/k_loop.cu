// The device-side test of the generation loop (pa_loop_*): a CUDA graph whose
// conditional WHILE node holds two Picard iterations (Sec. 2.1, Eq. 1: the
// window slides until every trajectory has reached T, Eq. 2) and, last in its
// body, this kernel. One thread reads the counters that the planning kernel
// published and sets the node's condition: run the body again while a
// trajectory is active, the device status is clean and fewer than `limit`
// passes have run. The pass limit bounds the loop whatever the counters say.
#include "pa_loop.h"

namespace pa {
namespace {

__global__ void k_loop_cond(cudaGraphConditionalHandle h, Ctl* ctl, int32_t limit) {
  pdl_wait();  // the counters come from the planning kernel just before
  if (threadIdx.x != 0) return;
  const int32_t c = ctl->loop_passes + 1;  // zeroed by pa_init's kernel before each launch
  ctl->loop_passes = c;
  const bool more = ctl->n_active > 0 && ctl->status == kDevOk && c < limit;
  cudaGraphSetConditional(h, more ? 1u : 0u);
}

}  // namespace

cudaError_t launch_loop_cond(cudaGraphConditionalHandle h, Ctl* ctl, int32_t limit, cudaStream_t st) {
  return launch_ex(k_loop_cond, dim3(1), dim3(32), 0, st, 0, h, ctl, limit);
}

}  // namespace pa
