// The generation loop's device-side test (k_loop.cu), launched last in the
// body of the conditional WHILE node that pa_loop_capture_end builds.
#pragma once
#include <cuda_runtime.h>

#include "pa_internal.h"

namespace pa {

// One thread: ctl->loop_passes += 1, then the node's condition := n_active > 0
// and the device status clean and loop_passes < limit.
cudaError_t launch_loop_cond(cudaGraphConditionalHandle h, Ctl* ctl, int32_t limit, cudaStream_t st);

}  // namespace pa
