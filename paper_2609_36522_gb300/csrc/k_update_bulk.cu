// Bulk-copy pipelined Picard update (placeholder until the pipeline lands).
#include "pa_internal.h"

namespace pa {

bool update_bulk_supported(const Dev&, const float*) { return false; }

cudaError_t launch_update_bulk(const Dev&, const float*, cudaStream_t, int*) {
  return cudaErrorNotSupported;
}

}  // namespace pa
