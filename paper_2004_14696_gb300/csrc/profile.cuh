// Internal hooks of the opt-in weight-gradient launch timing (profile.cu).
#pragma once

#include <cuda_runtime.h>

namespace dbw {
// Records a start event on ``st`` when timing is enabled; returns a token (NULL when disabled).
void* dw_profile_begin(cudaStream_t st, double algorithmic_bytes);
// Records the matching stop event.
void dw_profile_end(void* token, cudaStream_t st);
}  // namespace dbw
