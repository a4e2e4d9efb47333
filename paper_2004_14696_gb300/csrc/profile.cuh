// Internal hooks of the opt-in launch timing (profile.cu).
#pragma once

#include <cuda_runtime.h>

namespace dbw {
enum { PROF_DW = 0, PROF_GEMM = 1, PROF_CHANNELS = 2 };
// Records a start event on ``st`` when channel ``ch`` is enabled and attaches
// ``work`` to the launch; returns a token (NULL when disabled).
void* profile_begin(int ch, cudaStream_t st, double work);
// Records the matching stop event.
void profile_end(void* token, cudaStream_t st);
}  // namespace dbw
