// tcgen05 (5th-generation tensor core) bf16 GEMM for sm_103a, used by the
// worker-gradient pass.  Internal interface.
#pragma once

#include <cuda_bf16.h>
#include <stdint.h>

#include "common.cuh"

namespace dbw {

enum TcEpiKind { TC_HIDDEN = 0, TC_LOGITS = 1, TC_DX = 2, TC_DW = 3 };

// What the epilogue does with accumulator element (m, n) of batch z.
struct TcEpi {
    const float* bias;            // HIDDEN, LOGITS: + bias[n]
    __nv_bfloat16* out;           // HIDDEN, DX: out[m * ldo + n] (bf16, row-major)
    int64_t ldo;
    __nv_bfloat16* outT;          // HIDDEN, DX: outT[n * ldT + m] (bf16, transposed), nullable
    int64_t ldT;
    float* outF;                  // LOGITS: outF[m * ldF + n] (fp32)
    int64_t ldF;
    const __nv_bfloat16* act;     // DX: ReLU mask 1[act[m * ldact + n] > 0]
    int64_t ldact;
    float* G;                     // DW: G[z * ldG + off + m * ldrow + n] (fp32)
    int64_t ldG, off, ldrow;
};

// C[M, N] = sum_{k < K} A[m, z*kz + k] * B[n, z*kz + k] for z < batch, then the
// epilogue ``kind``.  A is [rowsA >= M, lda] and B is [rowsB >= N, ldb], both
// row-major bf16 with K contiguous (lda, ldb multiples of 8, bases 16-byte
// aligned, z*kz a multiple of 8).  colsA / colsB: the logical column count of A
// / B (reads past it are zero).  ``status`` (device int) gets bit 0 set if a
// pipeline wait ever times out; it must be zeroed by the caller.
int tc_gemm(int kind, const __nv_bfloat16* A, int64_t lda, int64_t rowsA, int64_t colsA, const __nv_bfloat16* B,
            int64_t ldb, int64_t rowsB, int64_t colsB, int M, int N, int K, int batch, int64_t kz, const TcEpi& epi,
            int* status, cudaStream_t st);

// True when tc_gemm can run this problem (alignment rules above).
bool tc_shape_ok(int64_t lda, int64_t ldb, int K, int64_t kz, const void* A, const void* B);

}  // namespace dbw
