// tcgen05 (5th-generation tensor core) bf16 GEMM for sm_103a, used by the
// worker-gradient pass.  Internal interface.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "common.cuh"

namespace dbw {

enum TcEpiKind { TC_HIDDEN = 0, TC_LOGITS = 1, TC_DX = 2, TC_DW = 3, TC_GBAR = 4 };

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
    // GBAR (mean over the received workers, Eqs. (3)-(4)): with g = acc / k,
    // W[off + m * ldrow + n] -= lr * g, gbar[off + m * ldrow + n] = g (nullable), and the
    // sums of g^2 (fp64) into pieces[(s * ceil(N / 256) + nt) * 8 + h * 4 + q]: rows
    // 128 s + 32 q .. +31 (s < ceil(M / 128)), columns 256 nt + 128 h .. +127.
    float* W;
    float* gbar;
    float lr;
    double* pieces;
    // Live row count on the device: when non-null, only (*kdev) * kmul rows of the
    // row dimension are computed (M for HIDDEN / LOGITS / DX, K for GBAR, where k =
    // *kdev); *kdev <= 0 runs no tile.
    const int* kdev;
    int kmul;
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

// 2-D TMA tensor map of a row-major bf16 matrix [rows, cols] with row stride ld
// (elements), box box_k x box_rows, 128-byte (box_k = 64) or 64-byte (32) swizzle;
// reads past the extents are zero.  False if the driver's encoder is unavailable
// or rejects the arguments.
bool tc_make_map(CUtensorMap* tm, const void* base, int64_t rows, int64_t cols, int64_t ld, int box_k, int box_rows);

// The same for a row-major fp32 matrix: box 32 (128 bytes, 128-byte swizzle) x box_rows;
// ld a multiple of 4 and base 16-byte aligned.
bool tc_make_map_f32(CUtensorMap* tm, const void* base, int64_t rows, int64_t cols, int64_t ld, int box_rows);

// True when tc_gemm can run this problem (alignment rules above).
bool tc_shape_ok(int64_t lda, int64_t ldb, int K, int64_t kz, const void* A, const void* B);

// Operands of one GEMM of tc_gemm_mean_dx (the same meaning as tc_gemm's arguments).
struct TcOperands {
    const __nv_bfloat16* A;
    int64_t lda, rowsA, colsA;
    const __nv_bfloat16* B;
    int64_t ldb, rowsB, colsB;
    int M, N, K;
};

// The mean-gradient GEMM (TC_GBAR, operands g, epilogue ge) and the input-gradient
// GEMM (TC_DX, operands x, epilogue xe) of one layer in one launch: both read dZ_l
// and neither writes what the other reads, so their tiles share the persistent
// grid (those of the mean gradient first).  Same rules as tc_gemm.
int tc_gemm_mean_dx(const TcOperands& g, const TcEpi& ge, const TcOperands& x, const TcEpi& xe, int* status,
                    cudaStream_t st);

// Per-worker squared gradient norms of L layers without forming the gradients, in one
// launch (the Gram identity ||D^T A||_F^2 = <D D^T, A A^T>_F, with the bias term
// ||1^T D||^2 = sum of D D^T added), for each layer l:
//   pieces[l][(r / 32) * CT + ct] = sum over rows r..r+31 of the 32-row group and the
//   columns c of the same worker (in column tile ct, CT = max(1, B / 128)) of
//   (D D^T)[r, c] * ((A A^T)[r, c] + 1)
// for the row groups of the first (*kdev) * B rows.  A = act[l] [rows, ldA[l]] (K =
// colsA[l]), D = dz[l] [rows, ldD] (K = colsD[l]), both bf16 row-major; B % 32 == 0 and
// either 128 % B == 0 or B % 128 == 0.  part: tc_gram_partial_floats(rows, B, L) floats
// of scratch for the partial products of the K ranges; cnt: tc_gram_items(rows, B, L)
// int32 counters, zero on entry and left zero on return.
int tc_gram(int L, const __nv_bfloat16* const* act, const int64_t* ldA, const int* colsA,
            const __nv_bfloat16* const* dz, int64_t ldD, const int* colsD, int rows, int B, const int* kdev,
            double* const* pieces, float* part, int* cnt, int* status, cudaStream_t st);
size_t tc_gram_partial_floats(int rows, int B, int L);
size_t tc_gram_items(int rows, int B, int L);

}  // namespace dbw
