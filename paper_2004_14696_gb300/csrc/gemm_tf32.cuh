// fp32 GEMMs on the tcgen05 tensor cores in three tf32 passes (3xTF32), for the fp32
// workloads: the forward GEMM (gemm_kernel, templated on its epilogue) and the per-worker
// weight gradient written into G (dw_kernel).  Internal header, included by grads.cu only.
//
// Every fp32 operand x is split into hi = x rounded to nearest tf32 (10 mantissa bits)
// and lo = x - hi (exact in fp32, |lo| <= 2^-11 |x|), itself stored rounded to nearest
// tf32, so that the tensor core reads both parts exactly.  Then
// x y ~ hi_x hi_y + hi_x lo_y + lo_x hi_y: the dropped lo_x lo_y and the rounding of lo
// are each at most 2^-22 of |x y|, and unbiased.
//
// The accumulation is split too, because the tensor core's fp32 accumulation is not
// assumed to round to nearest: the hi.hi products of 32-deep K block kb go to TMEM
// accumulator kb mod NMAIN, the two correction products of every block to one more
// accumulator (its terms are 2^-11 of the others, so its own rounding is negligible),
// and the epilogue adds the NMAIN + 1 partial sums in fp32, rounding to nearest.  Each
// accumulator then takes about K / (8 NMAIN) MMA additions instead of 3 K / 8.
//
// gemm_kernel: one CTA per 128 x BN output tile (the single-CTA layout of tc_gemm_kernel): a TMA
// producer thread, an MMA thread, four epilogue warps (one per 32-row TMEM lane
// quarter).  A stage holds 32-deep K slices of A_hi, A_lo (128 rows) and B_hi, B_lo
// (BN rows), 128-byte swizzled; its 4 K = 8 steps issue 3 MMAs each.  Every wait is
// bounded (2 s); if one runs out, bit 0 of ``status`` is set and the tile is skipped.
#pragma once

#include "gemm_tc.cuh"
#include "tc_ptx.cuh"

namespace dbw {
namespace tf32 {

// Instruction descriptor of kind::tf32: D fp32 (bits 4-5 = 1), A and B tf32 (bits 7-9 = 2,
// 10-12 = 2), both K-major, N >> 3 at bit 17, M >> 4 at bit 24.
__host__ __device__ constexpr uint32_t instr_desc_tf32(int m, int n) {
    return (1u << 4) | (2u << 7) | (2u << 10) | (static_cast<uint32_t>(n >> 3) << 17) |
           (static_cast<uint32_t>(m >> 4) << 24);
}
// D (TMEM) (+)= A (tf32, shared memory) x B (tf32, shared memory): one K = 8 step.
__device__ __forceinline__ void tc_mma_tf32(uint32_t d, uint64_t a, uint64_t b, uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n\t}" ::"r"(d),
        "l"(a), "l"(b), "r"(idesc), "r"(accumulate)
        : "memory");
}

constexpr int BM = 128;
constexpr int kThreads = 192;
constexpr int BK = 32;   // fp32 elements per 128-byte row

template <int BN, int STAGES, int NMAIN>
struct Cfg {
    static constexpr int A_BYTES = BM * BK * 4;    // one of A_hi / A_lo
    static constexpr int B_BYTES = BN * BK * 4;    // one of B_hi / B_lo
    static constexpr int STAGE_BYTES = 2 * A_BYTES + 2 * B_BYTES;
    static constexpr int SMEM = STAGES * STAGE_BYTES + 256 + 1024;
    static constexpr int ACC_COLS = (NMAIN + 1) * BN;   // NMAIN hi.hi accumulators, then the corrections
    static constexpr int TMEM_COLS = ACC_COLS <= 32 ? 32 : ACC_COLS <= 64 ? 64 : ACC_COLS <= 128 ? 128
                                   : ACC_COLS <= 256 ? 256 : 512;
    static_assert(BN % 32 == 0 && BN >= 32 && BN <= 256, "BN: a multiple of 32 up to 256");
    static_assert(ACC_COLS <= 512, "the accumulators exceed TMEM");
};

struct Operands {
    CUtensorMap a_hi, a_lo, b_hi, b_lo;   // A [M, K], B [N, K], fp32 row-major, K contiguous
};

// x rounded to the nearest tf32 value (10 mantissa bits; ties to even), for finite x; a
// value that would round up past the largest finite float is truncated instead.
__device__ __forceinline__ float round_tf32(float x) {
    const uint32_t u = __float_as_uint(x);
    const uint32_t r = (u + 0x0FFFu + ((u >> 13) & 1u)) & 0xFFFFE000u;
    return ((r & 0x7F800000u) == 0x7F800000u) ? __uint_as_float(u & 0xFFFFE000u) : __uint_as_float(r);
}
// hi = x rounded to nearest tf32, lo = x - hi (exact) rounded to nearest tf32.  A value
// that is not finite goes whole to hi (a NaN as the canonical quiet NaN), lo = 0.
__device__ __forceinline__ void split_value(float x, float& hi, float& lo) {
    if (isfinite(x)) {
        hi = round_tf32(x);
        lo = round_tf32(x - hi);
    } else {
        hi = isnan(x) ? __uint_as_float(0x7FC00000u) : x;
        lo = 0.f;
    }
}

// hi / lo parts of a row-major fp32 matrix [rows, cols] (row stride lds) into two
// matrices with row stride ldo.
__global__ void split_kernel(const float* __restrict__ src, int rows, int cols, int64_t lds,
                             float* __restrict__ hi, float* __restrict__ lo, int64_t ldo);
// The same four values at a time (cols, lds, ldo multiples of 4; src 16-byte aligned).
__global__ void split4_kernel(const float* __restrict__ src, int rows, int cols, int64_t lds,
                              float* __restrict__ hi, float* __restrict__ lo, int64_t ldo);
// Launches split4_kernel where its alignment holds, else split_kernel.
void split(const float* src, int rows, int cols, int64_t lds, float* hi, float* lo, int64_t ldo, cudaStream_t st);
// The same, transposed: hiT[c * ldt + r], loT[c * ldt + r] for r < rows, c < cols
// (32 x 32 tiles through shared memory; blocks of 32 x 8 threads).
__global__ void split_t_kernel(const float* __restrict__ src, int rows, int cols, int64_t lds,
                               float* __restrict__ hiT, float* __restrict__ loT, int64_t ldt);

template <int BN, int STAGES, int NMAIN, class Epi>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_kernel(const __grid_constant__ Operands op, int M, int N, int K, Epi epi, int* status) {
    using C = Cfg<BN, STAGES, NMAIN>;
    using namespace tcx;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    // stage s: A_hi, A_lo, B_hi, B_lo
    auto part = [&](int s, int which) {
        const int off = which < 2 ? which * C::A_BYTES : 2 * C::A_BYTES + (which - 2) * C::B_BYTES;
        return smem + s * C::STAGE_BYTES + off;
    };
    uint64_t* full_bar = reinterpret_cast<uint64_t*>(smem + STAGES * C::STAGE_BYTES);
    uint64_t* empty_bar = full_bar + STAGES;
    uint64_t* accum_bar = empty_bar + STAGES;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(accum_bar + 1);
    int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int m0 = blockIdx.y * BM, n0 = blockIdx.x * BN;
    const int nk = (K + BK - 1) / BK;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(smem_u32(full_bar + s), 1);
            mbar_init(smem_u32(empty_bar + s), 1);
        }
        mbar_init(smem_u32(accum_bar), 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 0) {
        tc_alloc(smem_u32(tmem_slot), C::TMEM_COLS);
        tc_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0 && lane == 0) {
        // ---------------- TMA producer
        int issued = 0;
        for (int kb = 0; kb < nk; ++kb) {
            const int s = kb % STAGES;
            const uint32_t ph = (kb / STAGES) & 1;
            if (!mbar_wait(smem_u32(empty_bar + s), ph ^ 1)) {
                atomicOr(status, 1);
                atomicExch(abort_flag, 1);
                break;
            }
            if (*reinterpret_cast<volatile int*>(abort_flag)) break;
            const uint32_t fb = smem_u32(full_bar + s);
            mbar_expect_tx(fb, C::STAGE_BYTES);
            tma_load_2d(smem_u32(part(s, 0)), &op.a_hi, kb * BK, m0, fb);
            tma_load_2d(smem_u32(part(s, 1)), &op.a_lo, kb * BK, m0, fb);
            tma_load_2d(smem_u32(part(s, 2)), &op.b_hi, kb * BK, n0, fb);
            tma_load_2d(smem_u32(part(s, 3)), &op.b_lo, kb * BK, n0, fb);
            issued = kb + 1;
        }
        if (*reinterpret_cast<volatile int*>(abort_flag)) {
            // this thread's copies that may still be in flight (the last STAGES issued)
            for (int kb = issued - STAGES < 0 ? 0 : issued - STAGES; kb < issued; ++kb)
                mbar_wait(smem_u32(full_bar + kb % STAGES), (kb / STAGES) & 1);
        }
    } else if (warp == 1 && lane == 0) {
        // ---------------- MMA issuer: per K = 8 step hi.hi (accumulator kb mod NMAIN),
        // hi.lo and lo.hi (the correction accumulator)
        constexpr uint32_t idesc = instr_desc_tf32(BM, BN);
        const uint32_t corr = tmem + NMAIN * BN;
        for (int kb = 0; kb < nk; ++kb) {
            const int s = kb % STAGES;
            const uint32_t ph = (kb / STAGES) & 1;
            if (!mbar_wait(smem_u32(full_bar + s), ph)) {
                atomicOr(status, 1);
                atomicExch(abort_flag, 1);
                break;
            }
            tc_fence_after();
            const uint32_t ah = smem_u32(part(s, 0)), al = smem_u32(part(s, 1));
            const uint32_t bh = smem_u32(part(s, 2)), bl = smem_u32(part(s, 3));
#pragma unroll
            for (int kk = 0; kk < BK / 8; ++kk) {
                const uint32_t o = kk * 32;   // 8 fp32 = 32 bytes of K per step
                tc_mma_tf32(tmem + (kb % NMAIN) * BN, smem_desc(ah + o, 128), smem_desc(bh + o, 128), idesc,
                            (kb >= NMAIN || kk > 0) ? 1u : 0u);
                tc_mma_tf32(corr, smem_desc(ah + o, 128), smem_desc(bl + o, 128), idesc, (kb > 0 || kk > 0) ? 1u : 0u);
                tc_mma_tf32(corr, smem_desc(al + o, 128), smem_desc(bh + o, 128), idesc, 1u);
            }
            tc_commit(smem_u32(empty_bar + s));   // frees the stage once these MMAs have read it
        }
        tc_commit(smem_u32(accum_bar));           // accumulator complete (or, after an abort, quiescent)
    } else if (warp >= 2) {
        // ---------------- epilogue: TMEM lane quarter q = rows m0 + 32 q ..
        if (!mbar_wait(smem_u32(accum_bar), 0)) {
            atomicOr(status, 1);
        } else if (!*reinterpret_cast<volatile int*>(abort_flag)) {
            tc_fence_after();
            const int q = warp & 3;
            const int row = m0 + q * 32 + lane;
            const uint32_t tbase = tmem + (static_cast<uint32_t>(q * 32) << 16);
            const int used = nk < NMAIN ? nk : NMAIN;   // hi.hi accumulators written
#pragma unroll 1
            for (int c = 0; c < BN / 32; ++c) {
                const int nb = n0 + c * 32;
                if (nb >= N) break;
                float v[32];
                uint32_t r[32];
#pragma unroll
                for (int j = 0; j < 32; ++j) v[j] = 0.f;
#pragma unroll 1
                for (int a = 0; a < used; ++a) {
                    tc_ld_32cols(tbase + a * BN + c * 32, r);
                    tc_wait_ld();
#pragma unroll
                    for (int j = 0; j < 32; ++j) v[j] += u2f(r[j]);
                }
                if (nk > 0) {
                    tc_ld_32cols(tbase + NMAIN * BN + c * 32, r);
                    tc_wait_ld();
#pragma unroll
                    for (int j = 0; j < 32; ++j) v[j] += u2f(r[j]);
                }
                if (row < M) epi.row32(row, nb, N, v);
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tc_dealloc(tmem, C::TMEM_COLS);
    }
}

constexpr int kBN = 64;
constexpr int kStages = 4;
constexpr int kMain = 7;   // (7 + 1) x 64 = 512 TMEM columns

// The epilogue functor takes a row's outputs 32 columns at a time:
// epi.row32(m, n0, N, v) for columns n0 .. n0 + 31 (those below N).
//
// Splits both operands into ws buffers (a_hi, a_lo: [M, lda2]; b_hi, b_lo: [N, ldb2],
// lda2 = ldb2 = K rounded up to 4) and runs C = A B^T into ``epi``.  A [M, K] (row
// stride lda) and B [N, K] (row stride ldb) are fp32 row-major.
// a_parts_ready: a_hi / a_lo already hold A's parts (written by the producer of A).
template <class Epi>
cudaError_t run(int M, int N, int K, const float* A, int64_t lda, const float* B, int64_t ldb, float* a_hi,
                float* a_lo, float* b_hi, float* b_lo, Epi epi, int* status, cudaStream_t st,
                bool a_parts_ready = false) {
    const int64_t ld2 = (K + 3) / 4 * 4;
    if (!a_parts_ready) split(A, M, K, lda, a_hi, a_lo, ld2, st);
    split(B, N, K, ldb, b_hi, b_lo, ld2, st);
    Operands op;
    if (!tc_make_map_f32(&op.a_hi, a_hi, M, K, ld2, BM) || !tc_make_map_f32(&op.a_lo, a_lo, M, K, ld2, BM) ||
        !tc_make_map_f32(&op.b_hi, b_hi, N, K, ld2, kBN) || !tc_make_map_f32(&op.b_lo, b_lo, N, K, ld2, kBN))
        return cudaErrorInvalidValue;
    using C = Cfg<kBN, kStages, kMain>;
    auto kern = gemm_kernel<kBN, kStages, kMain, Epi>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
    if (e != cudaSuccess) return e;
    dim3 grid((N + kBN - 1) / kBN, (M + BM - 1) / BM);
    kern<<<grid, kThreads, C::SMEM, st>>>(op, M, N, K, epi, status);
    return cudaGetLastError();
}


// ------------------------------------------------------------------ per-worker weight gradient
// G[z, off + o ldrow + c] = sum_{r < K} dZ[z K + r, o] act[z K + r, c] for every worker z,
// in three tf32 passes: A = the hi / lo parts of dZ^T [Mr = out rows, z K + r], B = those
// of act^T [Nr = in rows, z K + r], both K-major (the transposed parts are written by
// split_t_kernel).  A persistent grid walks 128 x 128 tiles (out x in) worker-major with
// the in-tiles fastest; each tile has a hi.hi accumulator and a correction accumulator
// (256 TMEM columns), two tiles in flight (512 columns), so that the MMAs of tile i + 1
// run while the epilogue drains tile i.  With K = B <= 256 the hi.hi accumulator takes at
// most 32 MMA additions.  Eight epilogue warps, two per TMEM lane quarter (32 G rows),
// each copy their 32 x 64 block TMEM -> registers (hi.hi + corrections, rounded to
// nearest; its four TMEM loads in flight together) -> shared memory (16-byte pieces
// XOR-swizzled by row) and then store it, 256 contiguous bytes of each of two G rows per
// instruction.
namespace dw {
constexpr int BN = 128;
constexpr int STAGES = 2;
constexpr int EPI_WARPS = 8;                             // two per TMEM lane quarter (16 measured slower)
constexpr int THREADS = 32 * (2 + EPI_WARPS);
constexpr int A_BYTES = BM * BK * 4;
constexpr int B_BYTES = BN * BK * 4;
constexpr int STAGE_BYTES = 2 * A_BYTES + 2 * B_BYTES;   // A_hi, A_lo, B_hi, B_lo
constexpr int WARP_COLS = BN / (EPI_WARPS / 4);          // columns of the tile per epilogue warp
constexpr int NSEG = WARP_COLS / 32;                     // its 32-column TMEM segments
constexpr int ROW_BYTES = WARP_COLS * 4;                 // a staged row
constexpr int LANES_PER_ROW = WARP_COLS / 4;             // 16-byte pieces of a row
constexpr int ROWS_PER_STORE = 32 / LANES_PER_ROW;       // rows one store instruction covers
constexpr int WARP_STAGING = 32 * ROW_BYTES;
static_assert(WARP_COLS % 32 == 0 && EPI_WARPS % 4 == 0, "whole 32-column segments per epilogue warp");
constexpr int SMEM = STAGES * STAGE_BYTES + EPI_WARPS * WARP_STAGING + 256 + 1024;
constexpr int TILE_COLS = 2 * BN;                         // hi.hi, then the corrections
constexpr int TMEM_COLS = 2 * TILE_COLS;
constexpr int kMaxK = 256;
}  // namespace dw

static __global__ void __launch_bounds__(dw::THREADS, 1)
    dw_kernel(const __grid_constant__ Operands op, int Mr, int Nr, int K, int batch, int* status,
              float* __restrict__ Gbase, int64_t ldrow, int64_t ldG) {
    using namespace tcx;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    auto part = [&](int s, int which) {
        const int off = which < 2 ? which * dw::A_BYTES : 2 * dw::A_BYTES + (which - 2) * dw::B_BYTES;
        return smem + s * dw::STAGE_BYTES + off;
    };
    uint8_t* staging = smem + dw::STAGES * dw::STAGE_BYTES;
    uint64_t* full_bar = reinterpret_cast<uint64_t*>(staging + dw::EPI_WARPS * dw::WARP_STAGING);
    uint64_t* empty_bar = full_bar + dw::STAGES;
    uint64_t* tfull_bar = empty_bar + dw::STAGES;   // [2] accumulator ready
    uint64_t* tempty_bar = tfull_bar + 2;           // [2] accumulator drained (every epilogue warp)
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tempty_bar + 2);
    int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int mt_n = (Mr + BM - 1) / BM, nt_n = (Nr + dw::BN - 1) / dw::BN;
    const int tiles_per_z = mt_n * nt_n;
    const long long total = static_cast<long long>(tiles_per_z) * batch;
    const int nk = (K + BK - 1) / BK;

    if (threadIdx.x == 0) {
        for (int s = 0; s < dw::STAGES; ++s) {
            mbar_init(smem_u32(full_bar + s), 1);
            mbar_init(smem_u32(empty_bar + s), 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(smem_u32(tfull_bar + a), 1);
            mbar_init(smem_u32(tempty_bar + a), dw::EPI_WARPS);
        }
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 0) {
        tc_alloc(smem_u32(tmem_slot), dw::TMEM_COLS);
        tc_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    volatile int* vabort = abort_flag;

    if (warp == 0 && lane == 0) {
        // ---------------- TMA producer
        long long g = 0, issued = 0;
        for (long long t = blockIdx.x; t < total && !*vabort; t += gridDim.x) {
            const int z = static_cast<int>(t / tiles_per_z);
            const int rem = static_cast<int>(t % tiles_per_z);
            const int m0 = (rem / nt_n) * BM, n0 = (rem % nt_n) * dw::BN;
            for (int kb = 0; kb < nk; ++kb, ++g) {
                const int s = static_cast<int>(g % dw::STAGES);
                const uint32_t ph = static_cast<uint32_t>((g / dw::STAGES) & 1);
                if (!mbar_wait(smem_u32(empty_bar + s), ph ^ 1)) {
                    atomicOr(status, 1);
                    *vabort = 1;
                    break;
                }
                const uint32_t fb = smem_u32(full_bar + s);
                mbar_expect_tx(fb, dw::STAGE_BYTES);
                const int kx = z * K + kb * BK;
                tma_load_2d(smem_u32(part(s, 0)), &op.a_hi, kx, m0, fb);
                tma_load_2d(smem_u32(part(s, 1)), &op.a_lo, kx, m0, fb);
                tma_load_2d(smem_u32(part(s, 2)), &op.b_hi, kx, n0, fb);
                tma_load_2d(smem_u32(part(s, 3)), &op.b_lo, kx, n0, fb);
                issued = g + 1;
            }
        }
        if (*vabort) {
            for (long long q = issued - dw::STAGES < 0 ? 0 : issued - dw::STAGES; q < issued; ++q)
                mbar_wait(smem_u32(full_bar + q % dw::STAGES), static_cast<uint32_t>((q / dw::STAGES) & 1));
        }
    } else if (warp == 1 && lane == 0) {
        // ---------------- MMA issuer
        constexpr uint32_t idesc = instr_desc_tf32(BM, dw::BN);
        long long g = 0;
        int i = 0;
        for (long long t = blockIdx.x; t < total && !*vabort; t += gridDim.x, ++i) {
            const int acc = i & 1;
            const uint32_t aph = static_cast<uint32_t>((i >> 1) & 1);
            if (!mbar_wait(smem_u32(tempty_bar + acc), aph ^ 1)) {
                atomicOr(status, 1);
                *vabort = 1;
                break;
            }
            tc_fence_after();
            const uint32_t dmain = tmem + static_cast<uint32_t>(acc * dw::TILE_COLS);
            const uint32_t dcorr = dmain + dw::BN;
            bool ok = true;
            for (int kb = 0; kb < nk; ++kb, ++g) {
                const int s = static_cast<int>(g % dw::STAGES);
                const uint32_t ph = static_cast<uint32_t>((g / dw::STAGES) & 1);
                if (!mbar_wait(smem_u32(full_bar + s), ph)) {
                    atomicOr(status, 1);
                    *vabort = 1;
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t ah = smem_u32(part(s, 0)), al = smem_u32(part(s, 1));
                const uint32_t bh = smem_u32(part(s, 2)), bl = smem_u32(part(s, 3));
#pragma unroll
                for (int kk = 0; kk < BK / 8; ++kk) {
                    const uint32_t o = kk * 32;
                    const uint32_t accum = (kb > 0 || kk > 0) ? 1u : 0u;
                    tc_mma_tf32(dmain, smem_desc(ah + o, 128), smem_desc(bh + o, 128), idesc, accum);
                    tc_mma_tf32(dcorr, smem_desc(ah + o, 128), smem_desc(bl + o, 128), idesc, accum);
                    tc_mma_tf32(dcorr, smem_desc(al + o, 128), smem_desc(bh + o, 128), idesc, 1u);
                }
                tc_commit(smem_u32(empty_bar + s));
            }
            tc_commit(smem_u32(tfull_bar + acc));
            if (!ok) break;
        }
    } else if (warp >= 2) {
        // ---------------- epilogue
        const int q = warp & 3;          // TMEM lanes 32 q .. 32 q + 31 = G rows m0 + 32 q ..
        const int h = (warp - 2) >> 2;   // columns [WARP_COLS h, WARP_COLS (h + 1)) of the tile
        uint8_t* buf = staging + (warp - 2) * dw::WARP_STAGING;
        int i = 0;
        for (long long t = blockIdx.x; t < total; t += gridDim.x, ++i) {
            const int acc = i & 1;
            const uint32_t aph = static_cast<uint32_t>((i >> 1) & 1);
            if (!mbar_wait(smem_u32(tfull_bar + acc), aph)) {
                atomicOr(status, 1);
                *vabort = 1;
                break;
            }
            if (*vabort) break;
            tc_fence_after();
            const int z = static_cast<int>(t / tiles_per_z);
            const int rem = static_cast<int>(t % tiles_per_z);
            const int m0 = (rem / nt_n) * BM, n0 = (rem % nt_n) * dw::BN;
            const uint32_t tbase =
                tmem + static_cast<uint32_t>(acc * dw::TILE_COLS) + (static_cast<uint32_t>(q * 32) << 16);
            const int row0 = m0 + q * 32;
            const int c0 = h * dw::WARP_COLS;   // this warp's first column of the tile
            if (row0 < Mr && n0 + c0 < Nr) {
                // TMEM -> smem, every segment's loads in flight together: lane = row; piece p of
                // 128-byte segment s of row r at r * ROW_BYTES + s * 128 + ((p ^ (r & 7)) * 16)
                uint32_t rm[dw::NSEG][32], rc[dw::NSEG][32];
#pragma unroll
                for (int sg = 0; sg < dw::NSEG; ++sg) {
                    tc_ld_32cols(tbase + c0 + 32 * sg, rm[sg]);
                    tc_ld_32cols(tbase + dw::BN + c0 + 32 * sg, rc[sg]);
                }
                tc_wait_ld();
#pragma unroll
                for (int sg = 0; sg < dw::NSEG; ++sg) {
#pragma unroll
                    for (int pc = 0; pc < 8; ++pc) {
                        float4 v;
                        v.x = u2f(rm[sg][4 * pc]) + u2f(rc[sg][4 * pc]);
                        v.y = u2f(rm[sg][4 * pc + 1]) + u2f(rc[sg][4 * pc + 1]);
                        v.z = u2f(rm[sg][4 * pc + 2]) + u2f(rc[sg][4 * pc + 2]);
                        v.w = u2f(rm[sg][4 * pc + 3]) + u2f(rc[sg][4 * pc + 3]);
                        *reinterpret_cast<float4*>(buf + lane * dw::ROW_BYTES + sg * 128 + ((pc ^ (lane & 7)) << 4)) =
                            v;
                    }
                }
                __syncwarp();
                // smem -> G, ROWS_PER_STORE rows per instruction: a lane writes columns
                // n0 + c0 + 4 piece .. + 3 of row rr + ro (ROW_BYTES contiguous bytes of each row)
                const int ro = lane / dw::LANES_PER_ROW, piece = lane % dw::LANES_PER_ROW;
                const int sg = piece >> 3, pc = piece & 7;
                const int col = n0 + c0 + 4 * piece;
                const bool col_ok = col + 3 < Nr;   // Nr % 4 == 0: whole pieces in or out
                float* gcol = Gbase + static_cast<int64_t>(z) * ldG + col;
#pragma unroll 4
                for (int rr = 0; rr < 32; rr += dw::ROWS_PER_STORE) {
                    const int r = rr + ro;
                    const float4 v =
                        *reinterpret_cast<const float4*>(buf + r * dw::ROW_BYTES + sg * 128 + ((pc ^ (r & 7)) << 4));
                    if (col_ok && row0 + r < Mr)
                        __stcs(reinterpret_cast<float4*>(gcol + static_cast<int64_t>(row0 + r) * ldrow), v);
                }
                __syncwarp();
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(tempty_bar + acc));
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tc_dealloc(tmem, dw::TMEM_COLS);
    }
}

// Per-worker weight gradient of one layer: dz [batch K, Mr] and act [batch K, Nr]
// (row-major fp32, row strides ldz / lda) -> G[z ldG + o ldrow + c] (Gbase = G + the
// layer's offset).  Needs K % 32 == 0, K <= 256, Nr % 4 == 0, ldrow % 4 == 0, ldG % 4 == 0
// and Gbase 16-byte aligned (the caller checks).  zt_hi / zt_lo: [Mr, batch K] scratch,
// at_hi / at_lo: [Nr, batch K] scratch.
// act_parts_ready: at_hi / at_lo already hold act's transposed parts (act is not read).
inline cudaError_t run_dw(int Mr, int Nr, int K, int batch, const float* dz, int64_t ldz, const float* act,
                          int64_t lda, float* zt_hi, float* zt_lo, float* at_hi, float* at_lo, float* Gbase,
                          int64_t ldrow, int64_t ldG, int* status, cudaStream_t st, bool act_parts_ready = false) {
    const int64_t Mt = static_cast<int64_t>(batch) * K;   // rows of dz / act = columns of the transposes
    const dim3 blk(32, 8);
    {
        const int64_t ry = (Mt + 31) / 32;
        dim3 g((Mr + 31) / 32, ry < 65535 ? static_cast<unsigned>(ry) : 65535u);
        split_t_kernel<<<g, blk, 0, st>>>(dz, static_cast<int>(Mt), Mr, ldz, zt_hi, zt_lo, Mt);
        if (!act_parts_ready) {
            dim3 g2((Nr + 31) / 32, g.y);
            split_t_kernel<<<g2, blk, 0, st>>>(act, static_cast<int>(Mt), Nr, lda, at_hi, at_lo, Mt);
        }
    }
    Operands op;
    if (!tc_make_map_f32(&op.a_hi, zt_hi, Mr, Mt, Mt, BM) || !tc_make_map_f32(&op.a_lo, zt_lo, Mr, Mt, Mt, BM) ||
        !tc_make_map_f32(&op.b_hi, at_hi, Nr, Mt, Mt, dw::BN) || !tc_make_map_f32(&op.b_lo, at_lo, Nr, Mt, Mt, dw::BN))
        return cudaErrorInvalidValue;
    cudaError_t e = cudaFuncSetAttribute(dw_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, dw::SMEM);
    if (e != cudaSuccess) return e;
    const long long tiles = static_cast<long long>((Mr + BM - 1) / BM) * ((Nr + dw::BN - 1) / dw::BN) * batch;
    const int grid = static_cast<int>(tiles < sm_count() ? tiles : sm_count());
    dw_kernel<<<grid, dw::THREADS, dw::SMEM, st>>>(op, Mr, Nr, K, batch, status, Gbase, ldrow, ldG);
    return cudaGetLastError();
}

}  // namespace tf32
}  // namespace dbw
