// Per-worker squared gradient norms without forming the gradients, on the
// tcgen05 tensor cores of sm_103a.
//
// Worker j's weight gradient of a layer is G_j = D_j^T A_j (D_j = its B rows of
// dZ, which already carry the 1/B of Eq. (2), A_j = its B rows of the layer
// input), and its bias gradient is 1^T D_j.  Both squared norms follow from two
// B x B Gram matrices:
//   ||D_j^T A_j||_F^2 + ||1^T D_j||^2 = sum_{r,c} (D_j D_j^T)[r,c] * ((A_j A_j^T)[r,c] + 1),
// which reads the B (in + out) inputs of the worker instead of the in x out
// gradient (the per-example-norm trick, applied per worker).
//
// One CTA per 128 x 128 Gram tile of one layer: rows m0 .. m0+127 of the stacked
// received rows against rows n0 .. n0+127 of the same worker block (the diagonal
// tile when B <= 128, so both operands are the same staged tile).  The TMA
// producer streams the K blocks of A (K = the layer's input width) and then of D
// (K = its output width) through one ring of stages; the MMA issuer accumulates
// A A^T into TMEM columns 0..127 and D D^T into 128..255; the four epilogue warps
// (one per TMEM lane quarter = 32 rows) combine the two within each worker block.
//
// Waits are bounded as in the GEMM kernels: a timeout sets bit 0 of *status,
// drains the loads in flight, frees TMEM and returns.
#include <cuda.h>

#include "gemm_tc.cuh"
#include "tc_ptx.cuh"

namespace dbw {

namespace {

using namespace tcx;

constexpr int GBM = 128;                        // tile rows = TMEM lanes = tile columns
constexpr int GBK = 64;                         // K block: 128 bytes of bf16, 128-byte swizzle
constexpr int GSTAGES = 4;
constexpr int GTHREADS = 192;                   // TMA warp, MMA warp, 4 epilogue warps
constexpr int GTILE = GBM * GBK * 2;            // 16 KB per operand tile
constexpr int GSMEM = GSTAGES * 2 * GTILE + 256 + 1024;

__global__ void __launch_bounds__(GTHREADS, 1)
    tc_gram_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmD, int colsA,
                   int colsD, int B, int CT, const int* __restrict__ kdev, double* __restrict__ pieces,
                   int* status) {
    const int k = *kdev;
    const long long live = static_cast<long long>(k > 0 ? k : 0) * B;   // received rows
    const int mb = blockIdx.x / CT, ct = blockIdx.x % CT;
    const int m0 = mb * GBM;
    if (m0 >= live) return;                     // whole CTA: no barrier or TMEM touched yet
    const int n0 = B <= GBM ? m0 : (m0 / B) * B + ct * GBM;
    const bool same = n0 == m0;

    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* sA = smem;
    uint8_t* sB = smem + GSTAGES * GTILE;
    uint64_t* full_bar = reinterpret_cast<uint64_t*>(smem + 2 * GSTAGES * GTILE);
    uint64_t* empty_bar = full_bar + GSTAGES;
    uint64_t* accum_bar = empty_bar + GSTAGES;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(accum_bar + 1);
    int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nk1 = (colsA + GBK - 1) / GBK, nk = nk1 + (colsD + GBK - 1) / GBK;
    const uint32_t stage_tx = same ? GTILE : 2 * GTILE;

    if (threadIdx.x == 0) {
        for (int s = 0; s < GSTAGES; ++s) {
            mbar_init(smem_u32(full_bar + s), 1);
            mbar_init(smem_u32(empty_bar + s), 1);
        }
        mbar_init(smem_u32(accum_bar), 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 0) {
        tc_alloc(smem_u32(tmem_slot), 2 * GBM);
        tc_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    volatile int* vabort = abort_flag;

    if (warp == 0 && lane == 0) {
        // ---------------- TMA producer: K blocks of A, then of D
        int issued = 0;
        for (int g = 0; g < nk; ++g) {
            const int s = g % GSTAGES;
            const uint32_t ph = (g / GSTAGES) & 1;
            if (!mbar_wait(smem_u32(empty_bar + s), ph ^ 1)) {
                atomicOr(status, 1);
                *vabort = 1;
                break;
            }
            if (*vabort) break;
            const CUtensorMap* tm = g < nk1 ? &tmA : &tmD;
            const int kx = (g < nk1 ? g : g - nk1) * GBK;
            mbar_expect_tx(smem_u32(full_bar + s), stage_tx);
            tma_load_2d(smem_u32(sA + s * GTILE), tm, kx, m0, smem_u32(full_bar + s));
            if (!same) tma_load_2d(smem_u32(sB + s * GTILE), tm, kx, n0, smem_u32(full_bar + s));
            issued = g + 1;
        }
        if (*vabort) {
            for (int g = issued - GSTAGES < 0 ? 0 : issued - GSTAGES; g < issued; ++g)
                mbar_wait(smem_u32(full_bar + g % GSTAGES), (g / GSTAGES) & 1);
        }
    } else if (warp == 1 && lane == 0) {
        // ---------------- MMA issuer: A A^T -> columns 0..127, D D^T -> 128..255
        constexpr uint32_t idesc = instr_desc_bf16(GBM, GBM);
        for (int g = 0; g < nk; ++g) {
            const int s = g % GSTAGES;
            const uint32_t ph = (g / GSTAGES) & 1;
            if (!mbar_wait(smem_u32(full_bar + s), ph)) {
                atomicOr(status, 1);
                *vabort = 1;
                break;
            }
            tc_fence_after();
            const uint32_t a0 = smem_u32(sA + s * GTILE);
            const uint32_t b0 = same ? a0 : smem_u32(sB + s * GTILE);
            const uint32_t dcol = tmem + (g < nk1 ? 0u : static_cast<uint32_t>(GBM));
            const bool first = (g == 0 || g == nk1);
#pragma unroll
            for (int kk = 0; kk < GBK / 16; ++kk)
                tc_mma(dcol, smem_desc(a0 + kk * 32, 128), smem_desc(b0 + kk * 32, 128), idesc,
                       (first && kk == 0) ? 0u : 1u);
            tc_commit(smem_u32(empty_bar + s));
        }
        tc_commit(smem_u32(accum_bar));
    } else if (warp >= 2) {
        // ---------------- epilogue: warp q holds rows m0 + 32q .. +31 (TMEM lanes 32q ..)
        const int q = warp & 3;
        if (!mbar_wait(smem_u32(accum_bar), 0)) {
            atomicOr(status, 1);
        } else if (!*vabort && m0 + 32 * q < live) {
            tc_fence_after();
            // columns of this row group's worker inside the tile
            const int c0 = B <= GBM ? (32 * q / B) * B : 0;
            const int c1 = B <= GBM ? c0 + B : GBM;
            const uint32_t lanes = static_cast<uint32_t>(q * 32) << 16;
            double acc = 0.0;
#pragma unroll 1
            for (int c = c0; c < c1; c += 32) {
                uint32_t p[32], d[32];
                tc_ld_32cols(tmem + lanes + c, p);
                tc_ld_32cols(tmem + lanes + GBM + c, d);
                tc_wait_ld();
                float s = 0.f;
#pragma unroll
                for (int j = 0; j < 32; ++j) s = fmaf(u2f(d[j]), u2f(p[j]) + 1.0f, s);
                acc += s;
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
            if (lane == 0) pieces[static_cast<int64_t>((m0 + 32 * q) / 32) * CT + ct] = acc;
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tc_dealloc(tmem, 2 * GBM);
    }
}

}  // namespace

int tc_gram(const __nv_bfloat16* act, int64_t ldA, int64_t colsA, const __nv_bfloat16* dz, int64_t ldD, int64_t colsD,
            int rows, int B, const int* kdev, double* pieces, int* status, cudaStream_t st) {
    if (B < 32 || B % 32 || (GBM % B && B % GBM)) return fail(DBW_EUNSUPPORTED, "tc_gram: unsupported B = %d", B);
    if ((ldA % 8) || (ldD % 8) || (reinterpret_cast<uintptr_t>(act) & 15u) || (reinterpret_cast<uintptr_t>(dz) & 15u))
        return fail(DBW_EALIGN, "tc_gram: unsupported operand alignment");
    CUtensorMap ta, td;
    if (!tc_make_map(&ta, act, rows, colsA, ldA, GBK, GBM) || !tc_make_map(&td, dz, rows, colsD, ldD, GBK, GBM))
        return fail(DBW_ECUDA, "tc_gram: cuTensorMapEncodeTiled failed");
    const int CT = B > GBM ? B / GBM : 1;
    const int items = (rows + GBM - 1) / GBM * CT;
    cudaError_t e = cudaFuncSetAttribute(tc_gram_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, GSMEM);
    if (e == cudaSuccess) {
        tc_gram_kernel<<<items, GTHREADS, GSMEM, st>>>(ta, td, static_cast<int>(colsA), static_cast<int>(colsD), B, CT,
                                                      kdev, pieces, status);
        e = cudaGetLastError();
    }
    if (e != cudaSuccess) return fail(DBW_ECUDA, "tc_gram launch: %s", cudaGetErrorString(e));
    return DBW_OK;
}

}  // namespace dbw
