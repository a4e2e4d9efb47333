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
// One launch covers every layer.  Work item = one 128 x 128 Gram tile of one layer:
// rows m0 .. m0+127 of the stacked received rows against rows n0 .. n0+127 of the
// same worker block (the
// diagonal tile when B <= 128, so both operands are the same staged tile).  The
// K blocks of A (K = the layer's input width) followed by those of D (K = its
// output width) are split into S contiguous ranges, one CTA per (item, range),
// S chosen on the device from k: for B < 128, as many ranges as the live items of
// all layers leave slots idle at two CTAs per SM (at most 8); S = 1 when the live
// items alone fill them or B >= 128.  A CTA's TMA producer streams its range through a ring of stages; the MMA
// issuer accumulates its part of A A^T into TMEM columns 0..127 and of D D^T into
// 128..255; the four epilogue warps (one per TMEM lane quarter = 32 rows) write
// the worker-block columns of both partial products to the workspace (with one
// range they combine them directly).  The CTA that finishes an item last (a
// counter per item) adds the S partials of each product in range order, combines
// them within each worker block and writes the item's pieces; the result does not
// depend on which CTA came last.
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
constexpr int GSMAX = 8;                        // most K ranges per item

// The layers of one launch: layer l's operands, widths and pieces.
struct GramLayers {
    CUtensorMap tmA[DBW_LMAX], tmD[DBW_LMAX];
    int colsA[DBW_LMAX], colsD[DBW_LMAX];
    double* pieces[DBW_LMAX];
    int L;
    int items;          // work items per layer: 128-row tiles x CT
};

__global__ void __launch_bounds__(GTHREADS, 1)
    tc_gram_kernel(const __grid_constant__ GramLayers G, int B, int CT, int target_ctas, const int* __restrict__ kdev,
                   float* __restrict__ part, int* __restrict__ cnt, int* status) {
    const int k = *kdev;
    const long long live = static_cast<long long>(k > 0 ? k : 0) * B;   // received rows
    const int item = blockIdx.x / GSMAX, s_id = blockIdx.x % GSMAX;    // item over all layers
    const int layer = item / G.items, litem = item % G.items;
    const int mb = litem / CT, ct = litem % CT;
    const int m0 = mb * GBM;
    if (m0 >= live) return;                     // whole CTA: no barrier or TMEM touched yet
    const CUtensorMap& tmA = G.tmA[layer];
    const CUtensorMap& tmD = G.tmD[layer];
    double* __restrict__ pieces = G.pieces[layer];
    const int colsA = G.colsA[layer], colsD = G.colsD[layer];
    const int nk1 = (colsA + GBK - 1) / GBK, nk = nk1 + (colsD + GBK - 1) / GBK;
    const long long live_items = (live + GBM - 1) / GBM * CT * G.L;   // over all layers of the launch
    // ranges only for worker blocks narrower than a tile: a 128-column block's
    // partials cost as much traffic as the split saves
    int S = B < GBM ? static_cast<int>(target_ctas / live_items) : 1;
    S = S < 1 ? 1 : (S > GSMAX ? GSMAX : S);
    S = S > nk ? nk : S;
    if (s_id >= S) return;
    const int g0 = static_cast<int>(static_cast<long long>(s_id) * nk / S);
    const int g1 = static_cast<int>(static_cast<long long>(s_id + 1) * nk / S);   // g0 < g1 since S <= nk
    const bool hasP = g0 < nk1, hasQ = g1 > nk1;
    const int n0 = B <= GBM ? m0 : (m0 / B) * B + ct * GBM;
    const bool same = n0 == m0;
    const int W = B <= GBM ? B : GBM;           // worker-block columns a tile row needs

    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* sA = smem;
    uint8_t* sB = smem + GSTAGES * GTILE;       // used when the two operand tiles differ
    uint8_t* tail = smem + (same ? 1 : 2) * GSTAGES * GTILE;
    uint64_t* full_bar = reinterpret_cast<uint64_t*>(tail);
    uint64_t* empty_bar = full_bar + GSTAGES;
    uint64_t* accum_bar = empty_bar + GSTAGES;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(accum_bar + 1);
    int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);
    int* last_flag = abort_flag + 1;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nblk = g1 - g0;
    const uint32_t stage_tx = same ? GTILE : 2 * GTILE;

    if (threadIdx.x == 0) {
        for (int s = 0; s < GSTAGES; ++s) {
            mbar_init(smem_u32(full_bar + s), 1);
            mbar_init(smem_u32(empty_bar + s), 1);
        }
        mbar_init(smem_u32(accum_bar), 1);
        *abort_flag = 0;
        *last_flag = 0;
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
        // ---------------- TMA producer: K blocks g0 .. g1-1 (A's, then D's)
        int issued = 0;
        for (int i = 0; i < nblk; ++i) {
            const int g = g0 + i;
            const int s = i % GSTAGES;
            const uint32_t ph = (i / GSTAGES) & 1;
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
            issued = i + 1;
        }
        if (*vabort) {
            for (int i = issued - GSTAGES < 0 ? 0 : issued - GSTAGES; i < issued; ++i)
                mbar_wait(smem_u32(full_bar + i % GSTAGES), (i / GSTAGES) & 1);
        }
    } else if (warp == 1 && lane == 0) {
        // ---------------- MMA issuer: A A^T -> columns 0..127, D D^T -> 128..255
        constexpr uint32_t idesc = instr_desc_bf16(GBM, GBM);
        for (int i = 0; i < nblk; ++i) {
            const int g = g0 + i;
            const int s = i % GSTAGES;
            const uint32_t ph = (i / GSTAGES) & 1;
            if (!mbar_wait(smem_u32(full_bar + s), ph)) {
                atomicOr(status, 1);
                *vabort = 1;
                break;
            }
            tc_fence_after();
            const uint32_t a0 = smem_u32(sA + s * GTILE);
            const uint32_t b0 = same ? a0 : smem_u32(sB + s * GTILE);
            const uint32_t dcol = tmem + (g < nk1 ? 0u : static_cast<uint32_t>(GBM));
            const bool first = (g == g0 || g == nk1);   // first block of this range in A, or in D
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
        const int row = 32 * q + lane;
        const int c0 = B <= GBM ? (32 * q / B) * B : 0;   // this row group's worker block in the tile
        const bool ok = mbar_wait(smem_u32(accum_bar), 0);
        if (!ok) {
            atomicOr(status, 1);
            *vabort = 1;
        }
        const bool rows_live = m0 + 32 * q < live;
        const uint32_t lanes = static_cast<uint32_t>(q * 32) << 16;
        if (S == 1) {
            // one range: combine straight from TMEM
            if (ok && !*vabort && rows_live) {
                tc_fence_after();
                double acc = 0.0;
#pragma unroll 1
                for (int c = 0; c < W; c += 32) {
                    uint32_t p[32], d[32];
                    tc_ld_32cols(tmem + lanes + c0 + c, p);
                    tc_ld_32cols(tmem + lanes + GBM + c0 + c, d);
                    tc_wait_ld();
                    float sdot = 0.f;
#pragma unroll
                    for (int j = 0; j < 32; ++j) sdot = fmaf(u2f(d[j]), u2f(p[j]) + 1.0f, sdot);
                    acc += sdot;
                }
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
                if (lane == 0) pieces[static_cast<int64_t>((m0 + 32 * q) / 32) * CT + ct] = acc;
            }
        } else {
            // 1) this range's partial products, column-major ([c][row]: a warp's stores and
            //    loads cover 128 contiguous bytes); a product the range does not touch is 0
            const long long slab = static_cast<long long>(W) * GBM;   // floats of one product
            if (ok && !*vabort && rows_live) {
                tc_fence_after();
                float* pp = part + ((static_cast<long long>(item) * GSMAX + s_id) * 2) * slab + row;
                float* pq = pp + slab;
#pragma unroll 1
                for (int c = 0; c < W; c += 32) {
                    uint32_t p[32], d[32];
                    tc_ld_32cols(tmem + lanes + c0 + c, p);
                    tc_ld_32cols(tmem + lanes + GBM + c0 + c, d);
                    tc_wait_ld();
#pragma unroll
                    for (int j = 0; j < 32; ++j) {
                        pp[static_cast<long long>(c + j) * GBM] = hasP ? u2f(p[j]) : 0.f;
                        pq[static_cast<long long>(c + j) * GBM] = hasQ ? u2f(d[j]) : 0.f;
                    }
                }
            }
            // 2) the last CTA of the item adds the ranges' partials in range order and
            //    combines them within each worker block
            __threadfence();
            asm volatile("bar.sync 1, 128;" ::: "memory");
            if (warp == 2 && lane == 0 && !*vabort) {
                const int prev = atomicAdd(cnt + item, 1);
                if (prev == S - 1) {
                    __threadfence();
                    *last_flag = 1;
                    cnt[item] = 0;   // ready for the next layer
                }
            }
            asm volatile("bar.sync 1, 128;" ::: "memory");
            if (*last_flag && rows_live) {
                const float* base = part + static_cast<long long>(item) * GSMAX * 2 * slab + row;
                double acc = 0.0;
#pragma unroll 1
                for (int c = 0; c < W; c += 8) {
                    float p[8], d[8];
#pragma unroll
                    for (int j = 0; j < 8; ++j) p[j] = d[j] = 0.f;
#pragma unroll
                    for (int r = 0; r < GSMAX; ++r) {
                        if (r < S) {
                            const float* bp = base + 2 * r * slab + static_cast<long long>(c) * GBM;
#pragma unroll
                            for (int j = 0; j < 8; ++j) {
                                p[j] += __ldcg(bp + j * GBM);
                                d[j] += __ldcg(bp + slab + j * GBM);
                            }
                        }
                    }
                    float sdot = 0.f;
#pragma unroll
                    for (int j = 0; j < 8; ++j) sdot = fmaf(d[j], p[j] + 1.0f, sdot);
                    acc += sdot;
                }
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
                if (lane == 0) pieces[static_cast<int64_t>((m0 + 32 * q) / 32) * CT + ct] = acc;
            }
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

int tc_gram(int L, const __nv_bfloat16* const* act, const int64_t* ldA, const int* colsA,
            const __nv_bfloat16* const* dz, int64_t ldD, const int* colsD, int rows, int B, const int* kdev,
            double* const* pieces, float* part, int* cnt, int* status, cudaStream_t st) {
    if (L < 1 || L > DBW_LMAX) return fail(DBW_EINVAL, "tc_gram: %d layers", L);
    if (B < 32 || B % 32 || (GBM % B && B % GBM)) return fail(DBW_EUNSUPPORTED, "tc_gram: unsupported B = %d", B);
    GramLayers G{};
    G.L = L;
    const int CT = B > GBM ? B / GBM : 1;
    G.items = (rows + GBM - 1) / GBM * CT;
    for (int l = 0; l < L; ++l) {
        if ((ldA[l] % 8) || (ldD % 8) || (reinterpret_cast<uintptr_t>(act[l]) & 15u) ||
            (reinterpret_cast<uintptr_t>(dz[l]) & 15u))
            return fail(DBW_EALIGN, "tc_gram: unsupported operand alignment");
        if (!tc_make_map(&G.tmA[l], act[l], rows, colsA[l], ldA[l], GBK, GBM) ||
            !tc_make_map(&G.tmD[l], dz[l], rows, colsD[l], ldD, GBK, GBM))
            return fail(DBW_ECUDA, "tc_gram: cuTensorMapEncodeTiled failed");
        G.colsA[l] = colsA[l];
        G.colsD[l] = colsD[l];
        G.pieces[l] = pieces[l];
    }
    // one or two operand rings; at least 80 KB so that at most two CTAs (2 x 256 TMEM
    // columns) share an SM
    const int ring = (B <= GBM ? 1 : 2) * GSTAGES * GTILE;
    const int need = ring + 256 + 1024;
    const int smem = need > 80 * 1024 ? need : 80 * 1024;
    cudaError_t e = cudaFuncSetAttribute(tc_gram_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e == cudaSuccess) {
        // ranges sized for two resident CTAs per SM
        tc_gram_kernel<<<G.items * L * GSMAX, GTHREADS, smem, st>>>(G, B, CT, 2 * sm_count(), kdev, part, cnt,
                                                                     status);
        e = cudaGetLastError();
    }
    if (e != cudaSuccess) return fail(DBW_ECUDA, "tc_gram launch: %s", cudaGetErrorString(e));
    return DBW_OK;
}

size_t tc_gram_partial_floats(int rows, int B, int L) {
    const int CT = B > GBM ? B / GBM : 1;
    const size_t items = static_cast<size_t>((rows + GBM - 1) / GBM) * CT * L;
    return items * GSMAX * 2 * GBM * static_cast<size_t>(B <= GBM ? B : GBM);
}

size_t tc_gram_items(int rows, int B, int L) {
    const int CT = B > GBM ? B / GBM : 1;
    return static_cast<size_t>((rows + GBM - 1) / GBM) * CT * L;
}

}  // namespace dbw
