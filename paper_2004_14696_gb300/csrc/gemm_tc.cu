// bf16 GEMM on the 5th-generation tensor cores of sm_103a (tcgen05), written
// with inline PTX: TMA (cp.async.bulk.tensor) loads into a ring of shared
// memory stages guarded by mbarriers, one thread issuing tcgen05.mma into a
// TMEM accumulator, and four epilogue warps reading TMEM with tcgen05.ld.
//
//   C[M, N] = sum_k A[m, k] * B[n, k]      (both operands K-major, bf16; fp32 accumulation)
//
// CTA = 6 warps:  warp 0  TMA producer (one lane) and TMEM owner
//                 warp 1  MMA issuer (one lane)
//                 warps 2-5  epilogue: warp w reads TMEM lanes 32*(w%4) .. +31,
//                            i.e. rows m0 + 32*(w%4) + lane of the 128-row tile.
// Tile 128 x BN x BK; K-major operands staged with the 128B (BK = 64) or 64B
// (BK = 32) swizzle that both TMA and the UMMA shared-memory descriptors use.
//
// Every wait on an mbarrier is bounded (2 s of %globaltimer).  A wait that runs
// out sets bit 0 of *status, the producer drains the TMA loads it still has in
// flight (again bounded), TMEM is freed and the CTA returns; the results of that
// launch are then undefined, never a fault or a hang.
#include <cuda.h>

#include <atomic>
#include <mutex>

#include "gemm_tc.cuh"
#include "profile.cuh"
#include "tc_ptx.cuh"

namespace dbw {

namespace {

using namespace tcx;

constexpr int BM = 128;
constexpr int kThreads = 192;

// ------------------------------------------------------------------ epilogues
// One thread: row ``row`` of the tile, 32 columns starting at ``nb`` (logits and the
// one-CTA-per-tile weight-gradient kernel).
template <int KIND>
__device__ __forceinline__ void epilogue_chunk(const TcEpi& e, int z, int row, int nb, int M, int N,
                                               const uint32_t (&r)[32]) {
    if (row >= M) return;
    const bool full = nb + 32 <= N;
    if constexpr (KIND == TC_LOGITS) {
        float* op = e.outF + static_cast<int64_t>(row) * e.ldF + nb;
        if (full && ((reinterpret_cast<uintptr_t>(op) & 15u) == 0)) {
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                float4 v;
                v.x = u2f(r[4 * q + 0]) + __ldg(e.bias + nb + 4 * q + 0);
                v.y = u2f(r[4 * q + 1]) + __ldg(e.bias + nb + 4 * q + 1);
                v.z = u2f(r[4 * q + 2]) + __ldg(e.bias + nb + 4 * q + 2);
                v.w = u2f(r[4 * q + 3]) + __ldg(e.bias + nb + 4 * q + 3);
                *reinterpret_cast<float4*>(op + 4 * q) = v;
            }
        } else {
#pragma unroll
            for (int j = 0; j < 32; ++j)
                if (nb + j < N) op[j] = u2f(r[j]) + __ldg(e.bias + nb + j);
        }
    } else {   // TC_DW: element (m, n) -> G[z*ldG + off + m*ldrow + n]
        static_assert(KIND == TC_DW, "epilogue_chunk serves TC_LOGITS and TC_DW");
        float* op = e.G + static_cast<int64_t>(z) * e.ldG + e.off + static_cast<int64_t>(row) * e.ldrow + nb;
#pragma unroll
        for (int j = 0; j < 32; ++j)
            if (nb + j < N) __stcs(op + j, u2f(r[j]));
    }
}

// ------------------------------------------------------------------ epilogues of the pair kernel
// One thread owns one output row and 128 columns of a tile (four 32-column chunks
// read from TMEM at ``taddr``).  The global loads a chunk needs (w for the SGD
// step, the layer input for the ReLU mask) are issued one chunk ahead, so that
// their latency overlaps the previous chunk's work.

// Per epilogue warp: a 32 x 32 bf16 chunk, transposed ([column][row], rows padded to 40
// elements), between TMEM and the transposed copy.
constexpr int kStageLd = 40;
constexpr int kStageBytes = 32 * kStageLd * 2;

// bf16 activation chunk -> out (row-major) and, when asked, outT (transposed).  The
// lanes of a warp hold 32 consecutive rows (row = row0 + lane; M is a multiple of 32,
// so a warp's rows are all inside or all outside the matrix); the transposed copy goes
// through the warp's staging chunk ``stg`` so that each global store writes 16 bytes
// and four lanes cover 64 contiguous bytes of one transposed row.
__device__ __forceinline__ void store_act_chunk(const TcEpi& e, int row, int nb, int N, const float (&x)[32],
                                                __nv_bfloat16* stg) {
    const int lane = threadIdx.x & 31;
    __nv_bfloat16* op = e.out + static_cast<int64_t>(row) * e.ldo + nb;
    if (nb + 32 <= N && ((reinterpret_cast<uintptr_t>(op) & 15u) == 0)) {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            uint4 w;
            w.x = pack_bf16(x[8 * q + 0], x[8 * q + 1]);
            w.y = pack_bf16(x[8 * q + 2], x[8 * q + 3]);
            w.z = pack_bf16(x[8 * q + 4], x[8 * q + 5]);
            w.w = pack_bf16(x[8 * q + 6], x[8 * q + 7]);
            *reinterpret_cast<uint4*>(op + 8 * q) = w;
        }
    } else {
#pragma unroll
        for (int j = 0; j < 32; ++j)
            if (nb + j < N) op[j] = __float2bfloat16_rn(x[j]);
    }
    if (e.outT) {
#pragma unroll
        for (int j = 0; j < 32; ++j) stg[j * kStageLd + lane] = __float2bfloat16_rn(x[j]);
        __syncwarp();
        const int row0 = row - lane;
        const bool vec = ((reinterpret_cast<uintptr_t>(e.outT) & 15u) == 0) && e.ldT % 8 == 0;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int idx = i * 32 + lane;
            const int j = idx >> 2, p = idx & 3;   // transposed row nb + j, rows row0 + 8p .. +7
            if (nb + j < N) {
                __nv_bfloat16* dst = e.outT + static_cast<int64_t>(nb + j) * e.ldT + row0 + 8 * p;
                const __nv_bfloat16* src = stg + j * kStageLd + 8 * p;
                if (vec) {
                    *reinterpret_cast<uint4*>(dst) = *reinterpret_cast<const uint4*>(src);
                } else {
#pragma unroll
                    for (int t = 0; t < 8; ++t) dst[t] = src[t];
                }
            }
        }
        __syncwarp();
    }
}

// TC_HIDDEN: A_l = ReLU(Z_l + b_l) in bf16.
__device__ __forceinline__ void hidden_cols(const TcEpi& e, int row, int nb0, int M, int N, uint32_t taddr,
                                            __nv_bfloat16* stg) {
#pragma unroll 1
    for (int c = 0; c < 4; ++c) {
        const int nb = nb0 + 32 * c;
        if (nb >= N) break;
        uint32_t r[32];
        tc_ld_32cols(taddr + 32 * c, r);
        tc_wait_ld();
        if (row >= M) continue;
        float x[32];
#pragma unroll
        for (int j = 0; j < 32; ++j) {
            const float v = u2f(r[j]) + (nb + j < N ? __ldg(e.bias + nb + j) : 0.f);
            x[j] = v > 0.f ? v : 0.f;
        }
        store_act_chunk(e, row, nb, N, x, stg);
    }
}

// TC_DX: dZ_{l-1} = (dZ_l W_l) * 1[A_{l-1} > 0] in bf16; ``avec``: the act rows allow
// 16-byte loads.
__device__ __forceinline__ void dx_cols(const TcEpi& e, int row, int nb0, int M, int N, uint32_t taddr, bool avec,
                                        __nv_bfloat16* stg) {
    const bool rowok = row < M;
    const __nv_bfloat16* ap = e.act + static_cast<int64_t>(row) * e.ldact + nb0;
    uint4 nxt[4];
    auto fetch = [&](int c) {
        if (rowok && avec && nb0 + 32 * c + 32 <= N) {
#pragma unroll
            for (int j = 0; j < 4; ++j) nxt[j] = *reinterpret_cast<const uint4*>(ap + 32 * c + 8 * j);
        }
    };
    fetch(0);
#pragma unroll
    for (int c = 0; c < 4; ++c) {
        const int nb = nb0 + 32 * c;
        if (nb >= N) break;
        uint4 cur[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) cur[j] = nxt[j];
        if (c + 1 < 4) fetch(c + 1);
        uint32_t r[32];
        tc_ld_32cols(taddr + 32 * c, r);
        tc_wait_ld();
        if (!rowok) continue;
        float x[32];
        if (avec && nb + 32 <= N) {
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const __nv_bfloat16* hv = reinterpret_cast<const __nv_bfloat16*>(&cur[q]);
#pragma unroll
                for (int t = 0; t < 8; ++t)
                    x[8 * q + t] = u2f(r[8 * q + t]) * (__bfloat162float(hv[t]) > 0.f ? 1.f : 0.f);
            }
        } else {
#pragma unroll
            for (int j = 0; j < 32; ++j)
                x[j] = (nb + j < N) ? u2f(r[j]) * (__bfloat162float(ap[32 * c + j]) > 0.f ? 1.f : 0.f) : 0.f;
        }
        store_act_chunk(e, row, nb, N, x, stg);
    }
}

// TC_GBAR: row ``row`` is an output unit; g = acc / k, w -= lr g, optional g out; returns
// the sum of g^2 over the 128 columns (fp32 per chunk, fp64 across chunks).  ``wvec``:
// w (and gbar) allow 16-byte accesses at every 32-column chunk.
__device__ __forceinline__ double gbar_cols(const TcEpi& e, int row, int nb0, int M, int N, float inv_k,
                                            uint32_t taddr, bool wvec) {
    const bool rowok = row < M;
    const int64_t at0 = e.off + static_cast<int64_t>(row) * e.ldrow + nb0;
    float* wp = e.W + at0;
    float* gp = e.gbar ? e.gbar + at0 : nullptr;
    float4 nxt[8];
    auto fetch = [&](int c) {
        if (rowok && wvec && nb0 + 32 * c + 32 <= N) {
#pragma unroll
            for (int j = 0; j < 8; ++j) nxt[j] = *reinterpret_cast<const float4*>(wp + 32 * c + 4 * j);
        }
    };
    fetch(0);
    double sq = 0.0;
#pragma unroll
    for (int c = 0; c < 4; ++c) {
        const int nb = nb0 + 32 * c;
        if (nb >= N) break;
        float4 cur[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) cur[j] = nxt[j];
        if (c + 1 < 4) fetch(c + 1);
        uint32_t r[32];
        tc_ld_32cols(taddr + 32 * c, r);
        tc_wait_ld();
        if (!rowok) continue;
        float part = 0.f;
        if (wvec && nb + 32 <= N) {
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                float4 g, wv = cur[q];
                g.x = u2f(r[4 * q + 0]) * inv_k;
                g.y = u2f(r[4 * q + 1]) * inv_k;
                g.z = u2f(r[4 * q + 2]) * inv_k;
                g.w = u2f(r[4 * q + 3]) * inv_k;
                wv.x = fmaf(-e.lr, g.x, wv.x);
                wv.y = fmaf(-e.lr, g.y, wv.y);
                wv.z = fmaf(-e.lr, g.z, wv.z);
                wv.w = fmaf(-e.lr, g.w, wv.w);
                *reinterpret_cast<float4*>(wp + 32 * c + 4 * q) = wv;
                if (gp) *reinterpret_cast<float4*>(gp + 32 * c + 4 * q) = g;
                part += g.x * g.x + g.y * g.y + g.z * g.z + g.w * g.w;
            }
        } else {
#pragma unroll
            for (int j = 0; j < 32; ++j) {
                if (nb + j < N) {
                    const float g = u2f(r[j]) * inv_k;
                    wp[32 * c + j] = fmaf(-e.lr, g, wp[32 * c + j]);
                    if (gp) gp[32 * c + j] = g;
                    part += g * g;
                }
            }
        }
        sq += part;
    }
    return sq;
}

// ------------------------------------------------------------------ kernel
template <int BN, int BK, int STAGES>
struct TcCfg {
    static constexpr int A_BYTES = BM * BK * 2;
    static constexpr int B_BYTES = BN * BK * 2;
    static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
    static constexpr int SW = BK * 2;   // swizzle span in bytes: 128 (BK = 64) or 64 (BK = 32)
    static constexpr int BAR_BYTES = 256;
    static constexpr int SMEM = STAGES * STAGE_BYTES + BAR_BYTES + 1024;   // + alignment slack
    static_assert(BK == 64 || BK == 32, "BK must be 64 or 32");
    static_assert(BN == 128 || BN == 256, "BN must be 128 or 256");
};

template <int BN, int BK, int STAGES, int KIND, int MINB>
__global__ void __launch_bounds__(kThreads, MINB)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB, int M, int N,
                   int K, int64_t kz, TcEpi epi, int* status) {
    using Cfg = TcCfg<BN, BK, STAGES>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* sA = smem;
    uint8_t* sB = smem + STAGES * Cfg::A_BYTES;
    uint64_t* full_bar = reinterpret_cast<uint64_t*>(smem + STAGES * Cfg::STAGE_BYTES);
    uint64_t* empty_bar = full_bar + STAGES;
    uint64_t* accum_bar = empty_bar + STAGES;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(accum_bar + 1);
    int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int m0 = blockIdx.y * BM, n0 = blockIdx.x * BN, z = blockIdx.z;
    const int nk = (K + BK - 1) / BK;
    const int kbase = static_cast<int>(z * kz);

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
        tc_alloc(smem_u32(tmem_slot), BN);
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
            mbar_expect_tx(smem_u32(full_bar + s), Cfg::STAGE_BYTES);
            tma_load_2d(smem_u32(sA + s * Cfg::A_BYTES), &tmA, kbase + kb * BK, m0, smem_u32(full_bar + s));
            tma_load_2d(smem_u32(sB + s * Cfg::B_BYTES), &tmB, kbase + kb * BK, n0, smem_u32(full_bar + s));
            issued = kb + 1;
        }
        if (*reinterpret_cast<volatile int*>(abort_flag)) {
            // drain this thread's copies that may still be in flight (the last STAGES issued)
            for (int kb = issued - STAGES < 0 ? 0 : issued - STAGES; kb < issued; ++kb)
                mbar_wait(smem_u32(full_bar + kb % STAGES), (kb / STAGES) & 1);
        }
    } else if (warp == 1 && lane == 0) {
        // ---------------- MMA issuer
        constexpr uint32_t idesc = instr_desc_bf16(BM, BN);
        for (int kb = 0; kb < nk; ++kb) {
            const int s = kb % STAGES;
            const uint32_t ph = (kb / STAGES) & 1;
            if (!mbar_wait(smem_u32(full_bar + s), ph)) {
                atomicOr(status, 1);
                atomicExch(abort_flag, 1);
                break;
            }
            tc_fence_after();
            const uint32_t a0 = smem_u32(sA + s * Cfg::A_BYTES);
            const uint32_t b0 = smem_u32(sB + s * Cfg::B_BYTES);
#pragma unroll
            for (int kk = 0; kk < BK / 16; ++kk) {
                tc_mma(tmem, smem_desc(a0 + kk * 32, Cfg::SW), smem_desc(b0 + kk * 32, Cfg::SW), idesc,
                       (kb > 0 || kk > 0) ? 1u : 0u);
            }
            tc_commit(smem_u32(empty_bar + s));   // frees the stage once these MMAs have read it
        }
        tc_commit(smem_u32(accum_bar));           // accumulator complete (or, after an abort, quiescent)
    } else if (warp >= 2) {
        // ---------------- epilogue
        if (!mbar_wait(smem_u32(accum_bar), 0)) {
            atomicOr(status, 1);
        } else if (!*reinterpret_cast<volatile int*>(abort_flag)) {
            tc_fence_after();
            const int q = warp & 3;
            const int row = m0 + q * 32 + lane;
            const uint32_t tbase = tmem + (static_cast<uint32_t>(q * 32) << 16);
#pragma unroll 1
            for (int c = 0; c < BN / 32; ++c) {
                if (n0 + c * 32 >= N) break;
                uint32_t r[32];
                tc_ld_32cols(tbase + c * 32, r);
                tc_wait_ld();
                epilogue_chunk<KIND>(epi, z, row, n0 + c * 32, M, N, r);
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tc_dealloc(tmem, BN);
    }
}

// ------------------------------------------------------------------ CTA-pair persistent kernel
// The persistent GEMM on CTA pairs: a cluster of two CTAs computes 256 x 256
// output tiles with tcgen05.mma.cta_group::2.  CTA r of the pair stages rows
// m0 + 128 r .. +127 of A and rows n0 + 128 r .. +127 of B (its half of the
// tile's B) in its own shared memory; one thread of the even CTA issues the
// MMAs, which read both CTAs' stages and accumulate output rows m0 + 128 r ..
// into CTA r's TMEM.  Per SM a 64-deep stage is 32 KB for 128 x 256 x 64 MACs,
// two thirds of what the single-CTA tile stages for the same work, so the ring
// is deeper in the same shared memory and each SM pulls fewer bytes per flop.
//
// One launch may carry two independent problems (nprob = 2, kinds KIND0 and
// KIND1): their tiles form one list, those of problem 0 first, dealt to the pairs
// in turn, so that the second problem fills the last partial wave of the first.
// Shared memory: the ring of STAGES stages, 256 bytes of barriers, then a 32 x 32
// bf16 transposing chunk per epilogue warp.
//
// Barriers (the same shared-memory offsets in both CTAs):
//   full[s]    even CTA only: its producer arrives with the byte count of both
//              CTAs' loads of stage s; the loads of both CTAs complete on it
//   empty[s]   both CTAs: the MMA issuer's commit arrives on both
//   tfull[a]   both CTAs: committed after the tile's last MMA into accumulator a
//   tempty[a]  even CTA only: the eight epilogue warps of each CTA arrive (16)
// Ten warps: 0 TMA producer and TMEM owner, 1 MMA issuer (even CTA), 2-9 epilogue:
// warp w reads TMEM lane quarter w % 4 (32 rows of the CTA's 128-row sub-tile) and
// the columns [128 h, 128 h + 128) of the tile, h = (w - 2) / 4.
constexpr int kPairThreads = 320;

struct PairProblem {
    CUtensorMap tmA, tmB;
    int M, N, K;
    TcEpi epi;
};
struct PairArgs {
    PairProblem p[2];
    int nprob;        // 1 or 2
    int* status;
};

// Live extent of one problem: rows past (*kdev) * kmul of the row dimension (M, or
// K for GBAR) are not computed.
struct PairShape {
    int Meff, Keff, live_k, mt_n, nt_n, msub_n, nk;
    long long tiles;
};
template <int KIND>
__device__ __forceinline__ PairShape pair_shape(const PairProblem& P) {
    constexpr int BN = 256, BK = 64;
    PairShape S;
    S.Meff = P.M;
    S.Keff = P.K;
    S.live_k = 1;
    if (P.epi.kdev) {
        S.live_k = *P.epi.kdev;
        const long long r = static_cast<long long>(S.live_k > 0 ? S.live_k : 0) * P.epi.kmul;
        if (KIND == TC_GBAR)
            S.Keff = r < P.K ? static_cast<int>(r) : P.K;
        else
            S.Meff = r < P.M ? static_cast<int>(r) : P.M;
    }
    S.mt_n = (S.Meff + 2 * BM - 1) / (2 * BM);
    S.nt_n = (P.N + BN - 1) / BN;
    S.msub_n = (P.M + BM - 1) / BM;   // 128-row sub-tiles of the full row extent
    S.tiles = S.live_k > 0 && S.Keff > 0 ? static_cast<long long>(S.mt_n) * S.nt_n : 0;
    S.nk = (S.Keff + BK - 1) / BK;
    return S;
}

// Epilogue of one tile for problem kind KIND (one thread: one row, 128 columns).
template <int KIND>
__device__ __forceinline__ void pair_epilogue(const PairProblem& P, const PairShape& S, long long t, int rank, int q,
                                              int h, int lane, uint32_t taddr, __nv_bfloat16* stg) {
    constexpr int BN = 256;
    const TcEpi& epi = P.epi;
    const int nt = static_cast<int>(t % S.nt_n);
    const int msub = static_cast<int>(t / S.nt_n) * 2 + rank;
    const int nb0 = nt * BN + h * (BN / 2);
    const int row = msub * BM + q * 32 + lane;
    if constexpr (KIND == TC_GBAR) {
        const bool wvec = ((reinterpret_cast<uintptr_t>(epi.W) & 15u) == 0) &&
                          ((reinterpret_cast<uintptr_t>(epi.gbar) & 15u) == 0) && epi.off % 4 == 0 &&
                          epi.ldrow % 4 == 0;
        double sq = gbar_cols(epi, row, nb0, P.M, P.N, 1.0f / static_cast<float>(S.live_k), taddr, wvec);
        // fixed-shape warp tree; one piece per (128-row sub-tile, column tile, half, quarter)
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
        if (lane == 0 && msub < S.msub_n) epi.pieces[(static_cast<long long>(msub) * S.nt_n + nt) * 8 + h * 4 + q] = sq;
    } else if constexpr (KIND == TC_DX) {
        const bool avec = ((reinterpret_cast<uintptr_t>(epi.act) & 15u) == 0) && epi.ldact % 8 == 0;
        dx_cols(epi, row, nb0, P.M, P.N, taddr, avec, stg);
    } else if constexpr (KIND == TC_HIDDEN) {
        hidden_cols(epi, row, nb0, P.M, P.N, taddr, stg);
    } else {
#pragma unroll 1
        for (int c = 0; c < 4; ++c) {
            if (nb0 + c * 32 >= P.N) break;
            uint32_t r[32];
            tc_ld_32cols(taddr + c * 32, r);
            tc_wait_ld();
            epilogue_chunk<KIND>(epi, 0, row, nb0 + c * 32, P.M, P.N, r);
        }
    }
}

template <int KIND0, int KIND1, int STAGES>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kPairThreads, 1)
    tc_gemm_pair_kernel(const __grid_constant__ PairArgs args) {
    constexpr int BN = 256, BK = 64, SW = 128;
    constexpr int A_BYTES = BM * BK * 2;          // 128 rows of A
    constexpr int B_BYTES = (BN / 2) * BK * 2;    // this CTA's 128 rows of B
    constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* sA = smem;
    uint8_t* sB = smem + STAGES * A_BYTES;
    uint64_t* full_bar = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
    uint64_t* empty_bar = full_bar + STAGES;
    uint64_t* tfull_bar = empty_bar + STAGES;    // [2]
    uint64_t* tempty_bar = tfull_bar + 2;        // [2]
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tempty_bar + 2);
    int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);
    // epilogue warps' transposing chunks, after the 256 bytes of barriers
    __nv_bfloat16* staging = reinterpret_cast<__nv_bfloat16*>(smem + STAGES * STAGE_BYTES + 256);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = cluster_rank();
    const long long pair = blockIdx.x >> 1, npairs = gridDim.x >> 1;
    int* status = args.status;
    const PairShape S0 = pair_shape<KIND0>(args.p[0]);
    PairShape S1 = S0;
    S1.tiles = 0;
    if (args.nprob > 1) S1 = pair_shape<KIND1>(args.p[1]);
    const long long total = S0.tiles + S1.tiles;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(smem_u32(full_bar + s), 1);
            mbar_init(smem_u32(empty_bar + s), 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(smem_u32(tfull_bar + a), 1);
            mbar_init(smem_u32(tempty_bar + a), 16);
        }
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 0) {
        tc2_alloc(smem_u32(tmem_slot), 2 * BN);
        tc2_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync();   // both CTAs' barriers exist before any remote arrive or load completes on them
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    volatile int* vabort = abort_flag;

    if (warp == 0 && lane == 0) {
        // ---------------- TMA producer (both CTAs)
        long long g = 0;
        for (long long t = pair; t < total && !*vabort; t += npairs) {
            const bool second = t >= S0.tiles;
            const long long u = second ? t - S0.tiles : t;
            const PairShape& S = second ? S1 : S0;
            const CUtensorMap* tmA = second ? &args.p[1].tmA : &args.p[0].tmA;
            const CUtensorMap* tmB = second ? &args.p[1].tmB : &args.p[0].tmB;
            const int ma = static_cast<int>(u / S.nt_n) * (2 * BM) + static_cast<int>(rank) * BM;
            const int nb = static_cast<int>(u % S.nt_n) * BN + static_cast<int>(rank) * (BN / 2);
            for (int kb = 0; kb < S.nk; ++kb, ++g) {
                const int s = static_cast<int>(g % STAGES);
                const uint32_t ph = static_cast<uint32_t>((g / STAGES) & 1);
                if (!mbar_wait(smem_u32(empty_bar + s), ph ^ 1)) {
                    atomicOr(status, 1);
                    *vabort = 1;
                    break;
                }
                if (rank == 0) mbar_expect_tx(smem_u32(full_bar + s), 2 * STAGE_BYTES);
                const uint32_t bar = map_to_rank(smem_u32(full_bar + s), 0);
                tma_load_2d_pair(smem_u32(sA + s * A_BYTES), tmA, kb * BK, ma, bar);
                tma_load_2d_pair(smem_u32(sB + s * B_BYTES), tmB, kb * BK, nb, bar);
            }
        }
        // the last use of every stage has been consumed: no load or commit is still
        // on its way into this CTA's shared memory
        if (!*vabort) {
            for (long long q = g - STAGES < 0 ? 0 : g - STAGES; q < g; ++q) {
                if (!mbar_wait(smem_u32(empty_bar + q % STAGES), static_cast<uint32_t>((q / STAGES) & 1))) {
                    atomicOr(status, 1);
                    *vabort = 1;
                    break;
                }
            }
        }
    } else if (warp == 1 && lane == 0 && rank == 0) {
        // ---------------- MMA issuer (even CTA)
        constexpr uint32_t idesc = instr_desc_bf16(2 * BM, BN);
        long long g = 0;
        int i = 0;
        for (long long t = pair; t < total && !*vabort; t += npairs, ++i) {
            const int nk = t >= S0.tiles ? S1.nk : S0.nk;
            const int acc = i & 1;
            const uint32_t aph = static_cast<uint32_t>((i >> 1) & 1);
            if (!mbar_wait(smem_u32(tempty_bar + acc), aph ^ 1)) {
                atomicOr(status, 1);
                *vabort = 1;
                break;
            }
            tc_fence_after();
            const uint32_t dcol = tmem + static_cast<uint32_t>(acc * BN);
            bool ok = true;
            for (int kb = 0; kb < nk; ++kb, ++g) {
                const int s = static_cast<int>(g % STAGES);
                const uint32_t ph = static_cast<uint32_t>((g / STAGES) & 1);
                if (!mbar_wait(smem_u32(full_bar + s), ph)) {
                    atomicOr(status, 1);
                    *vabort = 1;
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t a0 = smem_u32(sA + s * A_BYTES);
                const uint32_t b0 = smem_u32(sB + s * B_BYTES);
#pragma unroll
                for (int kk = 0; kk < BK / 16; ++kk)
                    tc2_mma(dcol, smem_desc(a0 + kk * 32, SW), smem_desc(b0 + kk * 32, SW), idesc,
                            (kb > 0 || kk > 0) ? 1u : 0u);
                tc2_commit_multicast(smem_u32(empty_bar + s), 0x3);
            }
            tc2_commit_multicast(smem_u32(tfull_bar + acc), 0x3);
            if (!ok) break;
        }
    } else if (warp >= 2) {
        // ---------------- epilogue (both CTAs): 128-row sub-tile msub, lane quarter q, column half h
        const int q = warp & 3, h = (warp - 2) >> 2;
        __nv_bfloat16* stg = staging + (warp - 2) * (kStageBytes / 2);
        int i = 0;
        for (long long t = pair; t < total; t += npairs, ++i) {
            const int acc = i & 1;
            const uint32_t aph = static_cast<uint32_t>((i >> 1) & 1);
            if (!mbar_wait(smem_u32(tfull_bar + acc), aph)) {
                atomicOr(status, 1);
                *vabort = 1;
                break;
            }
            if (*vabort) break;
            tc_fence_after();
            const uint32_t taddr = tmem + static_cast<uint32_t>(acc * BN + h * (BN / 2)) +
                                   (static_cast<uint32_t>(q * 32) << 16);
            if (t < S0.tiles)
                pair_epilogue<KIND0>(args.p[0], S0, t, static_cast<int>(rank), q, h, lane, taddr, stg);
            else
                pair_epilogue<KIND1>(args.p[1], S1, t - S0.tiles, static_cast<int>(rank), q, h, lane, taddr,
                                     stg);
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_remote(map_to_rank(smem_u32(tempty_bar + acc), 0));
        }
    }
    tc_fence_before();
    __syncthreads();
    if (*vabort && threadIdx.x == 0) {
        // a wait ran out: give the pair's loads and MMAs still in flight time to land
        // before the shared memory and the TMEM are released
        const uint64_t t0 = globaltimer();
        while (globaltimer() - t0 < 200000ull) {
        }
    }
    __syncthreads();
    cluster_sync();
    if (warp == 0) {
        tc_fence_after();
        tc2_dealloc(tmem, 2 * BN);
    }
}

// ------------------------------------------------------------------ persistent dW kernel
// Per-worker weight gradient G[z*ldG + m*ldrow + n] = sum_{k < K} A[m, z*K + k] B[n, z*K + k]
// (A = dZ^T [out, M], B = A_{l-1}^T [in, M], K = the worker's B samples).
//
// The kernel is bound by writing G (K is small), so it is built around that
// store.  A persistent grid (one CTA per SM) walks the tiles worker-major with n
// fastest; the MMA of tile i+1 runs into the second of two 256-column TMEM
// accumulators while the epilogue drains tile i.  Eight epilogue warps: two per
// TMEM lane quarter (32 rows of G), each owning 128 of the tile's 256 columns.
// A warp copies its 32 x 128 fp32 block TMEM -> registers -> shared memory
// (16-byte pieces XOR-swizzled by row, conflict-free) and then writes it row by
// row: each store instruction covers 512 contiguous bytes of one G row, the
// pattern that reaches the highest write bandwidth on this part.
constexpr int DW_BN = 256;
constexpr int DW_EPI_WARPS = 8;
constexpr int DW_THREADS = 32 * (2 + DW_EPI_WARPS);
constexpr int DW_WARP_COLS = 128;                         // columns of the tile per epilogue warp
constexpr int DW_STAGING_BYTES = 32 * DW_WARP_COLS * 4;   // 32 rows x 512 bytes per warp

template <int BK, int STAGES>
struct DwCfg {
    static constexpr int A_BYTES = BM * BK * 2;
    static constexpr int B_BYTES = DW_BN * BK * 2;
    static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
    static constexpr int SW = BK * 2;
    static constexpr int STAGING = DW_EPI_WARPS * DW_STAGING_BYTES;
    static constexpr int BAR_BYTES = 256;
    static constexpr int SMEM = STAGES * STAGE_BYTES + STAGING + BAR_BYTES + 1024;
};

// Tests of the bounded-wait path (the kTest instantiation, launched only when armed):
// the bound of the kernel's waits, and one pipeline stage whose TMA load the first CTA
// does not issue, so that the MMA's wait for it runs out as a lost copy would make it.
// The production instantiation ignores these: its waits are bounded by kWaitLimitNs.
struct DwWaits {
    unsigned long long limit_ns;   // every mbarrier wait of the launch
    long long skip_stage;          // stage counter g of block 0 left without its load; -1: none
};

template <int BK, int STAGES, bool kTest = false>
__global__ void __launch_bounds__(DW_THREADS, 1)
    tc_dw_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB, int Mr, int Nr,
                 int K, int batch, int* status, float* __restrict__ Gbase, int64_t ldrow, int64_t ldG, DwWaits wt) {
    const uint64_t wait_ns = kTest ? wt.limit_ns : kWaitLimitNs;
    using Cfg = DwCfg<BK, STAGES>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* sA = smem;
    uint8_t* sB = smem + STAGES * Cfg::A_BYTES;
    uint8_t* staging = smem + STAGES * Cfg::STAGE_BYTES;
    uint64_t* full_bar = reinterpret_cast<uint64_t*>(staging + Cfg::STAGING);
    uint64_t* empty_bar = full_bar + STAGES;
    uint64_t* tfull_bar = empty_bar + STAGES;    // [2] accumulator ready
    uint64_t* tempty_bar = tfull_bar + 2;        // [2] accumulator drained (all epilogue warps)
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tempty_bar + 2);
    int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int mt_n = (Mr + BM - 1) / BM, nt_n = (Nr + DW_BN - 1) / DW_BN;
    const int tiles_per_z = mt_n * nt_n;
    const long long total = static_cast<long long>(tiles_per_z) * batch;
    const int nk = (K + BK - 1) / BK;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(smem_u32(full_bar + s), 1);
            mbar_init(smem_u32(empty_bar + s), 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(smem_u32(tfull_bar + a), 1);
            mbar_init(smem_u32(tempty_bar + a), DW_EPI_WARPS);
        }
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 0) {
        tc_alloc(smem_u32(tmem_slot), 2 * DW_BN);
        tc_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    volatile int* vabort = abort_flag;

    if (warp == 0 && lane == 0) {
        // ---------------- TMA producer: every k block of every tile this CTA owns
        long long g = 0;
        long long issued = 0;
        for (long long t = blockIdx.x; t < total && !*vabort; t += gridDim.x) {
            const int z = static_cast<int>(t / tiles_per_z);
            const int rem = static_cast<int>(t % tiles_per_z);
            // n (out) fastest: consecutive tiles, run by neighbouring SMs at the same
            // time, fill the same G rows' line ranges together
            const int m0 = (rem / nt_n) * BM, n0 = (rem % nt_n) * DW_BN;
            for (int kb = 0; kb < nk; ++kb, ++g) {
                const int s = static_cast<int>(g % STAGES);
                const uint32_t ph = static_cast<uint32_t>((g / STAGES) & 1);
                if (!mbar_wait(smem_u32(empty_bar + s), ph ^ 1, wait_ns)) {
                    atomicOr(status, 1);
                    *vabort = 1;
                    break;
                }
                if (!(kTest && blockIdx.x == 0 && g == wt.skip_stage)) {
                    mbar_expect_tx(smem_u32(full_bar + s), Cfg::STAGE_BYTES);
                    const int kx = z * K + kb * BK;
                    tma_load_2d(smem_u32(sA + s * Cfg::A_BYTES), &tmA, kx, m0, smem_u32(full_bar + s));
                    tma_load_2d(smem_u32(sB + s * Cfg::B_BYTES), &tmB, kx, n0, smem_u32(full_bar + s));
                }
                issued = g + 1;
            }
        }
        if (*vabort) {
            // the loads of the last STAGES stages may still be landing: wait for them (a
            // stage whose load never started only runs out its bound)
            for (long long q = issued - STAGES < 0 ? 0 : issued - STAGES; q < issued; ++q)
                mbar_wait(smem_u32(full_bar + q % STAGES), static_cast<uint32_t>((q / STAGES) & 1), wait_ns);
        }
    } else if (warp == 1 && lane == 0) {
        // ---------------- MMA issuer
        constexpr uint32_t idesc = instr_desc_bf16(BM, DW_BN);
        long long g = 0;
        int i = 0;
        for (long long t = blockIdx.x; t < total && !*vabort; t += gridDim.x, ++i) {
            const int acc = i & 1;
            const uint32_t aph = static_cast<uint32_t>((i >> 1) & 1);
            if (!mbar_wait(smem_u32(tempty_bar + acc), aph ^ 1, wait_ns)) {
                atomicOr(status, 1);
                *vabort = 1;
                break;
            }
            tc_fence_after();
            const uint32_t dcol = tmem + static_cast<uint32_t>(acc * DW_BN);
            bool ok = true;
            for (int kb = 0; kb < nk; ++kb, ++g) {
                const int s = static_cast<int>(g % STAGES);
                const uint32_t ph = static_cast<uint32_t>((g / STAGES) & 1);
                if (!mbar_wait(smem_u32(full_bar + s), ph, wait_ns)) {
                    atomicOr(status, 1);
                    *vabort = 1;
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t a0 = smem_u32(sA + s * Cfg::A_BYTES);
                const uint32_t b0 = smem_u32(sB + s * Cfg::B_BYTES);
#pragma unroll
                for (int kk = 0; kk < BK / 16; ++kk)
                    tc_mma(dcol, smem_desc(a0 + kk * 32, Cfg::SW), smem_desc(b0 + kk * 32, Cfg::SW), idesc,
                           (kb > 0 || kk > 0) ? 1u : 0u);
                tc_commit(smem_u32(empty_bar + s));
            }
            tc_commit(smem_u32(tfull_bar + acc));
            if (!ok) break;
        }
    } else if (warp >= 2) {
        // ---------------- epilogue: TMEM -> registers -> swizzled smem -> 512-byte row stores
        const int q = warp & 3;                 // TMEM lanes 32q .. 32q+31 = G rows m0 + 32q ..
        const int half = (warp - 2) >> 2;       // columns [128 half, 128 half + 128) of the tile
        uint8_t* buf = staging + (warp - 2) * DW_STAGING_BYTES;
        int i = 0;
        for (long long t = blockIdx.x; t < total; t += gridDim.x, ++i) {
            const int acc = i & 1;
            const uint32_t aph = static_cast<uint32_t>((i >> 1) & 1);
            if (!mbar_wait(smem_u32(tfull_bar + acc), aph, wait_ns)) {
                atomicOr(status, 1);
                *vabort = 1;
                break;
            }
            if (*vabort) break;
            tc_fence_after();
            const int z = static_cast<int>(t / tiles_per_z);
            const int rem = static_cast<int>(t % tiles_per_z);
            const int m0 = (rem / nt_n) * BM, n0 = (rem % nt_n) * DW_BN;
            const uint32_t tbase = tmem + static_cast<uint32_t>(acc * DW_BN) + (static_cast<uint32_t>(q * 32) << 16);
            const int row0 = m0 + q * 32;
            const int colw = n0 + half * DW_WARP_COLS;      // first column of this warp's block
            if (row0 < Mr && colw < Nr) {
                // 1) TMEM -> smem: lane = row; 16-byte piece p of 128-byte segment sgm of row r
                //    lives at r*512 + sgm*128 + ((p ^ (r & 7)) * 16)
#pragma unroll 1
                for (int sgm = 0; sgm < DW_WARP_COLS / 32; ++sgm) {
                    uint32_t r[32];
                    tc_ld_32cols(tbase + half * DW_WARP_COLS + sgm * 32, r);
                    tc_wait_ld();
#pragma unroll
                    for (int pc = 0; pc < 8; ++pc)
                        *reinterpret_cast<uint4*>(buf + lane * 512 + sgm * 128 + ((pc ^ (lane & 7)) << 4)) =
                            make_uint4(r[4 * pc], r[4 * pc + 1], r[4 * pc + 2], r[4 * pc + 3]);
                }
                __syncwarp();
                // 2) smem -> G, one row per instruction: lane L writes columns colw + 4L .. +3
                const int sgm = lane >> 3, pc = lane & 7;
                const int col = colw + 4 * lane;
                const bool col_ok = col + 3 < Nr;   // Nr % 4 == 0 on this path: whole pieces in or out
                float* gcol = Gbase + static_cast<int64_t>(z) * ldG + col;
#pragma unroll 4
                for (int rr = 0; rr < 32; ++rr) {
                    const uint4 v = *reinterpret_cast<const uint4*>(buf + rr * 512 + sgm * 128 + ((pc ^ (rr & 7)) << 4));
                    if (col_ok && row0 + rr < Mr)
                        __stcs(reinterpret_cast<float4*>(gcol + static_cast<int64_t>(row0 + rr) * ldrow),
                               make_float4(__uint_as_float(v.x), __uint_as_float(v.y), __uint_as_float(v.z),
                                           __uint_as_float(v.w)));
                }
                __syncwarp();
            }
            // every tcgen05.ld of this accumulator has completed (wait::ld above)
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(tempty_bar + acc));
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tc_dealloc(tmem, 2 * DW_BN);
    }
}

// ------------------------------------------------------------------ host side
// One-shot arming of a lost load in the next launch of tc_dw_kernel (tests of the
// bounded-wait path; see dbw_test_arm_wait_timeout).
std::atomic<long long> g_dw_skip_stage{-1};
std::atomic<unsigned long long> g_dw_test_limit_ns{0};

template <int BK, int STAGES>
cudaError_t launch_dw(const CUtensorMap& a, const CUtensorMap& b, int Mr, int Nr, int K, int batch, int* status,
                      float* gbase, int64_t ldrow, int64_t ldG, cudaStream_t st) {
    using Cfg = DwCfg<BK, STAGES>;
    DwWaits wt{kWaitLimitNs, -1};
    const long long skip = g_dw_skip_stage.exchange(-1);
    const bool test = skip >= 0;
    if (test) {
        wt.skip_stage = skip;
        wt.limit_ns = g_dw_test_limit_ns.load();
    }
    auto kern = test ? tc_dw_kernel<BK, STAGES, true> : tc_dw_kernel<BK, STAGES, false>;
    // each CTA holds all 512 TMEM columns: ask for enough shared memory that a
    // second CTA can never be resident on the same SM (it would wait in tcgen05.alloc)
    const int smem = Cfg::SMEM > 120 * 1024 ? Cfg::SMEM : 120 * 1024;
    cudaError_t err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (err != cudaSuccess) return err;
    const long long tiles = static_cast<long long>((Mr + BM - 1) / BM) * ((Nr + DW_BN - 1) / DW_BN) * batch;
    const int grid = static_cast<int>(tiles < sm_count() ? tiles : sm_count());
    kern<<<grid, DW_THREADS, smem, st>>>(a, b, Mr, Nr, K, batch, status, gbase, ldrow, ldG, wt);
    return cudaGetLastError();
}

#ifndef DBW_PAIR_STAGES
#define DBW_PAIR_STAGES 6   // TMA ring depth of the CTA-pair GEMM (32 KB per stage and CTA)
#endif

// Co-resident 2-CTA clusters of the pair kernel (the persistent grid), once per kind.
template <class Kern>
int pair_slots(Kern kern, int smem) {
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.gridDim = dim3(2 * (sm_count() / 2), 1, 1);
    cfg.blockDim = dim3(kPairThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess || n < 1) {
        cudaGetLastError();
        n = sm_count() / 2;
    }
    return n;
}

template <int KIND0, int KIND1>
cudaError_t launch_pair(const PairArgs& args, cudaStream_t st) {
    constexpr int STAGES = DBW_PAIR_STAGES;
    constexpr int SMEM = STAGES * (2 * BM * 64 * 2) + 256 + 8 * kStageBytes + 1024;
    static_assert(SMEM <= 227 * 1024, "pair ring does not fit in shared memory");
    auto kern = tc_gemm_pair_kernel<KIND0, KIND1, STAGES>;
    cudaError_t err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM);
    if (err != cudaSuccess) return err;
    static int slots = 0;
    static std::once_flag once;
    std::call_once(once, [&] { slots = pair_slots(kern, SMEM); });
    long long tiles = 0;   // upper bound: the live extents are read on the device
    for (int i = 0; i < args.nprob; ++i)
        tiles += static_cast<long long>((args.p[i].M + 2 * BM - 1) / (2 * BM)) * ((args.p[i].N + 255) / 256);
    const int pairs = static_cast<int>(tiles < slots ? tiles : slots);
    if (pairs < 1) return cudaSuccess;
    kern<<<2 * pairs, kPairThreads, SMEM, st>>>(args);
    return cudaGetLastError();
}

template <int BN, int BK, int STAGES, int KIND, int MINB>
cudaError_t launch_cfg(const CUtensorMap& a, const CUtensorMap& b, int M, int N, int K, int batch, int64_t kz,
                       const TcEpi& e, int* status, cudaStream_t st, int min_smem) {
    using Cfg = TcCfg<BN, BK, STAGES>;
    auto kern = tc_gemm_kernel<BN, BK, STAGES, KIND, MINB>;
    const int smem = Cfg::SMEM > min_smem ? Cfg::SMEM : min_smem;
    cudaError_t err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (err != cudaSuccess) return err;
    dim3 grid((N + BN - 1) / BN, (M + BM - 1) / BM, batch);
    kern<<<grid, kThreads, smem, st>>>(a, b, M, N, K, kz, e, status);
    return cudaGetLastError();
}

}  // namespace

void arm_dw_wait_timeout(long long stage, unsigned long long limit_ns) {
    g_dw_test_limit_ns.store(limit_ns);
    g_dw_skip_stage.store(stage);
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    });
    return fn;
}

// 2-D tensor map of a row-major bf16 matrix [rows, cols] with row stride ld (elements).
bool tc_make_map(CUtensorMap* tm, const void* base, int64_t rows, int64_t cols, int64_t ld, int box_k, int box_rows) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
    cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld * 2)};
    cuuint32_t box[2] = {static_cast<cuuint32_t>(box_k), static_cast<cuuint32_t>(box_rows)};
    cuuint32_t estr[2] = {1, 1};
    const CUtensorMapSwizzle sw = box_k == 64 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B;
    return fn(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 2-D tensor map of a row-major fp32 matrix [rows, cols] with row stride ld (elements):
// box 32 x box_rows (128-byte rows, 128-byte swizzle); reads past the extents are zero.
bool tc_make_map_f32(CUtensorMap* tm, const void* base, int64_t rows, int64_t cols, int64_t ld, int box_rows) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
    cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld * 4)};
    cuuint32_t box[2] = {32u, static_cast<cuuint32_t>(box_rows)};
    cuuint32_t estr[2] = {1, 1};
    return fn(tm, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<void*>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool tc_shape_ok(int64_t lda, int64_t ldb, int K, int64_t kz, const void* A, const void* B) {
    if (!encode_fn()) return false;
    if ((lda % 8) || (ldb % 8) || (kz % 8)) return false;
    if ((reinterpret_cast<uintptr_t>(A) & 15u) || (reinterpret_cast<uintptr_t>(B) & 15u)) return false;
    if (kz > 0 && K % 32) return false;   // a batch's K must be whole K blocks (it is the column offset step)
    return K >= 1;
}

// One problem of the pair kernel: 256 x 256 tiles, each CTA stages 128 rows of A
// and 128 rows of B.
static int pair_problem(PairProblem* P, const __nv_bfloat16* A, int64_t lda, int64_t rowsA, int64_t colsA,
                        const __nv_bfloat16* B, int64_t ldb, int64_t rowsB, int64_t colsB, int M, int N, int K,
                        const TcEpi& epi) {
    if (!tc_shape_ok(lda, ldb, K, 0, A, B)) return fail(DBW_EALIGN, "tc_gemm: unsupported operand alignment");
    if (!tc_make_map(&P->tmA, A, rowsA, colsA, lda, 64, BM) || !tc_make_map(&P->tmB, B, rowsB, colsB, ldb, 64, 128))
        return fail(DBW_ECUDA, "tc_gemm: cuTensorMapEncodeTiled failed");
    P->M = M;
    P->N = N;
    P->K = K;
    P->epi = epi;
    return DBW_OK;
}

int tc_gemm_mean_dx(const TcOperands& g, const TcEpi& ge, const TcOperands& x, const TcEpi& xe, int* status,
                    cudaStream_t st) {
    PairArgs args{};
    args.nprob = 2;
    args.status = status;
    int rc = pair_problem(&args.p[0], g.A, g.lda, g.rowsA, g.colsA, g.B, g.ldb, g.rowsB, g.colsB, g.M, g.N, g.K, ge);
    if (rc) return rc;
    rc = pair_problem(&args.p[1], x.A, x.lda, x.rowsA, x.colsA, x.B, x.ldb, x.rowsB, x.colsB, x.M, x.N, x.K, xe);
    if (rc) return rc;
    void* prof = profile_begin(PROF_GEMM, st, 0.0);
    const cudaError_t e = launch_pair<TC_GBAR, TC_DX>(args, st);
    profile_end(prof, st);
    if (e != cudaSuccess) return fail(DBW_ECUDA, "tc_gemm_mean_dx launch: %s", cudaGetErrorString(e));
    return DBW_OK;
}

int tc_gemm(int kind, const __nv_bfloat16* A, int64_t lda, int64_t rowsA, int64_t colsA, const __nv_bfloat16* B,
            int64_t ldb, int64_t rowsB, int64_t colsB, int M, int N, int K, int batch, int64_t kz, const TcEpi& epi,
            int* status, cudaStream_t st) {
    cudaError_t e = cudaSuccess;
    if (kind == TC_DW) {
        if (!tc_shape_ok(lda, ldb, K, kz, A, B)) return fail(DBW_EALIGN, "tc_gemm: unsupported operand alignment");
        CUtensorMap ta, tb;
        // K = the per-worker sample count: 64-deep blocks when it allows, else 32
        const int bk = (K % 64 == 0) ? 64 : 32;
        // algorithmic bytes: G written once (fp32), both bf16 operands read once
        const double dw_bytes = 4.0 * batch * double(M) * N + 2.0 * batch * double(K) * (double(M) + N);
        if (!tc_make_map(&ta, A, rowsA, colsA, lda, bk, BM) || !tc_make_map(&tb, B, rowsB, colsB, ldb, bk, DW_BN))
            return fail(DBW_ECUDA, "tc_gemm: cuTensorMapEncodeTiled failed");
        float* gb = epi.G + epi.off;
        const bool vec_ok = ((reinterpret_cast<uintptr_t>(gb) & 15u) == 0) && epi.ldrow % 4 == 0 && epi.ldG % 4 == 0;
        // unaligned rows: the one-CTA-per-tile kernel (128-column tiles) with scalar stores
        if (!vec_ok && !tc_make_map(&tb, B, rowsB, colsB, ldb, bk, 128))
            return fail(DBW_ECUDA, "tc_gemm: cuTensorMapEncodeTiled failed");
        void* prof = profile_begin(PROF_DW, st, dw_bytes);
        if (!vec_ok) {
            e = bk == 64 ? launch_cfg<128, 64, 2, TC_DW, 4>(ta, tb, M, N, K, batch, kz, epi, status, st, 48 * 1024)
                         : launch_cfg<128, 32, 2, TC_DW, 4>(ta, tb, M, N, K, batch, kz, epi, status, st, 48 * 1024);
        } else {
            e = bk == 64 ? launch_dw<64, 2>(ta, tb, M, N, K, batch, status, gb, epi.ldrow, epi.ldG, st)
                         : launch_dw<32, 4>(ta, tb, M, N, K, batch, status, gb, epi.ldrow, epi.ldG, st);
        }
        profile_end(prof, st);
    } else {
        PairArgs args{};
        args.nprob = 1;
        args.status = status;
        const int rc = pair_problem(&args.p[0], A, lda, rowsA, colsA, B, ldb, rowsB, colsB, M, N, K, epi);
        if (rc) return rc;
        void* prof = profile_begin(PROF_GEMM, st, 0.0);
        if (kind == TC_HIDDEN)
            e = launch_pair<TC_HIDDEN, TC_HIDDEN>(args, st);
        else if (kind == TC_LOGITS)
            e = launch_pair<TC_LOGITS, TC_LOGITS>(args, st);
        else if (kind == TC_GBAR)
            e = launch_pair<TC_GBAR, TC_GBAR>(args, st);
        else
            e = launch_pair<TC_DX, TC_DX>(args, st);
        profile_end(prof, st);
    }
    if (e != cudaSuccess) return fail(DBW_ECUDA, "tc_gemm launch: %s", cudaGetErrorString(e));
    return DBW_OK;
}

}  // namespace dbw
