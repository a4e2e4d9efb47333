// The DBW estimator on the device (Sect. 3): end-of-iteration statistics
// (Eqs. (10)-(12), time bookkeeping of Sect. 3.2) and the choice of k_t
// (Eqs. (13)-(19)).  Everything is fp64 and runs in one CTA.
//
// This file is compiled with -fmad=false: every multiply and add below is a
// separately rounded IEEE operation, performed in the order written, so that a
// state reproduced elsewhere with the same operation order yields the same b_t
// bit for bit.  The sequential pieces (window sums, the loss mean) run in one
// thread on purpose: their summation order is part of that contract.  Their inputs
// are first loaded into shared memory by all threads, and so are the state's scalar
// fields (one round trip instead of one per field).
#include <math.h>
#include <math_constants.h>
#include <stddef.h>

#include "common.cuh"

namespace dbw {

namespace {

constexpr int kRedThreads = 256;

__device__ __forceinline__ int ring_slot(int cnt_minus_v) { return cnt_minus_v % DBW_DMAX; }

__device__ double window_mean(const double* ring, int cnt, int D) {
    const int m = cnt < D ? cnt : D;
    double acc = 0.0;
    for (int v = 1; v <= m; ++v) acc = acc + ring[ring_slot(cnt - v)];
    return acc / (double)m;
}

// The state's scalar fields (everything before the rings), copied into shared memory by
// the first threads in one round trip; the sequential code then reads the copy and
// writes its results to the state itself.
constexpr int kHeadWords = static_cast<int>(offsetof(dbw_state, ringV) / 8);
static_assert(offsetof(dbw_state, ringV) % 8 == 0, "the state's scalar fields are whole 8-byte words");

__device__ __forceinline__ const dbw_state* stage_head(const dbw_state* st, unsigned long long* head) {
    if (threadIdx.x < kHeadWords) head[threadIdx.x] = reinterpret_cast<const unsigned long long*>(st)[threadIdx.x];
    __syncthreads();
    return reinterpret_cast<const dbw_state*>(head);
}

// Sum of the per-block pieces of one quantity, in a fixed order: thread t adds
// blocks t, t + 256, ... sequentially, then a fixed pairwise tree.
__global__ void __launch_bounds__(kRedThreads) reduce_partials_kernel(double* __restrict__ partials, int n) {
    const int64_t* hdr = reinterpret_cast<const int64_t*>(partials);
    double* sums = partials + kPartialsHeader;
    if (hdr[0] != kPartialsMagic || hdr[2] != n || hdr[1] < 1 || hdr[1] > (1 << 20)) {
        // not written by dbw_aggregate_update for this n: poison instead of reading
        if (threadIdx.x == 0) sums[blockIdx.x] = CUDART_NAN;
        return;
    }
    const int blocks = (int)hdr[1];
    const double* vals = partials + kPartialsHeader + (n + 2) + (int64_t)blockIdx.x * blocks;
    __shared__ double red[kRedThreads];
    double s = 0.0;
    for (int i = threadIdx.x; i < blocks; i += kRedThreads) s = s + vals[i];
    red[threadIdx.x] = s;
    __syncthreads();
    for (int h = kRedThreads / 2; h > 0; h >>= 1) {
        if (threadIdx.x < h) red[threadIdx.x] = red[threadIdx.x] + red[threadIdx.x + h];
        __syncthreads();
    }
    if (threadIdx.x == 0) sums[blockIdx.x] = red[0];
}

__global__ void __launch_bounds__(1024) grad_stats_kernel(
    const double* __restrict__ sums, int n, const uint8_t* __restrict__ mask,
    const float* __restrict__ loss, const double* __restrict__ tsorted, double lr,
    dbw_state* __restrict__ st, double* __restrict__ stats_out, double* __restrict__ row_sqnorm) {
    __shared__ int k_s;
    // the mask and the losses, loaded by every thread at once; thread 0 then runs the
    // sequential sums from shared memory (n <= DBW_NMAX: checked by the caller)
    __shared__ uint8_t mask_s[DBW_NMAX];
    __shared__ float loss_s[DBW_NMAX];
    __shared__ unsigned long long head_s[kHeadWords];
    const int tid = threadIdx.x;
    for (int j = tid; j < n; j += blockDim.x) {
        mask_s[j] = mask[j] ? 1 : 0;
        loss_s[j] = loss[j];
    }
    const dbw_state* sh = stage_head(st, head_s);   // (its barrier also orders mask_s, loss_s)
    if (tid == 0) {
        int k = 0;
        for (int j = 0; j < n; ++j) k += mask_s[j];
        k_s = k;
        if (k == 0 || sh->n != n) {
            st->flags = sh->flags | (k == 0 ? DBW_FLAG_EMPTY_MASK : 0) | (sh->n != n ? DBW_FLAG_BAD_STATE : 0);
            k_s = 0;
        }
    }
    __syncthreads();
    if (k_s == 0) return;
    if (tid == 0) {
        const int k = k_s;
        double acc = 0.0;
        for (int j = 0; j < n; ++j)
            if (mask_s[j]) acc = acc + (double)loss_s[j];
        const double SS = sums[n];
        const double g2 = sums[n + 1];
        const double F = acc / (double)k;
        double V = CUDART_NAN, N = CUDART_NAN, L = CUDART_NAN;
        int flags = 0;
        if (k >= 2) {
            V = SS / (double)(k - 1);                         // Eq. (10)
            const double x = g2 - V / (double)k;              // Eq. (11)
            N = x > 0.0 ? x : 0.0;
        } else {
            flags |= DBW_FLAG_K1;
        }
        if (sh->t >= 1 && sh->has_last) {                     // Eq. (12)
            const double num = 2.0 * ((lr * sh->N_last) - (sh->F_last - F));
            const double den = (lr * lr) * (sh->N_last + (sh->V_last / (double)sh->k_last));
            if (den > 0.0) L = num / den;
            if (!(den > 0.0 && isfinite(L))) {
                L = CUDART_NAN;
                flags |= DBW_FLAG_L_SKIPPED;
            } else {
                st->ringL[sh->cntL % DBW_DMAX] = L;
                st->cntL = sh->cntL + 1;
            }
        }
        if (k >= 2) {
            st->ringV[sh->cntV % DBW_DMAX] = V;
            st->cntV = sh->cntV + 1;
            st->ringN[sh->cntN % DBW_DMAX] = N;
            st->cntN = sh->cntN + 1;
            st->N_last = N;
            st->V_last = V;
            st->has_last = 1;
        } else {
            st->N_last = CUDART_NAN;
            st->V_last = CUDART_NAN;
            st->has_last = 0;
        }
        st->c = sh->c + 1;
        const double vclock = sh->vclock + tsorted[k - 1];
        st->vclock = vclock;
        st->F_prev = sh->F_last;
        st->F_last = F;
        st->k_last = k;
        st->t = sh->t + 1;
        st->flags = sh->flags | flags;
        if (stats_out) {
            stats_out[DBW_STAT_K] = (double)k;
            stats_out[DBW_STAT_SS] = SS;
            stats_out[DBW_STAT_GBAR_SQ] = g2;
            stats_out[DBW_STAT_V] = V;
            stats_out[DBW_STAT_N] = N;
            stats_out[DBW_STAT_F] = F;
            stats_out[DBW_STAT_L] = L;
            stats_out[DBW_STAT_FLAGS] = (double)flags;
            stats_out[DBW_STAT_VCLOCK] = vclock;
        }
    }
    // Sect. 3.2: every arrival is observed, S[r] accumulates the r-th order statistic
    for (int r = tid; r < n; r += blockDim.x) st->S[r] = st->S[r] + tsorted[r];
    if (row_sqnorm) {
        // the partials header says whether the rows the mask left out were read too
        const bool all_rows = (reinterpret_cast<const int64_t*>(sums - kPartialsHeader)[3] & DBW_ALL_ROW_NORMS) != 0;
        for (int j = tid; j < n; j += blockDim.x) row_sqnorm[j] = (mask[j] || all_rows) ? sums[j] : CUDART_NAN;
    }
}

// T_ext (nullable): time estimates T^_k = T_ext[k-1] instead of S[k-1] / c; NaN in
// T_ext[0] means no estimate yet.
__global__ void __launch_bounds__(1024) choose_b_kernel(dbw_state* __restrict__ st, double lr, double beta,
                                                        int flags, int32_t* __restrict__ b_out,
                                                        double* __restrict__ ratio_out,
                                                        const double* __restrict__ T_ext) {
    __shared__ double Vh_s, Nh_s, q_s;
    __shared__ int ready_s;
    __shared__ double best_r[32];
    __shared__ int best_k[32];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    __shared__ unsigned long long head_s[kHeadWords];
    const dbw_state* sh = stage_head(st, head_s);
    const int n = sh->n;
    if (n < 1 || n > DBW_NMAX || sh->D < 1 || sh->D > DBW_DMAX || sh->cntV < 0 || sh->cntN < 0 ||
        sh->cntL < 0 || sh->c < 0) {
        if (tid == 0) st->flags = sh->flags | DBW_FLAG_BAD_STATE;
        return;
    }
    const bool blind = (flags & DBW_CHOOSE_BLIND) != 0;
    // the three windows' rings, loaded by every thread at once (window_mean then sums
    // them in its fixed order from shared memory)
    __shared__ double ring_s[3][DBW_DMAX];
    for (int e = tid; e < 3 * DBW_DMAX; e += blockDim.x) {
        const int r = e / DBW_DMAX, i = e - r * DBW_DMAX;
        ring_s[r][i] = (r == 0 ? st->ringV : r == 1 ? st->ringN : st->ringL)[i];
    }
    __syncthreads();
    if (tid == 0) {
        int ready;
        const bool have_T = T_ext ? !isnan(T_ext[0]) : sh->c > 0;
        if (blind) {
            ready = have_T;
        } else {
            ready = sh->cntV > 0 && sh->cntN > 0 && sh->cntL > 0 && sh->c > 0 && have_T;
            if (ready) {
                Vh_s = window_mean(ring_s[0], sh->cntV, sh->D);   // Eq. (13)
                Nh_s = window_mean(ring_s[1], sh->cntN, sh->D);   // Eq. (14)
                const double Lh = window_mean(ring_s[2], sh->cntL, sh->D);   // Eq. (15)
                q_s = ((Lh * lr) * lr) / 2.0;
            }
        }
        ready_s = ready;
    }
    __syncthreads();
    const int ready = ready_s;
    const double c = (double)sh->c;
    // candidate of this thread: k = tid + 1
    double my_r = -CUDART_INF;
    int my_k = 0;   // 0 = not eligible
    for (int k = tid + 1; k <= n; k += blockDim.x) {
        double ratio = CUDART_NAN;
        bool elig = false;
        if (ready) {
            const double T = T_ext ? T_ext[k - 1] : st->S[k - 1] / c;   // T^_k
            if (blind) {
                ratio = (double)k / T;
                elig = true;
            } else {
                const double gain = ((lr - q_s) * Nh_s) - (q_s * (Vh_s / (double)k));   // Eq. (16)
                ratio = gain / T;
                elig = gain > 0.0;
            }
        }
        if (ratio_out) ratio_out[k - 1] = ratio;
        if (elig && (my_k == 0 || ratio > my_r || (ratio == my_r && k > my_k))) {
            my_r = ratio;
            my_k = k;
        }
    }
    // Eq. (18): lexicographic max of (eligible, ratio, k) across the CTA
    for (int o = 16; o > 0; o >>= 1) {
        const double r2 = __shfl_xor_sync(0xffffffffu, my_r, o);
        const int k2 = __shfl_xor_sync(0xffffffffu, my_k, o);
        if (k2 != 0 && (my_k == 0 || r2 > my_r || (r2 == my_r && k2 > my_k))) {
            my_r = r2;
            my_k = k2;
        }
    }
    if (lane == 0) {
        best_r[warp] = my_r;
        best_k[warp] = my_k;
    }
    __syncthreads();
    if (tid == 0) {
        int kstar = 0;
        double rbest = -CUDART_INF;
        for (int wv = 0; wv < (int)(blockDim.x >> 5); ++wv) {
            const int k2 = best_k[wv];
            const double r2 = best_r[wv];
            if (k2 != 0 && (kstar == 0 || r2 > rbest || (r2 == rbest && k2 > kstar))) {
                rbest = r2;
                kstar = k2;
            }
        }
        if (kstar == 0) kstar = n;                                // R3 / R7: k = n
        if (sh->t >= 2 && sh->F_last > beta * sh->F_prev && sh->k_last < n) {   // Eq. (19)
            const int kg = sh->k_last + 1;
            if (kg > kstar) kstar = kg;
        }
        if (kstar > n) kstar = n;
        st->k_next = kstar;
        *b_out = n - kstar;
    }
}

__global__ void state_init_kernel(dbw_state* st, int n, int D) {
    double* raw = reinterpret_cast<double*>(st);
    const int nwords = (int)(sizeof(dbw_state) / sizeof(double));
    for (int i = threadIdx.x; i < nwords; i += blockDim.x) raw[i] = 0.0;
    __syncthreads();
    if (threadIdx.x == 0) {
        st->n = n;
        st->D = D;
        st->k_next = n;
        st->F_last = CUDART_NAN;
        st->F_prev = CUDART_NAN;
        st->N_last = CUDART_NAN;
        st->V_last = CUDART_NAN;
    }
}

}  // namespace

cudaError_t launch_state_init(dbw_state* s, int n, int D, cudaStream_t st) {
    state_init_kernel<<<1, 256, 0, st>>>(s, n, D);
    return cudaGetLastError();
}

cudaError_t launch_grad_stats(const double* partials, int n, const uint8_t* mask, const float* loss,
                              const double* tsorted, double lr, dbw_state* s, double* stats_out,
                              double* row_sqnorm, cudaStream_t st) {
    double* sums = const_cast<double*>(partials) + kPartialsHeader;
    reduce_partials_kernel<<<n + 2, kRedThreads, 0, st>>>(sums - kPartialsHeader, n);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    grad_stats_kernel<<<1, 1024, 0, st>>>(sums, n, mask, loss, tsorted, lr, s, stats_out, row_sqnorm);
    return cudaGetLastError();
}

cudaError_t launch_choose_b(dbw_state* s, double lr, double beta, int flags, int32_t* b_out,
                            double* ratio_out, const double* T_ext, cudaStream_t st) {
    choose_b_kernel<<<1, 1024, 0, st>>>(s, lr, beta, flags, b_out, ratio_out, T_ext);
    return cudaGetLastError();
}

}  // namespace dbw
