// Eq. (4): arrival order of the n gradients and the k = n - b the PS keeps.
//
// One CTA, one thread per worker.  The times are staged once in shared memory;
// worker i's arrival rank is the number of workers j with (T_j, j) < (T_i, i),
// counted by its warp in parallel (each lane scans a 1/32 slice of the workers
// and the counts meet in a warp reduction), so the comparison work is spread
// over all 32 lanes instead of being an O(n) loop per thread.  Ranks of a
// strict total order are a permutation, which gives order, mask and the order
// statistics directly.
//
// The comparisons run on 64-bit integer keys: a double's bits, with the sign bit
// flipped for non-negative values and all bits flipped for negative ones (-0 is
// first made +0), order exactly as the doubles do and are equal exactly when the
// doubles are.  On this part a dependent fp64 compare costs ~12x an integer one.
#include "common.cuh"

namespace dbw {

namespace {
__device__ __forceinline__ unsigned long long order_key(double t) {
    unsigned long long u = static_cast<unsigned long long>(__double_as_longlong(t));
    if (u == 0x8000000000000000ull) u = 0;   // -0 == +0
    return (u >> 63) ? ~u : (u | 0x8000000000000000ull);
}
}  // namespace

__global__ void __launch_bounds__(1024) select_fastest_kernel(
    const double* __restrict__ times, int n, const int32_t* __restrict__ b_ptr,
    int32_t* __restrict__ order, uint8_t* __restrict__ mask, double* __restrict__ tsorted,
    int32_t* __restrict__ k_out) {
    __shared__ double ts[DBW_NMAX];
    __shared__ unsigned long long key[DBW_NMAX];
    __shared__ int rank_s[DBW_NMAX];
    const int tid = threadIdx.x;
    for (int i = tid; i < n; i += blockDim.x) {
        const double t = times[i];
        ts[i] = t;
        key[i] = order_key(t);
    }
    __syncthreads();

    int b = *b_ptr;
    b = b < 0 ? 0 : (b > n - 1 ? n - 1 : b);
    const int k = n - b;

    // warp w ranks workers w, w + nwarps, ...; lane l compares against j = l, l + 32, ...
    const int lane = tid & 31, warp = tid >> 5, nwarps = blockDim.x >> 5;
    for (int i = warp; i < n; i += nwarps) {
        const unsigned long long ki = key[i];
        int cnt = 0;
        for (int j = lane; j < n; j += 32) {
            const unsigned long long kj = key[j];
            cnt += (kj < ki) || (kj == ki && j < i);
        }
        cnt = __reduce_add_sync(0xffffffffu, cnt);
        if (lane == 0) rank_s[i] = cnt;
    }
    __syncthreads();
    for (int i = tid; i < n; i += blockDim.x) {
        const int r = rank_s[i];
        order[r] = i;
        tsorted[r] = ts[i];
        mask[i] = r < k ? 1 : 0;
    }
    if (tid == 0 && k_out) *k_out = k;
}

cudaError_t launch_select(const double* times, int n, const int32_t* b, int32_t* order,
                          uint8_t* mask, double* tsorted, int32_t* k_out, cudaStream_t st) {
    int threads = ((n + 31) / 32) * 32;
    if (threads < 256) threads = 256;
    if (threads > 1024) threads = 1024;
    select_fastest_kernel<<<1, threads, 0, st>>>(times, n, b, order, mask, tsorted, k_out);
    return cudaGetLastError();
}

}  // namespace dbw
