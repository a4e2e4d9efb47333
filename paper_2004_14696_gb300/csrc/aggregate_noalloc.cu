// dbw_aggregate_update_noalloc: the fused aggregation of dbw_aggregate_update
// for callers that cannot hand the library any scratch memory.
//
// Who needs this: code that is not allowed to allocate device memory at all,
// for example a plugin running inside a host application that owns the whole
// GPU memory budget and gives its plugins only the tensors they work on, or a
// latency-critical loop in which cudaMalloc (which can synchronise the whole
// device) is not acceptable.  Such a caller passes only its inputs and outputs.
//
// Where the scratch lives instead: the per-block partial sums that
// dbw_aggregate_update writes into caller memory are written here into one
// file-scope device array of fixed size (kScratchBytes).  Every GPU that loads
// libdbw holds this array until the process exits.  All calls on a device share
// it and it keeps whatever the last call wrote.  Each call first clears the
// array's header (cudaMemsetAsync on the call's stream, which allocates
// nothing) and the aggregation kernel overwrites every other value the
// reduction later reads; so if the aggregation does not run, the reduction
// finds no valid header and writes NaN instead of the previous call's totals.
// Two calls whose work overlaps on the GPU (different streams without ordering
// between them) race on the array and corrupt each other's sums.
//
// Set-up: host code cannot use the array's name as a device address, so the
// first call on each device asks the runtime for the array's device address
// (cudaGetSymbolAddress) with that device current, caches it per device and
// passes it to the kernels.  That first call should come before any stream
// capture begins.
//
// This entry point calls no cudaMalloc, cudaFree or other allocating routine.
#include <math_constants.h>

#include <mutex>

#include "common.cuh"

namespace dbw {

namespace {

constexpr size_t kScratchBytes = DBW_NOALLOC_SCRATCH_BYTES;
static __device__ __align__(256) unsigned char g_agg_scratch[kScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void* g_scratch_ptr[kMaxDevices] = {nullptr};

// Device address of g_agg_scratch on the current device (looked up once per device).
int scratch_address(void** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return fail(DBW_ECUDA, "dbw_aggregate_update_noalloc: %s", cudaGetErrorString(e));
    if (dev < 0 || dev >= kMaxDevices)
        return fail(DBW_EUNSUPPORTED, "dbw_aggregate_update_noalloc: device index %d not supported", dev);
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_scratch_ptr[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_agg_scratch);
        if (e != cudaSuccess || !p)
            return fail(DBW_ECUDA, "dbw_aggregate_update_noalloc: cudaGetSymbolAddress failed: %s",
                        cudaGetErrorString(e));
        g_scratch_ptr[dev] = p;
    }
    *out = g_scratch_ptr[dev];
    return DBW_OK;
}

// sums_out[q] = total of quantity q over the per-block pieces, in the same fixed
// order dbw_grad_stats uses (256 strided partial sums, then a pairwise tree).  A
// header that the aggregation of this call did not write gives NaN.
constexpr int kRed = 256;
__global__ void __launch_bounds__(kRed) reduce_to_sums_kernel(const double* __restrict__ partials, int n,
                                                              double* __restrict__ sums_out) {
    const int64_t* hdr = reinterpret_cast<const int64_t*>(partials);
    if (hdr[0] != kPartialsMagic || hdr[2] != n || hdr[1] < 1 || hdr[1] > (1 << 20)) {
        if (threadIdx.x == 0) sums_out[blockIdx.x] = CUDART_NAN;
        return;
    }
    const int blocks = (int)hdr[1];
    const double* vals = partials + kPartialsHeader + (n + 2) + (int64_t)blockIdx.x * blocks;
    __shared__ double red[kRed];
    double s = 0.0;
    for (int i = threadIdx.x; i < blocks; i += kRed) s = s + vals[i];
    red[threadIdx.x] = s;
    __syncthreads();
    for (int h = kRed / 2; h > 0; h >>= 1) {
        if (threadIdx.x < h) red[threadIdx.x] = red[threadIdx.x] + red[threadIdx.x + h];
        __syncthreads();
    }
    if (threadIdx.x == 0) sums_out[blockIdx.x] = red[0];
}

}  // namespace

}  // namespace dbw

using namespace dbw;

extern "C" int dbw_aggregate_update_noalloc(const float* G, int64_t ld, int n, int64_t d, const uint8_t* mask,
                                            float lr, float* w, float* gbar, int flags, double* sums_out,
                                            void* stream) {
    clear_error();
    Call call("dbw_aggregate_update_noalloc", as_stream(stream));
    if (!G || !mask || !w || !sums_out)
        return fail(DBW_EINVAL, "dbw_aggregate_update_noalloc: NULL pointer argument");
    if (flags & ~DBW_ALL_ROW_NORMS) return fail(DBW_EINVAL, "dbw_aggregate_update_noalloc: unknown flags");
    if (n < 1 || n > DBW_NMAX)
        return fail(DBW_EINVAL, "dbw_aggregate_update_noalloc: n must be in [1, %d]", DBW_NMAX);
    if (d < 1) return fail(DBW_EINVAL, "dbw_aggregate_update_noalloc: d must be >= 1");
    if (ld < d || ld % 4 != 0)
        return fail(DBW_EALIGN, "dbw_aggregate_update_noalloc: ld must be >= d and a multiple of 4");
    if (!aligned16(G) || !aligned16(w) || (gbar && !aligned16(gbar)))
        return fail(DBW_EALIGN, "dbw_aggregate_update_noalloc: G, w, gbar must be 16-byte aligned");
    int rc = check_device();
    if (rc) return rc;
    const AggGeometry g = agg_geometry(n, d);
    if (g.bytes > kScratchBytes)
        return fail(DBW_EINVAL,
                    "dbw_aggregate_update_noalloc: n = %d needs %zu bytes of scratch on this device, more than the "
                    "built-in %zu; use dbw_aggregate_update with caller memory",
                    n, g.bytes, kScratchBytes);
    void* scratch = nullptr;
    rc = scratch_address(&scratch);
    if (rc) return rc;
    double* partials = static_cast<double*>(scratch);
    cudaStream_t st = as_stream(stream);
    cudaError_t e = cudaMemsetAsync(partials, 0, kPartialsHeader * sizeof(int64_t), st);
    if (e != cudaSuccess) return fail(DBW_ECUDA, "dbw_aggregate_update_noalloc: %s", cudaGetErrorString(e));
    e = launch_aggregate(G, ld, n, d, mask, lr, w, gbar, flags, partials, g, st);
    if (e != cudaSuccess) return fail(DBW_ECUDA, "dbw_aggregate_update_noalloc: %s", cudaGetErrorString(e));
    reduce_to_sums_kernel<<<n + 2, kRed, 0, st>>>(partials, n, sums_out);
    e = cudaGetLastError();
    if (e != cudaSuccess) return fail(DBW_ECUDA, "dbw_aggregate_update_noalloc: %s", cudaGetErrorString(e));
    return call.done(DBW_OK);
}
