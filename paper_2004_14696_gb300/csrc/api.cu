// extern "C" entry points of libdbw (declared in include/dbw.h): host-side
// argument checks, then launches on the caller's stream.  No entry point
// allocates device memory.
#include <nvtx3/nvToolsExt.h>
#include <stdarg.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include "common.cuh"

namespace dbw {

namespace {
thread_local char g_err[512] = "";

int device_sm_count_uncached(int dev) {
    int v = 0;
    cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev);
    return v > 0 ? v : 1;
}
}  // namespace

int fail(int code, const char* fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof(g_err), fmt, ap);
    va_end(ap);
    return code;
}

void clear_error() { g_err[0] = 0; }

int check_launch(const char* what) {
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return fail(DBW_ECUDA, "%s: %s", what, cudaGetErrorString(e));
    return DBW_OK;
}

int sm_count() {
    static int cache[64] = {0};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev < 0 || dev >= 64) return device_sm_count_uncached(dev);
    if (cache[dev] == 0) cache[dev] = device_sm_count_uncached(dev);
    return cache[dev];
}

Call::Call(const char* name, cudaStream_t st) : name_(name), st_(st) { nvtxRangePushA(name); }

Call::~Call() { nvtxRangePop(); }

int Call::done(int rc) {
    static const bool sync = [] {
        const char* v = getenv("DBW_DEBUG_SYNC");
        return v && v[0] == '1';
    }();
    if (rc != DBW_OK || !sync) return rc;
    cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(st_, &cap) != cudaSuccess || cap != cudaStreamCaptureStatusNone) return rc;
    const cudaError_t e = cudaStreamSynchronize(st_);
    if (e != cudaSuccess) return fail(DBW_ECUDA, "%s: %s (reported by the debug synchronisation)", name_,
                                      cudaGetErrorString(e));
    return rc;
}

int check_device() {
    static int cache[64] = {0};   // 0 unknown, 1 ok, 2 unsupported
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return fail(DBW_ECUDA, "no CUDA device");
    const int slot = dev >= 0 && dev < 64 ? dev : 0;
    if (cache[slot] == 0) {
        int major = 0, minor = 0;
        cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
        cache[slot] = (major == 10 && minor == 3) ? 1 : 2;
    }
    if (cache[slot] != 1) return fail(DBW_EUNSUPPORTED, "libdbw is built for sm_103 (GB300) only");
    return DBW_OK;
}

}  // namespace dbw

using namespace dbw;

extern "C" {

const char* dbw_last_error_string(void) { return g_err; }

int dbw_abi_version(void) { return 2; }

int64_t dbw_param_count(int num_layers, const int32_t* widths) {
    if (!widths || num_layers < 1 || num_layers > DBW_LMAX) return -1;
    int64_t d = 0;
    for (int l = 0; l < num_layers; ++l) {
        if (widths[l] < 1 || widths[l + 1] < 1) return -1;
        d += (int64_t)widths[l + 1] * ((int64_t)widths[l] + 1);
    }
    return d;
}

size_t dbw_worker_grads_workspace_bytes(int num_layers, const int32_t* widths, int n, int B, int prec) {
    if (!widths) return 0;
    return grads_workspace_bytes(num_layers, widths, n, B, prec);
}

int dbw_worker_grads_activations(int num_layers, const int32_t* widths, int n, int B, int prec, int layer,
                                 size_t* offset, int64_t* ld, int* elem_bytes) {
    g_err[0] = 0;
    if (!widths || !offset || !ld || !elem_bytes)
        return fail(DBW_EINVAL, "dbw_worker_grads_activations: NULL pointer argument");
    return grads_activations(num_layers, widths, n, B, prec, layer, offset, ld, elem_bytes);
}

int dbw_worker_grads(int num_layers, const int32_t* widths, int prec, const float* w, int64_t d, const float* pool,
                     int64_t S, const int32_t* labels, const int32_t* idx, int n, int B, float* G, int64_t ld,
                     float* loss, void* ws, size_t ws_bytes, void* stream) {
    g_err[0] = 0;
    Call call("dbw_worker_grads", as_stream(stream));
    if (!widths || !w || !pool || !labels || !idx || !G || !loss || !ws)
        return fail(DBW_EINVAL, "dbw_worker_grads: NULL pointer argument");
    if (S < 1) return fail(DBW_EINVAL, "dbw_worker_grads: S must be >= 1");
    if (ld < d || ld % 4 != 0) return fail(DBW_EALIGN, "dbw_worker_grads: ld must be >= d and a multiple of 4");
    if (!aligned16(w) || !aligned16(pool) || !aligned16(G) || !aligned256(ws))
        return fail(DBW_EALIGN, "dbw_worker_grads: w, pool, G must be 16-byte and ws 256-byte aligned");
    if (num_layers >= 1 && num_layers <= DBW_LMAX && widths[0] % 4 != 0)
        return fail(DBW_EALIGN, "dbw_worker_grads: widths[0] must be a multiple of 4");
    int rc = check_device();
    if (rc) return rc;
    return call.done(launch_worker_grads(num_layers, widths, prec, w, d, pool, S, labels, idx, n, B, G, ld, loss,
                                         ws, ws_bytes, as_stream(stream)));
}

int dbw_select_fastest(const double* times, int n, const int32_t* b, int32_t* order, uint8_t* mask, double* tsorted,
                       int32_t* k_out, void* stream) {
    g_err[0] = 0;
    Call call("dbw_select_fastest", as_stream(stream));
    if (!times || !b || !order || !mask || !tsorted)
        return fail(DBW_EINVAL, "dbw_select_fastest: NULL pointer argument");
    if (n < 1 || n > DBW_NMAX) return fail(DBW_EINVAL, "dbw_select_fastest: n must be in [1, %d]", DBW_NMAX);
    int rc = check_device();
    if (rc) return rc;
    cudaError_t e = launch_select(times, n, b, order, mask, tsorted, k_out, as_stream(stream));
    if (e != cudaSuccess) return fail(DBW_ECUDA, "dbw_select_fastest: %s", cudaGetErrorString(e));
    return call.done(DBW_OK);
}

size_t dbw_aggregate_partials_bytes(int n, int64_t d) {
    if (n < 1 || n > DBW_NMAX || d < 1) return 0;
    return agg_geometry(n, d).bytes;
}

int dbw_aggregate_update(const float* G, int64_t ld, int n, int64_t d, const uint8_t* mask, float lr, float* w,
                         float* gbar, int flags, double* partials, size_t partials_bytes, void* stream) {
    g_err[0] = 0;
    Call call("dbw_aggregate_update", as_stream(stream));
    if (!G || !mask || !w || !partials) return fail(DBW_EINVAL, "dbw_aggregate_update: NULL pointer argument");
    if (flags & ~DBW_ALL_ROW_NORMS) return fail(DBW_EINVAL, "dbw_aggregate_update: unknown flags");
    if (n < 1 || n > DBW_NMAX) return fail(DBW_EINVAL, "dbw_aggregate_update: n must be in [1, %d]", DBW_NMAX);
    if (d < 1) return fail(DBW_EINVAL, "dbw_aggregate_update: d must be >= 1");
    if (ld < d || ld % 4 != 0) return fail(DBW_EALIGN, "dbw_aggregate_update: ld must be >= d and a multiple of 4");
    if (!aligned16(G) || !aligned16(w) || (gbar && !aligned16(gbar)) || !aligned256(partials))
        return fail(DBW_EALIGN, "dbw_aggregate_update: G, w, gbar must be 16-byte and partials 256-byte aligned");
    int rc = check_device();
    if (rc) return rc;
    const AggGeometry g = agg_geometry(n, d);
    if (partials_bytes < g.bytes)
        return fail(DBW_EINVAL, "dbw_aggregate_update: partials %zu bytes < %zu needed", partials_bytes, g.bytes);
    cudaError_t e = launch_aggregate(G, ld, n, d, mask, lr, w, gbar, flags, partials, g, as_stream(stream));
    if (e != cudaSuccess) return fail(DBW_ECUDA, "dbw_aggregate_update: %s", cudaGetErrorString(e));
    return call.done(DBW_OK);
}

size_t dbw_received_grads_workspace_bytes(int num_layers, const int32_t* widths, int n, int B, int prec) {
    if (!widths) return 0;
    return received_workspace_bytes(num_layers, widths, n, B, prec);
}

size_t dbw_received_partials_bytes(int n) {
    if (n < 1 || n > DBW_NMAX) return 0;
    return sizeof(double) * (kPartialsHeader + 2 * ((size_t)n + 2));
}

int dbw_received_grads_update(int num_layers, const int32_t* widths, int prec, float* w, int64_t d, const float* pool,
                              int64_t S, const int32_t* labels, const int32_t* idx, int n, int B, const uint8_t* mask,
                              float lr, float* gbar, float* loss, double* partials, size_t partials_bytes, void* ws,
                              size_t ws_bytes, void* stream) {
    g_err[0] = 0;
    Call call("dbw_received_grads_update", as_stream(stream));
    if (!widths || !w || !pool || !labels || !idx || !mask || !loss || !partials || !ws)
        return fail(DBW_EINVAL, "dbw_received_grads_update: NULL pointer argument");
    if (S < 1) return fail(DBW_EINVAL, "dbw_received_grads_update: S must be >= 1");
    if (n < 1 || n > DBW_NMAX) return fail(DBW_EINVAL, "dbw_received_grads_update: n must be in [1, %d]", DBW_NMAX);
    if (partials_bytes < dbw_received_partials_bytes(n))
        return fail(DBW_EINVAL, "dbw_received_grads_update: partials %zu bytes < %zu needed", partials_bytes,
                    dbw_received_partials_bytes(n));
    if (!aligned16(w) || !aligned16(pool) || (gbar && !aligned16(gbar)) || !aligned256(partials) || !aligned256(ws))
        return fail(DBW_EALIGN,
                    "dbw_received_grads_update: w, pool, gbar must be 16-byte and partials, ws 256-byte aligned");
    if (num_layers >= 1 && num_layers <= DBW_LMAX && widths[0] % 4 != 0)
        return fail(DBW_EALIGN, "dbw_received_grads_update: widths[0] must be a multiple of 4");
    int rc = check_device();
    if (rc) return rc;
    return call.done(launch_received_grads(num_layers, widths, prec, w, d, pool, S, labels, idx, n, B, mask, lr,
                                           gbar, loss, partials, ws, ws_bytes, as_stream(stream)));
}

int dbw_state_init(dbw_state* state, int n, int D, void* stream) {
    g_err[0] = 0;
    Call call("dbw_state_init", as_stream(stream));
    if (!state) return fail(DBW_EINVAL, "dbw_state_init: NULL state");
    if (n < 1 || n > DBW_NMAX) return fail(DBW_EINVAL, "dbw_state_init: n must be in [1, %d]", DBW_NMAX);
    if (D < 1 || D > DBW_DMAX) return fail(DBW_EINVAL, "dbw_state_init: D must be in [1, %d]", DBW_DMAX);
    if (!aligned16(state)) return fail(DBW_EALIGN, "dbw_state_init: state must be 16-byte aligned");
    int rc = check_device();
    if (rc) return rc;
    cudaError_t e = launch_state_init(state, n, D, as_stream(stream));
    if (e != cudaSuccess) return fail(DBW_ECUDA, "dbw_state_init: %s", cudaGetErrorString(e));
    return call.done(DBW_OK);
}

int dbw_grad_stats(const double* partials, int n, const uint8_t* mask, const float* loss, const double* tsorted,
                   double lr, dbw_state* state, double* stats_out, double* row_sqnorm, void* stream) {
    g_err[0] = 0;
    Call call("dbw_grad_stats", as_stream(stream));
    if (!partials || !mask || !loss || !tsorted || !state)
        return fail(DBW_EINVAL, "dbw_grad_stats: NULL pointer argument");
    if (n < 1 || n > DBW_NMAX) return fail(DBW_EINVAL, "dbw_grad_stats: n must be in [1, %d]", DBW_NMAX);
    if (!(lr > 0.0)) return fail(DBW_EINVAL, "dbw_grad_stats: lr must be > 0");
    if (!aligned256(partials) || !aligned16(state)) return fail(DBW_EALIGN, "dbw_grad_stats: misaligned buffer");
    int rc = check_device();
    if (rc) return rc;
    cudaError_t e = launch_grad_stats(partials, n, mask, loss, tsorted, lr, state, stats_out, row_sqnorm,
                                      as_stream(stream));
    if (e != cudaSuccess) return fail(DBW_ECUDA, "dbw_grad_stats: %s", cudaGetErrorString(e));
    return call.done(DBW_OK);
}

int dbw_choose_b(dbw_state* state, double lr, double beta, int flags, int32_t* b_out, double* ratio_out,
                 void* stream) {
    g_err[0] = 0;
    Call call("dbw_choose_b", as_stream(stream));
    if (!state || !b_out) return fail(DBW_EINVAL, "dbw_choose_b: NULL pointer argument");
    if (!(lr > 0.0)) return fail(DBW_EINVAL, "dbw_choose_b: lr must be > 0");
    if (!(beta >= 1.0)) return fail(DBW_EINVAL, "dbw_choose_b: beta must be >= 1");
    if (flags & ~DBW_CHOOSE_BLIND) return fail(DBW_EINVAL, "dbw_choose_b: unknown flags");
    if (!aligned16(state)) return fail(DBW_EALIGN, "dbw_choose_b: state must be 16-byte aligned");
    int rc = check_device();
    if (rc) return rc;
    cudaError_t e = launch_choose_b(state, lr, beta, flags, b_out, ratio_out, nullptr, as_stream(stream));
    if (e != cudaSuccess) return fail(DBW_ECUDA, "dbw_choose_b: %s", cudaGetErrorString(e));
    return call.done(DBW_OK);
}

int dbw_choose_b_times(dbw_state* state, const double* T_hat, double lr, double beta, int flags, int32_t* b_out,
                       double* ratio_out, void* stream) {
    g_err[0] = 0;
    Call call("dbw_choose_b_times", as_stream(stream));
    if (!state || !T_hat || !b_out) return fail(DBW_EINVAL, "dbw_choose_b_times: NULL pointer argument");
    if (!(lr > 0.0)) return fail(DBW_EINVAL, "dbw_choose_b_times: lr must be > 0");
    if (!(beta >= 1.0)) return fail(DBW_EINVAL, "dbw_choose_b_times: beta must be >= 1");
    if (flags & ~DBW_CHOOSE_BLIND) return fail(DBW_EINVAL, "dbw_choose_b_times: unknown flags");
    if (!aligned16(state)) return fail(DBW_EALIGN, "dbw_choose_b_times: state must be 16-byte aligned");
    int rc = check_device();
    if (rc) return rc;
    cudaError_t e = launch_choose_b(state, lr, beta, flags, b_out, ratio_out, T_hat, as_stream(stream));
    if (e != cudaSuccess) return fail(DBW_ECUDA, "dbw_choose_b_times: %s", cudaGetErrorString(e));
    return call.done(DBW_OK);
}

int dbw_test_arm_wait_timeout(int stage, double wait_ms) {
    g_err[0] = 0;
    if (stage < 0) {
        arm_dw_wait_timeout(-1, 0);
        return DBW_OK;
    }
    if (!(wait_ms > 0.0 && wait_ms <= 2000.0))
        return fail(DBW_EINVAL, "dbw_test_arm_wait_timeout: wait_ms must be in (0, 2000]");
    arm_dw_wait_timeout(stage, static_cast<unsigned long long>(wait_ms * 1e6));
    return DBW_OK;
}

size_t dbw_psw_bytes(int n) {
    if (n < 1 || n > DBW_NMAX) return 0;
    return psw_bytes(n);
}

static int psw_args(const char* what, const void* psw, int n) {
    if (!psw) return fail(DBW_EINVAL, "%s: NULL state", what);
    if (n < 1 || n > DBW_NMAX) return fail(DBW_EINVAL, "%s: n must be in [1, %d]", what, DBW_NMAX);
    if (!aligned256(psw)) return fail(DBW_EALIGN, "%s: state must be 256-byte aligned", what);
    return check_device();
}

int dbw_psw_init(void* psw, int n, void* stream) {
    g_err[0] = 0;
    Call call("dbw_psw_init", as_stream(stream));
    int rc = psw_args("dbw_psw_init", psw, n);
    if (rc) return rc;
    cudaError_t e = launch_psw_init(psw, n, as_stream(stream));
    if (e != cudaSuccess) return fail(DBW_ECUDA, "dbw_psw_init: %s", cudaGetErrorString(e));
    return call.done(DBW_OK);
}

int dbw_psw_arrivals(const void* psw, int n, const double* omega, double* arrivals, void* stream) {
    g_err[0] = 0;
    Call call("dbw_psw_arrivals", as_stream(stream));
    if (!omega || !arrivals) return fail(DBW_EINVAL, "dbw_psw_arrivals: NULL pointer argument");
    int rc = psw_args("dbw_psw_arrivals", psw, n);
    if (rc) return rc;
    cudaError_t e = launch_psw_arrivals(psw, n, omega, arrivals, as_stream(stream));
    if (e != cudaSuccess) return fail(DBW_ECUDA, "dbw_psw_arrivals: %s", cudaGetErrorString(e));
    return call.done(DBW_OK);
}

int dbw_psw_record(void* psw, int n, const int32_t* order, const double* tsorted, const int32_t* k, void* stream) {
    g_err[0] = 0;
    Call call("dbw_psw_record", as_stream(stream));
    if (!order || !tsorted || !k) return fail(DBW_EINVAL, "dbw_psw_record: NULL pointer argument");
    int rc = psw_args("dbw_psw_record", psw, n);
    if (rc) return rc;
    cudaError_t e = launch_psw_record(psw, n, order, tsorted, k, as_stream(stream));
    if (e != cudaSuccess) return fail(DBW_ECUDA, "dbw_psw_record: %s", cudaGetErrorString(e));
    return call.done(DBW_OK);
}

int dbw_psw_estimate(void* psw, int n, double tol, int max_sweeps, double* T_hat, void* stream) {
    g_err[0] = 0;
    Call call("dbw_psw_estimate", as_stream(stream));
    if (!T_hat) return fail(DBW_EINVAL, "dbw_psw_estimate: NULL T_hat");
    if (!(tol > 0.0)) return fail(DBW_EINVAL, "dbw_psw_estimate: tol must be > 0");
    if (max_sweeps < 1) return fail(DBW_EINVAL, "dbw_psw_estimate: max_sweeps must be >= 1");
    int rc = psw_args("dbw_psw_estimate", psw, n);
    if (rc) return rc;
    cudaError_t e = launch_psw_estimate(psw, n, tol, max_sweeps, T_hat, as_stream(stream));
    if (e != cudaSuccess) return fail(DBW_ECUDA, "dbw_psw_estimate: %s", cudaGetErrorString(e));
    return call.done(DBW_OK);
}

}  // extern "C"
