// Internal helpers shared by the CUDA translation units of libdbw.
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "dbw.h"

namespace dbw {

// Records a message for dbw_last_error_string() and returns ``code``.
int fail(int code, const char* fmt, ...);
// Empties dbw_last_error_string() of the calling thread (every entry point starts with it).
void clear_error();
// Maps a pending launch error to DBW_ECUDA (with its text), else DBW_OK.
int check_launch(const char* what);
// Number of SMs of the current device (cached per device).
int sm_count();
// DBW_OK if the current device is sm_103 (compute capability 10.3), else DBW_EUNSUPPORTED.
int check_device();

// One C-ABI call: an NVTX range named after the entry point (seen by timeline tools,
// a no-op otherwise) and, with DBW_DEBUG_SYNC=1 in the environment, a
// synchronisation of the call's stream before it returns, so that an asynchronous
// fault is reported by the call that launched it (skipped while the stream is being
// captured into a graph).
class Call {
public:
    Call(const char* name, cudaStream_t st);
    ~Call();
    Call(const Call&) = delete;
    Call& operator=(const Call&) = delete;
    // rc, or DBW_ECUDA when the debug synchronisation reports an error.
    int done(int rc);

private:
    const char* name_;
    cudaStream_t st_;
};

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
inline bool aligned256(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 255u) == 0; }
inline cudaStream_t as_stream(void* s) { return reinterpret_cast<cudaStream_t>(s); }

// ----------------------------------------------------------------- launchers
// Selection (select.cu)
cudaError_t launch_select(const double* times, int n, const int32_t* b, int32_t* order,
                          uint8_t* mask, double* tsorted, int32_t* k_out, cudaStream_t st);

// Aggregation (aggregate.cu)
struct AggGeometry {
    int blocks;           // persistent grid size
    int rows_stride;      // n + 2: values per block in the partials
    size_t bytes;         // total partials bytes
};
AggGeometry agg_geometry(int n, int64_t d);
// flags: 0 or DBW_ALL_ROW_NORMS
cudaError_t launch_aggregate(const float* G, int64_t ld, int n, int64_t d, const uint8_t* mask,
                             float lr, float* w, float* gbar, int flags, double* partials,
                             const AggGeometry& g, cudaStream_t st);

// Estimator (estimator.cu)
cudaError_t launch_state_init(dbw_state* s, int n, int D, cudaStream_t st);
cudaError_t launch_grad_stats(const double* partials, int n, const uint8_t* mask, const float* loss,
                              const double* tsorted, double lr, dbw_state* s, double* stats_out,
                              double* row_sqnorm, cudaStream_t st);
cudaError_t launch_choose_b(dbw_state* s, double lr, double beta, int flags, int32_t* b_out,
                            double* ratio_out, const double* T_ext, cudaStream_t st);

// Push-and-wait clock and Eq. (17) (psw.cu)
size_t psw_bytes(int n);
cudaError_t launch_psw_init(void* psw, int n, cudaStream_t st);
cudaError_t launch_psw_arrivals(const void* psw, int n, const double* omega, double* e, cudaStream_t st);
cudaError_t launch_psw_record(void* psw, int n, const int32_t* order, const double* tsorted, const int32_t* k,
                              cudaStream_t st);
cudaError_t launch_psw_estimate(void* psw, int n, double tol, int max_sweeps, double* T_hat, cudaStream_t st);

// Worker gradients (grads.cu)
struct GradsPlan;
size_t grads_workspace_bytes(int L, const int32_t* widths, int n, int B, int prec);
int grads_activations(int L, const int32_t* widths, int n, int B, int prec, int layer, size_t* offset, int64_t* ld,
                      int* elem_bytes);
int launch_worker_grads(int L, const int32_t* widths, int prec, const float* w, int64_t d,
                        const float* pool, int64_t S, const int32_t* labels, const int32_t* idx,
                        int n, int B, float* G, int64_t ld, float* loss, void* ws, size_t ws_bytes,
                        cudaStream_t st);

// Tests of the bounded waits (gemm_tc.cu): the next weight-gradient launch bounds its
// waits by limit_ns and its first CTA does not issue the load of pipeline stage
// ``stage``; stage < 0 disarms.
void arm_dw_wait_timeout(long long stage, unsigned long long limit_ns);

// Received-workers pass (grads_tc.cu)
size_t received_workspace_bytes(int L, const int32_t* widths, int n, int B, int prec);
int launch_received_grads(int L, const int32_t* widths, int prec, float* w, int64_t d, const float* pool, int64_t S,
                          const int32_t* labels, const int32_t* idx, int n, int B, const uint8_t* mask, float lr,
                          float* gbar, float* loss, double* partials, void* ws, size_t ws_bytes, cudaStream_t st);

// Partials buffer layout shared by aggregate.cu, grads_tc.cu and estimator.cu:
//   int64 header[4] = {magic, blocks, n, flags (DBW_ALL_ROW_NORMS when every row's norm is in)}
//   double sums[n + 2]              reduced totals (written by dbw_grad_stats)
//   double vals[(n + 2) * blocks]   per-block pieces, by quantity: vals[q * blocks + blk]
//                                   q < n: ||g_q||^2, q = n: SS, q = n + 1: ||g_t||^2
constexpr int64_t kPartialsMagic = DBW_PARTIALS_MAGIC;  // "DBWPART"
constexpr int kPartialsHeader = 4;

}  // namespace dbw
