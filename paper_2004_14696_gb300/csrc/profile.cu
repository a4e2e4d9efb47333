// Opt-in timing of the per-worker weight-gradient launches (the kernel that
// writes G): CUDA events recorded on the launching stream around each launch,
// durations and algorithmic bytes accumulated for dbw_profile_dw_read.
#include <mutex>
#include <vector>

#include "common.cuh"
#include "profile.cuh"

namespace dbw {

namespace {
struct DwProfile {
    bool enabled = false;
    std::vector<cudaEvent_t> pool;     // 2 events per launch, reused
    size_t used = 0;                   // events recorded since the last read
    std::vector<double> bytes;         // algorithmic bytes of each recorded launch
};
std::mutex g_mu;
DwProfile g_prof;

cudaEvent_t next_event() {
    if (g_prof.used == g_prof.pool.size()) {
        cudaEvent_t e = nullptr;
        if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
        g_prof.pool.push_back(e);
    }
    return g_prof.pool[g_prof.used++];
}
}  // namespace

void* dw_profile_begin(cudaStream_t st, double algorithmic_bytes) {
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_prof.enabled) return nullptr;
    cudaEvent_t a = next_event();
    if (!a) return nullptr;
    cudaEventRecord(a, st);
    g_prof.bytes.push_back(algorithmic_bytes);
    return a;
}

void dw_profile_end(void* token, cudaStream_t st) {
    if (!token) return;
    std::lock_guard<std::mutex> lock(g_mu);
    cudaEvent_t b = next_event();
    if (b) cudaEventRecord(b, st);
}

}  // namespace dbw

using namespace dbw;

extern "C" int dbw_profile_dw(int enable) {
    std::lock_guard<std::mutex> lock(g_mu);
    g_prof.enabled = enable != 0;
    g_prof.used = 0;
    g_prof.bytes.clear();
    return DBW_OK;
}

extern "C" int dbw_profile_dw_read(double* total_ms, int64_t* launches, double* total_bytes) {
    if (!total_ms || !launches || !total_bytes) return fail(DBW_EINVAL, "dbw_profile_dw_read: NULL pointer argument");
    std::lock_guard<std::mutex> lock(g_mu);
    double ms = 0.0, bytes = 0.0;
    const size_t pairs = g_prof.used / 2;
    for (size_t i = 0; i < pairs; ++i) {
        float t = 0.f;
        cudaEvent_t a = g_prof.pool[2 * i], b = g_prof.pool[2 * i + 1];
        if (cudaEventSynchronize(b) != cudaSuccess || cudaEventElapsedTime(&t, a, b) != cudaSuccess)
            return fail(DBW_ECUDA, "dbw_profile_dw_read: event timing failed");
        ms += t;
        bytes += g_prof.bytes[i];
    }
    *total_ms = ms;
    *launches = static_cast<int64_t>(pairs);
    *total_bytes = bytes;
    g_prof.used = 0;
    g_prof.bytes.clear();
    return DBW_OK;
}
