// Opt-in launch timing of two kernel families: the per-worker weight-gradient
// launches that write G (channel DW), and the persistent tcgen05 GEMMs of the
// forward pass, the input gradient and the mean gradient (channel GEMM).  CUDA
// events are recorded on the launching stream around each launch; durations and
// the work the caller attached are accumulated until the channel is read.
#include <mutex>
#include <vector>

#include "common.cuh"
#include "profile.cuh"

namespace dbw {

namespace {
struct Channel {
    bool enabled = false;
    std::vector<cudaEvent_t> pool;     // 2 events per launch, reused
    size_t used = 0;                   // events recorded since the last read
    std::vector<double> work;          // work attached to each recorded launch
};
std::mutex g_mu;
Channel g_chan[PROF_CHANNELS];

cudaEvent_t next_event(Channel& c) {
    if (c.used == c.pool.size()) {
        cudaEvent_t e = nullptr;
        if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
        c.pool.push_back(e);
    }
    return c.pool[c.used++];
}

int enable(int ch, int on) {
    std::lock_guard<std::mutex> lock(g_mu);
    g_chan[ch].enabled = on != 0;
    g_chan[ch].used = 0;
    g_chan[ch].work.clear();
    return DBW_OK;
}

int read(int ch, const char* who, double* total_ms, int64_t* launches, double* total_work) {
    if (!total_ms || !launches) return fail(DBW_EINVAL, "%s: NULL pointer argument", who);
    std::lock_guard<std::mutex> lock(g_mu);
    Channel& c = g_chan[ch];
    double ms = 0.0, work = 0.0;
    const size_t pairs = c.used / 2;
    for (size_t i = 0; i < pairs; ++i) {
        float t = 0.f;
        cudaEvent_t a = c.pool[2 * i], b = c.pool[2 * i + 1];
        if (cudaEventSynchronize(b) != cudaSuccess || cudaEventElapsedTime(&t, a, b) != cudaSuccess)
            return fail(DBW_ECUDA, "%s: event timing failed", who);
        ms += t;
        work += c.work[i];
    }
    *total_ms = ms;
    *launches = static_cast<int64_t>(pairs);
    if (total_work) *total_work = work;
    c.used = 0;
    c.work.clear();
    return DBW_OK;
}
}  // namespace

void* profile_begin(int ch, cudaStream_t st, double work) {
    std::lock_guard<std::mutex> lock(g_mu);
    Channel& c = g_chan[ch];
    if (!c.enabled) return nullptr;
    cudaEvent_t a = next_event(c);
    if (!a) return nullptr;
    cudaEventRecord(a, st);
    c.work.push_back(work);
    return &c;
}

void profile_end(void* token, cudaStream_t st) {
    if (!token) return;
    std::lock_guard<std::mutex> lock(g_mu);
    Channel& c = *static_cast<Channel*>(token);
    cudaEvent_t b = next_event(c);
    if (b) cudaEventRecord(b, st);
}

}  // namespace dbw

using namespace dbw;

extern "C" int dbw_profile_dw(int on) { return enable(PROF_DW, on); }

extern "C" int dbw_profile_dw_read(double* total_ms, int64_t* launches, double* total_bytes) {
    if (!total_bytes) return fail(DBW_EINVAL, "dbw_profile_dw_read: NULL pointer argument");
    return read(PROF_DW, "dbw_profile_dw_read", total_ms, launches, total_bytes);
}

extern "C" int dbw_profile_gemm(int on) { return enable(PROF_GEMM, on); }

extern "C" int dbw_profile_gemm_read(double* total_ms, int64_t* launches) {
    return read(PROF_GEMM, "dbw_profile_gemm_read", total_ms, launches, nullptr);
}
