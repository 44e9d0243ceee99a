// Kernel-level tracing: when enabled, every kernel the library launches is bracketed by two
// CUDA events recorded on the launch stream; frac_trace_collect() waits for them and returns,
// per kernel name, the number of launches and the summed device time.  Disabled by default
// (no events, no overhead).
#include <cuda_runtime.h>

#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include "../../include/frac.h"
#include "kernels.h"

namespace {

struct Rec {
    const char *name;
    cudaEvent_t a, b;
};

std::mutex g_mu;
bool g_on = false;
std::vector<Rec> g_recs;
thread_local Rec g_open = {nullptr, nullptr, nullptr};

struct Agg {
    std::string name;
    int launches;
    double ms;
};
std::vector<Agg> g_agg;

}  // namespace

namespace frac {

void trace_begin(const char *name, cudaStream_t st) {
    if (!g_on) return;
    Rec r = {name, nullptr, nullptr};
    if (cudaEventCreate(&r.a) != cudaSuccess || cudaEventCreate(&r.b) != cudaSuccess) return;
    cudaEventRecord(r.a, st);
    g_open = r;
}

void trace_end(cudaStream_t st) {
    if (!g_on || !g_open.name) return;
    cudaEventRecord(g_open.b, st);
    std::lock_guard<std::mutex> lk(g_mu);
    g_recs.push_back(g_open);
    g_open = {nullptr, nullptr, nullptr};
}

}  // namespace frac

extern "C" {

frac_status frac_trace_enable(int on) {
    std::lock_guard<std::mutex> lk(g_mu);
    g_on = on != 0;
    return FRAC_OK;
}

frac_status frac_trace_collect(frac_trace_entry *out, int capacity, int *count) {
    std::lock_guard<std::mutex> lk(g_mu);
    for (const Rec &r : g_recs) {
        float ms = 0.f;
        if (cudaEventSynchronize(r.b) == cudaSuccess) cudaEventElapsedTime(&ms, r.a, r.b);
        cudaEventDestroy(r.a);
        cudaEventDestroy(r.b);
        bool found = false;
        for (Agg &g : g_agg)
            if (g.name == r.name) {
                g.launches += 1;
                g.ms += ms;
                found = true;
                break;
            }
        if (!found) g_agg.push_back({r.name, 1, double(ms)});
    }
    g_recs.clear();
    const int n = int(g_agg.size());
    if (count) *count = n;
    if (out) {
        for (int i = 0; i < n && i < capacity; ++i) {
            std::strncpy(out[i].name, g_agg[i].name.c_str(), sizeof(out[i].name) - 1);
            out[i].name[sizeof(out[i].name) - 1] = 0;
            out[i].launches = g_agg[i].launches;
            out[i].total_ms = g_agg[i].ms;
        }
    }
    return FRAC_OK;
}

frac_status frac_trace_reset(void) {
    std::lock_guard<std::mutex> lk(g_mu);
    for (const Rec &r : g_recs) {
        cudaEventDestroy(r.a);
        cudaEventDestroy(r.b);
    }
    g_recs.clear();
    g_agg.clear();
    return FRAC_OK;
}

}  // extern "C"
