// Launch accounting of the library: a per-kernel launch counter (always on) and optional
// CUDA-event timing of every launch on its own stream (cyfa_stats_* in include/cyfa.h).
#include <mutex>
#include <string>
#include <utility>
#include <vector>

#include "../../include/cyfa.h"
#include "kernels.h"

namespace cyfa {

namespace {

struct Entry {
    std::string name;
    long long launches = 0;
    double ms = 0.0;
    std::vector<std::pair<cudaEvent_t, cudaEvent_t>> pending;
};

std::mutex g_mu;
std::vector<Entry> g_entries;
std::vector<cudaEvent_t> g_pool;
bool g_timing = false;

cudaEvent_t take_event() {
    if (!g_pool.empty()) {
        cudaEvent_t e = g_pool.back();
        g_pool.pop_back();
        return e;
    }
    cudaEvent_t e = nullptr;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    return e;
}

int find_or_add(const char* name) {
    for (size_t i = 0; i < g_entries.size(); ++i)
        if (g_entries[i].name == name) return (int)i;
    g_entries.push_back(Entry{});
    g_entries.back().name = name;
    return (int)g_entries.size() - 1;
}

void resolve(Entry& e) {
    for (auto& pr : e.pending) {
        float ms = 0.f;
        if (cudaEventSynchronize(pr.second) == cudaSuccess &&
            cudaEventElapsedTime(&ms, pr.first, pr.second) == cudaSuccess)
            e.ms += ms;
        g_pool.push_back(pr.first);
        g_pool.push_back(pr.second);
    }
    e.pending.clear();
}

}  // namespace

LaunchScope::LaunchScope(const char* name, cudaStream_t st) : stream_(st) {
    std::lock_guard<std::mutex> lk(g_mu);
    idx_ = find_or_add(name);
    g_entries[idx_].launches++;
    if (g_timing) {
        start_ = take_event();
        if (start_) cudaEventRecord(start_, st);
    }
}

LaunchScope::~LaunchScope() {
    if (!start_) return;
    std::lock_guard<std::mutex> lk(g_mu);
    cudaEvent_t stop = take_event();
    if (!stop) return;
    cudaEventRecord(stop, stream_);
    g_entries[idx_].pending.emplace_back(start_, stop);
}

}  // namespace cyfa

using namespace cyfa;

extern "C" {

int cyfa_stats_reset(void) {
    std::lock_guard<std::mutex> lk(g_mu);
    for (auto& e : g_entries) resolve(e);
    g_entries.clear();
    return CYFA_OK;
}

int cyfa_stats_timing(int on) {
    std::lock_guard<std::mutex> lk(g_mu);
    g_timing = on != 0;
    return CYFA_OK;
}

int cyfa_stats_get(int index, char* name, int name_len, long long* launches, double* total_ms) {
    std::lock_guard<std::mutex> lk(g_mu);
    if (index < 0 || index >= (int)g_entries.size()) return CYFA_ERR_ARG;
    Entry& e = g_entries[index];
    resolve(e);
    if (name && name_len > 0) {
        const size_t n = std::min((size_t)name_len - 1, e.name.size());
        e.name.copy(name, n);
        name[n] = '\0';
    }
    if (launches) *launches = e.launches;
    if (total_ms) *total_ms = e.ms;
    return CYFA_OK;
}

}  // extern "C"
