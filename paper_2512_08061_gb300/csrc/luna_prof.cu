// Kernel timing hook: brackets every launch of one named kernel with CUDA
// events recorded on the launching stream (luna_profile_start / _stop).
#include <string.h>

#include <atomic>
#include <mutex>
#include <vector>

#include "luna_prof.cuh"

namespace luna {
namespace {

constexpr int kMaxRecords = 4096;

struct Profiler {
    std::mutex mu;
    std::atomic<bool> on{false};  // read without the lock on every launch; the name is compared under it
    char name[64] = {0};
    std::vector<cudaEvent_t> ev;  // 2 per record
    int used = 0;
    bool open = false;
};

Profiler &prof() {
    static Profiler p;
    return p;
}

std::atomic<unsigned long long> g_launches{0};

}  // namespace

void prof_before(const char *kernel, cudaStream_t s) {
    g_launches.fetch_add(1, std::memory_order_relaxed);
    Profiler &p = prof();
    if (!p.on.load(std::memory_order_acquire)) return;
    std::lock_guard<std::mutex> g(p.mu);
    if (!p.on.load(std::memory_order_relaxed) || strcmp(kernel, p.name) != 0 || p.used >= kMaxRecords) return;
    cudaEventRecord(p.ev[2 * p.used], s);
    p.open = true;
}

void prof_after(const char *kernel, cudaStream_t s) {
    Profiler &p = prof();
    if (!p.on.load(std::memory_order_acquire)) return;
    std::lock_guard<std::mutex> g(p.mu);
    if (!p.on.load(std::memory_order_relaxed) || strcmp(kernel, p.name) != 0 || !p.open || p.used >= kMaxRecords)
        return;
    cudaEventRecord(p.ev[2 * p.used + 1], s);
    p.used++;
    p.open = false;
}

}  // namespace luna

using namespace luna;

extern "C" {

uint64_t luna_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

luna_status luna_profile_start(const char *kernel) {
    if (!kernel || strlen(kernel) >= 64) return LUNA_ERR_INVALID_ARG;
    Profiler &p = prof();
    std::lock_guard<std::mutex> g(p.mu);
    if (p.ev.empty()) {
        p.ev.resize(2 * kMaxRecords);
        for (auto &e : p.ev)
            if (cudaEventCreate(&e) != cudaSuccess) {
                p.ev.clear();
                return LUNA_ERR_CUDA;
            }
    }
    strncpy(p.name, kernel, sizeof(p.name) - 1);
    p.used = 0;
    p.open = false;
    p.on.store(true, std::memory_order_release);
    return LUNA_OK;
}

luna_status luna_profile_stop(double *total_ms, int *launches) {
    if (!total_ms || !launches) return LUNA_ERR_INVALID_ARG;
    Profiler &p = prof();
    std::lock_guard<std::mutex> g(p.mu);
    p.on.store(false, std::memory_order_release);
    double tot = 0.0;
    for (int i = 0; i < p.used; ++i) {
        if (cudaEventSynchronize(p.ev[2 * i + 1]) != cudaSuccess) return LUNA_ERR_CUDA;
        float ms = 0.0f;
        if (cudaEventElapsedTime(&ms, p.ev[2 * i], p.ev[2 * i + 1]) != cudaSuccess) return LUNA_ERR_CUDA;
        tot += ms;
    }
    *total_ms = tot;
    *launches = p.used;
    p.used = 0;
    return LUNA_OK;
}

}  // extern "C"
