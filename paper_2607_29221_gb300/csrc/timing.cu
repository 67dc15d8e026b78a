// Optional per-kernel device timing for measurement (mosaic_kernel_timing /
// mosaic_kernel_times).  While timing is on, every launch that opens a
// KernelSpan on a stream that is not being captured into a graph is bracketed
// by a pair of CUDA events on that stream; the durations are summed per
// (calling entry point, kernel) when the caller asks for them.  Off by
// default: a disabled span costs one relaxed atomic load.
#include <string.h>

#include <map>
#include <mutex>
#include <string>
#include <vector>

#include "mosaic_internal.cuh"

namespace mosaic {
namespace {

std::atomic<int> g_timing{0};
thread_local const char *t_role = "other";

struct Pending {
    std::string key;
    int dev;
    cudaEvent_t e0, e1;
};
struct Total {
    uint64_t launches = 0;
    double ms = 0.0;
};

std::mutex g_mu;                                  // guards everything below
std::vector<Pending *> g_pending;                 // recorded, not yet read
std::vector<std::pair<int, cudaEvent_t>> g_pool;  // spare events, by device
std::map<std::string, Total> g_totals;

cudaEvent_t take_event_locked(int dev) {
    for (size_t i = g_pool.size(); i-- > 0;) {
        if (g_pool[i].first == dev) {
            const cudaEvent_t e = g_pool[i].second;
            g_pool.erase(g_pool.begin() + (ptrdiff_t)i);
            return e;
        }
    }
    cudaEvent_t e = nullptr;
    return cudaEventCreate(&e) == cudaSuccess ? e : nullptr;
}
void give_event_locked(int dev, cudaEvent_t e) {
    if (e) g_pool.emplace_back(dev, e);
}

}  // namespace

KernelSpan::KernelSpan(const char *kernel, cudaStream_t st) : st_(st) {
    if (!g_timing.load(std::memory_order_relaxed)) return;
    // A failed query here must not surface as the launch's own error, so the
    // error it leaves is cleared unless one was already pending.
    const bool clean = cudaPeekAtLastError() == cudaSuccess;
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(st, &cs) != cudaSuccess) {
        if (clean) cudaGetLastError();
        return;
    }
    if (cs != cudaStreamCaptureStatusNone) return;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        if (clean) cudaGetLastError();
        return;
    }
    Pending *p = new Pending{std::string(t_role) + ":" + kernel, dev, nullptr, nullptr};
    {
        std::lock_guard<std::mutex> lock(g_mu);
        p->e0 = take_event_locked(dev);
        p->e1 = take_event_locked(dev);
    }
    if (!p->e0 || !p->e1 || cudaEventRecord(p->e0, st) != cudaSuccess) {
        if (clean) cudaGetLastError();
        std::lock_guard<std::mutex> lock(g_mu);
        give_event_locked(dev, p->e0);
        give_event_locked(dev, p->e1);
        delete p;
        return;
    }
    slot_ = p;
}

KernelSpan::~KernelSpan() {
    if (!slot_) return;
    Pending *p = static_cast<Pending *>(slot_);
    const bool clean = cudaPeekAtLastError() == cudaSuccess;
    std::lock_guard<std::mutex> lock(g_mu);
    if (cudaEventRecord(p->e1, st_) != cudaSuccess) {
        if (clean) cudaGetLastError();
        give_event_locked(p->dev, p->e0);
        give_event_locked(p->dev, p->e1);
        delete p;
        return;
    }
    g_pending.push_back(p);
}

RoleScope::RoleScope(const char *role) : prev_(t_role) { t_role = role; }
RoleScope::~RoleScope() { t_role = prev_; }

}  // namespace mosaic

using namespace mosaic;

extern "C" {

int mosaic_kernel_timing(int enable) { return g_timing.exchange(enable ? 1 : 0); }

int mosaic_kernel_times(mosaic_kernel_time *out, int cap, int reset) {
    std::lock_guard<std::mutex> lock(g_mu);
    int cur = 0;
    cudaGetDevice(&cur);
    int rc = 0;
    for (Pending *p : g_pending) {
        float ms = 0.0f;
        if (cudaSetDevice(p->dev) != cudaSuccess || cudaEventSynchronize(p->e1) != cudaSuccess ||
            cudaEventElapsedTime(&ms, p->e0, p->e1) != cudaSuccess) {
            rc = -1;
        } else {
            Total &t = g_totals[p->key];
            t.launches += 1;
            t.ms += (double)ms;
        }
        give_event_locked(p->dev, p->e0);
        give_event_locked(p->dev, p->e1);
        delete p;
    }
    g_pending.clear();
    cudaSetDevice(cur);
    if (rc != 0) return rc;
    int n = 0;
    for (const auto &kv : g_totals) {
        if (out && n < cap) {
            memset(out[n].name, 0, sizeof out[n].name);
            strncpy(out[n].name, kv.first.c_str(), sizeof out[n].name - 1);
            out[n].launches = kv.second.launches;
            out[n].ms = kv.second.ms;
        }
        ++n;
    }
    if (reset) g_totals.clear();
    return n;
}

}  // extern "C"
