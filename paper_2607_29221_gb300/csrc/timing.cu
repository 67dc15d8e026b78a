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

// ---------------------------------------------------------------------------
// Integer ALU rate of the ChaCha20 mix (add, xor, rotate), for the draws'
// roofline: every thread runs the 8 quarter rounds of a double round on 16
// independent words, enough warps to fill every SM.
// ---------------------------------------------------------------------------
namespace mosaic {
namespace {

constexpr int kMixThreads = 256;
constexpr int kMixBlocksPerSm = 8;
constexpr int kMixIters = 2000;

__global__ void __launch_bounds__(kMixThreads) int_mix_kernel(uint32_t *out, int iters) {
    uint32_t x0 = threadIdx.x, x1 = blockIdx.x, x2 = 2, x3 = 3, x4 = 4, x5 = 5, x6 = 6, x7 = 7;
    uint32_t x8 = 8, x9 = 9, x10 = 10, x11 = 11, x12 = 12, x13 = 13, x14 = 14, x15 = 15;
    for (int it = 0; it < iters; ++it) {
        MOSAIC_QR(x0, x4, x8, x12);
        MOSAIC_QR(x1, x5, x9, x13);
        MOSAIC_QR(x2, x6, x10, x14);
        MOSAIC_QR(x3, x7, x11, x15);
        MOSAIC_QR(x0, x5, x10, x15);
        MOSAIC_QR(x1, x6, x11, x12);
        MOSAIC_QR(x2, x7, x8, x13);
        MOSAIC_QR(x3, x4, x9, x14);
    }
    out[(size_t)blockIdx.x * blockDim.x + threadIdx.x] =
        x0 ^ x1 ^ x2 ^ x3 ^ x4 ^ x5 ^ x6 ^ x7 ^ x8 ^ x9 ^ x10 ^ x11 ^ x12 ^ x13 ^ x14 ^ x15;
}

}  // namespace
}  // namespace mosaic

extern "C" mosaic_status mosaic_int_mix_rate(uint32_t *scratch, size_t scratch_bytes, double *ops_per_second,
                                             void *stream) {
    if (!ops_per_second) return MOSAIC_ERR_ARG;
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms < 1)
        return MOSAIC_ERR_CUDA;
    const int blocks = sms * kMixBlocksPerSm;
    if (!scratch || scratch_bytes < (size_t)blocks * kMixThreads * sizeof(uint32_t)) return MOSAIC_ERR_WORKSPACE;
    cudaStream_t st = as_stream(stream);
    cudaEvent_t e0 = nullptr, e1 = nullptr;
    if (cudaEventCreate(&e0) != cudaSuccess || cudaEventCreate(&e1) != cudaSuccess) {
        if (e0) cudaEventDestroy(e0);
        return MOSAIC_ERR_CUDA;
    }
    int_mix_kernel<<<blocks, kMixThreads, 0, st>>>(scratch, 8);   // warm-up
    cudaEventRecord(e0, st);
    int_mix_kernel<<<blocks, kMixThreads, 0, st>>>(scratch, kMixIters);
    cudaEventRecord(e1, st);
    float ms = 0.0f;
    const bool ok = cudaEventSynchronize(e1) == cudaSuccess && cudaEventElapsedTime(&ms, e0, e1) == cudaSuccess &&
                    cudaGetLastError() == cudaSuccess && ms > 0.0f;
    cudaEventDestroy(e0);
    cudaEventDestroy(e1);
    if (!ok) return MOSAIC_ERR_CUDA;
    // 8 quarter rounds of 12 add / xor / rotate per iteration and thread.
    *ops_per_second = (double)blocks * kMixThreads * kMixIters * 8.0 * 12.0 / ((double)ms * 1e-3);
    return MOSAIC_OK;
}

// ---------------------------------------------------------------------------
// Shared-memory read rate of the tiled gather's access: each group of 8 lanes
// reads one whole 128-byte line with 16-byte loads, the four groups of a warp
// four lines at scattered positions (conflict-free phases), for the gathers'
// roofline.  Volatile loads, so that none is merged or dropped.
// ---------------------------------------------------------------------------
namespace mosaic {
namespace {

constexpr int kSmemThreads = 512;
constexpr int kSmemWords = 16384;   // 64 KB = 512 lines per block
constexpr int kSmemIters = 4000;

__global__ void __launch_bounds__(kSmemThreads) smem_read_kernel(uint32_t *out, int iters) {
    extern __shared__ __align__(16) uint32_t buf[];
    for (int i = threadIdx.x; i < kSmemWords; i += blockDim.x) buf[i] = (uint32_t)i * 2654435761u;
    __syncthreads();
    const uint32_t base = (uint32_t)__cvta_generic_to_shared(buf);
    // Line of group (thread / 8) for load k: a hash of the group and k; the
    // iteration moves every line by 37 (mod 512), so no two loads of a thread
    // read the same line.
    uint32_t line[8];
    uint32_t h = (threadIdx.x >> 3) * 2654435761u + 0x9e3779b9u;
#pragma unroll
    for (int k = 0; k < 8; ++k) {
        h ^= h >> 13;
        h *= 0x5bd1e995u;
        h ^= h >> 15;
        line[k] = (h & ~63u) | (uint32_t)(k * 64);
    }
    const uint32_t chunk = (threadIdx.x & 7) * 16u;
    uint32_t a0 = 0, a1 = 0, a2 = 0, a3 = 0;
    for (int it = 0; it < iters; ++it) {
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const uint32_t addr = base + ((line[k] + (uint32_t)it * 37u) & 511u) * 128u + chunk;
            uint32_t v0, v1, v2, v3;
            asm volatile("ld.volatile.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                         : "=r"(v0), "=r"(v1), "=r"(v2), "=r"(v3)
                         : "r"(addr));
            a0 ^= v0; a1 ^= v1; a2 ^= v2; a3 ^= v3;
        }
    }
    out[(size_t)blockIdx.x * blockDim.x + threadIdx.x] = a0 ^ a1 ^ a2 ^ a3;
}

}  // namespace
}  // namespace mosaic

extern "C" mosaic_status mosaic_smem_read_rate(uint32_t *scratch, size_t scratch_bytes, double *bytes_per_second,
                                               void *stream) {
    if (!bytes_per_second) return MOSAIC_ERR_ARG;
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms < 1)
        return MOSAIC_ERR_CUDA;
    const int blocks = sms * 2;
    if (!scratch || scratch_bytes < (size_t)blocks * kSmemThreads * sizeof(uint32_t)) return MOSAIC_ERR_WORKSPACE;
    cudaStream_t st = as_stream(stream);
    cudaEvent_t e0 = nullptr, e1 = nullptr;
    if (cudaEventCreate(&e0) != cudaSuccess || cudaEventCreate(&e1) != cudaSuccess) {
        if (e0) cudaEventDestroy(e0);
        return MOSAIC_ERR_CUDA;
    }
    const size_t smem = (size_t)kSmemWords * 4;
    if (cudaFuncSetAttribute(smem_read_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
        cudaSuccess) {
        cudaEventDestroy(e0);
        cudaEventDestroy(e1);
        return MOSAIC_ERR_CUDA;
    }
    smem_read_kernel<<<blocks, kSmemThreads, smem, st>>>(scratch, 8);   // warm-up
    cudaEventRecord(e0, st);
    smem_read_kernel<<<blocks, kSmemThreads, smem, st>>>(scratch, kSmemIters);
    cudaEventRecord(e1, st);
    float ms = 0.0f;
    const bool ok = cudaEventSynchronize(e1) == cudaSuccess && cudaEventElapsedTime(&ms, e0, e1) == cudaSuccess &&
                    cudaGetLastError() == cudaSuccess && ms > 0.0f;
    cudaEventDestroy(e0);
    cudaEventDestroy(e1);
    if (!ok) return MOSAIC_ERR_CUDA;
    *bytes_per_second = (double)blocks * kSmemThreads * kSmemIters * 8.0 * 16.0 / ((double)ms * 1e-3);
    return MOSAIC_OK;
}
