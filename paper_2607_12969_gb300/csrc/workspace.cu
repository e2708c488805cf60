// workspace.cu -- device workspace of the split-phase apply: one buffer per
// (device, stream), allocated on first use and grown when a larger problem
// arrives.  Growing waits for the stream (work already queued may still use
// the old buffer) before the old buffer is freed.  Calls on different
// streams get different buffers, so they may run concurrently; calls on one
// stream are ordered by the stream.  lrc_shutdown() frees every buffer.
//
// Beside it each (device, stream) has a small buffer of arrival counters for
// kernels whose last CTA finishes a reduction: zeroed once when it is made
// (in stream order), and left at zero by every kernel that uses it; and a
// result slot in mapped pinned host memory, which the finishing kernel of a
// scalar reduction writes directly (the host reads it after the stream has
// synchronised), so a scalar result never queues behind bulk copies on the
// copy engines.
#include <map>
#include <mutex>
#include <utility>

#include "common.cuh"

namespace lrc {

namespace {

struct Buf {
    void* ptr = nullptr;
    size_t bytes = 0;
};

std::mutex g_ws_mu;
std::map<std::pair<int, cudaStream_t>, Buf> g_ws;
std::map<std::pair<int, cudaStream_t>, Buf> g_cnt;
struct Slot {
    double* host = nullptr;
    double* dev = nullptr;
};
std::map<std::pair<int, cudaStream_t>, Slot> g_slot;

}  // namespace

lrc_status stream_workspace(cudaStream_t s, size_t bytes, void** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    std::lock_guard<std::mutex> lock(g_ws_mu);
    Buf& b = g_ws[std::make_pair(dev, s)];
    if (b.bytes < bytes) {
        if (b.ptr) {
            e = cudaStreamSynchronize(s);
            if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize (workspace growth)");
            cudaFree(b.ptr);
            b.ptr = nullptr;
            b.bytes = 0;
        }
        const size_t want = (bytes + ((size_t)1 << 20) - 1) & ~(((size_t)1 << 20) - 1);   // whole MiB
        e = cudaMalloc(&b.ptr, want);
        if (e != cudaSuccess) {
            b.ptr = nullptr;
            cudaGetLastError();
            set_error("workspace allocation of %zu bytes failed: %s", want, cudaGetErrorString(e));
            return LRC_ERR_NOMEM;
        }
        b.bytes = want;
    }
    *out = b.ptr;
    return LRC_OK;
}

lrc_status stream_counters(cudaStream_t s, unsigned int** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    std::lock_guard<std::mutex> lock(g_ws_mu);
    Buf& b = g_cnt[std::make_pair(dev, s)];
    if (!b.ptr) {
        const size_t bytes = sizeof(unsigned int) * kStreamCounters;
        e = cudaMalloc(&b.ptr, bytes);
        if (e != cudaSuccess) {
            b.ptr = nullptr;
            cudaGetLastError();
            set_error("counter allocation failed: %s", cudaGetErrorString(e));
            return LRC_ERR_NOMEM;
        }
        e = cudaMemsetAsync(b.ptr, 0, bytes, s);
        if (e != cudaSuccess) {
            cudaFree(b.ptr);
            b.ptr = nullptr;
            return cuda_fail(e, "cudaMemsetAsync (counters)");
        }
        b.bytes = bytes;
    }
    *out = static_cast<unsigned int*>(b.ptr);
    return LRC_OK;
}

lrc_status stream_result_slot(cudaStream_t s, double** host, double** dev) {
    int d = 0;
    cudaError_t e = cudaGetDevice(&d);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    std::lock_guard<std::mutex> lock(g_ws_mu);
    Slot& sl = g_slot[std::make_pair(d, s)];
    if (!sl.host) {
        void* h = nullptr;
        e = cudaHostAlloc(&h, sizeof(double) * kResultSlots, cudaHostAllocMapped);
        if (e != cudaSuccess) {
            cudaGetLastError();
            set_error("result slot allocation failed: %s", cudaGetErrorString(e));
            return LRC_ERR_NOMEM;
        }
        void* dp = nullptr;
        e = cudaHostGetDevicePointer(&dp, h, 0);
        if (e != cudaSuccess) {
            cudaFreeHost(h);
            return cuda_fail(e, "cudaHostGetDevicePointer (result slot)");
        }
        sl.host = static_cast<double*>(h);
        sl.dev = static_cast<double*>(dp);
    }
    *host = sl.host;
    *dev = sl.dev;
    return LRC_OK;
}

void release_workspaces() {
    std::lock_guard<std::mutex> lock(g_ws_mu);
    int prev = -1;
    cudaGetDevice(&prev);
    for (auto* m : {&g_ws, &g_cnt}) {
        for (auto& kv : *m) {
            if (kv.second.ptr) {
                cudaSetDevice(kv.first.first);
                cudaFree(kv.second.ptr);
            }
        }
        m->clear();
    }
    for (auto& kv : g_slot)
        if (kv.second.host) cudaFreeHost(kv.second.host);
    g_slot.clear();
    if (prev >= 0) cudaSetDevice(prev);
}

}  // namespace lrc
