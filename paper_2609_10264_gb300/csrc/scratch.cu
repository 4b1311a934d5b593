// Host-side state kept per device.
//
// Grow-only device scratch held per (purpose, device, stream).
//
// The batched product's digit tiles and the small-batch product's digit
// planes live in library-owned buffers.  Keying them by stream lets calls on
// different streams overlap without sharing a buffer; calls on one stream
// are ordered, so they may share one.  A buffer that must grow is replaced
// after the stream has drained (the old one may still be read), which is
// not allowed while the stream is being captured: make one call of the
// largest shape before capturing.
#include <map>
#include <mutex>
#include <tuple>

#include "launch.h"

namespace pv {

cudaError_t stream_scratch(int purpose, size_t need, cudaStream_t s, void **out) {
    struct Buf {
        void *ptr = nullptr;
        size_t bytes = 0;
    };
    static std::mutex mu;
    static std::map<std::tuple<int, int, cudaStream_t>, Buf> bufs;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lock(mu);
    Buf &b = bufs[std::make_tuple(purpose, dev, s)];
    if (b.bytes < need) {
        if (b.ptr) {
            if ((e = cudaStreamSynchronize(s)) != cudaSuccess) return e;
            cudaFree(b.ptr);
            b.ptr = nullptr;
            b.bytes = 0;
        }
        if ((e = cudaMalloc(&b.ptr, need)) != cudaSuccess) return e;
        b.bytes = need;
    }
    *out = b.ptr;
    return cudaSuccess;
}

cudaError_t func_attr(const void *fn, cudaFuncAttribute attr, int value) {
    static std::mutex mu;
    static std::map<std::tuple<const void *, int, int>, std::pair<int, cudaError_t>> done;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lock(mu);
    auto key = std::make_tuple(fn, (int)attr, dev);
    auto it = done.find(key);
    if (it != done.end() && it->second.first == value) return it->second.second;
    e = cudaFuncSetAttribute(fn, attr, value);
    done[key] = std::make_pair(value, e);
    return e;
}

}  // namespace pv
