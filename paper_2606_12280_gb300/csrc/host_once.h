// host_once.h -- per-device, thread-safe one-time host set-up (internal).
//
// Launchers look up device properties and set kernel attributes once per
// device (the maximum dynamic shared memory, the resident blocks per SM, the
// registers ptxas gave a kernel).  Each result lives in a PerDevice slot that
// std::call_once fills, so host threads that launch at the same time never
// read a half-written value, and a process that drives several devices gets
// each device's own answer.
#pragma once

#include <mutex>
#include <cuda_runtime.h>

namespace w8a8 {

template <typename T>
struct PerDevice {
    static constexpr int kMaxDevices = 64;
    std::once_flag once[kMaxDevices];
    T value[kMaxDevices] = {};
    cudaError_t status[kMaxDevices] = {};

    // Runs f(T &) -> cudaError_t once for the current device, then returns
    // its status and (on success) the value in *out.
    template <typename F>
    cudaError_t get(F &&f, T *out) {
        int dev = 0;
        cudaError_t e = cudaGetDevice(&dev);
        if (e != cudaSuccess) return e;
        if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
        std::call_once(once[dev], [&] { status[dev] = f(value[dev]); });
        if (status[dev] != cudaSuccess) return status[dev];
        *out = value[dev];
        return cudaSuccess;
    }
};

// Number of SMs of the current device (cached per device).
inline int device_sms() {
    static PerDevice<int> sms;
    int n = 0;
    if (sms.get([](int &v) {
            int dev = 0;
            cudaError_t e = cudaGetDevice(&dev);
            if (e != cudaSuccess) return e;
            e = cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev);
            if (v <= 0) v = 1;
            return e;
        }, &n) != cudaSuccess)
        return 1;
    return n;
}

}  // namespace w8a8
