// Status strings, device checks and small shared host helpers of libgefen.
#include <mutex>

#include "internal.h"

namespace gefen {

int device_sm_count() {
    static std::mutex mu;
    static int cached[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 1;
    std::lock_guard<std::mutex> g(mu);
    if (cached[dev] == 0) {
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 1;
        cached[dev] = n;
    }
    return cached[dev];
}

gefen_status_t check_device() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return GEFEN_ECUDA;
    int major = 0, minor = 0;
    if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess)
        return GEFEN_ECUDA;
    return (major == 10 && minor == 3) ? GEFEN_OK : GEFEN_EUNSUPPORTED;
}

}  // namespace gefen

extern "C" const char* gefen_status_string(gefen_status_t s) {
    switch (s) {
        case GEFEN_OK: return "ok";
        case GEFEN_EINVAL: return "invalid argument";
        case GEFEN_ECUDA: return "CUDA error";
        case GEFEN_ENOMEM: return "workspace too small";
        case GEFEN_ETIMEOUT: return "device wait timed out";
        case GEFEN_EUNSUPPORTED: return "unsupported device or size";
        case GEFEN_EDEVICE: return "device-side data check failed";
    }
    return "unknown status";
}

extern "C" gefen_status_t gefen_sync_status(gefen_stream_t stream) {
    cudaError_t e = cudaStreamSynchronize(reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return GEFEN_ECUDA;
    e = cudaGetLastError();
    return e == cudaSuccess ? GEFEN_OK : GEFEN_ECUDA;
}
