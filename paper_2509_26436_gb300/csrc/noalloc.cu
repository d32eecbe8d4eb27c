// quartz_linear_noalloc: the W4A4 linear layer for callers that cannot
// allocate device memory.
//
// quartz_linear needs a scratch workspace (the operands expanded to tensor-core
// input plus transposed group scales) that its caller allocates.  Some callers
// cannot do that: a plugin running inside a host framework that owns all
// device memory through its own pool and forbids side allocations, or code on
// a latency-critical path where a cudaMalloc could synchronise the device.
// This entry point instead uses one scratch array that is part of the library
// image (a file-scope __device__ array), so it allocates nothing at call time.
//
// Properties a caller must know:
//   - The array holds QUARTZ_NOALLOC_SCRATCH_BYTES (32 MiB) on every GPU that loads
//     the library, for the lifetime of the process.  Problems whose workspace
//     (quartz_linear_workspace_size) exceeds that are rejected with
//     QUARTZ_ERR_WORKSPACE before anything is launched.
//   - The first call on a device looks up the device address of the array
//     (cudaGetSymbolAddress) with that device current; make that first call
//     before any stream capture.
//   - Every call on a device shares the same array and it keeps the previous
//     call's contents.  Calls that overlap on the GPU (different streams, no
//     ordering between them) race on it and give wrong results; serialise them.
//   - Nothing in the array needs to start at zero: each call rewrites every
//     byte it reads.
#include <mutex>

#include "quartz_internal.h"

namespace quartz {
namespace {

constexpr size_t kNoallocScratchBytes = QUARTZ_NOALLOC_SCRATCH_BYTES;
constexpr int kMaxDevices = 64;

__device__ __align__(256) unsigned char g_noalloc_scratch[kNoallocScratchBytes];

std::mutex g_noalloc_mutex;
void *g_noalloc_ptr[kMaxDevices] = {};

// Device address of the scratch array on the current device (looked up once
// per device; the host-side symbol itself is not a device address).
void *noalloc_scratch()
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
    std::lock_guard<std::mutex> lock(g_noalloc_mutex);
    if (!g_noalloc_ptr[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess) return nullptr;
        g_noalloc_ptr[dev] = p;
    }
    return g_noalloc_ptr[dev];
}

}  // namespace
}  // namespace quartz

using namespace quartz;

extern "C" int32_t quartz_linear_noalloc(const quartz_encoded_t *a, const quartz_encoded_t *w,
                                         const void *bias_f16, void *y, int32_t y_type,
                                         void *stream)
{
    // Reject problems whose workspace does not fit the array before anything
    // is launched; quartz_linear then validates every other argument.
    if (!a || !w) return QUARTZ_ERR_INVALID_ARG;
    const size_t need = quartz_linear_workspace_size(a->rows, w->rows, a->K, &a->p);
    if (a->rows > 0 && need == 0) return QUARTZ_ERR_INVALID_ARG;
    if (need > kNoallocScratchBytes) return QUARTZ_ERR_WORKSPACE;
    void *scratch = noalloc_scratch();
    if (!scratch) return QUARTZ_ERR_CUDA;
    return quartz_linear(a, w, bias_f16, y, y_type, scratch, kNoallocScratchBytes, stream);
}
