// noalloc.cu -- greedy vocabulary projection + argmax that allocates nothing.
//
// mnmt_linear_argmax needs a caller-provided buffer of packed keys, scratch
// the caller must allocate and zero.  Some callers cannot allocate device
// memory at all: a plugin whose host framework owns every byte of device
// memory through its own allocator (or a fixed memory budget), or code on a
// latency-critical thread where cudaMalloc's implicit device synchronisation
// is not acceptable.  mnmt_linear_argmax_ids_noalloc serves them: the keys
// live in the file-scope device array below, and the caller passes only the
// inputs and the int32 output ids.
#include <cuda_runtime.h>

#include <cstring>
#include <mutex>

#include "common.cuh"
#include "internal.h"

namespace {

// Maximum rows per call.  The array is 4096 x 8 = 32 KB of device memory that
// every GPU which loads this library holds until the process exits.
constexpr int NOALLOC_MAX_ROWS = 4096;
__device__ __align__(256) unsigned long long g_argmax_keys[NOALLOC_MAX_ROWS];

// In host code g_argmax_keys names a host-side stand-in, not device memory, so
// the kernels receive the array's device address, looked up once per device.
constexpr int MAX_DEVICES = 64;
std::mutex g_mu;
unsigned long long *g_keys_addr[MAX_DEVICES] = {nullptr};

__global__ void keys_to_ids(const unsigned long long *__restrict__ keys, int M, int32_t *__restrict__ ids) {
    int m = blockIdx.x * blockDim.x + threadIdx.x;
    if (m < M) ids[m] = (int32_t)key_index(keys[m]);
}

}  // namespace

extern "C" int mnmt_linear_argmax_ids_noalloc(const int8_t *A, const int8_t *W, const float *s_w,
                                              const float *bias, float s_x, int32_t M, int32_t N, int32_t K,
                                              int32_t *ids, void *cuda_stream) {
    if (!A || !W || !s_w || !bias || !ids || N < 1 || K < 16 || K % 16 || (M > 16 && K % 64) ||
        (M <= 16 && K > 2048))
        return mnmt::set_error(MNMT_EINVAL, "linear_argmax_ids_noalloc: bad pointer or shape");
    if (M < 1 || M > NOALLOC_MAX_ROWS)
        return mnmt::set_error(MNMT_EINVAL, "linear_argmax_ids_noalloc: M must be in [1, 4096] (fixed scratch)");
    if ((reinterpret_cast<uintptr_t>(A) | reinterpret_cast<uintptr_t>(W)) & 15)
        return mnmt::set_error(MNMT_EINVAL, "linear_argmax_ids_noalloc: A and W must be 16-byte aligned");
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= MAX_DEVICES)
        return mnmt::set_error(MNMT_ECUDA, "linear_argmax_ids_noalloc: no usable current device");
    unsigned long long *keys;
    {
        // first call on a device: look up the array's device address and opt
        // the GEMM kernels into their shared memory, with that device current
        std::lock_guard<std::mutex> lk(g_mu);
        if (!g_keys_addr[dev]) {
            void *p = nullptr;
            if (cudaGetSymbolAddress(&p, g_argmax_keys) != cudaSuccess || !p)
                return mnmt::set_error(MNMT_ECUDA, "linear_argmax_ids_noalloc: cudaGetSymbolAddress failed");
            if (mnmt::linear_init() != cudaSuccess)
                return mnmt::set_error(MNMT_ECUDA, "linear_argmax_ids_noalloc: kernel set-up failed");
            g_keys_addr[dev] = static_cast<unsigned long long *>(p);
        }
        keys = g_keys_addr[dev];
    }
    cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
    // the keys are combined with atomicMax: they must start at zero
    if (cudaMemsetAsync(keys, 0, (size_t)M * sizeof(unsigned long long), st) != cudaSuccess)
        return mnmt::set_error(MNMT_ECUDA, "linear_argmax_ids_noalloc: clearing the scratch failed");
    mnmt::Epi e;
    std::memset(&e, 0, sizeof(e));
    e.mode = mnmt::EPI_ARGMAX;
    e.s_x = s_x;
    e.s_w = s_w;
    e.bias = bias;
    e.keys = keys;
    if (mnmt::launch_linear(A, K, W, M, N, K, e, st) != cudaSuccess)
        return mnmt::set_error(MNMT_ECUDA, "linear_argmax_ids_noalloc: GEMM launch failed");
    keys_to_ids<<<(M + 255) / 256, 256, 0, st>>>(keys, M, ids);
    if (cudaGetLastError() != cudaSuccess)
        return mnmt::set_error(MNMT_ECUDA, "linear_argmax_ids_noalloc: key decode launch failed");
    return MNMT_OK;
}
