// Read-bandwidth probe for the benchmark's roofline denominators (a separate
// library, libpp_probe.so, not part of the planner): every thread streams
// 16-byte words of a buffer `iters` times.  With a buffer that fits in L2 the
// loop measures L2 read bandwidth, with one far larger than L2 it measures
// HBM read bandwidth.
#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>

#include "pp_probe.h"

namespace {

__global__ void __launch_bounds__(512) k_probe_read(const uint4 *__restrict__ p, size_t words, int iters,
                                                    unsigned long long *__restrict__ sink)
{
    uint32_t acc = 0;
    const size_t stride = (size_t)gridDim.x * blockDim.x;
    const size_t t0 = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
    for (int it = 0; it < iters; ++it) {
        size_t x = t0;
        // four independent loads in flight per thread
        for (; x + 3 * stride < words; x += 4 * stride) {
            const uint4 a = __ldcg(p + x), b = __ldcg(p + x + stride);
            const uint4 c = __ldcg(p + x + 2 * stride), d = __ldcg(p + x + 3 * stride);
            acc ^= a.x ^ a.y ^ a.z ^ a.w ^ b.x ^ b.y ^ b.z ^ b.w ^ c.x ^ c.y ^ c.z ^ c.w ^ d.x ^ d.y ^ d.z ^ d.w;
        }
        for (; x < words; x += stride) {
            const uint4 a = __ldcg(p + x);
            acc ^= a.x ^ a.y ^ a.z ^ a.w;
        }
    }
    if (acc == 0x9e3779b9u) atomicAdd(sink, 1ull);     // keeps the loads live
}

}  // namespace

extern "C" int pp_probe_read(const void *buf, size_t bytes, int32_t iters, uint64_t *sink, void *stream)
{
    if (!buf || !sink || iters < 0 || bytes % 16 || ((uintptr_t)buf & 15)) return 1;
    if (bytes == 0 || iters == 0) return 0;
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 2;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 2;
    k_probe_read<<<sms * 4, 512, 0, (cudaStream_t)stream>>>(reinterpret_cast<const uint4 *>(buf), bytes / 16,
                                                            iters, reinterpret_cast<unsigned long long *>(sink));
    return cudaGetLastError() == cudaSuccess ? 0 : 2;
}
