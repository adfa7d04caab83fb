// hbm_probe.cu -- read-only HBM bandwidth probe (a measuring aid).
//
// Streams `bytes` of device memory with 16-byte loads and folds them into one
// word per CTA, so the only DRAM traffic is the read.  The decode-attention
// kernel is a read-dominated stream; this kernel gives the pure-read ceiling
// next to the copy (read + write) peak.
#include "internal.h"

namespace cadkv {

namespace {

constexpr int kProbeThreads = 512;
constexpr int kProbeUnroll = 8;

__global__ void __launch_bounds__(kProbeThreads) hbm_read_kernel(const uint4 *__restrict__ src,
                                                                size_t n_vec,
                                                                unsigned long long *sink)
{
    uint32_t acc = 0;
    const size_t stride = (size_t)gridDim.x * kProbeThreads;
    size_t i = (size_t)blockIdx.x * kProbeThreads + threadIdx.x;
    for (; i + (kProbeUnroll - 1) * stride < n_vec; i += kProbeUnroll * stride) {
        uint4 v[kProbeUnroll];
#pragma unroll
        for (int u = 0; u < kProbeUnroll; ++u)
            v[u] = __ldcs(src + i + u * stride);
#pragma unroll
        for (int u = 0; u < kProbeUnroll; ++u)
            acc ^= v[u].x ^ v[u].y ^ v[u].z ^ v[u].w;
    }
    for (; i < n_vec; i += stride) {
        const uint4 v = __ldcs(src + i);
        acc ^= v.x ^ v.y ^ v.z ^ v.w;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
        acc ^= __shfl_xor_sync(0xffffffffu, acc, o);
    if ((threadIdx.x & 31) == 0)
        atomicXor(sink, (unsigned long long)acc);
}

}  // namespace

cudaError_t launch_hbm_read(const void *src, size_t bytes, unsigned long long *sink,
                            int num_sms, cudaStream_t stream)
{
    hbm_read_kernel<<<num_sms * 4, kProbeThreads, 0, stream>>>(
        static_cast<const uint4 *>(src), bytes / 16, sink);
    return cudaGetLastError();
}

}  // namespace cadkv
