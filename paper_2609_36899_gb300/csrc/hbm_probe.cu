// hbm_probe.cu -- diagnostics: a read-only HBM bandwidth probe (a measuring
// aid) and a self-test of the bounded-wait path.
//
// The probe streams `bytes` of device memory with 16-byte loads and folds them
// into one word per CTA, so the only DRAM traffic is the read.  The
// decode-attention kernel is a read-dominated stream; the probe gives the
// pure-read ceiling next to the copy (read + write) peak.
//
// The self-test runs, in one CTA, what every pipeline kernel does when a wait
// can never complete: it holds tensor memory, waits with the library's bounded
// wait on an mbarrier phase that nothing completes, records CADKV_ERR_TIMEOUT,
// raises the CTA's abort flag (the other warps, waiting on the same phase, see
// it and give up at once), frees the tensor memory and returns.  No fault, no
// hang: the wait ends after `limit_ns`.
#include "internal.h"
#include "ptx.cuh"

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

__global__ void __launch_bounds__(128) wait_selftest_kernel(WorkspaceHeader *hdr,
                                                             unsigned long long limit_ns)
{
    __shared__ uint64_t never_done;
    __shared__ uint32_t tmem_base;
    __shared__ int abort_flag;
    const int warp = threadIdx.x >> 5;
    if (threadIdx.x == 0) {
        mbar_init(&never_done, 1);  // nobody ever arrives
        abort_flag = 0;
        fence_mbarrier_init();
    }
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 32;" ::"r"(
                         smem_addr(&tmem_base))
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    volatile int *abort = &abort_flag;
    if (threadIdx.x == 0) {
        if (!mbar_wait_for(&never_done, 0, abort, limit_ns)) {
            *abort = 1;
            record_status(&hdr->status, CADKV_ERR_TIMEOUT);
        }
    } else {
        // the other warps wait on the same phase and leave on the abort flag
        const bool ok = mbar_wait_for(&never_done, 0, abort, 4 * limit_ns + 1000000);
        if (!ok && !*abort && (threadIdx.x & 31) == 0)
            record_status(&hdr->status, CADKV_ERR_TIMEOUT);
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (warp == 0) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 32;" ::"r"(tmem_base)
                     : "memory");
    }
}

}  // namespace

cudaError_t launch_wait_selftest(WorkspaceHeader *hdr, unsigned long long limit_ns,
                                 cudaStream_t stream)
{
    wait_selftest_kernel<<<1, 128, 0, stream>>>(hdr, limit_ns);
    return cudaGetLastError();
}

cudaError_t launch_hbm_read(const void *src, size_t bytes, unsigned long long *sink,
                            int num_sms, cudaStream_t stream)
{
    hbm_read_kernel<<<num_sms * 4, kProbeThreads, 0, stream>>>(
        static_cast<const uint4 *>(src), bytes / 16, sink);
    return cudaGetLastError();
}

}  // namespace cadkv
