// Test helper (not part of libpdb): a kernel that keeps thread blocks busy
// for a bounded time, so that another kernel launched on a second stream
// finds only part of the device free.  Each block asks for the largest
// dynamic shared memory a block may have, so no other block fits beside it
// on its SM; it sleeps in steps of 1 us until the global timer has advanced
// by `ns` (at most one second) and returns.
#include <cuda_runtime.h>
#include <stdint.h>

__global__ void k_hold(unsigned long long ns)
{
    extern __shared__ unsigned char smem[];
    unsigned long long t0, t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t0));
    do {
        __nanosleep(1000);
        asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    } while (t - t0 < ns);
    if (threadIdx.x == 0) smem[0] = 0;
}

extern "C" int hold_sms(int blocks, double seconds, void *stream)
{
    if (blocks < 1 || !(seconds > 0.0)) return -1;
    if (seconds > 1.0) seconds = 1.0;
    int dev = 0, smem = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return -2;
    if (cudaDeviceGetAttribute(&smem, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess) return -2;
    if (cudaFuncSetAttribute(k_hold, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess) return -2;
    k_hold<<<blocks, 32, smem, (cudaStream_t)stream>>>((unsigned long long)(seconds * 1e9));
    return cudaGetLastError() == cudaSuccess ? 0 : -3;
}
