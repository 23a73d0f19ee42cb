// ea_selftest.cu -- ea_selftest_bounded_wait: a check of the failure detection the staged server
// relies on.  Every wait of the server's producer and compute warps on an mbarrier is bounded:
// after its limit it gives up, the kernel records EA_E_TIMEOUT in a status word, and the host
// reads it (ea_sync_status).  Here one CTA waits, with the same mbar_wait and report_status, on an
// mbarrier that nothing arrives on (or, as the control, on one that completes first), so the
// limit runs out without any fault, trap or endless loop.
#include <cstdarg>
#include <cstdio>

#include "ea.h"
#include "ea_async.cuh"
#include "ea_internal.h"

namespace {

using namespace ea;

__device__ uint32_t g_selftest_status;

// One CTA of 32 threads; each thread waits on phase 0 of one mbarrier of arrival count 1.
__global__ void bounded_wait_kernel(long long limit_cycles, int arrive)
{
    __shared__ uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        mbar_init_fence();
    }
    __syncthreads();
    if (arrive && threadIdx.x == 0) mbar_arrive(&bar);
    __syncwarp();
    if (!mbar_wait(&bar, 0u, limit_cycles)) report_status(&g_selftest_status, kStatusTimeout);
}

int fail(int code, const char *fmt, ...)
{
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    set_last_error(buf);
    return code;
}

}  // namespace

extern "C" int ea_selftest_bounded_wait(int64_t limit_cycles, int32_t arrive, void *stream, int32_t *timed_out)
{
    if (timed_out == nullptr) return fail(EA_E_INVAL, "timed_out must not be NULL");
    if (limit_cycles < 1 || limit_cycles > kWaitLimitCycles)
        return fail(EA_E_INVAL, "limit_cycles must be in [1, %lld]", static_cast<long long>(kWaitLimitCycles));
    if (arrive != 0 && arrive != 1) return fail(EA_E_INVAL, "arrive is 0 or 1");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const uint32_t zero = 0;
    uint32_t status = 0;
    cudaError_t e = cudaMemcpyToSymbolAsync(g_selftest_status, &zero, sizeof zero, 0, cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess) {
        bounded_wait_kernel<<<1, 32, 0, s>>>(static_cast<long long>(limit_cycles), arrive);
        e = cudaGetLastError();
    }
    if (e == cudaSuccess)
        e = cudaMemcpyFromSymbolAsync(&status, g_selftest_status, sizeof status, 0, cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return fail(EA_E_CUDA, "bounded-wait self-test: %s", cudaGetErrorString(e));
    *timed_out = status == kStatusTimeout ? 1 : 0;
    return EA_OK;
}
