// The host<->device copies of a decode step (qx_decode_step*) as one small
// kernel per direction instead of one DMA copy per buffer.  A decode step
// moves tens of KB each way (x in, y out); at that size a copy engine's
// start-up, not the bytes, sets the time, while the SMs read and write pinned
// host memory directly through its mapped device address.  The kernel is
// launched with programmatic dependent launch where that is safe: the copy
// out waits (griddepcontrol.wait) for the matmuls that write y, and both let
// the next kernel in the stream start its set-up early.
#include "qx_kernels.cuh"

namespace qx {

namespace {

__global__ void __launch_bounds__(256) copy_kernel(const __grid_constant__ CopyList c) {
    // the previous kernel in the stream (under PDL) has finished and its
    // writes are visible; a no-op without PDL
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t nthreads = (int64_t)gridDim.x * blockDim.x;
    for (int i = 0; i < c.n; ++i) {
        const uint8_t *src = c.src[i];
        uint8_t *dst = c.dst[i];
        const int64_t bytes = c.bytes[i];
        if ((((uintptr_t)src | (uintptr_t)dst | (uintptr_t)bytes) & 15u) == 0) {
            const uint4 *s4 = reinterpret_cast<const uint4 *>(src);
            uint4 *d4 = reinterpret_cast<uint4 *>(dst);
            for (int64_t j = tid; j < bytes / 16; j += nthreads) d4[j] = s4[j];
        } else {
            for (int64_t j = tid; j < bytes; j += nthreads) dst[j] = src[j];
        }
    }
}

}  // namespace

cudaError_t launch_copies(const CopyList &c, int num_sms, bool pdl, cudaStream_t st) {
    if (c.n < 1 || c.n > kMaxCopies) return cudaErrorInvalidValue;
    int64_t total = 0;
    for (int i = 0; i < c.n; ++i) total += c.bytes[i];
    const int64_t blocks = std::max<int64_t>(1, std::min<int64_t>((total / 16 + 255) / 256, num_sms));
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)blocks);
    cfg.blockDim = dim3(256);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, copy_kernel, c);
}

}  // namespace qx
