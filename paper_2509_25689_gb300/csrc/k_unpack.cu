// Device dequantizer: packed tensor -> fp32, one thread per weight.
// Used for checking the packed-format decode on the GPU bit-for-bit
// against the host decode (every weight is exact up to one rounding).
#include "mq_internal.h"

namespace mq {
namespace {

__global__ void unpack_kernel(int fmt, const uint8_t* __restrict__ src, int64_t rows, int64_t cols,
                              float* __restrict__ dst) {
    const TensorLayout L = tensor_layout(fmt, rows, cols);
    const int64_t n = rows * cols;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        dst[i] = dequant_at(fmt, src, L, i / cols, i % cols);
}

}  // namespace

cudaError_t launch_unpack(int fmt, const uint8_t* src, int64_t rows, int64_t cols, float* dst, cudaStream_t s) {
    const int64_t n = rows * cols;
    if (n == 0) return cudaSuccess;
    int64_t blocks = (n + 255) / 256;
    if (blocks > 152 * 64) blocks = 152 * 64;
    prof_begin("unpack", s);
    unpack_kernel<<<(unsigned)blocks, 256, 0, s>>>(fmt, src, rows, cols, dst);
    prof_end(s);
    return cudaGetLastError();
}

}  // namespace mq
