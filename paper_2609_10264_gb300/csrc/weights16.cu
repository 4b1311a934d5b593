// 16-bit weights (Sec. 7.2 quantises FP8 weights as round(2^8 W), which can
// need more than 8 bits): M = 256 M_hi + M_lo with M_lo the low byte read as
// a signed byte (in [-128, 127]) and M_hi = (w - M_lo) / 256, which is in
// [-128, 127] for w in [-32768, 32639] (w = 32640 .. 32767 would need 128).  The server runs its int8 products on
// the two planes and combines y = 256 y_hi + y_lo over F_q.
#include "common.cuh"
#include "launch.h"

namespace pv {
namespace {

__global__ void k_split_i16(const int16_t *__restrict__ W, size_t n, int8_t *__restrict__ hi,
                            int8_t *__restrict__ lo) {
    const size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= n) return;
    const int w = W[i];
    const int l = (int)(int8_t)(w & 0xff);  // w - l is a multiple of 256
    lo[i] = (int8_t)l;
    hi[i] = (int8_t)((w - l) >> 8);
}

__global__ void k_lift_i16(const int16_t *__restrict__ W, size_t n, uint32_t *__restrict__ out) {
    const size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= n) return;
    const int w = W[i];
    out[i] = w < 0 ? kQ - (uint32_t)(-w) : (uint32_t)w;
}

// y = 256 y + y_lo over F_q (y holds y_hi on entry).
__global__ void k_combine_256(uint32_t *__restrict__ y, const uint32_t *__restrict__ ylo, size_t n) {
    const size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= n) return;
    y[i] = fadd(fmul(y[i], 256u), ylo[i]);
}

}  // namespace

static unsigned grid_of(size_t n) { return (unsigned)((n + 255) / 256); }

cudaError_t launch_split_i16(const int16_t *W, size_t n, int8_t *hi, int8_t *lo, cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    if ((n + 255) / 256 > 0x7fffffffu) return cudaErrorInvalidValue;
    k_split_i16<<<grid_of(n), 256, 0, s>>>(W, n, hi, lo); note_launch();
    return cudaGetLastError();
}

cudaError_t launch_lift_i16(const int16_t *W, size_t n, uint32_t *out, cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    if ((n + 255) / 256 > 0x7fffffffu) return cudaErrorInvalidValue;
    k_lift_i16<<<grid_of(n), 256, 0, s>>>(W, n, out); note_launch();
    return cudaGetLastError();
}

cudaError_t launch_combine_256(uint32_t *y, const uint32_t *ylo, size_t n, cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    if ((n + 255) / 256 > 0x7fffffffu) return cudaErrorInvalidValue;
    k_combine_256<<<grid_of(n), 256, 0, s>>>(y, ylo, n); note_launch();
    return cudaGetLastError();
}

}  // namespace pv
