// Batched field product Y_hat[b] = M x_hat[b] over F_q.
#include "common.cuh"
#include "launch.h"

namespace pv {

cudaError_t launch_batched(const int8_t *W, int m, int K, const uint32_t *Xhat, int B,
                           uint32_t *Yhat, uint32_t *err, cudaStream_t s) {
    (void)err;
    for (int b = 0; b < B; ++b) {
        cudaError_t e = launch_gemv(W, m, K, Xhat + (size_t)b * K, Yhat + (size_t)b * m, s);
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

}  // namespace pv
