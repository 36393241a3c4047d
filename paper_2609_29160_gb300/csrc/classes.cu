// Per-(model, SLO class) TSS from per-request classes. The paper gives each
// model one SLO class (Sec. II-A); with a class per request the signal is kept
// per (model, class) pair by treating every pair as a model of its own: record
// i's model becomes model[i] * n_classes + cls[i]. The reduction, scoring,
// calibration (one TTFT bound per pair) and selection then run unchanged over
// n_models * n_classes models.
#include <algorithm>

#include "internal.h"

namespace tre {
namespace {

__global__ void __launch_bounds__(256)
k_class_models(int64_t n, const int32_t* model, const int32_t* __restrict__ cls, int32_t M,
               int32_t C, int32_t* out) {
  for (int64_t i = (int64_t)blockIdx.x * 256 + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * 256) {
    const int32_t m = model[i], c = cls[i];
    // an id outside the grid stays outside it, so the reduction counts it
    out[i] = (m >= 0 && m < M && c >= 0 && c < C) ? m * C + c : -1;
  }
}

}  // namespace
}  // namespace tre

extern "C" tre_status tss_class_models(int64_t n, const int32_t* model, const int32_t* cls,
                                       int32_t n_models, int32_t n_classes, int32_t* model_out,
                                       tre_stream stream) {
  if (n < 0 || n_models < 1 || n_classes < 1 || (int64_t)n_models * n_classes > 1024)
    return TRE_EINVAL;
  if (n == 0) return TRE_OK;
  if (!model || !cls || !model_out) return TRE_EINVAL;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int64_t blocks = std::min<int64_t>((n + 255) / 256, 152 * 32);
  tre::k_class_models<<<(unsigned)blocks, 256, 0, s>>>(n, model, cls, n_models, n_classes,
                                                      model_out);
  return cudaGetLastError() == cudaSuccess ? TRE_OK : TRE_ECUDA;
}
