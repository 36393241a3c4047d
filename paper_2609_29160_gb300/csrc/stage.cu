// Stage-aware signal inputs (Sec. VIII: separate prefill and decode states;
// Sec. III-A ties prefill to time to first token and decode to time per output
// token). One pass over the request records gives, per record that the window
// reduction would keep:
//   - the +1/-1 window differences of the running gauge split at the first
//     token: prefill on [t_start, t_first), decode on [t_first, t_end);
//   - the packed calibration counts at the arrival window: arrivals and those
//     that met the TTFT bound (t_first - t_arr <= ttft[m]), and requests with
//     more than one output token and those that met the TPOT bound
//     ((t_end - t_first) <= tpot[m] * (L_out - 1), exact integer test).
// Counts pack as (count) + (met << 32) in one 64-bit word. All updates are
// integer atomics, so the result does not depend on record order.
#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace tre {
namespace {

constexpr int kThreads = 256;

__device__ __forceinline__ int64_t clamp_win(int64_t t, const FastDiv& fd, int K) {
  if (t < 0) return 0;
  const int64_t b = fd.div((uint32_t)t);
  return b > K ? K : b;
}

__global__ void __launch_bounds__(kThreads)
k_stage_requests(ReqCols r, int M, int win, FastDiv fd, int K, int32_t* __restrict__ dPre,
                 int32_t* __restrict__ dDec, unsigned long long* __restrict__ ttft,
                 unsigned long long* __restrict__ tpot, const int32_t* __restrict__ ttft_ms,
                 const int32_t* __restrict__ tpot_ms) {
  const int64_t span = (int64_t)K * win;
  for (int64_t i = (int64_t)blockIdx.x * kThreads + threadIdx.x; i < r.n;
       i += (int64_t)gridDim.x * kThreads) {
    const int m = r.model[i];
    const int64_t ta = r.t_arr[i], ts = r.t_start[i], tf = r.t_first[i], te = r.t_end[i];
    if (m < 0 || m >= M || ta < 0 || ta >= span) continue;
    const int32_t L_out = r.L_out[i];
    if (!(ta <= ts && ts <= tf && tf <= te) || r.L_in[i] < 0 || L_out < 1) continue;
    if (dPre) {
      const int64_t bs = clamp_win(ts, fd, K), bf = clamp_win(tf, fd, K),
                    be = clamp_win(te, fd, K);
      if (bs != bf) {
        atomicAdd(&dPre[bs * M + m], 1);
        atomicAdd(&dPre[bf * M + m], -1);
      }
      if (bf != be) {
        atomicAdd(&dDec[bf * M + m], 1);
        atomicAdd(&dDec[be * M + m], -1);
      }
    }
    if (ttft) {
      const size_t x = (size_t)fd.div((uint32_t)ta) * M + m;
      const unsigned long long met = (tf - ta <= (int64_t)ttft_ms[m]) ? 1ull : 0ull;
      atomicAdd(&ttft[x], 1ull + (met << 32));
      if (L_out >= 2) {
        const unsigned long long ok =
            (te - tf <= (int64_t)tpot_ms[m] * (int64_t)(L_out - 1)) ? 1ull : 0ull;
        atomicAdd(&tpot[x], 1ull + (ok << 32));
      }
    }
  }
}

template <class T> __global__ void k_fill(T* p, int64_t n, T v) {
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x)
    p[i] = v;
}

unsigned grid_of(int64_t n) {
  const int64_t b = (n + kThreads - 1) / kThreads;
  return (unsigned)std::max<int64_t>(1, std::min<int64_t>(b, (int64_t)device_sm_count() * 8));
}

}  // namespace

cudaError_t launch_stage_requests(const ReqCols& r, int M, int win, int K, int32_t* dPre,
                                  int32_t* dDec, unsigned long long* ttft,
                                  unsigned long long* tpot, const int32_t* ttft_ms,
                                  const int32_t* tpot_ms, cudaStream_t s) {
  const size_t cells1 = (size_t)(K + 1) * M, cells = (size_t)K * M;
  cudaError_t e = cudaSuccess;
  if (dPre) {
    if ((e = cudaMemsetAsync(dPre, 0, cells1 * sizeof(int32_t), s))) return e;
    if ((e = cudaMemsetAsync(dDec, 0, cells1 * sizeof(int32_t), s))) return e;
  }
  if (ttft) {
    if ((e = cudaMemsetAsync(ttft, 0, cells * sizeof(unsigned long long), s))) return e;
    if ((e = cudaMemsetAsync(tpot, 0, cells * sizeof(unsigned long long), s))) return e;
  }
  if (r.n == 0) return cudaSuccess;
  k_stage_requests<<<grid_of(r.n), kThreads, 0, s>>>(r, M, win, FastDiv(win), K, dPre, dDec,
                                                      ttft, tpot, ttft_ms, tpot_ms);
  return cudaGetLastError();
}

template <class T> cudaError_t launch_fill(T* p, int64_t n, T v, cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  k_fill<T><<<grid_of(n), kThreads, 0, s>>>(p, n, v);
  return cudaGetLastError();
}

template cudaError_t launch_fill<float>(float*, int64_t, float, cudaStream_t);
template cudaError_t launch_fill<double>(double*, int64_t, double, cudaStream_t);
template cudaError_t launch_fill<int32_t>(int32_t*, int64_t, int32_t, cudaStream_t);

}  // namespace tre
