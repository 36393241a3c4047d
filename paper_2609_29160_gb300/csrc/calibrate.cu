// Calibration of the healthy boundary theta (Sec. III-B: the lowest smoothed TSS
// value at which the SLO reliability target is still met).
//
// For model m, let the calibration windows be those with at least one arrival,
// not idle, S > 0. For a value s let C(s) be the number of calibration windows
// with S >= s and H(s) the healthy ones among them. theta is the smallest S
// value s with H(s) >= reliability * C(s).
//
// Instead of sorting, each model's (S, healthy) pairs are packed into unsigned
// keys (the bit pattern of a positive float orders like the float) and theta is
// found by a radix descent over 8-bit digits: at each level a histogram of
// counts, healthy counts and the smallest key per bucket; buckets are visited
// from the smallest values up. A bucket whose smallest value already satisfies
// the condition gives theta (nothing below it did). A bucket that could contain
// a qualifying value -- the bound that adds only its healthy windows passes --
// is refined one digit further; if the refinement finds nothing the scan
// resumes above it. All counts are exact integers and every comparison is the
// same double expression the definition uses, so theta is exact.
#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace tre {
namespace {

constexpr int kThrTable = 4096;
constexpr int kSearchThreads = 1024;

template <class T> struct KeyOf;
template <> struct KeyOf<float> {
  using U = uint32_t;
  static constexpr int kBits = 31;  // key bits of a non-negative float
};
template <> struct KeyOf<double> {
  using U = unsigned long long;
  static constexpr int kBits = 63;
};

// thr[a] = smallest integer n with (double)n >= ok_frac * (double)a
__global__ void k_thr(double ok_frac, int32_t* thr) {
  const int a = blockIdx.x * blockDim.x + threadIdx.x;
  if (a >= kThrTable) return;
  const double v = ok_frac * (double)a;
  int32_t t;
  if (!(v <= 2147483647.0)) t = 0x7fffffff;           // unreachable (or NaN)
  else if (v <= -2147483647.0) t = -0x7fffffff;
  else t = (int32_t)ceil(v);
  thr[a] = t;
}

__device__ __forceinline__ bool healthy(uint32_t n_arr, uint32_t n_met, const int32_t* thr,
                                        double ok_frac) {
  if (n_arr < (uint32_t)kThrTable) return (int64_t)n_met >= (int64_t)thr[n_arr];
  return (double)n_met >= ok_frac * (double)n_arr;
}

// [K][M] S, cls, packed SLO counts -> [M][K] packed keys (0 = not a calibration window)
template <class T>
__global__ void k_pack(int M, int K, const T* __restrict__ S, const uint8_t* __restrict__ cls,
                       const unsigned long long* __restrict__ slo, const int32_t* __restrict__ thr,
                       double ok_frac, typename KeyOf<T>::U* __restrict__ keys) {
  using U = typename KeyOf<T>::U;
  __shared__ U tile[32][33];
  const int k0 = blockIdx.x * 32, m0 = blockIdx.y * 32;
  for (int j = threadIdx.y; j < 32; j += blockDim.y) {
    const int k = k0 + j, m = m0 + threadIdx.x;
    U v = 0;
    if (k < K && m < M) {
      const size_t x = (size_t)k * M + m;
      const unsigned long long c = slo[x];
      const uint32_t n_arr = (uint32_t)c, n_met = (uint32_t)(c >> 32);
      const T s = S[x];
      if (cls[x] != kIdle && n_arr >= 1 && s > (T)0)
        v = ((U)key_of(s) << 1) | (U)(healthy(n_arr, n_met, thr, ok_frac) ? 1 : 0);
    }
    tile[j][threadIdx.x] = v;
  }
  __syncthreads();
  for (int j = threadIdx.y; j < 32; j += blockDim.y) {
    const int m = m0 + j, k = k0 + threadIdx.x;
    if (m < M && k < K) keys[(size_t)m * K + k] = tile[threadIdx.x][j];
  }
}

template <class T>
__global__ void __launch_bounds__(kSearchThreads)
k_search(int M, int K, const typename KeyOf<T>::U* __restrict__ keys, double reliability,
         T* theta, tre_diag* diag) {
  using U = typename KeyOf<T>::U;
  constexpr int NB = 256;
  constexpr int NL = (KeyOf<T>::kBits + 7) / 8;
  __shared__ int32_t cnt[NL][NB], hl[NL][NB];
  __shared__ int64_t tot_c[NL], tot_h[NL];
  __shared__ U mn[NL][NB];
  __shared__ int64_t cab[NL], hab[NL];
  __shared__ U prefix[NL];
  __shared__ int pos[NL];
  __shared__ int level, action, act_b;
  __shared__ U max_key;
  __shared__ U result;
  const int m = blockIdx.x;
  const U* mk = keys + (size_t)m * K;

  auto lo_bit = [](int l) { return max(0, KeyOf<T>::kBits - 8 * (l + 1)); };
  auto build = [&](int l) {
    for (int b = threadIdx.x; b < NB; b += blockDim.x) {
      cnt[l][b] = 0;
      hl[l][b] = 0;
      mn[l][b] = ~(U)0;
    }
    __syncthreads();
    const int lo = lo_bit(l);
    const int hi = KeyOf<T>::kBits - 8 * l;   // bits [lo, hi) are this level's digit
    const U pre = prefix[l];
    U local_max = 0;
    for (int64_t i = threadIdx.x; i < K; i += blockDim.x) {
      const U p = mk[i];
      if (!p) continue;
      const U key = p >> 1;
      if (l == 0) local_max = key > local_max ? key : local_max;
      if (hi < KeyOf<T>::kBits && (key >> hi) != pre) continue;
      const int b = (int)((key >> lo) & (U)(NB - 1));
      atomicAdd(&cnt[l][b], 1);
      if (p & 1) atomicAdd(&hl[l][b], 1);
      atomicMin(&mn[l][b], key);
    }
    if (l == 0 && local_max) atomicMax(&max_key, local_max);
    __syncthreads();
    if (threadIdx.x == 0) {
      int64_t tc = 0, th = 0;
      for (int b = 0; b < NB; ++b) {
        tc += cnt[l][b];
        th += hl[l][b];
      }
      tot_c[l] = tc;
      tot_h[l] = th;
      pos[l] = 0;
    }
    __syncthreads();
  };

  if (threadIdx.x == 0) {
    level = 0;
    prefix[0] = 0;
    cab[0] = 0;
    hab[0] = 0;
    max_key = 0;
  }
  __syncthreads();
  build(0);
  // action: 0 = descend into act_b, 1 = found, 2 = pop, 3 = none at all
  while (true) {
    if (threadIdx.x == 0) {
      const int l = level;
      action = 2;
      int64_t run_c = 0, run_h = 0;  // windows in buckets below b
      for (int b = 0; b < pos[l]; ++b) {
        run_c += cnt[l][b];
        run_h += hl[l][b];
      }
      for (int b = pos[l]; b < NB; ++b) {
        run_c += cnt[l][b];
        run_h += hl[l][b];
        if (!cnt[l][b]) continue;
        // windows of this range in buckets above b, plus everything above the range
        const int64_t Ca = cab[l] + tot_c[l] - run_c, Ha = hab[l] + tot_h[l] - run_h;
        const int64_t C = Ca + cnt[l][b], H = Ha + hl[l][b];
        if ((double)H >= reliability * (double)C) {
          action = 1;
          result = mn[l][b];
          break;
        }
        // a value inside the bucket has at most its healthy windows on top of
        // those above; one window of slack keeps the bound valid under rounding
        if (l + 1 < NL &&
            (double)(Ha + hl[l][b] + 1) >= reliability * (double)(Ca + hl[l][b])) {
          action = 0;
          act_b = b;
          pos[l] = b + 1;
          cab[l + 1] = Ca;
          hab[l + 1] = Ha;
          prefix[l + 1] = (prefix[l] << 8) | (U)b;
          level = l + 1;
          break;
        }
      }
      if (action == 2) {
        if (l == 0) action = 3;
        else level = l - 1;
      }
    }
    __syncthreads();
    const int a = action;
    if (a == 0) {
      build(level);
      continue;
    }
    if (a == 2) {
      __syncthreads();
      continue;
    }
    if (threadIdx.x == 0) {
      T th;
      if (a == 1) {
        th = [&] { U k = result; T v; memcpy(&v, &k, sizeof(T)); return v; }();
      } else if (max_key) {
        U k = max_key;
        memcpy(&th, &k, sizeof(T));
        atomicAdd(&diag->degenerate_calib, 1ull);
      } else {
        th = (T)1;
        atomicAdd(&diag->degenerate_calib, 1ull);
      }
      theta[m] = th;
    }
    break;
  }
}

}  // namespace

template <class T> void calib_ws_layout(Arena& a, int M, int K, CalibWs<T>& w) {
  w.keys = a.take<typename KeyOf<T>::U>((size_t)M * std::max(K, 1));
  w.thr = a.take<int32_t>(kThrTable);
}

template <class T>
cudaError_t launch_calibrate(int M, int K, const T* S, const uint8_t* cls,
                             const unsigned long long* slo, double ok_frac, double reliability,
                             T* theta, CalibWs<T>& w, tre_diag* diag, cudaStream_t s) {
  using U = typename KeyOf<T>::U;
  k_thr<<<kThrTable / 256, 256, 0, s>>>(ok_frac, w.thr);
  if (K > 0) {
    dim3 g((K + 31) / 32, (M + 31) / 32), b(32, 8);
    k_pack<T><<<g, b, 0, s>>>(M, K, S, cls, slo, w.thr, ok_frac, static_cast<U*>(w.keys));
  }
  k_search<T><<<M, kSearchThreads, 0, s>>>(M, K, static_cast<const U*>(w.keys), reliability,
                                           theta, diag);
  return cudaGetLastError();
}

template void calib_ws_layout<float>(Arena&, int, int, CalibWs<float>&);
template void calib_ws_layout<double>(Arena&, int, int, CalibWs<double>&);
template cudaError_t launch_calibrate<float>(int, int, const float*, const uint8_t*,
                                             const unsigned long long*, double, double, float*,
                                             CalibWs<float>&, tre_diag*, cudaStream_t);
template cudaError_t launch_calibrate<double>(int, int, const double*, const uint8_t*,
                                              const unsigned long long*, double, double, double*,
                                              CalibWs<double>&, tre_diag*, cudaStream_t);

}  // namespace tre
