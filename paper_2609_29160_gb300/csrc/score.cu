// Raw TSS (Eq. 1), exponential smoothing (Sec. III-B), Z = TSS / theta (Eq. 2),
// regions, and the per-window Eq. 3 receiver -- for a batch of series at once.
//
// Eq. 1 is evaluated for every (window, model) in one fully parallel pass. The
// smoothing S_k = alpha*raw_k + (1-alpha)*S_{k-1} is a sequential chain per
// model; to spread it over the GPU and still return exactly the values of the
// sequential definition (one rounding per operation, in order):
//   1. each segment of windows computes its affine summary (approximate);
//   2. a per-model scan of the summaries gives every segment an approximate
//      start state;
//   3. every segment runs the exact recurrence from that start;
//   4. every segment re-runs from its predecessor's computed end until its new
//      trajectory meets the stored one bit for bit (the recurrence is a
//      contraction, so they meet after a short stretch; from there on every
//      value is identical because each step depends only on the previous S);
//   5. one thread per model walks the segment boundaries in order and repairs
//      any segment whose start still differs from its predecessor's end.
// After step 5 each segment's stored trajectory starts from the exact end of
// the previous one, so the concatenation is the sequential result.
#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace tre {
namespace {

constexpr int kThreads = 256;
constexpr int kBatch = 16;  // windows loaded ahead in the sequential chains

template <class T> __device__ __forceinline__ T sub_rn(T a, T b);
template <> __device__ __forceinline__ float sub_rn<float>(float a, float b) { return __fsub_rn(a, b); }
template <> __device__ __forceinline__ double sub_rn<double>(double a, double b) { return __dsub_rn(a, b); }

__device__ __forceinline__ bool same_bits(float a, float b) {
  return __float_as_uint(a) == __float_as_uint(b);
}
__device__ __forceinline__ bool same_bits(double a, double b) {
  return __double_as_longlong(a) == __double_as_longlong(b);
}

struct Counts {
  const int32_t *P, *D, *A, *W;
};

// series of a global segment index (the table has at most 64 entries)
template <class T> __device__ __forceinline__ int series_of_seg(const SeriesTable<T>& t, int seg) {
  int s = 0;
  while (s + 1 < t.n && t.seg_base[s + 1] <= seg) ++s;
  return s;
}

template <class T> struct ModelParams {
  T a, b, th, tc, ts;
};

template <class T>
__device__ __forceinline__ ModelParams<T> load_params(const SeriesTable<T>& t, int s, int m,
                                                      const T* alpha, const T* theta,
                                                      const T* tau_crit, const T* tau_surp) {
  ModelParams<T> p;
  p.a = alpha ? alpha[m] : t.alpha[s];
  p.b = sub_rn<T>((T)1, p.a);
  p.th = theta ? theta[m] : (T)1;
  p.tc = tau_crit ? tau_crit[m] : (T)0;
  p.ts = tau_surp ? tau_surp[m] : (T)0;
  return p;
}

// ---- pass 0: Eq. 1 for every (window, model); idle windows marked ---------
template <class T>
__global__ void __launch_bounds__(kThreads)
k_raw(const __grid_constant__ SeriesTable<T> tab, Counts c, const T* __restrict__ w_p,
      const T* __restrict__ w_q, T* __restrict__ raw, uint8_t* __restrict__ cls) {
  const int s = blockIdx.y;
  const int M = tab.M;
  const int64_t n = (int64_t)tab.K[s] * M;
  const T dt = div_rn((T)tab.win[s], (T)1000);      // window length in seconds
  for (int64_t i = (int64_t)blockIdx.x * kThreads + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * kThreads) {
    const size_t x = (size_t)(tab.off[s] + i);
    const int m = (int)((uint32_t)i % (uint32_t)M);
    const int32_t p = c.P[x], d = c.D[x], a = c.A[x], w = c.W[x];
    if ((p | d | a | w) == 0) {
      cls[x] = kIdle;
      continue;
    }
    const T r_pre = div_rn(from_i32<T>(p), dt);
    const T r_dec = div_rn(from_i32<T>(d), dt);
    const T num = add_rn(mul_rn(w_p[m], r_pre), r_dec);
    T den = add_rn(from_i32<T>(a), mul_rn(w_q[m], from_i32<T>(w)));
    if (den < (T)1) den = (T)1;                       // demand floor of one request
    raw[x] = div_rn(num, den);
    cls[x] = kNom;
  }
}

// raw values and classes of windows [k, k + kBatch) clipped to k1 (idle past k1)
template <class T>
__device__ __forceinline__ void load_batch(const T* __restrict__ raw, const uint8_t* __restrict__ cls,
                                           size_t base, int M, int64_t k, int64_t k1,
                                           T (&r)[kBatch], uint8_t (&c)[kBatch]) {
  if (k + kBatch <= k1) {
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
      const size_t x = base + (size_t)(k + j) * M;
      c[j] = cls[x];
      r[j] = raw[x];
    }
  } else {
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
      c[j] = kIdle;
      r[j] = (T)0;
      if (k + j < k1) {
        const size_t x = base + (size_t)(k + j) * M;
        c[j] = cls[x];
        r[j] = raw[x];
      }
    }
  }
}

// ---- pass 1: affine summary of each segment -------------------------------
template <class T>
__global__ void __launch_bounds__(kThreads)
k_summary(const __grid_constant__ SeriesTable<T> tab, const T* __restrict__ raw,
          const uint8_t* __restrict__ cls, const T* __restrict__ alpha, T* sm, T* sc, T* sci,
          int32_t* sh) {
  const int M = tab.M;
  const int64_t t = (int64_t)blockIdx.x * kThreads + threadIdx.x;
  if (t >= (int64_t)tab.seg_base[tab.n] * M) return;
  const int m = (int)(t % M);
  const int seg = (int)(t / M);
  const int s = series_of_seg(tab, seg);
  const int L = tab.seg_len[s];
  const int64_t k0 = (int64_t)(seg - tab.seg_base[s]) * L, k1 = min64(k0 + L, tab.K[s]);
  const T a = alpha ? alpha[m] : tab.alpha[s];
  const T b = sub_rn<T>((T)1, a);
  const size_t base = (size_t)tab.off[s] + m;
  T mm = (T)1, cc = (T)0, ci = (T)0;
  int h = 0;
  T r[kBatch], rn[kBatch];
  uint8_t c[kBatch], cn[kBatch];
  load_batch(raw, cls, base, M, k0, k1, r, c);
  for (int64_t k = k0; k < k1; k += kBatch) {
    // next batch in flight while this one is folded
    load_batch(raw, cls, base, M, k + kBatch, k1, rn, cn);
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
      if (c[j] == kIdle) continue;
      const T ar = a * r[j];
      ci = h ? ci * b + ar : r[j];
      cc = cc * b + ar;
      mm = mm * b;
      h = 1;
    }
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
      r[j] = rn[j];
      c[j] = cn[j];
    }
  }
  sm[t] = mm;
  sc[t] = cc;
  sci[t] = ci;
  sh[t] = h;
}

template <class T> struct Sum {
  T m, c, ci;
  int h;
};

template <class T> __device__ __forceinline__ Sum<T> combine(const Sum<T>& a, const Sum<T>& b) {
  if (!b.h) return a;
  if (!a.h) return b;
  Sum<T> r;
  r.m = a.m * b.m;
  r.c = a.c * b.m + b.c;
  r.ci = a.ci * b.m + b.c;
  r.h = 1;
  return r;
}

template <class T> __device__ __forceinline__ void apply(const Sum<T>& u, T& S, int& init) {
  if (!u.h) return;
  S = init ? u.m * S + u.c : u.ci;
  init = 1;
}

// ---- pass 2: per-(series, model) exclusive scan -> approximate starts ------
template <class T>
__global__ void k_starts(const __grid_constant__ SeriesTable<T> tab, const T* sm, const T* sc,
                         const T* sci, const int32_t* sh, const T* S_carry,
                         const uint8_t* init_carry, T* start_S, int32_t* start_init) {
  const int M = tab.M;
  const int w = blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
  if (w >= tab.n * M) return;
  const int s = w / M, m = w % M;
  const int lane = threadIdx.x & 31;
  const int n_seg = tab.seg_base[s + 1] - tab.seg_base[s];
  const int per = (n_seg + 31) / 32;
  const int s0 = lane * per, s1 = min(n_seg, s0 + per);
  const size_t g0 = (size_t)tab.seg_base[s] * M + m;
  Sum<T> agg{(T)1, (T)0, (T)0, 0};
  for (int q = s0; q < s1; ++q) {
    const size_t x = g0 + (size_t)q * M;
    agg = combine(agg, Sum<T>{sm[x], sc[x], sci[x], sh[x]});
  }
  Sum<T> inc = agg;
  for (int o = 1; o < 32; o <<= 1) {
    Sum<T> v;
    v.m = __shfl_up_sync(0xffffffffu, inc.m, o);
    v.c = __shfl_up_sync(0xffffffffu, inc.c, o);
    v.ci = __shfl_up_sync(0xffffffffu, inc.ci, o);
    v.h = __shfl_up_sync(0xffffffffu, inc.h, o);
    if (lane >= o) inc = combine(v, inc);
  }
  Sum<T> exc;
  exc.m = __shfl_up_sync(0xffffffffu, inc.m, 1);
  exc.c = __shfl_up_sync(0xffffffffu, inc.c, 1);
  exc.ci = __shfl_up_sync(0xffffffffu, inc.ci, 1);
  exc.h = __shfl_up_sync(0xffffffffu, inc.h, 1);
  if (lane == 0) exc = Sum<T>{(T)1, (T)0, (T)0, 0};
  int init = (init_carry && init_carry[m]) ? 1 : 0;
  T S = init ? S_carry[m] : (T)0;
  apply(exc, S, init);
  for (int q = s0; q < s1; ++q) {
    const size_t x = g0 + (size_t)q * M;
    start_S[x] = S;
    start_init[x] = init;
    apply(Sum<T>{sm[x], sc[x], sci[x], sh[x]}, S, init);
  }
}

// Run windows [k0, k1) of model m exactly from (S, init), writing S and, with
// `with_z`, Z and the region (idle windows keep their class). With `verify`,
// stop at the first window whose new S equals the stored one with the same
// init state: from there the stored trajectory is the one this start produces.
// Returns true if it stopped early.
template <class T>
__device__ __forceinline__ bool run_segment(size_t base, int M, int64_t k0, int64_t k1,
                                            const T* __restrict__ raw, const ModelParams<T>& q,
                                            T& S, int& init, bool verify, int stored_init,
                                            T* S_out, T* Z_out, uint8_t* cls, bool with_z) {
  T r[kBatch], rn[kBatch];
  uint8_t c[kBatch], cn[kBatch];
  load_batch(raw, cls, base, M, k0, k1, r, c);
  for (int64_t k = k0; k < k1; k += kBatch) {
    T old[kBatch];
    if (verify) {
#pragma unroll
      for (int j = 0; j < kBatch; ++j)
        if (k + j < k1) old[j] = S_out[base + (size_t)(k + j) * M];
    }
    // next batch in flight while this one runs
    load_batch(raw, cls, base, M, k + kBatch, k1, rn, cn);
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
      if (k + j >= k1) break;
      const bool active = c[j] != kIdle;
      if (active) {
        if (!init) {
          S = r[j];
          init = 1;
        } else {
          S = add_rn(mul_rn(q.a, r[j]), mul_rn(q.b, S));
        }
        stored_init = 1;
      }
      if (verify && init == stored_init && same_bits(S, old[j])) return true;
      const size_t x = base + (size_t)(k + j) * M;
      const T Sv = init ? S : (T)0;
      S_out[x] = Sv;
      if (with_z) {
        const T Z = div_rn(Sv, q.th);
        Z_out[x] = Z;
        if (active) cls[x] = Z < q.tc ? kCrit : (Z > q.ts ? kSurp : kNom);
      }
    }
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
      r[j] = rn[j];
      c[j] = cn[j];
    }
  }
  return false;
}

// ---- pass 3: run every segment from its approximate start -------------------
template <class T>
__global__ void __launch_bounds__(kThreads)
k_run(const __grid_constant__ SeriesTable<T> tab, const T* __restrict__ raw, const T* alpha,
      const T* theta, const T* tau_crit, const T* tau_surp, const T* start_S,
      const int32_t* start_init, T* end_S, int32_t* end_init, T* S_out, T* Z_out, uint8_t* cls) {
  const int M = tab.M;
  const int64_t t = (int64_t)blockIdx.x * kThreads + threadIdx.x;
  if (t >= (int64_t)tab.seg_base[tab.n] * M) return;
  const int m = (int)(t % M);
  const int seg = (int)(t / M);
  const int s = series_of_seg(tab, seg);
  const ModelParams<T> q = load_params(tab, s, m, alpha, theta, tau_crit, tau_surp);
  const int L = tab.seg_len[s];
  const int64_t k0 = (int64_t)(seg - tab.seg_base[s]) * L, k1 = min64(k0 + L, tab.K[s]);
  T S = start_S[t];
  int init = start_init[t];
  run_segment<T>((size_t)tab.off[s] + m, M, k0, k1, raw, q, S, init, false, 0, S_out, Z_out, cls,
                 theta != nullptr);
  end_S[t] = S;
  end_init[t] = init;
}

// ---- pass 4: parallel verification from the predecessor's computed end ------
template <class T>
__global__ void __launch_bounds__(kThreads)
k_verify(const __grid_constant__ SeriesTable<T> tab, const T* __restrict__ raw, const T* alpha,
         const T* theta, const T* tau_crit, const T* tau_surp, T* start_S, int32_t* start_init,
         const T* end_S, const int32_t* end_init, T* end_S2, int32_t* end_init2, T* S_out,
         T* Z_out, uint8_t* cls, tre_diag* diag) {
  const int M = tab.M;
  const int64_t t = (int64_t)blockIdx.x * kThreads + threadIdx.x;
  if (t >= (int64_t)tab.seg_base[tab.n] * M) return;
  const int m = (int)(t % M);
  const int seg = (int)(t / M);
  const int s = series_of_seg(tab, seg);
  T eS = end_S[t];
  int eI = end_init[t];
  if (seg > tab.seg_base[s]) {
    const size_t p = t - M;
    T S = end_S[p];
    int init = end_init[p];
    if (init != start_init[t] || !same_bits(S, start_S[t])) {
      const ModelParams<T> q = load_params(tab, s, m, alpha, theta, tau_crit, tau_surp);
      const int L = tab.seg_len[s];
      const int64_t k0 = (int64_t)(seg - tab.seg_base[s]) * L, k1 = min64(k0 + L, tab.K[s]);
      const int stored_init = start_init[t];
      start_S[t] = S;
      start_init[t] = init;
      const bool met = run_segment<T>((size_t)tab.off[s] + m, M, k0, k1, raw, q, S, init, true,
                                      stored_init, S_out, Z_out, cls, theta != nullptr);
      if (!met) {
        eS = S;
        eI = init;
      }
      atomicAdd(&diag->ema_resolved, 1ull);
    }
  }
  end_S2[t] = eS;
  end_init2[t] = eI;
}

// ---- pass 5: in-order repair, one thread per (series, model) ---------------
template <class T>
__global__ void k_resolve(const __grid_constant__ SeriesTable<T> tab, const T* __restrict__ raw,
                          const T* alpha, const T* theta, const T* tau_crit, const T* tau_surp,
                          const T* start_S, const int32_t* start_init, const T* end_S,
                          const int32_t* end_init, T* S_out, T* Z_out, uint8_t* cls,
                          T* S_carry, uint8_t* init_carry, tre_diag* diag) {
  const int M = tab.M;
  const int w = blockIdx.x * blockDim.x + threadIdx.x;
  if (w >= tab.n * M) return;
  const int s = w / M, m = w % M;
  const int n_seg = tab.seg_base[s + 1] - tab.seg_base[s];
  if (n_seg == 0) return;
  const ModelParams<T> q = load_params(tab, s, m, alpha, theta, tau_crit, tau_surp);
  const int L = tab.seg_len[s];
  const size_t g0 = (size_t)tab.seg_base[s] * M + m;
  T S = end_S[g0];
  int init = end_init[g0];
  for (int q0 = 1; q0 < n_seg; q0 += kBatch) {
    // load the boundary states of a batch of segments ahead of the checks
    T bS[kBatch], bE[kBatch];
    int bI[kBatch], bEI[kBatch];
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
      if (q0 + j < n_seg) {
        const size_t x = g0 + (size_t)(q0 + j) * M;
        bS[j] = start_S[x];
        bI[j] = start_init[x];
        bE[j] = end_S[x];
        bEI[j] = end_init[x];
      }
    }
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
      const int qq = q0 + j;
      if (qq >= n_seg) break;
      if (init == bI[j] && same_bits(S, bS[j])) {
        S = bE[j];
        init = bEI[j];
        continue;
      }
      const int64_t k0 = (int64_t)qq * L, k1 = min64(k0 + L, tab.K[s]);
      const bool met = run_segment<T>((size_t)tab.off[s] + m, M, k0, k1, raw, q, S, init, true,
                                      bI[j], S_out, Z_out, cls, theta != nullptr);
      if (met) {
        S = bE[j];
        init = bEI[j];
      }
      atomicAdd(&diag->ema_resolved, 1ull);
    }
  }
  if (S_carry) {
    S_carry[m] = S;
    init_carry[m] = (uint8_t)init;
  }
}

// ---- Z and regions from S for every series ---------------------------------
template <class T>
__global__ void __launch_bounds__(kThreads)
k_normalize(const __grid_constant__ SeriesTable<T> tab, const T* S, const uint8_t* idle_cls,
            const T* theta, const T* tau_crit, T tau_crit_v, const T* tau_surp, T* Z,
            uint8_t* cls) {
  const int s = blockIdx.y;
  const int M = tab.M;
  const int64_t n = (int64_t)tab.K[s] * M;
  for (int64_t i = (int64_t)blockIdx.x * kThreads + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * kThreads) {
    const size_t x = (size_t)(tab.off[s] + i);
    const int m = (int)((uint32_t)i % (uint32_t)M);
    const T z = div_rn(S[x], theta[(size_t)s * M + m]);
    if (Z) Z[x] = z;
    if (cls) {
      uint8_t c;
      if (idle_cls[x] == kIdle) c = kIdle;
      else if (z < (tau_crit ? tau_crit[m] : tau_crit_v)) c = kCrit;
      else if (z > tau_surp[m]) c = kSurp;
      else c = kNom;
      cls[x] = c;
    }
  }
}

// ---- Eq. 3 receiver per window: warp per window ----------------------------
template <class T>
__global__ void k_receiver(int M, int K, const T* Z, const uint8_t* cls, int32_t* recv) {
  const int64_t k = (int64_t)blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
  if (k >= K) return;
  const int lane = threadIdx.x & 31;
  int best = -1;
  T bz = (T)0;
  for (int m = lane; m < M; m += 32) {
    const size_t x = (size_t)k * M + m;
    if (cls[x] == kIdle) continue;
    const T z = Z[x];
    if (best < 0 || z < bz) { best = m; bz = z; }
  }
  for (int o = 16; o > 0; o >>= 1) {
    const int ob = __shfl_down_sync(0xffffffffu, best, o);
    const T oz = __shfl_down_sync(0xffffffffu, bz, o);
    if (ob >= 0 && (best < 0 || oz < bz || (oz == bz && ob < best))) { best = ob; bz = oz; }
  }
  if (lane == 0) recv[k] = best;
}

template <class T> int64_t max_elems(const SeriesTable<T>& t) {
  int64_t mx = 0;
  for (int s = 0; s < t.n; ++s) mx = std::max<int64_t>(mx, (int64_t)t.K[s] * t.M);
  return mx;
}

unsigned blocks_for(int64_t n, int cap) {
  int64_t b = (n + kThreads - 1) / kThreads;
  return (unsigned)std::max<int64_t>(1, std::min<int64_t>(b, cap));
}

}  // namespace

template <class T> int series_segments(SeriesTable<T>& t) {
  int total = 0;
  for (int s = 0; s < t.n; ++s) {
    const int K = t.K[s];
    // Two trajectories of the smoothing that start a few dozen ulps apart meet
    // after about 4 / alpha windows; segments about twice that long let the
    // verification pass meet the stored trajectory inside one segment.
    const double a = (double)t.alpha[s];
    int base = 64;
    while (base < 512 && !(a > 0 && (double)base * a >= 8.0)) base *= 2;
    int L = (K + 1023) / 1024;
    L = L < base ? base : L;
    t.seg_len[s] = L;
    t.seg_base[s] = total;
    total += (K + L - 1) / L;
  }
  t.seg_base[t.n] = total;
  return total;
}

template <class T> void score_ws_layout(Arena& a, int M, int64_t elems, int n_seg, ScoreWs<T>& w) {
  w.raw = a.take<T>((size_t)std::max<int64_t>(elems, 1));
  w.cap_seg = std::max(n_seg, 1);
  const size_t n = (size_t)w.cap_seg * M;
  w.sum_m = a.take<T>(n);
  w.sum_c = a.take<T>(n);
  w.sum_ci = a.take<T>(n);
  w.sum_h = a.take<int32_t>(n);
  w.start_S = a.take<T>(n);
  w.start_init = a.take<int32_t>(n);
  w.end_S = a.take<T>(n);
  w.end_init = a.take<int32_t>(n);
  w.end_S2 = a.take<T>(n);
  w.end_init2 = a.take<int32_t>(n);
}

template <class T>
cudaError_t launch_score(const SeriesTable<T>& tab, const int32_t* P, const int32_t* D,
                         const int32_t* A, const int32_t* W, const T* w_p, const T* w_q,
                         const T* alpha, const T* theta, const T* tau_crit, const T* tau_surp,
                         T* S_carry, uint8_t* init_carry, T* S, T* Z, uint8_t* cls,
                         ScoreWs<T>& w, tre_diag* diag, cudaStream_t s) {
  const int M = tab.M;
  const int n_seg = tab.seg_base[tab.n];
  if (n_seg > w.cap_seg) return cudaErrorInvalidValue;
  const int64_t mx = max_elems(tab);
  if (mx == 0) return cudaSuccess;
  const Counts c{P, D, A, W};
  dim3 ge(blocks_for(mx, 2048), tab.n);
  k_raw<T><<<ge, kThreads, 0, s>>>(tab, c, w_p, w_q, w.raw, cls);
  const int64_t segs = (int64_t)n_seg * M;
  const unsigned g = (unsigned)((segs + kThreads - 1) / kThreads);
  k_summary<T><<<g, kThreads, 0, s>>>(tab, w.raw, cls, alpha, w.sum_m, w.sum_c, w.sum_ci, w.sum_h);
  const int warps = tab.n * M;
  k_starts<T><<<(warps + 3) / 4, 128, 0, s>>>(tab, w.sum_m, w.sum_c, w.sum_ci, w.sum_h, S_carry,
                                              init_carry, w.start_S, w.start_init);
  k_run<T><<<g, kThreads, 0, s>>>(tab, w.raw, alpha, theta, tau_crit, tau_surp, w.start_S,
                                  w.start_init, w.end_S, w.end_init, S, Z, cls);
  k_verify<T><<<g, kThreads, 0, s>>>(tab, w.raw, alpha, theta, tau_crit, tau_surp, w.start_S,
                                     w.start_init, w.end_S, w.end_init, w.end_S2, w.end_init2, S,
                                     Z, cls, diag);
  k_resolve<T><<<(warps + 63) / 64, 64, 0, s>>>(tab, w.raw, alpha, theta, tau_crit, tau_surp,
                                                w.start_S, w.start_init, w.end_S2, w.end_init2,
                                                S, Z, cls, S_carry, init_carry, diag);
  return cudaGetLastError();
}

template <class T>
cudaError_t launch_normalize(const SeriesTable<T>& tab, const T* S, const uint8_t* idle_cls,
                             const T* theta, const T* tau_crit, T tau_crit_v, const T* tau_surp,
                             T* Z, uint8_t* cls, cudaStream_t s) {
  const int64_t mx = max_elems(tab);
  if (mx == 0) return cudaSuccess;
  dim3 g(blocks_for(mx, 1024), tab.n);
  k_normalize<T><<<g, kThreads, 0, s>>>(tab, S, idle_cls, theta, tau_crit, tau_crit_v, tau_surp,
                                        Z, cls);
  return cudaGetLastError();
}

template <class T>
cudaError_t launch_receiver(int M, int K, const T* Z, const uint8_t* cls, int32_t* recv,
                            cudaStream_t s) {
  if (K == 0) return cudaSuccess;
  k_receiver<T><<<(unsigned)((K + 7) / 8), 256, 0, s>>>(M, K, Z, cls, recv);
  return cudaGetLastError();
}

#define TRE_INST(T)                                                                               \
  template int series_segments<T>(SeriesTable<T>&);                                               \
  template void score_ws_layout<T>(Arena&, int, int64_t, int, ScoreWs<T>&);                       \
  template cudaError_t launch_score<T>(const SeriesTable<T>&, const int32_t*, const int32_t*,      \
                                       const int32_t*, const int32_t*, const T*, const T*,         \
                                       const T*, const T*, const T*, const T*, T*, uint8_t*, T*,   \
                                       T*, uint8_t*, ScoreWs<T>&, tre_diag*, cudaStream_t);        \
  template cudaError_t launch_normalize<T>(const SeriesTable<T>&, const T*, const uint8_t*,        \
                                           const T*, const T*, T, const T*, T*, uint8_t*,          \
                                           cudaStream_t);                                          \
  template cudaError_t launch_receiver<T>(int, int, const T*, const uint8_t*, int32_t*,            \
                                          cudaStream_t);
TRE_INST(float)
TRE_INST(double)

}  // namespace tre
