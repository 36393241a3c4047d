// Raw TSS (Eq. 1), exponential smoothing (Sec. III-B), Z = TSS / theta (Eq. 2),
// regions, and the per-window Eq. 3 receiver.
//
// The smoothing S_k = alpha*raw_k + (1-alpha)*S_{k-1} is a sequential chain per
// model. To spread it over the GPU and still return exactly the values of the
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

template <class T> __device__ __forceinline__ T sub_rn(T a, T b);
template <> __device__ __forceinline__ float sub_rn<float>(float a, float b) { return __fsub_rn(a, b); }
template <> __device__ __forceinline__ double sub_rn<double>(double a, double b) { return __dsub_rn(a, b); }

__device__ __forceinline__ bool same_bits(float a, float b) {
  return __float_as_uint(a) == __float_as_uint(b);
}
__device__ __forceinline__ bool same_bits(double a, double b) {
  return __double_as_longlong(a) == __double_as_longlong(b);
}

template <class T> struct ModelParams {
  T wp, wq, a, b, th, tc, ts;
};

template <class T>
__device__ __forceinline__ ModelParams<T> load_params(const T* w_p, const T* w_q, const T* alpha,
                                                      T alpha_v, const T* theta,
                                                      const T* tau_crit, const T* tau_surp,
                                                      int m) {
  ModelParams<T> p;
  p.wp = w_p[m];
  p.wq = w_q[m];
  p.a = alpha ? alpha[m] : alpha_v;
  p.b = sub_rn<T>((T)1, p.a);
  p.th = theta ? theta[m] : (T)1;
  p.tc = tau_crit ? tau_crit[m] : (T)0;
  p.ts = tau_surp ? tau_surp[m] : (T)0;
  return p;
}

// Eq. 1 for one (window, model); returns false for an idle window
template <class T>
__device__ __forceinline__ bool raw_tss(int32_t p, int32_t d, int32_t a, int32_t w,
                                        const ModelParams<T>& q, T dt, T& raw) {
  if ((p | d | a | w) == 0) return false;
  const T r_pre = div_rn(from_i32<T>(p), dt);
  const T r_dec = div_rn(from_i32<T>(d), dt);
  const T num = add_rn(mul_rn(q.wp, r_pre), r_dec);
  T den = add_rn(from_i32<T>(a), mul_rn(q.wq, from_i32<T>(w)));
  if (den < (T)1) den = (T)1;
  raw = div_rn(num, den);
  return true;
}

template <class T>
__device__ __forceinline__ void ema_step(T& S, int& init, T raw, const ModelParams<T>& q) {
  if (!init) {
    S = raw;
    init = 1;
  } else {
    S = add_rn(mul_rn(q.a, raw), mul_rn(q.b, S));
  }
}

template <class T>
__device__ __forceinline__ uint8_t region(bool idle, T Z, const ModelParams<T>& q, bool classify) {
  if (idle) return kIdle;
  if (!classify) return kNom;
  if (Z < q.tc) return kCrit;
  if (Z > q.ts) return kSurp;
  return kNom;
}

struct Counts {
  const int32_t *P, *D, *A, *W;
};

// ---- pass 1: affine summary of each segment -------------------------------
template <class T>
__global__ void __launch_bounds__(kThreads)
k_summary(int M, int K, int L, int n_seg, Counts c, const T* w_p, const T* w_q, const T* alpha,
          T alpha_v, T dt, T* sm, T* sc, T* sci, int32_t* sh) {
  const int64_t t = (int64_t)blockIdx.x * kThreads + threadIdx.x;
  if (t >= (int64_t)n_seg * M) return;
  const int m = (int)(t % M);
  const int s = (int)(t / M);
  const ModelParams<T> q = load_params<T>(w_p, w_q, alpha, alpha_v, nullptr, nullptr, nullptr, m);
  T mm = (T)1, cc = (T)0, ci = (T)0;
  int h = 0;
  const int64_t k0 = (int64_t)s * L, k1 = min64(k0 + L, K);
  for (int64_t k = k0; k < k1; ++k) {
    const size_t x = (size_t)k * M + m;
    T raw;
    if (!raw_tss<T>(c.P[x], c.D[x], c.A[x], c.W[x], q, dt, raw)) continue;
    const T ar = q.a * raw;
    ci = h ? ci * q.b + ar : raw;
    cc = cc * q.b + ar;
    mm = mm * q.b;
    h = 1;
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

// ---- pass 2: per-model exclusive scan of summaries -> approximate starts ----
template <class T>
__global__ void k_starts(int M, int n_seg, const T* sm, const T* sc, const T* sci,
                         const int32_t* sh, const T* S_carry, const uint8_t* init_carry,
                         T* start_S, int32_t* start_init) {
  const int m = blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
  if (m >= M) return;
  const int lane = threadIdx.x & 31;
  const int per = (n_seg + 31) / 32;
  const int s0 = lane * per, s1 = min(n_seg, s0 + per);
  Sum<T> agg{(T)1, (T)0, (T)0, 0};
  for (int s = s0; s < s1; ++s) {
    const size_t x = (size_t)s * M + m;
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
  for (int s = s0; s < s1; ++s) {
    const size_t x = (size_t)s * M + m;
    start_S[x] = S;
    start_init[x] = init;
    apply(Sum<T>{sm[x], sc[x], sci[x], sh[x]}, S, init);
  }
}

// Run segment (s, m) exactly from (S, init) over windows [k0, k1), writing S,
// Z and the region. With `verify`, stop at the first window whose new S equals
// the stored one (same init state): from there the stored trajectory is the
// one this start produces. Returns true if it stopped early.
template <class T>
__device__ __forceinline__ bool run_segment(int M, int m, int64_t k0, int64_t k1, Counts c,
                                            const ModelParams<T>& q, T dt, T& S, int& init,
                                            bool verify, int stored_init, T* S_out, T* Z_out,
                                            uint8_t* cls_out, bool with_z) {
  for (int64_t k = k0; k < k1; ++k) {
    const size_t x = (size_t)k * M + m;
    T raw;
    const bool active = raw_tss<T>(c.P[x], c.D[x], c.A[x], c.W[x], q, dt, raw);
    if (active) {
      ema_step<T>(S, init, raw, q);
      stored_init = 1;
    }
    if (verify && init == stored_init && same_bits(S, S_out[x])) return true;
    const T Sv = init ? S : (T)0;
    S_out[x] = Sv;
    T Z = (T)0;
    if (with_z) {
      Z = div_rn(Sv, q.th);
      Z_out[x] = Z;
    }
    cls_out[x] = region<T>(!active, Z, q, with_z);
  }
  return false;
}

// ---- pass 3: run every segment from its approximate start -------------------
template <class T>
__global__ void __launch_bounds__(kThreads)
k_run(int M, int K, int L, int n_seg, Counts c, const T* w_p, const T* w_q, const T* alpha,
      T alpha_v, const T* theta, const T* tau_crit, const T* tau_surp, T dt,
      const T* start_S, const int32_t* start_init, T* end_S, int32_t* end_init, T* S_out,
      T* Z_out, uint8_t* cls_out) {
  const int64_t t = (int64_t)blockIdx.x * kThreads + threadIdx.x;
  if (t >= (int64_t)n_seg * M) return;
  const int m = (int)(t % M);
  const int s = (int)(t / M);
  const ModelParams<T> q = load_params<T>(w_p, w_q, alpha, alpha_v, theta, tau_crit, tau_surp, m);
  T S = start_S[t];
  int init = start_init[t];
  const int64_t k0 = (int64_t)s * L, k1 = min64(k0 + L, K);
  run_segment<T>(M, m, k0, k1, c, q, dt, S, init, false, 0, S_out, Z_out, cls_out,
                 theta != nullptr);
  end_S[t] = S;
  end_init[t] = init;
}

// ---- pass 4: parallel verification from the predecessor's computed end ------
template <class T>
__global__ void __launch_bounds__(kThreads)
k_verify(int M, int K, int L, int n_seg, Counts c, const T* w_p, const T* w_q, const T* alpha,
         T alpha_v, const T* theta, const T* tau_crit, const T* tau_surp, T dt, T* start_S,
         int32_t* start_init, const T* end_S, const int32_t* end_init, T* end_S2,
         int32_t* end_init2, T* S_out, T* Z_out, uint8_t* cls_out, tre_diag* diag) {
  const int64_t t = (int64_t)blockIdx.x * kThreads + threadIdx.x;
  if (t >= (int64_t)n_seg * M) return;
  const int m = (int)(t % M);
  const int s = (int)(t / M);
  T eS = end_S[t];
  int eI = end_init[t];
  if (s > 0) {
    const size_t p = t - M;
    T S = end_S[p];
    int init = end_init[p];
    if (init != start_init[t] || !same_bits(S, start_S[t])) {
      const ModelParams<T> q =
          load_params<T>(w_p, w_q, alpha, alpha_v, theta, tau_crit, tau_surp, m);
      const int64_t k0 = (int64_t)s * L, k1 = min64(k0 + L, K);
      const int stored_init = start_init[t];
      start_S[t] = S;
      start_init[t] = init;
      const bool met = run_segment<T>(M, m, k0, k1, c, q, dt, S, init, true, stored_init, S_out,
                                      Z_out, cls_out, theta != nullptr);
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

// ---- pass 5: in-order repair, one thread per model ---------------------------
template <class T>
__global__ void k_resolve(int M, int K, int L, int n_seg, Counts c, const T* w_p, const T* w_q,
                          const T* alpha, T alpha_v, const T* theta, const T* tau_crit,
                          const T* tau_surp, T dt, const T* start_S, const int32_t* start_init,
                          const T* end_S, const int32_t* end_init, T* S_out, T* Z_out,
                          uint8_t* cls_out, T* S_carry, uint8_t* init_carry, tre_diag* diag) {
  const int m = blockIdx.x * blockDim.x + threadIdx.x;
  if (m >= M) return;
  const ModelParams<T> q = load_params<T>(w_p, w_q, alpha, alpha_v, theta, tau_crit, tau_surp, m);
  T S = end_S[m];
  int init = end_init[m];
  for (int s = 1; s < n_seg; ++s) {
    const size_t x = (size_t)s * M + m;
    if (init == start_init[x] && same_bits(S, start_S[x])) {
      S = end_S[x];
      init = end_init[x];
      continue;
    }
    const int64_t k0 = (int64_t)s * L, k1 = min64(k0 + L, K);
    const bool met = run_segment<T>(M, m, k0, k1, c, q, dt, S, init, true, start_init[x], S_out,
                                    Z_out, cls_out, theta != nullptr);
    if (met) {
      S = end_S[x];
      init = end_init[x];
    }
    atomicAdd(&diag->ema_resolved, 1ull);
  }
  if (S_carry && n_seg > 0) {
    S_carry[m] = S;
    init_carry[m] = (uint8_t)init;
  }
}

// ---- Z and regions from S (one threshold for every model optional) ---------
template <class T>
__global__ void __launch_bounds__(kThreads)
k_normalize(int M, int64_t n, const T* S, const uint8_t* idle_cls, const T* theta,
            const T* tau_crit, T tau_crit_v, const T* tau_surp, T* Z, uint8_t* cls) {
  for (int64_t t = (int64_t)blockIdx.x * kThreads + threadIdx.x; t < n;
       t += (int64_t)gridDim.x * kThreads) {
    const int m = (int)(t % M);
    const T z = div_rn(S[t], theta[m]);
    if (Z) Z[t] = z;
    if (cls) {
      uint8_t c;
      if (idle_cls[t] == kIdle) c = kIdle;
      else if (z < (tau_crit ? tau_crit[m] : tau_crit_v)) c = kCrit;
      else if (z > tau_surp[m]) c = kSurp;
      else c = kNom;
      cls[t] = c;
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

int seg_len_for(int K) {
  const int L = (K + 1023) / 1024;
  return L < 256 ? 256 : L;
}

template <class T>
cudaError_t score_impl(int M, int win, int K, const int32_t* P, const int32_t* D, const int32_t* A,
                       const int32_t* W, const T* w_p, const T* w_q, const T* alpha, T alpha_v,
                       const T* theta, const T* tau_crit, const T* tau_surp, T* S_carry,
                       uint8_t* init_carry, T* S, T* Z, uint8_t* cls, ScoreWs<T>& w,
                       tre_diag* diag, cudaStream_t s) {
  if (K == 0) return cudaSuccess;
  const T dt = (T)win / (T)1000;
  // segmenting of this call; never more segments than the workspace was laid
  // out for (the count grows with K)
  const int L = seg_len_for(K), n = (K + L - 1) / L;
  if (n > w.n_seg) return cudaErrorInvalidValue;
  const int64_t segs = (int64_t)n * M;
  const unsigned g = (unsigned)((segs + kThreads - 1) / kThreads);
  const Counts c{P, D, A, W};
  k_summary<T><<<g, kThreads, 0, s>>>(M, K, L, n, c, w_p, w_q, alpha, alpha_v, dt, w.sum_m,
                                      w.sum_c, w.sum_ci, w.sum_h);
  k_starts<T><<<(M + 3) / 4, 128, 0, s>>>(M, n, w.sum_m, w.sum_c, w.sum_ci, w.sum_h, S_carry,
                                          init_carry, w.start_S, w.start_init);
  k_run<T><<<g, kThreads, 0, s>>>(M, K, L, n, c, w_p, w_q, alpha, alpha_v, theta, tau_crit,
                                  tau_surp, dt, w.start_S, w.start_init, w.end_S, w.end_init, S,
                                  Z, cls);
  k_verify<T><<<g, kThreads, 0, s>>>(M, K, L, n, c, w_p, w_q, alpha, alpha_v, theta, tau_crit,
                                     tau_surp, dt, w.start_S, w.start_init, w.end_S, w.end_init,
                                     w.end_S2, w.end_init2, S, Z, cls, diag);
  k_resolve<T><<<(M + 63) / 64, 64, 0, s>>>(M, K, L, n, c, w_p, w_q, alpha, alpha_v, theta,
                                            tau_crit, tau_surp, dt, w.start_S, w.start_init,
                                            w.end_S2, w.end_init2, S, Z, cls, S_carry,
                                            init_carry, diag);
  return cudaGetLastError();
}

}  // namespace

template <class T> void score_ws_layout(Arena& a, int M, int K, ScoreWs<T>& w) {
  w.seg_len = seg_len_for(K);
  w.n_seg = (K + w.seg_len - 1) / w.seg_len;
  const size_t n = (size_t)std::max(w.n_seg, 1) * M;
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
cudaError_t launch_score(int M, int win, int K, const int32_t* P, const int32_t* D,
                         const int32_t* A, const int32_t* W, const T* w_p, const T* w_q,
                         const T* alpha, const T* theta, const T* tau_crit, const T* tau_surp,
                         T* S_carry, uint8_t* init_carry, T* S, T* Z, uint8_t* cls,
                         ScoreWs<T>& w, tre_diag* diag, cudaStream_t s) {
  return score_impl<T>(M, win, K, P, D, A, W, w_p, w_q, alpha, (T)0, theta, tau_crit, tau_surp,
                       S_carry, init_carry, S, Z, cls, w, diag, s);
}

template <class T>
cudaError_t launch_score_alpha(int M, int win, int K, const int32_t* P, const int32_t* D,
                               const int32_t* A, const int32_t* W, const T* w_p, const T* w_q,
                               T alpha, T* S, uint8_t* cls, ScoreWs<T>& w, tre_diag* diag,
                               cudaStream_t s) {
  return score_impl<T>(M, win, K, P, D, A, W, w_p, w_q, nullptr, alpha, nullptr, nullptr, nullptr,
                       nullptr, nullptr, S, nullptr, cls, w, diag, s);
}

template <class T>
cudaError_t launch_normalize(int M, int K, const T* S, const uint8_t* idle_cls, const T* theta,
                             const T* tau_crit, T tau_crit_v, const T* tau_surp, T* Z,
                             uint8_t* cls, cudaStream_t s) {
  const int64_t n = (int64_t)K * M;
  if (n == 0) return cudaSuccess;
  int64_t b = (n + kThreads - 1) / kThreads;
  if (b > 152 * 32) b = 152 * 32;
  k_normalize<T><<<(unsigned)b, kThreads, 0, s>>>(M, n, S, idle_cls, theta, tau_crit, tau_crit_v,
                                                  tau_surp, Z, cls);
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
  template void score_ws_layout<T>(Arena&, int, int, ScoreWs<T>&);                                \
  template cudaError_t launch_score<T>(int, int, int, const int32_t*, const int32_t*,              \
                                       const int32_t*, const int32_t*, const T*, const T*,         \
                                       const T*, const T*, const T*, const T*, T*, uint8_t*, T*,   \
                                       T*, uint8_t*, ScoreWs<T>&, tre_diag*, cudaStream_t);        \
  template cudaError_t launch_score_alpha<T>(int, int, int, const int32_t*, const int32_t*,        \
                                             const int32_t*, const int32_t*, const T*, const T*,   \
                                             T, T*, uint8_t*, ScoreWs<T>&, tre_diag*,              \
                                             cudaStream_t);                                        \
  template cudaError_t launch_normalize<T>(int, int, const T*, const uint8_t*, const T*,           \
                                           const T*, T, const T*, T*, uint8_t*, cudaStream_t);     \
  template cudaError_t launch_receiver<T>(int, int, const T*, const uint8_t*, int32_t*,            \
                                          cudaStream_t);
TRE_INST(float)
TRE_INST(double)

}  // namespace tre
