// Raw TSS (Eq. 1), exponential smoothing (Sec. III-B), Z = TSS / theta (Eq. 2),
// regions, and the per-window Eq. 3 receiver -- for a batch of series at once.
//
// Eq. 1 is evaluated for every (window, model) in one fully parallel pass. The
// smoothing S_k = alpha*raw_k + (1-alpha)*S_{k-1} is a sequential chain per
// model; to spread it over the GPU and still return exactly the values of the
// sequential definition (one rounding per operation, in order):
//   1. the windows of each series are cut into chunks; one thread per (chunk,
//      model) first runs the recurrence over the B windows before its chunk
//      ("burn-in", started as if the series began there; B ~ c / -ln(1-alpha),
//      so a start error shrinks by e^-c before the chunk: c = 28 for float, 45
//      for double), records the state
//      it reached, then runs its chunk from that state and stores the result;
//   2. one thread per model walks the chunk boundaries in order: a chunk whose
//      recorded burn-in state equals its predecessor's exact end state (bit
//      for bit, with the same started/not-started flag) is exact, because
//      every step depends only on the previous state; any other chunk is run
//      again from the exact state until its new trajectory meets the stored
//      one. A chunk whose burn-in reaches window 0 starts from the true initial
//      state and is exact by construction.
// The result is therefore the sequential one in every case; the in-order pass
// only re-runs chunks when a burn-in did not converge (long idle stretches, a
// tiny alpha), counted in tre_diag.ema_resolved.
#include <algorithm>
#include <initializer_list>

#include "common.cuh"
#include "internal.h"

namespace tre {
namespace {

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
  const int64_t *A_ms, *W_ms;   // time-averaged occupancy (request-ms per window) or null
};

template <class T> __device__ __forceinline__ T from_i64(long long v);
template <> __device__ __forceinline__ float from_i64<float>(long long v) { return __ll2float_rn(v); }
template <> __device__ __forceinline__ double from_i64<double>(long long v) {
  return __ll2double_rn(v);
}

// series of a global segment index (the table has at most 64 entries)
template <class T> __device__ __forceinline__ int series_of_seg(const SeriesTable<T>& t, int seg) {
  return prefix_index(t.seg_base, t.n, seg);
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

// Eq. 1 values of idle windows carry this NaN pattern (arithmetic on the GPU
// only produces the canonical NaN), so the smoothing pass reads one array.
__device__ __forceinline__ float idle_raw(float) { return __uint_as_float(0xffc0deadu); }
__device__ __forceinline__ double idle_raw(double) {
  return __longlong_as_double((long long)0xfff8deaddeadbeefull);
}
__device__ __forceinline__ bool is_idle_raw(float r) { return __float_as_uint(r) == 0xffc0deadu; }
__device__ __forceinline__ bool is_idle_raw(double r) {
  return (unsigned long long)__double_as_longlong(r) == 0xfff8deaddeadbeefull;
}

// ---- pass 0: Eq. 1 for every (window, model) of every series ---------------
// Element-wise passes run over tiles of kTile consecutive elements of one
// series; a thread takes four consecutive elements, with 16-byte loads and
// stores when they are aligned (scalar ones otherwise), so that enough bytes
// are in flight to cover memory latency.
constexpr int kEwThreads = 256;
constexpr int kTile = 4 * kEwThreads;
struct TilePlan {
  int tile_base[kMaxSeries + 1];   // prefix of tiles per series
};

template <class T>
__device__ __forceinline__ T raw_tss(int32_t p, int32_t d, int32_t a, int32_t w, T dt, T wp,
                                     T wq) {
  const T r_pre = div_rn(from_i32<T>(p), dt);
  const T r_dec = div_rn(from_i32<T>(d), dt);
  const T num = add_rn(mul_rn(wp, r_pre), r_dec);
  T den = add_rn(from_i32<T>(a), mul_rn(wq, from_i32<T>(w)));
  if (den < (T)1) den = (T)1;                       // demand floor of one request
  return div_rn(num, den);
}

// Eq. 1 with the window means of the running and waiting counts: the
// request-milliseconds inside the window divided by its length
template <class T>
__device__ __forceinline__ T raw_tss_mean(int32_t p, int32_t d, long long a_ms, long long w_ms,
                                          T dt, T win, T wp, T wq) {
  const T r_pre = div_rn(from_i32<T>(p), dt);
  const T r_dec = div_rn(from_i32<T>(d), dt);
  const T num = add_rn(mul_rn(wp, r_pre), r_dec);
  const T a = div_rn(from_i64<T>(a_ms), win);
  const T w = div_rn(from_i64<T>(w_ms), win);
  T den = add_rn(a, mul_rn(wq, w));
  if (den < (T)1) den = (T)1;                       // demand floor of one request
  return div_rn(num, den);
}

template <class T, bool MEAN>
__global__ void __launch_bounds__(kEwThreads)
k_raw(const __grid_constant__ SeriesTable<T> tab, const __grid_constant__ TilePlan tp, FastDiv fm,
      bool vec, Counts c, const T* __restrict__ w_p, const T* __restrict__ w_q,
      T* __restrict__ raw, uint8_t* __restrict__ cls) {
  const int s = prefix_index(tp.tile_base, tab.n, blockIdx.x);
  const int M = tab.M;
  const int64_t n = (int64_t)tab.K[s] * M;
  const int64_t l0 = (int64_t)(blockIdx.x - tp.tile_base[s]) * kTile + 4 * threadIdx.x;
  if (l0 >= n) return;
  const size_t x0 = (size_t)(tab.off[s] + l0);
  const T dt = div_rn((T)tab.win[s], (T)1000);      // window length in seconds
  int32_t p[4], d[4], a[4], w[4];
  long long am[4], wm[4];
  const bool v4 = vec && l0 + 4 <= n;
  if (v4) {
    const int4 P4 = *reinterpret_cast<const int4*>(c.P + x0);
    const int4 D4 = *reinterpret_cast<const int4*>(c.D + x0);
    p[0] = P4.x; p[1] = P4.y; p[2] = P4.z; p[3] = P4.w;
    d[0] = D4.x; d[1] = D4.y; d[2] = D4.z; d[3] = D4.w;
    if (MEAN) {
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const longlong2 A2 = reinterpret_cast<const longlong2*>(c.A_ms + x0)[h];
        const longlong2 W2 = reinterpret_cast<const longlong2*>(c.W_ms + x0)[h];
        am[2 * h] = A2.x; am[2 * h + 1] = A2.y;
        wm[2 * h] = W2.x; wm[2 * h + 1] = W2.y;
      }
    } else {
      const int4 A4 = *reinterpret_cast<const int4*>(c.A + x0);
      const int4 W4 = *reinterpret_cast<const int4*>(c.W + x0);
      a[0] = A4.x; a[1] = A4.y; a[2] = A4.z; a[3] = A4.w;
      w[0] = W4.x; w[1] = W4.y; w[2] = W4.z; w[3] = W4.w;
    }
  } else {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const bool in = l0 + i < n;
      p[i] = in ? c.P[x0 + i] : 0;
      d[i] = in ? c.D[x0 + i] : 0;
      if (MEAN) {
        am[i] = in ? c.A_ms[x0 + i] : 0;
        wm[i] = in ? c.W_ms[x0 + i] : 0;
      } else {
        a[i] = in ? c.A[x0 + i] : 0;
        w[i] = in ? c.W[x0 + i] : 0;
      }
    }
  }
  int m = l0 <= 0xffffffffll ? (int)((uint32_t)l0 - fm.div((uint32_t)l0) * (uint32_t)M)
                             : (int)(l0 % M);
  T rv[4];
  uint8_t cv[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    bool idle;
    if (MEAN) {
      idle = (p[i] | d[i]) == 0 && (am[i] | wm[i]) == 0;
      rv[i] = idle ? idle_raw((T)0)
                   : raw_tss_mean<T>(p[i], d[i], am[i], wm[i], dt, (T)tab.win[s], w_p[m], w_q[m]);
    } else {
      idle = (p[i] | d[i] | a[i] | w[i]) == 0;
      rv[i] = idle ? idle_raw((T)0) : raw_tss<T>(p[i], d[i], a[i], w[i], dt, w_p[m], w_q[m]);
    }
    cv[i] = idle ? kIdle : kNom;
    if (++m == M) m = 0;
  }
  if (v4) {
#pragma unroll
    for (int i = 0; i < 4; ++i) raw[x0 + i] = rv[i];
    *reinterpret_cast<uchar4*>(cls + x0) = make_uchar4(cv[0], cv[1], cv[2], cv[3]);
  } else {
#pragma unroll
    for (int i = 0; i < 4; ++i)
      if (l0 + i < n) {
        raw[x0 + i] = rv[i];
        cls[x0 + i] = cv[i];
      }
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

// Run windows [k0, k1) of model m exactly from (S, init), writing S and, with
// `with_z`, Z and the region (idle windows keep their class). With `verify`,
// stop at the first window whose new S equals the stored one with the same
// init state: from there the stored trajectory is the one this start produces.
// Returns true if it stopped early.
template <class T, bool WRITE = true>
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
      if (!WRITE) continue;
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

// ---- non-idle windows per (chunk, model) ----------------------------------
// One CTA per chunk: its windows are consecutive rows of [K][M], read 16 bytes
// at a time; idle windows are counted per model in shared memory.
template <class T>
__global__ void __launch_bounds__(256)
k_active(const __grid_constant__ SeriesTable<T> tab, FastDiv fm, const uint8_t* __restrict__ cls,
         int32_t* __restrict__ active) {
  extern __shared__ int32_t s_idle[];
  const int seg = blockIdx.x;
  const int s = series_of_seg(tab, seg);
  const int M = tab.M, L = tab.seg_len[s];
  const int64_t k0 = (int64_t)(seg - tab.seg_base[s]) * L, k1 = min64(k0 + L, tab.K[s]);
  for (int m = threadIdx.x; m < M; m += blockDim.x) s_idle[m] = 0;
  __syncthreads();
  const uint8_t* base = cls + tab.off[s] + (size_t)k0 * M;
  const uint32_t n = (uint32_t)((k1 - k0) * M);
  // bytes before the first 16-byte boundary, then whole 16-byte words, then the rest
  const uint32_t head = min(n, (uint32_t)((16 - ((uintptr_t)base & 15)) & 15));
  const uint32_t n16 = (n - head) / 16;
  auto count = [&](uint32_t i, uint8_t v) {
    if (v == kIdle) atomicAdd(&s_idle[i - fm.div(i) * (uint32_t)M], 1);
  };
  for (uint32_t i = threadIdx.x; i < head; i += blockDim.x) count(i, base[i]);
  const uint4* q = reinterpret_cast<const uint4*>(base + head);
  for (uint32_t w = threadIdx.x; w < n16; w += blockDim.x) {
    const uint4 v = q[w];
    const uint32_t ws[4] = {v.x, v.y, v.z, v.w};
    // a word with no idle byte needs no per-byte work
    bool any = false;
#pragma unroll
    for (int h = 0; h < 4; ++h) any |= __vcmpeq4(ws[h], kIdle * 0x01010101u) != 0;
    if (!any) continue;
    const uint32_t i0 = head + 16 * w;
#pragma unroll
    for (int h = 0; h < 4; ++h)
#pragma unroll
      for (int j = 0; j < 4; ++j) count(i0 + 4 * h + j, (uint8_t)(ws[h] >> (8 * j)));
  }
  for (uint32_t i = head + 16 * n16 + threadIdx.x; i < n; i += blockDim.x) count(i, base[i]);
  __syncthreads();
  const int rows = (int)(n / (uint32_t)M);
  for (int m = threadIdx.x; m < M; m += blockDim.x)
    active[(size_t)seg * M + m] = rows - s_idle[m];
}

// ---- pass 1: burn-in and chunk run, one thread per (chunk, model) ----------
// Each thread streams its model's windows through its own slots of a shared
// memory ring with asynchronous copies (cp.async, kStages groups of kBlk
// windows in flight), so the dependent chain reads shared memory while the
// next windows are on their way.
constexpr int kEmaThreads = 32;    // few chains in all: spread them over every SM
constexpr int kBlk = 16;           // windows per copy group
constexpr int kStages = 8;         // copy groups in flight
constexpr int kRingStride = 64;    // chunk and burn-in lengths are multiples of this
constexpr int kMaxBurn = 16384;    // burn-in cap (tiny alpha: the in-order pass repairs)
constexpr int64_t kActiveMinCells = 1 << 22;   // series cells from which burn-ins skip idle chunks
constexpr int64_t kEmaChains = 32768;         // (chunk, model) chains a long table is cut into

template <int BYTES>
__device__ __forceinline__ void cp_async(void* smem, const void* gmem) {
  const unsigned sa = (unsigned)__cvta_generic_to_shared(smem);
  asm volatile("cp.async.ca.shared.global [%0], [%1], %2;\n" ::"r"(sa), "l"(gmem), "n"(BYTES)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;\n" ::: "memory");
}
template <int N> __device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory");
}

// One group of kBlk windows of the chain, read from its ring stage. FULL: all
// kBlk windows exist; STARTED: the chain has seen a non-idle window already
// (then the step is branch-free); STORE: write S (and Z, regions with WITHZ).
template <class T, bool FULL, bool STARTED, bool STORE, bool WITHZ>
__device__ __forceinline__ void ema_group(const T* src, int n, const ModelParams<T>& q, T& S,
                                          int& init, T*& sp, int M, T* S_out, T* Z_out,
                                          uint8_t* cls) {
  T r[kBlk];
#pragma unroll
  for (int j = 0; j < kBlk; ++j) r[j] = src[j * kEmaThreads];
#pragma unroll
  for (int j = 0; j < kBlk; ++j) {
    if (!FULL && j >= n) break;
    const bool idle = is_idle_raw(r[j]);
    if (STARTED) {
      const T nxt = add_rn(mul_rn(q.a, r[j]), mul_rn(q.b, S));
      S = idle ? S : nxt;
    } else if (!idle) {
      S = init ? add_rn(mul_rn(q.a, r[j]), mul_rn(q.b, S)) : r[j];
      init = 1;
    }
    if (STORE) {
      const T Sv = (STARTED || init) ? S : (T)0;
      *sp = Sv;
      if (WITHZ) {
        const size_t x = (size_t)(sp - S_out);
        const T Z = div_rn(Sv, q.th);
        Z_out[x] = Z;
        if (!idle) cls[x] = Z < q.tc ? kCrit : (Z > q.ts ? kSurp : kNom);
      }
      sp += M;
    }
  }
}

template <class T, bool WITHZ>
__global__ void __launch_bounds__(kEmaThreads)
k_ema(const __grid_constant__ SeriesTable<T> tab, const T* __restrict__ raw, const T* alpha,
      const T* theta, const T* tau_crit, const T* tau_surp, const T* S_carry,
      const uint8_t* init_carry, const int32_t* __restrict__ active, T* __restrict__ b_S,
      int32_t* __restrict__ b_init, T* __restrict__ e_S, int32_t* __restrict__ e_init,
      T* __restrict__ S_out, T* __restrict__ Z_out, uint8_t* __restrict__ cls) {
  __shared__ T ring[kStages * kBlk * kEmaThreads];
  const int M = tab.M;
  const int lane = threadIdx.x;
  const int64_t t = (int64_t)blockIdx.x * kEmaThreads + lane;
  if (t >= (int64_t)tab.seg_base[tab.n] * M) return;
  const int m = (int)(t % M);
  const int seg = (int)(t / M);
  const int s = series_of_seg(tab, seg);
  const ModelParams<T> q = load_params(tab, s, m, alpha, theta, tau_crit, tau_surp);
  const int L = tab.seg_len[s];
  const int64_t k0 = (int64_t)(seg - tab.seg_base[s]) * L, k1 = min64(k0 + L, tab.K[s]);
  // burn-in length, in updates (non-idle windows): (1 - alpha)^B <= e^-c, in
  // whole ring strides, with c well past the point where a start error falls
  // below the type's last bit, so that the rounded trajectories have met
  // (c = 28 for float's 6e-8 = e^-16.6, 45 for double's 1.1e-16 = e^-36.7)
  int B = kMaxBurn;
  {
    const float a = (float)q.a;
    const float c = sizeof(T) == 4 ? 28.f : 45.f;
    if (a >= 1.f) B = kRingStride;
    else if (a > 0.f) {
      const float x = c / -log1pf(-a);
      if (x < (float)kMaxBurn) B = (int)x + 1;
    }
    B = (B + kRingStride - 1) / kRingStride * kRingStride;
  }
  // The burn-in runs over spans of windows [sp_lo, sp_hi), ascending. Without
  // activity counts it is the one span [k0 - B, k0). With them (non-idle
  // windows per chunk) it walks back over the preceding chunks until they hold
  // B non-idle windows, leaving out chunks that are wholly idle: an idle window
  // leaves the state as it is, so the trajectory is the same without them,
  // and a burn-in across a long idle stretch still sees enough updates.
  constexpr int kSpans = 8;
  int64_t sp_lo[kSpans], sp_hi[kSpans];
  int nsp = 0;
  bool from_start = false;   // the burn-in covers every update since window 0
  if (active == nullptr) {
    int64_t kb = k0 - B;
    if (kb <= 0) {
      kb = 0;
      from_start = true;
    }
    if (kb < k0) {
      sp_lo[0] = kb;
      sp_hi[0] = k0;
      nsp = 1;
    }
  } else {
    int64_t acc = 0;
    int cb = seg - tab.seg_base[s];
    const int32_t* act = active + (size_t)tab.seg_base[s] * M + m;
    while (acc < B) {
      if (cb == 0) {
        from_start = true;
        break;
      }
      --cb;
      const int na = act[(size_t)cb * M];
      if (na == 0) continue;
      const int64_t hi = (int64_t)(cb + 1) * L;   // chunks before this one are whole
      int64_t lo = (int64_t)cb * L;
      if (na == L && acc + L > B)
        lo = hi - (B - acc + kRingStride - 1) / kRingStride * kRingStride;
      acc += na == L ? hi - lo : na;
      if (nsp > 0 && sp_lo[nsp - 1] == hi) {
        sp_lo[nsp - 1] = lo;
      } else if (nsp < kSpans) {
        sp_lo[nsp] = lo;
        sp_hi[nsp] = hi;
        ++nsp;
      } else {
        break;   // out of spans: a shorter burn-in, repaired by the in-order pass if short
      }
    }
    for (int i = 0; i < nsp / 2; ++i) {
      const int64_t l = sp_lo[i], h = sp_hi[i];
      sp_lo[i] = sp_lo[nsp - 1 - i];
      sp_hi[i] = sp_hi[nsp - 1 - i];
      sp_lo[nsp - 1 - i] = l;
      sp_hi[nsp - 1 - i] = h;
    }
  }
  T S = (T)0;
  int init = 0;
  if (from_start) {   // begin from the true state
    init = (init_carry && init_carry[m]) ? 1 : 0;
    S = init ? S_carry[m] : (T)0;
  }
  const size_t base = (size_t)tab.off[s] + m;
  int burn_grp = 0;
  for (int i = 0; i < nsp; ++i) burn_grp += (int)((sp_hi[i] - sp_lo[i]) / kBlk);
  const int n_grp = burn_grp + (int)((k1 - k0 + kBlk - 1) / kBlk);
  // groups are issued in order: the spans of the burn-in, then the chunk; a
  // group never straddles two spans (span lengths are multiples of kBlk)
  int cur = 0;
  int64_t cur_k = nsp > 0 ? sp_lo[0] : k0, cur_end = nsp > 0 ? sp_hi[0] : k1;
  const size_t step = (size_t)M;
  auto issue = [&](int g) {
    if (g < n_grp) {
      T* dst = ring + (size_t)(g % kStages) * kBlk * kEmaThreads + lane;
      const T* src = raw + base + (size_t)cur_k * M;
      const int64_t left = cur_end - cur_k;
      if (left >= kBlk) {
#pragma unroll
        for (int j = 0; j < kBlk; ++j) cp_async<sizeof(T)>(dst + j * kEmaThreads, src + j * step);
      } else {
#pragma unroll
        for (int j = 0; j < kBlk; ++j)
          if (j < left) cp_async<sizeof(T)>(dst + j * kEmaThreads, src + j * step);
      }
      cur_k += left < kBlk ? left : kBlk;
      if (cur_k >= cur_end && cur < nsp) {
        ++cur;
        cur_k = cur < nsp ? sp_lo[cur] : k0;
        cur_end = cur < nsp ? sp_hi[cur] : k1;
      }
    }
    cp_async_commit();
  };
#pragma unroll
  for (int g = 0; g < kStages - 1; ++g) issue(g);
  T* sp = S_out + base + (size_t)k0 * M;
  auto stage_of = [&](int g) { return ring + (size_t)(g % kStages) * kBlk * kEmaThreads + lane; };
  int g = 0;
  // burn-in: full groups, nothing stored
  for (; g < burn_grp; ++g) {
    issue(g + kStages - 1);
    cp_async_wait<kStages - 1>();
    if (init) ema_group<T, true, true, false, WITHZ>(stage_of(g), kBlk, q, S, init, sp, M, S_out, Z_out, cls);
    else ema_group<T, true, false, false, WITHZ>(stage_of(g), kBlk, q, S, init, sp, M, S_out, Z_out, cls);
  }
  b_S[t] = S;
  b_init[t] = init;
  // the chunk: full groups, then the last (possibly partial) one
  for (; g + 1 < n_grp; ++g) {
    issue(g + kStages - 1);
    cp_async_wait<kStages - 1>();
    if (init) ema_group<T, true, true, true, WITHZ>(stage_of(g), kBlk, q, S, init, sp, M, S_out, Z_out, cls);
    else ema_group<T, true, false, true, WITHZ>(stage_of(g), kBlk, q, S, init, sp, M, S_out, Z_out, cls);
  }
  cp_async_wait<0>();
  {
    const int n = (int)(k1 - (k0 + (int64_t)(g - burn_grp) * kBlk));
    ema_group<T, false, false, true, WITHZ>(stage_of(g), n, q, S, init, sp, M, S_out, Z_out, cls);
  }
  e_S[t] = S;
  e_init[t] = init;
}

// ---- pass 2: boundary check and repair, one warp per (series, model) -------
// Lanes check 32 chunk boundaries at a time. A chunk whose burn-in state
// differs from its predecessor's end state is run again from that end until its
// new trajectory meets the stored one; first as a dry run, so that a chunk is
// rewritten only when every chunk before it keeps its end state. A chunk whose
// re-run never meets its stored trajectory changes its end state, and from the
// next chunk on the boundaries are walked in order by one lane.
template <class T>
__global__ void k_resolve(const __grid_constant__ SeriesTable<T> tab, const T* __restrict__ raw,
                          const T* alpha, const T* theta, const T* tau_crit, const T* tau_surp,
                          const T* start_S, const int32_t* start_init, T* end_S,
                          int32_t* end_init, T* S_out, T* Z_out, uint8_t* cls,
                          T* S_carry, uint8_t* init_carry, tre_diag* diag) {
  const int M = tab.M;
  const int w = blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
  if (w >= tab.n * M) return;
  const int lane = threadIdx.x & 31;
  const int s = w / M, m = w % M;
  const int n_seg = tab.seg_base[s + 1] - tab.seg_base[s];
  if (n_seg == 0) return;
  const size_t g0 = (size_t)tab.seg_base[s] * M + m;
  const ModelParams<T> q = load_params(tab, s, m, alpha, theta, tau_crit, tau_surp);
  const bool with_z = theta != nullptr;
  const int L = tab.seg_len[s];
  const size_t base = (size_t)tab.off[s] + m;
  int first_bad = n_seg;   // the in-order walk starts here
  for (int c0 = 1; c0 < n_seg; c0 += 32) {
    const int c = c0 + lane;
    bool bad = false, moved = false;
    T pS = (T)0;
    int pI = 0, sI = 0;
    int64_t k0 = 0, k1 = 0;
    if (c < n_seg) {
      const size_t x = g0 + (size_t)c * M;
      pS = end_S[x - M];
      pI = end_init[x - M];
      sI = start_init[x];
      bad = sI != pI || !same_bits(start_S[x], pS);
      k0 = (int64_t)c * L;
      k1 = min64(k0 + L, tab.K[s]);
    }
    if (bad) {
      T S = pS;
      int init = pI;
      moved = !run_segment<T, false>(base, M, k0, k1, raw, q, S, init, true, sI, S_out, Z_out,
                                     cls, with_z);
    }
    const unsigned mv = __ballot_sync(0xffffffffu, moved);
    const int lim = mv ? c0 + __ffs(mv) - 1 : n_seg;   // predecessors final up to here
    if (bad && c <= lim) {
      T S = pS;
      int init = pI;
      const bool met = run_segment<T>(base, M, k0, k1, raw, q, S, init, true, sI, S_out, Z_out,
                                      cls, with_z);
      if (!met) {
        end_S[g0 + (size_t)c * M] = S;
        end_init[g0 + (size_t)c * M] = init;
      }
      atomicAdd(&diag->ema_resolved, 1ull);
    }
    if (mv) {
      first_bad = lim + 1;
      break;
    }
  }
  __syncwarp();
  if (lane != 0) return;
  const size_t last = g0 + (size_t)(min(first_bad, n_seg) - 1) * M;
  T S = end_S[last];
  int init = end_init[last];
  if (first_bad >= n_seg) {
    if (S_carry) {
      S_carry[m] = S;
      init_carry[m] = (uint8_t)init;
    }
    return;
  }
  for (int q0 = first_bad; q0 < n_seg; q0 += kBatch) {
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
__global__ void __launch_bounds__(kEwThreads)
k_normalize(const __grid_constant__ SeriesTable<T> tab, const __grid_constant__ TilePlan tp,
            FastDiv fm, bool vec, const T* S, const uint8_t* idle_cls, const T* theta,
            const T* tau_crit, T tau_crit_v, const T* tau_surp, T* Z, uint8_t* cls) {
  const int s = prefix_index(tp.tile_base, tab.n, blockIdx.x);
  const int M = tab.M;
  const int64_t n = (int64_t)tab.K[s] * M;
  const int64_t l0 = (int64_t)(blockIdx.x - tp.tile_base[s]) * kTile + 4 * threadIdx.x;
  if (l0 >= n) return;
  const size_t x0 = (size_t)(tab.off[s] + l0);
  const bool v4 = vec && l0 + 4 <= n;
  T sv[4];
  uint8_t ic[4];
  if (v4) {
#pragma unroll
    for (int i = 0; i < 4; ++i) sv[i] = S[x0 + i];
    const uchar4 c4 = *reinterpret_cast<const uchar4*>(idle_cls + x0);
    ic[0] = c4.x; ic[1] = c4.y; ic[2] = c4.z; ic[3] = c4.w;
  } else {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const bool in = l0 + i < n;
      sv[i] = in ? S[x0 + i] : (T)0;
      ic[i] = in ? idle_cls[x0 + i] : kIdle;
    }
  }
  int m = l0 <= 0xffffffffll ? (int)((uint32_t)l0 - fm.div((uint32_t)l0) * (uint32_t)M)
                             : (int)(l0 % M);
  T zv[4];
  uint8_t cv[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const T z = div_rn(sv[i], theta[(size_t)s * M + m]);
    zv[i] = z;
    uint8_t c;
    if (ic[i] == kIdle) c = kIdle;
    else if (z < (tau_crit ? tau_crit[m] : tau_crit_v)) c = kCrit;
    else if (z > tau_surp[m]) c = kSurp;
    else c = kNom;
    cv[i] = c;
    if (++m == M) m = 0;
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    if (!v4 && l0 + i >= n) break;
    if (Z) Z[x0 + i] = zv[i];
    if (cls && !v4) cls[x0 + i] = cv[i];
  }
  if (cls && v4) *reinterpret_cast<uchar4*>(cls + x0) = make_uchar4(cv[0], cv[1], cv[2], cv[3]);
}

// ---- Eq. 3 receiver per window: warp per window ----------------------------
template <class T>
__device__ __forceinline__ void load_quad_z(const T* p, T (&v)[4]);
template <> __device__ __forceinline__ void load_quad_z<float>(const float* p, float (&v)[4]) {
  const float4 q = *reinterpret_cast<const float4*>(p);
  v[0] = q.x; v[1] = q.y; v[2] = q.z; v[3] = q.w;
}
template <> __device__ __forceinline__ void load_quad_z<double>(const double* p, double (&v)[4]) {
  const double2 a = reinterpret_cast<const double2*>(p)[0];
  const double2 c = reinterpret_cast<const double2*>(p)[1];
  v[0] = a.x; v[1] = a.y; v[2] = c.x; v[3] = c.y;
}

// Eq. 3 receiver per window: argmin Z over non-idle models, lowest index on
// ties (the first minimum in index order), -1 when every model is idle. One
// thread per window; with QUAD (M a multiple of 4, 16-byte aligned rows) a
// row is read four models per load, several loads in flight.
template <class T, bool QUAD>
__global__ void __launch_bounds__(256)
k_receiver(int M, int K, const T* __restrict__ Z, const uint8_t* __restrict__ cls,
           int32_t* __restrict__ recv) {
  const int64_t k = (int64_t)blockIdx.x * 256 + threadIdx.x;
  if (k >= K) return;
  const T* z = Z + (size_t)k * M;
  const uint8_t* c = cls + (size_t)k * M;
  int best = -1;
  T bz = (T)0;
  if (QUAD) {
#pragma unroll 4
    for (int m0 = 0; m0 < M; m0 += 4) {
      T zv[4];
      load_quad_z<T>(z + m0, zv);
      const uchar4 c4 = *reinterpret_cast<const uchar4*>(c + m0);
      const uint8_t cv[4] = {c4.x, c4.y, c4.z, c4.w};
#pragma unroll
      for (int i = 0; i < 4; ++i)
        if (cv[i] != kIdle && (best < 0 || zv[i] < bz)) {
          best = m0 + i;
          bz = zv[i];
        }
    }
  } else {
#pragma unroll 4
    for (int m = 0; m < M; ++m) {
      const uint8_t cv = c[m];
      const T zv = z[m];
      if (cv != kIdle && (best < 0 || zv < bz)) {
        best = m;
        bz = zv;
      }
    }
  }
  recv[k] = best;
}

// ---- per-window donor preference order (Sec. IV-B), warp per window ---------
// Donor key: group (idle 0, surplus 1, nominal above the receiver 2), then Z
// descending within surplus and nominal, then index. Keys are distinct, so the
// r-th donor is the smallest key above the (r-1)-th: kRankDonors rounds of a
// warp-wide minimum, each over the models whose key exceeds the last one.
template <class T>
__device__ __forceinline__ bool donor_key_less(int ga, T za, int ia, int gb, T zb, int ib) {
  if (ga != gb) return ga < gb;
  if (ga != 0 && za != zb) return za > zb;
  return ia < ib;
}

template <class T>
__global__ void k_rank(int M, int K, const T* Z, const uint8_t* cls, int32_t* recv,
                       int32_t* donors) {
  const int64_t k = (int64_t)blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
  if (k >= K) return;
  const int lane = threadIdx.x & 31;
  const T* z = Z + (size_t)k * M;
  const uint8_t* c = cls + (size_t)k * M;
  int best = -1;
  T bz = (T)0;
  for (int m = lane; m < M; m += 32) {
    if (c[m] == kIdle) continue;
    const T zm = z[m];
    if (best < 0 || zm < bz) { best = m; bz = zm; }
  }
  for (int o = 16; o > 0; o >>= 1) {
    const int ob = __shfl_xor_sync(0xffffffffu, best, o);
    const T oz = __shfl_xor_sync(0xffffffffu, bz, o);
    if (ob >= 0 && (best < 0 || oz < bz || (oz == bz && ob < best))) { best = ob; bz = oz; }
  }
  if (lane == 0 && recv) recv[k] = best;
  if (!donors) return;
  int32_t* out = donors + (size_t)k * kRankDonors;
  int lg = -1, li = -1;
  T lzv = (T)0;
  int r = 0;
  for (; best >= 0 && r < kRankDonors; ++r) {
    int g = 3, i = -1;
    T zv = (T)0;
    for (int m = lane; m < M; m += 32) {
      if (m == best) continue;
      const uint8_t cm = c[m];
      const T zm = z[m];
      int gm;
      if (cm == kIdle) gm = 0;
      else if (cm == kSurp) gm = 1;
      else if (cm == kNom && zm > bz) gm = 2;
      else continue;
      if (lg >= 0 && !donor_key_less(lg, lzv, li, gm, zm, m)) continue;
      if (i < 0 || donor_key_less(gm, zm, m, g, zv, i)) { g = gm; zv = zm; i = m; }
    }
    for (int o = 16; o > 0; o >>= 1) {
      const int og = __shfl_xor_sync(0xffffffffu, g, o);
      const int oi = __shfl_xor_sync(0xffffffffu, i, o);
      const T oz = __shfl_xor_sync(0xffffffffu, zv, o);
      if (oi >= 0 && (i < 0 || donor_key_less(og, oz, oi, g, zv, i))) { g = og; zv = oz; i = oi; }
    }
    if (i < 0) break;
    if (lane == 0) out[r] = i;
    lg = g; lzv = zv; li = i;
  }
  if (lane >= r && lane < kRankDonors) out[lane] = -1;
}

// Up to 16 models: one thread per window, the row in registers. A donor's
// position is the number of donors with a smaller key; slot j takes the donor
// whose position is j.
template <class T, int MMAX>
__global__ void __launch_bounds__(256)
k_rank_small(int M, int K, const T* __restrict__ Z, const uint8_t* __restrict__ cls,
             int32_t* __restrict__ recv, int32_t* __restrict__ donors) {
  const int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (k >= K) return;
  const T* z = Z + (size_t)k * M;
  const uint8_t* c = cls + (size_t)k * M;
  T zv[MMAX];
  uint8_t cv[MMAX];
#pragma unroll
  for (int m = 0; m < MMAX; ++m) {
    zv[m] = m < M ? z[m] : (T)0;
    cv[m] = m < M ? c[m] : kIdle;
  }
  int best = -1;
  T bz = (T)0;
#pragma unroll
  for (int m = 0; m < MMAX; ++m)
    if (m < M && cv[m] != kIdle && (best < 0 || zv[m] < bz)) { best = m; bz = zv[m]; }
  if (recv) recv[k] = best;
  if (!donors) return;
  int32_t* out = donors + (size_t)k * kRankDonors;
  int g[MMAX];
#pragma unroll
  for (int m = 0; m < MMAX; ++m) {
    int gm = 3;
    if (m < M && m != best && best >= 0) {
      if (cv[m] == kIdle) gm = 0;
      else if (cv[m] == kSurp) gm = 1;
      else if (cv[m] == kNom && zv[m] > bz) gm = 2;
    }
    g[m] = gm;
  }
  int pos[MMAX];
#pragma unroll
  for (int a = 0; a < MMAX; ++a) {
    int r = 0;
#pragma unroll
    for (int b = 0; b < MMAX; ++b)
      if (b != a && g[b] < 3 && donor_key_less(g[b], zv[b], b, g[a], zv[a], a)) ++r;
    pos[a] = g[a] < 3 ? r : kRankDonors;
  }
#pragma unroll
  for (int j = 0; j < kRankDonors; ++j) {
    int d = -1;
#pragma unroll
    for (int a = 0; a < MMAX; ++a) d = pos[a] == j ? a : d;
    out[j] = d;
  }
}

template <class T> TilePlan tile_plan(const SeriesTable<T>& t, int& n_tiles) {
  TilePlan tp;
  n_tiles = 0;
  for (int s = 0; s < t.n; ++s) {
    tp.tile_base[s] = n_tiles;
    n_tiles += (int)(((int64_t)t.K[s] * t.M + kTile - 1) / kTile);
  }
  tp.tile_base[t.n] = n_tiles;
  return tp;
}

// 16-byte accesses need every series to start on a 4-element boundary and
// the arrays on 16-byte ones
template <class T> bool quad_aligned(const SeriesTable<T>& t, std::initializer_list<const void*> ps) {
  for (int s = 0; s < t.n; ++s)
    if (t.off[s] % 4) return false;
  for (const void* p : ps)
    if (p && ((uintptr_t)p % 16)) return false;
  return true;
}

template <class T> int64_t total_elems(const SeriesTable<T>& t) {
  int64_t n = 0;
  for (int s = 0; s < t.n; ++s) n += (int64_t)t.K[s] * t.M;
  return n;
}

}  // namespace

template <class T> int series_segments(SeriesTable<T>& t) {
  int total = 0;
  int64_t cells = 0;
  for (int s = 0; s < t.n; ++s) cells += (int64_t)t.K[s] * t.M;
  for (int s = 0; s < t.n; ++s) {
    const int K = t.K[s];
    // chunks of 256 windows, longer for very long series (to bound the count)
    // and for large tables: about kEmaChains chains keep the GPU busy, and
    // longer chunks re-read fewer windows in their burn-ins; a multiple of the
    // smoothing pass's ring stride
    int L = 256;
    int64_t need = std::max<int64_t>((K + 2047) / 2048, cells / kEmaChains);
    if (need > L) L = (int)((need + kRingStride - 1) / kRingStride * kRingStride);
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
  w.start_S = a.take<T>(n);
  w.start_init = a.take<int32_t>(n);
  w.end_S = a.take<T>(n);
  w.end_init = a.take<int32_t>(n);
  w.active = a.take<int32_t>(n);
}

template <class T> int score_launches(const SeriesTable<T>& tab) {
  return (total_elems(tab) >= kActiveMinCells ? 1 : 0) + 3;
}

template <class T>
cudaError_t launch_score(const SeriesTable<T>& tab, const int32_t* P, const int32_t* D,
                         const int32_t* A, const int32_t* W, const T* w_p, const T* w_q,
                         const T* alpha, const T* theta, const T* tau_crit, const T* tau_surp,
                         T* S_carry, uint8_t* init_carry, T* S, T* Z, uint8_t* cls,
                         ScoreWs<T>& w, tre_diag* diag, cudaStream_t s, const int64_t* A_ms,
                         const int64_t* W_ms) {
  const int M = tab.M;
  const int n_seg = tab.seg_base[tab.n];
  if (n_seg > w.cap_seg) return cudaErrorInvalidValue;
  if ((A_ms == nullptr) != (W_ms == nullptr)) return cudaErrorInvalidValue;
  const int64_t total = total_elems(tab);
  if (total == 0) return cudaSuccess;
  const Counts c{P, D, A, W, A_ms, W_ms};
  int n_tiles = 0;
  const TilePlan tp = tile_plan(tab, n_tiles);
  if (A_ms) {
    const bool vec = quad_aligned(tab, {P, D, A_ms, W_ms, w.raw, cls});
    k_raw<T, true><<<n_tiles, kEwThreads, 0, s>>>(tab, tp, FastDiv(M), vec, c, w_p, w_q, w.raw,
                                                  cls);
  } else {
    const bool vec = quad_aligned(tab, {P, D, A, W, w.raw, cls});
    k_raw<T, false><<<n_tiles, kEwThreads, 0, s>>>(tab, tp, FastDiv(M), vec, c, w_p, w_q, w.raw,
                                                   cls);
  }
  const int64_t segs = (int64_t)n_seg * M;
  const unsigned g = (unsigned)((segs + kEmaThreads - 1) / kEmaThreads);
  // activity counts for the burn-ins where the series are long enough that
  // idle stretches would otherwise send chunks to the in-order pass, and the
  // extra pass over the classes is small beside the smoothing
  const int32_t* active = nullptr;
  if (total >= kActiveMinCells) {
    k_active<T><<<n_seg, 256, (size_t)M * sizeof(int32_t), s>>>(tab, FastDiv(M), cls, w.active);
    active = w.active;
  }
  if (theta)
    k_ema<T, true><<<g, kEmaThreads, 0, s>>>(tab, w.raw, alpha, theta, tau_crit, tau_surp,
                                             S_carry, init_carry, active, w.start_S,
                                             w.start_init, w.end_S, w.end_init, S, Z, cls);
  else
    k_ema<T, false><<<g, kEmaThreads, 0, s>>>(tab, w.raw, alpha, theta, tau_crit, tau_surp,
                                              S_carry, init_carry, active, w.start_S,
                                              w.start_init, w.end_S, w.end_init, S, Z, cls);
  const int warps = tab.n * M;
  k_resolve<T><<<(warps + 1) / 2, 64, 0, s>>>(tab, w.raw, alpha, theta, tau_crit, tau_surp,
                                                w.start_S, w.start_init, w.end_S, w.end_init,
                                                S, Z, cls, S_carry, init_carry, diag);
  return cudaGetLastError();
}

template <class T>
cudaError_t launch_normalize(const SeriesTable<T>& tab, const T* S, const uint8_t* idle_cls,
                             const T* theta, const T* tau_crit, T tau_crit_v, const T* tau_surp,
                             T* Z, uint8_t* cls, cudaStream_t s) {
  const int64_t total = total_elems(tab);
  if (total == 0) return cudaSuccess;
  int n_tiles = 0;
  const TilePlan tp = tile_plan(tab, n_tiles);
  const bool vec = quad_aligned(tab, {S, idle_cls, Z, cls});
  k_normalize<T><<<n_tiles, kEwThreads, 0, s>>>(tab, tp, FastDiv(tab.M), vec, S, idle_cls, theta,
                                                tau_crit, tau_crit_v, tau_surp, Z, cls);
  return cudaGetLastError();
}

template <class T>
cudaError_t launch_receiver(int M, int K, const T* Z, const uint8_t* cls, int32_t* recv,
                            cudaStream_t s) {
  if (K == 0) return cudaSuccess;
  const unsigned g = (unsigned)((K + 255) / 256);
  if (M % 4 == 0 && (((uintptr_t)Z | (uintptr_t)cls) & 15) == 0)
    k_receiver<T, true><<<g, 256, 0, s>>>(M, K, Z, cls, recv);
  else
    k_receiver<T, false><<<g, 256, 0, s>>>(M, K, Z, cls, recv);
  return cudaGetLastError();
}

template <class T>
cudaError_t launch_rank(int M, int K, const T* Z, const uint8_t* cls, int32_t* recv,
                        int32_t* donors, cudaStream_t s) {
  if (K == 0 || (!recv && !donors)) return cudaSuccess;
  const unsigned thread_blocks = (unsigned)((K + 255) / 256);
  if (M <= 8)
    k_rank_small<T, 8><<<thread_blocks, 256, 0, s>>>(M, K, Z, cls, recv, donors);
  else if (M <= 16)
    k_rank_small<T, 16><<<thread_blocks, 256, 0, s>>>(M, K, Z, cls, recv, donors);
  else
    k_rank<T><<<(unsigned)((K + 7) / 8), 256, 0, s>>>(M, K, Z, cls, recv, donors);
  return cudaGetLastError();
}

#define TRE_INST(T)                                                                               \
  template int series_segments<T>(SeriesTable<T>&);                                               \
  template int score_launches<T>(const SeriesTable<T>&);                                          \
  template void score_ws_layout<T>(Arena&, int, int64_t, int, ScoreWs<T>&);                       \
  template cudaError_t launch_score<T>(const SeriesTable<T>&, const int32_t*, const int32_t*,      \
                                       const int32_t*, const int32_t*, const T*, const T*,         \
                                       const T*, const T*, const T*, const T*, T*, uint8_t*, T*,   \
                                       T*, uint8_t*, ScoreWs<T>&, tre_diag*, cudaStream_t,         \
                                       const int64_t*, const int64_t*);                            \
  template cudaError_t launch_normalize<T>(const SeriesTable<T>&, const T*, const uint8_t*,        \
                                           const T*, const T*, T, const T*, T*, uint8_t*,          \
                                           cudaStream_t);                                          \
  template cudaError_t launch_receiver<T>(int, int, const T*, const uint8_t*, int32_t*,            \
                                          cudaStream_t);                                          \
  template cudaError_t launch_rank<T>(int, int, const T*, const uint8_t*, int32_t*, int32_t*,      \
                                      cudaStream_t);
TRE_INST(float)
TRE_INST(double)

}  // namespace tre
