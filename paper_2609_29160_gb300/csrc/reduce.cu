// Window reduction of request telemetry: the inputs of Eq. 1 (Sec. III-A)
// collected as window deltas of prompt/decode token counters plus running and
// waiting gauges (Sec. V-B).
//
// Request records are sorted by arrival in practice, so the records of one CTA
// touch a short run of windows: the CTA accumulates into a shared-memory copy
// of those rows and flushes them once; targets outside the staged rows (long
// queue waits, unsorted input) go straight to global atomics. All arithmetic is
// integer and all atomics are integer adds, so the result does not depend on
// the order of the records.
#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace tre {
namespace {

constexpr int kThreads = 256;
constexpr int kStageBytes = 32 * 1024;   // start-side staging per CTA
constexpr int kSpill = 32;  // staged rows beyond the CTA's arrival range

// window of a millisecond time (int32 range), clamped to [0, K]
__device__ __forceinline__ int64_t win_clamp(int64_t t, const FastDiv& fd, int K) {
  if (t < 0) return 0;
  const int64_t b = fd.div((uint32_t)t);
  return b > K ? K : b;
}

template <class V>
__device__ __forceinline__ void stage_add(V* s, V* g, int64_t k, int64_t k_lo, int used, int M,
                                          int m, V v) {
  const int64_t rel = k - k_lo;
  if (rel >= 0 && rel < used) atomicAdd(&s[rel * M + m], v);
  else atomicAdd(&g[k * M + m], v);
}

// --------------------------------------------------------------------------
// request records -> P, D, gauge diffs, optional packed SLO counts, for a
// batch of traces on one grid (CTAs [cta_base[t], cta_base[t+1]) take trace t)
// --------------------------------------------------------------------------
constexpr int kMaxTraces = 64;
struct ReqBatch {
  int n;
  ReqCols cols[kMaxTraces];
  int64_t per_cta[kMaxTraces];
  int32_t cta_base[kMaxTraces + 1];
};

// Targets of one record fall in two places: the arrival side (the waiting
// gauge's +1 and the SLO counts at the arrival window) moves with the arrival
// order of the records, the start side (waiting -1 and running +1 at the
// start, prompt and decode tokens, running -1 at the end) with each model's
// FCFS start order. A CTA stages the arrival side over the windows its records
// arrive in, and the start side per model over a run of windows beginning at
// that model's earliest start among the CTA's records. Targets outside both
// go to global atomics.
struct Stage {
  int32_t *aW;                  // arrival side: [near_rows][M]
  unsigned long long* aS;       // arrival side SLO counts: [near_rows][M]
  int32_t *fP, *fD, *fA, *fW;   // start side: [M][far_rows]
  int32_t* far_lo;              // [M]
  int32_t* slo_lim;             // [M]
};

template <bool SLO>
__global__ void __launch_bounds__(kThreads)
k_reduce_requests(const __grid_constant__ ReqBatch bt, int M, int win, FastDiv fd, int K,
                  int near_rows, int far_rows, int32_t* __restrict__ P0, int32_t* __restrict__ D0,
                  int32_t* __restrict__ dA0, int32_t* __restrict__ dW0,
                  unsigned long long* __restrict__ slo0, const int32_t* __restrict__ slo_ms,
                  tre_diag* diag) {
  extern __shared__ unsigned long long smem[];
  int t = 0;
  while (t + 1 < bt.n && bt.cta_base[t + 1] <= (int)blockIdx.x) ++t;
  const ReqCols& r = bt.cols[t];
  const int64_t per_cta = bt.per_cta[t];
  const size_t cells0 = (size_t)K * M, cells1 = (size_t)(K + 1) * M;
  int32_t* P = P0 + t * cells0;
  int32_t* D = D0 + t * cells0;
  int32_t* dA = dA0 + t * cells1;
  int32_t* dW = dW0 + t * cells1;
  unsigned long long* slo = SLO ? slo0 + t * cells0 : nullptr;
  const int64_t i0 = (int64_t)(blockIdx.x - bt.cta_base[t]) * per_cta;
  const int64_t i1 = min(r.n, i0 + per_cta);
  if (i0 >= i1) return;
  const int64_t span = (int64_t)K * win;
  const int64_t k_lo = win_clamp(r.t_arr[i0], fd, K);
  const int64_t k_hi = win_clamp(r.t_arr[i1 - 1], fd, K);
  const int64_t need = (k_hi >= k_lo ? k_hi - k_lo + 1 : 1) + 1;
  const int used = (int)min64(near_rows, need);
  Stage st;
  st.aS = smem;
  st.aW = reinterpret_cast<int32_t*>(smem + (SLO ? (size_t)near_rows * M : 0));
  st.fP = st.aW + (size_t)near_rows * M;
  st.fD = st.fP + (size_t)far_rows * M;
  st.fA = st.fD + (size_t)far_rows * M;
  st.fW = st.fA + (size_t)far_rows * M;
  st.far_lo = st.fW + (size_t)far_rows * M;
  st.slo_lim = st.far_lo + M;
  const int ncell = used * M, fcell = far_rows * M;
  for (int c = threadIdx.x; c < ncell; c += kThreads) {
    st.aW[c] = 0;
    if (SLO) st.aS[c] = 0;
  }
  for (int c = threadIdx.x; c < fcell; c += kThreads) {
    st.fP[c] = 0; st.fD[c] = 0; st.fA[c] = 0; st.fW[c] = 0;
  }
  for (int m = threadIdx.x; m < M; m += kThreads) {
    st.far_lo[m] = 0x7fffffff;
    if (SLO) st.slo_lim[m] = slo_ms[m];
  }
  __syncthreads();
  // each model's earliest start window among this CTA's records
  for (int64_t i = i0 + threadIdx.x; i < i1; i += kThreads) {
    const int m = r.model[i];
    const int32_t ts = r.t_start[i];
    if (m >= 0 && m < M && ts >= 0) atomicMin(&st.far_lo[m], (int32_t)win_clamp(ts, fd, K));
  }
  __syncthreads();

  // arrival-side target (waiting +1, SLO counts)
  auto near_add = [&](auto* s_arr, auto* g_arr, int64_t k, int m, auto v) {
    const int64_t rel = k - k_lo;
    if (rel >= 0 && rel < used) atomicAdd(&s_arr[rel * M + m], v);
    else atomicAdd(&g_arr[k * M + m], v);
  };
  // start-side target of model m
  auto far_add = [&](int32_t* s_arr, int32_t* g_arr, int64_t k, int m, int32_t v) {
    const int64_t rel = k - st.far_lo[m];
    if (rel >= 0 && rel < far_rows) atomicAdd(&s_arr[m * far_rows + rel], v);
    else atomicAdd(&g_arr[k * M + m], v);
  };

  unsigned long long n_range = 0, n_model = 0, n_order = 0;
  int32_t nx[7];
  auto load_rec = [&](int64_t i) {
    if (i < i1) {
      nx[0] = r.model[i];
      nx[1] = r.t_arr[i];
      nx[2] = r.t_start[i];
      nx[3] = r.t_first[i];
      nx[4] = r.t_end[i];
      nx[5] = r.L_in[i];
      nx[6] = r.L_out[i];
    }
  };
  load_rec(i0 + threadIdx.x);
  for (int64_t i = i0 + threadIdx.x; i < i1; i += kThreads) {
    const int m = nx[0];
    const int64_t ta = nx[1], ts = nx[2], tf = nx[3], te = nx[4];
    const int32_t L_in = nx[5], L = nx[6];
    load_rec(i + kThreads);
    if (m < 0 || m >= M) { ++n_model; continue; }
    if (ta < 0 || ta >= span) { ++n_range; continue; }
    if (!(ta <= ts && ts <= tf && tf <= te) || L_in < 0 || L < 1) { ++n_order; continue; }

    const int64_t ba = fd.div((uint32_t)ta);
    const int64_t bs = win_clamp(ts, fd, K), be = win_clamp(te, fd, K);
    if (ba != bs) {
      near_add(st.aW, dW, ba, m, (int32_t)1);
      far_add(st.fW, dW, bs, m, -1);
    }
    if (bs != be) {
      far_add(st.fA, dA, bs, m, 1);
      far_add(st.fA, dA, be, m, -1);
    }
    if (SLO) {
      const unsigned long long met = (tf - ta <= (int64_t)st.slo_lim[m]) ? 1ull : 0ull;
      near_add(st.aS, slo, ba, m, 1ull + (met << 32));
    }
    if (tf < span) {
      const int64_t kf = fd.div((uint32_t)tf);
      // prompt tokens, all at the first-token time
      if (L_in) far_add(st.fP, P, kf, m, L_in);
      // decode tokens: N(T) = tokens emitted before T; D[k] = N((k+1)w) - N(kw)
      const int64_t ke_raw = fd.div((uint32_t)te);
      if (L == 1 || ke_raw == kf) {
        far_add(st.fD, D, kf, m, L);
      } else {
        const unsigned long long dur = (unsigned long long)(te - tf);
        const unsigned long long Lm1 = (unsigned long long)(L - 1);
        unsigned long long q, rem;
        // N at the first window boundary after tf: ceil((T - tf)(L-1)/dur)
        divmod((unsigned long long)((kf + 1) * win - tf) * Lm1, (uint32_t)dur, q, rem);
        const int32_t n1 = (int32_t)(q + (rem != 0));
        far_add(st.fD, D, kf, m, n1);
        if (ke_raw == kf + 1) {
          if (kf + 1 < K) far_add(st.fD, D, kf + 1, m, L - n1);
        } else {
          const int64_t ke = min64(ke_raw, K - 1);
          unsigned long long qs, rs;
          divmod((unsigned long long)win * Lm1, (uint32_t)dur, qs, rs);
          q += qs;
          rem += rs;
          if (rem >= dur) { rem -= dur; q += 1; }
          unsigned long long prevN = (unsigned long long)n1;
          for (int64_t k = kf + 1; k <= ke; ++k) {
            unsigned long long N;
            if ((k + 1) * win > te) {
              N = (unsigned long long)L;
            } else {
              N = q + (rem != 0);
              q += qs;
              rem += rs;
              if (rem >= dur) { rem -= dur; q += 1; }
            }
            const int32_t cnt = (int32_t)(N - prevN);
            if (cnt) far_add(st.fD, D, k, m, cnt);
            prevN = N;
          }
        }
      }
    }
  }
  __syncthreads();
  for (int c = threadIdx.x; c < ncell; c += kThreads) {
    const int64_t k = k_lo + c / M;
    const size_t g = (size_t)k * M + (c % M);
    if (k < K && SLO && st.aS[c]) atomicAdd(&slo[g], st.aS[c]);
    if (k <= K && st.aW[c]) atomicAdd(&dW[g], st.aW[c]);
  }
  for (int c = threadIdx.x; c < fcell; c += kThreads) {
    const int m = c / far_rows;
    const int lo = st.far_lo[m];
    if (lo == 0x7fffffff) continue;
    const int64_t k = (int64_t)lo + (c % far_rows);
    const size_t g = (size_t)k * M + m;
    if (k < K) {
      if (st.fP[c]) atomicAdd(&P[g], st.fP[c]);
      if (st.fD[c]) atomicAdd(&D[g], st.fD[c]);
    }
    if (k <= K) {
      if (st.fA[c]) atomicAdd(&dA[g], st.fA[c]);
      if (st.fW[c]) atomicAdd(&dW[g], st.fW[c]);
    }
  }
  warp_add_counter(&diag->dropped_range, n_range);
  warp_add_counter(&diag->dropped_model, n_model);
  warp_add_counter(&diag->dropped_order, n_order);
}

// SLO counts alone (for calibration from records whose counts exist already)
__global__ void __launch_bounds__(kThreads)
k_slo_requests(ReqCols r, int M, int win, int K, unsigned long long* __restrict__ slo,
               const int32_t* __restrict__ slo_ms) {
  const int64_t span = (int64_t)K * win;
  for (int64_t i = (int64_t)blockIdx.x * kThreads + threadIdx.x; i < r.n;
       i += (int64_t)gridDim.x * kThreads) {
    const int m = r.model[i];
    const int64_t ta = r.t_arr[i], ts = r.t_start[i], tf = r.t_first[i], te = r.t_end[i];
    if (m < 0 || m >= M || ta < 0 || ta >= span) continue;
    if (!(ta <= ts && ts <= tf && tf <= te) || r.L_in[i] < 0 || r.L_out[i] < 1) continue;
    const unsigned long long met = (tf - ta <= (int64_t)slo_ms[m]) ? 1ull : 0ull;
    atomicAdd(&slo[(size_t)(ta / win) * M + m], 1ull + (met << 32));
  }
}

// --------------------------------------------------------------------------
// token events -> P, D and per-request first/last tick
// --------------------------------------------------------------------------

// exact floor(t * 1000) of a float seconds value, as integer arithmetic on its
// significand; returns false for NaN, infinities and negative values (a
// negative zero is tick 0)
__device__ __forceinline__ bool ms_tick(float t, int64_t span, int64_t& tick) {
  const uint32_t b = __float_as_uint(t);
  if ((b & 0x7fffffffu) == 0) { tick = 0; return span > 0; }
  if (b >> 31) return false;
  const uint32_t ex = (b >> 23) & 0xffu;
  if (ex == 0xffu) return false;
  const unsigned long long mant = ex ? ((b & 0x7fffffu) | 0x800000u) : (b & 0x7fffffu);
  const int e = (ex ? (int)ex : 1) - 150;  // t = mant * 2^e
  const unsigned long long prod = mant * 1000ull;
  unsigned long long v;
  if (e >= 0) {
    if (e > 29) return false;                 // beyond any int32 millisecond
    v = prod << e;
  } else {
    v = (-e >= 64) ? 0ull : (prod >> (-e));
  }
  if ((long long)v >= span) return false;
  tick = (int64_t)v;
  return true;
}

__global__ void __launch_bounds__(kThreads)
k_reduce_events(EvCols e, int M, int win, FastDiv fd, int K, int64_t per_cta, int rows,
                int32_t* __restrict__ P, int32_t* __restrict__ D, int32_t* __restrict__ first,
                int32_t* __restrict__ last, tre_diag* diag) {
  extern __shared__ unsigned long long smem[];
  const int64_t i0 = (int64_t)blockIdx.x * per_cta;
  const int64_t i1 = min(e.n, i0 + per_cta);
  if (i0 >= i1) return;
  const int64_t span = (int64_t)K * win;
  int64_t t0, t1;
  const int64_t k_lo = ms_tick(e.t_s[i0], span, t0) ? fd.div((uint32_t)t0) : 0;
  const int64_t k_hi = ms_tick(e.t_s[i1 - 1], span, t1) ? fd.div((uint32_t)t1) : K;
  const int64_t need = (k_hi >= k_lo ? k_hi - k_lo + 1 : 1) + kSpill;
  const int used = (int)min64(rows, need);
  const int cells = used * M;
  int32_t* sP = reinterpret_cast<int32_t*>(smem);
  int32_t* sD = sP + (size_t)rows * M;
  for (int c = threadIdx.x; c < cells; c += kThreads) { sP[c] = 0; sD[c] = 0; }
  __syncthreads();

  const unsigned full = 0xffffffffu;
  const int lane = threadIdx.x & 31;
  unsigned long long n_range = 0, n_model = 0, n_order = 0;
  for (int64_t base = i0; base < i1; base += kThreads) {
    const int64_t i = base + threadIdx.x;
    bool ok = false;
    int64_t tick = 0;
    int rq = 0;
    if (i < i1) {
      const int m = e.model[i];
      rq = e.req[i];
      const float ts = e.t_s[i];
      const uint8_t ph = e.phase[i];
      if (m < 0 || m >= M || rq < 0 || rq >= e.n_req || e.req_model[rq] != m) {
        ++n_model;
      } else if (!ms_tick(ts, span, tick)) {
        ++n_range;
      } else if (ph > 1) {
        ++n_order;
      } else {
        ok = true;
        const int64_t k = fd.div((uint32_t)tick);
        stage_add<int32_t>(ph == 0 ? sP : sD, ph == 0 ? P : D, k, k_lo, used, M, m, 1);
      }
    }
    // first / last tick per request, one atomic per run of equal request ids
    const unsigned active = __ballot_sync(full, ok);
    if (ok) {
      const unsigned grp = __match_any_sync(active, rq);
      const int t32 = (int)tick;
      const int mn = __reduce_min_sync(grp, t32);
      const int mx = __reduce_max_sync(grp, t32);
      if (lane == __ffs(grp) - 1) {
        atomicMin(&first[rq], mn);
        atomicMax(&last[rq], mx);
      }
    }
  }
  __syncthreads();
  for (int c = threadIdx.x; c < cells; c += kThreads) {
    const int64_t k = k_lo + c / M;
    if (k >= K) continue;
    const size_t g = (size_t)k * M + (c % M);
    if (sP[c]) atomicAdd(&P[g], sP[c]);
    if (sD[c]) atomicAdd(&D[g], sD[c]);
  }
  warp_add_counter(&diag->dropped_range, n_range);
  warp_add_counter(&diag->dropped_model, n_model);
  warp_add_counter(&diag->dropped_order, n_order);
}

__global__ void k_fill_first_last(int32_t* first, int32_t* last, int64_t n) {
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    first[i] = 0x7fffffff;
    last[i] = -1;
  }
}

// per request with at least one valid event: waiting on [t_arr, first),
// running on [first, last)
__global__ void __launch_bounds__(kThreads)
k_event_gauges(EvCols e, int M, FastDiv fd, int K, const int32_t* __restrict__ first,
               const int32_t* __restrict__ last, int32_t* __restrict__ dA,
               int32_t* __restrict__ dW, tre_diag* diag) {
  unsigned long long n_order = 0;
  for (int64_t r = (int64_t)blockIdx.x * kThreads + threadIdx.x; r < e.n_req;
       r += (int64_t)gridDim.x * kThreads) {
    const int64_t lt = last[r];
    if (lt < 0) continue;
    const int64_t ft = first[r];
    const int m = e.req_model[r];
    const int64_t ta = e.req_t_arr[r];
    if (!(ta >= 0 && ta <= ft)) { ++n_order; continue; }
    const int64_t ba = win_clamp(ta, fd, K), bf = win_clamp(ft, fd, K), bl = win_clamp(lt, fd, K);
    if (ba != bf) {
      atomicAdd(&dW[ba * M + m], 1);
      atomicAdd(&dW[bf * M + m], -1);
    }
    if (bf != bl) {
      atomicAdd(&dA[bf * M + m], 1);
      atomicAdd(&dA[bl * M + m], -1);
    }
  }
  warp_add_counter(&diag->dropped_order, n_order);
}

__global__ void __launch_bounds__(kThreads)
k_slo_events(EvCols e, int M, int win, int K, unsigned long long* __restrict__ slo,
             const int32_t* __restrict__ slo_ms) {
  const int64_t span = (int64_t)K * win;
  for (int64_t r = (int64_t)blockIdx.x * kThreads + threadIdx.x; r < e.n_req;
       r += (int64_t)gridDim.x * kThreads) {
    const int m = e.req_model[r];
    const int64_t ta = e.req_t_arr[r];
    if (m < 0 || m >= M || ta < 0 || ta >= span) continue;
    const unsigned long long met = (e.req_ttft[r] <= slo_ms[m]) ? 1ull : 0ull;
    atomicAdd(&slo[(size_t)(ta / win) * M + m], 1ull + (met << 32));
  }
}

// --------------------------------------------------------------------------
// gauge scan: inclusive prefix over windows of the diff arrays, per model.
// Segment = (chunk of rows, model); adjacent threads take adjacent models so
// each row is read coalesced.
// --------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads)
k_scan_partials(int M, int K, int L, int n_chunks, const int32_t* __restrict__ dA,
                const int32_t* __restrict__ dW, int32_t* __restrict__ pA,
                int32_t* __restrict__ pW) {
  const int64_t t = (int64_t)blockIdx.x * kThreads + threadIdx.x;
  if (t >= (int64_t)n_chunks * M) return;
  dA += (size_t)blockIdx.y * (K + 1) * M;
  dW += (size_t)blockIdx.y * (K + 1) * M;
  pA += (size_t)blockIdx.y * n_chunks * M;
  pW += (size_t)blockIdx.y * n_chunks * M;
  const int m = (int)(t % M);
  const int c = (int)(t / M);
  const int64_t r0 = (int64_t)c * L, r1 = min64(r0 + L, K);
  int32_t a = 0, w = 0;
  for (int64_t k = r0; k < r1; ++k) {
    a += dA[k * M + m];
    w += dW[k * M + m];
  }
  pA[t] = a;
  pW[t] = w;
}

// exclusive scan over chunks, one warp per model (n_chunks <= 1024)
__global__ void k_scan_chunks(int M, int n_chunks, int32_t* __restrict__ pA,
                              int32_t* __restrict__ pW) {
  const int m = blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
  if (m >= M) return;
  pA += (size_t)blockIdx.y * n_chunks * M;
  pW += (size_t)blockIdx.y * n_chunks * M;
  const int lane = threadIdx.x & 31;
  const int per = (n_chunks + 31) / 32;
  const int c0 = lane * per, c1 = min(n_chunks, c0 + per);
  int32_t sa = 0, sw = 0;
  for (int c = c0; c < c1; ++c) { sa += pA[(size_t)c * M + m]; sw += pW[(size_t)c * M + m]; }
  int32_t ia = sa, iw = sw;
  for (int o = 1; o < 32; o <<= 1) {
    const int32_t xa = __shfl_up_sync(0xffffffffu, ia, o);
    const int32_t xw = __shfl_up_sync(0xffffffffu, iw, o);
    if (lane >= o) { ia += xa; iw += xw; }
  }
  int32_t ea = ia - sa, ew = iw - sw;
  for (int c = c0; c < c1; ++c) {
    const size_t x = (size_t)c * M + m;
    const int32_t va = pA[x], vw = pW[x];
    pA[x] = ea;
    pW[x] = ew;
    ea += va;
    ew += vw;
  }
}

__global__ void __launch_bounds__(kThreads)
k_scan_apply(int M, int K, int L, int n_chunks, const int32_t* __restrict__ dA,
             const int32_t* __restrict__ dW, const int32_t* __restrict__ pA,
             const int32_t* __restrict__ pW, int32_t* __restrict__ A, int32_t* __restrict__ W) {
  const int64_t t = (int64_t)blockIdx.x * kThreads + threadIdx.x;
  if (t >= (int64_t)n_chunks * M) return;
  dA += (size_t)blockIdx.y * (K + 1) * M;
  dW += (size_t)blockIdx.y * (K + 1) * M;
  pA += (size_t)blockIdx.y * n_chunks * M;
  pW += (size_t)blockIdx.y * n_chunks * M;
  A += (size_t)blockIdx.y * K * M;
  W += (size_t)blockIdx.y * K * M;
  const int m = (int)(t % M);
  const int c = (int)(t / M);
  const int64_t r0 = (int64_t)c * L, r1 = min64(r0 + L, K);
  int32_t a = pA[t], w = pW[t];
  for (int64_t k = r0; k < r1; ++k) {
    a += dA[k * M + m];
    w += dW[k * M + m];
    A[k * M + m] = a;
    W[k * M + m] = w;
  }
}

// exact coarsening: counts add over q base windows, gauges are read at the
// last base window of each coarse window (blockIdx.y = window length,
// blockIdx.z = trace)
__global__ void __launch_bounds__(kThreads)
k_aggregate(const __grid_constant__ AggPlan pl, const int32_t* __restrict__ P,
            const int32_t* __restrict__ D, const int32_t* __restrict__ A,
            const int32_t* __restrict__ W, const unsigned long long* __restrict__ slo,
            int32_t* __restrict__ Pq, int32_t* __restrict__ Dq, int32_t* __restrict__ Aq,
            int32_t* __restrict__ Wq, unsigned long long* __restrict__ sloq) {
  const int w = blockIdx.y, tr = blockIdx.z;
  const int M = pl.M, q = pl.q[w];
  const int64_t n = (int64_t)pl.Kq[w] * M;
  const size_t in0 = (size_t)tr * pl.Kb * M;
  const size_t o0 = (size_t)pl.out_off[tr][w];
  for (int64_t t = (int64_t)blockIdx.x * kThreads + threadIdx.x; t < n;
       t += (int64_t)gridDim.x * kThreads) {
    const uint32_t k = (uint32_t)t / (uint32_t)M;
    const int m = (int)((uint32_t)t - k * (uint32_t)M);
    int32_t p = 0, d = 0;
    unsigned long long sl = 0;
    for (int j = 0; j < q; ++j) {
      const size_t x = in0 + ((size_t)k * q + j) * M + m;
      p += P[x];
      d += D[x];
      if (slo) sl += slo[x];
    }
    const size_t last = in0 + ((size_t)k * q + q - 1) * M + m;
    Pq[o0 + t] = p;
    Dq[o0 + t] = d;
    Aq[o0 + t] = A[last];
    Wq[o0 + t] = W[last];
    if (sloq) sloq[o0 + t] = sl;
  }
}

int num_sms() {
  static int n = 0;
  if (!n) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 1;
  }
  return n;
}

int64_t per_cta_records(int64_t n, int lo, int hi) {
  int64_t per = (n + (int64_t)num_sms() * 4 - 1) / ((int64_t)num_sms() * 4);
  per = std::max<int64_t>(lo, std::min<int64_t>(hi, per));
  return (per + kThreads - 1) / kThreads * kThreads;
}

unsigned grid_for(int64_t work, int per_thread = 1) {
  const int64_t b = (work + (int64_t)kThreads * per_thread - 1) / ((int64_t)kThreads * per_thread);
  return (unsigned)std::max<int64_t>(1, std::min<int64_t>(b, (int64_t)num_sms() * 16));
}

int scan_chunk_rows(int K) {
  int L = (K + 1023) / 1024;
  return L < 16 ? 16 : L;
}

}  // namespace

void reduce_ws_layout(Arena& a, int M, int K, int n_traces, int64_t n_req, ReduceWs& w) {
  const size_t cells = (size_t)(K + 1) * M * n_traces;
  w.n_traces = n_traces;
  w.dA = a.take<int32_t>(cells);
  w.dW = a.take<int32_t>(cells);
  w.first = n_req > 0 ? a.take<int32_t>((size_t)n_req) : nullptr;
  w.last = n_req > 0 ? a.take<int32_t>((size_t)n_req) : nullptr;
  const int L = scan_chunk_rows(K);
  const int n_chunks = (K + L - 1) / L;
  w.partA = a.take<int32_t>((size_t)std::max(n_chunks, 1) * M * n_traces);
  w.partW = a.take<int32_t>((size_t)std::max(n_chunks, 1) * M * n_traces);
}

cudaError_t launch_reduce_requests(const ReqCols* traces, int n_traces, int M, int win, int K,
                                   int32_t* P, int32_t* D, ReduceWs& w, unsigned long long* slo,
                                   const int32_t* slo_ms, tre_diag* diag, cudaStream_t s) {
  if (n_traces < 1 || n_traces > kMaxTraces || n_traces > w.n_traces)
    return cudaErrorInvalidValue;
  const size_t cells = (size_t)K * M * n_traces;
  cudaError_t e;
  if ((e = cudaMemsetAsync(P, 0, cells * sizeof(int32_t), s))) return e;
  if ((e = cudaMemsetAsync(D, 0, cells * sizeof(int32_t), s))) return e;
  if ((e = cudaMemsetAsync(w.dA, 0, (cells + (size_t)M * n_traces) * sizeof(int32_t), s))) return e;
  if ((e = cudaMemsetAsync(w.dW, 0, (cells + (size_t)M * n_traces) * sizeof(int32_t), s))) return e;
  if (slo && (e = cudaMemsetAsync(slo, 0, cells * sizeof(unsigned long long), s))) return e;
  ReqBatch bt;
  bt.n = n_traces;
  int64_t total_n = 0;
  for (int t = 0; t < n_traces; ++t) total_n += traces[t].n;
  int ctas = 0;
  for (int t = 0; t < n_traces; ++t) {
    bt.cols[t] = traces[t];
    // records per CTA sized on the whole batch so the grid fills the GPU
    const int64_t per = per_cta_records(std::max<int64_t>(total_n / n_traces, 1), 1024, 8192);
    bt.per_cta[t] = per;
    bt.cta_base[t] = ctas;
    ctas += (int)((traces[t].n + per - 1) / per);
  }
  bt.cta_base[n_traces] = ctas;
  if (ctas == 0) return cudaSuccess;
  // arrival-side rows cover the CTA's arrival span; start-side rows per model
  const int64_t per = bt.per_cta[0];
  const int64_t near_cap = 48 * 1024 / ((4 + (slo ? 8 : 0)) * M);   // arrival-stage budget
  const int near_rows = (int)std::max<int64_t>(
      1, std::min<int64_t>(near_cap,
                           (int64_t)(3.0 * per / std::max<int64_t>(total_n / n_traces, 1) * K) +
                               34));   // 3x the mean arrival span
  const int far_rows = std::max(8, std::min(512, (int)(kStageBytes / (16 * M))));
  const size_t smem = (size_t)near_rows * M * (4 + (slo ? 8 : 0)) + (size_t)far_rows * M * 16 +
                      (size_t)M * 8;
  if (smem > 200 * 1024) return cudaErrorInvalidValue;
  static bool attr = false;
  if (!attr) {
    cudaError_t e1 = cudaFuncSetAttribute(k_reduce_requests<true>,
                                          cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
    cudaError_t e2 = cudaFuncSetAttribute(k_reduce_requests<false>,
                                          cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
    if (e1 || e2) return e1 ? e1 : e2;
    attr = true;
  }
  if (slo)
    k_reduce_requests<true><<<ctas, kThreads, smem, s>>>(bt, M, win, FastDiv(win), K, near_rows,
                                                         far_rows, P, D, w.dA, w.dW, slo, slo_ms,
                                                         diag);
  else
    k_reduce_requests<false><<<ctas, kThreads, smem, s>>>(bt, M, win, FastDiv(win), K, near_rows,
                                                          far_rows, P, D, w.dA, w.dW, nullptr,
                                                          nullptr, diag);
  return cudaGetLastError();
}

cudaError_t launch_slo_requests(const ReqCols& r, int M, int win, int K,
                                unsigned long long* slo, const int32_t* slo_ms, cudaStream_t s) {
  cudaError_t e = cudaMemsetAsync(slo, 0, (size_t)K * M * sizeof(unsigned long long), s);
  if (e || r.n == 0) return e;
  k_slo_requests<<<grid_for(r.n, 4), kThreads, 0, s>>>(r, M, win, K, slo, slo_ms);
  return cudaGetLastError();
}

cudaError_t launch_reduce_events(const EvCols& ev, int M, int win, int K, int32_t* P, int32_t* D,
                                 ReduceWs& w, tre_diag* diag, cudaStream_t s) {
  const size_t cells = (size_t)K * M;
  cudaError_t e;
  if ((e = cudaMemsetAsync(P, 0, cells * sizeof(int32_t), s))) return e;
  if ((e = cudaMemsetAsync(D, 0, cells * sizeof(int32_t), s))) return e;
  if ((e = cudaMemsetAsync(w.dA, 0, (cells + M) * sizeof(int32_t), s))) return e;
  if ((e = cudaMemsetAsync(w.dW, 0, (cells + M) * sizeof(int32_t), s))) return e;
  if (ev.n_req > 0) {
    k_fill_first_last<<<grid_for(ev.n_req, 4), kThreads, 0, s>>>(w.first, w.last, ev.n_req);
    if ((e = cudaGetLastError())) return e;
  }
  if (ev.n > 0) {
    const int rows = std::max(1, kStageBytes / (8 * M));
    const int64_t per = per_cta_records(ev.n, 2048, 16384);
    const unsigned grid = (unsigned)((ev.n + per - 1) / per);
    k_reduce_events<<<grid, kThreads, (size_t)rows * M * 8, s>>>(ev, M, win, FastDiv(win), K, per,
                                                                 rows, P, D, w.first, w.last, diag);
    if ((e = cudaGetLastError())) return e;
  }
  if (ev.n_req > 0) {
    k_event_gauges<<<grid_for(ev.n_req, 4), kThreads, 0, s>>>(ev, M, FastDiv(win), K, w.first,
                                                               w.last, w.dA, w.dW, diag);
    if ((e = cudaGetLastError())) return e;
  }
  return cudaSuccess;
}

cudaError_t launch_slo_events(const EvCols& ev, int M, int win, int K, unsigned long long* slo,
                              const int32_t* slo_ms, cudaStream_t s) {
  cudaError_t e = cudaMemsetAsync(slo, 0, (size_t)K * M * sizeof(unsigned long long), s);
  if (e || ev.n_req == 0) return e;
  k_slo_events<<<grid_for(ev.n_req, 4), kThreads, 0, s>>>(ev, M, win, K, slo, slo_ms);
  return cudaGetLastError();
}

cudaError_t launch_gauge_scan(int M, int K, ReduceWs& w, int32_t* A, int32_t* W,
                              cudaStream_t s) {
  if (K == 0) return cudaSuccess;
  const int L = scan_chunk_rows(K);
  const int n_chunks = (K + L - 1) / L;
  const int64_t segs = (int64_t)n_chunks * M;
  dim3 g((unsigned)((segs + kThreads - 1) / kThreads), w.n_traces);
  k_scan_partials<<<g, kThreads, 0, s>>>(M, K, L, n_chunks, w.dA, w.dW, w.partA, w.partW);
  k_scan_chunks<<<dim3((M + 3) / 4, w.n_traces), 128, 0, s>>>(M, n_chunks, w.partA, w.partW);
  k_scan_apply<<<g, kThreads, 0, s>>>(M, K, L, n_chunks, w.dA, w.dW, w.partA, w.partW, A, W);
  return cudaGetLastError();
}

cudaError_t launch_aggregate(const AggPlan& pl, const int32_t* P, const int32_t* D,
                             const int32_t* A, const int32_t* W, const unsigned long long* slo,
                             int32_t* Pq, int32_t* Dq, int32_t* Aq, int32_t* Wq,
                             unsigned long long* sloq, cudaStream_t s) {
  int64_t mx = 0;
  for (int w = 0; w < pl.n_win; ++w) mx = std::max<int64_t>(mx, (int64_t)pl.Kq[w] * pl.M);
  if (mx == 0) return cudaSuccess;
  dim3 g(grid_for(mx), pl.n_win, pl.n_traces);
  k_aggregate<<<g, kThreads, 0, s>>>(pl, P, D, A, W, slo, Pq, Dq, Aq, Wq, sloq);
  return cudaGetLastError();
}

}  // namespace tre
