// CPU oracle for the Token Service Share (TSS) signal and TRE move selection.
//
// TEST INFRASTRUCTURE ONLY. This file is the slow, plain reference that the
// CUDA library is checked against. Only the tests, the smoke check and the
// CPU-baseline leg of the benchmark may load it; the library never does, and
// it shares no code, header, table or helper with the library.
//
// Every step follows the paper's definitions in the paper's order, with the
// readings listed below where the paper is silent. Floating-point expressions
// are evaluated one IEEE operation at a time in the caller's precision T
// (float or double); build with -ffp-contract=off so no multiply-add is fused.
//
// Readings (the paper does not fix these):
//  * time base: all times are integer milliseconds; window k covers
//    [k*win, (k+1)*win), windows start at t = 0 (Eq. 1 observes counts over
//    windows of a fixed length).
//  * prompt tokens of a request are all counted at its first-token time; decode
//    token j (0 <= j < L_out) is emitted at t_first + floor(j*(t_end-t_first)/(L_out-1))
//    (a single decode token is at t_first). Counters become window deltas
//    (Sec. V-B).
//  * running (A) and waiting (W) counts are gauges read at the last millisecond
//    of each window: running on [t_start, t_end), waiting on [t_arr, t_start)
//    (Sec. III-A, Sec. V-B).
//  * the demand denominator is floored at one request (Sec. II-B: the raw
//    inverse is clamped at one request); a window with no tokens and no
//    requests is IDLE.
//  * EMA: S = alpha*raw + (1-alpha)*S_prev, started at the first non-idle window
//    and held through idle windows (Sec. III-B).
//  * regions: critical if Z < tau_crit, surplus if Z > tau_surplus, else nominal
//    (Sec. III-B); idle windows form their own class.
//  * theta: the smallest smoothed TSS value s such that, among calibration
//    windows with S >= s, the healthy fraction reaches the reliability target
//    (Sec. III-B: theta is the lowest smoothed TSS at which the SLO reliability
//    target is still met).
//  * control ticks: a window ends a fast (slow) tick when a multiple of
//    fast_ms (slow_ms) falls in (k*win, (k+1)*win] (Sec. IV-B, Sec. V-B).
//  * rescue, rebalance and bounded transfer as in Sec. IV-B/IV-C, Eq. 3.

#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <functional>
#include <queue>
#include <utility>
#include <vector>

namespace {

constexpr uint8_t kCrit = 0, kNom = 1, kSurp = 2, kIdle = 3;
constexpr int kRescue = 1, kRebalance = 2;

struct Move {          // one released donor replica (or pool draw) of a transition
  int32_t window, recv, donor, kind, seq;
};

// window of a non-negative millisecond time, clamped to [0, K]
int64_t win_of(int64_t t, int64_t win, int64_t K) {
  int64_t b = t / win;
  return b > K ? K : b;
}

// --------------------------------------------------------------------------
// Window reduction of request records (Eq. 1 inputs, Sec. V-B).
// drops[0] = arrival outside [0, K*win), drops[1] = bad model id,
// drops[2] = times out of order or bad lengths.
// --------------------------------------------------------------------------
int reduce_requests(int32_t M, int32_t win, int32_t K, int64_t n, const int32_t* model,
                    const int32_t* t_arr, const int32_t* t_start, const int32_t* t_first,
                    const int32_t* t_end, const int32_t* L_in, const int32_t* L_out,
                    int32_t* P, int32_t* D, int32_t* A, int32_t* W, int64_t* drops) {
  if (M < 1 || win < 1 || K < 0 || n < 0) return 1;
  const int64_t span = (int64_t)K * win;
  std::vector<uint32_t> p((size_t)K * M, 0), d((size_t)K * M, 0);
  std::vector<int64_t> dA((size_t)(K + 1) * M, 0), dW((size_t)(K + 1) * M, 0);
  for (int64_t i = 0; i < n; ++i) {
    const int64_t m = model[i];
    if (m < 0 || m >= M) { drops[1]++; continue; }
    const int64_t ta = t_arr[i], ts = t_start[i], tf = t_first[i], te = t_end[i];
    if (ta < 0 || ta >= span) { drops[0]++; continue; }
    if (!(ta <= ts && ts <= tf && tf <= te) || L_in[i] < 0 || L_out[i] < 1) {
      drops[2]++;
      continue;
    }
    // prompt tokens, all at the first-token time
    if (tf < span) p[(size_t)(tf / win) * M + m] += (uint32_t)L_in[i];
    // decode tokens, one at a time at their emission times
    const int64_t L = L_out[i], dur = te - tf;
    for (int64_t j = 0; j < L; ++j) {
      const int64_t tj = (L == 1) ? tf : tf + (j * dur) / (L - 1);
      if (tj < span) d[(size_t)(tj / win) * M + m] += 1u;
    }
    // gauges: +1 where a state begins, -1 where it ends (window of the
    // transition time); the running sum over windows is the gauge value at
    // each window's last millisecond
    dW[(size_t)win_of(ta, win, K) * M + m] += 1;
    dW[(size_t)win_of(ts, win, K) * M + m] -= 1;
    dA[(size_t)win_of(ts, win, K) * M + m] += 1;
    dA[(size_t)win_of(te, win, K) * M + m] -= 1;
  }
  for (int64_t m = 0; m < M; ++m) {
    int64_t a = 0, w = 0;
    for (int64_t k = 0; k < K; ++k) {
      a += dA[(size_t)k * M + m];
      w += dW[(size_t)k * M + m];
      A[(size_t)k * M + m] = (int32_t)a;
      W[(size_t)k * M + m] = (int32_t)w;
    }
  }
  for (size_t x = 0; x < (size_t)K * M; ++x) {
    P[x] = (int32_t)p[x];
    D[x] = (int32_t)d[x];
  }
  return 0;
}

// Time-averaged occupancy of request records (the window-mean reading of the
// running and waiting counts in Eq. 1, Sec. III-A; Sec. II-B speaks of an
// average waiting queue): per (window, model) the request-milliseconds spent
// running ([t_start, t_end)) and waiting ([t_arr, t_start)) inside the window.
// The mean count is that sum divided by the window length. Records are taken
// or skipped by the same rules as reduce_requests (nothing is counted here).
int occupancy_mean_requests(int32_t M, int32_t win, int32_t K, int64_t n, const int32_t* model,
                            const int32_t* t_arr, const int32_t* t_start,
                            const int32_t* t_first, const int32_t* t_end, const int32_t* L_in,
                            const int32_t* L_out, int64_t* A_ms, int64_t* W_ms) {
  if (M < 1 || win < 1 || K < 0 || n < 0) return 1;
  const int64_t span = (int64_t)K * win;
  for (size_t x = 0; x < (size_t)K * M; ++x) A_ms[x] = W_ms[x] = 0;
  // add the part of [a, e) inside every window it touches
  auto add_span = [&](int64_t a, int64_t e, int64_t m, int64_t* out) {
    if (e > span) e = span;
    if (a >= e) return;
    for (int64_t k = a / win; k * win < e; ++k) {
      const int64_t lo = std::max(a, k * win), hi = std::min(e, (k + 1) * win);
      out[(size_t)k * M + m] += hi - lo;
    }
  };
  for (int64_t i = 0; i < n; ++i) {
    const int64_t m = model[i];
    if (m < 0 || m >= M) continue;
    const int64_t ta = t_arr[i], ts = t_start[i], tf = t_first[i], te = t_end[i];
    if (ta < 0 || ta >= span) continue;
    if (!(ta <= ts && ts <= tf && tf <= te) || L_in[i] < 0 || L_out[i] < 1) continue;
    add_span(ts, te, m, A_ms);
    add_span(ta, ts, m, W_ms);
  }
  return 0;
}

// Calibration counts of request records: arrivals per (arrival window, model)
// and how many of them met the TTFT bound of their model's SLO class.
int slo_counts_requests(int32_t M, int32_t win, int32_t K, int64_t n, const int32_t* model,
                        const int32_t* t_arr, const int32_t* t_start, const int32_t* t_first,
                        const int32_t* t_end, const int32_t* L_in, const int32_t* L_out,
                        const int32_t* slo_ttft_ms, int32_t* n_arr, int32_t* n_met) {
  if (M < 1 || win < 1 || K < 0 || n < 0) return 1;
  const int64_t span = (int64_t)K * win;
  for (size_t x = 0; x < (size_t)K * M; ++x) n_arr[x] = n_met[x] = 0;
  for (int64_t i = 0; i < n; ++i) {
    const int64_t m = model[i];
    if (m < 0 || m >= M) continue;
    const int64_t ta = t_arr[i], ts = t_start[i], tf = t_first[i], te = t_end[i];
    if (ta < 0 || ta >= span) continue;
    if (!(ta <= ts && ts <= tf && tf <= te) || L_in[i] < 0 || L_out[i] < 1) continue;
    const size_t x = (size_t)(ta / win) * M + m;
    n_arr[x] += 1;
    if (tf - ta <= slo_ttft_ms[m]) n_met[x] += 1;
  }
  return 0;
}

// Running gauge split at the first token for a stage-aware signal (Sec. VIII:
// separate prefill and decode states): among the records reduce_requests
// keeps, a request is prefilling on [t_start, t_first) and decoding on
// [t_first, t_end); both gauges are read at the last millisecond of each
// window, by the same +1/-1 difference and running sum as A and W.
int stage_gauges_requests(int32_t M, int32_t win, int32_t K, int64_t n, const int32_t* model,
                          const int32_t* t_arr, const int32_t* t_start, const int32_t* t_first,
                          const int32_t* t_end, const int32_t* L_in, const int32_t* L_out,
                          int32_t* A_pre, int32_t* A_dec) {
  if (M < 1 || win < 1 || K < 0 || n < 0) return 1;
  const int64_t span = (int64_t)K * win;
  std::vector<int64_t> dP((size_t)(K + 1) * M, 0), dD((size_t)(K + 1) * M, 0);
  for (int64_t i = 0; i < n; ++i) {
    const int64_t m = model[i];
    if (m < 0 || m >= M) continue;
    const int64_t ta = t_arr[i], ts = t_start[i], tf = t_first[i], te = t_end[i];
    if (ta < 0 || ta >= span) continue;
    if (!(ta <= ts && ts <= tf && tf <= te) || L_in[i] < 0 || L_out[i] < 1) continue;
    dP[(size_t)win_of(ts, win, K) * M + m] += 1;
    dP[(size_t)win_of(tf, win, K) * M + m] -= 1;
    dD[(size_t)win_of(tf, win, K) * M + m] += 1;
    dD[(size_t)win_of(te, win, K) * M + m] -= 1;
  }
  for (int64_t m = 0; m < M; ++m) {
    int64_t a = 0, d = 0;
    for (int64_t k = 0; k < K; ++k) {
      a += dP[(size_t)k * M + m];
      d += dD[(size_t)k * M + m];
      A_pre[(size_t)k * M + m] = (int32_t)a;
      A_dec[(size_t)k * M + m] = (int32_t)d;
    }
  }
  return 0;
}

// Decode-side SLO counts for a stage-aware signal (Sec. VIII: separate prefill
// and decode states; Sec. III-A: decode determines TPOT): per (arrival window,
// model) the requests with more than one output token and how many of them
// met the model's TPOT bound, (t_end - t_first) <= tpot_ms * (L_out - 1)
// (exact integer test). Records taken or skipped as in reduce_requests.
int slo_tpot_counts_requests(int32_t M, int32_t win, int32_t K, int64_t n, const int32_t* model,
                             const int32_t* t_arr, const int32_t* t_start,
                             const int32_t* t_first, const int32_t* t_end, const int32_t* L_in,
                             const int32_t* L_out, const int32_t* tpot_ms, int32_t* n_dec,
                             int32_t* n_met) {
  if (M < 1 || win < 1 || K < 0 || n < 0) return 1;
  const int64_t span = (int64_t)K * win;
  for (size_t x = 0; x < (size_t)K * M; ++x) n_dec[x] = n_met[x] = 0;
  for (int64_t i = 0; i < n; ++i) {
    const int64_t m = model[i];
    if (m < 0 || m >= M) continue;
    const int64_t ta = t_arr[i], ts = t_start[i], tf = t_first[i], te = t_end[i];
    if (ta < 0 || ta >= span) continue;
    if (!(ta <= ts && ts <= tf && tf <= te) || L_in[i] < 0 || L_out[i] < 1) continue;
    if (L_out[i] < 2) continue;                      // no inter-token gap
    const size_t x = (size_t)(ta / win) * M + m;
    n_dec[x] += 1;
    if (te - tf <= (int64_t)tpot_ms[m] * (L_out[i] - 1)) n_met[x] += 1;
  }
  return 0;
}

// --------------------------------------------------------------------------
// Window reduction of token-level events (one record per emitted token).
// --------------------------------------------------------------------------
int reduce_events(int32_t M, int32_t win, int32_t K, int64_t n, const int32_t* model,
                  const int32_t* req, const float* t_s, const uint8_t* phase, int64_t n_req,
                  const int32_t* req_model, const int32_t* req_t_arr, int32_t* P, int32_t* D,
                  int32_t* A, int32_t* W, int64_t* drops) {
  if (M < 1 || win < 1 || K < 0 || n < 0 || n_req < 0) return 1;
  const double span = (double)((int64_t)K * win);
  std::vector<uint32_t> p((size_t)K * M, 0), d((size_t)K * M, 0);
  std::vector<int64_t> first((size_t)n_req, INT64_MAX), last((size_t)n_req, -1);
  for (int64_t i = 0; i < n; ++i) {
    const int64_t m = model[i], r = req[i];
    if (m < 0 || m >= M || r < 0 || r >= n_req || req_model[r] != m) { drops[1]++; continue; }
    // exact millisecond tick of the float timestamp: the product of a float
    // and 1000 is exact in double
    const double ms = std::floor((double)t_s[i] * 1000.0);
    if (!(ms >= 0.0 && ms < span)) { drops[0]++; continue; }
    if (phase[i] > 1) { drops[2]++; continue; }
    const int64_t t = (int64_t)ms;
    const size_t x = (size_t)(t / win) * M + m;
    if (phase[i] == 0) p[x] += 1u; else d[x] += 1u;
    if (t < first[r]) first[r] = t;
    if (t > last[r]) last[r] = t;
  }
  std::vector<int64_t> dA((size_t)(K + 1) * M, 0), dW((size_t)(K + 1) * M, 0);
  for (int64_t r = 0; r < n_req; ++r) {
    if (last[r] < 0) continue;                       // no valid event
    const int64_t m = req_model[r], ta = req_t_arr[r];
    if (!(ta >= 0 && ta <= first[r])) { drops[2]++; continue; }
    dW[(size_t)win_of(ta, win, K) * M + m] += 1;
    dW[(size_t)win_of(first[r], win, K) * M + m] -= 1;
    dA[(size_t)win_of(first[r], win, K) * M + m] += 1;
    dA[(size_t)win_of(last[r], win, K) * M + m] -= 1;
  }
  for (int64_t m = 0; m < M; ++m) {
    int64_t a = 0, w = 0;
    for (int64_t k = 0; k < K; ++k) {
      a += dA[(size_t)k * M + m];
      w += dW[(size_t)k * M + m];
      A[(size_t)k * M + m] = (int32_t)a;
      W[(size_t)k * M + m] = (int32_t)w;
    }
  }
  for (size_t x = 0; x < (size_t)K * M; ++x) {
    P[x] = (int32_t)p[x];
    D[x] = (int32_t)d[x];
  }
  return 0;
}

// Time-averaged occupancy of token events: a request runs from its first to
// its last valid event and waits from its arrival to its first event (the
// spans reduce_events reads at each window's last millisecond); per (window,
// model) the request-milliseconds of each span inside the window. Events and
// requests are taken or skipped by reduce_events' rules (nothing is counted).
int occupancy_mean_events(int32_t M, int32_t win, int32_t K, int64_t n, const int32_t* model,
                          const int32_t* req, const float* t_s, const uint8_t* phase,
                          int64_t n_req, const int32_t* req_model, const int32_t* req_t_arr,
                          int64_t* A_ms, int64_t* W_ms) {
  if (M < 1 || win < 1 || K < 0 || n < 0 || n_req < 0) return 1;
  const int64_t span = (int64_t)K * win;
  for (size_t x = 0; x < (size_t)K * M; ++x) A_ms[x] = W_ms[x] = 0;
  std::vector<int64_t> first((size_t)n_req, INT64_MAX), last((size_t)n_req, -1);
  for (int64_t i = 0; i < n; ++i) {
    const int64_t m = model[i], r = req[i];
    if (m < 0 || m >= M || r < 0 || r >= n_req || req_model[r] != m) continue;
    const double ms = std::floor((double)t_s[i] * 1000.0);
    if (!(ms >= 0.0 && ms < (double)span) || phase[i] > 1) continue;
    const int64_t t = (int64_t)ms;
    if (t < first[r]) first[r] = t;
    if (t > last[r]) last[r] = t;
  }
  auto add_span = [&](int64_t a, int64_t e, int64_t m, int64_t* out) {
    if (e > span) e = span;
    if (a >= e) return;
    for (int64_t k = a / win; k * win < e; ++k) {
      const int64_t lo = std::max(a, k * win), hi = std::min(e, (k + 1) * win);
      out[(size_t)k * M + m] += hi - lo;
    }
  };
  for (int64_t r = 0; r < n_req; ++r) {
    if (last[r] < 0) continue;
    const int64_t m = req_model[r], ta = req_t_arr[r];
    if (!(ta >= 0 && ta <= first[r])) continue;
    add_span(first[r], last[r], m, A_ms);
    add_span(ta, first[r], m, W_ms);
  }
  return 0;
}

int slo_counts_events(int32_t M, int32_t win, int32_t K, int64_t n_req, const int32_t* req_model,
                      const int32_t* req_t_arr, const int32_t* req_ttft,
                      const int32_t* slo_ttft_ms, int32_t* n_arr, int32_t* n_met) {
  if (M < 1 || win < 1 || K < 0 || n_req < 0) return 1;
  const int64_t span = (int64_t)K * win;
  for (size_t x = 0; x < (size_t)K * M; ++x) n_arr[x] = n_met[x] = 0;
  for (int64_t r = 0; r < n_req; ++r) {
    const int64_t m = req_model[r], ta = req_t_arr[r];
    if (m < 0 || m >= M || ta < 0 || ta >= span) continue;
    const size_t x = (size_t)(ta / win) * M + m;
    n_arr[x] += 1;
    if (req_ttft[r] <= slo_ttft_ms[m]) n_met[x] += 1;
  }
  return 0;
}

// --------------------------------------------------------------------------
// Eq. 1 (raw TSS), EMA smoothing, Eq. 2 (Z = S / theta) and the regions.
// S_carry / init_carry (may be null) hold the smoothing state across calls.
// recv (may be null): per window, the Eq. 3 receiver argmin Z over non-idle
// models (lowest index on ties), -1 if every model is idle.
// A_ms / W_ms (both null or both given): the time-averaged occupancy in place
// of the sampled A / W -- the mean counts A_ms / win and W_ms / win enter the
// demand term, and a window is idle when P, D, A_ms and W_ms are all zero.
// --------------------------------------------------------------------------
template <class T>
int score(int32_t M, int32_t win, int32_t K, const int32_t* P, const int32_t* D,
          const int32_t* A, const int32_t* W, const T* w_p, const T* w_q, const T* alpha,
          const T* theta, const T* tau_crit, const T* tau_surplus, T* S_carry,
          uint8_t* init_carry, T* S_out, T* Z_out, uint8_t* cls_out, int32_t* recv,
          const int64_t* A_ms, const int64_t* W_ms) {
  if ((A_ms == nullptr) != (W_ms == nullptr)) return 1;
  if (M < 1 || win < 1 || K < 0) return 1;
  const T dt = (T)win / (T)1000;                     // window length in seconds
  for (int64_t m = 0; m < M; ++m) {
    T S = S_carry ? S_carry[m] : (T)0;
    bool init = init_carry ? init_carry[m] != 0 : false;
    if (!init) S = (T)0;
    const T a = alpha[m];
    const T b = (T)1 - a;
    for (int64_t k = 0; k < K; ++k) {
      const size_t x = (size_t)k * M + m;
      const bool idle = A_ms ? P[x] == 0 && D[x] == 0 && A_ms[x] == 0 && W_ms[x] == 0
                             : P[x] == 0 && D[x] == 0 && A[x] == 0 && W[x] == 0;
      if (!idle) {
        const T r_pre = (T)P[x] / dt;                  // prefill token rate
        const T r_dec = (T)D[x] / dt;                  // decode token rate
        const T svc = w_p[m] * r_pre;
        const T num = svc + r_dec;
        // running and waiting counts: sampled, or window means
        const T a_cnt = A_ms ? (T)A_ms[x] / (T)win : (T)A[x];
        const T w_cnt = A_ms ? (T)W_ms[x] / (T)win : (T)W[x];
        const T qw = w_q[m] * w_cnt;
        T den = a_cnt + qw;
        if (den < (T)1) den = (T)1;                    // demand floor of one request
        const T raw = num / den;
        if (!init) {
          S = raw;
          init = true;
        } else {
          const T x1 = a * raw;
          const T x2 = b * S;
          S = x1 + x2;
        }
      }
      const T Z = S / theta[m];
      S_out[x] = S;
      Z_out[x] = Z;
      uint8_t c;
      if (idle) c = kIdle;
      else if (Z < tau_crit[m]) c = kCrit;
      else if (Z > tau_surplus[m]) c = kSurp;
      else c = kNom;
      cls_out[x] = c;
    }
    if (S_carry) S_carry[m] = S;
    if (init_carry) init_carry[m] = init ? 1 : 0;
  }
  if (recv) {
    for (int64_t k = 0; k < K; ++k) {
      int32_t best = -1;
      for (int64_t m = 0; m < M; ++m) {
        const size_t x = (size_t)k * M + m;
        if (cls_out[x] == kIdle) continue;
        if (best < 0 || Z_out[x] < Z_out[(size_t)k * M + best]) best = (int32_t)m;
      }
      recv[k] = best;
    }
  }
  return 0;
}

// --------------------------------------------------------------------------
// theta calibration (Sec. III-B): per model, among windows that had at least
// one arrival, are not idle and have S > 0, find the smallest S value s such
// that the windows with S >= s are healthy in at least a `reliability`
// fraction. A window is healthy when at least `ok_frac` of its arrivals met
// the TTFT bound. Falls back to max S (no s qualifies) or 1 (no candidate),
// counting the model in *degenerate.
// --------------------------------------------------------------------------
template <class T>
int calibrate(int32_t M, int32_t K, const T* S, const uint8_t* cls, const int32_t* n_arr,
              const int32_t* n_met, double ok_frac, double reliability, T* theta,
              int64_t* degenerate) {
  if (M < 1 || K < 0) return 1;
  for (int64_t m = 0; m < M; ++m) {
    std::vector<std::pair<T, int>> cand;
    for (int64_t k = 0; k < K; ++k) {
      const size_t x = (size_t)k * M + m;
      if (cls[x] == kIdle || n_arr[x] < 1 || !(S[x] > (T)0)) continue;
      const int healthy = (double)n_met[x] >= ok_frac * (double)n_arr[x] ? 1 : 0;
      cand.push_back({S[x], healthy});
    }
    if (cand.empty()) {
      theta[m] = (T)1;
      (*degenerate)++;
      continue;
    }
    std::sort(cand.begin(), cand.end(),
              [](const std::pair<T, int>& u, const std::pair<T, int>& v) { return u.first > v.first; });
    int64_t H = 0, C = 0;
    bool found = false;
    T best = (T)0;
    size_t i = 0;
    while (i < cand.size()) {                // one step per distinct value, descending
      const T s = cand[i].first;
      while (i < cand.size() && cand[i].first == s) {
        C += 1;
        H += cand[i].second;
        ++i;
      }
      if ((double)H >= reliability * (double)C) {
        best = s;
        found = true;
      }
    }
    if (found) {
      theta[m] = best;
    } else {
      theta[m] = cand.front().first;
      (*degenerate)++;
    }
  }
  return 0;
}

// --------------------------------------------------------------------------
// TRE move selection (Sec. IV-B dual-speed control, Eq. 3, Sec. IV-C bounded
// pairwise transfer), open loop over a scored trace. Z and the idle class come
// from the scored windows; the critical/surplus regions are re-derived here
// from the given thresholds so one scored series serves many settings.
// r (in/out) holds routable replicas; the idle pool is budget - sum(g*r).
// Emits one Move per released donor replica, or one with donor = -1 for a
// transition served from the idle pool. Returns 4 if more than `cap` moves.
// --------------------------------------------------------------------------
template <class T>
struct Walk {
  int32_t M;
  const T* Zk;                 // Z of the current window
  const uint8_t* ck;           // class of the current window (only kIdle is used)
  const T* tau_crit;
  const T* tau_surplus;
  const int32_t* r_min;
  const int32_t* g;
  const uint8_t* guard = nullptr;   // closed loop: donors whose latency guard is breached

  uint8_t region(int32_t m) const {
    if (ck[m] == kIdle) return kIdle;
    if (Zk[m] < tau_crit[m]) return kCrit;
    if (Zk[m] > tau_surplus[m]) return kSurp;
    return kNom;
  }
  // donor preference: idle models (lowest index), then surplus by Z
  // descending, then nominal by Z descending (nominal only above the
  // receiver's Z when `nom_above` is set); never critical, never the receiver,
  // never below the replica floor.
  // A donor whose local latency guard is breached (closed loop only) is not
  // released at this tick (Sec. IV-C donor-side release guard).
  bool held(int32_t m) const { return guard && guard[m]; }
  int32_t pick_donor(const std::vector<int64_t>& r, int32_t recv, bool nom_above) const {
    for (int32_t m = 0; m < M; ++m)
      if (m != recv && region(m) == kIdle && r[m] > r_min[m] && !held(m)) return m;
    int32_t best = -1;
    for (int32_t m = 0; m < M; ++m)
      if (m != recv && region(m) == kSurp && r[m] > r_min[m] && !held(m) &&
          (best < 0 || Zk[m] > Zk[best]))
        best = m;
    if (best >= 0) return best;
    for (int32_t m = 0; m < M; ++m) {
      if (m == recv || region(m) != kNom || r[m] <= r_min[m] || held(m)) continue;
      if (nom_above && !(Zk[m] > Zk[recv])) continue;
      if (best < 0 || Zk[m] > Zk[best]) best = m;
    }
    return best;
  }
};

// --------------------------------------------------------------------------
// Per-window ranking (Eq. 3 receiver, Sec. IV-B acquisition order): the
// receiver is the non-idle model of smallest Z (lowest index on ties), -1 if
// every model is idle. Its donors, in the order they would be released: idle
// models by index, then surplus models by Z descending, then nominal models
// whose Z is above the receiver's, by Z descending (equal Z: lower index
// first); never a critical model, never the receiver. The first 8 are
// written, -1 in the slots left over (all of them without a receiver).
// Regions come from cls (as scored with the profile's thresholds).
// --------------------------------------------------------------------------
template <class T>
int rank_windows(int32_t M, int32_t K, const T* Z, const uint8_t* cls, int32_t* recv_out,
                 int32_t* order_out) {
  if (M < 1 || K < 0) return 1;
  std::vector<int32_t> surp, nom;
  for (int64_t k = 0; k < K; ++k) {
    const T* z = Z + k * M;
    const uint8_t* c = cls + k * M;
    int32_t recv = -1;
    for (int32_t m = 0; m < M; ++m)
      if (c[m] != kIdle && (recv < 0 || z[m] < z[recv])) recv = m;
    if (recv_out) recv_out[k] = recv;
    if (!order_out) continue;
    int32_t* o = order_out + k * 8;
    for (int i = 0; i < 8; ++i) o[i] = -1;
    if (recv < 0) continue;
    std::vector<int32_t> order;
    for (int32_t m = 0; m < M; ++m)
      if (m != recv && c[m] == kIdle) order.push_back(m);
    surp.clear();
    nom.clear();
    for (int32_t m = 0; m < M; ++m) {
      if (m == recv) continue;
      if (c[m] == kSurp) surp.push_back(m);
      else if (c[m] == kNom && z[m] > z[recv]) nom.push_back(m);
    }
    auto by_z_desc = [&](int32_t a, int32_t b) { return z[a] > z[b] || (z[a] == z[b] && a < b); };
    std::sort(surp.begin(), surp.end(), by_z_desc);
    std::sort(nom.begin(), nom.end(), by_z_desc);
    order.insert(order.end(), surp.begin(), surp.end());
    order.insert(order.end(), nom.begin(), nom.end());
    for (size_t i = 0; i < order.size() && i < 8; ++i) o[i] = order[i];
  }
  return 0;
}

// The controller of Sec. IV-B/IV-C, one control tick at a time: replica
// state r (routable replicas per model), the idle pool, and the move list.
template <class T>
struct Controller {
  int32_t M;
  const T* tau_crit;
  const T* tau_surplus;
  const int32_t* r_min;
  const int32_t* footprint;
  int32_t pacing_cap;
  std::vector<int64_t> r;
  int64_t free_pool = 0;
  Move* moves;
  int64_t cap;
  int64_t nm = 0;
  // transitions of the last tick: receiver and the donor replicas it released
  struct Transition {
    int32_t recv;
    std::vector<int32_t> donors;
  };
  std::vector<Transition> last;

  // false on an inconsistent initial state (negative counts, footprints
  // below one, more replicas than the budget holds)
  bool init(int64_t budget, const int32_t* r0) {
    r.assign(M, 0);
    int64_t used = 0;
    for (int32_t m = 0; m < M; ++m) {
      if (r0[m] < 0 || footprint[m] < 1 || r_min[m] < 0) return false;
      r[m] = r0[m];
      used += (int64_t)footprint[m] * r[m];
    }
    if (used > budget) return false;
    free_pool = budget - used;
    return true;
  }

  void emit(int64_t k, int32_t recv, int32_t donor, int kind, int seq) {
    if (nm < cap) moves[nm] = Move{(int32_t)k, recv, donor, kind, seq};
    ++nm;
  }

  // window k ends a fast and/or a slow tick; Zk, ck: that window's Z and class.
  // Closed loop only (null / false in the open-loop walk): guard[m] set when
  // model m breached its latency guard in the window, lost[m] when it has
  // requests waiting and no routable replica, busy when a rebalance transfer
  // is still in progress. Returns the kind of transition the tick made (0:
  // none) -- a rescue deferred behind a rebalance in progress returns 0.
  int tick(int64_t k, const T* Zk, const uint8_t* ck, bool fast, bool slow,
           const uint8_t* guard = nullptr, const uint8_t* lost = nullptr, bool busy = false) {
    last.clear();
    Walk<T> wk{M, Zk, ck, tau_crit, tau_surplus, r_min, footprint, guard};
    int32_t recv = -1;
    int kind = 0;
    bool nom_above = false;
    if (fast) {
      // rescue (Sec. IV-B): a hard latency-guard breach pre-empts every other
      // event (the breaching model of lowest Z); otherwise the lowest Z among
      // critical models and models that lost their routable capacity
      bool hard = false;
      if (guard)
        for (int32_t m = 0; m < M; ++m)
          if (guard[m] && (recv < 0 || wk.Zk[m] < wk.Zk[recv])) recv = m;
      if (recv >= 0) {
        hard = true;
      } else {
        for (int32_t m = 0; m < M; ++m) {
          const bool want = wk.region(m) == kCrit || (lost && lost[m]);
          if (want && (recv < 0 || wk.Zk[m] < wk.Zk[recv])) recv = m;
        }
      }
      if (recv >= 0) {
        // a rebalance transfer in progress is not pre-empted unless the
        // receiver breaches a hard guard; the pending rescue still keeps the
        // slow loop out of this tick
        if (busy && !hard) return 0;
        kind = kRescue;
      }
    }
    if (kind == 0 && recv < 0 && slow) {         // rebalance: Eq. 3 over non-idle models
      for (int32_t m = 0; m < M; ++m)
        if (wk.region(m) != kIdle && (recv < 0 || wk.Zk[m] < wk.Zk[recv])) recv = m;
      if (recv >= 0 && wk.Zk[recv] < (T)1) {
        kind = kRebalance;
        nom_above = true;
      }
    }
    if (kind == 0) return 0;
    for (int32_t seq = 0; seq < pacing_cap; ++seq) {
      const int64_t need = footprint[recv];
      if (free_pool >= need) {                   // idle capacity first
        free_pool -= need;
        r[recv] += 1;
        emit(k, recv, -1, kind, seq);
        last.push_back({recv, {}});
        continue;
      }
      // release donors one replica at a time until the receiver's footprint
      // fits; abandon the transition if the eligible donors cannot cover it
      std::vector<int64_t> rr = r;
      int64_t f = free_pool;
      std::vector<int32_t> rel;
      bool ok = true;
      while (f < need) {
        const int32_t d = wk.pick_donor(rr, recv, nom_above);
        if (d < 0) { ok = false; break; }
        rr[d] -= 1;
        f += footprint[d];
        rel.push_back(d);
      }
      if (!ok) break;
      r = rr;
      free_pool = f - need;
      r[recv] += 1;
      for (int32_t d : rel) emit(k, recv, d, kind, seq);
      last.push_back({recv, rel});
    }
    return kind;
  }
};

// window k ends a tick of cadence c when a multiple of c falls in (k*win, (k+1)*win]
inline bool ends_tick(int64_t k, int32_t win, int32_t c) {
  return ((k + 1) * (int64_t)win) / c > (k * (int64_t)win) / c;
}

template <class T>
int select_moves(int32_t M, int32_t win, int32_t K, const T* Z, const uint8_t* cls,
                 const T* tau_crit, const T* tau_surplus, int64_t budget, const int32_t* r_min,
                 const int32_t* footprint, int32_t fast_ms, int32_t slow_ms, int32_t pacing_cap,
                 int32_t* r_inout, Move* moves, int64_t cap, int64_t* n_moves) {
  if (M < 1 || win < 1 || K < 0 || fast_ms < 1 || slow_ms < 1 || pacing_cap < 0) return 1;
  Controller<T> ctl{M, tau_crit, tau_surplus, r_min, footprint, pacing_cap, {}, 0, moves, cap, 0, {}};
  if (!ctl.init(budget, r_inout)) return 1;
  for (int64_t k = 0; k < K; ++k) {
    const bool fast = ends_tick(k, win, fast_ms), slow = ends_tick(k, win, slow_ms);
    if (fast || slow) ctl.tick(k, Z + (size_t)k * M, cls + (size_t)k * M, fast, slow);
  }
  for (int32_t m = 0; m < M; ++m) r_inout[m] = (int32_t)ctl.r[m];
  *n_moves = ctl.nm;
  return ctl.nm > cap ? 4 : 0;
}

// --------------------------------------------------------------------------
// Closed-loop replay: the controller's moves change the capacity that serves
// the requests, and the telemetry it scores comes from the requests as they
// are served. Readings:
//  * each routable replica of a model is one server; a model's requests are
//    served in input order (FCFS when sorted by arrival) by whichever server
//    frees first; a request needs d_first ms to its first token and d_total
//    ms to its last once started;
//  * window k is processed at T = (k+1)*win: every request that starts before
//    T is started first, then window k's telemetry (same attribution as
//    reduce_requests) is scored (carry across windows) and, on a control
//    tick, the controller acts with the replica counts as they are;
//  * a transition commits at its tick T (the controller's replica counts and
//    pool change then); each donor replica it releases is the donor's server
//    that frees first: it takes no request from T on, finishes the one it is
//    serving (drain) and returns its GPU sleep_ms after that; the receiver's
//    new replica starts waking when its GPU is free -- at T when the idle
//    pool paid for it, else when the last of the transition's released
//    donor replicas has returned its GPU -- and serves requests wake_ms
//    later (Sec. VI-D measures sleep and wake; with both zero a drained
//    donor's GPU passes straight to the receiver);
//  * a request not started by the end of the grid reports
//    t_start = t_first = t_end = K*win; invalid latent records (model out of
//    range, arrival outside [0, K*win), negative durations, d_first > d_total,
//    L_in < 0, L_out < 1) are not served and report -1.
// --------------------------------------------------------------------------
template <class T>
int closed_loop(int32_t M, int32_t win, int32_t K, int64_t n, const int32_t* model,
                const int32_t* t_arr, const int32_t* d_first, const int32_t* d_total,
                const int32_t* L_in, const int32_t* L_out, const T* w_p, const T* w_q,
                const T* alpha, const T* theta, const T* tau_crit, const T* tau_surplus,
                int64_t budget, const int32_t* r0, const int32_t* r_min, const int32_t* footprint,
                int32_t fast_ms, int32_t slow_ms, int32_t pacing_cap, int32_t wake_ms,
                int32_t sleep_ms, const int32_t* guard_ms, int32_t* t_start, int32_t* t_first,
                int32_t* t_end, int32_t* r_out, Move* moves, int64_t cap, int64_t* n_moves,
                T* Z_out, uint8_t* cls_out) {
  if (M < 1 || win < 1 || K < 0 || n < 0 || fast_ms < 1 || slow_ms < 1 || pacing_cap < 0 ||
      wake_ms < 0 || sleep_ms < 0)
    return 1;
  const int64_t span = (int64_t)K * win;
  Controller<T> ctl{M, tau_crit, tau_surplus, r_min, footprint, pacing_cap, {}, 0, moves, cap, 0, {}};
  if (!ctl.init(budget, r0)) return 1;
  using MinHeap = std::priority_queue<int64_t, std::vector<int64_t>, std::greater<int64_t>>;
  std::vector<MinHeap> servers(M);
  for (int32_t m = 0; m < M; ++m)
    for (int64_t j = 0; j < ctl.r[m]; ++j) servers[m].push(0);
  std::vector<std::vector<int64_t>> queue(M);
  std::vector<size_t> head(M, 0);
  std::vector<int64_t> arr_cnt((size_t)K * M, 0);     // arrivals per (window, model)
  for (int64_t i = 0; i < n; ++i) {
    t_start[i] = t_first[i] = t_end[i] = -1;
    const int64_t m = model[i];
    if (m < 0 || m >= M || t_arr[i] < 0 || t_arr[i] >= span) continue;
    if (d_first[i] < 0 || d_total[i] < d_first[i] || L_in[i] < 0 || L_out[i] < 1) continue;
    queue[m].push_back(i);
    t_start[i] = t_first[i] = t_end[i] = (int32_t)span;   // until it starts
    arr_cnt[(size_t)(t_arr[i] / win) * M + m] += 1;
  }
  // telemetry accumulated as requests start (windows at or after the current)
  std::vector<uint32_t> P((size_t)K * M, 0), D((size_t)K * M, 0);
  std::vector<int64_t> end_cnt((size_t)(K + 1) * M, 0);
  std::vector<int64_t> cum_arr(M, 0), cum_start(M, 0), cum_end(M, 0);
  std::vector<T> S_carry(M, (T)0), S_row(M), Z_row(M);
  std::vector<uint8_t> init_carry(M, 0), cls_row(M);
  std::vector<int32_t> Pk(M), Dk(M), Ak(M), Wk(M);
  // latency guard: first tokens per (window, model) later than the model's
  // guard bound after arrival; the tick's guard and lost-capacity flags
  std::vector<int64_t> late((size_t)K * M, 0);
  std::vector<uint8_t> guard_row(M, 0), lost_row(M, 0);
  int64_t reb_until = 0;                         // a rebalance transfer serves from here on
  for (int64_t k = 0; k < K; ++k) {
    const int64_t Tk = (k + 1) * (int64_t)win;
    for (int32_t m = 0; m < M; ++m) {
      while (head[m] < queue[m].size() && !servers[m].empty()) {
        const int64_t i = queue[m][head[m]];
        const int64_t st = std::max<int64_t>(t_arr[i], servers[m].top());
        if (st >= Tk) break;
        const int64_t tf = std::min<int64_t>(st + d_first[i], INT32_MAX);
        const int64_t te = std::min<int64_t>(st + d_total[i], INT32_MAX);
        servers[m].pop();
        servers[m].push(st + d_total[i]);
        ++head[m];
        t_start[i] = (int32_t)st;
        t_first[i] = (int32_t)tf;
        t_end[i] = (int32_t)te;
        cum_start[m] += 1;
        // tokens and the end of the running span, as reduce_requests counts them
        if (tf < span) P[(size_t)(tf / win) * M + m] += (uint32_t)L_in[i];
        if (guard_ms && tf < span && tf - t_arr[i] > guard_ms[m]) late[(size_t)(tf / win) * M + m] += 1;
        const int64_t L = L_out[i], dur = te - tf;
        for (int64_t j = 0; j < L; ++j) {
          const int64_t tj = (L == 1) ? tf : tf + (j * dur) / (L - 1);
          if (tj < span) D[(size_t)(tj / win) * M + m] += 1u;
        }
        end_cnt[(size_t)win_of(te, win, K) * M + m] += 1;
      }
    }
    for (int32_t m = 0; m < M; ++m) {
      const size_t x = (size_t)k * M + m;
      cum_arr[m] += arr_cnt[x];
      cum_end[m] += end_cnt[x];
      Pk[m] = (int32_t)P[x];
      Dk[m] = (int32_t)D[x];
      Ak[m] = (int32_t)(cum_start[m] - cum_end[m]);
      Wk[m] = (int32_t)(cum_arr[m] - cum_start[m]);
    }
    score<T>(M, win, 1, Pk.data(), Dk.data(), Ak.data(), Wk.data(), w_p, w_q, alpha, theta,
             tau_crit, tau_surplus, S_carry.data(), init_carry.data(), S_row.data(), Z_row.data(),
             cls_row.data(), nullptr, nullptr, nullptr);
    if (Z_out) std::copy(Z_row.begin(), Z_row.end(), Z_out + (size_t)k * M);
    if (cls_out) std::copy(cls_row.begin(), cls_row.end(), cls_out + (size_t)k * M);
    const bool fast = ends_tick(k, win, fast_ms), slow = ends_tick(k, win, slow_ms);
    if (!fast && !slow) continue;
    for (int32_t m = 0; m < M; ++m) {
      guard_row[m] = late[(size_t)k * M + m] > 0 ? 1 : 0;
      lost_row[m] = ctl.r[m] == 0 && Wk[m] > 0 ? 1 : 0;
    }
    const int kind = ctl.tick(k, Z_row.data(), cls_row.data(), fast, slow,
                              guard_ms ? guard_row.data() : nullptr, lost_row.data(),
                              Tk < reb_until);
    for (const auto& tr : ctl.last) {
      int64_t gpu_free = Tk;                     // when the receiver's GPU is free
      for (int32_t d : tr.donors) {
        const int64_t drained = std::max<int64_t>(servers[d].top(), Tk);
        servers[d].pop();
        gpu_free = std::max<int64_t>(gpu_free, drained + sleep_ms);
      }
      servers[tr.recv].push(gpu_free + wake_ms);
      if (kind == kRebalance) reb_until = std::max<int64_t>(reb_until, gpu_free + wake_ms);
    }
  }
  for (int32_t m = 0; m < M; ++m) r_out[m] = (int32_t)ctl.r[m];
  *n_moves = ctl.nm;
  return ctl.nm > cap ? 4 : 0;
}

}  // namespace

extern "C" {

int orc_reduce_requests(int32_t M, int32_t win, int32_t K, int64_t n, const int32_t* model,
                        const int32_t* t_arr, const int32_t* t_start, const int32_t* t_first,
                        const int32_t* t_end, const int32_t* L_in, const int32_t* L_out,
                        int32_t* P, int32_t* D, int32_t* A, int32_t* W, int64_t* drops) {
  return reduce_requests(M, win, K, n, model, t_arr, t_start, t_first, t_end, L_in, L_out, P, D,
                         A, W, drops);
}

int orc_occupancy_mean_requests(int32_t M, int32_t win, int32_t K, int64_t n,
                                const int32_t* model, const int32_t* t_arr,
                                const int32_t* t_start, const int32_t* t_first,
                                const int32_t* t_end, const int32_t* L_in, const int32_t* L_out,
                                int64_t* A_ms, int64_t* W_ms) {
  return occupancy_mean_requests(M, win, K, n, model, t_arr, t_start, t_first, t_end, L_in, L_out,
                                 A_ms, W_ms);
}

int orc_stage_gauges_requests(int32_t M, int32_t win, int32_t K, int64_t n,
                              const int32_t* model, const int32_t* t_arr,
                              const int32_t* t_start, const int32_t* t_first,
                              const int32_t* t_end, const int32_t* L_in, const int32_t* L_out,
                              int32_t* A_pre, int32_t* A_dec) {
  return stage_gauges_requests(M, win, K, n, model, t_arr, t_start, t_first, t_end, L_in, L_out,
                               A_pre, A_dec);
}

int orc_slo_tpot_counts_requests(int32_t M, int32_t win, int32_t K, int64_t n,
                                 const int32_t* model, const int32_t* t_arr,
                                 const int32_t* t_start, const int32_t* t_first,
                                 const int32_t* t_end, const int32_t* L_in, const int32_t* L_out,
                                 const int32_t* tpot, int32_t* n_dec, int32_t* n_met) {
  return slo_tpot_counts_requests(M, win, K, n, model, t_arr, t_start, t_first, t_end, L_in,
                                  L_out, tpot, n_dec, n_met);
}

int orc_occupancy_mean_events(int32_t M, int32_t win, int32_t K, int64_t n, const int32_t* model,
                              const int32_t* req, const float* t_s, const uint8_t* phase,
                              int64_t n_req, const int32_t* req_model, const int32_t* req_t_arr,
                              int64_t* A_ms, int64_t* W_ms) {
  return occupancy_mean_events(M, win, K, n, model, req, t_s, phase, n_req, req_model, req_t_arr,
                               A_ms, W_ms);
}

int orc_slo_counts_requests(int32_t M, int32_t win, int32_t K, int64_t n, const int32_t* model,
                            const int32_t* t_arr, const int32_t* t_start, const int32_t* t_first,
                            const int32_t* t_end, const int32_t* L_in, const int32_t* L_out,
                            const int32_t* slo, int32_t* n_arr, int32_t* n_met) {
  return slo_counts_requests(M, win, K, n, model, t_arr, t_start, t_first, t_end, L_in, L_out,
                             slo, n_arr, n_met);
}

int orc_reduce_events(int32_t M, int32_t win, int32_t K, int64_t n, const int32_t* model,
                      const int32_t* req, const float* t_s, const uint8_t* phase, int64_t n_req,
                      const int32_t* req_model, const int32_t* req_t_arr, int32_t* P, int32_t* D,
                      int32_t* A, int32_t* W, int64_t* drops) {
  return reduce_events(M, win, K, n, model, req, t_s, phase, n_req, req_model, req_t_arr, P, D,
                       A, W, drops);
}

int orc_slo_counts_events(int32_t M, int32_t win, int32_t K, int64_t n_req,
                          const int32_t* req_model, const int32_t* req_t_arr,
                          const int32_t* req_ttft, const int32_t* slo, int32_t* n_arr,
                          int32_t* n_met) {
  return slo_counts_events(M, win, K, n_req, req_model, req_t_arr, req_ttft, slo, n_arr, n_met);
}

#define ORC_TYPED(SUF, T)                                                                          \
  int orc_score_##SUF(int32_t M, int32_t win, int32_t K, const int32_t* P, const int32_t* D,      \
                      const int32_t* A, const int32_t* W, const T* w_p, const T* w_q,             \
                      const T* alpha, const T* theta, const T* tau_crit, const T* tau_surplus,    \
                      T* S_carry, uint8_t* init_carry, T* S, T* Z, uint8_t* cls, int32_t* recv,   \
                      const int64_t* A_ms, const int64_t* W_ms) {                                  \
    return score<T>(M, win, K, P, D, A, W, w_p, w_q, alpha, theta, tau_crit, tau_surplus,         \
                    S_carry, init_carry, S, Z, cls, recv, A_ms, W_ms);                             \
  }                                                                                                \
  int orc_calibrate_##SUF(int32_t M, int32_t K, const T* S, const uint8_t* cls,                   \
                          const int32_t* n_arr, const int32_t* n_met, double ok_frac,             \
                          double reliability, T* theta, int64_t* degenerate) {                    \
    return calibrate<T>(M, K, S, cls, n_arr, n_met, ok_frac, reliability, theta, degenerate);     \
  }                                                                                                \
  int orc_select_##SUF(int32_t M, int32_t win, int32_t K, const T* Z, const uint8_t* cls,         \
                       const T* tau_crit, const T* tau_surplus, int64_t budget,                   \
                       const int32_t* r_min, const int32_t* footprint, int32_t fast_ms,           \
                       int32_t slow_ms, int32_t pacing_cap, int32_t* r_inout, void* moves,        \
                       int64_t cap, int64_t* n_moves) {                                            \
    return select_moves<T>(M, win, K, Z, cls, tau_crit, tau_surplus, budget, r_min, footprint,    \
                           fast_ms, slow_ms, pacing_cap, r_inout, static_cast<Move*>(moves), cap, \
                           n_moves);                                                               \
  }

ORC_TYPED(f32, float)
ORC_TYPED(f64, double)

// Per-(model, SLO class) signal with a class per request (Sec. II-A gives
// each model one class): every (model, class) pair becomes a model of its own,
// id model * n_classes + class; ids outside the grid become -1.
int orc_class_models(int64_t n, const int32_t* model, const int32_t* cls, int32_t M, int32_t C,
                     int32_t* out) {
  if (n < 0 || M < 1 || C < 1) return 1;
  for (int64_t i = 0; i < n; ++i) {
    const bool ok = model[i] >= 0 && model[i] < M && cls[i] >= 0 && cls[i] < C;
    out[i] = ok ? model[i] * C + cls[i] : -1;
  }
  return 0;
}

int orc_rank_f32(int32_t M, int32_t K, const float* Z, const uint8_t* cls, int32_t* recv,
                 int32_t* order) {
  return rank_windows<float>(M, K, Z, cls, recv, order);
}
int orc_rank_f64(int32_t M, int32_t K, const double* Z, const uint8_t* cls, int32_t* recv,
                 int32_t* order) {
  return rank_windows<double>(M, K, Z, cls, recv, order);
}

#define ORC_CLOSED_LOOP(SUF, T)                                                                   \
  int orc_closed_loop_##SUF(                                                                       \
      int32_t M, int32_t win, int32_t K, int64_t n, const int32_t* model, const int32_t* t_arr,    \
      const int32_t* d_first, const int32_t* d_total, const int32_t* L_in, const int32_t* L_out,   \
      const T* w_p, const T* w_q, const T* alpha, const T* theta, const T* tau_crit,               \
      const T* tau_surplus, int64_t budget, const int32_t* r0, const int32_t* r_min,               \
      const int32_t* footprint, int32_t fast_ms, int32_t slow_ms, int32_t pacing_cap,              \
      int32_t wake_ms, int32_t sleep_ms, const int32_t* guard_ms, int32_t* t_start,                \
      int32_t* t_first, int32_t* t_end, int32_t* r_out, Move* moves, int64_t cap,                  \
      int64_t* n_moves, T* Z_out, uint8_t* cls_out) {                                              \
    return closed_loop<T>(M, win, K, n, model, t_arr, d_first, d_total, L_in, L_out, w_p, w_q,     \
                          alpha, theta, tau_crit, tau_surplus, budget, r0, r_min, footprint,       \
                          fast_ms, slow_ms, pacing_cap, wake_ms, sleep_ms, guard_ms, t_start,      \
                          t_first, t_end, r_out, moves, cap, n_moves, Z_out, cls_out);             \
  }
ORC_CLOSED_LOOP(f32, float)
ORC_CLOSED_LOOP(f64, double)

int orc_move_size(void) { return (int)sizeof(Move); }

}  // extern "C"
