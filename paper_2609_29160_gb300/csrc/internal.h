// Host-side launchers shared between the library's translation units.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "tre.h"

namespace tre {

// Bump allocator over the caller's workspace. With base == nullptr it only
// measures (the query pass of every entry point).
struct Arena {
  char* base;
  size_t off = 0;
  explicit Arena(void* b) : base(static_cast<char*>(b)) {}
  template <class T> T* take(size_t count) {
    off = (off + 255) & ~size_t(255);
    T* p = base ? reinterpret_cast<T*>(base + off) : nullptr;
    off += count * sizeof(T);
    return p;
  }
};

struct ReqCols {
  const int32_t *model, *t_arr, *t_start, *t_first, *t_end, *L_in, *L_out;
  int64_t n;
};

struct EvCols {
  const int32_t *model, *req;
  const float* t_s;
  const uint8_t* phase;
  int64_t n, n_req;
  const int32_t *req_model, *req_t_arr, *req_ttft;
};

// ---- reduce.cu ------------------------------------------------------------
// Reduction scratch: diff arrays [K+1][M] for the gauges, per-request first and
// last event ticks, scan partials.
struct ReduceWs {
  int32_t *dA, *dW;
  int32_t *first, *last;       // events only, [n_req]
  int32_t *partA, *partW;      // [n_chunks][M]
};
void reduce_ws_layout(Arena& a, int M, int K, int64_t n_req, ReduceWs& w);
// slo (may be null): packed per-(window, model) arrivals (low 32 bits) and
// arrivals that met the TTFT bound (high 32 bits), added to.
cudaError_t launch_reduce_requests(const ReqCols& r, int M, int win, int K, int32_t* P,
                                   int32_t* D, ReduceWs& w, unsigned long long* slo,
                                   const int32_t* slo_ms, tre_diag* diag, cudaStream_t s);
cudaError_t launch_reduce_events(const EvCols& e, int M, int win, int K, int32_t* P, int32_t* D,
                                 ReduceWs& w, tre_diag* diag, cudaStream_t s);
cudaError_t launch_slo_requests(const ReqCols& r, int M, int win, int K,
                                unsigned long long* slo, const int32_t* slo_ms, cudaStream_t s);
cudaError_t launch_slo_events(const EvCols& e, int M, int win, int K, unsigned long long* slo,
                              const int32_t* slo_ms, cudaStream_t s);
// inclusive scan of the diff arrays over windows -> A, W
cudaError_t launch_gauge_scan(int M, int K, ReduceWs& w, int32_t* A, int32_t* W, cudaStream_t s);
// exact aggregation of a base grid to a coarser one (q base windows per window)
cudaError_t launch_aggregate(int M, int Kq, int q, const int32_t* P, const int32_t* D,
                             const int32_t* A, const int32_t* W, const unsigned long long* slo,
                             int32_t* Pq, int32_t* Dq, int32_t* Aq, int32_t* Wq,
                             unsigned long long* sloq, cudaStream_t s);

// ---- score.cu -------------------------------------------------------------
template <class T> struct ScoreWs {
  T *sum_m, *sum_c, *sum_ci;   // per-segment affine summaries [n_seg][M]
  int32_t* sum_h;
  T* start_S;                  // start state used by the stored trajectory [n_seg][M]
  int32_t* start_init;
  T *end_S, *end_S2;           // end states (double buffered) [n_seg][M]
  int32_t *end_init, *end_init2;
  int n_seg, seg_len;
};
template <class T> void score_ws_layout(Arena& a, int M, int K, ScoreWs<T>& w);
// profile arrays are device pointers of T; theta may be null (Z not written)
template <class T>
cudaError_t launch_score(int M, int win, int K, const int32_t* P, const int32_t* D,
                         const int32_t* A, const int32_t* W, const T* w_p, const T* w_q,
                         const T* alpha, const T* theta, const T* tau_crit, const T* tau_surp,
                         T* S_carry, uint8_t* init_carry, T* S, T* Z, uint8_t* cls,
                         ScoreWs<T>& w, tre_diag* diag, cudaStream_t s);
// same, with one alpha value for all models given on the host
template <class T>
cudaError_t launch_score_alpha(int M, int win, int K, const int32_t* P, const int32_t* D,
                               const int32_t* A, const int32_t* W, const T* w_p, const T* w_q,
                               T alpha, T* S, uint8_t* cls, ScoreWs<T>& w, tre_diag* diag,
                               cudaStream_t s);
// Z = S / theta and regions (tau arrays device, or one host value when the
// pointer is null)
template <class T>
cudaError_t launch_normalize(int M, int K, const T* S, const uint8_t* idle_cls, const T* theta,
                             const T* tau_crit, T tau_crit_v, const T* tau_surp, T* Z,
                             uint8_t* cls, cudaStream_t s);
template <class T>
cudaError_t launch_receiver(int M, int K, const T* Z, const uint8_t* cls, int32_t* recv,
                            cudaStream_t s);

// ---- calibrate.cu ---------------------------------------------------------
template <class T> struct CalibWs {
  void* keys;                  // [M][K] packed keys (u32 for float, u64 for double)
  int32_t* thr;                // healthy threshold table
};
template <class T> void calib_ws_layout(Arena& a, int M, int K, CalibWs<T>& w);
template <class T>
cudaError_t launch_calibrate(int M, int K, const T* S, const uint8_t* cls,
                             const unsigned long long* slo, double ok_frac, double reliability,
                             T* theta, CalibWs<T>& w, tre_diag* diag, cudaStream_t s);

// ---- select.cu ------------------------------------------------------------
// One controller instance per (series, tau, cap). The small per-series tables
// travel by value in the kernel parameters.
constexpr int kMaxSeries = 64, kMaxTau = 32, kMaxCap = 32;
template <class T> struct WalkBatch {
  int M, n_inst, n_series, n_tau, n_cap;
  int64_t series_off[kMaxSeries];  // element offset of each series in Z / cls
  int32_t series_K[kMaxSeries];
  int32_t series_win[kMaxSeries];
  T tau_list[kMaxTau];             // used when tau_crit == null
  int32_t cap_list[kMaxCap];
  const T* Z;
  const uint8_t* cls;
  const T* tau_crit;               // device [M] or null
  const T* tau_surp;               // device [M]
  int64_t budget;
  const int32_t *r_min, *footprint, *r0;
  int32_t fast_ms, slow_ms;
  int32_t* r_out;                  // [n_inst][M] (may alias r0 for one instance)
  tre_move* moves;
  int64_t moves_cap;
  int64_t* n_moves;                // [n_inst]
  tre_diag* diag;
};
template <class T> cudaError_t launch_walk(const WalkBatch<T>& b, cudaStream_t s);

}  // namespace tre
