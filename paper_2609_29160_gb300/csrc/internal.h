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

// ---- device.cu ------------------------------------------------------------
// Launch state kept per GPU (the device current on the calling thread), safe to
// call from several host threads.
// SM count of the current device.
int device_sm_count();
// Raises fn's dynamic shared-memory limit to `bytes` (and, with max_carveout,
// asks for the largest shared-memory carveout) once per (device, function).
cudaError_t func_smem_once(const void* fn, int bytes, bool max_carveout);

// ---- api.cu: argument checks shared by the entry points ---------------------
bool grid_ok(const tre_grid* g);
bool counts_ok(const tre_counts* c);
bool prof_ok(const tre_profile* p, bool need_theta_tau);

// ---- api.cu: phase tracing (tre_trace_enable / tre_trace_collect) -----------
enum Phase { kReduce, kScan, kAggregate, kScore, kReceiver, kSlo, kCalibrate, kNormalize,
             kSelect, kOccupancy, kReplay };
// While tracing is on, brackets the launches of one phase with a pair of
// events recorded on the stream (constructed before, destroyed after them).
class Scope {
 public:
  Scope(int phase, int launches, cudaStream_t st);
  ~Scope();
  Scope(const Scope&) = delete;
  Scope& operator=(const Scope&) = delete;
  void set_launches(int launches) { n = launches; }

 private:
  cudaStream_t s;
  cudaEvent_t a = nullptr, b = nullptr;
  int ph = 0, n = 0;
  bool live = false;
};

// ---- reduce.cu ------------------------------------------------------------
// Reduction scratch for a batch of traces on one grid: diff arrays
// [trace][K+1][M] for the gauges, per-request first and last event ticks, scan
// partials [trace][chunk][M].
struct ReduceWs {
  int32_t *dA, *dW;
  int32_t *first, *last;       // events only, [n_req]
  int32_t *partA, *partW;
  int64_t part_cap;            // partial entries per trace
  int n_traces;
};
constexpr int kGaugeMinBlk = 16;   // shortest row block of the fused gauge pass
constexpr int kGaugeMaxWin = 8;    // most window lengths the fused gauge pass takes
void reduce_ws_layout(Arena& a, int M, int K, int n_traces, int64_t n_req, ReduceWs& w);
// Request records of n_traces traces (host array of column sets) on one grid;
// trace t writes P, D (and the packed SLO counts when slo != null) at element
// offset out_off[t] (host array; null: t*K*M). slo packs per-(window, model)
// arrivals (low 32 bits) and the arrivals that met the TTFT bound (high 32
// bits).
cudaError_t launch_reduce_requests(const ReqCols* traces, int n_traces, int M, int win, int K,
                                   int32_t* P, int32_t* D, ReduceWs& w, unsigned long long* slo,
                                   const int32_t* slo_ms, tre_diag* diag, cudaStream_t s,
                                   const int64_t* out_off = nullptr);
cudaError_t launch_reduce_events(const EvCols& e, int M, int win, int K, int32_t* P, int32_t* D,
                                 ReduceWs& w, tre_diag* diag, cudaStream_t s);
cudaError_t launch_slo_requests(const ReqCols& r, int M, int win, int K,
                                unsigned long long* slo, const int32_t* slo_ms, cudaStream_t s);
cudaError_t launch_slo_events(const EvCols& e, int M, int win, int K, unsigned long long* slo,
                              const int32_t* slo_ms, cudaStream_t s);
// inclusive scan of the diff arrays over windows -> A, W (trace t at t*K*M)
cudaError_t launch_gauge_scan(int M, int K, ReduceWs& w, int32_t* A, int32_t* W, cudaStream_t s);
// Time-averaged occupancy of one trace's request records: request-milliseconds
// running and waiting per (window, model), int64 [K][M]; reuses the gauge
// diff and partial arrays of w (call after the gauge scan of the same trace)
cudaError_t launch_occupancy_mean(const ReqCols& r, int M, int win, int K, ReduceWs& w,
                                  int64_t* A_ms, int64_t* W_ms, cudaStream_t s);
// The same for token events: spans from the per-request first/last ticks the
// event reduction left in w (call after launch_reduce_events and the gauge scan)
cudaError_t launch_occupancy_mean_events(const EvCols& ev, int M, int win, int K, ReduceWs& w,
                                         int64_t* A_ms, int64_t* W_ms, cudaStream_t s);
// exact coarsening of every trace's base grid to every window length: counts
// add over q base windows, gauges are read at the last base window
struct AggPlan {
  int n_traces, n_win, M, Kb;
  int32_t q[16], Kq[16];
  int64_t out_off[64][16];      // element offset of (trace, window length) in the outputs
};
// Gauge scan and coarsening in one pass over row blocks (sweeps): inputs are
// the diff arrays in the reduction scratch and the base P, D, SLO counts at
// in_off[trace]; the base window length (base_w >= 0) gets its gauges written
// in place, every other length its counts and gauges at out_off.
struct GaugePlan {
  int n_traces, n_win, M, Kb;
  int blk, nblk, base_w;
  int32_t q[16];
  int64_t out_off[64][16];
  int64_t in_off[64];
};
// passes 1-2: block sums of the diffs and their exclusive prefixes
cudaError_t launch_gauge_prefix(const GaugePlan& gp, ReduceWs& w, cudaStream_t s);
// pass 3: base gauges and every coarser window length
cudaError_t launch_gauge_apply(const GaugePlan& gp, ReduceWs& w, const int32_t* Pin,
                               const int32_t* Din, const unsigned long long* sloin, int32_t* P,
                               int32_t* D, int32_t* A, int32_t* W, unsigned long long* slo,
                               cudaStream_t s);
cudaError_t launch_aggregate(const AggPlan& plan, const int32_t* P, const int32_t* D,
                             const int32_t* A, const int32_t* W, const unsigned long long* slo,
                             int32_t* Pq, int32_t* Dq, int32_t* Aq, int32_t* Wq,
                             unsigned long long* sloq, cudaStream_t s);

// ---- stage.cu -------------------------------------------------------------
// One pass over request records kept by the reduction's rules: the +1/-1
// window differences of the running gauge split at the first token (prefill
// [t_start, t_first) into dPre, decode [t_first, t_end) into dDec, each
// [K+1][M], cleared here; both null = skipped) and the packed TTFT and TPOT
// calibration counts at the arrival window (count + met << 32, [K][M], cleared
// here; both null = skipped).
cudaError_t launch_stage_requests(const ReqCols& r, int M, int win, int K, int32_t* dPre,
                                  int32_t* dDec, unsigned long long* ttft,
                                  unsigned long long* tpot, const int32_t* ttft_ms,
                                  const int32_t* tpot_ms, cudaStream_t s);
template <class T> cudaError_t launch_fill(T* p, int64_t n, T v, cudaStream_t s);

// ---- series tables ----------------------------------------------------------
// A batch of series (one per (trace, window length) in a sweep, one for the
// single-trace entry points) laid out back to back: series s occupies elements
// [off[s], off[s] + K[s]*M) of every per-window array. Passed by value.
constexpr int kMaxSeries = 64, kMaxTau = 32, kMaxCap = 32;
template <class T> struct SeriesTable {
  int n, M;
  int64_t off[kMaxSeries];
  int32_t K[kMaxSeries];
  int32_t win[kMaxSeries];
  T alpha[kMaxSeries];            // per series, used when the per-model alpha is null
  int32_t seg_len[kMaxSeries];    // smoothing chunk length of the series
  int32_t seg_base[kMaxSeries + 1];  // prefix sum of segments per series
};
// fill seg_len / seg_base from K (returns the total segment count)
template <class T> int series_segments(SeriesTable<T>& t);

// ---- score.cu -------------------------------------------------------------
template <class T> struct ScoreWs {
  T* raw;                      // Eq. 1 value per element (idle windows: a marker NaN)
  T* start_S;                  // per (segment, model): state the stored run started from
  int32_t* start_init;
  T* end_S;                    // per (segment, model): state after the segment
  int32_t* end_init;
  int32_t* active;             // per (segment, model): non-idle windows (long tables)
  int cap_seg;                 // segments the arrays hold (per model)
};
template <class T> void score_ws_layout(Arena& a, int M, int64_t elems, int n_seg, ScoreWs<T>& w);
// Eq. 1, smoothing and (when theta is given) Z and regions for every series
// of the table. Profile arrays are device [M]; alpha may be null (then the
// table's per-series value is used); theta null = S only (cls = IDLE / NOM).
// The carries (device [M], may be null) apply to a one-series table.
// kernels one launch_score call issues (for the phase trace)
template <class T> int score_launches(const SeriesTable<T>& tab);
template <class T>
cudaError_t launch_score(const SeriesTable<T>& tab, const int32_t* P, const int32_t* D,
                         const int32_t* A, const int32_t* W, const T* w_p, const T* w_q,
                         const T* alpha, const T* theta, const T* tau_crit, const T* tau_surp,
                         T* S_carry, uint8_t* init_carry, T* S, T* Z, uint8_t* cls,
                         ScoreWs<T>& w, tre_diag* diag, cudaStream_t s,
                         const int64_t* A_ms = nullptr, const int64_t* W_ms = nullptr);
// Z = S / theta[series][m] and regions for every series (tau_crit device [M] or
// one value for all)
template <class T>
cudaError_t launch_normalize(const SeriesTable<T>& tab, const T* S, const uint8_t* idle_cls,
                             const T* theta, const T* tau_crit, T tau_crit_v, const T* tau_surp,
                             T* Z, uint8_t* cls, cudaStream_t s);
// donors listed per window by tss_rank
constexpr int kRankDonors = 8;
template <class T>
cudaError_t launch_rank(int M, int K, const T* Z, const uint8_t* cls, int32_t* recv,
                        int32_t* donors, cudaStream_t s);
template <class T>
cudaError_t launch_receiver(int M, int K, const T* Z, const uint8_t* cls, int32_t* recv,
                            cudaStream_t s);

// ---- calibrate.cu ---------------------------------------------------------
template <class T> struct CalibWs {
  void* keys;                  // packed keys, same element offsets as the series
  int32_t* thr;                // healthy threshold table
  void *kmin, *kmax;           // per (series, model): candidate key range
  uint32_t* ncand;             // per (series, model): candidate count
  int n_sm;                    // (series, model) pairs the range arrays hold
};
template <class T> void calib_ws_layout(Arena& a, int64_t elems, int n_sm, CalibWs<T>& w);
// theta[s*M + m] for every series of the table
template <class T>
cudaError_t launch_calibrate(const SeriesTable<T>& tab, const T* S, const uint8_t* cls,
                             const unsigned long long* slo, double ok_frac, double reliability,
                             T* theta, CalibWs<T>& w, tre_diag* diag, cudaStream_t s);

// ---- select.cu ------------------------------------------------------------
// One controller instance per (series, tau, cap). The small per-series tables
// travel by value in the kernel parameters.
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
  int32_t ent_base[kMaxSeries + 1];  // tick entries (fast then slow) per series, prefix
};
// per-(series, tau, tick) receiver and per-model donor ranks
struct WalkWs {
  int16_t* recv;
  int16_t* n_donor;   // donors with a rank at the tick
  uint16_t* rank;     // [entry][model] position in the donor order
  uint16_t* order;    // [entry][position] model at that position
  unsigned long long* packed;  // [entry] donor order, 4 bits per position (M <= 16)
  uint32_t* dmask;             // [entry] bitmask of the models with a rank (M <= 16)
  unsigned long long* dm64;    // [entry] the same for up to 64 models (warp walk)
};
// lays out the tick tables and fills b.ent_base
template <class T> void walk_ws_layout(Arena& a, WalkBatch<T>& b, WalkWs& w);
// *launches (may be null): kernels it issued
template <class T> cudaError_t launch_walk(const WalkBatch<T>& b, WalkWs& w, cudaStream_t s,
                                          int* launches = nullptr);

// ---- replay.cu ------------------------------------------------------------
// Latent requests of a closed-loop replay (what a request needs once started).
struct ReplayLatent {
  int64_t n;
  const int32_t *model, *t_arr, *d_first, *d_total, *L_in, *L_out;
};
// One controller instance per (rescue threshold, pacing cap); passed by value.
template <class T> struct ReplayBatch {
  int M, win, K, n_inst, n_tau, n_cap;
  T tau_list[kMaxTau];             // used when n_tau > 0, else tau_crit per model
  int32_t cap_list[kMaxCap];
  const T *w_p, *w_q, *alpha, *theta, *tau_crit, *tau_surp;   // device [M]
  int64_t budget;
  const int32_t *r0, *r_min, *footprint;
  int32_t fast_ms, slow_ms, wake_ms, sleep_ms;
  ReplayLatent lat;
  const int32_t* slo_ms;           // device [M] or null
  const int32_t* guard_ms;         // device [M] or null: latency guard per model
  // scratch
  const int32_t* list;             // valid request indices grouped by model
  const int4* grp;                 // per grouped request: (t_arr, d_first, d_total, index),
                                   // (L_in, L_out, -, -)
  const int32_t* base;             // [M + 1]
  const int32_t* arr_cnt;          // [K][M] arrivals
  uint32_t* acc;                   // per instance: P, D, ends, late first tokens, [K + 1][M] each
  long long* gheap;                // per instance [M][hcap] when the heaps are global
  int hcap;
  int warps_per_cta;
  int warp_bytes, heap_off;        // shared memory per warp, heap offset in it
  int act_off, acap;               // decoding-request lists: offset, entries per model
  int ring_off;                    // per-model window rings and pending far windows
  int q_off;                       // per-model staged requests
  // outputs
  int32_t *o_ts, *o_tf, *o_te;     // [n_inst][n] or null
  T* Z;                            // [n_inst][K][M] or null (with cls)
  uint8_t* cls;
  tre_move* moves;
  int64_t moves_cap;
  int64_t* n_moves;
  int32_t* r_final;
  int64_t *slo_met, *served;       // [n_inst][M] or null
  tre_diag* diag;
};
struct ReplayWs {
  int8_t* vm;
  int32_t *arr_cnt, *n_valid, *base, *list;
  int4* grp;
  uint32_t* acc;
  long long* gheap;
  bool shared_heaps;
  int warps_per_cta;
};
// lays out the scratch and fills the batch's shared-memory plan
template <class T> void replay_ws_layout(Arena& a, ReplayBatch<T>& b, ReplayWs& w);
template <class T> cudaError_t launch_replay(ReplayBatch<T>& b, ReplayWs& w, cudaStream_t s);

}  // namespace tre
