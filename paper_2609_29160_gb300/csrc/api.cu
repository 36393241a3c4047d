// C ABI of the library: argument checks, workspace layout and the launch order
// of each entry point. Every array argument is a device pointer owned by the
// caller; nothing here allocates.
#include <algorithm>
#include <cstring>
#include <numeric>
#include <vector>

#include "internal.h"

using namespace tre;

namespace {

// ---- phase tracing ----------------------------------------------------------
const char* const kPhaseName[TRE_TRACE_PHASES] = {"reduce", "gauge_scan", "aggregate", "score",
                                                  "receiver", "slo_counts", "calibrate",
                                                  "normalize", "select", "occupancy",
                                                  "replay"};
struct TraceRec {
  int phase, launches;
  cudaEvent_t a, b;
};
struct Tracer {
  bool on = false;
  std::vector<cudaEvent_t> pool;
  size_t used = 0;
  std::vector<TraceRec> recs;
  cudaEvent_t next() {
    if (used == pool.size()) {
      cudaEvent_t e;
      if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
      pool.push_back(e);
    }
    return pool[used++];
  }
};
Tracer g_trace;


// A column the kernels may read: device memory, or host memory the GPU
// addresses (pinned and mapped). Plain pageable host memory is refused here,
// since a kernel reading it would fault. When the runtime cannot tell (no
// device), the launch decides.
bool gpu_addressable(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return true;
  }
  return a.type != cudaMemoryTypeUnregistered;
}

bool req_ok(const tre_requests* r) {
  if (!r || r->n < 0) return false;
  if (r->n == 0) return true;
  const void* cols[7] = {r->model, r->t_arr_ms, r->t_start_ms, r->t_first_ms, r->t_end_ms,
                         r->L_in, r->L_out};
  for (const void* c : cols)
    if (!c || !gpu_addressable(c)) return false;
  return true;
}

bool ev_ok(const tre_events* e) {
  if (!e || e->n < 0 || e->n_req < 0) return false;
  if (e->n > 0 && !(e->model && e->req && e->t_s && e->phase)) return false;
  if ((e->n > 0 || e->n_req > 0) && !(e->req_model && e->req_t_arr_ms && e->req_ttft_ms))
    return false;
  return true;
}

ReqCols cols_of(const tre_requests* r) {
  return ReqCols{r->model, r->t_arr_ms, r->t_start_ms, r->t_first_ms, r->t_end_ms, r->L_in,
                 r->L_out, r->n};
}

EvCols cols_of(const tre_events* e) {
  return EvCols{e->model, e->req, e->t_s, e->phase, e->n, e->n_req, e->req_model,
                e->req_t_arr_ms, e->req_ttft_ms};
}

// Workspace protocol shared by every entry point: with ws == NULL report the
// size, else check it.
tre_status ws_check(const Arena& a, void* ws, size_t* ws_bytes, bool& query) {
  query = ws == nullptr;
  if (query) {
    *ws_bytes = a.off ? a.off : 256;
    return TRE_OK;
  }
  if (reinterpret_cast<uintptr_t>(ws) & 255) return TRE_EINVAL;
  if (*ws_bytes < a.off) return TRE_ENOMEM;
  return TRE_OK;
}

tre_status cuda_status(cudaError_t e) { return e == cudaSuccess ? TRE_OK : TRE_ECUDA; }

}  // namespace

namespace tre {

bool grid_ok(const tre_grid* g) {
  return g && g->n_models >= 1 && g->n_models <= 1024 && g->window_ms >= 1 && g->n_windows >= 0 &&
         (int64_t)g->n_windows * g->window_ms < (int64_t)2147483647;
}

bool counts_ok(const tre_counts* c) {
  return c && c->P && c->D && c->A && c->W && (!c->A_ms) == (!c->W_ms);
}

bool prof_ok(const tre_profile* p, bool need_theta_tau) {
  if (!p || (p->dtype != TRE_F32 && p->dtype != TRE_F64)) return false;
  if (!(p->w_p && p->w_q && p->alpha)) return false;
  if (need_theta_tau && !(p->theta && p->tau_crit && p->tau_surplus)) return false;
  return true;
}

// An event recorded while the stream is being captured into a CUDA graph is
// recorded as a graph node (the external flag), so a replay of the graph
// records it and the phase can be timed from the replay.
static cudaError_t record(cudaEvent_t e, cudaStream_t s) {
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(s, &cs) != cudaSuccess) {
    cudaGetLastError();
    cs = cudaStreamCaptureStatusNone;
  }
  return cs == cudaStreamCaptureStatusActive ? cudaEventRecordWithFlags(e, s, cudaEventRecordExternal)
                                             : cudaEventRecord(e, s);
}

Scope::Scope(int phase, int launches, cudaStream_t st) : s(st) {
  if (!g_trace.on) return;
  a = g_trace.next();
  b = g_trace.next();
  if (!a || !b) return;
  ph = phase;
  n = launches;
  live = record(a, s) == cudaSuccess;
}

Scope::~Scope() {
  if (live && record(b, s) == cudaSuccess) g_trace.recs.push_back(TraceRec{ph, n, a, b});
}

}  // namespace tre

namespace {

template <class T> T to_t(double v) { return (T)v; }

// ---- tss_score --------------------------------------------------------------
// one-series table over a whole grid (per-model alpha comes from the profile)
template <class T> SeriesTable<T> single_series(const tre_grid* g) {
  SeriesTable<T> t;
  std::memset(&t, 0, sizeof(t));
  t.n = 1;
  t.M = g->n_models;
  t.off[0] = 0;
  t.K[0] = g->n_windows;
  t.win[0] = g->window_ms;
  t.alpha[0] = (T)0.01;  // alpha is per model on the device: size segments for slow smoothing
  series_segments(t);
  return t;
}

template <class T>
tre_status score_typed(const tre_grid* g, const tre_counts* in, const tre_profile* p,
                       void* S_carry, uint8_t* init_carry, void* S_out, void* Z_out,
                       uint8_t* cls_out, int32_t* recv_out, void* ws, size_t* ws_bytes,
                       tre_diag* diag, cudaStream_t s) {
  const int M = g->n_models, K = g->n_windows;
  SeriesTable<T> tab = single_series<T>(g);
  Arena a(ws);
  ScoreWs<T> w;
  score_ws_layout<T>(a, M, (int64_t)K * M, tab.seg_base[1], w);
  bool query;
  tre_status st = ws_check(a, ws, ws_bytes, query);
  if (st != TRE_OK || query) return st;
  cudaError_t e;
  {
    Scope sc(kScore, score_launches(tab), s);
    e = launch_score<T>(tab, in->P, in->D, in->A, in->W, static_cast<const T*>(p->w_p),
                        static_cast<const T*>(p->w_q), static_cast<const T*>(p->alpha),
                        static_cast<const T*>(p->theta), static_cast<const T*>(p->tau_crit),
                        static_cast<const T*>(p->tau_surplus), static_cast<T*>(S_carry),
                        init_carry, static_cast<T*>(S_out), static_cast<T*>(Z_out), cls_out, w,
                        diag, s, in->A_ms, in->W_ms);
  }
  if (!e && recv_out) {
    Scope sc(kReceiver, 1, s);
    e = launch_receiver<T>(M, K, static_cast<const T*>(Z_out), cls_out, recv_out, s);
  }
  return cuda_status(e);
}

// ---- tss_calibrate ----------------------------------------------------------
template <class T>
tre_status calibrate_typed(const tre_grid* g, const tre_requests* req, const tre_events* ev,
                           const tre_counts* in, const tre_profile* p, const int32_t* slo_ms,
                           double ok_frac, double rel, void* theta, void* S_out,
                           uint8_t* cls_out, void* ws, size_t* ws_bytes, tre_diag* diag,
                           cudaStream_t s) {
  const int M = g->n_models, K = g->n_windows;
  SeriesTable<T> tab = single_series<T>(g);
  Arena a(ws);
  unsigned long long* slo = a.take<unsigned long long>((size_t)K * M);
  T* S_ws = a.take<T>((size_t)K * M);
  uint8_t* cls_ws = a.take<uint8_t>((size_t)K * M);
  // the smoothed series and idle classes go to the caller's arrays when given
  T* S = S_out ? static_cast<T*>(S_out) : S_ws;
  uint8_t* cls = cls_out ? cls_out : cls_ws;
  ScoreWs<T> sw;
  score_ws_layout<T>(a, M, (int64_t)K * M, tab.seg_base[1], sw);
  CalibWs<T> cw;
  calib_ws_layout<T>(a, (int64_t)K * M, M, cw);
  bool query;
  tre_status st = ws_check(a, ws, ws_bytes, query);
  if (st != TRE_OK || query) return st;
  cudaError_t e;
  {
    Scope sc(kSlo, 1, s);
    e = req ? launch_slo_requests(cols_of(req), M, g->window_ms, K, slo, slo_ms, s)
            : launch_slo_events(cols_of(ev), M, g->window_ms, K, slo, slo_ms, s);
  }
  if (!e) {
    Scope sc(kScore, score_launches(tab), s);
    e = launch_score<T>(tab, in->P, in->D, in->A, in->W, static_cast<const T*>(p->w_p),
                        static_cast<const T*>(p->w_q), static_cast<const T*>(p->alpha), nullptr,
                        nullptr, nullptr, nullptr, nullptr, S, nullptr, cls, sw, diag, s,
                        in->A_ms, in->W_ms);
  }
  if (!e) {
    Scope sc(kCalibrate, 3, s);
    e = launch_calibrate<T>(tab, S, cls, slo, ok_frac, rel, static_cast<T*>(theta), cw, diag, s);
  }
  return cuda_status(e);
}

// ---- tre_select_moves -------------------------------------------------------
template <class T>
tre_status select_typed(const tre_grid* g, const void* Z, const uint8_t* cls,
                        const tre_profile* p, const tre_ctrl* c, int32_t* r_inout, tre_move* moves,
                        int64_t cap, int64_t* n_moves, void* ws, size_t* ws_bytes, tre_diag* diag,
                        cudaStream_t s) {
  WalkBatch<T> b;
  std::memset(&b, 0, sizeof(b));
  b.M = g->n_models;
  b.n_inst = 1;
  b.n_series = 1;
  b.n_tau = 1;
  b.n_cap = 1;
  b.series_off[0] = 0;
  b.series_K[0] = g->n_windows;
  b.series_win[0] = g->window_ms;
  b.cap_list[0] = c->pacing_cap;
  b.Z = static_cast<const T*>(Z);
  b.cls = cls;
  b.tau_crit = static_cast<const T*>(p->tau_crit);
  b.tau_surp = static_cast<const T*>(p->tau_surplus);
  b.budget = c->budget;
  b.r_min = c->r_min;
  b.footprint = c->footprint;
  b.r0 = r_inout;
  b.fast_ms = c->fast_ms;
  b.slow_ms = c->slow_ms;
  b.r_out = r_inout;
  b.moves = moves;
  b.moves_cap = cap;
  b.n_moves = n_moves;
  b.diag = diag;
  Arena a(ws);
  WalkWs w;
  walk_ws_layout<T>(a, b, w);
  bool query;
  tre_status st = ws_check(a, ws, ws_bytes, query);
  if (st != TRE_OK || query) return st;
  Scope sc(kSelect, 2, s);
  int n_launch = 0;
  const cudaError_t e = launch_walk<T>(b, w, s, &n_launch);
  sc.set_launches(n_launch);
  return cuda_status(e);
}

// ---- tre_sweep --------------------------------------------------------------
struct SweepPlan {
  int M, n_series, base_win, Kb;
  std::vector<int> K, q;           // per window length
  std::vector<int64_t> off;        // per series element offset
  int64_t total;                   // sum over series of K*M
  int Kmax;
};

bool sweep_plan(const tre_sweep_spec* sp, SweepPlan& pl) {
  if (!sp || sp->n_models < 1 || sp->n_models > 1024 || sp->duration_ms < 1) return false;
  if (sp->n_traces < 1 || !sp->traces || sp->n_win < 1 || sp->n_win > 16 || !sp->window_ms ||
      !sp->alpha)
    return false;
  if (sp->n_tau < 1 || sp->n_tau > kMaxTau || !sp->tau_crit) return false;
  if (sp->n_cap < 1 || sp->n_cap > kMaxCap || !sp->pacing_cap) return false;
  if ((int64_t)sp->n_traces * sp->n_win > kMaxSeries) return false;
  if (sp->dtype != TRE_F32 && sp->dtype != TRE_F64) return false;
  if (!(sp->w_p && sp->w_q && sp->tau_surplus && sp->slo_ttft_ms && sp->r0)) return false;
  if (!(sp->ctrl.r_min && sp->ctrl.footprint) || sp->ctrl.fast_ms < 1 || sp->ctrl.slow_ms < 1)
    return false;
  for (int c = 0; c < sp->n_cap; ++c)
    if (sp->pacing_cap[c] < 0 || sp->pacing_cap[c] > 255) return false;
  for (int t = 0; t < sp->n_traces; ++t)
    if (!req_ok(&sp->traces[t])) return false;
  pl.M = sp->n_models;
  pl.base_win = *std::min_element(sp->window_ms, sp->window_ms + sp->n_win);
  if (pl.base_win < 1 || sp->duration_ms % pl.base_win) return false;
  pl.Kb = sp->duration_ms / pl.base_win;
  pl.K.resize(sp->n_win);
  pl.q.resize(sp->n_win);
  pl.Kmax = 0;
  for (int w = 0; w < sp->n_win; ++w) {
    const int win = sp->window_ms[w];
    if (win < 1 || win % pl.base_win || sp->duration_ms % win) return false;
    pl.q[w] = win / pl.base_win;
    pl.K[w] = sp->duration_ms / win;
    pl.Kmax = std::max(pl.Kmax, pl.K[w]);
  }
  pl.n_series = sp->n_traces * sp->n_win;
  pl.off.resize(pl.n_series);
  int64_t o = 0;
  for (int s = 0; s < pl.n_series; ++s) {
    pl.off[s] = o;
    o += (int64_t)pl.K[s % sp->n_win] * pl.M;
  }
  pl.total = o;
  return true;
}

template <class T>
tre_status sweep_typed(const tre_sweep_spec* sp, const SweepPlan& pl, const tre_sweep_out* out,
                       void* ws, size_t* ws_bytes, tre_diag* diag, cudaStream_t s) {
  const int M = pl.M;
  const int NT = sp->n_traces;
  // series table: series si = trace * n_win + w
  SeriesTable<T> tab;
  std::memset(&tab, 0, sizeof(tab));
  tab.n = pl.n_series;
  tab.M = M;
  for (int si = 0; si < pl.n_series; ++si) {
    const int w = si % sp->n_win;
    tab.off[si] = pl.off[si];
    tab.K[si] = pl.K[w];
    tab.win[si] = sp->window_ms[w];
    tab.alpha[si] = to_t<T>(sp->alpha[w]);
  }
  const int n_seg = series_segments(tab);
  AggPlan ag;
  std::memset(&ag, 0, sizeof(ag));
  ag.n_traces = NT;
  ag.n_win = sp->n_win;
  ag.M = M;
  ag.Kb = pl.Kb;
  for (int w = 0; w < sp->n_win; ++w) {
    ag.q[w] = pl.q[w];
    ag.Kq[w] = pl.K[w];
  }
  for (int t = 0; t < NT; ++t)
    for (int w = 0; w < sp->n_win; ++w) ag.out_off[t][w] = pl.off[t * sp->n_win + w];

  // Gauge scan and coarsening in one blocked pass when the ratios allow a
  // short common block; the reduction then writes the base window length's
  // counts in place (if it is one of the lengths).
  GaugePlan gp;
  std::memset(&gp, 0, sizeof(gp));
  gp.n_traces = NT;
  gp.n_win = sp->n_win;
  gp.M = M;
  gp.Kb = pl.Kb;
  gp.base_w = -1;
  int64_t lcm = 1;
  for (int w = 0; w < sp->n_win; ++w) {
    gp.q[w] = pl.q[w];
    if (pl.q[w] == 1 && gp.base_w < 0) gp.base_w = w;
    lcm = lcm / std::gcd<int64_t>(lcm, pl.q[w]) * pl.q[w];
    if (lcm > 4096) break;
  }
  const bool fused = lcm <= 4096 && sp->n_win <= kGaugeMaxWin;
  if (fused) {
    // the shortest row block that holds whole coarse windows of every length
    // and at least kGaugeMinBlk rows: more (trace, block, model) threads keep
    // more loads in flight
    gp.blk = (int)(lcm * ((kGaugeMinBlk + lcm - 1) / lcm));
    gp.nblk = (pl.Kb + gp.blk - 1) / gp.blk;
    for (int t = 0; t < NT; ++t) {
      for (int w = 0; w < sp->n_win; ++w) gp.out_off[t][w] = pl.off[t * sp->n_win + w];
      gp.in_off[t] = gp.base_w >= 0 ? gp.out_off[t][gp.base_w] : (int64_t)t * pl.Kb * M;
    }
  }
  const bool in_place = fused && gp.base_w >= 0;

  Arena a(ws);
  const size_t nb = (size_t)pl.Kb * M * NT;
  int32_t* Pb = in_place ? nullptr : a.take<int32_t>(nb);
  int32_t* Db = in_place ? nullptr : a.take<int32_t>(nb);
  int32_t* Ab = fused ? nullptr : a.take<int32_t>(nb);
  int32_t* Wb = fused ? nullptr : a.take<int32_t>(nb);
  unsigned long long* slob = in_place ? nullptr : a.take<unsigned long long>(nb);
  ReduceWs rw;
  reduce_ws_layout(a, M, pl.Kb, NT, 0, rw);
  const size_t tot = (size_t)pl.total;
  int32_t* P = out->P ? out->P : a.take<int32_t>(tot);
  int32_t* D = out->D ? out->D : a.take<int32_t>(tot);
  int32_t* A = out->A ? out->A : a.take<int32_t>(tot);
  int32_t* W = out->W ? out->W : a.take<int32_t>(tot);
  T* S = out->S ? static_cast<T*>(out->S) : a.take<T>(tot);
  T* Z = out->Z ? static_cast<T*>(out->Z) : a.take<T>(tot);
  uint8_t* idle = a.take<uint8_t>(tot);
  unsigned long long* slo = a.take<unsigned long long>(tot);
  if (in_place) {
    Pb = P;
    Db = D;
    slob = slo;
  }
  ScoreWs<T> sw;
  score_ws_layout<T>(a, M, (int64_t)tot, n_seg, sw);
  CalibWs<T> cw;
  calib_ws_layout<T>(a, (int64_t)tot, tab.n * M, cw);
  WalkBatch<T> b;
  std::memset(&b, 0, sizeof(b));
  b.M = M;
  b.n_series = pl.n_series;
  b.n_tau = sp->n_tau;
  b.n_cap = sp->n_cap;
  b.n_inst = pl.n_series * sp->n_tau * sp->n_cap;
  for (int si = 0; si < pl.n_series; ++si) {
    b.series_off[si] = pl.off[si];
    b.series_K[si] = pl.K[si % sp->n_win];
    b.series_win[si] = sp->window_ms[si % sp->n_win];
  }
  for (int t = 0; t < sp->n_tau; ++t) b.tau_list[t] = to_t<T>(sp->tau_crit[t]);
  for (int c = 0; c < sp->n_cap; ++c) b.cap_list[c] = sp->pacing_cap[c];
  b.Z = Z;
  b.cls = idle;
  b.tau_crit = nullptr;
  b.tau_surp = static_cast<const T*>(sp->tau_surplus);
  b.budget = sp->ctrl.budget;
  b.r_min = sp->ctrl.r_min;
  b.footprint = sp->ctrl.footprint;
  b.r0 = sp->r0;
  b.fast_ms = sp->ctrl.fast_ms;
  b.slow_ms = sp->ctrl.slow_ms;
  b.r_out = out->r_final;
  b.moves = out->moves;
  b.moves_cap = out->moves_cap;
  b.n_moves = out->n_moves;
  b.diag = diag;
  WalkWs wk;
  walk_ws_layout<T>(a, b, wk);
  bool query;
  tre_status st = ws_check(a, ws, ws_bytes, query);
  if (st != TRE_OK || query) return st;

  T* theta = static_cast<T*>(out->theta);
  std::vector<ReqCols> cols(NT);
  for (int t = 0; t < NT; ++t) cols[t] = cols_of(&sp->traces[t]);
  cudaError_t e;
  {
    Scope sc(kReduce, 2, s);
    std::vector<int64_t> red_off(NT);
    for (int t = 0; t < NT; ++t) red_off[t] = in_place ? gp.in_off[t] : (int64_t)t * pl.Kb * M;
    e = launch_reduce_requests(cols.data(), NT, M, pl.base_win, pl.Kb, Pb, Db, rw, slob,
                               sp->slo_ttft_ms, diag, s, red_off.data());
  }
  if (fused) {
    if (!e) {
      Scope sc(kScan, 2, s);
      e = launch_gauge_prefix(gp, rw, s);
    }
    if (!e) {
      Scope sc(kAggregate, 1, s);
      e = launch_gauge_apply(gp, rw, Pb, Db, slob, P, D, A, W, slo, s);
    }
  } else {
    if (!e) {
      Scope sc(kScan, 3, s);
      e = launch_gauge_scan(M, pl.Kb, rw, Ab, Wb, s);
    }
    if (!e) {
      Scope sc(kAggregate, 1, s);
      e = launch_aggregate(ag, Pb, Db, Ab, Wb, slob, P, D, A, W, slo, s);
    }
  }
  if (!e) {
    Scope sc(kScore, score_launches(tab), s);
    e = launch_score<T>(tab, P, D, A, W, static_cast<const T*>(sp->w_p),
                        static_cast<const T*>(sp->w_q), nullptr, nullptr, nullptr, nullptr,
                        nullptr, nullptr, S, nullptr, idle, sw, diag, s);
  }
  if (!e) {
    Scope sc(kCalibrate, 3, s);
    e = launch_calibrate<T>(tab, S, idle, slo, sp->ok_frac, sp->reliability, theta, cw, diag, s);
  }
  if (!e) {
    Scope sc(kNormalize, 1, s);
    e = launch_normalize<T>(tab, S, idle, theta, nullptr, to_t<T>(sp->tau_crit[0]),
                            static_cast<const T*>(sp->tau_surplus), Z, out->cls, s);
  }
  if (e) return TRE_ECUDA;
  Scope sc(kSelect, 2, s);
  int n_launch = 0;
  const cudaError_t e2 = launch_walk<T>(b, wk, s, &n_launch);
  sc.set_launches(n_launch);
  return cuda_status(e2);
}

}  // namespace

namespace {

// ---- stage-aware signal (Sec. VIII) ----------------------------------------
template <class T>
tre_status stage_calibrate_typed(const tre_grid* g, const tre_requests* req, const tre_counts* in,
                                 const int32_t* A_pre, const int32_t* A_dec,
                                 const tre_profile* p, const int32_t* ttft_ms,
                                 const int32_t* tpot_ms, double ok_frac, double rel,
                                 void* th_pre, void* th_dec, void* ws, size_t* ws_bytes,
                                 tre_diag* diag, cudaStream_t s) {
  const int M = g->n_models, K = g->n_windows;
  const size_t cells = (size_t)K * M;
  SeriesTable<T> tab = single_series<T>(g);
  Arena a(ws);
  unsigned long long* ttft = a.take<unsigned long long>(cells);
  unsigned long long* tpot = a.take<unsigned long long>(cells);
  int32_t* zero = a.take<int32_t>(cells);
  T* ones = a.take<T>((size_t)M);
  T* S = a.take<T>(cells);
  uint8_t* cls = a.take<uint8_t>(cells);
  ScoreWs<T> sw;
  score_ws_layout<T>(a, M, (int64_t)cells, tab.seg_base[1], sw);
  CalibWs<T> cw;
  calib_ws_layout<T>(a, (int64_t)cells, M, cw);
  bool query;
  tre_status st = ws_check(a, ws, ws_bytes, query);
  if (st != TRE_OK || query) return st;
  const T* w_p = static_cast<const T*>(p->w_p);
  const T* w_q = static_cast<const T*>(p->w_q);
  const T* alpha = static_cast<const T*>(p->alpha);
  cudaError_t e;
  {
    Scope sc(kSlo, 1, s);
    e = launch_stage_requests(cols_of(req), M, g->window_ms, K, nullptr, nullptr, ttft, tpot,
                              ttft_ms, tpot_ms, s);
  }
  if (!e) e = cudaMemsetAsync(zero, 0, cells * sizeof(int32_t), s);
  if (!e) e = launch_fill<T>(ones, M, (T)1, s);
  // prefill: (P/dt) / max(A_prefill + w_q W, 1), calibrated on TTFT
  if (!e) {
    Scope sc(kScore, score_launches(tab), s);
    e = launch_score<T>(tab, in->P, zero, A_pre, in->W, ones, w_q, alpha, nullptr, nullptr,
                        nullptr, nullptr, nullptr, S, nullptr, cls, sw, diag, s);
  }
  if (!e) {
    Scope sc(kCalibrate, 3, s);
    e = launch_calibrate<T>(tab, S, cls, ttft, ok_frac, rel, static_cast<T*>(th_pre), cw, diag, s);
  }
  // decode: (D/dt) / max(A_decode, 1), calibrated on TPOT
  if (!e) {
    Scope sc(kScore, score_launches(tab), s);
    e = launch_score<T>(tab, zero, in->D, A_dec, zero, w_p, w_q, alpha, nullptr, nullptr,
                        nullptr, nullptr, nullptr, S, nullptr, cls, sw, diag, s);
  }
  if (!e) {
    Scope sc(kCalibrate, 3, s);
    e = launch_calibrate<T>(tab, S, cls, tpot, ok_frac, rel, static_cast<T*>(th_dec), cw, diag, s);
  }
  return cuda_status(e);
}

template <class T>
tre_status stage_score_typed(const tre_grid* g, const tre_counts* in, const int32_t* A_pre,
                             const int32_t* A_dec, const tre_profile* p, const void* th_pre,
                             const void* th_dec, void* S_pre, void* Z_pre, uint8_t* cls_pre,
                             void* S_dec, void* Z_dec, uint8_t* cls_dec, void* ws,
                             size_t* ws_bytes, tre_diag* diag, cudaStream_t s) {
  const int M = g->n_models, K = g->n_windows;
  const size_t cells = (size_t)K * M;
  SeriesTable<T> tab = single_series<T>(g);
  Arena a(ws);
  int32_t* zero = a.take<int32_t>(cells);
  T* ones = a.take<T>((size_t)M);
  ScoreWs<T> sw;
  score_ws_layout<T>(a, M, (int64_t)cells, tab.seg_base[1], sw);
  bool query;
  tre_status st = ws_check(a, ws, ws_bytes, query);
  if (st != TRE_OK || query) return st;
  const T* w_q = static_cast<const T*>(p->w_q);
  const T* alpha = static_cast<const T*>(p->alpha);
  const T* tc = static_cast<const T*>(p->tau_crit);
  const T* tsu = static_cast<const T*>(p->tau_surplus);
  cudaError_t e = cudaMemsetAsync(zero, 0, cells * sizeof(int32_t), s);
  if (!e) e = launch_fill<T>(ones, M, (T)1, s);
  if (!e) {
    Scope sc(kScore, score_launches(tab), s);
    e = launch_score<T>(tab, in->P, zero, A_pre, in->W, ones, w_q, alpha,
                        static_cast<const T*>(th_pre), tc, tsu, nullptr, nullptr,
                        static_cast<T*>(S_pre), static_cast<T*>(Z_pre), cls_pre, sw, diag, s);
  }
  if (!e) {
    Scope sc(kScore, score_launches(tab), s);
    e = launch_score<T>(tab, zero, in->D, A_dec, zero, static_cast<const T*>(p->w_p), w_q,
                        alpha, static_cast<const T*>(th_dec), tc, tsu, nullptr, nullptr,
                        static_cast<T*>(S_dec), static_cast<T*>(Z_dec), cls_dec, sw, diag, s);
  }
  return cuda_status(e);
}

}  // namespace

namespace {

// ---- tre_replay -------------------------------------------------------------
template <class T>
tre_status replay_typed(const tre_grid* g, const tre_latent* lat, const tre_profile* p,
                        const tre_ctrl* c, const int32_t* r0, const tre_replay_spec* sp,
                        const int32_t* slo_ms, const tre_replay_out* out, void* ws,
                        size_t* ws_bytes, tre_diag* diag, cudaStream_t s) {
  ReplayBatch<T> b;
  std::memset(&b, 0, sizeof(b));
  b.M = g->n_models;
  b.win = g->window_ms;
  b.K = g->n_windows;
  const int n_tau = sp ? sp->n_tau : 0, n_cap = sp ? sp->n_cap : 0;
  b.n_tau = n_tau;
  b.n_cap = n_cap > 0 ? n_cap : 1;
  for (int t = 0; t < n_tau; ++t) b.tau_list[t] = (T)sp->tau_crit[t];
  for (int q = 0; q < b.n_cap; ++q) b.cap_list[q] = n_cap > 0 ? sp->pacing_cap[q] : c->pacing_cap;
  b.n_inst = (n_tau > 0 ? n_tau : 1) * b.n_cap;
  b.w_p = static_cast<const T*>(p->w_p);
  b.w_q = static_cast<const T*>(p->w_q);
  b.alpha = static_cast<const T*>(p->alpha);
  b.theta = static_cast<const T*>(p->theta);
  b.tau_crit = static_cast<const T*>(p->tau_crit);
  b.tau_surp = static_cast<const T*>(p->tau_surplus);
  b.budget = c->budget;
  b.r0 = r0;
  b.r_min = c->r_min;
  b.footprint = c->footprint;
  b.fast_ms = c->fast_ms;
  b.slow_ms = c->slow_ms;
  b.wake_ms = sp ? sp->wake_ms : 0;
  b.sleep_ms = sp ? sp->sleep_ms : 0;
  b.guard_ms = sp ? sp->guard_ttft_ms : nullptr;
  b.lat = ReplayLatent{lat->n, lat->model, lat->t_arr_ms, lat->d_first_ms, lat->d_total_ms,
                       lat->L_in, lat->L_out};
  b.slo_ms = slo_ms;
  b.hcap = (int)c->budget;
  b.o_ts = out->t_start_ms;
  b.o_tf = out->t_first_ms;
  b.o_te = out->t_end_ms;
  b.Z = static_cast<T*>(out->Z);
  b.cls = out->cls;
  b.moves = out->moves;
  b.moves_cap = out->moves_cap;
  b.n_moves = out->n_moves;
  b.r_final = out->r_final;
  b.slo_met = out->slo_met;
  b.served = out->served;
  b.diag = diag;
  Arena a(ws);
  ReplayWs w;
  replay_ws_layout<T>(a, b, w);
  bool query;
  tre_status st = ws_check(a, ws, ws_bytes, query);
  if (st != TRE_OK || query) return st;
  Scope sc(kReplay, 4, s);
  return cuda_status(launch_replay<T>(b, w, s));
}

}  // namespace

extern "C" {

void tre_trace_enable(int on) {
  g_trace.on = on != 0;
  g_trace.recs.clear();
  g_trace.used = 0;
}

tre_status tre_trace_collect(tre_trace* out) {
  if (!out) return TRE_EINVAL;
  std::memset(out, 0, sizeof(*out));
  out->n_phases = TRE_TRACE_PHASES;
  for (int i = 0; i < TRE_TRACE_PHASES; ++i) out->name[i] = kPhaseName[i];
  tre_status st = TRE_OK;
  for (const TraceRec& r : g_trace.recs) {
    float ms = 0.f;
    if (cudaEventSynchronize(r.b) != cudaSuccess || cudaEventElapsedTime(&ms, r.a, r.b)) {
      st = TRE_ECUDA;
      continue;
    }
    out->ms[r.phase] += ms;
    out->calls[r.phase] += 1;
    out->launches[r.phase] += r.launches;
  }
  g_trace.recs.clear();
  g_trace.used = 0;
  return st;
}

const char* tre_status_str(tre_status s) {
  switch (s) {
    case TRE_OK: return "ok";
    case TRE_EINVAL: return "invalid argument";
    case TRE_ENOMEM: return "workspace too small";
    case TRE_ECUDA: return "CUDA error";
    case TRE_EOVERFLOW: return "move list overflow";
    case TRE_ETIMEOUT: return "device wait timed out";
  }
  return "unknown status";
}

tre_status tss_window_reduce(const tre_grid* grid, const tre_requests* req, const tre_events* ev,
                             tre_counts out, void* ws, size_t* ws_bytes, tre_diag* diag,
                             tre_stream stream) {
  if (!grid_ok(grid) || !ws_bytes || (!req) == (!ev)) return TRE_EINVAL;
  if (req ? !req_ok(req) : !ev_ok(ev)) return TRE_EINVAL;
  if (!counts_ok(&out)) return TRE_EINVAL;
  if (ws && !diag) return TRE_EINVAL;
  const int M = grid->n_models, K = grid->n_windows;
  Arena a(ws);
  ReduceWs w;
  reduce_ws_layout(a, M, K, 1, ev ? ev->n_req : 0, w);
  bool query;
  tre_status st = ws_check(a, ws, ws_bytes, query);
  if (st != TRE_OK || query) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e;
  {
    Scope sc(kReduce, req ? 2 : 3, s);   // clearing + reduction; or three event passes
    const ReqCols rc = req ? cols_of(req) : ReqCols{};
    e = req ? launch_reduce_requests(&rc, 1, M, grid->window_ms, K, out.P, out.D, w, nullptr,
                                     nullptr, diag, s)
            : launch_reduce_events(cols_of(ev), M, grid->window_ms, K, out.P, out.D, w, diag, s);
  }
  if (!e) {
    Scope sc(kScan, 3, s);
    e = launch_gauge_scan(M, K, w, out.A, out.W, s);
  }
  if (!e && out.A_ms) {
    Scope sc(kOccupancy, 3 + (req ? req->n > 0 : ev->n_req > 0), s);
    e = req ? launch_occupancy_mean(cols_of(req), M, grid->window_ms, K, w, out.A_ms, out.W_ms, s)
            : launch_occupancy_mean_events(cols_of(ev), M, grid->window_ms, K, w, out.A_ms,
                                           out.W_ms, s);
  }
  return cuda_status(e);
}

tre_status tss_score(const tre_grid* grid, const tre_counts* in, const tre_profile* prof,
                     void* S_carry, uint8_t* init_carry, void* S_out, void* Z_out,
                     uint8_t* cls_out, int32_t* recv_out, void* ws, size_t* ws_bytes,
                     tre_diag* diag, tre_stream stream) {
  if (!grid_ok(grid) || !ws_bytes || !counts_ok(in) || !prof_ok(prof, true)) return TRE_EINVAL;
  if (!S_out || !Z_out || !cls_out || (!S_carry) != (!init_carry)) return TRE_EINVAL;
  if (ws && !diag) return TRE_EINVAL;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (prof->dtype == TRE_F32)
    return score_typed<float>(grid, in, prof, S_carry, init_carry, S_out, Z_out, cls_out,
                              recv_out, ws, ws_bytes, diag, s);
  return score_typed<double>(grid, in, prof, S_carry, init_carry, S_out, Z_out, cls_out, recv_out,
                             ws, ws_bytes, diag, s);
}

tre_status tss_rank(const tre_grid* grid, tre_dtype dtype, const void* Z, const uint8_t* cls,
                    int32_t* recv_out, int32_t* donors_out, tre_stream stream) {
  if (!grid_ok(grid) || (dtype != TRE_F32 && dtype != TRE_F64)) return TRE_EINVAL;
  if (grid->n_windows > 0 && (recv_out || donors_out) && (!Z || !cls)) return TRE_EINVAL;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int M = grid->n_models, K = grid->n_windows;
  Scope sc(kReceiver, 1, s);
  return cuda_status(
      dtype == TRE_F32
          ? launch_rank<float>(M, K, static_cast<const float*>(Z), cls, recv_out, donors_out, s)
          : launch_rank<double>(M, K, static_cast<const double*>(Z), cls, recv_out, donors_out,
                                s));
}

tre_status tss_calibrate(const tre_grid* grid, const tre_requests* req, const tre_events* ev,
                         const tre_counts* in, const tre_profile* prof, const int32_t* slo_ttft_ms,
                         double ok_frac, double reliability, void* theta_out, void* S_out,
                         uint8_t* cls_out, void* ws, size_t* ws_bytes, tre_diag* diag,
                         tre_stream stream) {
  if (!grid_ok(grid) || !ws_bytes || (!req) == (!ev) || !counts_ok(in) || !prof_ok(prof, false))
    return TRE_EINVAL;
  if (req ? !req_ok(req) : !ev_ok(ev)) return TRE_EINVAL;
  if (!slo_ttft_ms || !theta_out) return TRE_EINVAL;
  if (ws && !diag) return TRE_EINVAL;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (prof->dtype == TRE_F32)
    return calibrate_typed<float>(grid, req, ev, in, prof, slo_ttft_ms, ok_frac, reliability,
                                  theta_out, S_out, cls_out, ws, ws_bytes, diag, s);
  return calibrate_typed<double>(grid, req, ev, in, prof, slo_ttft_ms, ok_frac, reliability,
                                 theta_out, S_out, cls_out, ws, ws_bytes, diag, s);
}

tre_status tss_normalize(const tre_grid* grid, const tre_profile* prof, const void* S,
                         const uint8_t* idle_cls, void* Z_out, uint8_t* cls_out,
                         int32_t* recv_out, tre_stream stream) {
  if (!grid_ok(grid) || !prof_ok(prof, true)) return TRE_EINVAL;
  if (grid->n_windows > 0 && (!S || !idle_cls || !Z_out || !cls_out)) return TRE_EINVAL;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int M = grid->n_models, K = grid->n_windows;
  if (K == 0) return TRE_OK;
  cudaError_t e;
  if (prof->dtype == TRE_F32) {
    const SeriesTable<float> tab = single_series<float>(grid);
    {
      Scope sc(kNormalize, 1, s);
      e = launch_normalize<float>(tab, static_cast<const float*>(S), idle_cls,
                                  static_cast<const float*>(prof->theta),
                                  static_cast<const float*>(prof->tau_crit), 0.f,
                                  static_cast<const float*>(prof->tau_surplus),
                                  static_cast<float*>(Z_out), cls_out, s);
    }
    if (!e && recv_out) {
      Scope sc(kReceiver, 1, s);
      e = launch_receiver<float>(M, K, static_cast<const float*>(Z_out), cls_out, recv_out, s);
    }
  } else {
    const SeriesTable<double> tab = single_series<double>(grid);
    {
      Scope sc(kNormalize, 1, s);
      e = launch_normalize<double>(tab, static_cast<const double*>(S), idle_cls,
                                   static_cast<const double*>(prof->theta),
                                   static_cast<const double*>(prof->tau_crit), 0.0,
                                   static_cast<const double*>(prof->tau_surplus),
                                   static_cast<double*>(Z_out), cls_out, s);
    }
    if (!e && recv_out) {
      Scope sc(kReceiver, 1, s);
      e = launch_receiver<double>(M, K, static_cast<const double*>(Z_out), cls_out, recv_out,
                                  s);
    }
  }
  return cuda_status(e);
}

tre_status tre_select_moves(const tre_grid* grid, const void* Z, const uint8_t* cls,
                            const tre_profile* prof, const tre_ctrl* ctrl, int32_t* r_inout,
                            tre_move* moves, int64_t moves_cap, int64_t* n_moves_out, void* ws,
                            size_t* ws_bytes, tre_diag* diag, tre_stream stream) {
  if (!grid_ok(grid) || !ws_bytes || !Z || !cls || !prof || !ctrl || !r_inout || !n_moves_out)
    return TRE_EINVAL;
  if (prof->dtype != TRE_F32 && prof->dtype != TRE_F64) return TRE_EINVAL;
  if (!prof->tau_crit || !prof->tau_surplus || !ctrl->r_min || !ctrl->footprint) return TRE_EINVAL;
  if (ctrl->fast_ms < 1 || ctrl->slow_ms < 1 || ctrl->pacing_cap < 0 || ctrl->pacing_cap > 255)
    return TRE_EINVAL;
  if (moves_cap < 0 || (moves_cap > 0 && !moves)) return TRE_EINVAL;
  if (ws && !diag) return TRE_EINVAL;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (prof->dtype == TRE_F32)
    return select_typed<float>(grid, Z, cls, prof, ctrl, r_inout, moves, moves_cap, n_moves_out,
                               ws, ws_bytes, diag, s);
  return select_typed<double>(grid, Z, cls, prof, ctrl, r_inout, moves, moves_cap, n_moves_out,
                              ws, ws_bytes, diag, s);
}

tre_status tre_sweep(const tre_sweep_spec* spec, const tre_sweep_out* out, void* ws,
                     size_t* ws_bytes, tre_diag* diag, tre_stream stream) {
  SweepPlan pl;
  if (!ws_bytes || !sweep_plan(spec, pl) || !out) return TRE_EINVAL;
  if (!out->theta || !out->n_moves || !out->r_final || out->moves_cap < 0 ||
      (out->moves_cap > 0 && !out->moves))
    return TRE_EINVAL;
  if (ws && !diag) return TRE_EINVAL;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (spec->dtype == TRE_F32) return sweep_typed<float>(spec, pl, out, ws, ws_bytes, diag, s);
  return sweep_typed<double>(spec, pl, out, ws, ws_bytes, diag, s);
}

tre_status tss_stage_gauges(const tre_grid* grid, const tre_requests* req, int32_t* A_prefill,
                            int32_t* A_decode, void* ws, size_t* ws_bytes, tre_diag* diag,
                            tre_stream stream) {
  if (!grid_ok(grid) || !ws_bytes || !req_ok(req) || !A_prefill || !A_decode) return TRE_EINVAL;
  if (ws && !diag) return TRE_EINVAL;
  const int M = grid->n_models, K = grid->n_windows;
  Arena a(ws);
  ReduceWs w;
  reduce_ws_layout(a, M, K, 1, 0, w);
  bool query;
  tre_status st = ws_check(a, ws, ws_bytes, query);
  if (st != TRE_OK || query) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e;
  {
    // the prefill differences take the running slot and the decode ones the
    // waiting slot of the gauge scan
    Scope sc(kReduce, 1, s);
    e = launch_stage_requests(cols_of(req), M, grid->window_ms, K, w.dA, w.dW, nullptr, nullptr,
                              nullptr, nullptr, s);
  }
  if (!e) {
    Scope sc(kScan, 3, s);
    e = launch_gauge_scan(M, K, w, A_prefill, A_decode, s);
  }
  return cuda_status(e);
}

tre_status tss_stage_calibrate(const tre_grid* grid, const tre_requests* req,
                               const tre_counts* in, const int32_t* A_prefill,
                               const int32_t* A_decode, const tre_profile* prof,
                               const int32_t* slo_ttft_ms, const int32_t* slo_tpot_ms,
                               double ok_frac, double reliability, void* theta_prefill,
                               void* theta_decode, void* ws, size_t* ws_bytes, tre_diag* diag,
                               tre_stream stream) {
  if (!grid_ok(grid) || !ws_bytes || !req_ok(req) || !counts_ok(in) || in->A_ms ||
      !prof_ok(prof, false))
    return TRE_EINVAL;
  if (!A_prefill || !A_decode || !slo_ttft_ms || !slo_tpot_ms || !theta_prefill || !theta_decode)
    return TRE_EINVAL;
  if (ws && !diag) return TRE_EINVAL;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (prof->dtype == TRE_F32)
    return stage_calibrate_typed<float>(grid, req, in, A_prefill, A_decode, prof, slo_ttft_ms,
                                        slo_tpot_ms, ok_frac, reliability, theta_prefill,
                                        theta_decode, ws, ws_bytes, diag, s);
  return stage_calibrate_typed<double>(grid, req, in, A_prefill, A_decode, prof, slo_ttft_ms,
                                       slo_tpot_ms, ok_frac, reliability, theta_prefill,
                                       theta_decode, ws, ws_bytes, diag, s);
}

tre_status tss_stage_score(const tre_grid* grid, const tre_counts* in, const int32_t* A_prefill,
                           const int32_t* A_decode, const tre_profile* prof,
                           const void* theta_prefill, const void* theta_decode, void* S_prefill,
                           void* Z_prefill, uint8_t* cls_prefill, void* S_decode, void* Z_decode,
                           uint8_t* cls_decode, void* ws, size_t* ws_bytes, tre_diag* diag,
                           tre_stream stream) {
  if (!grid_ok(grid) || !ws_bytes || !counts_ok(in) || in->A_ms || !prof_ok(prof, false))
    return TRE_EINVAL;
  if (!prof->tau_crit || !prof->tau_surplus || !A_prefill || !A_decode || !theta_prefill ||
      !theta_decode)
    return TRE_EINVAL;
  if (!S_prefill || !Z_prefill || !cls_prefill || !S_decode || !Z_decode || !cls_decode)
    return TRE_EINVAL;
  if (ws && !diag) return TRE_EINVAL;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (prof->dtype == TRE_F32)
    return stage_score_typed<float>(grid, in, A_prefill, A_decode, prof, theta_prefill,
                                    theta_decode, S_prefill, Z_prefill, cls_prefill, S_decode,
                                    Z_decode, cls_decode, ws, ws_bytes, diag, s);
  return stage_score_typed<double>(grid, in, A_prefill, A_decode, prof, theta_prefill,
                                   theta_decode, S_prefill, Z_prefill, cls_prefill, S_decode,
                                   Z_decode, cls_decode, ws, ws_bytes, diag, s);
}

tre_status tre_replay(const tre_grid* grid, const tre_latent* lat, const tre_profile* prof,
                      const tre_ctrl* ctrl, const int32_t* r0, const tre_replay_spec* spec,
                      const int32_t* slo_ttft_ms, const tre_replay_out* out, void* ws,
                      size_t* ws_bytes, tre_diag* diag, tre_stream stream) {
  if (!grid_ok(grid) || grid->n_models > 64 || !ws_bytes || !lat || lat->n < 0 || !ctrl || !r0 ||
      !out)
    return TRE_EINVAL;
  if (lat->n > 0 && !(lat->model && lat->t_arr_ms && lat->d_first_ms && lat->d_total_ms &&
                      lat->L_in && lat->L_out))
    return TRE_EINVAL;
  if (lat->n > 2147483647ll) return TRE_EINVAL;
  if (!prof_ok(prof, true)) return TRE_EINVAL;
  if (!ctrl->r_min || !ctrl->footprint || ctrl->fast_ms < 1 || ctrl->slow_ms < 1 ||
      ctrl->budget < 0 || ctrl->budget > 65536)
    return TRE_EINVAL;
  if (spec) {
    if (spec->n_tau < 0 || spec->n_tau > kMaxTau || (spec->n_tau > 0 && !spec->tau_crit))
      return TRE_EINVAL;
    if (spec->n_cap < 0 || spec->n_cap > kMaxCap || (spec->n_cap > 0 && !spec->pacing_cap))
      return TRE_EINVAL;
    for (int q = 0; q < spec->n_cap; ++q)
      if (spec->pacing_cap[q] < 0 || spec->pacing_cap[q] > 255) return TRE_EINVAL;
    if (spec->wake_ms < 0 || spec->sleep_ms < 0) return TRE_EINVAL;
  }
  if ((!spec || spec->n_cap == 0) && (ctrl->pacing_cap < 0 || ctrl->pacing_cap > 255))
    return TRE_EINVAL;
  if (!out->n_moves || !out->r_final || out->moves_cap < 0 || (out->moves_cap > 0 && !out->moves))
    return TRE_EINVAL;
  if ((!out->t_start_ms) != (!out->t_first_ms) || (!out->t_start_ms) != (!out->t_end_ms))
    return TRE_EINVAL;
  if ((!out->Z) != (!out->cls) || (out->slo_met && !slo_ttft_ms)) return TRE_EINVAL;
  if (ws && !diag) return TRE_EINVAL;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (prof->dtype == TRE_F32)
    return replay_typed<float>(grid, lat, prof, ctrl, r0, spec, slo_ttft_ms, out, ws, ws_bytes,
                               diag, s);
  return replay_typed<double>(grid, lat, prof, ctrl, r0, spec, slo_ttft_ms, out, ws, ws_bytes,
                              diag, s);
}

}  // extern "C"
