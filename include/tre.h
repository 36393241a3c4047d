/*
 * tre.h -- C ABI of the GB300 Token Service Share / TRE library (libtre.so).
 *
 * The library computes, in batch over request telemetry, the control signal and
 * the capacity moves of "Cross-Model Autoscaling for Shared LLM Serving"
 * (arXiv 2609.29160):
 *   - per-(window, model) prompt/decode token counts and running/waiting gauges
 *     (the inputs of Eq. 1, collected as in Sec. V-B),
 *   - raw Token Service Share (Eq. 1), its exponential smoothing (Sec. III-B),
 *     Z = TSS / theta (Eq. 2) and the critical / nominal / surplus regions,
 *   - the SLO calibration of the healthy boundary theta (Sec. III-B),
 *   - the per-window Eq. 3 receiver and donor release order (Sec. IV-B),
 *   - the open-loop rescue / rebalance move selection with bounded pairwise
 *     transfer under a fixed replica budget (Sec. IV-B, Eq. 3, Sec. IV-C),
 *   - a batched sweep of all of the above over many traces and settings,
 *   - and, beside the paper's signal: the time-averaged occupancy variant of
 *     Eq. 1's demand term, per-(model, SLO class) scoring through pair ids,
 *     and a scoring entry point that needs no workspace.
 *
 * Conventions (every entry point):
 *   - Array arguments are DEVICE pointers owned by the caller, unless a field
 *     says "host". The library allocates nothing and keeps no state; scratch
 *     memory comes in through `ws`.
 *   - Workspace query: call with ws == NULL; the required size is written to
 *     *ws_bytes and TRE_OK is returned without touching the device. With
 *     ws != NULL, *ws_bytes must be at least that size (else TRE_ENOMEM). `ws`
 *     must be 256-byte aligned.
 *   - Work is enqueued on `stream` (NULL = legacy default stream) and is
 *     asynchronous. Argument errors are detected on the host before anything
 *     is enqueued and returned as TRE_EINVAL. Launch failures return TRE_ECUDA.
 *   - Data problems never trap: malformed records are dropped and counted in
 *     the device-resident `tre_diag` (added to, never reset by the library:
 *     zero it before the first call), valid after the stream is synchronised.
 *   - Layout of every per-window array is row-major [n_windows][n_models].
 *   - Floating-point results are computed in the profile's dtype with one
 *     correctly rounded IEEE operation per step and no fused multiply-add, in
 *     the same order as the sequential definitions; results are reproducible
 *     bit for bit.
 * Limits: 1 <= n_models <= 1024; window_ms >= 1; n_windows * window_ms < 2^31.
 */
#ifndef TRE_H
#define TRE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* tre_stream; /* a cudaStream_t */

typedef enum {
  TRE_OK = 0,
  TRE_EINVAL = 1,    /* bad argument (host-side check, nothing enqueued) */
  TRE_ENOMEM = 2,    /* workspace smaller than the queried size */
  TRE_ECUDA = 3,     /* a CUDA launch or runtime call failed */
  TRE_EOVERFLOW = 4, /* move list longer than its capacity (reported in diag.err) */
  TRE_ETIMEOUT = 5   /* reserved: a bounded device wait gave up (reported in diag.err) */
} tre_status;

typedef enum { TRE_F32 = 0, TRE_F64 = 1 } tre_dtype;

/* Region of a model in a window (Sec. III-B): Z < tau_crit critical, Z > tau_surplus
 * surplus, otherwise nominal. A window with no tokens and no running or waiting
 * request is IDLE: never a receiver, the first donor candidate. */
enum { TRE_CRIT = 0, TRE_NOM = 1, TRE_SURP = 2, TRE_IDLE = 3 };
/* Kind of a move: fast-loop rescue or slow-loop rebalance (Sec. IV-B). */
enum { TRE_RESCUE = 1, TRE_REBALANCE = 2 };

/* Window grid: window k covers [k*window_ms, (k+1)*window_ms) milliseconds. */
typedef struct {
  int32_t n_models;
  int32_t window_ms;
  int32_t n_windows;
} tre_grid;

/* Request records, structure of arrays (int32, length n), in device memory or
 * in pinned host memory that the GPU addresses directly (cudaHostAlloc'd
 * memory under unified addressing; the kernels then read it over the host
 * link, with no separate copy; pageable host memory is refused with
 * TRE_EINVAL). Columns on 16-byte boundaries are read 16 bytes at a time.
 * Times in ms.
 * A record is valid when 0 <= model < n_models, 0 <= t_arr < n_windows*window_ms,
 * t_arr <= t_start <= t_first <= t_end, L_in >= 0 and L_out >= 1. Prompt tokens
 * count at t_first; decode token j is emitted at
 * t_first + floor(j*(t_end-t_first)/(L_out-1)) (at t_first when L_out == 1). */
typedef struct {
  int64_t n;
  const int32_t *model, *t_arr_ms, *t_start_ms, *t_first_ms, *t_end_ms, *L_in, *L_out;
} tre_requests;

/* Token-level events (device, length n): one record per emitted token, phase 0 =
 * prompt (prefill), 1 = decode; t_s in float seconds (tick = floor(t_s*1000) ms,
 * exact). The request table (device, length n_req) gives each request's model,
 * arrival ms and TTFT ms. An event is valid when its model matches
 * req_model[req], its tick lies inside the grid and phase <= 1. A request runs
 * from its first to its last valid event and waits from t_arr to its first. */
typedef struct {
  int64_t n;
  const int32_t *model, *req;
  const float* t_s;
  const uint8_t* phase;
  int64_t n_req;
  const int32_t *req_model, *req_t_arr_ms, *req_ttft_ms;
} tre_events;

/* Per-window counts (device, int32, [n_windows][n_models] each):
 * P prompt tokens, D decode tokens, A running and W waiting requests read at
 * the last millisecond of the window. Counts wrap modulo 2^32.
 * A_ms, W_ms (device, int64, [n_windows][n_models]; both NULL or both set):
 * the time-averaged occupancy -- request-milliseconds spent running
 * ([t_start, t_end)) and waiting ([t_arr, t_start)) inside the window, so that
 * A_ms / window_ms is the window's mean running count (Sec. III-A defines the
 * counts at a time t; Sec. II-B speaks of an average waiting queue).
 * tss_window_reduce fills them when they are set, from request records or from
 * token events (a request runs from its first to its last valid event and
 * waits from t_arr to its first); tss_score, tss_score_noalloc and tss_calibrate then use
 * the means A_ms / window_ms and W_ms / window_ms in Eq. 1's demand term in
 * place of A and W, and a window is IDLE when P, D, A_ms and W_ms are zero. */
typedef struct {
  int32_t *P, *D, *A, *W;
  int64_t *A_ms, *W_ms;
} tre_counts;

/* Control profile (Sec. III-B, Sec. V-B): six scalars per model, device arrays
 * of length n_models in `dtype`. */
typedef struct {
  tre_dtype dtype;
  const void *w_p, *w_q, *alpha, *theta, *tau_crit, *tau_surplus;
} tre_profile;

/* Controller (Sec. IV-B, IV-C): fixed budget in footprint units, per-model
 * replica floor and footprint (device int32 [n_models]), cadences of the fast
 * (rescue) and slow (rebalance) loops in ms, and the pacing cap: the most
 * transitions per control tick (the paper's rule is 1). */
typedef struct {
  int64_t budget;
  const int32_t *r_min, *footprint;
  int32_t fast_ms, slow_ms, pacing_cap;
} tre_ctrl;

/* One move. A transition activates one receiver replica; it is served from the
 * idle pool (donor = -1) or by releasing donor replicas, one entry per released
 * replica, all with the same (window, seq). */
typedef struct {
  int32_t window;
  int16_t recv, donor;
  uint8_t kind, seq;
  uint16_t reserved;
} tre_move;

/* Device-resident diagnostics (accumulated). */
typedef struct {
  unsigned long long dropped_range; /* record time outside the grid */
  unsigned long long dropped_model; /* model id out of range / event-request mismatch */
  unsigned long long dropped_order; /* times out of order, bad lengths, bad phase */
  unsigned long long degenerate_calib; /* models whose theta fell back */
  unsigned long long ema_resolved;  /* smoothing segments re-run to exactness */
  int32_t err;                      /* last data-dependent error status, 0 if none */
  int32_t reserved;
} tre_diag;

/*
 * tss_window_reduce -- window telemetry (Sec. III-A Eq. 1 inputs; Sec. V-B:
 * counters become window deltas, running/waiting counts are the demand).
 * Exactly one of `req` / `ev` is non-NULL (host pointer to the descriptor).
 * Writes out.P, out.D, out.A, out.W (all four required).
 */
tre_status tss_window_reduce(const tre_grid* grid, const tre_requests* req, const tre_events* ev,
                             tre_counts out, void* ws, size_t* ws_bytes, tre_diag* diag,
                             tre_stream stream);

/*
 * tss_score -- Eq. 1 raw TSS = (w_p*P/dt + D/dt) / max(A + w_q*W, 1) with dt the
 * window length in seconds; smoothing S = alpha*raw + (1-alpha)*S_prev started at
 * a model's first non-idle window and held through idle ones (Sec. III-B);
 * Z = S / theta (Eq. 2); region per window.
 * S_carry (dtype[n_models]) and init_carry (uint8[n_models]) carry the smoothing
 * state in and out across calls on consecutive window ranges; both NULL = fresh.
 * S_out, Z_out (dtype), cls_out (uint8) are [n_windows][n_models] and required.
 * recv_out (int32[n_windows], may be NULL): the Eq. 3 receiver argmin Z over
 * non-idle models, lowest index on ties, -1 if all idle.
 */
tre_status tss_score(const tre_grid* grid, const tre_counts* in, const tre_profile* prof,
                     void* S_carry, uint8_t* init_carry, void* S_out, void* Z_out,
                     uint8_t* cls_out, int32_t* recv_out, void* ws, size_t* ws_bytes,
                     tre_diag* diag, tre_stream stream);

/*
 * tss_rank -- per window, the Eq. 3 receiver and the donors it would draw on,
 * in the order the controller releases them (Sec. IV-B): idle models by index,
 * then surplus models by Z descending, then nominal models whose Z is above the
 * receiver's, by Z descending; equal Z puts the lower index first; critical
 * models and the receiver are never donors. The receiver is argmin Z over
 * non-idle models, lowest index on ties, -1 if every model is idle (the same
 * value as tss_score's recv_out). Replica floors, footprints and the idle pool
 * are not applied here; tre_select_moves applies them on control ticks.
 * Z (`dtype`) and cls (uint8) are [n_windows][n_models] in device memory, as
 * tss_score writes them; Z must not be NaN where cls is not TRE_IDLE.
 * recv_out: int32[n_windows]; donors_out: int32[n_windows][TRE_RANK_DONORS],
 * the first TRE_RANK_DONORS donors of each window and -1 in the slots left
 * over (every slot of a window without a receiver). Either may be NULL; Z and
 * cls are required when one is not. Needs no workspace and touches no diag.
 */
#define TRE_RANK_DONORS 8
tre_status tss_rank(const tre_grid* grid, tre_dtype dtype, const void* Z, const uint8_t* cls,
                    int32_t* recv_out, int32_t* donors_out, tre_stream stream);

/*
 * tss_class_models -- per-(model, SLO class) TSS with a class per request. The
 * paper gives each model one SLO class (Sec. II-A); to keep the signal per
 * (model, class) pair, every pair is treated as a model of its own:
 * model_out[i] = model[i] * n_classes + cls[i], or -1 when model[i] is outside
 * [0, n_models) or cls[i] outside [0, n_classes) (the reduction then drops the
 * record as a bad model id). Pass model_out as the records' model column and
 * n_models * n_classes as the grid's model count; slo_ttft_ms then holds one
 * bound per pair. model, cls, model_out: device int32[n] (model_out may alias
 * model). Limit: n_models * n_classes <= 1024. No workspace.
 */
tre_status tss_class_models(int64_t n, const int32_t* model, const int32_t* cls, int32_t n_models,
                            int32_t n_classes, int32_t* model_out, tre_stream stream);

/*
 * tss_calibrate -- healthy boundary theta (Sec. III-B: the lowest smoothed TSS at
 * which the SLO reliability target is still met). Calibration windows have at least
 * one arrival, are not idle and have S > 0. A window is healthy when at least
 * ok_frac of the requests arriving in it met the TTFT bound slo_ttft_ms[model]
 * (device int32[n_models]). theta[m] is the smallest S value s for which the
 * windows with S >= s are healthy in at least a `reliability` fraction; if none
 * qualifies theta = max S, if there is no calibration window theta = 1 (both
 * counted in diag.degenerate_calib). S uses w_p, w_q, alpha of `prof` (theta
 * and thresholds are ignored). Exactly one of req / ev non-NULL; `in` holds the
 * counts of the same telemetry. theta_out: dtype[n_models] on the device.
 * S_out (dtype) and cls_out (uint8), [n_windows][n_models] on the device, may
 * be NULL; when given they receive the smoothed series the boundary was taken
 * from (the S tss_score returns for the same counts and profile) and the idle
 * classes (TRE_IDLE for idle windows, TRE_NOM otherwise), which tss_normalize
 * turns into Z and regions without smoothing the series again.
 */
tre_status tss_calibrate(const tre_grid* grid, const tre_requests* req, const tre_events* ev,
                         const tre_counts* in, const tre_profile* prof, const int32_t* slo_ttft_ms,
                         double ok_frac, double reliability, void* theta_out, void* S_out,
                         uint8_t* cls_out, void* ws, size_t* ws_bytes, tre_diag* diag,
                         tre_stream stream);

/*
 * tss_normalize -- Z = S / theta (Eq. 2), the regions (Sec. IV-A: critical
 * below tau_crit, surplus above tau_surplus, idle windows stay idle) and the
 * Eq. 3 receiver, for a series smoothed already (tss_calibrate's S_out and
 * cls_out): with them it returns exactly tss_score's Z, cls and recv. S
 * (dtype) and idle_cls (uint8, TRE_IDLE marks idle windows) are
 * [n_windows][n_models] on the device; prof supplies theta, tau_crit and
 * tau_surplus (w_p, w_q, alpha are not read). Z_out (dtype) and cls_out
 * (uint8, may be idle_cls itself) are [n_windows][n_models]; recv_out
 * (int32[n_windows]) may be NULL. Needs no workspace and touches no diag.
 */
tre_status tss_normalize(const tre_grid* grid, const tre_profile* prof, const void* S,
                         const uint8_t* idle_cls, void* Z_out, uint8_t* cls_out,
                         int32_t* recv_out, tre_stream stream);

/*
 * Stage-aware signal (Sec. VIII: separate prefill and decode states; Sec. III-A
 * ties prefill to the time to first token and decode to the time per output
 * token). Request records only; records are taken or skipped by
 * tss_window_reduce's rules (drops are not counted again here).
 *
 * tss_stage_gauges -- the running gauge split at the first token, read at the
 * last millisecond of each window: A_prefill counts requests on
 * [t_start, t_first), A_decode on [t_first, t_end) (device int32
 * [n_windows][n_models] each); the two sum to tss_window_reduce's A.
 */
tre_status tss_stage_gauges(const tre_grid* grid, const tre_requests* req, int32_t* A_prefill,
                            int32_t* A_decode, void* ws, size_t* ws_bytes, tre_diag* diag,
                            tre_stream stream);

/*
 * tss_stage_calibrate -- one healthy boundary per stage, by tss_calibrate's
 * rule (Sec. III-B) on each stage's smoothed signal: the prefill signal
 * (P/dt) / max(A_prefill + w_q*W, 1) against TTFT (t_first - t_arr <=
 * slo_ttft_ms[m]) and the decode signal (D/dt) / max(A_decode, 1) against TPOT
 * (a request with L_out > 1 meets it when t_end - t_first <=
 * slo_tpot_ms[m] * (L_out - 1)), both counted at the arrival window. `in`
 * supplies P, D and W of tss_window_reduce on the same records (A is not read;
 * A_ms / W_ms must be NULL); w_q and alpha come from `prof`. theta_prefill,
 * theta_decode: dtype[n_models] on the device.
 */
tre_status tss_stage_calibrate(const tre_grid* grid, const tre_requests* req,
                               const tre_counts* in, const int32_t* A_prefill,
                               const int32_t* A_decode, const tre_profile* prof,
                               const int32_t* slo_ttft_ms, const int32_t* slo_tpot_ms,
                               double ok_frac, double reliability, void* theta_prefill,
                               void* theta_decode, void* ws, size_t* ws_bytes, tre_diag* diag,
                               tre_stream stream);

/*
 * tss_stage_score -- both stage signals, each smoothed as tss_score smooths
 * (alpha of `prof`), normalised by its own theta (Eq. 2) and classified with
 * the profile's thresholds: prefill (P/dt) / max(A_prefill + w_q*W, 1) and
 * decode (D/dt) / max(A_decode, 1). A stage window is IDLE when its tokens,
 * its running gauge and (prefill) W are all zero. Outputs [n_windows][n_models]
 * (S, Z in dtype, cls uint8), all required.
 */
tre_status tss_stage_score(const tre_grid* grid, const tre_counts* in, const int32_t* A_prefill,
                           const int32_t* A_decode, const tre_profile* prof,
                           const void* theta_prefill, const void* theta_decode, void* S_prefill,
                           void* Z_prefill, uint8_t* cls_prefill, void* S_decode, void* Z_decode,
                           uint8_t* cls_decode, void* ws, size_t* ws_bytes, tre_diag* diag,
                           tre_stream stream);

/*
 * tre_select_moves -- open-loop TRE controller over a scored trace (Sec. IV-B,
 * Eq. 3, Sec. IV-C). A window ends a fast (slow) tick when a multiple of
 * fast_ms (slow_ms) falls in (k*window_ms, (k+1)*window_ms]. At a fast tick with
 * a critical model: rescue the critical model with the lowest Z. Otherwise at a
 * slow tick: rebalance toward argmin Z over non-idle models if its Z < 1. Up to
 * pacing_cap transitions per tick toward that receiver; each takes the idle
 * pool if it covers the receiver's footprint, else releases donor replicas in
 * the order idle models (by index), surplus by Z descending, nominal by Z
 * descending (in rebalance only nominal models with Z above the receiver's);
 * never a critical model, never below its floor; an uncoverable transition
 * releases nothing and ends the tick. Regions are re-derived from Z with the
 * profile's thresholds; only the IDLE class is taken from cls.
 * r_inout (device int32[n_models]): routable replicas in, final replicas out;
 * the idle pool is budget - sum(footprint*r). moves: device tre_move[moves_cap];
 * n_moves_out (device int64[1]): number of moves produced; when it exceeds
 * moves_cap only the first moves_cap are written and diag.err = TRE_EOVERFLOW.
 */
tre_status tre_select_moves(const tre_grid* grid, const void* Z, const uint8_t* cls,
                            const tre_profile* prof, const tre_ctrl* ctrl, int32_t* r_inout,
                            tre_move* moves, int64_t moves_cap, int64_t* n_moves_out, void* ws,
                            size_t* ws_bytes, tre_diag* diag, tre_stream stream);

/*
 * tss_score_noalloc -- the same computation and outputs as tss_score, for
 * callers that cannot allocate device memory (no cudaMalloc where they run, or
 * a host that owns every allocation), so they cannot supply `ws`. It takes no
 * workspace: its scratch is a 12 MiB buffer compiled into the library, one
 * copy on every GPU that loads the library, held until the process exits. The
 * paper has no counterpart; this is a deployment variant of the scoring call.
 * Limit: n_windows * n_models <= 1048576 (for example 36000 windows x 8 models
 * or 16384 x 64); larger problems return TRE_ENOMEM before anything is
 * enqueued. The first call on a device
 * looks up the buffer's device address (make it before any stream capture);
 * the address is kept for the life of the process, so do not call this entry
 * point on a device after cudaDeviceReset of that device.
 * All calls share the one buffer: calls whose GPU work overlaps in time (other
 * streams, other host threads) race on it and must be serialised by the
 * caller. Nothing in the buffer needs to start at zero; every call writes what
 * it later reads. diag is required.
 */
tre_status tss_score_noalloc(const tre_grid* grid, const tre_counts* in, const tre_profile* prof,
                             void* S_carry, uint8_t* init_carry, void* S_out, void* Z_out,
                             uint8_t* cls_out, int32_t* recv_out, tre_diag* diag,
                             tre_stream stream);

/* Sweep description. Host fields are read during the call only. */
typedef struct {
  int32_t n_models;
  int32_t duration_ms;               /* every window length divides it */
  int32_t n_traces;
  const tre_requests* traces;        /* host array [n_traces] of device column sets */
  int32_t n_win;
  const int32_t* window_ms;          /* host [n_win]; each a multiple of the smallest */
  const double* alpha;               /* host [n_win]: smoothing weight per window length */
  int32_t n_tau;
  const double* tau_crit;            /* host [n_tau] rescue thresholds */
  int32_t n_cap;
  const int32_t* pacing_cap;         /* host [n_cap] */
  tre_dtype dtype;
  const void *w_p, *w_q, *tau_surplus; /* device [n_models] of dtype */
  const int32_t* slo_ttft_ms;        /* device [n_models] */
  double ok_frac, reliability;
  tre_ctrl ctrl;                     /* budget, floors, footprints, cadences (pacing_cap unused) */
  const int32_t* r0;                 /* device [n_models] initial replicas */
} tre_sweep_spec;

/* Sweep outputs (device). Series s = trace*n_win + w has K_s = duration_ms /
 * window_ms[w] windows; per-window arrays concatenate the series in that order
 * (series s starts at element n_models * sum_{s'<s} K_s'). Instance
 * i = (s*n_tau + t)*n_cap + c. Optional arrays may be NULL. */
typedef struct {
  int32_t *P, *D, *A, *W; /* optional counts */
  void *S, *Z;            /* optional dtype */
  uint8_t* cls;           /* optional: regions with tau_crit[0] */
  void* theta;            /* required: dtype [n_series][n_models] */
  tre_move* moves;        /* required: [n_instances][moves_cap] */
  int64_t moves_cap;
  int64_t* n_moves;       /* required: [n_instances] */
  int32_t* r_final;       /* required: [n_instances][n_models] */
} tre_sweep_out;

/*
 * tre_sweep -- the open-loop sweep: for every trace and window length, the
 * window reduction, calibration of theta, scoring, and then the move selection
 * for every (rescue threshold, pacing cap) setting (controller cadences of
 * Sec. IV-B, bounded transfer of Sec. IV-C). Equivalent, bit for bit, to calling
 * the four entry points above per (trace, window length, setting).
 */
tre_status tre_sweep(const tre_sweep_spec* spec, const tre_sweep_out* out, void* ws,
                     size_t* ws_bytes, tre_diag* diag, tre_stream stream);

/*
 * Closed-loop replay (Sec. IV-B: rescue and rebalance act on live capacity;
 * Sec. IV-C: bounded transfer; Sec. VI-D: measured sleep and wake latencies).
 * The controller's moves change the servers that serve the requests, and the
 * telemetry it scores comes from the requests as they are served:
 *  - each routable replica of a model is one server; a model's requests are
 *    served in input order (FCFS when sorted by arrival) by whichever of its
 *    servers frees first; once started a request needs d_first_ms to its first
 *    token and d_total_ms to its last;
 *  - window k is processed at T = (k+1)*window_ms: every request that can start
 *    before T starts, then window k's telemetry (tss_window_reduce's token
 *    attribution and gauges) is scored as tss_score scores it, with the
 *    smoothing carried across windows, and on a control tick the controller of
 *    tre_select_moves acts on the replica counts as they are;
 *  - a transition commits at its tick; each donor replica it releases is the
 *    donor's server that frees first: it takes no request from T on, finishes
 *    the request it serves (drain) and returns its GPU sleep_ms later; the
 *    receiver's new server starts waking when its GPU is free -- at T when the
 *    idle pool paid, else when the transition's last released donor replica
 *    has returned its GPU -- and serves wake_ms after that.
 * A latent record is served when 0 <= model < n_models, 0 <= t_arr <
 * n_windows*window_ms, 0 <= d_first <= d_total, L_in >= 0 and L_out >= 1.
 */
typedef struct {
  int64_t n;                 /* < 2^31 */
  const int32_t *model, *t_arr_ms, *d_first_ms, *d_total_ms, *L_in, *L_out;  /* device [n] */
} tre_latent;

/* Settings replayed side by side, instance i = t * n_cap + c. n_tau == 0: one
 * threshold set, the profile's tau_crit per model; else tau_crit[t] (host) for
 * every model. n_cap == 0: the control's pacing_cap; else pacing_cap[c] (host,
 * 0..255). Limits: n_tau, n_cap <= 32. wake_ms, sleep_ms >= 0.
 * guard_ttft_ms (device int32[n_models], NULL = no guard): a model breaches its
 * latency guard in window k when one of its requests got its first token in
 * window k more than guard_ttft_ms[m] after arriving. At a fast tick a breach
 * pre-empts every other rescue reason (receiver: the breaching model of lowest
 * Z); otherwise rescue takes the lowest Z among critical models and models with
 * requests waiting and no routable replica (lost capacity). A model whose guard
 * is breached is not released as a donor at that tick (Sec. IV-C release
 * guard). While a rebalance transfer is in progress (until its receiver's new
 * server serves) a rescue without a breach is deferred, and the slow loop stays
 * out of that tick (Sec. IV-B: the loops are mutually exclusive). */
typedef struct {
  int32_t n_tau;
  const double* tau_crit;
  int32_t n_cap;
  const int32_t* pacing_cap;
  int32_t wake_ms, sleep_ms;
  const int32_t* guard_ttft_ms;
} tre_replay_spec;

/* Replay outputs (device). Optional arrays may be NULL.
 * t_start_ms, t_first_ms, t_end_ms: [n_inst][n] served times (all three or
 *   none): K*window_ms for a request not started within the grid, -1 for a
 *   record that is not served;
 * Z (dtype), cls: [n_inst][n_windows][n_models] the signal the controller saw;
 * moves [n_inst][moves_cap], n_moves [n_inst] (required; n_moves above
 *   moves_cap sets diag.err = TRE_EOVERFLOW), r_final [n_inst][n_models]
 *   (required);
 * slo_met [n_inst][n_models]: served requests whose first token came within
 *   slo_ttft_ms[m] of arrival, counting a request never started as getting it
 *   at the end of the grid (needs slo_ttft_ms); served [n_inst][n_models]:
 *   requests started within the grid. */
typedef struct {
  int32_t *t_start_ms, *t_first_ms, *t_end_ms;
  void* Z;
  uint8_t* cls;
  tre_move* moves;
  int64_t moves_cap;
  int64_t* n_moves;
  int32_t* r_final;
  int64_t *slo_met, *served;
} tre_replay_out;

/*
 * tre_replay -- the closed-loop replay of one latent trace for every setting of
 * `spec` (NULL: one instance with the profile's thresholds, the control's
 * pacing cap and no actuation delay). prof: w_p, w_q, alpha, theta, tau_crit,
 * tau_surplus (device [n_models], all required); ctrl: budget (<= 65536),
 * floors, footprints, cadences; r0: device int32[n_models] initial replicas.
 * Limits: n_models <= 64. An inconsistent initial state (negative replicas or
 * floors, footprints below one, more replicas than the budget holds) is found
 * on the device: diag.err = TRE_EINVAL and nothing is replayed.
 */
tre_status tre_replay(const tre_grid* grid, const tre_latent* lat, const tre_profile* prof,
                      const tre_ctrl* ctrl, const int32_t* r0, const tre_replay_spec* spec,
                      const int32_t* slo_ttft_ms, const tre_replay_out* out, void* ws,
                      size_t* ws_bytes, tre_diag* diag, tre_stream stream);

/* Kernel-phase tracing (host side, not thread safe). While enabled, every
 * kernel phase an entry point enqueues is bracketed by a pair of CUDA events
 * recorded on the call's stream, so phases can be timed on the device inside
 * a caller's timed region. tre_trace_collect synchronises the recorded events,
 * returns per-phase device milliseconds and kernel-launch counts accumulated
 * since tracing was enabled (or since the last collect), and starts over.
 * Phases: reduce, gauge_scan, aggregate, score, receiver, slo_counts,
 * calibrate, normalize, select, occupancy (the time-averaged occupancy pass of
 * tss_window_reduce), replay (tre_replay). Calls captured into a CUDA graph
 * while tracing is on record their events as graph nodes: after a replay of
 * the graph, tre_trace_collect returns that replay's phase times. No
 * counterpart in the paper (instrumentation). */
#define TRE_TRACE_PHASES 11
typedef struct {
  int32_t n_phases;
  const char* name[TRE_TRACE_PHASES];
  double ms[TRE_TRACE_PHASES];
  int64_t calls[TRE_TRACE_PHASES];
  int64_t launches[TRE_TRACE_PHASES];
} tre_trace;
void tre_trace_enable(int on);
tre_status tre_trace_collect(tre_trace* out);

/* Human-readable name of a status. */
const char* tre_status_str(tre_status s);

#ifdef __cplusplus
}
#endif

#endif /* TRE_H */
