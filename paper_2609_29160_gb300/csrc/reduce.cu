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
constexpr int kStageBytes = 32 * 1024;   // event staging per CTA
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
constexpr int kVec = 4;               // records per thread per pass
constexpr int kMaxPerCta = 16384;     // bound that keeps the packed shared counters exact
constexpr int kFarScan = 1024;        // records that place a CTA's start-side rows
struct ReqBatch {
  int n;
  ReqCols cols[kMaxTraces];
  int64_t per_cta[kMaxTraces];
  int32_t cta_base[kMaxTraces + 1];
  unsigned long long vec_ok;          // bit t: trace t's columns allow 16-byte loads
  int64_t out_off[kMaxTraces];        // element offset of trace t's P, D, SLO counts
};

// Targets of one record fall in two places: the arrival side (the waiting
// gauge's +1 and the SLO counts at the arrival window) moves with the arrival
// order of the records, the start side (waiting -1 and running +1 at the
// start, prompt and decode tokens, running -1 at the end) with each model's
// FCFS start order. A CTA stages the arrival side over the windows its records
// arrive in, and the start side per model over a run of windows beginning at
// that model's earliest start among the CTA's records. Targets outside both
// go to global atomics.
//
// Two counters share one 32-bit shared word where both stay small: a CTA
// holds at most kMaxPerCta records, so the SLO pair (arrivals, met) packs as
// arrivals + met * 2^16, and the running/waiting gauge deltas of one start
// window pack as running + waiting * 2^16 (both signed, each bounded by the
// CTA's record count; the low half is recovered by sign extension).
struct Stage {
  int32_t* aW;        // arrival side, waiting +1: [near_rows][Mp]
  uint32_t* aS;       // arrival side, packed SLO counts: [near_rows][Mp]
  int32_t *fP, *fD;   // start side, tokens: [M][F + 1]
  int32_t* fAW;       // start side, packed gauge deltas: [M][F + 1]
  int32_t* far_lo;    // [M]
  int32_t* slo_lim;   // [M]
  uint16_t* queue;    // long decodes of this warp: record indices in the CTA
};

// Long decodes (beyond the window after the first-token window) are queued per
// warp -- the record's index in the CTA, at most one entry per record -- and,
// after the warp's last pass, walked one record per lane without a division
// per window: with y the emitted-token bound shifted so that N(T) =
// floor(y / dur), moving one window boundary adds win*(L-1) = Q*dur + R to y,
// so a window gets Q or Q + 1 tokens.


template <bool SLO, bool COPY>
__global__ void __launch_bounds__(kThreads, 4)
k_reduce_requests(const __grid_constant__ ReqBatch bt, int M, int lgMp, int win, FastDiv fd,
                  int K, int near_rows, int lgF, int32_t* __restrict__ P0,
                  int32_t* __restrict__ D0, int32_t* __restrict__ dA0, int32_t* __restrict__ dW0,
                  unsigned long long* __restrict__ slo0, const int32_t* __restrict__ slo_ms,
                  tre_diag* diag) {
  extern __shared__ unsigned long long smem[];
  unsigned long long n_range = 0, n_model = 0, n_order = 0;
  // a CTA takes slices blockIdx.x, blockIdx.x + gridDim.x, ...: one slice when
  // the grid holds them all; a smaller grid leaves SMs to other streams' work
  // (records read over the host link keep fewer SMs busy just as well)
  for (int vb = blockIdx.x; vb < bt.cta_base[bt.n]; vb += gridDim.x) {
    int t = 0;
    while (t + 1 < bt.n && bt.cta_base[t + 1] <= vb) ++t;
    const ReqCols& r = bt.cols[t];
    const bool vec = (bt.vec_ok >> t) & 1ull;
    const size_t cells1 = (size_t)(K + 1) * M;
    int32_t* P = P0 + bt.out_off[t];
    int32_t* D = D0 + bt.out_off[t];
    int32_t* dA = dA0 + t * cells1;
    int32_t* dW = dW0 + t * cells1;
    unsigned long long* slo = SLO ? slo0 + bt.out_off[t] : nullptr;
    const int64_t i0 = (int64_t)(vb - bt.cta_base[t]) * bt.per_cta[t];
    const int n_loc = (int)min64(r.n - i0, bt.per_cta[t]);
    if (n_loc <= 0) continue;
    const int Mp = 1 << lgMp, F = 1 << lgF, F1 = F + 1;
    const uint32_t span = (uint32_t)K * (uint32_t)win;
    // Columns of this CTA's records: read in place, or (COPY, for records in
    // host memory) first copied once into shared memory so that no column is
    // read twice over the host link.
    const int32_t* gcol[7] = {r.model + i0, r.t_arr + i0, r.t_start + i0, r.t_first + i0,
                              r.t_end + i0, r.L_in + i0, r.L_out + i0};
    const int32_t* colp[7];
    int32_t* recs = reinterpret_cast<int32_t*>(smem);
    const int cap_rec = COPY ? (int)bt.per_cta[t] : 0;
    if (COPY) {
#pragma unroll
      for (int c = 0; c < 7; ++c) {
        int32_t* dst = recs + (size_t)c * cap_rec;
        for (int i = threadIdx.x * 4; i < n_loc; i += kThreads * 4) {
          if (vec && i + 4 <= n_loc) {
            *reinterpret_cast<int4*>(dst + i) = *reinterpret_cast<const int4*>(gcol[c] + i);
          } else {
            for (int u = 0; u < 4 && i + u < n_loc; ++u) dst[i + u] = gcol[c][i + u];
          }
        }
        colp[c] = dst;
      }
    } else {
#pragma unroll
      for (int c = 0; c < 7; ++c) colp[c] = gcol[c];
    }
    const bool vec4 = COPY || vec;
    const int a_first = gcol[1][0], a_last = gcol[1][n_loc - 1];
    const int k_lo = a_first < 0 ? 0 : (int)min(fd.div((uint32_t)a_first), (uint32_t)K);
    const int k_hi = a_last < 0 ? 0 : (int)min(fd.div((uint32_t)a_last), (uint32_t)K);
    const int used = min(near_rows, (k_hi >= k_lo ? k_hi - k_lo + 1 : 1) + 1);
    Stage st;
    st.aW = reinterpret_cast<int32_t*>(smem + (size_t)cap_rec * 7 / 2);
    st.aS = reinterpret_cast<uint32_t*>(st.aW + (size_t)near_rows * Mp);
    st.fP = reinterpret_cast<int32_t*>(st.aS + (SLO ? (size_t)near_rows * Mp : 0));
    st.fD = st.fP + (size_t)M * F1;
    st.fAW = st.fD + (size_t)M * F1;
    st.far_lo = st.fAW + (size_t)M * F1;
    st.slo_lim = st.far_lo + M;
    st.queue = reinterpret_cast<uint16_t*>((reinterpret_cast<uintptr_t>(st.slo_lim + M) + 15) &
                                           ~(uintptr_t)15) +
               (size_t)(threadIdx.x >> 5) * (bt.per_cta[t] / (kThreads / 32));
    const int ncell = used * Mp, fcell = M * F1;
    for (int c = threadIdx.x; c < ncell; c += kThreads) {
      st.aW[c] = 0;
      if (SLO) st.aS[c] = 0;
    }
    for (int c = threadIdx.x; c < fcell; c += kThreads) { st.fP[c] = 0; st.fD[c] = 0; st.fAW[c] = 0; }
    for (int m = threadIdx.x; m < M; m += kThreads) {
      st.far_lo[m] = 0x7fffffff;
      if (SLO) st.slo_lim[m] = slo_ms[m];
    }
    __syncthreads();
    // each model's earliest start window among the CTA's first kFarScan
    // records: records come in arrival order and each model starts its requests
    // in arrival order (first come, first served), so its earliest starts are
    // among its first records; a record that starts before this window takes
    // the global path (the tests below check both ends)
    for (int b = threadIdx.x * kVec; b < min(n_loc, kFarScan); b += kThreads * kVec) {
      int mm[kVec], ss[kVec];
      if (vec4 && b + kVec <= n_loc) {
        const int4 a = *reinterpret_cast<const int4*>(colp[0] + b);
        const int4 s = *reinterpret_cast<const int4*>(colp[2] + b);
        mm[0] = a.x; mm[1] = a.y; mm[2] = a.z; mm[3] = a.w;
        ss[0] = s.x; ss[1] = s.y; ss[2] = s.z; ss[3] = s.w;
      } else {
#pragma unroll
        for (int u = 0; u < kVec; ++u) {
          const bool in = b + u < n_loc;
          mm[u] = in ? colp[0][b + u] : -1;
          ss[u] = in ? colp[2][b + u] : -1;
        }
      }
#pragma unroll
      for (int u = 0; u < kVec; ++u)
        if (mm[u] >= 0 && mm[u] < M && ss[u] >= 0)
          atomicMin(&st.far_lo[mm[u]], (int)min(fd.div((uint32_t)ss[u]), (uint32_t)K));
    }
    __syncthreads();

    // arrival-side target
    auto near_idx = [&](int k, int m) -> int {
      const unsigned rel = (unsigned)(k - k_lo);
      return rel < (unsigned)used ? (int)(rel << lgMp) + m : -1;
    };
    // start-side target of model m: shared cell index, or -1 when outside
    auto far_idx = [&](int k, int m, int lo) -> int {
      const unsigned rel = (unsigned)(k - lo);
      return rel < (unsigned)F ? m * F1 + (int)rel : -1;
    };
    auto add_tok = [&](int32_t* s_arr, int32_t* g_arr, int k, int m, int lo, int32_t v) {
      const int c = far_idx(k, m, lo);
      if (c >= 0) atomicAdd(&s_arr[c], v);
      else atomicAdd(&g_arr[(size_t)k * M + m], v);
    };
    auto add_aw = [&](int k, int m, int lo, int32_t a, int32_t w) {
      const int c = far_idx(k, m, lo);
      if (c >= 0) {
        atomicAdd(&st.fAW[c], a + w * 65536);
      } else {
        if (a) atomicAdd(&dA[(size_t)k * M + m], a);
        if (w) atomicAdd(&dW[(size_t)k * M + m], w);
      }
    };

    const unsigned full = 0xffffffffu;
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    // warp-uniform passes: lane l of a pass takes records b + l*kVec + u
    int qn = 0;   // entries in the warp's queue
    for (int wb = warp * 32 * kVec; wb < n_loc; wb += kThreads * kVec) {
      const int b = wb + lane * kVec;
      int v[7][kVec];
      if (vec4 && b + kVec <= n_loc) {
#pragma unroll
        for (int c = 0; c < 7; ++c) {
          // streaming loads, except the four columns the long-decode walk reads
          // again (model, first-token and end times, output length)
          const bool again = c == 0 || c == 3 || c == 4 || c == 6;
          const int4 q = COPY ? *reinterpret_cast<const int4*>(colp[c] + b)
                         : again ? *reinterpret_cast<const int4*>(colp[c] + b)
                                 : __ldcs(reinterpret_cast<const int4*>(colp[c] + b));
          v[c][0] = q.x; v[c][1] = q.y; v[c][2] = q.z; v[c][3] = q.w;
        }
      } else {
#pragma unroll
        for (int u = 0; u < kVec; ++u) {
          const bool in = b + u < n_loc;
#pragma unroll
          for (int c = 0; c < 7; ++c) v[c][u] = in ? colp[c][b + u] : 0;
          if (!in) v[0][u] = -1;   // marks "no record" (not counted as a drop)
        }
      }
#pragma unroll
      for (int u = 0; u < kVec; ++u) {
        const bool present = b + u < n_loc;
        const int m = v[0][u], ta = v[1][u], ts = v[2][u], tf = v[3][u], te = v[4][u];
        const int L_in = v[5][u], L = v[6][u];
        bool ok = false;
        if (present) {
          if (m < 0 || m >= M) ++n_model;
          else if (ta < 0 || (uint32_t)ta >= span) ++n_range;
          else if (!(ta <= ts && ts <= tf && tf <= te) || L_in < 0 || L < 1) ++n_order;
          else ok = true;
        }
        // decode windows after the first-token window go to the warp's queue
        bool lng = false;
        int kf = 0;
        if (ok) {
          const int lo = st.far_lo[m];
          const int ba = (int)fd.div((uint32_t)ta);
          const int bs = (int)min(fd.div((uint32_t)ts), (uint32_t)K);
          const int be_raw = (int)fd.div((uint32_t)te);
          const int be = min(be_raw, K);
          const bool tok = (uint32_t)tf < span;
          kf = tok ? (int)fd.div((uint32_t)tf) : 0;
          // decode tokens of the first-token window (d0) and, for a decode that
          // ends in the next window, of that window (d1); longer decodes leave
          // their later windows to the queue walk below
          int d0 = L, d1 = 0;
          if (tok && L != 1 && be_raw != kf) {
            // N(T) = tokens emitted before T = ceil((T - tf)(L-1)/dur)
            unsigned long long qq, rr;
            divmod((unsigned long long)((uint32_t)(kf + 1) * (uint32_t)win - (uint32_t)tf) *
                       (uint32_t)(L - 1),
                   (uint32_t)(te - tf), qq, rr);
            const int n1 = (int)(qq + (rr != 0));
            d0 = n1;
            if (be_raw == kf + 1) d1 = L - n1;
            else lng = kf + 1 < K;   // windows kf+1 .. min(be, K-1)
          }
          const int wait = ba != bs ? 1 : 0, run = bs != be ? 1 : 0;
          const uint32_t met = SLO && (tf - ta <= st.slo_lim[m]) ? 1u : 0u;
          const uint32_t rel_a = (uint32_t)(ba - k_lo);
          // bs <= kf <= be: the two ends bound every start-side target
          if (rel_a < (uint32_t)used && (uint32_t)(be - lo) < (uint32_t)F && bs >= lo) {
            const int na = (int)(rel_a << lgMp) + m;
            const int fb = m * F1 - lo;
            atomicAdd(&st.aW[na], wait);
            if (SLO) atomicAdd(&st.aS[na], 1u + (met << 16));
            atomicAdd(&st.fAW[fb + bs], run - wait * 65536);
            if (run) atomicAdd(&st.fAW[fb + be], -1);
            if (tok) {
              if (L_in) atomicAdd(&st.fP[fb + kf], L_in);
              atomicAdd(&st.fD[fb + kf], d0);
              if (d1) atomicAdd(&st.fD[fb + kf + 1], d1);
            }
          } else {
            const int na = near_idx(ba, m);
            if (wait) {
              if (na >= 0) atomicAdd(&st.aW[na], 1);
              else atomicAdd(&dW[(size_t)ba * M + m], 1);
            }
            if (SLO) {
              if (na >= 0) atomicAdd(&st.aS[na], 1u + (met << 16));
              else atomicAdd(&slo[(size_t)ba * M + m], 1ull + ((unsigned long long)met << 32));
            }
            if (run | wait) add_aw(bs, m, lo, run, -wait);
            if (run) add_aw(be, m, lo, -1, 0);
            if (tok) {
              if (L_in) add_tok(st.fP, P, kf, m, lo, L_in);
              add_tok(st.fD, D, kf, m, lo, d0);
              if (d1 && kf + 1 < K) add_tok(st.fD, D, kf + 1, m, lo, d1);
            }
          }
        }
        const unsigned qb = __ballot_sync(full, lng);
        if (lng) st.queue[qn + __popc(qb & ((1u << lane) - 1u))] = (uint16_t)(b + u);
        qn += __popc(qb);
      }
    }
    // walk the warp's long decodes, one record per lane
    __syncwarp();
    for (int i = lane; i < qn; i += 32) {
      const int j = st.queue[i];
      const int m = colp[0][j], tf = colp[3][j], te = colp[4][j], L = colp[6][j];
      const int kf = (int)fd.div((uint32_t)tf), be_raw = (int)fd.div((uint32_t)te);
      const uint32_t dur = (uint32_t)(te - tf);
      unsigned long long qq, rr;
      divmod((unsigned long long)((uint32_t)(kf + 1) * (uint32_t)win - (uint32_t)tf) *
                 (uint32_t)(L - 1),
             dur, qq, rr);
      const uint32_t q1 = (uint32_t)qq, r1 = (uint32_t)rr;
      {
        // y = x + dur - 1 at the end of window kf: N = floor(y / dur), rem = y mod dur
        uint32_t n = q1 + (r1 != 0);
        uint32_t rem = r1 ? r1 - 1 : dur - 1;
        unsigned long long Q64, R64;
        divmod((unsigned long long)(uint32_t)win * (uint32_t)(L - 1), dur, Q64, R64);
        const uint32_t Q = (uint32_t)Q64, R = (uint32_t)R64;   // Q < L: dur > win here
        const int lo = st.far_lo[m];
        const int k_full = min(be_raw - 1, K - 1);   // windows ending at or before t_end
        const int k_end = min(be_raw, K - 1);
        if ((uint32_t)(k_end - lo) < (uint32_t)F && kf + 1 >= lo) {
          int32_t* fd_row = st.fD + m * F1 - lo;
          for (int k = kf + 1; k <= k_full; ++k) {
            const uint32_t t = rem + R;
            const uint32_t c = t >= dur ? 1u : 0u;
            rem = t - (c ? dur : 0u);
            const uint32_t d = Q + c;
            n += d;
            if (d) atomicAdd(&fd_row[k], (int32_t)d);
          }
          if (be_raw <= K - 1 && (uint32_t)L != n) atomicAdd(&fd_row[be_raw], (int32_t)(L - n));
        } else {
          for (int k = kf + 1; k <= k_full; ++k) {
            const uint32_t t = rem + R;
            const uint32_t c = t >= dur ? 1u : 0u;
            rem = t - (c ? dur : 0u);
            const uint32_t d = Q + c;
            n += d;
            if (d) add_tok(st.fD, D, k, m, lo, (int32_t)d);
          }
          if (be_raw <= K - 1 && (uint32_t)L != n) add_tok(st.fD, D, be_raw, m, lo, (int32_t)(L - n));
        }
      }
    }
    __syncthreads();
    for (int c = threadIdx.x; c < ncell; c += kThreads) {
      const int m = c & (Mp - 1);
      if (m >= M) continue;
      const int k = k_lo + (c >> lgMp);
      const size_t g = (size_t)k * M + m;
      if (SLO && k < K) {
        const uint32_t s = st.aS[c];
        if (s) atomicAdd(&slo[g], (unsigned long long)(s & 0xffffu) + ((unsigned long long)(s >> 16) << 32));
      }
      if (k <= K && st.aW[c]) atomicAdd(&dW[g], st.aW[c]);
    }
    for (int c = threadIdx.x; c < M * F; c += kThreads) {
      const int m = c >> lgF;
      const int lo = st.far_lo[m];
      if (lo == 0x7fffffff) continue;
      const int k = lo + (c & (F - 1));
      const int cell = m * F1 + (c & (F - 1));
      const size_t g = (size_t)k * M + m;
      if (k < K) {
        if (st.fP[cell]) atomicAdd(&P[g], st.fP[cell]);
        if (st.fD[cell]) atomicAdd(&D[g], st.fD[cell]);
      }
      const int32_t aw = st.fAW[cell];
      if (k <= K && aw) {
        const int32_t a = (int32_t)(int16_t)(aw & 0xffff);
        const int32_t w = (aw - a) / 65536;
        if (a) atomicAdd(&dA[g], a);
        if (w) atomicAdd(&dW[g], w);
      }
    }
    __syncthreads();   // the next slice reuses the shared memory
  }
  warp_add_counter(&diag->dropped_range, n_range);
  warp_add_counter(&diag->dropped_model, n_model);
  warp_add_counter(&diag->dropped_order, n_order);
}

// SLO counts alone (for calibration from records whose counts exist already).
// Records sorted by arrival put a CTA's slice into a short run of arrival
// windows: the CTA adds into a shared copy of those rows, two 16-bit counts
// (arrivals, met) per 32-bit word (a slice holds at most kSloPer records), and
// flushes them once; records outside the run (unsorted input) go to global
// atomics.
constexpr int kSloPer = 4096;
__global__ void __launch_bounds__(kThreads)
k_slo_requests(ReqCols r, int M, int win, FastDiv fd, int K, int rows, bool vec,
               unsigned long long* __restrict__ slo, const int32_t* __restrict__ slo_ms) {
  extern __shared__ uint32_t s_slo[];   // [rows][M]
  const int64_t i0 = (int64_t)blockIdx.x * kSloPer;
  const int n_loc = (int)min64(r.n - i0, (int64_t)kSloPer);
  if (n_loc <= 0) return;
  const uint32_t span = (uint32_t)K * (uint32_t)win;
  const int a_first = r.t_arr[i0];
  const int k_lo = (a_first < 0 || (uint32_t)a_first >= span) ? 0 : (int)fd.div((uint32_t)a_first);
  const int used = min(rows, K - k_lo);
  for (int c = threadIdx.x; c < used * M; c += kThreads) s_slo[c] = 0;
  __syncthreads();
  // every column of four consecutive records is loaded before any test, so
  // that the loads are in flight together
  const int32_t* col[7] = {r.model + i0, r.t_arr + i0, r.t_start + i0, r.t_first + i0,
                           r.t_end + i0, r.L_in + i0, r.L_out + i0};
  for (int b = 4 * threadIdx.x; b < n_loc; b += 4 * kThreads) {
    int v[7][4];
    if (vec && b + 4 <= n_loc) {
#pragma unroll
      for (int c = 0; c < 7; ++c) {
        const int4 q = __ldcs(reinterpret_cast<const int4*>(col[c] + b));
        v[c][0] = q.x; v[c][1] = q.y; v[c][2] = q.z; v[c][3] = q.w;
      }
    } else {
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const bool in = b + u < n_loc;
#pragma unroll
        for (int c = 0; c < 7; ++c) v[c][u] = in ? col[c][b + u] : 0;
        if (!in) v[0][u] = -1;
      }
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int m = v[0][u], ta = v[1][u], ts = v[2][u], tf = v[3][u], te = v[4][u];
      const bool ok = m >= 0 && m < M && ta >= 0 && (uint32_t)ta < span && ta <= ts && ts <= tf &&
                      tf <= te && v[5][u] >= 0 && v[6][u] >= 1;
      if (!ok) continue;
      const uint32_t met = (int64_t)tf - ta <= (int64_t)slo_ms[m] ? 1u : 0u;
      const int k = (int)fd.div((uint32_t)ta);
      const uint32_t rel = (uint32_t)(k - k_lo);
      if (rel < (uint32_t)used) atomicAdd(&s_slo[rel * M + m], 1u + (met << 16));
      else atomicAdd(&slo[(size_t)k * M + m], 1ull + ((unsigned long long)met << 32));
    }
  }
  __syncthreads();
  for (int c = threadIdx.x; c < used * M; c += kThreads) {
    const uint32_t v = s_slo[c];
    if (v)
      atomicAdd(&slo[(size_t)k_lo * M + c],
                (unsigned long long)(v & 0xffffu) + ((unsigned long long)(v >> 16) << 32));
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

// First and last valid tick of each request: the events of a CTA's slice (a
// few seconds of a time-ordered stream) come from a few hundred requests,
// each with many events, so the CTA keeps a shared-memory table of them (open
// addressing on the request id, with the request's model cached beside it)
// and flushes one min and one max per request; requests that find no slot
// within kProbe probes go to global atomics directly.
constexpr int kReqSlots = 1024;
constexpr int kProbe = 32;
constexpr int32_t kNoReq = -1;
constexpr int32_t kModelUnread = -2;

__global__ void __launch_bounds__(kThreads)
k_reduce_events(EvCols e, int M, int win, FastDiv fd, int K, int64_t per_cta, int rows,
                bool vec, int32_t* __restrict__ P, int32_t* __restrict__ D,
                int32_t* __restrict__ first, int32_t* __restrict__ last, tre_diag* diag) {
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
  int32_t* s_key = sD + (size_t)rows * M;
  int32_t* s_first = s_key + kReqSlots;
  int32_t* s_last = s_first + kReqSlots;
  int32_t* s_model = s_last + kReqSlots;
  for (int c = threadIdx.x; c < cells; c += kThreads) { sP[c] = 0; sD[c] = 0; }
  for (int c = threadIdx.x; c < kReqSlots; c += kThreads) {
    s_key[c] = kNoReq;
    s_first[c] = 0x7fffffff;
    s_last[c] = -1;
    s_model[c] = kModelUnread;
  }
  __syncthreads();

  unsigned long long n_range = 0, n_model = 0, n_order = 0;
  auto one = [&](int m, int rq, float ts, uint8_t ph) {
    if (m < 0 || m >= M || rq < 0 || rq >= e.n_req) {
      ++n_model;
      return;
    }
    // the request's slot (or -1: none free within kProbe probes)
    int slot = -1;
    {
      uint32_t h = ((uint32_t)rq * 0x9E3779B1u) >> (32 - 10);
      for (int p = 0; p < kProbe; ++p, h = (h + 1) & (kReqSlots - 1)) {
        const int32_t k = s_key[h];
        if (k == rq) { slot = (int)h; break; }
        if (k == kNoReq) {
          const int32_t prev = atomicCAS(&s_key[h], kNoReq, rq);
          if (prev == kNoReq || prev == rq) { slot = (int)h; break; }
        }
      }
    }
    int rm = slot >= 0 ? s_model[slot] : kModelUnread;
    if (rm == kModelUnread) {
      rm = e.req_model[rq];
      if (slot >= 0) s_model[slot] = rm;
    }
    int64_t tick = 0;
    if (rm != m) {
      ++n_model;
    } else if (!ms_tick(ts, span, tick)) {
      ++n_range;
    } else if (ph > 1) {
      ++n_order;
    } else {
      const int64_t k = fd.div((uint32_t)tick);
      stage_add<int32_t>(ph == 0 ? sP : sD, ph == 0 ? P : D, k, k_lo, used, M, m, 1);
      if (slot >= 0) {
        atomicMin(&s_first[slot], (int)tick);
        atomicMax(&s_last[slot], (int)tick);
      } else {
        atomicMin(&first[rq], (int)tick);
        atomicMax(&last[rq], (int)tick);
      }
    }
  };
  // four consecutive events per thread and pass, with 16-byte loads of the
  // columns when they are aligned, so that enough bytes are in flight
  for (int64_t b = i0 + 4 * threadIdx.x; b < i1; b += 4 * kThreads) {
    int mm[4], rr[4];
    float tt[4];
    uint8_t pp[4];
    if (vec && b + 4 <= i1) {
      const int4 a4 = *reinterpret_cast<const int4*>(e.model + b);
      const int4 q4 = *reinterpret_cast<const int4*>(e.req + b);
      const float4 t4 = *reinterpret_cast<const float4*>(e.t_s + b);
      const uchar4 p4 = *reinterpret_cast<const uchar4*>(e.phase + b);
      mm[0] = a4.x; mm[1] = a4.y; mm[2] = a4.z; mm[3] = a4.w;
      rr[0] = q4.x; rr[1] = q4.y; rr[2] = q4.z; rr[3] = q4.w;
      tt[0] = t4.x; tt[1] = t4.y; tt[2] = t4.z; tt[3] = t4.w;
      pp[0] = p4.x; pp[1] = p4.y; pp[2] = p4.z; pp[3] = p4.w;
#pragma unroll
      for (int u = 0; u < 4; ++u) one(mm[u], rr[u], tt[u], pp[u]);
    } else {
      for (int u = 0; u < 4 && b + u < i1; ++u)
        one(e.model[b + u], e.req[b + u], e.t_s[b + u], e.phase[b + u]);
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
  for (int c = threadIdx.x; c < kReqSlots; c += kThreads) {
    const int rq = s_key[c];
    if (rq == kNoReq || s_last[c] < 0) continue;
    atomicMin(&first[rq], s_first[c]);
    atomicMax(&last[rq], s_last[c]);
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
constexpr int kScanBatch = 16;
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
  int64_t k = r0;
  // kScanBatch rows' loads issued together, so that enough bytes are in flight
  for (; k + kScanBatch <= r1; k += kScanBatch) {
    int32_t xa[kScanBatch], xw[kScanBatch];
#pragma unroll
    for (int j = 0; j < kScanBatch; ++j) {
      xa[j] = dA[(k + j) * M + m];
      xw[j] = dW[(k + j) * M + m];
    }
#pragma unroll
    for (int j = 0; j < kScanBatch; ++j) {
      a += xa[j];
      w += xw[j];
    }
  }
  for (; k < r1; ++k) {
    a += dA[k * M + m];
    w += dW[k * M + m];
  }
  pA[t] = a;
  pW[t] = w;
}

// exclusive scan over chunks, one CTA per model, one thread per chunk
// (n_chunks <= 1024)
__global__ void __launch_bounds__(1024)
k_scan_chunks(int M, int n_chunks, int32_t* __restrict__ pA, int32_t* __restrict__ pW) {
  __shared__ int32_t wa[32], ww[32];
  const int m = blockIdx.x;
  pA += (size_t)blockIdx.y * n_chunks * M;
  pW += (size_t)blockIdx.y * n_chunks * M;
  const int c = threadIdx.x, lane = c & 31, wid = c >> 5;
  const int32_t va = c < n_chunks ? pA[(size_t)c * M + m] : 0;
  const int32_t vw = c < n_chunks ? pW[(size_t)c * M + m] : 0;
  int32_t ia = va, iw = vw;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int32_t xa = __shfl_up_sync(0xffffffffu, ia, o);
    const int32_t xw = __shfl_up_sync(0xffffffffu, iw, o);
    if (lane >= o) { ia += xa; iw += xw; }
  }
  if (lane == 31) { wa[wid] = ia; ww[wid] = iw; }
  __syncthreads();
  if (wid == 0) {
    int32_t sa = lane < (int)(blockDim.x >> 5) ? wa[lane] : 0;
    int32_t sw = lane < (int)(blockDim.x >> 5) ? ww[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int32_t xa = __shfl_up_sync(0xffffffffu, sa, o);
      const int32_t xw = __shfl_up_sync(0xffffffffu, sw, o);
      if (lane >= o) { sa += xa; sw += xw; }
    }
    wa[lane] = sa;   // inclusive over warps
    ww[lane] = sw;
  }
  __syncthreads();
  const int32_t base_a = wid ? wa[wid - 1] : 0, base_w = wid ? ww[wid - 1] : 0;
  if (c < n_chunks) {
    pA[(size_t)c * M + m] = base_a + ia - va;
    pW[(size_t)c * M + m] = base_w + iw - vw;
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
  int64_t k = r0;
  for (; k + kScanBatch <= r1; k += kScanBatch) {
    int32_t xa[kScanBatch], xw[kScanBatch];
#pragma unroll
    for (int j = 0; j < kScanBatch; ++j) {
      xa[j] = dA[(k + j) * M + m];
      xw[j] = dW[(k + j) * M + m];
    }
#pragma unroll
    for (int j = 0; j < kScanBatch; ++j) {
      a += xa[j];
      w += xw[j];
      A[(k + j) * M + m] = a;
      W[(k + j) * M + m] = w;
    }
  }
  for (; k < r1; ++k) {
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

// Clears a list of 32-bit word ranges in one launch: every CTA clears one
// chunk of kZeroChunk words of one range (16-byte stores where the range's
// alignment allows them), the chunks of all ranges numbered back to back.
constexpr int kMaxZero = 3 * kMaxTraces + 2;
constexpr int kZeroChunk = kThreads * 16;   // words per CTA
struct ZeroList {
  int n;
  uint32_t* ptr[kMaxZero];
  int64_t words[kMaxZero];
  int32_t cta_base[kMaxZero + 1];
};

__global__ void __launch_bounds__(kThreads) k_zero(const __grid_constant__ ZeroList zl) {
  const int r = prefix_index(zl.cta_base, zl.n, blockIdx.x);
  uint32_t* p = zl.ptr[r];
  const int64_t n = zl.words[r];
  const int64_t w0 = (int64_t)(blockIdx.x - zl.cta_base[r]) * kZeroChunk;
  const int64_t w1 = min64(n, w0 + kZeroChunk);
  // words up to the first 16-byte boundary of the chunk, 16-byte groups, tail
  const int64_t head = min64(w1 - w0, (int64_t)((16 - ((uintptr_t)(p + w0) & 15)) & 15) / 4);
  if (threadIdx.x < head) p[w0 + threadIdx.x] = 0u;
  uint4* q = reinterpret_cast<uint4*>(p + w0 + head);
  const int64_t nq = (w1 - w0 - head) / 4;
  for (int64_t i = threadIdx.x; i < nq; i += kThreads) q[i] = make_uint4(0u, 0u, 0u, 0u);
  const int64_t t0 = w0 + head + nq * 4;
  if (threadIdx.x < w1 - t0) p[t0 + threadIdx.x] = 0u;
}

// ---- gauge scan fused with the exact coarsening (sweeps) --------------------
// Base windows are cut into blocks of `blk` rows (a multiple of every window
// length's ratio q, so no coarse window straddles two blocks). Pass 1 sums the
// gauge diffs of every (trace, block, model); pass 2 turns those sums into
// exclusive prefixes per (trace, model); pass 3 runs each block from its
// prefix, writes the base gauges, and for every coarser window length adds the
// counts over q base windows and reads the gauges at the last of them.
__global__ void __launch_bounds__(kThreads)
k_gauge_blocks(const __grid_constant__ GaugePlan gp, const int32_t* __restrict__ dA,
               const int32_t* __restrict__ dW, int32_t* __restrict__ pA,
               int32_t* __restrict__ pW) {
  const int M = gp.M, Kb = gp.Kb;
  const int64_t t = (int64_t)blockIdx.x * kThreads + threadIdx.x;
  if (t >= (int64_t)gp.n_traces * gp.nblk * M) return;
  const int m = (int)(t % M);
  const int64_t rest = t / M;
  const int b = (int)(rest % gp.nblk), tr = (int)(rest / gp.nblk);
  const int k0 = b * gp.blk, k1 = min(Kb, k0 + gp.blk);
  const size_t base = (size_t)tr * (Kb + 1) * M + m;
  int32_t a = 0, w = 0;
#pragma unroll 4
  for (int k = k0; k < k1; ++k) {
    a += dA[base + (size_t)k * M];
    w += dW[base + (size_t)k * M];
  }
  pA[t] = a;
  pW[t] = w;
}

// exclusive scan of the block sums of one (trace, model) per CTA
__global__ void __launch_bounds__(kThreads)
k_gauge_block_scan(const __grid_constant__ GaugePlan gp, int32_t* __restrict__ pA,
                   int32_t* __restrict__ pW) {
  __shared__ int32_t wa[kThreads / 32], ww[kThreads / 32];
  const int M = gp.M, nb = gp.nblk;
  const int tr = blockIdx.x / M, m = blockIdx.x % M;
  const size_t base = (size_t)tr * nb * M + m;
  const int per = (nb + kThreads - 1) / kThreads;
  const int b0 = threadIdx.x * per, b1 = min(nb, b0 + per);
  int32_t sa = 0, sw = 0;
  for (int b = b0; b < b1; ++b) {
    sa += pA[base + (size_t)b * M];
    sw += pW[base + (size_t)b * M];
  }
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  int32_t ia = sa, iw = sw;
  for (int o = 1; o < 32; o <<= 1) {
    const int32_t xa = __shfl_up_sync(0xffffffffu, ia, o);
    const int32_t xw = __shfl_up_sync(0xffffffffu, iw, o);
    if (lane >= o) { ia += xa; iw += xw; }
  }
  if (lane == 31) { wa[wid] = ia; ww[wid] = iw; }
  __syncthreads();
  int32_t ea = ia - sa, ew = iw - sw;
  for (int q = 0; q < wid; ++q) { ea += wa[q]; ew += ww[q]; }
  for (int b = b0; b < b1; ++b) {
    const size_t x = base + (size_t)b * M;
    const int32_t va = pA[x], vw = pW[x];
    pA[x] = ea;
    pW[x] = ew;
    ea += va;
    ew += vw;
  }
}

// NW: the most window lengths the launch serves (their running sums live in
// registers; four cover the sweep's usual lengths with fewer registers)
template <int NW>
__global__ void __launch_bounds__(kThreads)
k_gauge_apply(const __grid_constant__ GaugePlan gp, const int32_t* __restrict__ dA,
              const int32_t* __restrict__ dW, const int32_t* __restrict__ pA,
              const int32_t* __restrict__ pW, const int32_t* __restrict__ Pin,
              const int32_t* __restrict__ Din, const unsigned long long* __restrict__ sloin,
              int32_t* __restrict__ P, int32_t* __restrict__ D, int32_t* __restrict__ A,
              int32_t* __restrict__ W, unsigned long long* __restrict__ slo) {
  constexpr int RB = 4;   // rows whose loads are issued together
  const int M = gp.M, Kb = gp.Kb;
  const int64_t t = (int64_t)blockIdx.x * kThreads + threadIdx.x;
  if (t >= (int64_t)gp.n_traces * gp.nblk * M) return;
  const int m = (int)(t % M);
  const int64_t rest = t / M;
  const int b = (int)(rest % gp.nblk), tr = (int)(rest / gp.nblk);
  const int k0 = b * gp.blk, k1 = min(Kb, k0 + gp.blk);
  const size_t dbase = (size_t)tr * (Kb + 1) * M + m;
  const size_t ibase = (size_t)gp.in_off[tr] + m;
  int32_t a = pA[t], w = pW[t];
  int32_t ap[NW], ad[NW], cnt[NW], kq[NW];
  unsigned long long as[NW];
#pragma unroll
  for (int j = 0; j < NW; ++j) {
    ap[j] = 0; ad[j] = 0; as[j] = 0;
    cnt[j] = j < gp.n_win ? gp.q[j] : 0;
    kq[j] = j < gp.n_win ? k0 / gp.q[j] : 0;
  }
  for (int kb = k0; kb < k1; kb += RB) {
    int32_t va[RB], vw[RB], vp[RB], vd[RB];
    unsigned long long vs[RB];
#pragma unroll
    for (int r = 0; r < RB; ++r) {
      const int k = kb + r;
      const bool in = k < k1;
      const size_t xd = dbase + (size_t)k * M, xi = ibase + (size_t)k * M;
      va[r] = in ? dA[xd] : 0;
      vw[r] = in ? dW[xd] : 0;
      vp[r] = in ? Pin[xi] : 0;
      vd[r] = in ? Din[xi] : 0;
      vs[r] = in && sloin ? sloin[xi] : 0ull;
    }
#pragma unroll
    for (int r = 0; r < RB; ++r) {
      const int k = kb + r;
      if (k >= k1) break;
      a += va[r];
      w += vw[r];
#pragma unroll
      for (int j = 0; j < NW; ++j) {
        if (j >= gp.n_win) break;
        if (j == gp.base_w) {
          const size_t o = (size_t)gp.out_off[tr][j] + (size_t)k * M + m;
          A[o] = a;
          W[o] = w;
          continue;
        }
        ap[j] += vp[r];
        ad[j] += vd[r];
        as[j] += vs[r];
        if (--cnt[j] == 0) {
          const size_t o = (size_t)gp.out_off[tr][j] + (size_t)kq[j] * M + m;
          P[o] = ap[j];
          D[o] = ad[j];
          A[o] = a;
          W[o] = w;
          if (slo) slo[o] = as[j];
          ap[j] = 0; ad[j] = 0; as[j] = 0;
          cnt[j] = gp.q[j];
          ++kq[j];
        }
      }
    }
  }
}

int num_sms() { return device_sm_count(); }

int64_t per_cta_records(int64_t n, int lo, int hi, int quantum = kThreads) {
  int64_t per = (n + (int64_t)num_sms() * 4 - 1) / ((int64_t)num_sms() * 4);
  per = std::max<int64_t>(lo, std::min<int64_t>(hi, per));
  return (per + quantum - 1) / quantum * quantum;
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
  const int n_chunks = std::max((K + L - 1) / L, (K + kGaugeMinBlk - 1) / kGaugeMinBlk);
  w.part_cap = (int64_t)std::max(n_chunks, 1) * M;
  w.partA = a.take<int32_t>((size_t)w.part_cap * n_traces);
  w.partW = a.take<int32_t>((size_t)w.part_cap * n_traces);
}

cudaError_t launch_reduce_requests(const ReqCols* traces, int n_traces, int M, int win, int K,
                                   int32_t* P, int32_t* D, ReduceWs& w, unsigned long long* slo,
                                   const int32_t* slo_ms, tre_diag* diag, cudaStream_t s,
                                   const int64_t* out_off) {
  if (n_traces < 1 || n_traces > kMaxTraces || n_traces > w.n_traces)
    return cudaErrorInvalidValue;
  const size_t cells = (size_t)K * M * n_traces;
  ReqBatch bt;
  bt.n = n_traces;
  bt.vec_ok = 0;
  // every output the kernel adds into starts at zero: one clearing launch
  ZeroList zl;
  zl.n = 0;
  for (int t = 0; t < n_traces; ++t) {
    bt.out_off[t] = out_off ? out_off[t] : (int64_t)t * K * M;
    zl.ptr[zl.n] = reinterpret_cast<uint32_t*>(P + bt.out_off[t]);
    zl.words[zl.n++] = (int64_t)K * M;
    zl.ptr[zl.n] = reinterpret_cast<uint32_t*>(D + bt.out_off[t]);
    zl.words[zl.n++] = (int64_t)K * M;
    if (slo) {
      zl.ptr[zl.n] = reinterpret_cast<uint32_t*>(slo + bt.out_off[t]);
      zl.words[zl.n++] = (int64_t)K * M * 2;
    }
  }
  zl.ptr[zl.n] = reinterpret_cast<uint32_t*>(w.dA);
  zl.words[zl.n++] = (int64_t)(cells + (size_t)M * n_traces);
  zl.ptr[zl.n] = reinterpret_cast<uint32_t*>(w.dW);
  zl.words[zl.n++] = (int64_t)(cells + (size_t)M * n_traces);
  int zctas = 0;
  for (int r = 0; r < zl.n; ++r) {
    zl.cta_base[r] = zctas;
    zctas += (int)((zl.words[r] + kZeroChunk - 1) / kZeroChunk);
  }
  zl.cta_base[zl.n] = zctas;
  if (zctas > 0) k_zero<<<zctas, kThreads, 0, s>>>(zl);
  int64_t total_n = 0;
  for (int t = 0; t < n_traces; ++t) total_n += traces[t].n;
  // records that live in host memory (pinned, mapped) are copied into shared
  // memory once per CTA rather than read twice over the host link; any column
  // in host memory selects the copying variant (it reads device columns too)
  bool copy_records = false;
  for (int t = 0; t < n_traces; ++t) {
    const ReqCols& c = traces[t];
    if (c.n == 0) continue;
    const void* cols[7] = {c.model, c.t_arr, c.t_start, c.t_first, c.t_end, c.L_in, c.L_out};
    for (const void* p : cols) {
      cudaPointerAttributes pa;
      if (cudaPointerGetAttributes(&pa, p) != cudaSuccess) {
        cudaGetLastError();
        continue;
      }
      if (pa.type == cudaMemoryTypeHost) copy_records = true;
    }
  }
  const int64_t mean_n = std::max<int64_t>(total_n / n_traces, 1);
  // model rows padded to a power of two on the arrival side; start side runs
  // of F (power of two) windows per model
  int lgMp = 0;
  while ((1 << lgMp) < M) ++lgMp;
  const int Mp = 1 << lgMp;
  const int64_t near_cap = 32 * 1024 / ((4 + (slo ? 4 : 0)) * Mp);   // arrival-stage budget
  int lgF = 3;
  while (lgF < 8 && (size_t)12 * M * ((2 << lgF) + 1) <= 16 * 1024) ++lgF;
  const int F = 1 << lgF;
  // arrival-side rows (3x the mean arrival span of a CTA's records) and the
  // shared memory a CTA of `p` records needs
  auto rows_for = [&](int64_t p) {
    return (int)std::max<int64_t>(
        1, std::min<int64_t>(near_cap, (int64_t)(3.0 * p / mean_n * K) + 34));
  };
  auto smem_for = [&](int64_t p) {
    const size_t stage = (size_t)rows_for(p) * Mp * (4 + (slo ? 4 : 0)) +
                         (size_t)12 * M * (F + 1) + (size_t)M * 8 + 16 +
                         (size_t)p * sizeof(uint16_t);
    return stage + (copy_records ? (size_t)p * 7 * 4 : 0);
  };
  constexpr size_t kSmemMax = 200 * 1024;
  // records per CTA sized on the whole batch so the grid fills the GPU, in
  // whole passes of every warp; with copied records, fewer per CTA when many
  // models leave less room beside the staging
  int64_t per = per_cta_records(mean_n, 1024, copy_records ? 2048 : 8192, kThreads * kVec);
  while (per > kThreads * kVec && smem_for(per) > kSmemMax) per -= kThreads * kVec;
  static_assert(8192 <= kMaxPerCta, "packed shared counters need <= kMaxPerCta records per CTA");
  const int near_rows = rows_for(per);
  const size_t smem = smem_for(per);
  if (smem > kSmemMax) return cudaErrorInvalidValue;
  int ctas = 0;
  for (int t = 0; t < n_traces; ++t) {
    const ReqCols& c = traces[t];
    bt.cols[t] = c;
    bt.per_cta[t] = per;
    bt.cta_base[t] = ctas;
    ctas += (int)((c.n + per - 1) / per);
    const uintptr_t ptr_or = (uintptr_t)c.model | (uintptr_t)c.t_arr | (uintptr_t)c.t_start |
                             (uintptr_t)c.t_first | (uintptr_t)c.t_end | (uintptr_t)c.L_in |
                             (uintptr_t)c.L_out;
    if ((ptr_or & 15u) == 0) bt.vec_ok |= 1ull << t;
  }
  bt.cta_base[n_traces] = ctas;
  if (ctas == 0) return cudaSuccess;
  // the largest shared-memory carveout, so that four CTAs with their staging
  // and queues share an SM
  const void* fns[4] = {(const void*)k_reduce_requests<true, false>,
                        (const void*)k_reduce_requests<false, false>,
                        (const void*)k_reduce_requests<true, true>,
                        (const void*)k_reduce_requests<false, true>};
  for (const void* f : fns) {
    cudaError_t e = func_smem_once(f, 200 * 1024, true);
    if (e) return e;
  }
  const FastDiv fd(win);
  // Records read over the host link: one CTA per slice would hold every SM for
  // the length of the transfer. CTAs on two thirds of the SMs (two each) still
  // keep the link busy -- a CTA spends most of a slice copying it in -- and
  // leave the other SMs to work on other streams, such as the later phases of
  // the step before.
  const unsigned grid = copy_records
                            ? (unsigned)std::min(ctas, 2 * std::max(1, device_sm_count() * 2 / 3))
                            : (unsigned)ctas;
  if (slo && copy_records)
    k_reduce_requests<true, true><<<grid, kThreads, smem, s>>>(bt, M, lgMp, win, fd, K,
                                                               near_rows, lgF, P, D, w.dA, w.dW,
                                                               slo, slo_ms, diag);
  else if (slo)
    k_reduce_requests<true, false><<<grid, kThreads, smem, s>>>(bt, M, lgMp, win, fd, K,
                                                                near_rows, lgF, P, D, w.dA, w.dW,
                                                                slo, slo_ms, diag);
  else if (copy_records)
    k_reduce_requests<false, true><<<grid, kThreads, smem, s>>>(bt, M, lgMp, win, fd, K,
                                                                near_rows, lgF, P, D, w.dA, w.dW,
                                                                nullptr, nullptr, diag);
  else
    k_reduce_requests<false, false><<<grid, kThreads, smem, s>>>(bt, M, lgMp, win, fd, K,
                                                                 near_rows, lgF, P, D, w.dA, w.dW,
                                                                 nullptr, nullptr, diag);
  return cudaGetLastError();
}

cudaError_t launch_slo_requests(const ReqCols& r, int M, int win, int K,
                                unsigned long long* slo, const int32_t* slo_ms, cudaStream_t s) {
  cudaError_t e = cudaMemsetAsync(slo, 0, (size_t)K * M * sizeof(unsigned long long), s);
  if (e || r.n == 0) return e;
  // arrival rows staged per CTA: the mean arrival span of a slice, three times
  // over, plus a margin, within 32 KB
  const int64_t mean_rows = (int64_t)kSloPer * K / std::max<int64_t>(r.n, 1);
  const int rows = (int)std::max<int64_t>(1, std::min<int64_t>(3 * mean_rows + 34,
                                                               32 * 1024 / (4 * M)));
  const unsigned grid = (unsigned)((r.n + kSloPer - 1) / kSloPer);
  const bool vec = (((uintptr_t)r.model | (uintptr_t)r.t_arr | (uintptr_t)r.t_start |
                     (uintptr_t)r.t_first | (uintptr_t)r.t_end | (uintptr_t)r.L_in |
                     (uintptr_t)r.L_out) & 15) == 0;
  k_slo_requests<<<grid, kThreads, (size_t)rows * M * 4, s>>>(r, M, win, FastDiv(win), K, rows,
                                                              vec, slo, slo_ms);
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
    // per is a multiple of four, so every CTA's first event keeps the alignment
    const bool vec = ((((uintptr_t)ev.model | (uintptr_t)ev.req | (uintptr_t)ev.t_s) & 15) |
                      ((uintptr_t)ev.phase & 3)) == 0;
    k_reduce_events<<<grid, kThreads, (size_t)rows * M * 8 + (size_t)kReqSlots * 16, s>>>(
        ev, M, win, FastDiv(win), K, per, rows, vec, P, D, w.first, w.last, diag);
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
  k_scan_chunks<<<dim3(M, w.n_traces), 1024, 0, s>>>(M, n_chunks, w.partA, w.partW);
  k_scan_apply<<<g, kThreads, 0, s>>>(M, K, L, n_chunks, w.dA, w.dW, w.partA, w.partW, A, W);
  return cudaGetLastError();
}

// Time-averaged occupancy (the window-mean reading of Eq. 1's running and
// waiting counts, Sec. III-A): the request-milliseconds that running
// ([t_start, t_end)) and waiting ([t_arr, t_start)) requests spend inside each
// window. A span adds its partial first and last windows directly (64-bit
// sums) and marks the windows it covers completely in a +1/-1 difference
// array; the prefix of that array times the window length is added
// afterwards. Records are taken or skipped by the reduction's rules.
// One CTA per chunk of consecutive records, staged in shared memory like the
// token reduction: the waiting span's first window sits on the arrival side
// (rows from the chunk's first arrival window), every other target near the
// record's start (per model, a run of F windows from the earliest start among
// the chunk's records). Targets outside both go to global atomics. Staged
// partial sums are 32-bit (a chunk adds at most kOccPerCta * win to a cell,
// staged only for win <= 2^20); the covered-window difference counts of
// running and waiting share one word per start-side cell (each bounded by the
// chunk's record count). Each thread reads four consecutive records per pass
// with 16-byte loads when the columns allow it.
constexpr int kOccPerCta = 2048;
__global__ void __launch_bounds__(kThreads)
k_occ_staged(ReqCols r, bool vec, bool stage, int M, int lgMp, int win, FastDiv fd, int K,
             int near_rows, int lgF, unsigned long long* __restrict__ pA,
             unsigned long long* __restrict__ pW, int32_t* __restrict__ fA,
             int32_t* __restrict__ fW) {
  extern __shared__ uint32_t osm32[];
  const int64_t i0 = (int64_t)blockIdx.x * kOccPerCta;
  const int n_loc = (int)min64(r.n - i0, kOccPerCta);
  if (n_loc <= 0) return;
  const int Mp = 1 << lgMp, F = 1 << lgF;
  const uint32_t span = (uint32_t)K * (uint32_t)win;
  const uint32_t uw = (uint32_t)win;
  uint32_t* sWp = osm32;                                             // [near_rows][Mp]
  int32_t* sWf = reinterpret_cast<int32_t*>(sWp + (size_t)near_rows * Mp);
  uint32_t* sAp = reinterpret_cast<uint32_t*>(sWf + (size_t)near_rows * Mp);  // [M][F]
  uint32_t* sWq = sAp + (size_t)M * F;                               // [M][F]
  int32_t* sAWf = reinterpret_cast<int32_t*>(sWq + (size_t)M * F);   // [M][F]
  int32_t* slo = sAWf + (size_t)M * F;                               // [M]
  const int32_t* col[7] = {r.model + i0, r.t_arr + i0, r.t_start + i0, r.t_first + i0,
                           r.t_end + i0, r.L_in + i0, r.L_out + i0};
  const int a_first = col[1][0], a_last = col[1][n_loc - 1];
  const int k_lo = a_first < 0 ? 0 : (int)min(fd.div((uint32_t)a_first), (uint32_t)K);
  const int k_hi = a_last < 0 ? 0 : (int)min(fd.div((uint32_t)a_last), (uint32_t)K);
  const int used = stage ? min(near_rows, (k_hi >= k_lo ? k_hi - k_lo + 1 : 1) + 1) : 0;
  const int Fs = stage ? F : 0;
  for (int c = threadIdx.x; c < used * Mp; c += kThreads) { sWp[c] = 0; sWf[c] = 0; }
  for (int c = threadIdx.x; c < M * Fs; c += kThreads) { sAp[c] = 0; sWq[c] = 0; sAWf[c] = 0; }
  for (int m = threadIdx.x; m < M; m += kThreads) slo[m] = 0x7fffffff;
  __syncthreads();
  // each model's earliest start-side window: the window before its first start
  for (int b = threadIdx.x * kVec; b < n_loc; b += kThreads * kVec) {
    int mm[kVec], ss[kVec];
    if (vec && b + kVec <= n_loc) {
      const int4 a = *reinterpret_cast<const int4*>(col[0] + b);
      const int4 q = *reinterpret_cast<const int4*>(col[2] + b);
      mm[0] = a.x; mm[1] = a.y; mm[2] = a.z; mm[3] = a.w;
      ss[0] = q.x; ss[1] = q.y; ss[2] = q.z; ss[3] = q.w;
    } else {
#pragma unroll
      for (int u = 0; u < kVec; ++u) {
        const bool in = b + u < n_loc;
        mm[u] = in ? col[0][b + u] : -1;
        ss[u] = in ? col[2][b + u] : -1;
      }
    }
#pragma unroll
    for (int u = 0; u < kVec; ++u) {
      if (mm[u] < 0 || mm[u] >= M || ss[u] < 0) continue;
      const uint32_t s1 = min((uint32_t)ss[u], span);
      atomicMin(&slo[mm[u]], s1 > 0 ? (int)fd.div(s1 - 1) : 0);
    }
  }
  __syncthreads();
  for (int b = threadIdx.x * kVec; b < n_loc; b += kThreads * kVec) {
    int v[7][kVec];
    if (vec && b + kVec <= n_loc) {
#pragma unroll
      for (int c = 0; c < 7; ++c) {
        const int4 q = *reinterpret_cast<const int4*>(col[c] + b);
        v[c][0] = q.x; v[c][1] = q.y; v[c][2] = q.z; v[c][3] = q.w;
      }
    } else {
#pragma unroll
      for (int u = 0; u < kVec; ++u) {
        const bool in = b + u < n_loc;
#pragma unroll
        for (int c = 0; c < 7; ++c) v[c][u] = in ? col[c][b + u] : 0;
        if (!in) v[0][u] = -1;
      }
    }
#pragma unroll
    for (int u = 0; u < kVec; ++u) {
      const int m = v[0][u], ta = v[1][u], ts = v[2][u], tf = v[3][u], te = v[4][u];
      if (m < 0 || m >= M) continue;
      if (ta < 0 || (uint32_t)ta >= span) continue;
      if (!(ta <= ts && ts <= tf && tf <= te) || v[5][u] < 0 || v[6][u] < 1) continue;
      const int lo = slo[m];
      auto near_part = [&](uint32_t k, uint32_t val) {
        const uint32_t rel = k - (uint32_t)k_lo;
        if (rel < (uint32_t)used) atomicAdd(&sWp[(rel << lgMp) + m], val);
        else atomicAdd(&pW[(size_t)k * M + m], (unsigned long long)val);
      };
      auto near_full = [&](uint32_t k) {
        const uint32_t rel = k - (uint32_t)k_lo;
        if (rel < (uint32_t)used) atomicAdd(&sWf[(rel << lgMp) + m], 1);
        else atomicAdd(&fW[(size_t)k * M + m], 1);
      };
      auto far_part = [&](uint32_t* st, unsigned long long* g, uint32_t k, uint32_t val) {
        const uint32_t rel = k - (uint32_t)lo;
        if (rel < (uint32_t)Fs) atomicAdd(&st[(m << lgF) + rel], val);
        else atomicAdd(&g[(size_t)k * M + m], (unsigned long long)val);
      };
      auto far_full = [&](uint32_t k, int32_t a, int32_t w) {
        const uint32_t rel = k - (uint32_t)lo;
        if (rel < (uint32_t)Fs) {
          atomicAdd(&sAWf[(m << lgF) + rel], a + w * 65536);
        } else {
          if (a) atomicAdd(&fA[(size_t)k * M + m], a);
          if (w) atomicAdd(&fW[(size_t)k * M + m], w);
        }
      };
      // waiting on [ta, ts)
      const uint32_t ew = min((uint32_t)ts, span);
      if ((uint32_t)ta < ew) {
        const uint32_t ka = fd.div((uint32_t)ta), kw = fd.div(ew - 1);
        if (ka == kw) {
          near_part(ka, ew - (uint32_t)ta);
        } else {
          near_part(ka, (ka + 1) * uw - (uint32_t)ta);
          far_part(sWq, pW, kw, ew - kw * uw);
          if (kw > ka + 1) {
            near_full(ka + 1);
            far_full(kw, 0, -1);
          }
        }
      }
      // running on [ts, te)
      const uint32_t er = min((uint32_t)te, span);
      if ((uint32_t)ts < er) {
        const uint32_t ks = fd.div((uint32_t)ts), ke = fd.div(er - 1);
        if (ks == ke) {
          far_part(sAp, pA, ks, er - (uint32_t)ts);
        } else {
          far_part(sAp, pA, ks, (ks + 1) * uw - (uint32_t)ts);
          far_part(sAp, pA, ke, er - ke * uw);
          if (ke > ks + 1) {
            far_full(ks + 1, 1, 0);
            far_full(ke, -1, 0);
          }
        }
      }
    }
  }
  __syncthreads();
  for (int c = threadIdx.x; c < used * Mp; c += kThreads) {
    const int m = c & (Mp - 1);
    const int k = k_lo + (c >> lgMp);
    if (m >= M || k >= K) continue;
    if (sWp[c]) atomicAdd(&pW[(size_t)k * M + m], (unsigned long long)sWp[c]);
    if (sWf[c]) atomicAdd(&fW[(size_t)k * M + m], sWf[c]);
  }
  for (int c = threadIdx.x; c < M * Fs; c += kThreads) {
    const int m = c >> lgF;
    const int lo = slo[m];
    if (lo == 0x7fffffff) continue;
    const int k = lo + (c & (F - 1));
    if (k >= K) continue;
    const size_t g = (size_t)k * M + m;
    if (sAp[c]) atomicAdd(&pA[g], (unsigned long long)sAp[c]);
    if (sWq[c]) atomicAdd(&pW[g], (unsigned long long)sWq[c]);
    const int32_t aw = sAWf[c];
    if (aw) {
      const int32_t a = (int32_t)(int16_t)(aw & 0xffff);
      const int32_t w = (aw - a) / 65536;
      if (a) atomicAdd(&fA[g], a);
      if (w) atomicAdd(&fW[g], w);
    }
  }
}

// adds the full-window counts (chunk prefixes from the gauge scan's first
// two passes) times the window length to the partial sums
__global__ void __launch_bounds__(kThreads)
k_occ_apply(int M, int K, int L, int n_chunks, int win, const int32_t* __restrict__ fA,
            const int32_t* __restrict__ fW, const int32_t* __restrict__ pA,
            const int32_t* __restrict__ pW, long long* __restrict__ A_ms,
            long long* __restrict__ W_ms) {
  const int64_t t = (int64_t)blockIdx.x * kThreads + threadIdx.x;
  if (t >= (int64_t)n_chunks * M) return;
  const int m = (int)(t % M);
  const int c = (int)(t / M);
  const int64_t r0 = (int64_t)c * L, r1 = min64(r0 + L, K);
  int32_t a = pA[t], w = pW[t];
  constexpr int B = 8;
  for (int64_t k0 = r0; k0 < r1; k0 += B) {
    int32_t da[B], dw[B];
    long long am[B], wm[B];
#pragma unroll
    for (int j = 0; j < B; ++j) {
      const bool in = k0 + j < r1;
      const int64_t x = (k0 + j) * M + m;
      da[j] = in ? fA[x] : 0;
      dw[j] = in ? fW[x] : 0;
      am[j] = in ? A_ms[x] : 0;
      wm[j] = in ? W_ms[x] : 0;
    }
#pragma unroll
    for (int j = 0; j < B; ++j) {
      a += da[j];
      w += dw[j];
      if (k0 + j < r1) {
        const int64_t x = (k0 + j) * M + m;
        A_ms[x] = am[j] + (long long)a * win;
        W_ms[x] = wm[j] + (long long)w * win;
      }
    }
  }
}

// Time-averaged occupancy of token events: per request with at least one
// valid event (first/last tick from the event pass) and 0 <= t_arr <= first,
// waiting on [t_arr, first) and running on [first, last), cut at the end of the
// grid. One thread per request (the request table is small beside the event
// stream): partial first and last windows are added to the 64-bit sums, the
// windows a span covers completely are marked +1/-1 in the difference arrays.
__global__ void __launch_bounds__(kThreads)
k_occ_events(EvCols ev, int M, int win, FastDiv fd, int K, const int32_t* __restrict__ first,
             const int32_t* __restrict__ last, unsigned long long* __restrict__ pA,
             unsigned long long* __restrict__ pW, int32_t* __restrict__ fA,
             int32_t* __restrict__ fW) {
  const uint32_t span = (uint32_t)K * (uint32_t)win, uw = (uint32_t)win;
  for (int64_t r = (int64_t)blockIdx.x * kThreads + threadIdx.x; r < ev.n_req;
       r += (int64_t)gridDim.x * kThreads) {
    const int32_t lt = last[r];
    if (lt < 0) continue;
    const int m = ev.req_model[r];
    const int32_t ta = ev.req_t_arr[r], f = first[r];
    if (m < 0 || m >= M || ta < 0 || ta > f) continue;
    auto add_span = [&](uint32_t a, uint32_t e, unsigned long long* part, int32_t* full) {
      e = min(e, span);
      if (a >= e) return;
      const uint32_t k0 = fd.div(a), k1 = fd.div(e - 1);
      if (k0 == k1) {
        atomicAdd(&part[(size_t)k0 * M + m], (unsigned long long)(e - a));
        return;
      }
      atomicAdd(&part[(size_t)k0 * M + m], (unsigned long long)((k0 + 1) * uw - a));
      atomicAdd(&part[(size_t)k1 * M + m], (unsigned long long)(e - k1 * uw));
      if (k1 > k0 + 1) {
        atomicAdd(&full[(size_t)(k0 + 1) * M + m], 1);
        atomicAdd(&full[(size_t)k1 * M + m], -1);
      }
    };
    add_span((uint32_t)ta, (uint32_t)f, pW, fW);
    add_span((uint32_t)f, (uint32_t)lt, pA, fA);
  }
}

// last step of both occupancy passes: the covered-window counts (inclusive
// prefix of the difference arrays) times the window length added to the
// partial sums
cudaError_t occ_finish(int M, int win, int K, ReduceWs& w, int64_t* A_ms, int64_t* W_ms,
                       cudaStream_t s) {
  const int L = scan_chunk_rows(K);
  const int n_chunks = (K + L - 1) / L;
  const int64_t segs = (int64_t)n_chunks * M;
  const unsigned g = (unsigned)((segs + kThreads - 1) / kThreads);
  k_scan_partials<<<dim3(g, 1), kThreads, 0, s>>>(M, K, L, n_chunks, w.dA, w.dW, w.partA,
                                                  w.partW);
  k_scan_chunks<<<dim3(M, 1), 1024, 0, s>>>(M, n_chunks, w.partA, w.partW);
  k_occ_apply<<<g, kThreads, 0, s>>>(M, K, L, n_chunks, win, w.dA, w.dW, w.partA, w.partW,
                                     reinterpret_cast<long long*>(A_ms),
                                     reinterpret_cast<long long*>(W_ms));
  return cudaGetLastError();
}

cudaError_t launch_occupancy_mean(const ReqCols& r, int M, int win, int K, ReduceWs& w,
                                  int64_t* A_ms, int64_t* W_ms, cudaStream_t s) {
  if (K == 0) return cudaSuccess;
  const size_t cells = (size_t)K * M, cells1 = (size_t)(K + 1) * M;
  cudaError_t e = cudaMemsetAsync(A_ms, 0, cells * sizeof(int64_t), s);
  if (!e) e = cudaMemsetAsync(W_ms, 0, cells * sizeof(int64_t), s);
  if (!e) e = cudaMemsetAsync(w.dA, 0, cells1 * sizeof(int32_t), s);
  if (!e) e = cudaMemsetAsync(w.dW, 0, cells1 * sizeof(int32_t), s);
  if (e) return e;
  if (r.n > 0) {
    int lgMp = 0;
    while ((1 << lgMp) < M) ++lgMp;
    const int Mp = 1 << lgMp;
    // arrival-side rows: 3x the mean arrival span of a chunk, within 16 KB
    const int64_t near_cap = std::max<int64_t>(1, 16 * 1024 / (8 * Mp));
    const int near_rows = (int)std::max<int64_t>(
        1, std::min<int64_t>(near_cap, (int64_t)(3.0 * kOccPerCta / r.n * K) + 34));
    // start-side run per model: the longest power of two within 24 KB
    int lgF = 0;
    while (lgF < 8 && (size_t)12 * M * (2u << lgF) <= 24 * 1024) ++lgF;
    const size_t smem = (size_t)near_rows * Mp * 8 + (size_t)12 * M * (1u << lgF) +
                        (size_t)4 * M;
    const bool vec = ((uintptr_t)r.model | (uintptr_t)r.t_arr | (uintptr_t)r.t_start |
                      (uintptr_t)r.t_first | (uintptr_t)r.t_end | (uintptr_t)r.L_in |
                      (uintptr_t)r.L_out) % 16 == 0;
    const bool stage = win <= (1 << 20);   // 32-bit staged sums cannot overflow
    e = func_smem_once((const void*)k_occ_staged, 96 * 1024, false);
    if (e) return e;
    if (smem > 96 * 1024) return cudaErrorInvalidValue;
    const unsigned ctas = (unsigned)((r.n + kOccPerCta - 1) / kOccPerCta);
    k_occ_staged<<<ctas, kThreads, smem, s>>>(r, vec, stage, M, lgMp, win, FastDiv(win), K,
                                              near_rows, lgF,
                                              reinterpret_cast<unsigned long long*>(A_ms),
                                              reinterpret_cast<unsigned long long*>(W_ms), w.dA,
                                              w.dW);
  }
  return occ_finish(M, win, K, w, A_ms, W_ms, s);
}

cudaError_t launch_occupancy_mean_events(const EvCols& ev, int M, int win, int K, ReduceWs& w,
                                         int64_t* A_ms, int64_t* W_ms, cudaStream_t s) {
  if (K == 0) return cudaSuccess;
  const size_t cells = (size_t)K * M, cells1 = (size_t)(K + 1) * M;
  cudaError_t e = cudaMemsetAsync(A_ms, 0, cells * sizeof(int64_t), s);
  if (!e) e = cudaMemsetAsync(W_ms, 0, cells * sizeof(int64_t), s);
  if (!e) e = cudaMemsetAsync(w.dA, 0, cells1 * sizeof(int32_t), s);
  if (!e) e = cudaMemsetAsync(w.dW, 0, cells1 * sizeof(int32_t), s);
  if (e) return e;
  if (ev.n_req > 0) {
    k_occ_events<<<grid_for(ev.n_req, 4), kThreads, 0, s>>>(
        ev, M, win, FastDiv(win), K, w.first, w.last,
        reinterpret_cast<unsigned long long*>(A_ms), reinterpret_cast<unsigned long long*>(W_ms),
        w.dA, w.dW);
    if ((e = cudaGetLastError())) return e;
  }
  return occ_finish(M, win, K, w, A_ms, W_ms, s);
}

cudaError_t launch_gauge_prefix(const GaugePlan& gp, ReduceWs& w, cudaStream_t s) {
  if (gp.n_traces > w.n_traces || (int64_t)gp.nblk * gp.M > w.part_cap) return cudaErrorInvalidValue;
  const int64_t n = (int64_t)gp.n_traces * gp.nblk * gp.M;
  if (n == 0) return cudaSuccess;
  k_gauge_blocks<<<(unsigned)((n + kThreads - 1) / kThreads), kThreads, 0, s>>>(gp, w.dA, w.dW,
                                                                                w.partA, w.partW);
  k_gauge_block_scan<<<gp.n_traces * gp.M, kThreads, 0, s>>>(gp, w.partA, w.partW);
  return cudaGetLastError();
}

cudaError_t launch_gauge_apply(const GaugePlan& gp, ReduceWs& w, const int32_t* Pin,
                               const int32_t* Din, const unsigned long long* sloin, int32_t* P,
                               int32_t* D, int32_t* A, int32_t* W, unsigned long long* slo,
                               cudaStream_t s) {
  const int64_t n = (int64_t)gp.n_traces * gp.nblk * gp.M;
  if (n == 0) return cudaSuccess;
  const unsigned g = (unsigned)((n + kThreads - 1) / kThreads);
  if (gp.n_win <= 4)
    k_gauge_apply<4><<<g, kThreads, 0, s>>>(gp, w.dA, w.dW, w.partA, w.partW, Pin, Din, sloin,
                                            P, D, A, W, slo);
  else
    k_gauge_apply<kGaugeMaxWin><<<g, kThreads, 0, s>>>(gp, w.dA, w.dW, w.partA, w.partW, Pin, Din,
                                                       sloin, P, D, A, W, slo);
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
