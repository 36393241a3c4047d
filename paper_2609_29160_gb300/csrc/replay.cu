// Closed-loop replay (Sec. IV-B rescue and rebalance acting on live capacity,
// Sec. IV-C bounded transfer, Sec. VI-D actuation delays): the controller's
// moves change the servers that serve the requests, and the telemetry it
// scores comes from the requests as they are served.
//
// Readings (shared with the oracle's replay):
//  * each routable replica of a model is one server; a model's requests are
//    served in input order by whichever of its servers frees first; a request
//    needs d_first ms to its first token and d_total ms to its last once
//    started;
//  * window k is processed at T = (k+1)*win: every request that can start
//    before T starts first, then window k's telemetry (the window reduction's
//    token attribution and gauges) is scored with the smoothing carried over
//    windows, and on a control tick the controller acts on the replica counts
//    as they are;
//  * a transition commits at its tick; each donor replica it releases is the
//    donor's server that frees first: it takes no request from T on, finishes
//    the one it serves and returns its GPU sleep_ms after that; the receiver's
//    new server starts waking when its GPU is free (at T when the idle pool
//    paid, else when the transition's last released donor replica has
//    returned its GPU) and serves wake_ms later;
//  * a request not started by the end of the grid reports K*win for its
//    times; an invalid latent record reports -1 and is not served.
//
// GPU layout: one warp per controller instance (a rescue threshold and a
// pacing cap), one lane per model (two for more than 32 models). A lane keeps
// its model's request cursor, gauge counters and smoothing state in
// registers and its servers as a binary min-heap of free times (shared memory
// when the instance's heaps fit, else the workspace). Tokens are attributed to
// future windows in per-instance accumulators; lane 0 runs the controller on
// control ticks from the window's Z and regions staged in shared memory.
#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace tre {
namespace {

constexpr int kFillThreads = 1024;

// ---- latent records grouped by model, input order kept ----------------------
// valid model id per record (-1 when the record is not served) and arrivals
// per (window, model)
__global__ void k_rp_valid(ReplayLatent lat, int M, int win, int K, int8_t* __restrict__ vm,
                           int32_t* __restrict__ arr_cnt, int32_t* __restrict__ n_valid) {
  const int64_t span = (int64_t)K * win;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < lat.n;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int m = lat.model[i];
    const int64_t ta = lat.t_arr[i];
    bool ok = m >= 0 && m < M && ta >= 0 && ta < span;
    ok = ok && lat.d_first[i] >= 0 && lat.d_total[i] >= lat.d_first[i] && lat.L_in[i] >= 0 &&
         lat.L_out[i] >= 1;
    vm[i] = ok ? (int8_t)m : (int8_t)-1;
    if (ok) {
      atomicAdd(&arr_cnt[(ta / win) * M + m], 1);
      atomicAdd(&n_valid[m], 1);
    }
  }
}

// one CTA per model: the model's record indices in input order
__global__ void __launch_bounds__(kFillThreads)
k_rp_fill(int64_t n, int M, const int8_t* __restrict__ vm, const int32_t* __restrict__ n_valid,
          int32_t* __restrict__ list, int32_t* __restrict__ base_out) {
  __shared__ int32_t wcnt[kFillThreads / 32];
  __shared__ int32_t s_base;
  const int m = blockIdx.x;
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  if (threadIdx.x == 0) {
    int32_t b = 0;
    for (int j = 0; j < m; ++j) b += n_valid[j];
    s_base = b;
    base_out[m] = b;
    if (m == M - 1) base_out[M] = b + n_valid[m];
  }
  __syncthreads();
  int32_t base = s_base;
  for (int64_t i0 = 0; i0 < n; i0 += kFillThreads) {
    const int64_t i = i0 + threadIdx.x;
    const bool f = i < n && vm[i] == m;
    const unsigned b = __ballot_sync(0xffffffffu, f);
    if (lane == 0) wcnt[wid] = __popc(b);
    __syncthreads();
    int32_t before = 0, total = 0;
    for (int w = 0; w < kFillThreads / 32; ++w) {
      const int32_t c = wcnt[w];
      before += w < wid ? c : 0;
      total += c;
    }
    if (f) list[base + before + __popc(b & ((1u << lane) - 1u))] = (int32_t)i;
    base += total;
    __syncthreads();
  }
}

// the model-grouped columns a lane walks: arrival, time to first and last
// token, prompt and output lengths, in the grouped order
__global__ void k_rp_gather(int64_t n_valid_total, ReplayLatent lat,
                            const int32_t* __restrict__ list, const int32_t* __restrict__ base,
                            int M, int4* __restrict__ g) {
  const int64_t n = base[M];
  for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < n;
       p += (int64_t)gridDim.x * blockDim.x) {
    const int32_t i = list[p];
    g[2 * p] = make_int4(lat.t_arr[i], lat.d_first[i], lat.d_total[i], i);
    g[2 * p + 1] = make_int4(lat.L_in[i], lat.L_out[i], 0, 0);
  }
}

// served records start as "not started" (K*win) or "not served" (-1)
__global__ void k_rp_init_records(int64_t n, int n_inst, int32_t span, const int8_t* __restrict__ vm,
                                  int32_t* ts, int32_t* tf, int32_t* te) {
  const int64_t total = n * n_inst;
  for (int64_t x = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; x < total;
       x += (int64_t)gridDim.x * blockDim.x) {
    const int32_t v = vm[x % n] >= 0 ? span : -1;
    ts[x] = v;
    tf[x] = v;
    te[x] = v;
  }
}

// ---- per-model server heaps -----------------------------------------------
struct Heap {
  long long* h;
  int n;
  __device__ void sift_down(int i) {
    const long long v = h[i];
    for (;;) {
      int c = 2 * i + 1;
      if (c >= n) break;
      if (c + 1 < n && h[c + 1] < h[c]) ++c;
      if (h[c] >= v) break;
      h[i] = h[c];
      i = c;
    }
    h[i] = v;
  }
  __device__ void replace_top(long long v) {
    h[0] = v;
    sift_down(0);
  }
  __device__ void pop() {
    --n;
    if (n > 0) {
      h[0] = h[n];
      sift_down(0);
    }
  }
  __device__ void push(long long v) {
    int i = n++;
    while (i > 0) {
      const int p = (i - 1) >> 1;
      if (h[p] <= v) break;
      h[i] = h[p];
      i = p;
    }
    h[i] = v;
  }
};

// tokens emitted strictly before tick t by a request with first token at tf,
// last at te and L output tokens (token j at tf + floor(j*(te-tf)/(L-1)))
__device__ __forceinline__ long long tokens_before(long long t, long long tf, long long te,
                                                   long long L) {
  if (t <= tf) return 0;
  if (t > te) return L;
  if (L == 1) return 1;
  const unsigned long long num = (unsigned long long)(t - tf) * (unsigned long long)(L - 1);
  const unsigned long long dur = (unsigned long long)(te - tf);
  const unsigned long long y = num + dur - 1;
  if ((y >> 32) == 0) return (long long)((uint32_t)y / (uint32_t)dur);   // 32-bit divide
  return (long long)(y / dur);
}

// A request still emitting decode tokens after its first-token window: the
// window from which it contributes, its last window (within the grid), its
// last token time, output length and tokens counted so far. With
// y = (T - tf)(L - 1) + dur - 1 the tokens before T are floor(y / dur) while
// T <= te; moving T one window on adds win * (L - 1) = qd * dur + rd to y, so
// the count is carried as a quotient and remainder without dividing.
struct Decoding {
  int32_t k_from, k_last, te, L, done;
  int32_t q, r;            // floor and remainder of y / dur at T = k_from * win
  int32_t qd, rd, dur;
};
// per-model window ring (power of two) and pending far-window list sizes; the
// four counts a window collects
constexpr int kRing = 64, kFar = 32, kQ = 32;
enum { kP = 0, kD = 1, kEnd = 2, kLate = 3 };

// window k ends a tick of cadence c when a multiple of c falls in (k*win, (k+1)*win]
__device__ __forceinline__ bool ends_tick(long long k, int win, int c) {
  return ((k + 1) * (long long)win) / c > (k * (long long)win) / c;
}

template <class T> struct Ctl {
  const ReplayBatch<T>& b;
  const T* z;
  const uint8_t* c;
  const uint8_t* flag;   // bit 0: latency guard breached in the window; bit 1: lost capacity
  int32_t* r;
  T tc;            // the instance's rescue threshold (NaN: per model from the profile)
  __device__ T tcrit(int m) const { return tc == tc ? tc : b.tau_crit[m]; }
  __device__ uint8_t region(int m) const {
    if (c[m] == TRE_IDLE) return TRE_IDLE;
    if (z[m] < tcrit(m)) return TRE_CRIT;
    if (z[m] > b.tau_surp[m]) return TRE_SURP;
    return TRE_NOM;
  }
  __device__ bool held(int m) const { return flag[m] & 1; }
  // donor preference: idle models (lowest index), then surplus by Z
  // descending, then nominal by Z descending (with nom_above only above the
  // receiver's Z); never critical, never the receiver, never below the floor,
  // never a donor whose latency guard is breached (its release is deferred)
  __device__ int pick(const int32_t* rr, int recv, bool nom_above) const {
    const int M = b.M;
    for (int m = 0; m < M; ++m)
      if (m != recv && region(m) == TRE_IDLE && rr[m] > b.r_min[m] && !held(m)) return m;
    int best = -1;
    for (int m = 0; m < M; ++m)
      if (m != recv && region(m) == TRE_SURP && rr[m] > b.r_min[m] && !held(m) &&
          (best < 0 || z[m] > z[best]))
        best = m;
    if (best >= 0) return best;
    for (int m = 0; m < M; ++m) {
      if (m == recv || region(m) != TRE_NOM || rr[m] <= b.r_min[m] || held(m)) continue;
      if (nom_above && !(z[m] > z[recv])) continue;
      if (best < 0 || z[m] > z[best]) best = m;
    }
    return best;
  }
};

template <class T, int MPL, bool SHEAP>
__global__ void __launch_bounds__(256, 1)
k_replay(const __grid_constant__ ReplayBatch<T> b) {
  extern __shared__ unsigned long long rsm[];
  const int wid = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int inst = blockIdx.x * b.warps_per_cta + wid;
  if (inst >= b.n_inst) return;                 // whole warps only
  const int M = b.M, win = b.win, K = b.K;
  const long long span = (long long)K * win;
  // this warp's shared region: Z row, class row, replicas, dry-run replicas,
  // heap sizes, then (shared heaps) the heaps
  char* base = reinterpret_cast<char*>(rsm) + (size_t)wid * b.warp_bytes;
  T* zrow = reinterpret_cast<T*>(base);
  int32_t* r = reinterpret_cast<int32_t*>(zrow + M);
  int32_t* rr = r + M;
  int32_t* hs = rr + M;
  uint8_t* crow = reinterpret_cast<uint8_t*>(hs + M);
  uint8_t* frow = crow + M;                     // guard / lost-capacity flags
  long long* heaps = SHEAP ? reinterpret_cast<long long*>(base + b.heap_off)
                           : b.gheap + (size_t)inst * M * b.hcap;
  // per model, the requests still decoding past their first-token window
  Decoding* act = reinterpret_cast<Decoding*>(base + b.act_off);
  const int ti = inst / b.n_cap, ci = inst % b.n_cap;
  const int pacing = b.cap_list[ci];
  const T tc = b.n_tau > 0 ? b.tau_list[ti] : (T)NAN;
  // per-window prompt tokens, decode tokens, running-span ends and late first
  // tokens beyond the ring, [4][K + 1][M]
  uint32_t* Gacc = b.acc + (size_t)inst * 4 * (K + 1) * M;
  uint32_t* ring = reinterpret_cast<uint32_t*>(base + b.ring_off);   // [4][M][kRing]
  int32_t* farl = reinterpret_cast<int32_t*>(ring + (size_t)4 * M * kRing);  // [M][kFar]
  // each model's next requests, staged from the grouped columns: grouped
  // positions [qend - kQ, qend) sit in slot position % kQ; qhead mirrors the
  // owning lane's cursor for the refill
  int4* qbuf = reinterpret_cast<int4*>(base + b.q_off);              // [M][kQ][2]
  int32_t* qhead = reinterpret_cast<int32_t*>(qbuf + (size_t)M * kQ * 2);
  int32_t* qend = qhead + M;
  for (int c = lane; c < 4 * M * kRing; c += 32) ring[c] = 0;
  // initial replicas: one server free at t = 0 per replica
  long long used = 0;
  bool bad = false;
  for (int j = 0; j < MPL; ++j) {
    const int m = lane + 32 * j;
    if (m >= M) continue;
    const int32_t r0 = b.r0[m], g = b.footprint[m];
    bad |= r0 < 0 || g < 1 || b.r_min[m] < 0;
    used += (long long)g * r0;
    r[m] = r0;
    hs[m] = r0;
  }
  for (int o = 16; o > 0; o >>= 1) used += __shfl_xor_sync(0xffffffffu, used, o);
  bad = __any_sync(0xffffffffu, bad) || used > b.budget;
  if (bad) {
    if (lane == 0) {
      b.diag->err = TRE_EINVAL;
      b.n_moves[inst] = 0;
    }
    return;
  }
  for (int j = 0; j < MPL; ++j) {
    const int m = lane + 32 * j;
    if (m >= M) continue;
    for (int q = 0; q < r[m]; ++q) heaps[(size_t)m * b.hcap + q] = 0;
  }
  // per-model state of this lane
  int32_t head[MPL], end[MPL], n_act[MPL], n_far[MPL];
  bool far_all[MPL];
  uint32_t arr_next[MPL];
  T pw[MPL], pq[MPL], pa[MPL], pth[MPL], ptc[MPL], pts[MPL];   // the profile, per model
  long long cum_arr[MPL], cum_start[MPL], cum_end[MPL], met[MPL];
  T S[MPL];
  bool init[MPL];
  const T dt = (T)win / (T)1000;
  for (int j = 0; j < MPL; ++j) {
    const int m = lane + 32 * j;
    head[j] = m < M ? b.base[m] : 0;
    end[j] = m < M ? b.base[m + 1] : 0;
    n_act[j] = 0;
    n_far[j] = 0;
    far_all[j] = false;
    arr_next[j] = m < M && K > 0 ? (uint32_t)b.arr_cnt[m] : 0u;
    if (m < M) {
      pw[j] = b.w_p[m];
      pq[j] = b.w_q[m];
      pa[j] = b.alpha[m];
      pth[j] = b.theta[m];
      ptc[j] = tc == tc ? tc : b.tau_crit[m];
      pts[j] = b.tau_surp[m];
    }
    if (m < M) {
      qhead[m] = head[j];
      qend[m] = head[j];
    }
    cum_arr[j] = cum_start[j] = cum_end[j] = met[j] = 0;
    S[j] = (T)0;
    init[j] = false;
  }
  long long free_pool = b.budget - used;        // lane 0's copy is the live one
  long long reb_until = 0;                      // a rebalance transfer serves from here on
  int64_t nm = 0;
  __syncwarp();
  for (int k = 0; k < K; ++k) {
    const long long Tk = (long long)(k + 1) * win;
    // top up the staged requests of every model that has used half of them:
    // the warp loads up to kQ of a model's next requests at once
    for (int j = 0; j < MPL; ++j) {
      const int m = lane + 32 * j;
      const bool want = m < M && qend[m] < end[j] && qend[m] - head[j] < kQ / 2 &&
                        head[j] < end[j];
      unsigned need = __ballot_sync(0xffffffffu, want);
      while (need) {
        const int l = __ffs(need) - 1;
        need &= need - 1;
        const int mm = l + 32 * j;
        const int h = __shfl_sync(0xffffffffu, head[j], l);
        const int ne = __shfl_sync(0xffffffffu, end[j], l);
        const int e = max(qend[mm], h);          // the owner may have read past them
        const int upto = min(h + kQ, ne);
        const int p = e + lane;
        if (p < upto) {
          int4* slot = qbuf + ((size_t)mm * kQ + (p & (kQ - 1))) * 2;
          slot[0] = b.grp[2 * (size_t)p];
          slot[1] = b.grp[2 * (size_t)p + 1];
        }
        __syncwarp();
        if (lane == 0) qend[mm] = upto;
        __syncwarp();
      }
    }
    for (int j = 0; j < MPL; ++j) {
      const int m = lane + 32 * j;
      if (m >= M) continue;
      Heap hp{heaps + (size_t)m * b.hcap, hs[m]};
      Decoding* am = act + (size_t)m * b.acap;
      int32_t* fl = farl + (size_t)m * kFar;
      // per-window counts of this model: windows k .. k+kRing-1 in the shared
      // ring, later ones in the instance's global accumulators (their windows
      // listed, or every row reads them once the list has overflowed)
      auto add = [&](int arr, long long kt, uint32_t v) {
        if (kt - k < kRing) {
          ring[((size_t)arr * M + m) * kRing + (kt & (kRing - 1))] += v;
          return;
        }
        Gacc[(size_t)arr * (K + 1) * M + kt * M + m] += v;
        if (far_all[j]) return;
        for (int q = 0; q < n_far[j]; ++q)
          if (fl[q] == (int32_t)kt) return;
        if (n_far[j] < kFar) fl[n_far[j]++] = (int32_t)kt;
        else far_all[j] = true;
      };
      // start every request of the model that can start before T, in order
      const int staged_end = qend[m];
      while (head[j] < end[j] && hp.n > 0) {
        int4 c0, c1;
        if (head[j] < staged_end) {
          const int4* slot = qbuf + ((size_t)m * kQ + (head[j] & (kQ - 1))) * 2;
          c0 = slot[0];
          c1 = slot[1];
        } else {                                 // beyond the staged ones
          c0 = b.grp[2 * (size_t)head[j]];
          c1 = b.grp[2 * (size_t)head[j] + 1];
        }
        const long long ta = c0.x;
        const long long st = max(ta, hp.h[0]);
        if (st >= Tk) break;
        const long long dtot = c0.z;
        const long long tf = min(st + (long long)c0.y, 2147483647ll);
        const long long te = min(st + dtot, 2147483647ll);
        const int32_t i = c0.w, L_in = c1.x, L_out = c1.y;
        hp.replace_top(st + dtot);
        ++head[j];
        ++cum_start[j];
        if (b.o_ts) {
          const size_t x = (size_t)inst * b.lat.n + i;
          b.o_ts[x] = (int32_t)st;
          b.o_tf[x] = (int32_t)tf;
          b.o_te[x] = (int32_t)te;
        }
        if (b.slo_ms && tf - ta <= (long long)b.slo_ms[m]) ++met[j];
        bool ends_via_list = false;
        if (tf < span) {
          // times fit 31 bits: 32-bit divisions
          const long long kf = (uint32_t)tf / (uint32_t)win;
          const long long ke = min((long long)((uint32_t)te / (uint32_t)win), (long long)K - 1);
          if (b.guard_ms && tf - ta > (long long)b.guard_ms[m]) add(kLate, kf, 1u);
          add(kP, kf, (uint32_t)L_in);
          const long long first = tokens_before((kf + 1) * win, tf, te, L_out);
          if (first) add(kD, kf, (uint32_t)first);
          if (ke > kf && L_out >= 2) {
            if (n_act[j] < b.acap) {             // later windows: counted window by window
              // here te >= (kf + 1) * win > tf and L_out >= 2 (else every token
              // of the request falls in window kf)
              const unsigned long long dur = (unsigned long long)(te - tf);
              const unsigned long long y = (unsigned long long)((kf + 1) * win - tf) *
                                               (unsigned long long)(L_out - 1) + dur - 1;
              const unsigned long long step = (unsigned long long)win * (L_out - 1);
              Decoding d;
              d.k_from = (int32_t)kf + 1;
              d.k_last = (int32_t)ke;
              d.te = (int32_t)te;
              d.L = L_out;
              d.done = (int32_t)first;
              d.q = (int32_t)(y / dur);
              d.r = (int32_t)(y - (unsigned long long)d.q * dur);
              // a step of more than L tokens ends the request in the next
              // window, where the count is L: the clamp never shows
              const unsigned long long qd = step / dur;
              d.qd = (int32_t)min(qd, (unsigned long long)L_out + 1);
              d.rd = (int32_t)(step - qd * dur);
              d.dur = (int32_t)dur;
              am[n_act[j]++] = d;
              ends_via_list = true;
            } else {                             // no room: add them all now
              long long prev = first;
              for (long long kk = kf + 1; kk <= ke; ++kk) {
                const long long nxt = tokens_before((kk + 1) * win, tf, te, L_out);
                if (nxt != prev) add(kD, kk, (uint32_t)(nxt - prev));
                prev = nxt;
              }
            }
          }
        }
        // the running span ends in window te / win (never read when te is
        // past the grid); a listed request counts its end when it retires
        if (!ends_via_list && te < span) add(kEnd, (uint32_t)te / (uint32_t)win, 1u);
      }
      qhead[m] = head[j];
      // decode tokens of the requests still decoding, for window k, and the
      // ends of those that retire in it
      uint32_t d_live = 0, e_live = 0;
      for (int q = 0; q < n_act[j];) {
        Decoding& e = am[q];
        if (e.k_from > k) {
          ++q;
          continue;
        }
        // y at the end of window k
        e.q += e.qd;
        e.r += e.rd;
        if (e.r >= e.dur) {
          e.r -= e.dur;
          e.q += 1;
        }
        const int32_t nxt = (long long)(k + 1) * win > (long long)e.te ? e.L : e.q;
        d_live += (uint32_t)(nxt - e.done);
        e.done = nxt;
        if (e.k_last <= k) {
          if ((long long)e.te < span) ++e_live;
          am[q] = am[--n_act[j]];
        } else {
          ++q;
        }
      }
      // window k's counts: the ring slot (cleared for window k + kRing) plus
      // any later-window contributions made before the ring reached it
      uint32_t v[4];
      bool far = far_all[j];
      for (int q = 0; q < n_far[j]; ++q)
        if (fl[q] == k) {
          far = true;
          fl[q] = fl[--n_far[j]];
          break;
        }
#pragma unroll
      for (int a = 0; a < 4; ++a) {
        uint32_t* slot = &ring[((size_t)a * M + m) * kRing + (k & (kRing - 1))];
        v[a] = *slot;
        *slot = 0;
        if (far) v[a] += Gacc[(size_t)a * (K + 1) * M + (size_t)k * M + m];
      }
      const size_t x = (size_t)k * M + m;
      cum_arr[j] += arr_next[j];
      if (k + 1 < K) arr_next[j] = b.arr_cnt[x + M];   // the next window's arrivals, early
      cum_end[j] += v[kEnd] + e_live;
      const int32_t P = (int32_t)v[kP], D = (int32_t)(v[kD] + d_live);
      const int32_t A = (int32_t)(cum_start[j] - cum_end[j]);
      const int32_t W = (int32_t)(cum_arr[j] - cum_start[j]);
      const bool idle = P == 0 && D == 0 && A == 0 && W == 0;
      if (!idle) {
        const T r_pre = (T)P / dt;
        const T r_dec = (T)D / dt;
        const T svc = pw[j] * r_pre;
        const T num = svc + r_dec;
        const T qw = pq[j] * (T)W;
        T den = (T)A + qw;
        if (den < (T)1) den = (T)1;
        const T raw = num / den;
        if (!init[j]) {
          S[j] = raw;
          init[j] = true;
        } else {
          const T x1 = pa[j] * raw;
          const T x2 = ((T)1 - pa[j]) * S[j];
          S[j] = x1 + x2;
        }
      }
      const T Z = S[j] / pth[j];
      uint8_t cl;
      if (idle) cl = TRE_IDLE;
      else if (Z < ptc[j]) cl = TRE_CRIT;
      else if (Z > pts[j]) cl = TRE_SURP;
      else cl = TRE_NOM;
      zrow[m] = Z;
      crow[m] = cl;
      // latency guard breached in the window; requests waiting with no
      // routable replica (lost capacity)
      frow[m] = (uint8_t)((b.guard_ms && v[kLate] ? 1 : 0) | (r[m] == 0 && W > 0 ? 2 : 0));
      if (b.Z) {
        const size_t y = (size_t)inst * K * M + x;
        b.Z[y] = Z;
        b.cls[y] = cl;
      }
    }
    const bool fast = ends_tick(k, win, b.fast_ms), slow = ends_tick(k, win, b.slow_ms);
    if (!fast && !slow) continue;
    __threadfence_block();
    __syncwarp();
    if (lane == 0) {
      Ctl<T> ctl{b, zrow, crow, frow, r, tc};
      int recv = -1, kind = 0;
      bool nom_above = false, deferred = false;
      if (fast) {
        // rescue: a latency-guard breach pre-empts every other event (lowest
        // Z among the breaching models); otherwise the lowest Z among critical
        // models and models that lost their routable capacity. A rebalance
        // transfer in progress defers a rescue without a breach; the pending
        // rescue keeps the slow loop out of the tick.
        bool hard = false;
        for (int m = 0; m < M; ++m)
          if ((frow[m] & 1) && (recv < 0 || zrow[m] < zrow[recv])) recv = m;
        if (recv >= 0) {
          hard = true;
        } else {
          for (int m = 0; m < M; ++m)
            if ((ctl.region(m) == TRE_CRIT || (frow[m] & 2)) && (recv < 0 || zrow[m] < zrow[recv]))
              recv = m;
        }
        if (recv >= 0) {
          if (Tk < reb_until && !hard) deferred = true;
          else kind = TRE_RESCUE;
        }
      }
      if (kind == 0 && recv < 0 && slow) {       // rebalance: Eq. 3 over non-idle models
        for (int m = 0; m < M; ++m)
          if (ctl.region(m) != TRE_IDLE && (recv < 0 || zrow[m] < zrow[recv])) recv = m;
        if (recv >= 0 && zrow[recv] < (T)1) {
          kind = TRE_REBALANCE;
          nom_above = true;
        }
      }
      auto emit = [&](int recv_m, int donor, int seq) {
        if (nm < b.moves_cap) {
          tre_move mv;
          mv.window = k;
          mv.recv = (int16_t)recv_m;
          mv.donor = (int16_t)donor;
          mv.kind = (uint8_t)kind;
          mv.seq = (uint8_t)seq;
          mv.reserved = 0;
          b.moves[(size_t)inst * b.moves_cap + nm] = mv;
        }
        ++nm;
      };
      if (deferred) kind = 0;
      for (int seq = 0; kind && seq < pacing; ++seq) {
        const long long need = b.footprint[recv];
        Heap hr{heaps + (size_t)recv * b.hcap, hs[recv]};
        if (free_pool >= need) {                 // idle capacity first
          free_pool -= need;
          r[recv] += 1;
          emit(recv, -1, seq);
          hr.push(Tk + b.wake_ms);
          hs[recv] = hr.n;
          if (kind == TRE_REBALANCE) reb_until = max(reb_until, Tk + (long long)b.wake_ms);
          continue;
        }
        // dry run: can the eligible donors cover the receiver's footprint?
        for (int m = 0; m < M; ++m) rr[m] = r[m];
        long long f = free_pool;
        bool ok = true;
        while (f < need) {
          const int d = ctl.pick(rr, recv, nom_above);
          if (d < 0) {
            ok = false;
            break;
          }
          rr[d] -= 1;
          f += b.footprint[d];
        }
        if (!ok) break;
        // commit: the same releases, each the donor's server that frees first
        f = free_pool;
        long long gpu_free = Tk;
        while (f < need) {
          const int d = ctl.pick(r, recv, nom_above);
          r[d] -= 1;
          f += b.footprint[d];
          emit(recv, d, seq);
          Heap hd{heaps + (size_t)d * b.hcap, hs[d]};
          const long long drained = max(hd.h[0], Tk);
          hd.pop();
          hs[d] = hd.n;
          gpu_free = max(gpu_free, drained + b.sleep_ms);
        }
        free_pool = f - need;
        r[recv] += 1;
        hr.push(gpu_free + b.wake_ms);
        hs[recv] = hr.n;
        if (kind == TRE_REBALANCE) reb_until = max(reb_until, gpu_free + (long long)b.wake_ms);
      }
    }
    __threadfence_block();
    __syncwarp();
  }
  // requests never started count against the SLO with their first token at
  // the end of the grid
  for (int j = 0; j < MPL; ++j) {
    const int m = lane + 32 * j;
    if (m >= M) continue;
    if (b.slo_ms) {
      for (int32_t q = head[j]; q < end[j]; ++q)
        if (span - (long long)b.grp[2 * q].x <= (long long)b.slo_ms[m]) ++met[j];
      if (b.slo_met) b.slo_met[(size_t)inst * M + m] = met[j];
    }
    if (b.served) b.served[(size_t)inst * M + m] = cum_start[j];
    b.r_final[(size_t)inst * M + m] = r[m];
  }
  if (lane == 0) {
    b.n_moves[inst] = nm;
    if (nm > b.moves_cap) b.diag->err = TRE_EOVERFLOW;
  }
}

constexpr size_t kReplaySmemMax = 160 * 1024;

template <class T> int warp_base_bytes(int M) {
  size_t o = ((size_t)M * sizeof(T) + 15) & ~(size_t)15;   // Z row
  o += (size_t)M * 4 * 3;                                   // r, dry-run r, heap sizes
  o += (size_t)M * 2;                                       // class and flag rows
  return (int)((o + 15) & ~(size_t)15);
}

}  // namespace

template <class T> void replay_ws_layout(Arena& a, ReplayBatch<T>& b, ReplayWs& w) {
  const int M = b.M, K = b.K;
  w.vm = a.take<int8_t>((size_t)std::max<int64_t>(b.lat.n, 1));
  w.arr_cnt = a.take<int32_t>((size_t)K * M + 1);
  w.n_valid = a.take<int32_t>((size_t)M);
  w.base = a.take<int32_t>((size_t)M + 1);
  w.list = a.take<int32_t>((size_t)std::max<int64_t>(b.lat.n, 1));
  w.acc = a.take<uint32_t>((size_t)b.n_inst * 4 * (K + 1) * M);
  w.grp = a.take<int4>((size_t)std::max<int64_t>(b.lat.n, 1) * 2);
  // warps per CTA: spread the instances over the SMs first
  const int sms = device_sm_count();
  int W = (int)std::min<int64_t>(8, std::max<int64_t>(1, (b.n_inst + sms - 1) / sms));
  auto a16 = [](size_t x) { return (x + 15) & ~(size_t)15; };
  const size_t wb = (size_t)warp_base_bytes<T>(M);
  const size_t hb = a16((size_t)M * b.hcap * 8);
  const size_t ring_bytes = a16((size_t)M * (4 * kRing + kFar) * 4);
  const size_t q_bytes = a16((size_t)M * kQ * 32 + (size_t)M * 8);
  // decoding requests per model: room for as many as the budget has replicas
  // (more are added straight to the accumulators), at least 8
  int acap = std::max(8, std::min(b.hcap, 256));
  auto act_bytes = [&](int c) { return a16((size_t)M * c * sizeof(Decoding)); };
  w.shared_heaps = false;
  for (int tw = W; tw >= 1; tw >>= 1) {
    if ((wb + hb + q_bytes + ring_bytes + act_bytes(8)) * tw <= kReplaySmemMax) {
      w.shared_heaps = true;
      W = tw;
      break;
    }
  }
  const size_t fixed = wb + (w.shared_heaps ? hb : 0) + q_bytes + ring_bytes;
  if (!w.shared_heaps) W = 1;
  while (acap > 8 && (fixed + act_bytes(acap)) * W > kReplaySmemMax) acap >>= 1;
  w.warps_per_cta = W;
  b.warps_per_cta = W;
  // per warp: base rows | heaps (when shared) | staged requests | rings | lists
  b.heap_off = (int)wb;
  b.q_off = (int)(wb + (w.shared_heaps ? hb : 0));
  b.ring_off = (int)(b.q_off + q_bytes);
  b.act_off = (int)(b.ring_off + ring_bytes);
  b.acap = acap;
  b.warp_bytes = (int)(fixed + act_bytes(acap));
  w.gheap = w.shared_heaps ? nullptr
                           : a.take<long long>((size_t)b.n_inst * M * b.hcap);
  b.list = w.list;
  b.grp = w.grp;
  b.base = w.base;
  b.arr_cnt = w.arr_cnt;
  b.acc = w.acc;
  b.gheap = w.gheap;
}

template <class T> cudaError_t launch_replay(ReplayBatch<T>& b, ReplayWs& w, cudaStream_t s) {
  const int M = b.M, K = b.K;
  cudaError_t e = cudaMemsetAsync(w.arr_cnt, 0, ((size_t)K * M + 1) * sizeof(int32_t), s);
  if (!e) e = cudaMemsetAsync(w.n_valid, 0, (size_t)M * sizeof(int32_t), s);
  if (!e) e = cudaMemsetAsync(w.acc, 0, (size_t)b.n_inst * 4 * (K + 1) * M * sizeof(uint32_t), s);
  if (e) return e;
  const int sms = device_sm_count();
  const unsigned g1 = (unsigned)std::max<int64_t>(
      1, std::min<int64_t>((b.lat.n + 255) / 256, (int64_t)sms * 8));
  if (b.lat.n > 0) k_rp_valid<<<g1, 256, 0, s>>>(b.lat, M, b.win, K, w.vm, w.arr_cnt, w.n_valid);
  k_rp_fill<<<M, kFillThreads, 0, s>>>(b.lat.n, M, w.vm, w.n_valid, w.list, w.base);
  if (b.lat.n > 0) k_rp_gather<<<g1, 256, 0, s>>>(b.lat.n, b.lat, w.list, w.base, M, w.grp);
  if ((e = cudaGetLastError())) return e;
  if (b.o_ts && b.lat.n > 0) {
    k_rp_init_records<<<(unsigned)sms * 8, 256, 0, s>>>(b.lat.n, b.n_inst, (int32_t)(K * b.win),
                                                        w.vm, b.o_ts, b.o_tf, b.o_te);
    if ((e = cudaGetLastError())) return e;
  }
  const int W = w.warps_per_cta;
  const unsigned grid = (unsigned)((b.n_inst + W - 1) / W);
  const size_t smem = (size_t)b.warp_bytes * W;
  const void* fn;
  if (M <= 32)
    fn = w.shared_heaps ? (const void*)k_replay<T, 1, true> : (const void*)k_replay<T, 1, false>;
  else
    fn = w.shared_heaps ? (const void*)k_replay<T, 2, true> : (const void*)k_replay<T, 2, false>;
  if ((e = func_smem_once(fn, (int)kReplaySmemMax, false))) return e;
  if (M <= 32) {
    if (w.shared_heaps) k_replay<T, 1, true><<<grid, 32 * W, smem, s>>>(b);
    else k_replay<T, 1, false><<<grid, 32 * W, smem, s>>>(b);
  } else {
    if (w.shared_heaps) k_replay<T, 2, true><<<grid, 32 * W, smem, s>>>(b);
    else k_replay<T, 2, false><<<grid, 32 * W, smem, s>>>(b);
  }
  return cudaGetLastError();
}

template void replay_ws_layout<float>(Arena&, ReplayBatch<float>&, ReplayWs&);
template void replay_ws_layout<double>(Arena&, ReplayBatch<double>&, ReplayWs&);
template cudaError_t launch_replay<float>(ReplayBatch<float>&, ReplayWs&, cudaStream_t);
template cudaError_t launch_replay<double>(ReplayBatch<double>&, ReplayWs&, cudaStream_t);

}  // namespace tre
