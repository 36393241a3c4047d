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
  const long long num = (t - tf) * (L - 1), dur = te - tf;
  return (num + dur - 1) / dur;
}

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
__global__ void __launch_bounds__(256)
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
  const int ti = inst / b.n_cap, ci = inst % b.n_cap;
  const int pacing = b.cap_list[ci];
  const T tc = b.n_tau > 0 ? b.tau_list[ti] : (T)NAN;
  uint32_t* Pacc = b.acc + (size_t)inst * 4 * (K + 1) * M;
  uint32_t* Dacc = Pacc + (size_t)(K + 1) * M;
  uint32_t* Eacc = Dacc + (size_t)(K + 1) * M;
  uint32_t* Lacc = Eacc + (size_t)(K + 1) * M;  // first tokens later than the guard
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
  int32_t head[MPL], end[MPL];
  long long cum_arr[MPL], cum_start[MPL], cum_end[MPL], met[MPL];
  T S[MPL];
  bool init[MPL];
  const T dt = (T)win / (T)1000;
  for (int j = 0; j < MPL; ++j) {
    const int m = lane + 32 * j;
    head[j] = m < M ? b.base[m] : 0;
    end[j] = m < M ? b.base[m + 1] : 0;
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
    for (int j = 0; j < MPL; ++j) {
      const int m = lane + 32 * j;
      if (m >= M) continue;
      Heap hp{heaps + (size_t)m * b.hcap, hs[m]};
      // start every request of the model that can start before T, in order
      while (head[j] < end[j] && hp.n > 0) {
        const int32_t i = b.list[head[j]];
        const long long ta = b.lat.t_arr[i];
        const long long st = max(ta, hp.h[0]);
        if (st >= Tk) break;
        const long long dtot = b.lat.d_total[i];
        const long long tf = min(st + (long long)b.lat.d_first[i], 2147483647ll);
        const long long te = min(st + dtot, 2147483647ll);
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
        if (b.guard_ms && tf < span && tf - ta > (long long)b.guard_ms[m])
          Lacc[(tf / win) * M + m] += 1u;
        if (tf < span) {
          const long long kf = tf / win, ke = min(te / win, (long long)K - 1);
          Pacc[kf * M + m] += (uint32_t)b.lat.L_in[i];
          const long long L = b.lat.L_out[i];
          long long prev = tokens_before(kf * win, tf, te, L);
          for (long long kk = kf; kk <= ke; ++kk) {
            const long long nxt = tokens_before((kk + 1) * win, tf, te, L);
            if (nxt != prev) Dacc[kk * M + m] += (uint32_t)(nxt - prev);
            prev = nxt;
          }
        }
        Eacc[min(te / win, (long long)K) * M + m] += 1u;
      }
      // window k's telemetry, scored with the carried smoothing state
      const size_t x = (size_t)k * M + m;
      cum_arr[j] += b.arr_cnt[x];
      cum_end[j] += Eacc[x];
      const int32_t P = (int32_t)Pacc[x], D = (int32_t)Dacc[x];
      const int32_t A = (int32_t)(cum_start[j] - cum_end[j]);
      const int32_t W = (int32_t)(cum_arr[j] - cum_start[j]);
      const bool idle = P == 0 && D == 0 && A == 0 && W == 0;
      if (!idle) {
        const T r_pre = (T)P / dt;
        const T r_dec = (T)D / dt;
        const T svc = b.w_p[m] * r_pre;
        const T num = svc + r_dec;
        const T qw = b.w_q[m] * (T)W;
        T den = (T)A + qw;
        if (den < (T)1) den = (T)1;
        const T raw = num / den;
        if (!init[j]) {
          S[j] = raw;
          init[j] = true;
        } else {
          const T a = b.alpha[m];
          const T x1 = a * raw;
          const T x2 = ((T)1 - a) * S[j];
          S[j] = x1 + x2;
        }
      }
      const T Z = S[j] / b.theta[m];
      uint8_t cl;
      const T tcm = tc == tc ? tc : b.tau_crit[m];
      if (idle) cl = TRE_IDLE;
      else if (Z < tcm) cl = TRE_CRIT;
      else if (Z > b.tau_surp[m]) cl = TRE_SURP;
      else cl = TRE_NOM;
      zrow[m] = Z;
      crow[m] = cl;
      // latency guard breached in the window; requests waiting with no
      // routable replica (lost capacity)
      frow[m] = (uint8_t)((b.guard_ms && Lacc[x] ? 1 : 0) | (r[m] == 0 && W > 0 ? 2 : 0));
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
        if (span - (long long)b.lat.t_arr[b.list[q]] <= (long long)b.slo_ms[m]) ++met[j];
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
  // warps per CTA: spread the instances over the SMs first
  const int sms = device_sm_count();
  int W = (int)std::min<int64_t>(8, std::max<int64_t>(1, (b.n_inst + sms - 1) / sms));
  const size_t wb = (size_t)warp_base_bytes<T>(M);
  const size_t hb = (size_t)M * b.hcap * 8;
  w.shared_heaps = false;
  for (int tw = W; tw >= 1; tw >>= 1) {
    if ((wb + hb) * tw <= kReplaySmemMax) {
      w.shared_heaps = true;
      W = tw;
      break;
    }
  }
  w.warps_per_cta = W;
  b.warps_per_cta = W;
  b.heap_off = (int)wb;
  b.warp_bytes = (int)(w.shared_heaps ? wb + hb : wb);
  w.gheap = w.shared_heaps ? nullptr
                           : a.take<long long>((size_t)b.n_inst * M * b.hcap);
  b.list = w.list;
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
