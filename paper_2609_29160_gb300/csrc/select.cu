// Open-loop TRE move selection (Sec. IV-B dual-speed control, Eq. 3 receiver,
// Sec. IV-C bounded pairwise transfer under a fixed budget).
//
// Everything that does not depend on the replica state is computed first, in
// parallel, for every (series, rescue threshold, control tick):
//   - at each fast tick: whether any model is critical, the rescue receiver
//     (lowest Z among critical models, lowest index on ties) and every model's
//     rank in the rescue donor order;
//   - at each slow tick: the Eq. 3 receiver over non-idle models, whether its
//     Z is below 1, and every model's rank in the rebalance donor order.
// Donor order: idle models by index, then surplus by Z descending, then
// nominal by Z descending (in rebalance only those above the receiver's Z);
// critical models and the receiver get no rank.
// The serial part -- one warp per controller instance walking its ticks with
// the replica counts in registers (models m = lane + 32*j) -- then only picks,
// per released replica, the lowest-ranked model still above its floor.
#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace tre {
namespace {

constexpr int kWarpsPerBlock = 4;
constexpr uint16_t kNoRank = 0xffff;

__device__ __forceinline__ int64_t tick_window(int64_t j, int64_t cadence, int64_t win) {
  // window whose right edge passes the j-th multiple of the cadence (j >= 1)
  return (j * cadence + win - 1) / win - 1;
}

template <class T>
__device__ __forceinline__ uint8_t region_of(uint8_t c, T z, T tc, T ts) {
  if (c == kIdle) return kIdle;
  if (z < tc) return kCrit;
  if (z > ts) return kSurp;
  return kNom;
}

// One thread per (series, tau, tick entry, model). Entries [0, nf) of a series
// are its fast ticks, [nf, nf + ns) its slow ticks.
template <class T>
__global__ void __launch_bounds__(256)
k_tick_rank(const __grid_constant__ WalkBatch<T> b, int16_t* recv_out, uint16_t* rank) {
  const int M = b.M;
  const int64_t gid = (int64_t)blockIdx.x * 256 + threadIdx.x;
  const int64_t total_ent = (int64_t)b.ent_base[b.n_series] * b.n_tau;
  if (gid >= total_ent * M) return;
  const int m = (int)(gid % M);
  const int64_t e = gid / M;                       // entry over (series, tau, tick)
  int s = 0;
  while (s + 1 < b.n_series && (int64_t)b.ent_base[s + 1] * b.n_tau <= e) ++s;
  const int64_t local = e - (int64_t)b.ent_base[s] * b.n_tau;
  const int n_ent = b.ent_base[s + 1] - b.ent_base[s];
  const int ti = (int)(local / n_ent);
  const int j = (int)(local % n_ent);
  const int64_t win = b.series_win[s];
  const int64_t K = b.series_K[s];
  const int64_t nf = K * win / b.fast_ms;
  const bool fast = j < nf;
  const int64_t k =
      fast ? tick_window(j + 1, b.fast_ms, win) : tick_window(j - nf + 1, b.slow_ms, win);
  const T* Zk = b.Z + b.series_off[s] + (size_t)k * M;
  const uint8_t* Ck = b.cls + b.series_off[s] + (size_t)k * M;
  const bool tau_dev = b.tau_crit != nullptr;
  const T tau_v = b.tau_list[tau_dev ? 0 : ti];
  auto reg = [&](int q) {
    return region_of(Ck[q], Zk[q], tau_dev ? b.tau_crit[q] : tau_v, b.tau_surp[q]);
  };
  // receiver: rescue -> lowest Z among critical; rebalance -> lowest Z among non-idle
  int recv = -1;
  T zr = (T)0;
  for (int q = 0; q < M; ++q) {
    const uint8_t rg = reg(q);
    const bool cand = fast ? rg == kCrit : rg != kIdle;
    if (cand && (recv < 0 || Zk[q] < zr)) {
      recv = q;
      zr = Zk[q];
    }
  }
  const bool act = recv >= 0 && (fast || zr < (T)1);
  // donor group of model q, -1 = not a donor at this tick
  auto group = [&](int q, uint8_t rg) -> int {
    if (q == recv || rg == kCrit) return -1;
    if (rg == kIdle) return 0;
    if (rg == kSurp) return 1;
    if (!fast && !(Zk[q] > zr)) return -1;       // rebalance: nominal donors above the receiver
    return 2;
  };
  const int gm = act ? group(m, reg(m)) : -1;
  uint16_t r = kNoRank;
  if (gm >= 0) {
    const T zm = Zk[m];
    int before = 0;
    for (int q = 0; q < M; ++q) {
      if (q == m) continue;
      const int gq = group(q, reg(q));
      if (gq < 0) continue;
      bool prec;
      if (gq != gm) prec = gq < gm;
      else if (gq == 0) prec = q < m;
      else prec = Zk[q] > zm || (Zk[q] == zm && q < m);
      before += prec;
    }
    r = (uint16_t)before;
  }
  const size_t row = (size_t)b.ent_base[s] * b.n_tau + (size_t)ti * n_ent + j;
  rank[row * M + m] = r;
  if (m == 0) recv_out[row] = (int16_t)(act ? recv : -1);
}

template <int MPL>
__device__ __forceinline__ int lane_of_min_rank(const uint16_t (&rk)[MPL], const int (&r)[MPL],
                                                const int (&rmin)[MPL], int lane, int M,
                                                int& model) {
  uint32_t best = 0xffffffffu;
  int bj = 0;
#pragma unroll
  for (int j = 0; j < MPL; ++j) {
    const bool ok = lane + 32 * j < M && rk[j] != kNoRank && r[j] > rmin[j];
    if (ok && rk[j] < best) {
      best = rk[j];
      bj = j;
    }
  }
  const uint32_t wmin = __reduce_min_sync(0xffffffffu, best);
  if (wmin == 0xffffffffu) return -1;
  const unsigned who = __ballot_sync(0xffffffffu, best == wmin);
  const int src = __ffs(who) - 1;            // ranks are distinct within a tick
  model = src + 32 * __shfl_sync(0xffffffffu, bj, src);
  return src;
}

template <class T, int MPL>
__global__ void __launch_bounds__(kWarpsPerBlock * 32)
k_walk(const __grid_constant__ WalkBatch<T> b, const int16_t* recv_tab, const uint16_t* rank) {
  const int inst = blockIdx.x * kWarpsPerBlock + threadIdx.x / 32;
  if (inst >= b.n_inst) return;
  const int lane = threadIdx.x & 31;
  const int M = b.M;
  const int ci = inst % b.n_cap;
  const int ti = (inst / b.n_cap) % b.n_tau;
  const int si = inst / (b.n_cap * b.n_tau);
  const int K = b.series_K[si];
  const int64_t win = b.series_win[si];
  const int Kp = b.cap_list[ci];
  const int64_t cap = b.moves_cap;
  tre_move* mv = b.moves + (size_t)inst * cap;
  const int n_ent = b.ent_base[si + 1] - b.ent_base[si];
  const size_t row0 = (size_t)b.ent_base[si] * b.n_tau + (size_t)ti * n_ent;
  const int16_t* rv_tab = recv_tab + row0;
  const uint16_t* rk0 = rank + row0 * M;
  const int64_t F = b.fast_ms, Sl = b.slow_ms;
  const int64_t nf = (int64_t)K * win / F;

  int r[MPL], rmin[MPL], g[MPL];
  int64_t used = 0;
  bool bad = false;
#pragma unroll
  for (int j = 0; j < MPL; ++j) {
    const int m = lane + 32 * j;
    if (m < M) {
      r[j] = b.r0[m];
      rmin[j] = b.r_min[m];
      g[j] = b.footprint[m];
      used += (int64_t)g[j] * r[j];
      if (r[j] < 0 || g[j] < 1 || rmin[j] < 0) bad = true;
    } else {
      r[j] = 0; rmin[j] = 0; g[j] = 0;
    }
  }
  for (int o = 16; o > 0; o >>= 1) used += __shfl_xor_sync(0xffffffffu, used, o);
  int64_t free_pool = b.budget - used;
  // an inconsistent controller state (negative replicas or floors, footprint
  // below one, replicas beyond the budget) produces no moves
  if (__any_sync(0xffffffffu, bad) || free_pool < 0) {
#pragma unroll
    for (int j = 0; j < MPL; ++j)
      if (lane + 32 * j < M) b.r_out[(size_t)inst * M + lane + 32 * j] = r[j];
    if (lane == 0) {
      b.n_moves[inst] = 0;
      b.diag->err = TRE_EINVAL;
    }
    return;
  }
  int64_t nm = 0;
  int64_t jf = 1, js = 1;
  while (true) {
    const int64_t kf = tick_window(jf, F, win);
    const int64_t ks = tick_window(js, Sl, win);
    const int64_t k = kf < ks ? kf : ks;
    if (k >= K) break;
    const bool fast = kf == k, slow = ks == k;
    const int64_t ef = jf - 1, es = nf + js - 1;   // entries of this tick
    while (tick_window(jf, F, win) <= k) ++jf;
    while (tick_window(js, Sl, win) <= k) ++js;
    int recv = -1, kind = 0;
    int64_t ent = -1;
    if (fast) {
      const int rv = rv_tab[ef];
      if (rv >= 0) { recv = rv; ent = ef; kind = TRE_RESCUE; }
    }
    if (!kind && slow) {
      const int rv = rv_tab[es];
      if (rv >= 0) { recv = rv; ent = es; kind = TRE_REBALANCE; }
    }
    if (!kind) continue;
    uint16_t rk[MPL];
#pragma unroll
    for (int j = 0; j < MPL; ++j)
      rk[j] = lane + 32 * j < M ? rk0[(size_t)ent * M + lane + 32 * j] : kNoRank;
    int g_own = 0;
#pragma unroll
    for (int j = 0; j < MPL; ++j)
      if (lane + 32 * j == recv) g_own = g[j];
    const int need = __shfl_sync(0xffffffffu, g_own, recv & 31);
    for (int seq = 0; seq < Kp; ++seq) {
      if (free_pool >= need) {
        free_pool -= need;
#pragma unroll
        for (int j = 0; j < MPL; ++j)
          if (lane + 32 * j == recv) r[j] += 1;
        if (lane == 0 && nm < cap)
          mv[nm] = tre_move{(int32_t)k, (int16_t)recv, (int16_t)-1, (uint8_t)kind, (uint8_t)seq, 0};
        ++nm;
        continue;
      }
      // release donor replicas one at a time until the receiver's footprint
      // fits; an uncoverable transition releases nothing and ends the tick
      int rr[MPL];
#pragma unroll
      for (int j = 0; j < MPL; ++j) rr[j] = r[j];
      int64_t f = free_pool;
      const int64_t nm0 = nm;
      bool ok = true;
      while (f < need) {
        int d = -1;
        const int src = lane_of_min_rank<MPL>(rk, rr, rmin, lane, M, d);
        if (src < 0) { ok = false; break; }
        int gd = 0;
#pragma unroll
        for (int j = 0; j < MPL; ++j)
          if (lane + 32 * j == d) { rr[j] -= 1; gd = g[j]; }
        gd = __shfl_sync(0xffffffffu, gd, src);
        f += gd;
        if (lane == 0 && nm < cap)
          mv[nm] = tre_move{(int32_t)k, (int16_t)recv, (int16_t)d, (uint8_t)kind, (uint8_t)seq, 0};
        ++nm;
      }
      if (!ok) {
        nm = nm0;
        break;
      }
#pragma unroll
      for (int j = 0; j < MPL; ++j) {
        r[j] = rr[j];
        if (lane + 32 * j == recv) r[j] += 1;
      }
      free_pool = f - need;
    }
  }
#pragma unroll
  for (int j = 0; j < MPL; ++j) {
    const int m = lane + 32 * j;
    if (m < M) b.r_out[(size_t)inst * M + m] = r[j];
  }
  if (lane == 0) {
    b.n_moves[inst] = nm;
    if (nm > cap) b.diag->err = TRE_EOVERFLOW;
  }
}

}  // namespace

template <class T> void walk_ws_layout(Arena& a, WalkBatch<T>& b, WalkWs& w) {
  int64_t total = 0;
  for (int s = 0; s < b.n_series; ++s) {
    b.ent_base[s] = (int32_t)total;
    const int64_t span = (int64_t)b.series_K[s] * b.series_win[s];
    total += span / b.fast_ms + span / b.slow_ms;
  }
  b.ent_base[b.n_series] = (int32_t)total;
  w.recv = a.take<int16_t>((size_t)std::max<int64_t>(total * b.n_tau, 1));
  w.rank = a.take<uint16_t>((size_t)std::max<int64_t>(total * b.n_tau * b.M, 1));
}

template <class T> cudaError_t launch_walk(const WalkBatch<T>& b, WalkWs& w, cudaStream_t s) {
  if (b.n_inst == 0) return cudaSuccess;
  const int64_t ents = (int64_t)b.ent_base[b.n_series] * b.n_tau;
  if (ents > 0) {
    const int64_t th = ents * b.M;
    k_tick_rank<T><<<(unsigned)((th + 255) / 256), 256, 0, s>>>(b, w.recv, w.rank);
  }
  const unsigned grid = (unsigned)((b.n_inst + kWarpsPerBlock - 1) / kWarpsPerBlock);
  const int mpl = (b.M + 31) / 32;
  const unsigned th = kWarpsPerBlock * 32;
  if (mpl <= 1) k_walk<T, 1><<<grid, th, 0, s>>>(b, w.recv, w.rank);
  else if (mpl <= 2) k_walk<T, 2><<<grid, th, 0, s>>>(b, w.recv, w.rank);
  else if (mpl <= 4) k_walk<T, 4><<<grid, th, 0, s>>>(b, w.recv, w.rank);
  else if (mpl <= 8) k_walk<T, 8><<<grid, th, 0, s>>>(b, w.recv, w.rank);
  else if (mpl <= 16) k_walk<T, 16><<<grid, th, 0, s>>>(b, w.recv, w.rank);
  else k_walk<T, 32><<<grid, th, 0, s>>>(b, w.recv, w.rank);
  return cudaGetLastError();
}

template void walk_ws_layout<float>(Arena&, WalkBatch<float>&, WalkWs&);
template void walk_ws_layout<double>(Arena&, WalkBatch<double>&, WalkWs&);
template cudaError_t launch_walk<float>(const WalkBatch<float>&, WalkWs&, cudaStream_t);
template cudaError_t launch_walk<double>(const WalkBatch<double>&, WalkWs&, cudaStream_t);

}  // namespace tre
