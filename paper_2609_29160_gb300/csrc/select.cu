// Open-loop TRE move selection (Sec. IV-B dual-speed control, Eq. 3 receiver,
// Sec. IV-C bounded pairwise transfer under a fixed budget).
//
// One warp runs one controller instance serially over its control ticks; the
// models are spread over the lanes (models m = lane + 32*j, j < MPL) with their
// replica counts in registers. Receiver and donor choices are warp arg-min /
// arg-max reductions with the lowest model index winning ties. Only the windows
// that end a fast or slow tick are visited.
#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace tre {
namespace {

constexpr int kWarpsPerBlock = 4;

// candidate ordering: smaller `grp` first, then larger `z` (when by_z),
// then smaller index
template <class T> struct Cand {
  int grp;   // INT_MAX = none
  T z;
  int m;
};

template <class T> __device__ __forceinline__ bool better(const Cand<T>& a, const Cand<T>& b,
                                                          bool hi_z) {
  if (a.grp != b.grp) return a.grp < b.grp;
  if (a.grp == 0x7fffffff) return false;
  if (a.z != b.z) return hi_z ? (a.z > b.z) : (a.z < b.z);
  return a.m < b.m;
}

template <class T> __device__ __forceinline__ Cand<T> warp_best(Cand<T> c, bool hi_z) {
  for (int o = 16; o > 0; o >>= 1) {
    Cand<T> x;
    x.grp = __shfl_xor_sync(0xffffffffu, c.grp, o);
    x.z = __shfl_xor_sync(0xffffffffu, c.z, o);
    x.m = __shfl_xor_sync(0xffffffffu, c.m, o);
    if (better(x, c, hi_z)) c = x;
  }
  return c;
}

template <class T, int MPL>
__global__ void __launch_bounds__(kWarpsPerBlock * 32)
k_walk(const __grid_constant__ WalkBatch<T> b) {
  const int inst = blockIdx.x * kWarpsPerBlock + threadIdx.x / 32;
  if (inst >= b.n_inst) return;
  const int lane = threadIdx.x & 31;
  const int M = b.M;
  const int ci = inst % b.n_cap;
  const int ti = (inst / b.n_cap) % b.n_tau;
  const int si = inst / (b.n_cap * b.n_tau);
  const int64_t off = b.series_off[si];
  const int K = b.series_K[si];
  const int64_t win = b.series_win[si];
  const T* Zs = b.Z + off;
  const uint8_t* Cs = b.cls + off;
  const int Kp = b.cap_list[ci];
  const T tau_v = b.tau_crit ? (T)0 : b.tau_list[ti];
  const int64_t cap = b.moves_cap;
  tre_move* mv = b.moves + (size_t)inst * cap;

  int r[MPL], rmin[MPL], g[MPL];
  T tc[MPL], ts[MPL];
  int64_t used = 0;
#pragma unroll
  for (int j = 0; j < MPL; ++j) {
    const int m = lane + 32 * j;
    if (m < M) {
      r[j] = b.r0[m];
      rmin[j] = b.r_min[m];
      g[j] = b.footprint[m];
      tc[j] = b.tau_crit ? b.tau_crit[m] : tau_v;
      ts[j] = b.tau_surp[m];
      used += (int64_t)g[j] * r[j];
    } else {
      r[j] = 0; rmin[j] = 0; g[j] = 0; tc[j] = (T)0; ts[j] = (T)0;
    }
  }
  for (int o = 16; o > 0; o >>= 1) used += __shfl_xor_sync(0xffffffffu, used, o);
  int64_t free_pool = b.budget - used;
  int64_t nm = 0;
  bool bad = false;
#pragma unroll
  for (int j = 0; j < MPL; ++j)
    if (lane + 32 * j < M && (r[j] < 0 || g[j] < 1 || rmin[j] < 0)) bad = true;
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

  const int64_t F = b.fast_ms, Sl = b.slow_ms;
  int64_t jf = 1, js = 1;
  while (true) {
    // next window that ends a fast / slow tick: smallest k with (k+1)*win >= j*cadence
    const int64_t kf = (jf * F + win - 1) / win - 1;
    const int64_t ks = (js * Sl + win - 1) / win - 1;
    const int64_t k = kf < ks ? kf : ks;
    if (k >= K) break;
    const bool fast = kf == k, slow = ks == k;
    while ((jf * F + win - 1) / win - 1 <= k) ++jf;
    while ((js * Sl + win - 1) / win - 1 <= k) ++js;

    T z[MPL];
    uint8_t reg[MPL];
#pragma unroll
    for (int j = 0; j < MPL; ++j) {
      const int m = lane + 32 * j;
      if (m < M) {
        const size_t x = (size_t)k * M + m;
        z[j] = Zs[x];
        if (Cs[x] == kIdle) reg[j] = kIdle;
        else if (z[j] < tc[j]) reg[j] = kCrit;
        else if (z[j] > ts[j]) reg[j] = kSurp;
        else reg[j] = kNom;
      } else {
        z[j] = (T)0;
        reg[j] = 0xff;
      }
    }
    int kind = 0;
    Cand<T> rc{0x7fffffff, (T)0, 0};
    if (fast) {
#pragma unroll
      for (int j = 0; j < MPL; ++j) {
        const Cand<T> c{reg[j] == kCrit ? 0 : 0x7fffffff, z[j], lane + 32 * j};
        if (better(c, rc, false)) rc = c;
      }
      rc = warp_best(rc, false);
      if (rc.grp == 0) kind = TRE_RESCUE;
    }
    bool nom_above = false;
    if (!kind && slow) {
      rc = Cand<T>{0x7fffffff, (T)0, 0};
#pragma unroll
      for (int j = 0; j < MPL; ++j) {
        const bool ok = reg[j] != kIdle && reg[j] != 0xff;
        const Cand<T> c{ok ? 0 : 0x7fffffff, z[j], lane + 32 * j};
        if (better(c, rc, false)) rc = c;
      }
      rc = warp_best(rc, false);
      if (rc.grp == 0 && rc.z < (T)1) {
        kind = TRE_REBALANCE;
        nom_above = true;
      }
    }
    if (!kind) continue;
    const int recv = rc.m;
    const T zr = rc.z;
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
      int rr[MPL];
#pragma unroll
      for (int j = 0; j < MPL; ++j) rr[j] = r[j];
      int64_t f = free_pool;
      const int64_t nm0 = nm;
      bool ok = true;
      while (f < need) {
        Cand<T> dc{0x7fffffff, (T)0, 0};
#pragma unroll
        for (int j = 0; j < MPL; ++j) {
          const int m = lane + 32 * j;
          if (m == recv || reg[j] == kCrit || reg[j] == 0xff || rr[j] <= rmin[j]) continue;
          int grp;
          if (reg[j] == kIdle) grp = 0;
          else if (reg[j] == kSurp) grp = 1;
          else if (!nom_above || z[j] > zr) grp = 2;
          else continue;
          // idle donors go by index only
          const Cand<T> c{grp, grp == 0 ? (T)0 : z[j], m};
          if (better(c, dc, true)) dc = c;
        }
        dc = warp_best(dc, true);
        if (dc.grp == 0x7fffffff) { ok = false; break; }
        const int d = dc.m;
        int gd = 0;
#pragma unroll
        for (int j = 0; j < MPL; ++j)
          if (lane + 32 * j == d) { rr[j] -= 1; gd = g[j]; }
        gd = __shfl_sync(0xffffffffu, gd, d & 31);
        f += gd;
        if (lane == 0 && nm < cap)
          mv[nm] = tre_move{(int32_t)k, (int16_t)recv, (int16_t)d, (uint8_t)kind, (uint8_t)seq, 0};
        ++nm;
      }
      if (!ok) {
        nm = nm0;   // an uncoverable transition releases nothing
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

template <class T> cudaError_t launch_walk(const WalkBatch<T>& b, cudaStream_t s) {
  if (b.n_inst == 0) return cudaSuccess;
  const unsigned grid = (unsigned)((b.n_inst + kWarpsPerBlock - 1) / kWarpsPerBlock);
  const int mpl = (b.M + 31) / 32;
  const unsigned th = kWarpsPerBlock * 32;
  if (mpl <= 1) k_walk<T, 1><<<grid, th, 0, s>>>(b);
  else if (mpl <= 2) k_walk<T, 2><<<grid, th, 0, s>>>(b);
  else if (mpl <= 4) k_walk<T, 4><<<grid, th, 0, s>>>(b);
  else if (mpl <= 8) k_walk<T, 8><<<grid, th, 0, s>>>(b);
  else if (mpl <= 16) k_walk<T, 16><<<grid, th, 0, s>>>(b);
  else k_walk<T, 32><<<grid, th, 0, s>>>(b);
  return cudaGetLastError();
}

template cudaError_t launch_walk<float>(const WalkBatch<float>&, cudaStream_t);
template cudaError_t launch_walk<double>(const WalkBatch<double>&, cudaStream_t);

}  // namespace tre
