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
#include <cstddef>

#include "common.cuh"
#include "internal.h"

namespace tre {
namespace {

constexpr uint16_t kNoRank = 0xffff;

__device__ __forceinline__ int64_t tick_window(int64_t j, int64_t cadence, int64_t win) {
  // window whose right edge passes the j-th multiple of the cadence (j >= 1)
  return (j * cadence + win - 1) / win - 1;
}

// successive multiples j*c of a cadence c as quotient and remainder of win
struct TickSeq {
  int32_t q, r, qc, rc, win;
  __device__ __forceinline__ TickSeq(int32_t c, int32_t w) : win(w) {
    qc = c / w;
    rc = c - qc * w;
    q = qc;
    r = rc;
  }
  // window whose right edge passes the current multiple (windows end before 2^31 ms)
  __device__ __forceinline__ int32_t window() const { return q + (r > 0) - 1; }
  __device__ __forceinline__ void next() {
    q += qc;
    r += rc;
    if (r >= win) { r -= win; q += 1; }
  }
};

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
k_tick_rank(const __grid_constant__ WalkBatch<T> b, int16_t* recv_out, int16_t* ndon_out,
            uint16_t* rank, uint16_t* order, unsigned long long* dm64) {
  const int M = b.M;
  const int64_t gid = (int64_t)blockIdx.x * 256 + threadIdx.x;
  const int64_t total_ent = (int64_t)b.ent_base[b.n_series] * b.n_tau;
  if (gid >= total_ent * M) return;
  const int m = (int)(gid % M);
  const int64_t e = gid / M;                       // entry over (series, tau, tick)
  const int s = prefix_index(b.ent_base, b.n_series, e, b.n_tau);
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
  if (r != kNoRank) order[row * M + r] = (uint16_t)m;
  if (m == 0) {
    int nd = 0;
    unsigned long long dm = 0;
    if (act)
      for (int q = 0; q < M; ++q)
        if (group(q, reg(q)) >= 0) {
          ++nd;
          if (q < 64) dm |= 1ull << q;
        }
    recv_out[row] = (int16_t)(act ? recv : -1);
    ndon_out[row] = (int16_t)nd;
    if (dm64) dm64[row] = dm;                      // models that are donors at the tick
  }
}

__device__ __forceinline__ void load_quad(const float* p, float* v) {
  const float4 q = *reinterpret_cast<const float4*>(p);
  v[0] = q.x; v[1] = q.y; v[2] = q.z; v[3] = q.w;
}
__device__ __forceinline__ void load_quad(const double* p, double* v) {
  const double2 a = reinterpret_cast<const double2*>(p)[0];
  const double2 c = reinterpret_cast<const double2*>(p)[1];
  v[0] = a.x; v[1] = a.y; v[2] = c.x; v[3] = c.y;
}

// The action of one control tick of (series s, tau ti) at window k, for
// M <= MMAX: regions from the window's Z and class rows; the receiver (rescue:
// lowest Z among critical models; rebalance: lowest Z among non-idle models,
// acting only below Z = 1; lowest index on ties; -1 when the tick does
// nothing); each model's rank in the donor order (kNoRank when not a donor),
// the donor order packed four bits a position (M <= 16), the donor mask and
// the donor count. With QUAD (M a multiple of 4, 16-byte aligned rows) the
// rows are read four models per load.
template <class T, int MMAX, bool QUAD>
struct TickAction {
  int recv, nd;
  unsigned long long pk, dmw;
  uint32_t dm;
  uint16_t rk[MMAX];
};

template <class T, int MMAX, bool QUAD>
__device__ __forceinline__ void tick_row(const WalkBatch<T>& b, int s, uint32_t k, T (&z)[MMAX],
                                         uint8_t (&cl)[MMAX]) {
  const int M = b.M;
  const T* Zk = b.Z + b.series_off[s] + (size_t)k * M;
  const uint8_t* Ck = b.cls + b.series_off[s] + (size_t)k * M;
#pragma unroll
  for (int q = 0; q < MMAX; ++q) {
    z[q] = (T)0;
    cl[q] = kIdle;
  }
  if (QUAD) {
#pragma unroll
    for (int q = 0; q < MMAX; q += 4) {
      if (q < M) {
        load_quad(Zk + q, z + q);
        const uchar4 c4 = *reinterpret_cast<const uchar4*>(Ck + q);
        cl[q] = c4.x; cl[q + 1] = c4.y; cl[q + 2] = c4.z; cl[q + 3] = c4.w;
      }
    }
  } else {
#pragma unroll
    for (int q = 0; q < MMAX; ++q)
      if (q < M) {
        z[q] = Zk[q];
        cl[q] = Ck[q];
      }
  }
}

template <class T, int MMAX, bool QUAD>
__device__ __forceinline__ void tick_action(const WalkBatch<T>& b, int ti, bool fast,
                                            const T (&z)[MMAX], const uint8_t (&cl)[MMAX],
                                            TickAction<T, MMAX, QUAD>& out) {
  const int M = b.M;
  const bool tau_dev = b.tau_crit != nullptr;
  const T tau_v = b.tau_list[tau_dev ? 0 : ti];
  uint8_t rg[MMAX];
  int recv = -1;
  T zr = (T)0;
#pragma unroll
  for (int q = 0; q < MMAX; ++q) {
    rg[q] = 0xff;
    if (q < M) {
      rg[q] = region_of(cl[q], z[q], tau_dev ? b.tau_crit[q] : tau_v, b.tau_surp[q]);
      const bool cand = fast ? rg[q] == kCrit : rg[q] != kIdle;
      if (cand && (recv < 0 || z[q] < zr)) {
        recv = q;
        zr = z[q];
      }
    }
  }
  const bool act = recv >= 0 && (fast || zr < (T)1);
  int grp[MMAX];
  int nd = 0;
#pragma unroll
  for (int q = 0; q < MMAX; ++q) {
    int g = -1;
    if (act && q < M && q != recv && rg[q] != kCrit) {
      if (rg[q] == kIdle) g = 0;
      else if (rg[q] == kSurp) g = 1;
      else if (fast || z[q] > zr) g = 2;       // rebalance: nominal donors above the receiver
    }
    grp[q] = g;
    nd += g >= 0;
  }
  unsigned long long pk = 0, dmw = 0;
  uint32_t dm = 0;
#pragma unroll
  for (int m = 0; m < MMAX; ++m) {
    uint16_t r = kNoRank;
    if (m < M && grp[m] >= 0) {
      int before = 0;
#pragma unroll
      for (int q = 0; q < MMAX; ++q) {
        if (q >= M || q == m || grp[q] < 0) continue;
        bool prec;
        if (grp[q] != grp[m]) prec = grp[q] < grp[m];
        else if (grp[q] == 0) prec = q < m;
        else prec = z[q] > z[m] || (z[q] == z[m] && q < m);
        before += prec;
      }
      r = (uint16_t)before;
      dmw |= 1ull << m;
      if (MMAX <= 16) {
        pk |= (unsigned long long)m << (4 * before);
        dm |= 1u << m;
      }
    }
    out.rk[m] = r;
  }
  out.recv = act ? recv : -1;
  out.nd = nd;
  out.pk = pk;
  out.dm = dm;
  out.dmw = dmw;
}

// One thread per (series, tau, tick entry) for M <= MMAX: the regions are
// computed once per model and the ranks in registers; the per-model rank and
// order tables are written only when the walk that follows reads them.
template <class T, int MMAX, bool QUAD>
__global__ void __launch_bounds__(128)
k_tick_rank_small(const __grid_constant__ WalkBatch<T> b, int16_t* recv_out, int16_t* ndon_out,
                  uint16_t* rank, uint16_t* order, unsigned long long* packed, uint32_t* dmask,
                  bool need_rank, unsigned long long* dm64) {
  const int M = b.M;
  const int64_t e = (int64_t)blockIdx.x * 128 + threadIdx.x;
  if (e >= (int64_t)b.ent_base[b.n_series] * b.n_tau) return;
  const int s = prefix_index(b.ent_base, b.n_series, e, b.n_tau);
  const int local = (int)(e - (int64_t)b.ent_base[s] * b.n_tau);
  const int n_ent = b.ent_base[s + 1] - b.ent_base[s];
  const int ti = local / n_ent;
  const int j = local - ti * n_ent;
  // K * win < 2^31, so every tick time below fits 32 unsigned bits
  const uint32_t win = (uint32_t)b.series_win[s];
  const uint32_t nf = (uint32_t)b.series_K[s] * win / (uint32_t)b.fast_ms;
  const bool fast = (uint32_t)j < nf;
  const uint32_t tj = fast ? ((uint32_t)j + 1) * (uint32_t)b.fast_ms
                           : ((uint32_t)j - nf + 1) * (uint32_t)b.slow_ms;
  const uint32_t k = (tj + win - 1) / win - 1;   // window whose right edge passes tj
  T z[MMAX];
  uint8_t cl[MMAX];
  tick_row<T, MMAX, QUAD>(b, s, k, z, cl);
  TickAction<T, MMAX, QUAD> a;
  tick_action<T, MMAX, QUAD>(b, ti, fast, z, cl, a);
  const size_t row = (size_t)b.ent_base[s] * b.n_tau + (size_t)ti * n_ent + j;
  if (need_rank) {
#pragma unroll
    for (int m = 0; m < MMAX; ++m) {
      if (m >= M) break;
      rank[row * M + m] = a.rk[m];
      if (a.rk[m] != kNoRank) order[row * M + a.rk[m]] = (uint16_t)m;
    }
    dm64[row] = a.dmw;                             // for the warp walk
  }
  recv_out[row] = (int16_t)a.recv;
  ndon_out[row] = (int16_t)a.nd;
  if (MMAX <= 16) {
    packed[row] = a.pk;
    dmask[row] = a.dm;
  }
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

// One CTA per (series, tau) and group of up to kCapWarps pacing caps, one warp
// per cap: the warps share the tick tables of their (series, tau), staged in
// shared memory when they fit. (Eight warps a CTA leave each thread the
// registers the walk's state needs.)
constexpr int kCapWarps = 8;
template <class T, int MPL, bool STAGED>
__global__ void __launch_bounds__(kCapWarps * 32)
k_walk(const __grid_constant__ WalkBatch<T> b, const int16_t* recv_tab, const int16_t* ndon_tab,
       const uint16_t* rank, const uint16_t* order, const unsigned long long* dm64) {
  extern __shared__ __align__(16) unsigned char dyn[];
  const int grp = blockIdx.x;                       // (series, tau)
  const int ti = grp % b.n_tau;
  const int si = grp / b.n_tau;
  const int ci = blockIdx.y * kCapWarps + threadIdx.x / 32;   // pacing cap index
  const int lane = threadIdx.x & 31;
  const int M = b.M;
  const int K = b.series_K[si];
  const int64_t win = b.series_win[si];
  const int n_ent = b.ent_base[si + 1] - b.ent_base[si];
  const size_t row0 = (size_t)b.ent_base[si] * b.n_tau + (size_t)ti * n_ent;
  const int16_t* rv_tab = recv_tab + row0;
  const int16_t* nd_tab = ndon_tab + row0;
  const unsigned long long* dm_tab = dm64 + row0;
  const uint16_t* rk0 = rank + row0 * M;
  const uint16_t* od0 = order + row0 * M;
  if (STAGED) {
    const size_t a2 = ((size_t)n_ent * 2 + 15) & ~(size_t)15;
    const size_t am = ((size_t)n_ent * M * 2 + 15) & ~(size_t)15;
    int16_t* srv = reinterpret_cast<int16_t*>(dyn);
    int16_t* snd = reinterpret_cast<int16_t*>(dyn + a2);
    uint16_t* srk = reinterpret_cast<uint16_t*>(dyn + 2 * a2);
    uint16_t* sod = reinterpret_cast<uint16_t*>(dyn + 2 * a2 + am);
    for (int i = threadIdx.x; i < n_ent; i += blockDim.x) {
      srv[i] = rv_tab[i];
      snd[i] = nd_tab[i];
    }
    for (int64_t i = threadIdx.x; i < (int64_t)n_ent * M; i += blockDim.x) {
      srk[i] = rk0[i];
      sod[i] = od0[i];
    }
    __syncthreads();
    rv_tab = srv;
    nd_tab = snd;
    rk0 = srk;
    od0 = sod;
  }
  if (ci >= b.n_cap) return;
  const int inst = (si * b.n_tau + ti) * b.n_cap + ci;
  const int Kp = b.cap_list[ci];
  const int64_t cap = b.moves_cap;
  tre_move* mv = b.moves + (size_t)inst * cap;
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
  // With unit footprints and one model per lane a tick is closed form: pool
  // draws first, then donors drain in rank order down to their floors.
  bool unit = true;
#pragma unroll
  for (int j = 0; j < MPL; ++j)
    if (lane + 32 * j < M && g[j] != 1) unit = false;
  const bool closed = MPL == 1 && __all_sync(0xffffffffu, unit);
  // tick windows without division: the j-th tick of a cadence c ends window
  // ceil(j*c / win) - 1; keep j*c as quotient and remainder of win
  TickSeq sf((int32_t)F, (int32_t)win), ss((int32_t)Sl, (int32_t)win);
  int32_t jf = 1, js = 1;
  // the receivers of the coming 32 fast and 32 slow ticks, one per lane: most
  // ticks move nothing, and a tick then costs a shuffle instead of a load
  int32_t fb0 = -64, sb0 = -64;                 // entries >= 0: the first access loads
  int fbuf = -1, sbuf = -1;
  auto rv_at = [&](int32_t e, int32_t& b0, int& buf) {
    if ((uint32_t)(e - b0) >= 32u) {
      b0 = e;
      buf = e + lane < n_ent ? rv_tab[e + lane] : -1;
    }
    return __shfl_sync(0xffffffffu, buf, e - b0);
  };
  // the donor sets of the same ticks (models with a rank), for up to 64
  // models: a tick whose receiver the pool cannot serve and whose donors all
  // sit at their floors moves nothing, and costs no row load
  int32_t fm0 = -64, sm0 = -64;
  unsigned long long fmb = 0, smb = 0;
  auto dm_at = [&](int32_t e, int32_t& b0, unsigned long long& buf) {
    if ((uint32_t)(e - b0) >= 32u) {
      b0 = e;
      buf = e + lane < n_ent ? dm_tab[e + lane] : 0ull;
    }
    return __shfl_sync(0xffffffffu, buf, e - b0);
  };
  // the transitions of one tick: window k, receiver recv, table entry ent
  auto act = [&](int32_t k, int recv, int kind, int32_t ent) {
    if (closed) {
      const int nd = nd_tab[ent];
      const int mo = lane < nd ? od0[(size_t)ent * M + lane] : -1;
      const int r_src = __shfl_sync(0xffffffffu, r[0] - rmin[0], mo < 0 ? 0 : mo);
      const int cap_p = mo < 0 ? 0 : (r_src > 0 ? r_src : 0);
      int incl = cap_p;
      for (int o = 1; o < 32; o <<= 1) {
        const int x = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += x;
      }
      const int excl = incl - cap_p;
      const int total_cap = __shfl_sync(0xffffffffu, incl, 31);
      const int n_pool = (int)(free_pool < Kp ? free_pool : Kp);
      const int t_d = min(Kp - n_pool, total_cap);
      const int give = max(0, min(t_d - excl, cap_p));
      // moves: pool draws take seq 0.., donors follow in rank order
      for (int q = lane; q < n_pool; q += 32)
        if (nm + q < cap)
          mv[nm + q] = tre_move{(int32_t)k, (int16_t)recv, (int16_t)-1, (uint8_t)kind,
                                (uint8_t)q, 0};
      for (int i = 0; i < give; ++i) {
        const int64_t q = n_pool + excl + i;
        if (nm + q < cap)
          mv[nm + q] = tre_move{(int32_t)k, (int16_t)recv, (int16_t)mo, (uint8_t)kind,
                                (uint8_t)q, 0};
      }
      // my model's position in the donor order, then what it gave
      const uint16_t my_rank = lane < M ? rk0[(size_t)ent * M + lane] : kNoRank;
      const int given = __shfl_sync(0xffffffffu, give, my_rank == kNoRank ? 0 : (my_rank & 31));
      if (my_rank != kNoRank) r[0] -= given;
      if (lane == recv) r[0] += n_pool + t_d;
      free_pool -= n_pool;
      nm += n_pool + t_d;
      return;
    }
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
  };
  // Nested cadences (the slow tick a multiple of the fast one, the fast tick
  // at least a window): the ticks are the fast ticks u = 0 .. nf-1, and fast
  // tick u also carries slow tick (u+1)/ratio when ratio divides u+1. The
  // replica state only changes where a tick moves something, so 32 ticks are
  // tested at once against the current state (a receiver, and either room in
  // the pool for its footprint or a donor above its floor) and the walk jumps
  // to the first that can act.
  if (MPL <= 2 && F >= win && Sl % F == 0) {
    const int64_t ratio = Sl / F;
    // tick windows by multiply-high division (tick times stay below 2^31 ms)
    const FastDiv fwin((uint32_t)win);
    // the table entries of 32 consecutive fast ticks, one per lane: receivers
    // and donor masks of the tick and of the slow tick it carries
    struct Ent {
      int rf, rs;
      unsigned long long df, ds;
    };
    // entry of the slow tick carried by fast tick u
    auto slow_ent = [&](int64_t u) { return (int32_t)(nf + (u + 1) / ratio - 1); };
    auto load = [&](int64_t base, Ent& e) {
      const int64_t u = base + lane;
      const int32_t es = slow_ent(u);
      const bool in = u < nf;
      const bool has_slow = in && (u + 1) % ratio == 0 && es < n_ent;
      e.rf = in ? rv_tab[u] : -1;
      e.df = in ? dm_tab[u] : 0ull;
      e.rs = has_slow ? rv_tab[es] : -1;
      e.ds = has_slow ? dm_tab[es] : 0ull;
    };
    // the next group's entries are loaded while the current group is tested
    // and acted on; after a tick acts, the rest of its group is tested again
    // against the new state without loading anything
    Ent cur, nxt;
    int64_t base = 0;
    int start = 0;   // lanes of the current group before it are done
    load(0, cur);
    load(32, nxt);
    while (base < nf) {
      unsigned long long above = 0;
#pragma unroll
      for (int j = 0; j < MPL; ++j)
        above |= (unsigned long long)__ballot_sync(0xffffffffu, lane + 32 * j < M && r[j] > rmin[j])
                 << (32 * j);
      int rv = -1, kind = 0;
      int32_t ent = -1;
      unsigned long long dn = 0;
      if (cur.rf >= 0) {
        rv = cur.rf; kind = TRE_RESCUE; ent = (int32_t)(base + lane); dn = cur.df;
      } else if (cur.rs >= 0) {
        rv = cur.rs; kind = TRE_REBALANCE; ent = slow_ent(base + lane); dn = cur.ds;
      }
      // the receiver's footprint sits in lane rv % 32, slot rv / 32
      int g_rv = 0;
#pragma unroll
      for (int j = 0; j < MPL; ++j) {
        const int x = __shfl_sync(0xffffffffu, g[j], rv & 31);
        if (rv >= 0 && (rv >> 5) == j) g_rv = x;
      }
      const bool can = lane >= start && rv >= 0 && (free_pool >= g_rv || (dn & above) != 0);
      const unsigned hit = __ballot_sync(0xffffffffu, can);
      int next_start = 32;
      if (hit) {
        const int src = __ffs(hit) - 1;
        const int32_t e_t = __shfl_sync(0xffffffffu, ent, src);
        const int rv_t = __shfl_sync(0xffffffffu, rv, src);
        const int kd_t = __shfl_sync(0xffffffffu, kind, src);
        act((int32_t)fwin.div((uint32_t)(base + src + 1) * (uint32_t)F + (uint32_t)win - 1u) - 1,
            rv_t, kd_t, e_t);
        next_start = src + 1;
      }
      if (next_start < 32) {
        start = next_start;
      } else {
        base += 32;
        cur = nxt;
        load(base + 32, nxt);
        start = 0;
      }
    }
  } else {
    while (true) {
      const int32_t kf = sf.window(), ks = ss.window();
      const int32_t k = kf < ks ? kf : ks;
      if (k >= K) break;
      const bool fast = kf == k, slow = ks == k;
      const int32_t ef = jf - 1, es = (int32_t)nf + js - 1;   // entries of this tick
      while (sf.window() <= k) { sf.next(); ++jf; }
      while (ss.window() <= k) { ss.next(); ++js; }
      int recv = -1, kind = 0;
      int32_t ent = -1;
      if (fast) {
        const int rv = rv_at(ef, fb0, fbuf);
        if (rv >= 0) { recv = rv; ent = ef; kind = TRE_RESCUE; }
      }
      if (!kind && slow) {
        const int rv = rv_at(es, sb0, sbuf);
        if (rv >= 0) { recv = rv; ent = es; kind = TRE_REBALANCE; }
      }
      if (!kind) continue;
      if (MPL <= 2) {
        const unsigned long long donors =
            ent < (int32_t)nf ? dm_at(ent, fm0, fmb) : dm_at(ent, sm0, smb);
        unsigned long long above = 0;
#pragma unroll
        for (int j = 0; j < MPL; ++j)
          above |= (unsigned long long)__ballot_sync(0xffffffffu, lane + 32 * j < M && r[j] > rmin[j])
                   << (32 * j);
        int g_rv = 0;
#pragma unroll
        for (int j = 0; j < MPL; ++j)
          if (lane + 32 * j == recv) g_rv = g[j];
        const int need_rv = __shfl_sync(0xffffffffu, g_rv, recv & 31);
        if (free_pool < need_rv && !(donors & above)) continue;
      }
      act(k, recv, kind, ent);
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

// One thread per controller instance (M <= 16): the threads of a CTA are the
// pacing caps of one (series, tau) and share its staged tick tables. A
// transition draws on the idle pool if it covers the receiver's footprint,
// else releases donor replicas in the tick's donor order (lowest rank first,
// each down to its floor). The models still above their floors are a bit
// mask in a register, so a tick whose donors are all at their floors costs one
// AND; the donor order is a packed 4-bit list per tick.
template <class T, int MMAX>
__device__ __forceinline__ int sel(const int (&a)[MMAX], int m) {
  int v = 0;
#pragma unroll
  for (int q = 0; q < MMAX; ++q) v = q == m ? a[q] : v;
  return v;
}
template <class T, int MMAX>
__device__ __forceinline__ void add_at(int (&a)[MMAX], int m, int d) {
#pragma unroll
  for (int q = 0; q < MMAX; ++q) a[q] += q == m ? d : 0;
}

template <class T, int MMAX>
__global__ void __launch_bounds__(32)
k_walk_thread(const __grid_constant__ WalkBatch<T> b, const int16_t* recv_tab,
              const unsigned long long* packed, const uint32_t* dmask) {
  extern __shared__ __align__(16) unsigned char dyn[];
  const int grp = blockIdx.x;
  const int ti = grp % b.n_tau;
  const int si = grp / b.n_tau;
  const int M = b.M;
  const int K = b.series_K[si];
  const int32_t win = b.series_win[si];
  const int n_ent = b.ent_base[si + 1] - b.ent_base[si];
  const size_t row0 = (size_t)b.ent_base[si] * b.n_tau + (size_t)ti * n_ent;
  unsigned long long* spk = reinterpret_cast<unsigned long long*>(dyn);
  uint32_t* sdm = reinterpret_cast<uint32_t*>(spk + n_ent);
  int16_t* srv = reinterpret_cast<int16_t*>(sdm + n_ent);
  for (int i = threadIdx.x; i < n_ent; i += blockDim.x) {
    spk[i] = packed[row0 + i];
    sdm[i] = dmask[row0 + i];
    srv[i] = recv_tab[row0 + i];
  }
  __syncthreads();
  const int ci = threadIdx.x;
  if (ci >= b.n_cap) return;
  const int inst = (si * b.n_tau + ti) * b.n_cap + ci;
  const int Kp = b.cap_list[ci];
  const int64_t cap = b.moves_cap;
  tre_move* mv = b.moves + (size_t)inst * cap;
  const int32_t nf = (int32_t)((int64_t)K * win / b.fast_ms);
  int r[MMAX], rmin[MMAX], g[MMAX];
  int64_t used = 0;
  bool bad = false, unit = true;
  uint32_t avail = 0;                           // models above their floor
#pragma unroll
  for (int m = 0; m < MMAX; ++m) {
    r[m] = 0;
    rmin[m] = 0;
    g[m] = 1;
    if (m < M) {
      r[m] = b.r0[m];
      rmin[m] = b.r_min[m];
      g[m] = b.footprint[m];
      used += (int64_t)g[m] * r[m];
      if (r[m] < 0 || rmin[m] < 0 || g[m] < 1) bad = true;
      if (g[m] != 1) unit = false;
      if (r[m] > rmin[m]) avail |= 1u << m;
    }
  }
  int64_t free_pool = b.budget - used;
  if (bad || free_pool < 0) {
    for (int m = 0; m < M && m < MMAX; ++m) b.r_out[(size_t)inst * M + m] = sel<T, MMAX>(r, m);
    b.n_moves[inst] = 0;
    b.diag->err = TRE_EINVAL;
    return;
  }
  auto emit = [&](int64_t at, int32_t k, int recv, int donor, int kind, int sq) {
    if (at < cap) mv[at] = tre_move{k, (int16_t)recv, (int16_t)donor, (uint8_t)kind, (uint8_t)sq, 0};
  };
  int64_t nm = 0;
  TickSeq sf(b.fast_ms, win), ss(b.slow_ms, win);
  int32_t jf = 1, js = 1;
  while (true) {
    const int32_t kf = sf.window(), ks = ss.window();
    const int32_t k = kf < ks ? kf : ks;
    if (k >= K) break;
    const bool fast = kf == k, slow = ks == k;
    const int32_t ef = jf - 1, es = nf + js - 1;
    while (sf.window() <= k) { sf.next(); ++jf; }
    while (ss.window() <= k) { ss.next(); ++js; }
    int recv = -1, kind = 0;
    int32_t ent = -1;
    if (fast) {
      const int rv = srv[ef];
      if (rv >= 0) { recv = rv; ent = ef; kind = TRE_RESCUE; }
    }
    if (!kind && slow) {
      const int rv = srv[es];
      if (rv >= 0) { recv = rv; ent = es; kind = TRE_REBALANCE; }
    }
    if (!kind) continue;
    const uint32_t usable = avail & sdm[ent];
    const int need = unit ? 1 : sel<T, MMAX>(g, recv);
    if (free_pool < need && !usable) continue;        // nothing can move this tick
    unsigned long long pk = spk[ent];
    if (unit) {
      const int n_pool = (int)(free_pool < Kp ? free_pool : Kp);
      for (int q = 0; q < n_pool; ++q) emit(nm + q, k, recv, -1, kind, q);
      int sq = n_pool;
      uint32_t left = usable;
      while (sq < Kp && left) {
        int m = (int)(pk & 15);                      // next model in donor order
        pk >>= 4;
        if (!(left >> m & 1)) continue;
        left &= ~(1u << m);
        const int c = sel<T, MMAX>(r, m) - sel<T, MMAX>(rmin, m);
        const int take = min(c, Kp - sq);
        add_at<T, MMAX>(r, m, -take);
        if (take == c) avail &= ~(1u << m);
        for (int i = 0; i < take; ++i, ++sq) emit(nm + sq, k, recv, m, kind, sq);
      }
      add_at<T, MMAX>(r, recv, sq);
      if (sel<T, MMAX>(r, recv) > sel<T, MMAX>(rmin, recv)) avail |= 1u << recv;
      free_pool -= n_pool;
      nm += sq;
      continue;
    }
    for (int sq = 0; sq < Kp; ++sq) {
      if (free_pool >= need) {
        free_pool -= need;
        add_at<T, MMAX>(r, recv, 1);
        if (sel<T, MMAX>(r, recv) > sel<T, MMAX>(rmin, recv)) avail |= 1u << recv;
        emit(nm++, k, recv, -1, kind, sq);
        continue;
      }
      // plan the releases; an uncoverable transition releases nothing
      int64_t f = free_pool;
      const int64_t nm0 = nm;
      int taken[MMAX];
#pragma unroll
      for (int m = 0; m < MMAX; ++m) taken[m] = 0;
      unsigned long long order = pk;
      uint32_t left = avail & sdm[ent];
      while (f < need && left) {
        const int m = (int)(order & 15);
        order >>= 4;
        if (!(left >> m & 1)) continue;
        left &= ~(1u << m);
        int c = sel<T, MMAX>(r, m) - sel<T, MMAX>(rmin, m);
        const int gm = sel<T, MMAX>(g, m);
        while (f < need && c > 0) {
          add_at<T, MMAX>(taken, m, 1);
          --c;
          f += gm;
          emit(nm++, k, recv, m, kind, sq);
        }
      }
      if (f < need) {
        nm = nm0;
        break;
      }
#pragma unroll
      for (int m = 0; m < MMAX; ++m) {
        r[m] -= taken[m];
        if (m < M && !(r[m] > rmin[m])) avail &= ~(1u << m);
      }
      add_at<T, MMAX>(r, recv, 1);
      if (sel<T, MMAX>(r, recv) > sel<T, MMAX>(rmin, recv)) avail |= 1u << recv;
      free_pool = f - need;
    }
  }
  for (int m = 0; m < M && m < MMAX; ++m) b.r_out[(size_t)inst * M + m] = sel<T, MMAX>(r, m);
  b.n_moves[inst] = nm;
  if (nm > cap) b.diag->err = TRE_EOVERFLOW;
}

// Jumping walk for nested cadences (slow_ms a multiple of fast_ms, so every
// slow tick is a fast tick): the action of each tick (rescue entry, else
// rebalance entry, else none) does not depend on the replica state, and the
// state changes only when something moves. A tick can move something only if
// the idle pool is non-empty or a model above its floor is a donor there; per
// model, the next tick where it is a donor is precomputed, so the walk jumps
// from one possible move to the next instead of visiting every tick.
// Smallest of a tick row's next-donor ticks over the models in `avail`: the
// row holds MMAX 16-bit entries; models outside the mask are lifted to 0xffff
// and the row is reduced with per-halfword minima.
template <int MMAX>
__device__ __forceinline__ int next_donor_tick(const uint16_t* row, uint32_t avail) {
  const uint4* q = reinterpret_cast<const uint4*>(row);
  uint32_t acc = 0xffffffffu;
#pragma unroll
  for (int h = 0; h < MMAX / 8; ++h) {
    const uint4 w = q[h];
    const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int m = h * 8 + 2 * i;
      const uint32_t lift = ((avail >> m) & 1u ? 0u : 0xffffu) |
                            ((avail >> (m + 1)) & 1u ? 0u : 0xffff0000u);
      acc = __vminu2(acc, ws[i] | lift);
    }
  }
  return (int)min(acc & 0xffffu, acc >> 16);
}

// One move record, written as three 32-bit words (window; receiver and donor;
// kind and position in the tick) when it fits the caller's list.
static_assert(sizeof(tre_move) == 12 && offsetof(tre_move, recv) == 4 &&
                  offsetof(tre_move, donor) == 6 && offsetof(tre_move, kind) == 8 &&
                  offsetof(tre_move, seq) == 9 && offsetof(tre_move, reserved) == 10,
              "tre_move layout");
__device__ __forceinline__ void put_move(tre_move* mv, int64_t at, int64_t cap, int32_t k,
                                         int recv, int donor, int kind, int sq) {
  if (at < cap) {
    uint32_t* p = reinterpret_cast<uint32_t*>(mv + at);
    p[0] = (uint32_t)k;
    p[1] = (uint32_t)(uint16_t)recv | ((uint32_t)(uint16_t)donor << 16);
    p[2] = (uint32_t)(uint8_t)kind | ((uint32_t)(uint8_t)sq << 8);
  }
}

// One tick's action as the walk reads it: donor order (4 bits a position),
// donor mask, receiver (-1: nothing acts) and kind, in one 16-byte load.
struct __align__(16) TickRec {
  unsigned long long pk;
  uint32_t dm;
  int16_t recv;
  uint8_t kind, pad;
};

// RANK: the CTA of a (series, tau) finds its ticks' actions itself from the Z
// and class rows (tick_action) while it builds the tables -- one launch, for
// batches with a CTA per SM or more; otherwise it reads them from the tick
// tables k_tick_rank_small wrote (the ranking then spreads over many CTAs).
template <class T, int MMAX, bool RANK, bool QUAD>
__global__ void __launch_bounds__(256, 1)
k_walk_jump(const __grid_constant__ WalkBatch<T> b, const int16_t* recv_tab,
            const unsigned long long* packed, const uint32_t* dmask, bool store_win) {
  extern __shared__ __align__(16) unsigned char dyn[];
  const int grp = blockIdx.x;
  const int ti = grp % b.n_tau;
  const int si = grp / b.n_tau;
  const int M = b.M;
  const int K = b.series_K[si];
  const int64_t win = b.series_win[si];
  const int n_ent = b.ent_base[si + 1] - b.ent_base[si];
  const size_t row0 = (size_t)b.ent_base[si] * b.n_tau + (size_t)ti * n_ent;
  const int nf = (int)((int64_t)K * win / b.fast_ms);   // fast ticks = all ticks
  const int ratio = b.slow_ms / b.fast_ms;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, n_warps = blockDim.x >> 5;
  // shared layout: per tick u < nf: action record and window; per tick
  // u <= nf: for every model the next tick >= u where it is a donor (one
  // 2*MMAX-byte row per tick, so a row is read with 16-byte loads), and the
  // next tick >= u where anything acts
  // (the window of each tick is staged when there is room, else recomputed
  // at each visit)
  TickRec* srec = reinterpret_cast<TickRec*>(dyn);
  int32_t* swin = reinterpret_cast<int32_t*>(srec + nf);
  uint16_t* snx = store_win ? reinterpret_cast<uint16_t*>(swin + ((nf + 3) & ~3))
                            : reinterpret_cast<uint16_t*>(swin);           // [nf + 1][MMAX]
  // window of fast tick u, ceil((u + 1) * fast / win) - 1, without a divide
  // instruction (the tick times stay below 2^31 ms)
  const FastDiv fwin((uint32_t)win);
  auto tick_of = [&](int u) -> int32_t {
    return (int32_t)fwin.div((uint32_t)(u + 1) * (uint32_t)b.fast_ms + (uint32_t)win - 1u) - 1;
  };
  auto tick_win = [&](int u) -> int32_t {
    return store_win ? swin[u] : tick_of(u);
  };
  uint16_t* sany = snx + (size_t)(nf + 1) * MMAX;                          // [nf + 1]
  __shared__ int s_cap[8][MMAX];   // unit footprints: replicas above the floor, per warp
#pragma unroll 4
  for (int u = threadIdx.x; u < nf; u += blockDim.x) {
    int kd = 0, rv = -1;
    unsigned long long pk = 0;
    uint32_t dm = 0;
    if (!RANK) {
      // both entries' loads issued before either is used
      const bool has_slow = (u + 1) % ratio == 0;
      const int es = nf + (u + 1) / ratio - 1;
      const int rf = recv_tab[row0 + u];
      const unsigned long long pf = packed[row0 + u];
      const uint32_t df = dmask[row0 + u];
      const int rs = has_slow ? recv_tab[row0 + es] : -1;
      const unsigned long long ps = has_slow ? packed[row0 + es] : 0ull;
      const uint32_t ds = has_slow ? dmask[row0 + es] : 0u;
      if (rf >= 0) {
        kd = TRE_RESCUE; rv = rf; pk = pf; dm = df;
      } else if (rs >= 0) {
        kd = TRE_REBALANCE; rv = rs; pk = ps; dm = ds;
      }
    } else {
      // a slow tick falls on the window of the fast tick it coincides with;
      // a rescue at a tick takes precedence over its rebalance
      T z[MMAX];
      uint8_t cl[MMAX];
      tick_row<T, MMAX, QUAD>(b, si, (uint32_t)tick_of(u), z, cl);
      TickAction<T, MMAX, QUAD> a;
      tick_action<T, MMAX, QUAD>(b, ti, true, z, cl, a);
      if (a.recv >= 0) {
        kd = TRE_RESCUE; rv = a.recv; pk = a.pk; dm = a.dm;
      } else if ((u + 1) % ratio == 0) {
        tick_action<T, MMAX, QUAD>(b, ti, false, z, cl, a);
        if (a.recv >= 0) { kd = TRE_REBALANCE; rv = a.recv; pk = a.pk; dm = a.dm; }
      }
    }
    TickRec t;
    t.pk = pk;
    t.dm = dm;
    t.recv = (int16_t)rv;
    t.kind = (uint8_t)kd;
    t.pad = 0;
    srec[u] = t;
    if (store_win) swin[u] = tick_of(u);
  }
  __syncthreads();
  // next-tick tables, a suffix minimum per column (MMAX models, then "any"):
  // the CTA's threads split each column into segments of consecutive ticks;
  // each finds its segment's first acting tick, then writes its segment
  // backwards from the first acting tick of the segments after it
  constexpr int NC = MMAX + 1;
  const int n_seg = (int)blockDim.x / NC;              // segments per column
  // a segment length of 1 mod 8 puts the segments' tick records (16 bytes, so
  // 8 to a bank cycle) of one step on different banks
  int seg_len = (nf + n_seg - 1) / n_seg;
  seg_len += (9 - seg_len % 8) % 8;
  __shared__ int s_first[256];                         // [NC][n_seg]
  const int my_c = threadIdx.x / n_seg, my_s = threadIdx.x % n_seg;
  const bool has_seg = my_c < NC;
  auto acts = [&](int u, int c) -> bool {
    const TickRec& t = srec[u];
    if (t.recv < 0) return false;
    if (c == MMAX) return true;                        // anything acts
    return c < M && (t.dm >> c & 1u);                  // padding columns never give
  };
  const int u_lo = my_s * seg_len, u_hi = min(nf, u_lo + seg_len);
  if (has_seg) {
    int f = nf;
    for (int u = u_lo; u < u_hi; ++u)
      if (acts(u, my_c)) {
        f = u;
        break;
      }
    s_first[threadIdx.x] = f;
  }
  __syncthreads();
  if (has_seg) {
    uint16_t* col = my_c < MMAX ? snx + my_c : sany;
    const int cs = my_c < MMAX ? MMAX : 1;             // column stride
    int v = nf;
    for (int j = my_s + 1; j < n_seg; ++j) v = min(v, s_first[my_c * n_seg + j]);
    if (my_s == n_seg - 1) col[(size_t)nf * cs] = (uint16_t)nf;
    for (int u = u_hi - 1; u >= u_lo; --u) {
      if (acts(u, my_c)) v = u;
      col[(size_t)u * cs] = (uint16_t)v;
    }
  }
  __syncthreads();
  // one instance per warp, walked by its first lane
  if (lane != 0) return;
  for (int ci = warp; ci < b.n_cap; ci += n_warps) {
  const int inst = (si * b.n_tau + ti) * b.n_cap + ci;
  const int Kp = b.cap_list[ci];
  const int64_t cap = b.moves_cap;
  tre_move* mv = b.moves + (size_t)inst * cap;
  int r[MMAX], rmin[MMAX], g[MMAX];
  int64_t used = 0;
  bool bad = false, unit = true;
  uint32_t avail = 0;
#pragma unroll
  for (int m = 0; m < MMAX; ++m) {
    r[m] = 0;
    rmin[m] = 0;
    g[m] = 1;
    if (m < M) {
      r[m] = b.r0[m];
      rmin[m] = b.r_min[m];
      g[m] = b.footprint[m];
      used += (int64_t)g[m] * r[m];
      if (r[m] < 0 || rmin[m] < 0 || g[m] < 1) bad = true;
      if (g[m] != 1) unit = false;
      if (r[m] > rmin[m]) avail |= 1u << m;
    }
  }
  int64_t free_pool = b.budget - used;
  if (bad || free_pool < 0) {
    for (int m = 0; m < M && m < MMAX; ++m) b.r_out[(size_t)inst * M + m] = sel<T, MMAX>(r, m);
    b.n_moves[inst] = 0;
    b.diag->err = TRE_EINVAL;
    continue;
  }
  auto emit = [&](int64_t at, int32_t k, int recv, int donor, int kind, int sq) {
    if (at < cap) mv[at] = tre_move{k, (int16_t)recv, (int16_t)donor, (uint8_t)kind, (uint8_t)sq, 0};
  };
  int64_t nm = 0;
  int u = 0;
  if (unit) {
    // unit footprints: a transition is one replica, so a tick moves up to
    // K_p replicas from the pool, then from donors in order
    int* scap = s_cap[warp];
    for (int m = 0; m < M && m < MMAX; ++m) scap[m] = sel<T, MMAX>(r, m) - sel<T, MMAX>(rmin, m);
    // next-donor rows are masked by `avail` with these halfword lifts, rebuilt
    // only when `avail` changes
    uint32_t lw[MMAX / 2];
    uint32_t lw_for = ~avail;
    auto next_tick = [&](int uu) -> int {
      if (free_pool > 0) return sany[uu];
      if (lw_for != avail) {
#pragma unroll
        for (int i = 0; i < MMAX / 2; ++i)
          lw[i] = ((avail >> (2 * i)) & 1u ? 0u : 0xffffu) |
                  ((avail >> (2 * i + 1)) & 1u ? 0u : 0xffff0000u);
        lw_for = avail;
      }
      const uint4* q = reinterpret_cast<const uint4*>(snx + (size_t)uu * MMAX);
      uint32_t acc = 0xffffffffu;
#pragma unroll
      for (int h = 0; h < MMAX / 8; ++h) {
        const uint4 w = q[h];
        acc = __vminu2(acc, w.x | lw[4 * h]);
        acc = __vminu2(acc, w.y | lw[4 * h + 1]);
        acc = __vminu2(acc, w.z | lw[4 * h + 2]);
        acc = __vminu2(acc, w.w | lw[4 * h + 3]);
      }
      return (int)min(acc & 0xffffu, acc >> 16);
    };
    if (Kp == 1 && MMAX == 8 && b.budget <= 255) {
      // as below, with the replicas above the floor packed one byte per model
      // in a register (a model never holds more than the budget)
      unsigned long long cp = 0;
      for (int m = 0; m < M; ++m) cp |= (unsigned long long)scap[m] << (8 * m);
      int32_t nm1 = 0;
      while (true) {
        const int nxt = next_tick(u);
        if (nxt >= nf) break;
        u = nxt + 1;
        const TickRec tr = srec[nxt];
        const int32_t k = tick_win(nxt);
        const int recv = tr.recv;
        int donor = -1;
        if (free_pool > 0) {
          --free_pool;
        } else {
          const uint32_t left = avail & tr.dm;
          const uint32_t tl = ((left & 0xFu) * 0x00204081u) & 0x01010101u;
          const uint32_t th = (((left >> 4) & 0xFu) * 0x00204081u) & 0x01010101u;
          const uint32_t pl = (uint32_t)tr.pk;
          const int nd = __popc(tr.dm);
          uint32_t f0 = __byte_perm(tl, th, pl & 0xFFFFu);
          uint32_t f1 = __byte_perm(tl, th, pl >> 16);
          if (nd < 4) f0 &= (1u << (8 * nd)) - 1u;
          if (nd < 8) f1 &= nd <= 4 ? 0u : (1u << (8 * (nd - 4))) - 1u;
          const int j = f0 ? (__ffs(f0) - 1) >> 3 : 4 + ((__ffs(f1) - 1) >> 3);
          donor = (int)((pl >> (4 * j)) & 15u);
          cp -= 1ull << (8 * donor);
          if (((cp >> (8 * donor)) & 0xFFull) == 0) avail &= ~(1u << donor);
        }
        put_move(mv, nm1, cap, k, recv, donor, tr.kind, 0);
        ++nm1;
        cp += 1ull << (8 * recv);
        avail |= 1u << recv;
      }
      for (int m = 0; m < M; ++m) scap[m] = (int)((cp >> (8 * m)) & 0xFFull);
      nm = nm1;
      u = nf;
    }
    if (Kp == 1 && MMAX == 16 && b.budget <= 255) {
      // as above for up to 16 models: the replicas above the floor packed a
      // byte per model in two registers, and the donor the first model of
      // the tick's order that can still give (the jump only lands on ticks
      // that have one when the pool is empty)
      unsigned long long c0 = 0ull, c1 = 0ull;
      for (int m = 0; m < M; ++m) {
        const unsigned long long v = (unsigned long long)scap[m] << (8 * (m & 7));
        if (m < 8) c0 |= v; else c1 |= v;
      }
      int32_t nm1 = 0;
      while (true) {
        const int nxt = next_tick(u);
        if (nxt >= nf) break;
        u = nxt + 1;
        const TickRec tr = srec[nxt];
        const int32_t k = tick_win(nxt);
        const int recv = tr.recv;
        int donor = -1;
        if (free_pool > 0) {
          --free_pool;
        } else {
          const uint32_t left = avail & tr.dm;
          unsigned long long pk = tr.pk;
          int d = (int)(pk & 15u);
          for (int p = 1; p < MMAX && !((left >> d) & 1u); ++p) {
            pk >>= 4;
            d = (int)(pk & 15u);
          }
          donor = d;
          const int sh = 8 * (d & 7);
          const unsigned long long c = (d < 8 ? c0 : c1) - (1ull << sh);
          if (d < 8) c0 = c; else c1 = c;
          if (((c >> sh) & 0xFFull) == 0) avail &= ~(1u << d);
        }
        put_move(mv, nm1, cap, k, recv, donor, tr.kind, 0);
        ++nm1;
        if (recv < 8) c0 += 1ull << (8 * recv);
        else c1 += 1ull << (8 * (recv - 8));
        avail |= 1u << recv;
      }
      for (int m = 0; m < M; ++m)
        scap[m] = (int)(((m < 8 ? c0 : c1) >> (8 * (m & 7))) & 0xFFull);
      nm = nm1;
      u = nf;
    }
    if (Kp == 1 && MMAX == 8 && u < nf) {
      // one transition per tick: every tick the jump lands on moves exactly
      // one replica (it has a receiver, and a usable donor when the pool is
      // empty), so the visit is straight-line code
      int32_t nm1 = 0;
      while (true) {
        const int nxt = next_tick(u);
        if (nxt >= nf) break;
        u = nxt + 1;
        const TickRec tr = srec[nxt];
        const int32_t k = tick_win(nxt);
        const int recv = tr.recv;
        int donor = -1;
        if (free_pool > 0) {
          --free_pool;
        } else {
          const uint32_t left = avail & tr.dm;
          const uint32_t tl = ((left & 0xFu) * 0x00204081u) & 0x01010101u;
          const uint32_t th = (((left >> 4) & 0xFu) * 0x00204081u) & 0x01010101u;
          const uint32_t pl = (uint32_t)tr.pk;
          const int nd = __popc(tr.dm);
          uint32_t f0 = __byte_perm(tl, th, pl & 0xFFFFu);
          uint32_t f1 = __byte_perm(tl, th, pl >> 16);
          if (nd < 4) f0 &= (1u << (8 * nd)) - 1u;
          if (nd < 8) f1 &= nd <= 4 ? 0u : (1u << (8 * (nd - 4))) - 1u;
          const int j = f0 ? (__ffs(f0) - 1) >> 3 : 4 + ((__ffs(f1) - 1) >> 3);
          donor = (int)((pl >> (4 * j)) & 15u);
          const int c = scap[donor] - 1;
          scap[donor] = c;
          if (c == 0) avail &= ~(1u << donor);
        }
        put_move(mv, nm1, cap, k, recv, donor, tr.kind, 0);
        ++nm1;
        scap[recv] += 1;
        avail |= 1u << recv;
      }
      nm = nm1;
      u = nf;
    }
    while (u < nf) {
      const int nxt = next_tick(u);
      if (nxt >= nf) break;
      u = nxt;
      const TickRec tr = srec[u];
      const int32_t k = tick_win(u);
      ++u;
      const int recv = tr.recv;
      if (recv < 0) continue;
      uint32_t left = avail & tr.dm;
      if (free_pool <= 0 && !left) continue;
      const int kind = tr.kind;
      const int n_pool = free_pool < Kp ? (int)free_pool : Kp;
      for (int q = 0; q < n_pool; ++q) put_move(mv, nm + q, cap, k, recv, -1, kind, q);
      int sq = n_pool;
      unsigned long long pk = tr.pk;
      if (MMAX == 8) {
        // usable donors by position in the order, one flag byte per position:
        // spread the usable bits to bytes, then gather them by the order's
        // model nibbles; positions past the tick's donor count are masked
        const uint32_t tl = ((left & 0xFu) * 0x00204081u) & 0x01010101u;
        const uint32_t th = (((left >> 4) & 0xFu) * 0x00204081u) & 0x01010101u;
        const uint32_t pl = (uint32_t)pk;
        const int nd = __popc(tr.dm);
        uint32_t f0 = __byte_perm(tl, th, pl & 0xFFFFu);
        uint32_t f1 = __byte_perm(tl, th, pl >> 16);
        if (nd < 4) f0 &= (1u << (8 * nd)) - 1u;
        if (nd < 8) f1 &= nd <= 4 ? 0u : (1u << (8 * (nd - 4))) - 1u;
        while (sq < Kp && (f0 | f1)) {
          int j;
          if (f0) {
            j = (__ffs(f0) - 1) >> 3;
            f0 &= ~(0xFFu << (8 * j));
          } else {
            const int j1 = (__ffs(f1) - 1) >> 3;
            f1 &= ~(0xFFu << (8 * j1));
            j = 4 + j1;
          }
          const int m = (int)((pl >> (4 * j)) & 15u);
          const int c = scap[m];
          const int take = min(c, Kp - sq);
          scap[m] = c - take;
          if (take == c) avail &= ~(1u << m);
          for (int i = 0; i < take; ++i, ++sq) put_move(mv, nm + sq, cap, k, recv, m, kind, sq);
        }
      } else {
        while (sq < Kp && left) {
          const int m = (int)(pk & 15);
          pk >>= 4;
          if (!(left >> m & 1)) continue;
          left &= ~(1u << m);
          const int c = scap[m];
          const int take = min(c, Kp - sq);
          scap[m] = c - take;
          if (take == c) avail &= ~(1u << m);
          for (int i = 0; i < take; ++i, ++sq) put_move(mv, nm + sq, cap, k, recv, m, kind, sq);
        }
      }
      const int cr = scap[recv] + sq;
      scap[recv] = cr;
      if (cr > 0) avail |= 1u << recv;
      free_pool -= n_pool;
      nm += sq;
    }
    for (int m = 0; m < M && m < MMAX; ++m)
      b.r_out[(size_t)inst * M + m] = scap[m] + sel<T, MMAX>(rmin, m);
    b.n_moves[inst] = nm;
    if (nm > cap) b.diag->err = TRE_EOVERFLOW;
    continue;
  }
  while (u < nf) {
    // the next tick where something may move
    int nxt;
    if (free_pool > 0) nxt = sany[u];
    else nxt = next_donor_tick<MMAX>(snx + (size_t)u * MMAX, avail);
    if (nxt >= nf) break;
    u = nxt;
    const TickRec tr = srec[u];
    const int recv = tr.recv;
    const int kind = tr.kind;
    const int32_t k = tick_win(u);
    ++u;
    if (recv < 0) continue;
    const uint32_t usable = avail & tr.dm;
    const int need = unit ? 1 : sel<T, MMAX>(g, recv);
    if (free_pool < need && !usable) continue;
    unsigned long long pk = tr.pk;
    if (unit) {
      const int n_pool = (int)(free_pool < Kp ? free_pool : Kp);
      for (int q = 0; q < n_pool; ++q) emit(nm + q, k, recv, -1, kind, q);
      int sq = n_pool;
      uint32_t left = usable;
      while (sq < Kp && left) {
        const int m = (int)(pk & 15);
        pk >>= 4;
        if (!(left >> m & 1)) continue;
        left &= ~(1u << m);
        const int c = sel<T, MMAX>(r, m) - sel<T, MMAX>(rmin, m);
        const int take = min(c, Kp - sq);
        add_at<T, MMAX>(r, m, -take);
        if (take == c) avail &= ~(1u << m);
        for (int i = 0; i < take; ++i, ++sq) emit(nm + sq, k, recv, m, kind, sq);
      }
      add_at<T, MMAX>(r, recv, sq);
      if (sel<T, MMAX>(r, recv) > sel<T, MMAX>(rmin, recv)) avail |= 1u << recv;
      free_pool -= n_pool;
      nm += sq;
      continue;
    }
    for (int sq = 0; sq < Kp; ++sq) {
      if (free_pool >= need) {
        free_pool -= need;
        add_at<T, MMAX>(r, recv, 1);
        if (sel<T, MMAX>(r, recv) > sel<T, MMAX>(rmin, recv)) avail |= 1u << recv;
        emit(nm++, k, recv, -1, kind, sq);
        continue;
      }
      int64_t f = free_pool;
      const int64_t nm0 = nm;
      int taken[MMAX];
#pragma unroll
      for (int m = 0; m < MMAX; ++m) taken[m] = 0;
      unsigned long long order = pk;
      uint32_t left = avail & tr.dm;
      while (f < need && left) {
        const int m = (int)(order & 15);
        order >>= 4;
        if (!(left >> m & 1)) continue;
        left &= ~(1u << m);
        int c = sel<T, MMAX>(r, m) - sel<T, MMAX>(rmin, m);
        const int gm = sel<T, MMAX>(g, m);
        while (f < need && c > 0) {
          add_at<T, MMAX>(taken, m, 1);
          --c;
          f += gm;
          emit(nm++, k, recv, m, kind, sq);
        }
      }
      if (f < need) {
        nm = nm0;
        break;
      }
#pragma unroll
      for (int m = 0; m < MMAX; ++m) {
        r[m] -= taken[m];
        if (m < M && !(r[m] > rmin[m])) avail &= ~(1u << m);
      }
      add_at<T, MMAX>(r, recv, 1);
      if (sel<T, MMAX>(r, recv) > sel<T, MMAX>(rmin, recv)) avail |= 1u << recv;
      free_pool = f - need;
    }
  }
  for (int m = 0; m < M && m < MMAX; ++m) b.r_out[(size_t)inst * M + m] = sel<T, MMAX>(r, m);
  b.n_moves[inst] = nm;
  if (nm > cap) b.diag->err = TRE_EOVERFLOW;
  }
}

constexpr size_t kStageMax = 160 * 1024;

template <class T, int MPL>
cudaError_t walk_launch(const WalkBatch<T>& b, WalkWs& w, cudaStream_t s) {
  int max_ent = 0;
  for (int i = 0; i < b.n_series; ++i) max_ent = std::max(max_ent, b.ent_base[i + 1] - b.ent_base[i]);
  const size_t smem = 2 * (((size_t)max_ent * 2 + 15) & ~(size_t)15) +
                      2 * (((size_t)max_ent * b.M * 2 + 15) & ~(size_t)15);
  const dim3 grid((unsigned)(b.n_series * b.n_tau),
                  (unsigned)((b.n_cap + kCapWarps - 1) / kCapWarps));
  const unsigned th = (unsigned)(std::min(b.n_cap, kCapWarps) * 32);
  if (smem <= kStageMax) {
    cudaError_t e = func_smem_once((const void*)k_walk<T, MPL, true>, (int)kStageMax, false);
    if (e) return e;
    k_walk<T, MPL, true><<<grid, th, smem, s>>>(b, w.recv, w.n_donor, w.rank, w.order, w.dm64);
  } else {
    k_walk<T, MPL, false><<<grid, th, 0, s>>>(b, w.recv, w.n_donor, w.rank, w.order, w.dm64);
  }
  return cudaGetLastError();
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
  w.n_donor = a.take<int16_t>((size_t)std::max<int64_t>(total * b.n_tau, 1));
  w.rank = a.take<uint16_t>((size_t)std::max<int64_t>(total * b.n_tau * b.M, 1));
  w.order = a.take<uint16_t>((size_t)std::max<int64_t>(total * b.n_tau * b.M, 1));
  w.packed = a.take<unsigned long long>((size_t)std::max<int64_t>(total * b.n_tau, 1));
  w.dmask = a.take<uint32_t>((size_t)std::max<int64_t>(total * b.n_tau, 1));
  w.dm64 = a.take<unsigned long long>((size_t)std::max<int64_t>(total * b.n_tau, 1));
}

// unit footprints and few models: thread-per-instance walk with staged tables
// Whether the jump walk applies (nested cadences, a fast tick not shorter
// than a window, tick tables within the opt-in shared-memory limit) and its
// shared memory: the tables, with or without the staged tick windows.
struct JumpPlan {
  bool ok, store_win;
  size_t smem, lim;
};
template <class T, int MMAX> JumpPlan jump_plan(const WalkBatch<T>& b) {
  JumpPlan p{false, false, 0, 0};
  if (b.slow_ms % b.fast_ms != 0 || b.fast_ms < b.series_win[0]) return p;
  bool ok = true;
  size_t jsmem = 0, wsmem = 0;
  for (int i = 0; i < b.n_series; ++i) {
    if (b.fast_ms < b.series_win[i]) ok = false;
    const int64_t nf = (int64_t)b.series_K[i] * b.series_win[i] / b.fast_ms;
    if (nf >= 32767) ok = false;
    const size_t need = (size_t)nf * sizeof(TickRec) + (size_t)(nf + 1) * MMAX * 2 +
                        (size_t)(nf + 1) * 2;
    jsmem = std::max(jsmem, need);
    wsmem = std::max(wsmem, (size_t)((nf + 3) & ~3) * 4);
  }
  // the largest dynamic shared memory a block may opt into, beside the
  // kernel's static per-warp counts
  int dev = 0, optin = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) !=
          cudaSuccess || optin <= 4096) {
    cudaGetLastError();
    return p;
  }
  p.lim = (size_t)optin - 2048;
  p.store_win = jsmem + wsmem <= p.lim;
  p.smem = p.store_win ? jsmem + wsmem : jsmem;
  p.ok = ok && p.smem <= p.lim;
  return p;
}

// The jump walk; RANK: it ranks its own ticks (one launch for the selection).
template <class T, int MMAX, bool RANK, bool QUAD>
cudaError_t jump_launch(const WalkBatch<T>& b, const WalkWs& w, const JumpPlan& p,
                        cudaStream_t s) {
  cudaError_t e =
      func_smem_once((const void*)k_walk_jump<T, MMAX, RANK, QUAD>, (int)p.lim, false);
  if (e) return e;
  // eight warps build the tables; the first n_cap of them walk
  k_walk_jump<T, MMAX, RANK, QUAD><<<b.n_series * b.n_tau, 256, p.smem, s>>>(
      b, w.recv, w.packed, w.dmask, p.store_win);
  return cudaGetLastError();
}

template <class T, int MMAX>
cudaError_t walk_thread_launch(const WalkBatch<T>& b, WalkWs& w, size_t smem, cudaStream_t s) {
  cudaError_t e = func_smem_once((const void*)k_walk_thread<T, MMAX>, (int)kStageMax, false);
  if (e) return e;
  k_walk_thread<T, MMAX><<<b.n_series * b.n_tau, 32, smem, s>>>(b, w.recv, w.packed, w.dmask);
  return cudaGetLastError();
}

template <class T>
cudaError_t launch_walk(const WalkBatch<T>& b, WalkWs& w, cudaStream_t s, int* launches) {
  if (launches) *launches = 0;
  if (b.n_inst == 0) return cudaSuccess;
  const int64_t ents = (int64_t)b.ent_base[b.n_series] * b.n_tau;
  // which walk runs decides whether the per-model rank tables are needed
  int max_ent = 0;
  for (int i = 0; i < b.n_series; ++i)
    max_ent = std::max(max_ent, b.ent_base[i + 1] - b.ent_base[i]);
  const size_t thread_smem = (size_t)max_ent * (8 + 4 + 2) + 16;
  const bool thread_walk = b.M <= 16 && b.n_cap <= 32 && thread_smem <= kStageMax;
  // rows start on 16-byte boundaries when M is a multiple of 4 (series
  // offsets are multiples of M) and both arrays are 16-byte aligned
  const bool quad = b.M % 4 == 0 && (((uintptr_t)b.Z | (uintptr_t)b.cls) & 15) == 0;
  JumpPlan jp{false, false, 0, 0};
  if (thread_walk && ents > 0) jp = b.M <= 8 ? jump_plan<T, 8>(b) : jump_plan<T, 16>(b);
  // with a CTA per SM or more, the jump walk ranks its own ticks: one launch
  if (jp.ok && b.n_series * b.n_tau >= device_sm_count()) {
    if (launches) *launches = 1;
    if (b.M <= 8)
      return quad ? jump_launch<T, 8, true, true>(b, w, jp, s)
                  : jump_launch<T, 8, true, false>(b, w, jp, s);
    return quad ? jump_launch<T, 16, true, true>(b, w, jp, s)
                : jump_launch<T, 16, true, false>(b, w, jp, s);
  }
  // the tick ranking, then the walk
  if (launches) *launches = (ents > 0 ? 1 : 0) + 1;
  if (ents > 0) {
    const unsigned g = (unsigned)((ents + 127) / 128);
    if (b.M <= 8 && quad) {
      k_tick_rank_small<T, 8, true><<<g, 128, 0, s>>>(b, w.recv, w.n_donor, w.rank, w.order,
                                                      w.packed, w.dmask, !thread_walk, w.dm64);
    } else if (b.M <= 8) {
      k_tick_rank_small<T, 8, false><<<g, 128, 0, s>>>(b, w.recv, w.n_donor, w.rank, w.order,
                                                       w.packed, w.dmask, !thread_walk, w.dm64);
    } else if (b.M <= 16) {
      k_tick_rank_small<T, 16, false><<<g, 128, 0, s>>>(b, w.recv, w.n_donor, w.rank, w.order,
                                                        w.packed, w.dmask, !thread_walk, w.dm64);
    } else if (b.M <= 32) {
      k_tick_rank_small<T, 32, false><<<g, 128, 0, s>>>(b, w.recv, w.n_donor, w.rank, w.order,
                                                        w.packed, w.dmask, true, w.dm64);
    } else {
      const int64_t th = ents * b.M;
      k_tick_rank<T><<<(unsigned)((th + 255) / 256), 256, 0, s>>>(b, w.recv, w.n_donor, w.rank,
                                                                   w.order, w.dm64);
    }
  }
  if (jp.ok)
    return b.M <= 8 ? jump_launch<T, 8, false, false>(b, w, jp, s)
                    : jump_launch<T, 16, false, false>(b, w, jp, s);
  if (thread_walk)
    return b.M <= 8 ? walk_thread_launch<T, 8>(b, w, thread_smem, s)
                    : walk_thread_launch<T, 16>(b, w, thread_smem, s);
  const int mpl = (b.M + 31) / 32;
  if (mpl <= 1) return walk_launch<T, 1>(b, w, s);
  if (mpl <= 2) return walk_launch<T, 2>(b, w, s);
  if (mpl <= 4) return walk_launch<T, 4>(b, w, s);
  if (mpl <= 8) return walk_launch<T, 8>(b, w, s);
  if (mpl <= 16) return walk_launch<T, 16>(b, w, s);
  return walk_launch<T, 32>(b, w, s);
}

template void walk_ws_layout<float>(Arena&, WalkBatch<float>&, WalkWs&);
template void walk_ws_layout<double>(Arena&, WalkBatch<double>&, WalkWs&);
template cudaError_t launch_walk<float>(const WalkBatch<float>&, WalkWs&, cudaStream_t, int*);
template cudaError_t launch_walk<double>(const WalkBatch<double>&, WalkWs&, cudaStream_t, int*);

}  // namespace tre
