// Calibration of the healthy boundary theta (Sec. III-B: the lowest smoothed TSS
// value at which the SLO reliability target is still met), for a batch of
// series at once.
//
// For model m, let the calibration windows be those with at least one arrival,
// not idle, S > 0. For a value s let C(s) be the number of calibration windows
// with S >= s and H(s) the healthy ones among them. theta is the smallest S
// value s with H(s) >= reliability * C(s).
//
// Instead of sorting, each (series, model) packs its (S, healthy) pairs into
// unsigned keys (the bit pattern of a positive float orders like the float)
// and one CTA finds theta by a descent over the key range: the current range
// is split linearly into buckets; a histogram gives per bucket the count, the
// healthy count and the smallest key; per bucket, in parallel, the exact test
// at its smallest value (everything at or above it included) and an upper
// bound for any value inside it (only its healthy windows added). The lowest
// bucket that passes either gives theta directly (its smallest value
// qualifies and nothing below did) or is refined; a refinement that finds
// nothing resumes with the buckets above it. Counts are exact integers and the
// final test is the definition's double expression, so theta is exact.
#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace tre {
namespace {

constexpr int kThrTable = 4096;
constexpr int kNB = 1024;           // buckets per level = threads per CTA
constexpr int kWarps = kNB / 32;

template <class T> struct KeyOf;
template <> struct KeyOf<float> {
  using U = uint32_t;
  static constexpr int kLevels = 4;   // 31 key bits, >= 10 bits resolved per level
};
template <> struct KeyOf<double> {
  using U = unsigned long long;
  static constexpr int kLevels = 7;   // 63 key bits
};

__device__ __forceinline__ float value_of(uint32_t k) { return __uint_as_float(k); }
__device__ __forceinline__ double value_of(unsigned long long k) {
  return __longlong_as_double((long long)k);
}

// thr[a] = smallest integer n with (double)n >= ok_frac * (double)a; also
// resets the per-(series, model) candidate key ranges filled by k_pack
template <class U>
__global__ void k_thr(double ok_frac, int32_t* thr, int n_sm, U* kmin, U* kmax, uint32_t* ncand) {
  const int a = blockIdx.x * blockDim.x + threadIdx.x;
  if (a < n_sm) {
    kmin[a] = ~(U)0;
    kmax[a] = 0;
    ncand[a] = 0;
  }
  if (a >= kThrTable) return;
  const double v = ok_frac * (double)a;
  int32_t t;
  if (!(v <= 2147483647.0)) t = 0x7fffffff;           // unreachable (or NaN)
  else if (v <= -2147483647.0) t = -0x7fffffff;
  else t = (int32_t)ceil(v);
  thr[a] = t;
}

__device__ __forceinline__ bool healthy(uint32_t n_arr, uint32_t n_met, const int32_t* thr,
                                        double ok_frac) {
  if (n_arr < (uint32_t)kThrTable) return (int64_t)n_met >= (int64_t)thr[n_arr];
  return (double)n_met >= ok_frac * (double)n_arr;
}

// [K][M] S, class, packed SLO counts of every series -> [M][K] packed keys
// (0 = not a calibration window) at the series' element offset, plus each
// (series, model)'s smallest and largest candidate key and candidate count.
// A CTA transposes one tile of TK windows x TM models (TM = the model count
// rounded up to a power of two, at most 32; TK * TM = 1024) through shared
// memory; every thread of a CTA keeps to one model of the tile.
constexpr int kPackThreads = 256;
constexpr int kPackTile = 1024;
struct PackPlan {
  int lg_tm, tm, lg_tk, tk, m_tiles;
  int tile_base[kMaxSeries + 1];   // prefix of tiles per series
};

__device__ __forceinline__ uint32_t warp_min(uint32_t v) { return __reduce_min_sync(0xffffffffu, v); }
__device__ __forceinline__ uint32_t warp_max(uint32_t v) { return __reduce_max_sync(0xffffffffu, v); }
__device__ __forceinline__ unsigned long long warp_min(unsigned long long v) {
  for (int o = 16; o > 0; o >>= 1) {
    const unsigned long long y = __shfl_xor_sync(0xffffffffu, v, o);
    v = y < v ? y : v;
  }
  return v;
}
__device__ __forceinline__ unsigned long long warp_max(unsigned long long v) {
  for (int o = 16; o > 0; o >>= 1) {
    const unsigned long long y = __shfl_xor_sync(0xffffffffu, v, o);
    v = y > v ? y : v;
  }
  return v;
}

__device__ __forceinline__ void load4(const float* p, float (&v)[4]) {
  const float4 q = *reinterpret_cast<const float4*>(p);
  v[0] = q.x; v[1] = q.y; v[2] = q.z; v[3] = q.w;
}
__device__ __forceinline__ void load4(const double* p, double (&v)[4]) {
  const double2 a = reinterpret_cast<const double2*>(p)[0];
  const double2 b = reinterpret_cast<const double2*>(p)[1];
  v[0] = a.x; v[1] = a.y; v[2] = b.x; v[3] = b.y;
}

// The same packing with 16-byte loads, for model counts that fill whole tile
// rows (M a multiple of TM and of 4, 16-byte aligned arrays): a thread reads
// four consecutive models of one window; the candidate range and count of a
// tile row come from warp reductions over the transposed tile.
template <class T>
__global__ void __launch_bounds__(kPackThreads)
k_pack_vec(const __grid_constant__ SeriesTable<T> tab, const __grid_constant__ PackPlan pp,
           const T* __restrict__ S, const uint8_t* __restrict__ cls,
           const unsigned long long* __restrict__ slo, const int32_t* __restrict__ thr,
           double ok_frac, typename KeyOf<T>::U* __restrict__ keys,
           typename KeyOf<T>::U* kmin_g, typename KeyOf<T>::U* kmax_g, uint32_t* ncand_g) {
  using U = typename KeyOf<T>::U;
  static_assert(kPackTile == 4 * kPackThreads, "four elements per thread");
  __shared__ U tile[kPackTile + 32];
  __shared__ U smin[32], smax[32];
  __shared__ uint32_t scnt[32];
  const int s = prefix_index(pp.tile_base, tab.n, blockIdx.x);
  const int M = tab.M, K = tab.K[s];
  const int t_loc = blockIdx.x - pp.tile_base[s];
  const int kt = pp.m_tiles == 1 ? t_loc : t_loc / pp.m_tiles;
  const int k0 = kt * pp.tk, m0 = (t_loc - kt * pp.m_tiles) * pp.tm;
  const size_t off = (size_t)tab.off[s];
  const int tid = threadIdx.x;
  if (tid < 32) {
    smin[tid] = ~(U)0;
    smax[tid] = 0;
    scnt[tid] = 0;
  }
  const int TKp = pp.tk + 1;
  const int e4 = tid * 4;
  const int kk = e4 >> pp.lg_tm, mm = e4 & (pp.tm - 1);
  const int k = k0 + kk;
  U v[4] = {0, 0, 0, 0};
  if (k < K) {
    const size_t x = off + (size_t)k * M + m0 + mm;
    T sv[4];
    load4(S + x, sv);
    const uchar4 c4 = *reinterpret_cast<const uchar4*>(cls + x);
    const ulonglong2 a = reinterpret_cast<const ulonglong2*>(slo + x)[0];
    const ulonglong2 b = reinterpret_cast<const ulonglong2*>(slo + x)[1];
    const unsigned long long cv[4] = {a.x, a.y, b.x, b.y};
    const uint8_t iv[4] = {c4.x, c4.y, c4.z, c4.w};
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const uint32_t n_arr = (uint32_t)cv[u];
      if (iv[u] != kIdle && n_arr >= 1 && sv[u] > (T)0) {
        const bool h = healthy(n_arr, (uint32_t)(cv[u] >> 32), thr, ok_frac);
        v[u] = ((U)key_of(sv[u]) << 1) | (U)(h ? 1 : 0);
      }
    }
  }
#pragma unroll
  for (int u = 0; u < 4; ++u) tile[(mm + u) * TKp + kk] = v[u];
  __syncthreads();
  // tile rows are models: a warp's 32 consecutive elements share one row
#pragma unroll
  for (int j = 0; j < kPackTile / kPackThreads; ++j) {
    const int e = tid + j * kPackThreads;
    const int r = e >> pp.lg_tk, kr = e & (pp.tk - 1);
    const int kg = k0 + kr;
    const U w = tile[r * TKp + kr];
    const bool in = kg < K;
    if (in) keys[off + (size_t)(m0 + r) * K + kg] = w;
    const bool cand = in && w != 0;
    const U lo = warp_min(cand ? (U)(w >> 1) : ~(U)0);
    const U hi = warp_max(cand ? (U)(w >> 1) : (U)0);
    const uint32_t nc = __popc(__ballot_sync(0xffffffffu, cand));
    if ((tid & 31) == 0 && nc) {
      atomicMin(&smin[r], lo);
      atomicMax(&smax[r], hi);
      atomicAdd(&scnt[r], nc);
    }
  }
  __syncthreads();
  if (tid < pp.tm && scnt[tid]) {
    const size_t g = (size_t)s * M + m0 + tid;
    atomicMin(&kmin_g[g], smin[tid]);
    atomicMax(&kmax_g[g], smax[tid]);
    atomicAdd(&ncand_g[g], scnt[tid]);
  }
}

template <class T>
__global__ void __launch_bounds__(kPackThreads)
k_pack(const __grid_constant__ SeriesTable<T> tab, const __grid_constant__ PackPlan pp,
       const T* __restrict__ S, const uint8_t* __restrict__ cls,
       const unsigned long long* __restrict__ slo, const int32_t* __restrict__ thr,
       double ok_frac, typename KeyOf<T>::U* __restrict__ keys, typename KeyOf<T>::U* kmin_g,
       typename KeyOf<T>::U* kmax_g, uint32_t* ncand_g) {
  using U = typename KeyOf<T>::U;
  __shared__ U tile[kPackTile + 32];
  __shared__ U smin[32], smax[32];
  __shared__ uint32_t scnt[32];
  const int s = prefix_index(pp.tile_base, tab.n, blockIdx.x);
  const int M = tab.M, K = tab.K[s];
  const int t_loc = blockIdx.x - pp.tile_base[s];
  const int kt = pp.m_tiles == 1 ? t_loc : t_loc / pp.m_tiles;
  const int k0 = kt * pp.tk, m0 = (t_loc - kt * pp.m_tiles) * pp.tm;
  const size_t off = (size_t)tab.off[s];
  const int tid = threadIdx.x;
  const int mm = tid & (pp.tm - 1);
  const int m = m0 + mm;
  if (tid < 32) {
    smin[tid] = ~(U)0;
    smax[tid] = 0;
    scnt[tid] = 0;
  }
  U lmin = ~(U)0, lmax = 0;
  uint32_t lc = 0;
  const int TKp = pp.tk + 1;   // padded row of the transposed tile
  constexpr int J = kPackTile / kPackThreads;
  // every load of the thread's elements first, then the threshold lookups,
  // then the keys: more requests in flight per thread
  unsigned long long cj[J];
  T sj[J];
  uint8_t ij[J];
  bool in[J];
#pragma unroll
  for (int j = 0; j < J; ++j) {
    const int k = k0 + ((tid + j * kPackThreads) >> pp.lg_tm);
    in[j] = k < K && m < M;
    const size_t x = off + (size_t)k * M + m;
    cj[j] = in[j] ? slo[x] : 0ull;
    sj[j] = in[j] ? S[x] : (T)0;
    ij[j] = in[j] ? cls[x] : kIdle;
  }
  bool hj[J];
#pragma unroll
  for (int j = 0; j < J; ++j) hj[j] = healthy((uint32_t)cj[j], (uint32_t)(cj[j] >> 32), thr, ok_frac);
#pragma unroll
  for (int j = 0; j < J; ++j) {
    const int kk = (tid + j * kPackThreads) >> pp.lg_tm;
    U v = 0;
    if (in[j] && ij[j] != kIdle && (uint32_t)cj[j] >= 1 && sj[j] > (T)0) {
      const U key = (U)key_of(sj[j]);
      v = (key << 1) | (U)(hj[j] ? 1 : 0);
      lmin = key < lmin ? key : lmin;
      lmax = key > lmax ? key : lmax;
      ++lc;
    }
    tile[mm * TKp + kk] = v;
  }
  __syncthreads();
  if (lc) {
    atomicMin(&smin[mm], lmin);
    atomicMax(&smax[mm], lmax);
    atomicAdd(&scnt[mm], lc);
  }
#pragma unroll
  for (int j = 0; j < kPackTile / kPackThreads; ++j) {
    const int e = tid + j * kPackThreads;
    const int r = e >> pp.lg_tk, kk = e & (pp.tk - 1);
    const int mo = m0 + r, k = k0 + kk;
    if (mo < M && k < K) keys[off + (size_t)mo * K + k] = tile[r * TKp + kk];
  }
  __syncthreads();
  if (tid < pp.tm && m0 + tid < M && scnt[tid]) {
    const size_t g = (size_t)s * M + m0 + tid;
    atomicMin(&kmin_g[g], smin[tid]);
    atomicMax(&kmax_g[g], smax[tid]);
    atomicAdd(&ncand_g[g], scnt[tid]);
  }
}

// exclusive suffix sums over the block: out = sum of v over threads > tid
__device__ __forceinline__ int64_t block_suffix(int64_t v, int64_t* red) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x / 32;
  // inclusive suffix within the warp (lanes above)
  int64_t inc = v;
  for (int o = 1; o < 32; o <<= 1) {
    const int64_t x = __shfl_down_sync(0xffffffffu, inc, o);
    if (lane + o < 32) inc += x;
  }
  if (lane == 0) red[wid] = inc;
  __syncthreads();
  int64_t above = 0;
  for (int w = wid + 1; w < kWarps; ++w) above += red[w];
  __syncthreads();
  return inc - v + above;
}

__device__ __forceinline__ int block_min(int v, int* red) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x / 32;
  v = __reduce_min_sync(0xffffffffu, v);
  if (lane == 0) red[wid] = v;
  __syncthreads();
  int r = 0x7fffffff;
  for (int w = 0; w < kWarps; ++w) r = min(r, red[w]);
  __syncthreads();
  return r;
}

constexpr int kFine = 4096;     // buckets of the first histogram
constexpr int kUnroll = 8;      // keys per thread whose loads are issued together
constexpr int kCap = 2048;      // most keys the exact pass sorts in shared memory

template <class T> size_t search_smem_bytes() {
  using U = typename KeyOf<T>::U;
  const size_t fast = (size_t)kFine * (5 * 4) + (size_t)kCap * (sizeof(U) + 4);
  const size_t descent = (size_t)KeyOf<T>::kLevels * kNB * (4 + 4 + sizeof(U));
  return fast > descent ? fast : descent;
}

template <class T>
__global__ void __launch_bounds__(kNB)
k_search(const __grid_constant__ SeriesTable<T> tab, const typename KeyOf<T>::U* __restrict__ keys,
         const typename KeyOf<T>::U* kmin_g, const typename KeyOf<T>::U* kmax_g,
         const uint32_t* ncand_g, double reliability, T* theta, tre_diag* diag) {
  using U = typename KeyOf<T>::U;
  constexpr int NL = KeyOf<T>::kLevels;
  extern __shared__ __align__(16) unsigned char dyn[];
  __shared__ U lo_s[NL], hi_s[NL];
  __shared__ int shift_s[NL], pos_s[NL];
  __shared__ int64_t cab_s[NL], hab_s[NL];
  __shared__ int64_t red64[kWarps];
  __shared__ int red32[kWarps];
  __shared__ int nsel_s;
  __shared__ U bfmin_s;
  const int M = tab.M;
  const int s = blockIdx.x / M, m = blockIdx.x % M;
  const int K = tab.K[s];
  const U* mk = keys + (size_t)tab.off[s] + (size_t)m * K;
  const int tid = threadIdx.x, lane = tid & 31;
  const size_t out = (size_t)s * M + m;

  // ---- range of candidate keys (from the packing pass) ---------------------
  if (ncand_g[out] == 0) {
    if (tid == 0) {
      theta[out] = (T)1;
      atomicAdd(&diag->degenerate_calib, 1ull);
    }
    return;
  }
  const U kmin = kmin_g[out], kmax = kmax_g[out];

  // ---- fast path -----------------------------------------------------------
  // A fine histogram over [kmin, kmax]; per bucket the exact test at its
  // smallest value ("found") and the bound for values inside it ("maybe").
  // With bf the lowest found bucket, theta is either a value inside a maybe
  // bucket below bf or the smallest value of bf. Those maybe buckets' keys are
  // gathered, sorted and tested one distinct value at a time.
  {
    int32_t* fcnt = reinterpret_cast<int32_t*>(dyn);
    int32_t* fhl = fcnt + kFine;
    int32_t* fst = fhl + kFine;                 // run start of a selected bucket, -1 if not
    int32_t* fca = fst + kFine;                 // windows in buckets above
    int32_t* fha = fca + kFine;                 // healthy windows in buckets above
    U* list = reinterpret_cast<U*>(fha + kFine);
    int32_t* hpre = reinterpret_cast<int32_t*>(list + kCap);
    int sh = 0;
    while (sh < 63 && ((kmax - kmin) >> sh) >= (U)kFine) ++sh;
    for (int b = tid; b < kFine; b += kNB) {
      fcnt[b] = 0;
      fhl[b] = 0;
    }
    if (tid == 0) bfmin_s = ~(U)0;
    __syncthreads();
    // with fewer than 2^16 candidates, a bucket's count and healthy count
    // share one 32-bit word (one atomic per key)
    const bool packed = ncand_g[out] < 65536u;
    uint32_t* fpk = reinterpret_cast<uint32_t*>(fcnt);
    for (int i0 = 0; i0 < K; i0 += kNB * kUnroll) {
      U pv[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int i = i0 + u * kNB + tid;
        pv[u] = i < K ? mk[i] : (U)0;
      }
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const U p = pv[u];
        if (!p) continue;
        const int b = (int)(((p >> 1) - kmin) >> sh);
        if (packed) {
          atomicAdd(&fpk[b], 1u + ((uint32_t)(p & 1) << 16));
        } else {
          atomicAdd(&fcnt[b], 1);
          if (p & 1) atomicAdd(&fhl[b], 1);
        }
      }
    }
    __syncthreads();
    constexpr int PER = kFine / kNB;            // consecutive buckets per thread
    const int b0 = tid * PER;
    if (packed) {
      for (int j = 0; j < PER; ++j) {
        const uint32_t v = fpk[b0 + j];
        fcnt[b0 + j] = (int32_t)(v & 0xffffu);
        fhl[b0 + j] = (int32_t)(v >> 16);
      }
    }
    int64_t tc = 0, th = 0;
    for (int j = 0; j < PER; ++j) {
      tc += fcnt[b0 + j];
      th += fhl[b0 + j];
    }
    int64_t c_above = block_suffix(tc, red64), h_above = block_suffix(th, red64);
    int my_found = 0x7fffffff;
    uint32_t maybe_bits = 0;
    for (int j = PER - 1; j >= 0; --j) {
      const int b = b0 + j;
      const int32_t c = fcnt[b], h = fhl[b];
      fca[b] = (int32_t)c_above;
      fha[b] = (int32_t)h_above;
      if (c > 0) {
        if ((double)(h_above + h) >= reliability * (double)(c_above + c)) {
          my_found = b;
        } else if ((double)(h_above + h + 1) >= reliability * (double)(c_above + h)) {
          // a value inside adds at most the bucket's healthy windows to those
          // above; one window of slack keeps the bound valid under rounding
          maybe_bits |= 1u << j;
        }
      }
      c_above += c;
      h_above += h;
    }
    const int bf = block_min(my_found, red32);
    int64_t my_sel = 0;
    for (int j = 0; j < PER; ++j)
      if ((maybe_bits >> j & 1) && b0 + j < bf) my_sel += fcnt[b0 + j];
    const int64_t sel_above = block_suffix(my_sel, red64);
    if (tid == 0) nsel_s = 0;
    __syncthreads();
    if (my_sel) atomicAdd(&nsel_s, (int)my_sel);
    __syncthreads();
    const int nsel = nsel_s;
    // smallest key of the found bucket bf, by a pass over the keys (the gather
    // pass below does it on the way when there are keys to gather)
    auto bucket_min_pass = [&]() {
      U lm = ~(U)0;
      for (int i = tid; i < K; i += kNB) {
        const U p = mk[i];
        if (p && (int)(((p >> 1) - kmin) >> sh) == bf && (p >> 1) < lm) lm = p >> 1;
      }
      if (lm != ~(U)0) atomicMin(&bfmin_s, lm);
      __syncthreads();
    };
    if (nsel <= kCap) {
      if (nsel == 0) {
        if (bf != 0x7fffffff) bucket_min_pass();
        if (tid == 0) {
          if (bf != 0x7fffffff) {
            theta[out] = value_of(bfmin_s);
          } else {
            theta[out] = value_of(kmax);
            atomicAdd(&diag->degenerate_calib, 1ull);
          }
        }
        return;
      }
      // where each selected bucket's keys start in ascending order
      int64_t run = nsel - sel_above - my_sel;
      for (int j = 0; j < PER; ++j) {
        const int b = b0 + j;
        if ((maybe_bits >> j & 1) && b < bf) {
          fst[b] = (int32_t)run;
          run += fcnt[b];
        } else {
          fst[b] = -1;
        }
      }
      if (tid == 0) nsel_s = 0;
      __syncthreads();
      U lmin = ~(U)0;
      for (int i0 = 0; i0 < K; i0 += kNB * kUnroll) {
        U pv[kUnroll];
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
          const int i = i0 + u * kNB + tid;
          pv[u] = i < K ? mk[i] : (U)0;
        }
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
          const U p = pv[u];
          if (!p) continue;
          const int b = (int)(((p >> 1) - kmin) >> sh);
          if (fst[b] >= 0) list[atomicAdd(&nsel_s, 1)] = p;
          if (b == bf && (p >> 1) < lmin) lmin = p >> 1;
        }
      }
      if (lmin != ~(U)0) atomicMin(&bfmin_s, lmin);
      int n2 = 32;
      while (n2 < nsel) n2 <<= 1;
      for (int i = nsel + tid; i < n2; i += kNB) list[i] = ~(U)0;
      __syncthreads();
      for (int k2 = 2; k2 <= n2; k2 <<= 1) {       // bitonic sort, ascending
        for (int j2 = k2 >> 1; j2 > 0; j2 >>= 1) {
          for (int i = tid; i < n2; i += kNB) {
            const int ixj = i ^ j2;
            if (ixj > i) {
              const U a = list[i], c = list[ixj];
              if ((a > c) == ((i & k2) == 0)) {
                list[i] = c;
                list[ixj] = a;
              }
            }
          }
          __syncthreads();
        }
      }
      // inclusive healthy prefix over the sorted keys
      constexpr int PERC = kCap / kNB;
      int hs = 0;
      for (int j = 0; j < PERC; ++j) {
        const int i = tid * PERC + j;
        if (i < nsel) hs += (int)(list[i] & 1);
      }
      const int64_t h_after = block_suffix(hs, red64);
      if (tid == 0) red64[0] = h_after + hs;       // total
      __syncthreads();
      int64_t hp = red64[0] - (h_after + hs);
      __syncthreads();
      for (int j = 0; j < PERC; ++j) {
        const int i = tid * PERC + j;
        if (i < nsel) hp += (int64_t)(list[i] & 1);
        hpre[i] = (int32_t)hp;
      }
      __syncthreads();
      // exact test at the first position of every distinct value
      int best = 0x7fffffff;
      for (int i = tid; i < nsel; i += kNB) {
        const U key = list[i] >> 1;
        if (i > 0 && (list[i - 1] >> 1) == key) continue;
        const int b = (int)((key - kmin) >> sh);
        const int end = fst[b] + fcnt[b];
        const int64_t C = (int64_t)fca[b] + (end - i);
        const int64_t H = (int64_t)fha[b] + hpre[end - 1] - (i > 0 ? hpre[i - 1] : 0);
        if ((double)H >= reliability * (double)C) best = min(best, i);
      }
      best = block_min(best, red32);
      if (tid == 0) {
        if (best != 0x7fffffff) {
          theta[out] = value_of(list[best] >> 1);
        } else if (bf != 0x7fffffff) {
          theta[out] = value_of(bfmin_s);
        } else {
          theta[out] = value_of(kmax);
          atomicAdd(&diag->degenerate_calib, 1ull);
        }
      }
      return;
    }
  }
  __syncthreads();

  // ---- fallback: radix descent over the key range (many candidate keys) ----
  int32_t (*cnt)[kNB] = reinterpret_cast<int32_t (*)[kNB]>(dyn);
  int32_t (*hl)[kNB] = reinterpret_cast<int32_t (*)[kNB]>(dyn + (size_t)NL * kNB * 4);
  U (*mn)[kNB] = reinterpret_cast<U (*)[kNB]>(dyn + (size_t)NL * kNB * 8);
  auto build = [&](int l) {
    cnt[l][tid] = 0;
    hl[l][tid] = 0;
    mn[l][tid] = ~(U)0;
    __syncthreads();
    const U lo = lo_s[l], hi = hi_s[l];
    const int sh = shift_s[l];
    for (int i0 = 0; i0 < K; i0 += kNB) {
      const int i = i0 + tid;
      const U p = i < K ? mk[i] : (U)0;
      const U key = p >> 1;
      const bool in = p != 0 && key >= lo && key <= hi;
      const int b = in ? (int)((key - lo) >> sh) : -1;
      const unsigned act = __ballot_sync(0xffffffffu, in);
      if (in) {
        const unsigned grp = __match_any_sync(act, b);
        const unsigned hgrp = __ballot_sync(grp, (p & 1) != 0);
        if (lane == __ffs(grp) - 1) {
          atomicAdd(&cnt[l][b], __popc(grp));
          if (hgrp) atomicAdd(&hl[l][b], __popc(hgrp));
        }
        if (key < mn[l][b]) atomicMin(&mn[l][b], key);
      }
    }
    __syncthreads();
  };
  auto set_range = [&](int l, U lo, U hi, int64_t ca, int64_t ha) {
    int sh = 0;
    while (sh < 63 && ((hi - lo) >> sh) >= (U)kNB) ++sh;
    lo_s[l] = lo;
    hi_s[l] = hi;
    shift_s[l] = sh;
    pos_s[l] = 0;
    cab_s[l] = ca;
    hab_s[l] = ha;
  };
  if (tid == 0) set_range(0, kmin, kmax, 0, 0);
  __syncthreads();
  build(0);
  int l = 0;
  while (true) {
    const int64_t c_above = block_suffix(cnt[l][tid], red64) + cab_s[l];
    const int64_t h_above = block_suffix(hl[l][tid], red64) + hab_s[l];
    const int32_t c = cnt[l][tid], h = hl[l][tid];
    int cand = 0x7fffffff;
    int kind = 0;   // 1 = its smallest value qualifies, 2 = may contain one
    if (c > 0 && tid >= pos_s[l]) {
      if ((double)(h_above + h) >= reliability * (double)(c_above + c)) {
        kind = 1;
      } else if (shift_s[l] > 0 &&
                 (double)(h_above + h + 1) >= reliability * (double)(c_above + h)) {
        kind = 2;
      }
      if (kind) cand = tid;
    }
    const int b = block_min(cand, red32);
    if (b == 0x7fffffff) {
      if (l == 0) {
        if (tid == 0) {
          theta[out] = value_of(kmax);
          atomicAdd(&diag->degenerate_calib, 1ull);
        }
        return;
      }
      --l;
      __syncthreads();
      continue;
    }
    if (tid == b) red32[0] = kind;
    __syncthreads();
    const int kb = red32[0];
    if (kb == 1) {
      if (tid == 0) theta[out] = value_of(mn[l][b]);
      return;
    }
    if (tid == b) {
      const U lo = lo_s[l] + ((U)b << shift_s[l]);
      const U hi = lo + (((U)1 << shift_s[l]) - 1);
      pos_s[l] = b + 1;
      set_range(l + 1, lo, hi, c_above, h_above);
    }
    __syncthreads();
    ++l;
    build(l);
  }
}

}  // namespace

template <class T> void calib_ws_layout(Arena& a, int64_t elems, int n_sm, CalibWs<T>& w) {
  using U = typename KeyOf<T>::U;
  w.keys = a.take<U>((size_t)std::max<int64_t>(elems, 1));
  w.thr = a.take<int32_t>(kThrTable);
  const size_t n = (size_t)std::max(n_sm, 1);
  w.kmin = a.take<U>(n);
  w.kmax = a.take<U>(n);
  w.ncand = a.take<uint32_t>(n);
  w.n_sm = n_sm;
}

template <class T>
cudaError_t launch_calibrate(const SeriesTable<T>& tab, const T* S, const uint8_t* cls,
                             const unsigned long long* slo, double ok_frac, double reliability,
                             T* theta, CalibWs<T>& w, tre_diag* diag, cudaStream_t s) {
  using U = typename KeyOf<T>::U;
  const int n_sm = tab.n * tab.M;
  if (n_sm > w.n_sm) return cudaErrorInvalidValue;
  U* kmin = static_cast<U*>(w.kmin);
  U* kmax = static_cast<U*>(w.kmax);
  const int thr_n = std::max(kThrTable, n_sm);
  k_thr<U><<<(thr_n + 255) / 256, 256, 0, s>>>(ok_frac, w.thr, n_sm, kmin, kmax, w.ncand);
  PackPlan pp;
  pp.lg_tm = 0;
  while ((1 << pp.lg_tm) < tab.M && pp.lg_tm < 5) ++pp.lg_tm;
  pp.tm = 1 << pp.lg_tm;
  pp.lg_tk = 10 - pp.lg_tm;
  pp.tk = 1 << pp.lg_tk;
  static_assert(kPackTile == 1024, "tile of 2^10 elements");
  pp.m_tiles = (tab.M + pp.tm - 1) / pp.tm;
  int tiles = 0;
  for (int i = 0; i < tab.n; ++i) {
    pp.tile_base[i] = tiles;
    tiles += (tab.K[i] + pp.tk - 1) / pp.tk * pp.m_tiles;
  }
  pp.tile_base[tab.n] = tiles;
  const bool vec = tab.M % pp.tm == 0 && tab.M % 4 == 0 &&
                   (((uintptr_t)S | (uintptr_t)cls | (uintptr_t)slo) & 15) == 0;
  if (tiles > 0 && vec)
    k_pack_vec<T><<<tiles, kPackThreads, 0, s>>>(tab, pp, S, cls, slo, w.thr, ok_frac,
                                                 static_cast<U*>(w.keys), kmin, kmax, w.ncand);
  else if (tiles > 0)
    k_pack<T><<<tiles, kPackThreads, 0, s>>>(tab, pp, S, cls, slo, w.thr, ok_frac,
                                             static_cast<U*>(w.keys), kmin, kmax, w.ncand);
  const size_t smem = search_smem_bytes<T>();
  // the largest carveout lets two searches share an SM where their tables fit
  cudaError_t e = func_smem_once((const void*)k_search<T>, (int)smem, true);
  if (e) return e;
  k_search<T><<<tab.n * tab.M, kNB, smem, s>>>(tab, static_cast<const U*>(w.keys), kmin, kmax,
                                               w.ncand, reliability, theta, diag);
  return cudaGetLastError();
}

template void calib_ws_layout<float>(Arena&, int64_t, int, CalibWs<float>&);
template void calib_ws_layout<double>(Arena&, int64_t, int, CalibWs<double>&);
template cudaError_t launch_calibrate<float>(const SeriesTable<float>&, const float*,
                                             const uint8_t*, const unsigned long long*, double,
                                             double, float*, CalibWs<float>&, tre_diag*,
                                             cudaStream_t);
template cudaError_t launch_calibrate<double>(const SeriesTable<double>&, const double*,
                                              const uint8_t*, const unsigned long long*, double,
                                              double, double*, CalibWs<double>&, tre_diag*,
                                              cudaStream_t);

}  // namespace tre
