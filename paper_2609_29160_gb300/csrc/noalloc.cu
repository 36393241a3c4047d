// tss_score_noalloc: the scoring entry point for callers that cannot allocate
// device memory (for example code running where cudaMalloc is forbidden or
// unavailable, such as inside a host callback, a plug-in host that owns every
// allocation, or a process whose allocator is locked down). Its scratch lives in
// a fixed buffer compiled into this library instead of a caller workspace.
#include <cuda_runtime.h>

#include <cstring>
#include <mutex>

#include "internal.h"

using namespace tre;

namespace {

// Scratch of one scoring call: the Eq. 1 value of every (window, model) and the
// per-(segment, model) smoothing state, in double precision at most
// 8 * K*M + 64 * segments*M bytes plus alignment.
constexpr int64_t kMaxElems = 1 << 20;        // K * M
constexpr int64_t kMaxSegModels = 65536;      // segments * M
constexpr size_t kScratchBytes = (size_t)kMaxElems * 8 + (size_t)kMaxSegModels * 64 + 16 * 256;

// One copy per GPU that loads this library; it stays allocated until the
// process exits. In host code this name is only a host-side stand-in: kernels
// get the device address obtained with cudaGetSymbolAddress below.
static __device__ __align__(256) unsigned char g_score_scratch[kScratchBytes];

constexpr int kMaxDevices = 256;
void* g_scratch_addr[kMaxDevices];
std::mutex g_scratch_mu;

// Device address of the scratch for the current device, looked up once per
// device with that device current (the first call on a device does this; make
// it before any stream capture). Guarded for concurrent host threads. The
// address belongs to the device's current context: cudaDeviceReset loads the
// module anew and may move the buffer, so a process that resets a device must
// not call tss_score_noalloc on it afterwards (tre.h says so).
tre_status scratch_address(void** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return TRE_ECUDA;
  std::lock_guard<std::mutex> lk(g_scratch_mu);
  if (!g_scratch_addr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_score_scratch) != cudaSuccess || !p) return TRE_ECUDA;
    g_scratch_addr[dev] = p;
  }
  *out = g_scratch_addr[dev];
  return TRE_OK;
}

template <class T>
tre_status run(const tre_grid* g, const tre_counts* in, const tre_profile* p, void* S_carry,
               uint8_t* init_carry, void* S_out, void* Z_out, uint8_t* cls_out,
               int32_t* recv_out, tre_diag* diag, cudaStream_t s) {
  const int M = g->n_models, K = g->n_windows;
  SeriesTable<T> tab;
  memset(&tab, 0, sizeof(tab));
  tab.n = 1;
  tab.M = M;
  tab.K[0] = K;
  tab.win[0] = g->window_ms;
  tab.alpha[0] = (T)0.01;  // alpha is per model on the device: size segments for slow smoothing
  const int n_seg = series_segments(tab);
  const int64_t elems = (int64_t)K * M;
  Arena measure(nullptr);
  ScoreWs<T> w;
  score_ws_layout<T>(measure, M, elems, n_seg, w);
  if (elems > kMaxElems || (int64_t)n_seg * M > kMaxSegModels || measure.off > kScratchBytes)
    return TRE_ENOMEM;
  void* base = nullptr;
  tre_status st = scratch_address(&base);
  if (st != TRE_OK) return st;
  Arena a(base);
  score_ws_layout<T>(a, M, elems, n_seg, w);
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
  return e == cudaSuccess ? TRE_OK : TRE_ECUDA;
}

}  // namespace

extern "C" tre_status tss_score_noalloc(const tre_grid* grid, const tre_counts* in,
                                        const tre_profile* prof, void* S_carry,
                                        uint8_t* init_carry, void* S_out, void* Z_out,
                                        uint8_t* cls_out, int32_t* recv_out, tre_diag* diag,
                                        tre_stream stream) {
  // the same argument checks as tss_score (which additionally needs ws_bytes)
  if (!grid_ok(grid) || !counts_ok(in) || !prof_ok(prof, true) || !diag) return TRE_EINVAL;
  if (!S_out || !Z_out || !cls_out || (!S_carry) != (!init_carry)) return TRE_EINVAL;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (prof->dtype == TRE_F32)
    return run<float>(grid, in, prof, S_carry, init_carry, S_out, Z_out, cls_out, recv_out, diag,
                      s);
  return run<double>(grid, in, prof, S_carry, init_carry, S_out, Z_out, cls_out, recv_out, diag,
                     s);
}
