// C ABI of the library (include/molt.h): argument validation, workspace
// layout, TMA tensor maps and the launch sequence of each entry point.
#include <atomic>
#include <cstdint>
#include <cstring>
#include <mutex>
#include <string>

#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include "../../include/molt.h"
#include "molt_internal.cuh"
#include "ptx.cuh"

// Per-device status word set by the kernels (MOLT_DEV_* bits).
__device__ unsigned g_molt_status_word;

namespace molt {

std::atomic<unsigned long long> g_kernel_launches{0};
void note_launches(int n) { g_kernel_launches.fetch_add(static_cast<unsigned long long>(n), std::memory_order_relaxed); }

namespace {

thread_local std::string t_last_error;

// benchmark timing hook (molt_set_timing_events)
thread_local cudaEvent_t* t_ev_start = nullptr;
thread_local cudaEvent_t* t_ev_stop = nullptr;
thread_local int t_ev_n = 0;

inline void ev_start(int k, cudaStream_t s) {
  if (k < t_ev_n && t_ev_start && t_ev_start[k]) cudaEventRecord(t_ev_start[k], s);
}
inline void ev_stop(int k, cudaStream_t s) {
  if (k < t_ev_n && t_ev_stop && t_ev_stop[k]) cudaEventRecord(t_ev_stop[k], s);
}

molt_status fail(molt_status s, const std::string& msg) {
  t_last_error = msg;
  return s;
}
molt_status cuda_fail(cudaError_t e, const char* what) {
  t_last_error = std::string(what) + ": " + cudaGetErrorString(e);
  return MOLT_ERR_CUDA;
}

constexpr int kMaxDevices = 64;
struct DeviceInfo {
  std::once_flag once;
  int n_sm = 0;
  unsigned* status = nullptr;
  cudaError_t err = cudaSuccess;
};
DeviceInfo g_dev[kMaxDevices];

// SM count and the address of the status word on the current device
const DeviceInfo* device_info(molt_status* st) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) {
    *st = cuda_fail(e, "cudaGetDevice");
    return nullptr;
  }
  if (dev < 0 || dev >= kMaxDevices) {
    *st = fail(MOLT_ERR_CUDA, "device ordinal out of range");
    return nullptr;
  }
  DeviceInfo& d = g_dev[dev];
  std::call_once(d.once, [&d, dev]() {
    d.err = cudaDeviceGetAttribute(&d.n_sm, cudaDevAttrMultiProcessorCount, dev);
    if (d.err == cudaSuccess) d.err = cudaGetSymbolAddress(reinterpret_cast<void**>(&d.status), g_molt_status_word);
  });
  if (d.err != cudaSuccess) {
    *st = cuda_fail(d.err, "device query");
    return nullptr;
  }
  *st = MOLT_OK;
  return &d;
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static std::once_flag once;
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  std::call_once(once, []() {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// 2-D row-major tensor map: `rows` x `cols` elements, box `box_cols` x `box_rows`
molt_status make_tmap(CUtensorMap* m, CUtensorMapDataType dt, int elem_bytes, const void* base, uint64_t rows,
                      uint64_t cols, uint32_t box_cols, uint32_t box_rows,
                      CUtensorMapSwizzle swizzle = CU_TENSOR_MAP_SWIZZLE_128B) {
  auto fn = encode_fn();
  if (!fn) return fail(MOLT_ERR_CUDA, "cuTensorMapEncodeTiled entry point unavailable");
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * static_cast<uint64_t>(elem_bytes)};
  cuuint32_t box[2] = {box_cols, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, dt, 2, const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(MOLT_ERR_CUDA, "cuTensorMapEncodeTiled failed (" + std::to_string((int)r) + ")");
  return MOLT_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

inline size_t up256(size_t x) { return (x + 255) & ~size_t(255); }

int64_t round_tiles(int64_t T) { return ((T + kTileM - 1) / kTileM) * kTileM; }

// vocab splits of the forward pass: enough units for ~16 waves of CTAs when
// every row is active, never more splits than vocab tiles
int choose_splits(int64_t Tcap, int64_t V, int n_sm) {
  const int64_t n_vt = (V + kFwdBN - 1) / kFwdBN;
  const int64_t n_mt = Tcap / kTileM;
  int64_t S = (16 * static_cast<int64_t>(n_sm) + n_mt - 1) / n_mt;
  if (S < 1) S = 1;
  if (S > n_vt) S = n_vt;
  return static_cast<int>(S);
}

struct Layout {
  size_t counts, row_map, pos, tok_p, b_p, adv_p, h_p, part, zx, lse, coef, tile_flag, tile_list, red, dh32, turns;
  size_t lp_p, ent_p, ecoef, mu, gate_p;
  size_t live_map, live_of, h_l, tok_l, lse_l, coef_l, ecoef_l, mu_l, total;
};

constexpr size_t kNoRegion = ~size_t(0);   // a Layout region that is not allocated

// turn counters of the deterministic schedule: an abort word (padded to 64
// words), then [token quads, H jobs, 32] for dhidden and [vocab blocks, H jobs,
// 32] for dW
struct TurnLayout {
  int64_t dh_off, dw_off, words;
};
TurnLayout turn_layout(int64_t Tcap, int64_t H, int64_t V) {
  const int64_t n_jobs = (H + 255) / 256;
  const int64_t n_quads = (Tcap / kTileM + 3) / 4;
  const int64_t n_blocks = (V + 511) / 512;
  TurnLayout t;
  t.dh_off = 64;
  t.dw_off = t.dh_off + n_quads * n_jobs * 32;
  t.words = t.dw_off + n_blocks * n_jobs * 32;
  return t;
}

Layout layout(int64_t T, int64_t H, int64_t V, int S, bool with_bwd, bool det = false) {
  const int64_t Tcap = round_tiles(T);
  const int64_t ntile = Tcap / kTileM;
  Layout L{};
  size_t o = 0;
  auto take = [&o](size_t bytes) {
    size_t r = o;
    o += up256(bytes);
    return r;
  };
  L.counts = take(64);
  L.row_map = take(T * 4);
  L.pos = take(T * 4);
  L.tok_p = take(Tcap * 4);
  L.b_p = take(Tcap * 4);
  L.adv_p = take(Tcap * 4);
  L.h_p = take(Tcap * H * 2);
  L.part = take(static_cast<size_t>(S) * Tcap * 16);
  L.zx = take(Tcap * 4);
  L.lse = take(Tcap * 4);
  L.coef = take(Tcap * 4);
  L.tile_flag = take(ntile * 4);
  L.tile_list = take(ntile * 4);
  L.red = take(ntile * kRedSlots * 8);
  L.dh32 = with_bwd ? take(static_cast<size_t>(Tcap) * H * 4) : o;
  L.turns = (with_bwd && det) ? take(static_cast<size_t>(turn_layout(Tcap, H, V).words) * 4) : kNoRegion;
  L.lp_p = with_bwd ? take(Tcap * 4) : o;
  L.ent_p = with_bwd ? take(Tcap * 4) : o;
  L.ecoef = with_bwd ? take(Tcap * 4) : o;
  L.mu = with_bwd ? take(Tcap * 4) : o;
  L.gate_p = with_bwd ? take(Tcap) : o;
  L.live_map = with_bwd ? take(Tcap * 4) : o;
  L.live_of = with_bwd ? take(Tcap * 4) : o;
  L.h_l = with_bwd ? take(Tcap * H * 2) : o;
  L.tok_l = with_bwd ? take(Tcap * 4) : o;
  L.lse_l = with_bwd ? take(Tcap * 4) : o;
  L.coef_l = with_bwd ? take(Tcap * 4) : o;
  L.ecoef_l = with_bwd ? take(Tcap * 4) : o;
  L.mu_l = with_bwd ? take(Tcap * 4) : o;
  L.total = o + 256;   // slack for aligning the caller's base pointer
  return L;
}

// Workspace of the shard merge (molt_vp_loss): the active-row compaction,
// per-row m c / D, the tile partial sums and finalize's row list.
Layout vp_loss_layout(int64_t T) {
  const int64_t Tcap = round_tiles(T);
  const int64_t ntile = Tcap / kTileM;
  Layout L{};
  size_t o = 0;
  auto take = [&o](size_t bytes) {
    size_t r = o;
    o += up256(bytes);
    return r;
  };
  L.counts = take(64);
  L.row_map = take(T * 4);
  L.pos = take(T * 4);
  L.coef = take(Tcap * 4);
  L.tile_flag = take(ntile * 4);
  L.tile_list = take(ntile * 4);
  L.red = take(ntile * kRedSlots * 8);
  L.live_map = take(Tcap * 4);
  L.live_of = take(Tcap * 4);
  L.tok_p = L.b_p = L.adv_p = L.h_p = L.part = L.zx = L.lse = L.dh32 = L.lp_p = L.ent_p = L.ecoef = L.mu = L.gate_p =
      L.h_l = L.tok_l = L.lse_l = L.coef_l = L.ecoef_l = L.mu_l = o;
  L.turns = kNoRegion;
  L.total = o + 256;
  return L;
}

// Workspace of one shard's backward (molt_vp_backward): the rows with a
// gradient, packed (hidden, token, lse, m c / D), and the fp32 dhidden
// accumulator by backward row.
Layout vp_backward_layout(int64_t T, int64_t H) {
  const int64_t Tcap = round_tiles(T);
  const int64_t ntile = Tcap / kTileM;
  Layout L{};
  size_t o = 0;
  auto take = [&o](size_t bytes) {
    size_t r = o;
    o += up256(bytes);
    return r;
  };
  L.counts = take(64);
  L.tile_list = take(ntile * 4);
  L.live_map = take(Tcap * 4);
  L.live_of = take(Tcap * 4);
  L.h_l = take(Tcap * H * 2);
  L.tok_l = take(Tcap * 4);
  L.lse_l = take(Tcap * 4);
  L.coef_l = take(Tcap * 4);
  L.dh32 = take(static_cast<size_t>(Tcap) * H * 4);
  L.row_map = L.pos = L.tok_p = L.b_p = L.adv_p = L.h_p = L.part = L.zx = L.lse = L.coef = L.tile_flag = L.red =
      L.lp_p = L.ent_p = L.ecoef = L.mu = L.gate_p = L.ecoef_l = L.mu_l = o;
  L.turns = kNoRegion;
  L.total = o + 256;
  return L;
}

Workspace carve(void* base, const Layout& L) {
  uint8_t* p = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(base) + 255) & ~uintptr_t(255));
  Workspace w{};
  w.counts = reinterpret_cast<int32_t*>(p + L.counts);
  w.row_map = reinterpret_cast<int32_t*>(p + L.row_map);
  w.pos_of_row = reinterpret_cast<int32_t*>(p + L.pos);
  w.tok_p = reinterpret_cast<int32_t*>(p + L.tok_p);
  w.b_p = reinterpret_cast<float*>(p + L.b_p);
  w.adv_p = reinterpret_cast<float*>(p + L.adv_p);
  w.h_p = reinterpret_cast<uint16_t*>(p + L.h_p);
  w.part = reinterpret_cast<float4*>(p + L.part);
  w.zx = reinterpret_cast<float*>(p + L.zx);
  w.lse = reinterpret_cast<float*>(p + L.lse);
  w.coef = reinterpret_cast<float*>(p + L.coef);
  w.tile_flag = reinterpret_cast<int32_t*>(p + L.tile_flag);
  w.tile_list = reinterpret_cast<int32_t*>(p + L.tile_list);
  w.red = reinterpret_cast<double*>(p + L.red);
  w.dh32 = reinterpret_cast<float*>(p + L.dh32);
  w.turns = L.turns != kNoRegion ? reinterpret_cast<uint32_t*>(p + L.turns) : nullptr;
  w.lp_p = reinterpret_cast<float*>(p + L.lp_p);
  w.ent_p = reinterpret_cast<float*>(p + L.ent_p);
  w.ecoef = reinterpret_cast<float*>(p + L.ecoef);
  w.mu = reinterpret_cast<float*>(p + L.mu);
  w.gate_p = p + L.gate_p;
  w.live_map = reinterpret_cast<int32_t*>(p + L.live_map);
  w.live_of = reinterpret_cast<int32_t*>(p + L.live_of);
  w.h_l = reinterpret_cast<uint16_t*>(p + L.h_l);
  w.tok_l = reinterpret_cast<int32_t*>(p + L.tok_l);
  w.lse_l = reinterpret_cast<float*>(p + L.lse_l);
  w.coef_l = reinterpret_cast<float*>(p + L.coef_l);
  w.ecoef_l = reinterpret_cast<float*>(p + L.ecoef_l);
  w.mu_l = reinterpret_cast<float*>(p + L.mu_l);
  return w;
}

molt_status check_shape(int64_t T, int64_t H, int64_t V) {
  if (T < 0 || V < 1 || H < 1) return fail(MOLT_ERR_INVALID_ARG, "sizes must satisfy T >= 0, H >= 1, V >= 1");
  if (H % 64 != 0) return fail(MOLT_ERR_UNSUPPORTED_SHAPE, "H must be a multiple of 64");
  if (T >= (int64_t(1) << 31) - kTileM || V >= (int64_t(1) << 31) || H > 65536)
    return fail(MOLT_ERR_UNSUPPORTED_SHAPE, "T and V must be below 2^31 and H at most 65536");
  return MOLT_OK;
}

// Scratch memory of one call: the caller's buffer, or a stream-ordered allocation.
struct Scratch {
  void* ptr = nullptr;
  bool owned = false;
  cudaStream_t s = nullptr;
  ~Scratch() {
    if (owned && ptr) cudaFreeAsync(ptr, s);
  }
};

// Vocab split of the raster backward (see the side lanes below): the first
// Vq columns go to the cluster kernel, the rest to the single-CTA kernel on the
// `spare` SMs.  Vq is the multiple of 512 that minimises the later of the two
// kernels' predicted finish times, in units per cluster (512 x 512 units over
// `clusters`) against units per spare SM (128 x 256 units, measured at 0.84 of
// a cluster unit's time); T stands in for the active rows.  Returns V for no
// split.
int64_t choose_vocab_split(int64_t T, int64_t V, int clusters, int spare) {
  if (spare <= 0 || clusters <= 0 || V < 16 * 512) return V;
  const int64_t n_t = (T + kTileM - 1) / kTileM, n_tq = (n_t + 3) / 4;
  auto cdiv = [](int64_t a, int64_t b) { return (a + b - 1) / b; };
  auto finish = [&](int64_t vq) {
    const double quad = static_cast<double>(cdiv(cdiv(vq, 512) * n_tq, clusters));
    const double side = vq < V ? 0.84 * static_cast<double>(cdiv(cdiv(V - vq, kBwdBV) * n_t, spare)) : 0.0;
    return quad > side ? quad : side;
  };
  int64_t best = V;
  double best_t = finish(V) * 0.995;   // a split must gain at least 0.5 %
  for (int64_t vq = (V - 1) / 512 * 512; vq >= V - V / 8 && vq > 0; vq -= 512) {
    const double t = finish(vq);
    if (t < best_t) {
      best_t = t;
      best = vq;
    }
  }
  return best;
}

molt_status get_scratch(Scratch& sc, void* ws, size_t ws_bytes, size_t need, cudaStream_t s) {
  sc.s = s;
  if (ws) {
    if (ws_bytes < need)
      return fail(MOLT_ERR_WORKSPACE, "workspace of " + std::to_string(ws_bytes) + " bytes, need " +
                                          std::to_string(need));
    sc.ptr = ws;
    return MOLT_OK;
  }
  cudaError_t e = cudaMallocAsync(&sc.ptr, need, s);
  if (e != cudaSuccess) {
    cudaGetLastError();
    sc.ptr = nullptr;
    return fail(MOLT_ERR_NO_MEMORY, std::string("cudaMallocAsync: ") + cudaGetErrorString(e));
  }
  sc.owned = true;
  return MOLT_OK;
}

// Side lanes of the loss call.  Clusters of four leave the SMs that cannot
// hold a whole cluster idle (8 of 152 on a GB300); the single-CTA backward runs
// there concurrently on a slice of the vocabulary.  The backward's reduce-add
// targets are zeroed on the same lane while the forward runs (the memset
// kernels fit beside the forward's one CTA per SM).  One low-priority side
// stream and fork / join / zeroed events per (device, caller stream), created
// on first use and kept for the life of the process; at most kMaxSideLanes of
// them (further streams run without the split and zero in line).
struct SideLane {
  int dev = -1;
  cudaStream_t caller = nullptr;
  cudaStream_t side = nullptr;
  cudaEvent_t fork = nullptr, join = nullptr, zeroed = nullptr;
};
constexpr int kMaxSideLanes = 64;
std::mutex g_side_mu;
SideLane g_side[kMaxSideLanes];
int g_side_n = 0;

// the side lane of `caller` on the current device, or nullptr (no lane: run
// the cluster kernel alone)
const SideLane* side_lane(cudaStream_t caller) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  std::lock_guard<std::mutex> lk(g_side_mu);
  for (int i = 0; i < g_side_n; ++i)
    if (g_side[i].dev == dev && g_side[i].caller == caller) return &g_side[i];
  if (g_side_n == kMaxSideLanes) return nullptr;
  // no new streams or events while the caller's stream is being captured
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(caller, &cap) != cudaSuccess || cap != cudaStreamCaptureStatusNone) {
    cudaGetLastError();
    return nullptr;
  }
  SideLane l;
  l.dev = dev;
  l.caller = caller;
  int least = 0, greatest = 0;
  bool ok = cudaDeviceGetStreamPriorityRange(&least, &greatest) == cudaSuccess &&
            cudaStreamCreateWithPriority(&l.side, cudaStreamNonBlocking, least) == cudaSuccess;
  ok = ok && cudaEventCreateWithFlags(&l.fork, cudaEventDisableTiming) == cudaSuccess;
  ok = ok && cudaEventCreateWithFlags(&l.join, cudaEventDisableTiming) == cudaSuccess;
  ok = ok && cudaEventCreateWithFlags(&l.zeroed, cudaEventDisableTiming) == cudaSuccess;
  if (!ok) {
    cudaGetLastError();
    if (l.zeroed) cudaEventDestroy(l.zeroed);
    if (l.join) cudaEventDestroy(l.join);
    if (l.fork) cudaEventDestroy(l.fork);
    if (l.side) cudaStreamDestroy(l.side);
    return nullptr;
  }
  g_side[g_side_n] = l;
  return &g_side[g_side_n++];
}

// Makes `stream` wait for a side lane's zeroing (its `zeroed` event) once:
// by join(), or when it goes out of scope on an early return (declared after
// the call's Scratch, so before the workspace is released).
struct ZeroJoin {
  const SideLane* lane = nullptr;
  cudaStream_t stream = nullptr;
  bool pending = false;
  cudaError_t join() {
    if (!pending) return cudaSuccess;
    pending = false;
    return cudaStreamWaitEvent(stream, lane->zeroed, 0);
  }
  ~ZeroJoin() {
    if (join() != cudaSuccess) cudaGetLastError();
  }
};

#define MOLT_CUDA(call, what)                        \
  do {                                               \
    cudaError_t e_ = (call);                         \
    if (e_ != cudaSuccess) return cuda_fail(e_, what); \
  } while (0)

// a kernel launch: as MOLT_CUDA, and counted on success
#define MOLT_LAUNCH(call, what)                        \
  do {                                                 \
    cudaError_t e_ = (call);                           \
    if (e_ != cudaSuccess) return cuda_fail(e_, what); \
    note_launches(1);                                  \
  } while (0)

#define MOLT_TRY(call)                   \
  do {                                   \
    molt_status s_ = (call);             \
    if (s_ != MOLT_OK) return s_;        \
  } while (0)

// Shared front half of both LM-head calls: compaction, packed gather and the
// forward kernel (tensor maps already encoded by the caller).
// tok_shift is subtracted from the tokens (a vocabulary shard's first column).
molt_status run_forward(const DeviceInfo* di, const uint16_t* hidden, const int32_t* tokens, const uint8_t* mask,
                        const float* b, const float* adv, int64_t T, int64_t H, int64_t V, int S,
                        const Workspace& w, const CUtensorMap& tm_h, const CUtensorMap& tm_w, cudaStream_t s,
                        int tok_shift = 0) {
  const int64_t Tcap = round_tiles(T);
  ev_start(0, s);
  MOLT_LAUNCH(launch_compact(mask, static_cast<int>(T), w, s), "compact");
  MOLT_LAUNCH(launch_gather(hidden, tokens, b, adv, static_cast<int>(T), static_cast<int>(Tcap), static_cast<int>(H),
                          w, di->n_sm, s, tok_shift),
            "gather");
  ev_stop(0, s);
  FwdArgs fa{};
  fa.tok_p = w.tok_p;
  fa.counts = w.counts;
  fa.rows_cap = static_cast<int>(Tcap);
  fa.V = static_cast<int>(V);
  fa.H = static_cast<int>(H);
  fa.n_split = S;
  fa.n_vtiles = static_cast<int>((V + kFwdBN - 1) / kFwdBN);
  fa.part = w.part;
  fa.zx = w.zx;
  fa.err = di->status;
  ev_start(1, s);
  MOLT_LAUNCH(launch_lmhead_fwd(tm_h, tm_w, fa, di->n_sm, s), "lmhead forward");
  ev_stop(1, s);
  return MOLT_OK;
}

// Zero the backward's fp32 reduce-add targets on stream s: the dhidden
// accumulator, the deterministic schedule's turn counters and, unless the call
// accumulates into it, dW.
molt_status zero_backward_targets(const Workspace& w, int64_t T, int64_t H, int64_t V, bool det, float* dW_out,
                                  int accumulate_dW, cudaStream_t s) {
  const int64_t Tcap = round_tiles(T);
  MOLT_CUDA(cudaMemsetAsync(w.dh32, 0, static_cast<size_t>(Tcap) * H * sizeof(float), s), "memset dh32");
  if (det) {
    const TurnLayout tl = turn_layout(Tcap, H, V);
    MOLT_CUDA(cudaMemsetAsync(w.turns, 0, static_cast<size_t>(tl.words) * 4, s), "memset turns");
  }
  if (!accumulate_dW) MOLT_CUDA(cudaMemsetAsync(dW_out, 0, static_cast<size_t>(V) * H * sizeof(float), s), "memset dW");
  return MOLT_OK;
}

// Back half of the loss calls: the backward kernels over the rows with a
// gradient, packed in w (h_l, tok_l, lse_l, coef_l and, with an entropy bonus,
// ecoef_l and mu_l; counts[1] tiles of them), reduce-adding into the fp32
// accumulator w.dh32 (by backward row) and dW (zeroed first unless
// accumulate_dW; `zeroed`: the caller has zeroed them already, ordered before
// this point on `stream`).  det: the deterministic schedule on n_det clusters.
molt_status run_backward(const DeviceInfo* di, const uint16_t* W, int64_t T, int64_t H, int64_t V,
                         const Workspace& w, bool det, int n_det, bool with_ecoef, float* dW_out, int accumulate_dW,
                         bool zeroed, cudaStream_t stream) {
  const int64_t Tcap = round_tiles(T);
  const bool pair_bwd = (H % 128) == 0;   // the cluster backward
  CUtensorMap tm_wz, tm_wn, tm_dh, tm_dw;
  MOLT_TRY(make_tmap(&tm_wz, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, W, V, H, kBK, pair_bwd ? 128 : kBwdBV));
  MOLT_TRY(make_tmap(&tm_wn, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, W, V, H, kBK, 64));
  // the backward reads the rows with a gradient, packed again into h_l:
  // 128-row boxes for the single-CTA kernel, 64-byte-swizzled K = 32 boxes of
  // h and W for the logit recompute on CTA pairs, and 64-row boxes of h (a dW
  // stage of the cluster backward is 64 token rows)
  CUtensorMap tm_hb, tm_hz, tm_wz32, tm_h64;
  MOLT_TRY(make_tmap(&tm_hb, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, w.h_l, Tcap, H, kBK, kTileM));
  MOLT_TRY(make_tmap(&tm_hz, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, w.h_l, Tcap, H, 32, kTileM,
                     CU_TENSOR_MAP_SWIZZLE_64B));
  MOLT_TRY(make_tmap(&tm_wz32, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, W, V, H, 32, 128, CU_TENSOR_MAP_SWIZZLE_64B));
  MOLT_TRY(make_tmap(&tm_h64, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, w.h_l, Tcap, H, kBK, 64));
  MOLT_TRY(make_tmap(&tm_dh, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, w.dh32, Tcap, H, 32, 32));
  MOLT_TRY(make_tmap(&tm_dw, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, dW_out, V, H, 32, 32));
  if (!zeroed) MOLT_TRY(zero_backward_targets(w, T, H, V, det, dW_out, accumulate_dW, stream));
  const TurnLayout tl = turn_layout(Tcap, H, V);
  BwdArgs ba{};
  ba.tok_p = w.tok_l;
  ba.lse = w.lse_l;
  ba.coef = w.coef_l;
  ba.counts = w.counts;
  ba.tile_list = w.tile_list;
  ba.V = static_cast<int>(V);
  ba.H = static_cast<int>(H);
  ba.n_vchunks = static_cast<int>((V + kBwdBV - 1) / kBwdBV);
  ba.tile_group = pair_bwd ? 4 : 16;
  ba.dh32 = w.dh32;
  ba.dW = dW_out;
  ba.det_clusters = n_det;
  if (det) {
    ba.det_abort = w.turns;
    ba.det_dh_turns = w.turns + tl.dh_off;
    ba.det_dw_turns = w.turns + tl.dw_off;
  }
  if (with_ecoef) {
    ba.ecoef = w.ecoef_l;
    ba.mu = w.mu_l;
  }
  ba.err = di->status;
  ev_start(3, stream);
  if (pair_bwd) {
    // vocab split with the single-CTA kernel on the SMs no cluster can use
    // (raster schedule only: the deterministic order needs every vocab block
    // reduced by its owner clusters)
    const int clusters = lmhead_bwd_quad_clusters(di->n_sm);
    const int spare = di->n_sm - 4 * clusters;
    int64_t Vq = V;
    const SideLane* lane = nullptr;
    if (!det) {
      const int64_t vq = choose_vocab_split(T, V, clusters, spare);
      if (vq < V && (lane = side_lane(stream)) != nullptr) Vq = vq;
    }
    if (Vq < V) {
      CUtensorMap tm_wz256;
      MOLT_TRY(make_tmap(&tm_wz256, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, W, V, H, kBK, kBwdBV));
      BwdArgs bq = ba;
      bq.V = static_cast<int>(Vq);   // columns from Vq on count as padding for the cluster kernel
      BwdArgs bs = ba;
      bs.vc_begin = static_cast<int>(Vq / kBwdBV);
      bs.n_vchunks = static_cast<int>((V - Vq + kBwdBV - 1) / kBwdBV);
      bs.tile_group = 16;
      // the cluster kernel is enqueued first so that its clusters take their
      // SMs before the side kernel's CTAs fill the rest
      MOLT_CUDA(cudaEventRecord(lane->fork, stream), "backward fork");
      MOLT_LAUNCH(launch_lmhead_bwd_quad(tm_hz, tm_wz32, tm_h64, tm_wn, tm_dh, tm_dw, bq, di->n_sm, stream),
                "lmhead backward");
      MOLT_CUDA(cudaStreamWaitEvent(lane->side, lane->fork, 0), "backward fork");
      // the join is made whatever the side launch returned, so that nothing on
      // the caller's stream (the workspace release included) can overtake it
      const cudaError_t e_side = launch_lmhead_bwd(tm_hb, tm_wz256, tm_wn, tm_dh, tm_dw, bs, spare, lane->side);
      if (e_side == cudaSuccess) note_launches(1);
      cudaError_t e_join = cudaEventRecord(lane->join, lane->side);
      if (e_join == cudaSuccess) e_join = cudaStreamWaitEvent(stream, lane->join, 0);
      if (e_side != cudaSuccess) return cuda_fail(e_side, "lmhead backward (side)");
      if (e_join != cudaSuccess) return cuda_fail(e_join, "backward join");
    } else {
      MOLT_LAUNCH(launch_lmhead_bwd_quad(tm_hz, tm_wz32, tm_h64, tm_wn, tm_dh, tm_dw, ba, di->n_sm, stream),
                "lmhead backward");
    }
  } else
    MOLT_LAUNCH(launch_lmhead_bwd(tm_hb, tm_wz, tm_wn, tm_dh, tm_dw, ba, di->n_sm, stream), "lmhead backward");
  ev_stop(3, stream);
  return MOLT_OK;
}

// Both loss entry points.  opts == nullptr runs the plain clipped surrogate
// (one merge kernel computes the loss rows); otherwise the merge only writes
// the packed log-probs and entropies, the sequence gate runs on them, and a
// second row kernel forms the extended loss and the backward coefficients.
molt_status policy_loss_impl(const uint16_t* hidden, const uint16_t* W, const int32_t* tokens,
                             const float* behavior_logp, const float* adv, const uint8_t* mask, int64_t T,
                             int64_t H, int64_t V, float clip_lo, float clip_hi, double denom,
                             const molt_loss_options* opts, float* loss_out, uint16_t* dhidden_out, float* dW_out,
                             int accumulate_dW, float* logp_out, float* entropy_out, float* token_loss_out,
                             molt_stats* stats_out, molt_stats_ex* stats_ex_out, void* workspace,
                             size_t workspace_bytes, cudaStream_t stream) {
  MOLT_TRY(check_shape(T, H, V));
  if (!hidden || !W || !tokens || !behavior_logp || !adv || !loss_out || !dhidden_out || !dW_out)
    return fail(MOLT_ERR_INVALID_ARG, "null pointer");
  if (!aligned16(hidden) || !aligned16(W) || !aligned16(dhidden_out) || !aligned16(dW_out))
    return fail(MOLT_ERR_INVALID_ARG, "hidden, W, dhidden and dW must be 16-byte aligned");
  if (!(clip_lo >= 0.f && clip_lo < 1.f) || !(clip_hi >= 0.f) || clip_hi != clip_hi || clip_hi > 1e30f)
    return fail(MOLT_ERR_INVALID_ARG, "clip bounds must satisfy 0 <= clip_lo < 1 and clip_hi >= 0");
  if (denom != denom) return fail(MOLT_ERR_INVALID_ARG, "denom is NaN");
  LossEx ex{};
  if (opts) {
    ex.kl_coef = opts->kl_coef;
    ex.entropy_coef = opts->entropy_coef;
    ex.ref_logp = opts->ref_logp;
    ex.seq = opts->seq_of_token;
    ex.gate_lo = opts->gate_lo;
    ex.gate_hi = opts->gate_hi;
    if (!(ex.kl_coef >= 0.f) || ex.kl_coef > 1e30f) return fail(MOLT_ERR_INVALID_ARG, "kl_coef must be finite and >= 0");
    if (ex.kl_coef != 0.f && !ex.ref_logp) return fail(MOLT_ERR_INVALID_ARG, "kl_coef > 0 needs ref_logp");
    if (!(ex.entropy_coef >= -1e30f && ex.entropy_coef <= 1e30f))
      return fail(MOLT_ERR_INVALID_ARG, "entropy_coef must be finite");
    if (ex.seq && !(ex.gate_lo >= 0.0 && ex.gate_hi >= ex.gate_lo))
      return fail(MOLT_ERR_INVALID_ARG, "the gate band must satisfy 0 <= gate_lo <= gate_hi");
  }
  const bool det = opts && opts->deterministic;
  if (det && H % 128 != 0) return fail(MOLT_ERR_UNSUPPORTED_SHAPE, "deterministic mode needs H % 128 == 0");
  molt_status st;
  const DeviceInfo* di = device_info(&st);
  if (!di) return st;
  if (T == 0) {
    // nothing to compute: loss 0, stats zero, dW untouched or zeroed
    MOLT_CUDA(cudaMemsetAsync(loss_out, 0, sizeof(float), stream), "memset loss");
    if (!accumulate_dW) MOLT_CUDA(cudaMemsetAsync(dW_out, 0, V * H * sizeof(float), stream), "memset dW");
    if (stats_out) MOLT_CUDA(cudaMemsetAsync(stats_out, 0, sizeof(molt_stats), stream), "memset stats");
    if (stats_ex_out) MOLT_CUDA(cudaMemsetAsync(stats_ex_out, 0, sizeof(molt_stats_ex), stream), "memset stats");
    return MOLT_OK;
  }
  const int64_t Tcap = round_tiles(T);
  const int S = choose_splits(Tcap, V, di->n_sm);
  // deterministic schedule: n_det clusters (a multiple of 4), all resident at
  // once, whose reduce-adds take turns
  int n_det = det ? lmhead_bwd_quad_det_clusters(di->n_sm) : 0;
  if (det && n_det < 4) return fail(MOLT_ERR_UNSUPPORTED_SHAPE, "deterministic mode needs 4 clusters of 4 CTAs");
  if (det && opts->det_clusters != 0) {
    // fewer clusters (a multiple of 4); the results do not depend on the count
    const int want = opts->det_clusters;
    if (want < 4 || want % 4 != 0 || want > n_det)
      return fail(MOLT_ERR_INVALID_ARG,
                  "det_clusters must be 0 or a multiple of 4 from 4 to " + std::to_string(n_det));
    n_det = want;
  }
  const Layout L = layout(T, H, V, S, true, det);
  Scratch sc;
  MOLT_TRY(get_scratch(sc, workspace, workspace_bytes, L.total, stream));
  const Workspace w = carve(sc.ptr, L);
  CUtensorMap tm_h, tm_w;
  MOLT_TRY(make_tmap(&tm_h, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, w.h_p, Tcap, H, kBK, kTileM));
  MOLT_TRY(make_tmap(&tm_w, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, W, V, H, kBK, kFwdBN));
  // the backward's targets are zeroed on the side lane while the forward runs;
  // the caller's stream waits for them before the backward, or on any early
  // return before the workspace is released
  ZeroJoin zj;
  if (const SideLane* zl = side_lane(stream)) {
    MOLT_CUDA(cudaEventRecord(zl->fork, stream), "zero fork");
    MOLT_CUDA(cudaStreamWaitEvent(zl->side, zl->fork, 0), "zero fork");
    const molt_status zs = zero_backward_targets(w, T, H, V, det, dW_out, accumulate_dW, zl->side);
    const cudaError_t e = cudaEventRecord(zl->zeroed, zl->side);
    if (e != cudaSuccess) {
      cudaStreamSynchronize(zl->side);
      cudaGetLastError();
      return cuda_fail(e, "zero join");
    }
    zj.lane = zl;
    zj.stream = stream;
    zj.pending = true;
    if (zs != MOLT_OK) return zs;
  }
  MOLT_TRY(run_forward(di, hidden, tokens, mask, behavior_logp, adv, T, H, V, S, w, tm_h, tm_w, stream));
  if (logp_out) MOLT_CUDA(cudaMemsetAsync(logp_out, 0, T * sizeof(float), stream), "memset logp");
  if (entropy_out) MOLT_CUDA(cudaMemsetAsync(entropy_out, 0, T * sizeof(float), stream), "memset entropy");
  if (token_loss_out) MOLT_CUDA(cudaMemsetAsync(token_loss_out, 0, T * sizeof(float), stream), "memset token loss");
  ev_start(2, stream);
  if (opts) {
    MOLT_LAUNCH(launch_merge_stats_ex(static_cast<int>(Tcap), static_cast<int>(V), S, w, logp_out, entropy_out,
                                    di->status, stream),
              "merge");
    MOLT_LAUNCH(launch_seq_gate(static_cast<int>(T), static_cast<int>(Tcap), ex, w, di->status, stream), "gate");
    MOLT_LAUNCH(launch_loss_rows_ex(static_cast<int>(Tcap), denom, clip_lo, clip_hi, ex, w, token_loss_out, stream),
              "loss rows");
  } else {
    MOLT_LAUNCH(launch_merge(true, static_cast<int>(Tcap), static_cast<int>(V), S, denom, clip_lo, clip_hi, w,
                           logp_out, entropy_out, token_loss_out, di->status, stream),
              "merge");
  }
  // rows whose gradient coefficient is 0 (masked out already; clipped, A = 0,
  // rejected) are left out of the backward
  const bool with_ecoef = opts && ex.entropy_coef != 0.f;
  MOLT_LAUNCH(launch_finalize(static_cast<int>(Tcap), denom, with_ecoef, w, loss_out, stats_out, stats_ex_out,
                              di->status, stream),
              "finalize");
  MOLT_LAUNCH(launch_live_gather(static_cast<int>(H), with_ecoef, w, di->n_sm, stream), "live gather");
  ev_stop(2, stream);
  MOLT_CUDA(zj.join(), "zero join");
  MOLT_TRY(run_backward(di, W, T, H, V, w, det, n_det, with_ecoef, dW_out, accumulate_dW, zj.lane != nullptr, stream));
  ev_start(4, stream);
  MOLT_LAUNCH(launch_cast_dh(w, static_cast<int>(T), static_cast<int>(H), dhidden_out, di->n_sm, stream), "cast dh");
  ev_stop(4, stream);
  return MOLT_OK;
}

}  // namespace

void set_last_error(const std::string& msg) { t_last_error = msg; }

void timing_event(int k, bool stop, cudaStream_t s) {
  if (stop)
    ev_stop(k, s);
  else
    ev_start(k, s);
}

unsigned* device_status_word(molt_status* st) {
  const DeviceInfo* di = device_info(st);
  return di ? di->status : nullptr;
}

int device_sm_count() {
  molt_status st;
  const DeviceInfo* di = device_info(&st);
  return di ? di->n_sm : 1;
}

molt_status encode_tmap_2d(CUtensorMap* m, CUtensorMapDataType dt, int elem_bytes, const void* base, uint64_t rows,
                           uint64_t cols, uint32_t box_cols, uint32_t box_rows) {
  return make_tmap(m, dt, elem_bytes, base, rows, cols, box_cols, box_rows);
}

}  // namespace molt

using namespace molt;

extern "C" {

const char* molt_status_string(molt_status s) {
  switch (s) {
    case MOLT_OK: return "ok";
    case MOLT_ERR_INVALID_ARG: return "invalid argument";
    case MOLT_ERR_UNSUPPORTED_SHAPE: return "unsupported shape";
    case MOLT_ERR_UNSORTED_GROUPS: return "group ids are not sorted";
    case MOLT_ERR_ZERO_DENOM: return "zero token-mean denominator";
    case MOLT_ERR_CUDA: return "CUDA error";
    case MOLT_ERR_DEVICE_TIMEOUT: return "device pipeline wait timed out";
    case MOLT_ERR_NO_MEMORY: return "out of device memory";
    case MOLT_ERR_TOKEN_RANGE: return "token id out of range";
    case MOLT_ERR_WORKSPACE: return "workspace too small";
  }
  return "unknown status";
}

const char* molt_last_error(void) { return t_last_error.c_str(); }

int molt_version(void) { return 1; }

uint64_t molt_kernel_launches(void) { return molt::g_kernel_launches.load(std::memory_order_relaxed); }

void molt_set_timing_events(cudaEvent_t* starts, cudaEvent_t* stops, int n) {
  t_ev_start = starts;
  t_ev_stop = stops;
  t_ev_n = (starts && stops && n > 0) ? n : 0;
}

molt_status molt_selftest_wait_timeout(cudaStream_t stream) {
  molt_status st;
  const DeviceInfo* di = device_info(&st);
  if (!di) return st;
  void* words = nullptr;
  MOLT_CUDA(cudaMallocAsync(&words, 16, stream), "cudaMallocAsync");
  cudaError_t e = cudaMemsetAsync(words, 0, 16, stream);
  if (e == cudaSuccess) {
    e = molt::launch_wait_selftest(static_cast<uint32_t*>(words), di->status, stream);
    if (e == cudaSuccess) molt::note_launches(1);
  }
  const cudaError_t e_free = cudaFreeAsync(words, stream);
  if (e != cudaSuccess) return cuda_fail(e, "wait self-test");
  if (e_free != cudaSuccess) return cuda_fail(e_free, "cudaFreeAsync");
  return MOLT_OK;
}

molt_status molt_device_status(cudaStream_t stream, uint32_t* flags) {
  if (!flags) return fail(MOLT_ERR_INVALID_ARG, "flags is NULL");
  molt_status st;
  const DeviceInfo* di = device_info(&st);
  if (!di) return st;
  MOLT_CUDA(cudaStreamSynchronize(stream), "cudaStreamSynchronize");
  unsigned v = 0;
  MOLT_CUDA(cudaMemcpy(&v, di->status, sizeof(v), cudaMemcpyDeviceToHost), "read status word");
  MOLT_CUDA(cudaMemset(di->status, 0, sizeof(unsigned)), "clear status word");
  *flags = v;
  if (v & MOLT_DEV_TIMEOUT) return fail(MOLT_ERR_DEVICE_TIMEOUT, "a pipeline wait timed out");
  if (v & MOLT_DEV_TOKEN_RANGE) return fail(MOLT_ERR_TOKEN_RANGE, "a token id on an active row is outside [0, V)");
  if (v & MOLT_DEV_ZERO_DENOM) return fail(MOLT_ERR_ZERO_DENOM, "no active token and no window denominator");
  if (v & MOLT_DEV_UNSORTED_GROUPS) return fail(MOLT_ERR_UNSORTED_GROUPS, "group ids decrease somewhere");
  return MOLT_OK;
}

molt_status molt_group_advantages(const float* rewards, const int32_t* group_ids, int64_t n_resp, double eps,
                                  float* adv_out, cudaStream_t stream) {
  if (n_resp < 0 || n_resp >= (int64_t(1) << 26)) return fail(MOLT_ERR_INVALID_ARG, "n_resp out of range");
  if (n_resp == 0) return MOLT_OK;
  if (!rewards || !group_ids || !adv_out) return fail(MOLT_ERR_INVALID_ARG, "null pointer");
  if (!(eps >= 0.0) || eps != eps) return fail(MOLT_ERR_INVALID_ARG, "eps must be >= 0");
  molt_status st;
  const DeviceInfo* di = device_info(&st);
  if (!di) return st;
  MOLT_LAUNCH(launch_group_advantages(rewards, group_ids, static_cast<int>(n_resp), eps, adv_out, di->status, stream),
            "group advantages");
  return MOLT_OK;
}

molt_status molt_advantages(const float* rewards, const int32_t* group_ids, int64_t n_resp, int estimator,
                            double eps, float* adv_out, cudaStream_t stream) {
  if (estimator < MOLT_ADV_GRPO || estimator > MOLT_ADV_REINFORCE_PP)
    return fail(MOLT_ERR_INVALID_ARG, "unknown advantage estimator");
  if (n_resp < 0 || n_resp >= (int64_t(1) << 26)) return fail(MOLT_ERR_INVALID_ARG, "n_resp out of range");
  if (n_resp == 0) return MOLT_OK;
  if (!rewards || !adv_out || (!group_ids && estimator != MOLT_ADV_REINFORCE_PP))
    return fail(MOLT_ERR_INVALID_ARG, "null pointer");
  if (!(eps >= 0.0)) return fail(MOLT_ERR_INVALID_ARG, "eps must be >= 0");
  molt_status st;
  const DeviceInfo* di = device_info(&st);
  if (!di) return st;
  MOLT_LAUNCH(launch_advantages(rewards, group_ids, static_cast<int>(n_resp), estimator, eps, adv_out, di->status,
                              stream),
            "advantages");
  return MOLT_OK;
}

molt_status molt_broadcast_advantages(const float* adv_resp, const int32_t* resp_of_token, int64_t n_resp,
                                      int64_t T, float* adv_tok, cudaStream_t stream) {
  if (T < 0 || n_resp < 0 || T >= (int64_t(1) << 31) || n_resp >= (int64_t(1) << 31))
    return fail(MOLT_ERR_INVALID_ARG, "sizes out of range");
  if (T == 0) return MOLT_OK;
  if (!adv_resp || !resp_of_token || !adv_tok) return fail(MOLT_ERR_INVALID_ARG, "null pointer");
  MOLT_LAUNCH(launch_broadcast(adv_resp, resp_of_token, static_cast<int>(n_resp), static_cast<int>(T), adv_tok, stream),
            "broadcast");
  return MOLT_OK;
}

molt_status molt_mask_count(const uint8_t* mask, int64_t T, int64_t* count_out, cudaStream_t stream) {
  if (T < 0) return fail(MOLT_ERR_INVALID_ARG, "T < 0");
  if (!count_out || (T > 0 && !mask)) return fail(MOLT_ERR_INVALID_ARG, "null pointer");
  if (T > 0 && !aligned16(mask)) return fail(MOLT_ERR_INVALID_ARG, "mask must be 16-byte aligned");
  if ((reinterpret_cast<uintptr_t>(count_out) & 7u) != 0) return fail(MOLT_ERR_INVALID_ARG, "count_out misaligned");
  MOLT_LAUNCH(launch_mask_count(mask, T, count_out, stream), "mask count");
  return MOLT_OK;
}

size_t molt_token_logprobs_workspace_bytes(int64_t T, int64_t H, int64_t V) {
  if (check_shape(T, H, V) != MOLT_OK) return 0;
  molt_status st;
  const DeviceInfo* di = device_info(&st);
  const int n_sm = di ? di->n_sm : 152;
  const int64_t Tcap = round_tiles(T);
  return layout(T, H, V, choose_splits(Tcap > 0 ? Tcap : kTileM, V, n_sm), false).total;
}

size_t molt_policy_loss_workspace_bytes(int64_t T, int64_t H, int64_t V) {
  if (check_shape(T, H, V) != MOLT_OK) return 0;
  molt_status st;
  const DeviceInfo* di = device_info(&st);
  const int n_sm = di ? di->n_sm : 152;
  const int64_t Tcap = round_tiles(T);
  return layout(T, H, V, choose_splits(Tcap > 0 ? Tcap : kTileM, V, n_sm), true).total;
}

size_t molt_policy_loss_workspace_bytes_ex(int64_t T, int64_t H, int64_t V, const molt_loss_options* opts) {
  if (check_shape(T, H, V) != MOLT_OK) return 0;
  const bool det = opts && opts->deterministic;
  if (det && H % 128 != 0) return 0;
  molt_status st;
  const DeviceInfo* di = device_info(&st);
  const int n_sm = di ? di->n_sm : 152;
  const int64_t Tcap = round_tiles(T);
  return layout(T, H, V, choose_splits(Tcap > 0 ? Tcap : kTileM, V, n_sm), true, det).total;
}

molt_status molt_token_logprobs_fwd(const uint16_t* hidden, const uint16_t* W, const int32_t* tokens,
                                    const uint8_t* mask, int64_t T, int64_t H, int64_t V, float* logp_out,
                                    float* entropy_out, void* workspace, size_t workspace_bytes,
                                    cudaStream_t stream) {
  MOLT_TRY(check_shape(T, H, V));
  if (T == 0) return MOLT_OK;
  if (!hidden || !W || !tokens || !logp_out) return fail(MOLT_ERR_INVALID_ARG, "null pointer");
  if (!aligned16(hidden) || !aligned16(W)) return fail(MOLT_ERR_INVALID_ARG, "hidden and W must be 16-byte aligned");
  molt_status st;
  const DeviceInfo* di = device_info(&st);
  if (!di) return st;
  const int64_t Tcap = round_tiles(T);
  const int S = choose_splits(Tcap, V, di->n_sm);
  const Layout L = layout(T, H, V, S, false);
  Scratch sc;
  MOLT_TRY(get_scratch(sc, workspace, workspace_bytes, L.total, stream));
  const Workspace w = carve(sc.ptr, L);
  CUtensorMap tm_h, tm_w;
  MOLT_TRY(make_tmap(&tm_h, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, w.h_p, Tcap, H, kBK, kTileM));
  MOLT_TRY(make_tmap(&tm_w, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, W, V, H, kBK, kFwdBN));
  MOLT_TRY(run_forward(di, hidden, tokens, mask, nullptr, nullptr, T, H, V, S, w, tm_h, tm_w, stream));
  MOLT_CUDA(cudaMemsetAsync(logp_out, 0, T * sizeof(float), stream), "memset logp");
  if (entropy_out) MOLT_CUDA(cudaMemsetAsync(entropy_out, 0, T * sizeof(float), stream), "memset entropy");
  ev_start(2, stream);
  MOLT_LAUNCH(launch_merge(false, static_cast<int>(Tcap), static_cast<int>(V), S, 0.0, 0.f, 0.f, w, logp_out,
                         entropy_out, nullptr, di->status, stream),
            "merge");
  ev_stop(2, stream);
  return MOLT_OK;
}

molt_status molt_policy_loss_fwd_bwd(const uint16_t* hidden, const uint16_t* W, const int32_t* tokens,
                                     const float* behavior_logp, const float* adv, const uint8_t* mask,
                                     int64_t T, int64_t H, int64_t V, float clip_lo, float clip_hi,
                                     double denom, float* loss_out, uint16_t* dhidden_out, float* dW_out,
                                     int accumulate_dW, float* logp_out, float* entropy_out,
                                     float* token_loss_out, molt_stats* stats_out, void* workspace,
                                     size_t workspace_bytes, cudaStream_t stream) {
  return policy_loss_impl(hidden, W, tokens, behavior_logp, adv, mask, T, H, V, clip_lo, clip_hi, denom, nullptr,
                          loss_out, dhidden_out, dW_out, accumulate_dW, logp_out, entropy_out, token_loss_out,
                          stats_out, nullptr, workspace, workspace_bytes, stream);
}

molt_status molt_policy_loss_fwd_bwd_ex(const uint16_t* hidden, const uint16_t* W, const int32_t* tokens,
                                        const float* behavior_logp, const float* adv, const uint8_t* mask,
                                        int64_t T, int64_t H, int64_t V, float clip_lo, float clip_hi,
                                        double denom, const molt_loss_options* opts, float* loss_out,
                                        uint16_t* dhidden_out, float* dW_out, int accumulate_dW,
                                        float* logp_out, float* entropy_out, float* token_loss_out,
                                        molt_stats_ex* stats_out, void* workspace, size_t workspace_bytes,
                                        cudaStream_t stream) {
  molt_loss_options none{};
  none.gate_hi = 0.0;
  return policy_loss_impl(hidden, W, tokens, behavior_logp, adv, mask, T, H, V, clip_lo, clip_hi, denom,
                          opts ? opts : &none, loss_out, dhidden_out, dW_out, accumulate_dW, logp_out, entropy_out,
                          token_loss_out, nullptr, stats_out, workspace, workspace_bytes, stream);
}


// ------------------------------------------------ vocabulary-parallel calls
size_t molt_vp_partials_workspace_bytes(int64_t T, int64_t H, int64_t V_shard) {
  return molt_token_logprobs_workspace_bytes(T, H, V_shard);
}

molt_status molt_vp_partials(const uint16_t* hidden, const uint16_t* W_shard, const int32_t* tokens,
                             const uint8_t* mask, int64_t T, int64_t H, int64_t V_shard, int64_t v_begin,
                             float* partials_out, void* workspace, size_t workspace_bytes, cudaStream_t stream) {
  MOLT_TRY(check_shape(T, H, V_shard));
  if (v_begin < 0 || v_begin + V_shard >= (int64_t(1) << 31))
    return fail(MOLT_ERR_INVALID_ARG, "v_begin must satisfy 0 <= v_begin and v_begin + V_shard < 2^31");
  if (T == 0) return MOLT_OK;
  if (!hidden || !W_shard || !tokens || !partials_out) return fail(MOLT_ERR_INVALID_ARG, "null pointer");
  if (!aligned16(hidden) || !aligned16(W_shard) || !aligned16(partials_out))
    return fail(MOLT_ERR_INVALID_ARG, "hidden, W_shard and partials_out must be 16-byte aligned");
  molt_status st;
  const DeviceInfo* di = device_info(&st);
  if (!di) return st;
  const int64_t Tcap = round_tiles(T);
  const int S = choose_splits(Tcap, V_shard, di->n_sm);
  const Layout L = layout(T, H, V_shard, S, false);
  Scratch sc;
  MOLT_TRY(get_scratch(sc, workspace, workspace_bytes, L.total, stream));
  const Workspace w = carve(sc.ptr, L);
  CUtensorMap tm_h, tm_w;
  MOLT_TRY(make_tmap(&tm_h, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, w.h_p, Tcap, H, kBK, kTileM));
  MOLT_TRY(make_tmap(&tm_w, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, W_shard, V_shard, H, kBK, kFwdBN));
  MOLT_TRY(run_forward(di, hidden, tokens, mask, nullptr, nullptr, T, H, V_shard, S, w, tm_h, tm_w, stream,
                       static_cast<int>(v_begin)));
  ev_start(2, stream);
  MOLT_LAUNCH(launch_vp_local(static_cast<int>(T), static_cast<int>(Tcap), static_cast<int>(V_shard), S, w,
                              reinterpret_cast<float4*>(partials_out), stream),
              "shard statistics");
  ev_stop(2, stream);
  return MOLT_OK;
}

size_t molt_vp_loss_workspace_bytes(int64_t T) {
  if (T < 0 || T >= (int64_t(1) << 31) - kTileM) return 0;
  return vp_loss_layout(T).total;
}

molt_status molt_vp_loss(const float* partials, int n_shards, const float* behavior_logp, const float* adv,
                         const uint8_t* mask, int64_t T, float clip_lo, float clip_hi, double denom, float* loss_out,
                         float* lse_out, float* coef_out, float* logp_out, float* entropy_out, float* token_loss_out,
                         molt_stats* stats_out, void* workspace, size_t workspace_bytes, cudaStream_t stream) {
  if (T < 0 || T >= (int64_t(1) << 31) - kTileM) return fail(MOLT_ERR_INVALID_ARG, "T out of range");
  if (n_shards < 1 || n_shards > 65536) return fail(MOLT_ERR_INVALID_ARG, "n_shards must be in [1, 65536]");
  if (!loss_out) return fail(MOLT_ERR_INVALID_ARG, "null pointer");
  if (T > 0 && (!partials || !behavior_logp || !adv || !lse_out || !coef_out))
    return fail(MOLT_ERR_INVALID_ARG, "null pointer");
  if (T > 0 && !aligned16(partials)) return fail(MOLT_ERR_INVALID_ARG, "partials must be 16-byte aligned");
  if (!(clip_lo >= 0.f && clip_lo < 1.f) || !(clip_hi >= 0.f) || clip_hi != clip_hi || clip_hi > 1e30f)
    return fail(MOLT_ERR_INVALID_ARG, "clip bounds must satisfy 0 <= clip_lo < 1 and clip_hi >= 0");
  if (denom != denom) return fail(MOLT_ERR_INVALID_ARG, "denom is NaN");
  molt_status st;
  const DeviceInfo* di = device_info(&st);
  if (!di) return st;
  if (T == 0) {
    MOLT_CUDA(cudaMemsetAsync(loss_out, 0, sizeof(float), stream), "memset loss");
    if (stats_out) MOLT_CUDA(cudaMemsetAsync(stats_out, 0, sizeof(molt_stats), stream), "memset stats");
    return MOLT_OK;
  }
  const int64_t Tcap = round_tiles(T);
  const Layout L = vp_loss_layout(T);
  Scratch sc;
  MOLT_TRY(get_scratch(sc, workspace, workspace_bytes, L.total, stream));
  const Workspace w = carve(sc.ptr, L);
  MOLT_CUDA(cudaMemsetAsync(lse_out, 0, T * sizeof(float), stream), "memset lse");
  MOLT_CUDA(cudaMemsetAsync(coef_out, 0, T * sizeof(float), stream), "memset coef");
  if (logp_out) MOLT_CUDA(cudaMemsetAsync(logp_out, 0, T * sizeof(float), stream), "memset logp");
  if (entropy_out) MOLT_CUDA(cudaMemsetAsync(entropy_out, 0, T * sizeof(float), stream), "memset entropy");
  if (token_loss_out) MOLT_CUDA(cudaMemsetAsync(token_loss_out, 0, T * sizeof(float), stream), "memset token loss");
  ev_start(0, stream);
  MOLT_LAUNCH(launch_compact(mask, static_cast<int>(T), w, stream), "compact");
  ev_stop(0, stream);
  ev_start(2, stream);
  MOLT_LAUNCH(launch_vp_merge(static_cast<int>(T), static_cast<int>(Tcap), n_shards, denom, clip_lo, clip_hi,
                              reinterpret_cast<const float4*>(partials), behavior_logp, adv, w, lse_out, coef_out,
                              logp_out, entropy_out, token_loss_out, di->status, stream),
              "shard merge");
  MOLT_LAUNCH(launch_finalize(static_cast<int>(Tcap), denom, false, w, loss_out, stats_out, nullptr, di->status,
                              stream),
              "finalize");
  ev_stop(2, stream);
  return MOLT_OK;
}

size_t molt_vp_backward_workspace_bytes(int64_t T, int64_t H, int64_t V_shard) {
  if (check_shape(T, H, V_shard) != MOLT_OK) return 0;
  return vp_backward_layout(T, H).total;
}

molt_status molt_vp_backward(const uint16_t* hidden, const uint16_t* W_shard, const int32_t* tokens,
                             const float* lse, const float* coef, int64_t T, int64_t H, int64_t V_shard,
                             int64_t v_begin, float* dhidden_partial_out, float* dW_shard_out, int accumulate_dW,
                             void* workspace, size_t workspace_bytes, cudaStream_t stream) {
  MOLT_TRY(check_shape(T, H, V_shard));
  if (v_begin < 0 || v_begin + V_shard >= (int64_t(1) << 31))
    return fail(MOLT_ERR_INVALID_ARG, "v_begin must satisfy 0 <= v_begin and v_begin + V_shard < 2^31");
  if (!W_shard || !dW_shard_out || (T > 0 && (!hidden || !tokens || !lse || !coef || !dhidden_partial_out)))
    return fail(MOLT_ERR_INVALID_ARG, "null pointer");
  if (!aligned16(W_shard) || !aligned16(dW_shard_out) || (T > 0 && (!aligned16(hidden) ||
                                                                   !aligned16(dhidden_partial_out))))
    return fail(MOLT_ERR_INVALID_ARG, "hidden, W_shard, dhidden_partial_out and dW_shard_out must be 16-byte aligned");
  molt_status st;
  const DeviceInfo* di = device_info(&st);
  if (!di) return st;
  if (T == 0) {
    if (!accumulate_dW)
      MOLT_CUDA(cudaMemsetAsync(dW_shard_out, 0, V_shard * H * sizeof(float), stream), "memset dW");
    return MOLT_OK;
  }
  const Layout L = vp_backward_layout(T, H);
  Scratch sc;
  MOLT_TRY(get_scratch(sc, workspace, workspace_bytes, L.total, stream));
  const Workspace w = carve(sc.ptr, L);
  ev_start(2, stream);
  MOLT_LAUNCH(launch_vp_live(static_cast<int>(T), coef, w, stream), "shard rows");
  MOLT_LAUNCH(launch_vp_gather(hidden, tokens, lse, coef, static_cast<int>(v_begin), static_cast<int>(H), w,
                               di->n_sm, stream),
              "shard gather");
  ev_stop(2, stream);
  MOLT_TRY(
      run_backward(di, W_shard, T, H, V_shard, w, false, 0, false, dW_shard_out, accumulate_dW, false, stream));
  ev_start(4, stream);
  MOLT_LAUNCH(launch_vp_dh_out(w, static_cast<int>(T), static_cast<int>(H), dhidden_partial_out, di->n_sm, stream),
              "shard dhidden");
  ev_stop(4, stream);
  return MOLT_OK;
}

}  // extern "C"
