// molt_token_logprobs_fwd_noalloc: the log-probability / entropy forward for
// callers that must not allocate device memory.
//
// Some callers cannot let a library call cudaMalloc (or cudaMallocAsync): a
// training runtime that reserves the whole HBM budget up front and hands out
// memory only through its own pool, or a process whose memory limits leave no
// room outside that pool.  For them this entry point keeps its scratch in one
// file-scope device array, sized for at most kNoAllocMaxRows tokens, that every
// GPU loading the library holds until the process exits.  The caller still owns
// and passes every input and output; the call allocates nothing.
//
// Differences from molt_token_logprobs_fwd: no active-row compaction (masked
// rows are computed and then written as 0), at most kNoAllocMaxSplits vocab
// splits, and T <= kNoAllocMaxRows.  The same forward kernel does the work.
#include <cstdint>
#include <mutex>
#include <string>

#include <cuda.h>
#include <cuda_runtime.h>

#include "../../include/molt.h"
#include "molt_internal.cuh"
#include "ptx.cuh"

namespace molt {
namespace {

constexpr int kNoAllocMaxRows = MOLT_NOALLOC_MAX_TOKENS;
constexpr int kNoAllocMaxSplits = 8;
constexpr size_t kCountsBytes = 256;
constexpr size_t kPartBytes = static_cast<size_t>(kNoAllocMaxSplits) * kNoAllocMaxRows * sizeof(float4);
constexpr size_t kZxBytes = static_cast<size_t>(kNoAllocMaxRows) * sizeof(float);
constexpr size_t kScratchBytes = kCountsBytes + kPartBytes + kZxBytes;   // ~4.1 MB

constexpr float kLog2e = 1.4426950408889634f;

}  // namespace
}  // namespace molt

// The scratch shared by every call on a device (counts, split partials, target
// logits).  Host code must not take its address directly: it is resolved per
// device with cudaGetSymbolAddress.
static __device__ __align__(256) unsigned char g_noalloc_scratch[molt::kScratchBytes];

namespace molt {
namespace {

// Device address of the scratch array per device, looked up on the first call
// that succeeds in doing so (a failed lookup is not remembered: the next call
// tries again).
std::mutex g_noalloc_mu;
unsigned char* g_noalloc_addr[64] = {};

// rows [0, T): counts[0] = T and the target logits start at 0 (so a row whose
// target is out of range never reads a previous call's value)
__global__ void noalloc_init_kernel(int T, int32_t* counts, float* zx) {
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t == 0) {
    counts[0] = T;
    counts[1] = 0;
  }
  if (t < T) zx[t] = 0.f;
}

// merge the per-split partials of each row into logp and entropy; masked rows
// are written as 0, active rows with an out-of-range token raise the status flag
__global__ void noalloc_merge_kernel(int T, int V, int S, int rows_cap, const int32_t* __restrict__ tokens,
                                     const uint8_t* __restrict__ mask, const float4* __restrict__ part,
                                     const float* __restrict__ zx, float* __restrict__ logp_out,
                                     float* __restrict__ ent_out, unsigned* err) {
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= T) return;
  if (mask != nullptr && mask[t] == 0) {
    logp_out[t] = 0.f;
    if (ent_out) ent_out[t] = 0.f;
    return;
  }
  float M = -INFINITY;
  for (int s = 0; s < S; ++s) M = fmaxf(M, part[static_cast<int64_t>(s) * rows_cap + t].x);
  float Ssum = 0.f, Q = 0.f;
  for (int s = 0; s < S; ++s) {
    const float4 p = part[static_cast<int64_t>(s) * rows_cap + t];
    if (p.y > 0.f) {
      const float d = p.x - M;
      const float f = ex2_approx(d * kLog2e);
      Ssum += f * p.y;
      Q += f * (p.z + d * p.y);
    }
  }
  const int x = tokens[t];
  if (x < 0 || x >= V) atomicOr(err, kDevErrTokenRange);
  const float logS = logf(Ssum);
  logp_out[t] = zx[t] - (M + logS);
  if (ent_out) ent_out[t] = logS - Q / Ssum;
}

molt_status noalloc_fail(molt_status s, const std::string& msg) {
  set_last_error(msg);
  return s;
}

#define MOLT_TRY_STATUS(call)        \
  do {                               \
    molt_status s_ = (call);         \
    if (s_ != MOLT_OK) return s_;    \
  } while (0)

}  // namespace
}  // namespace molt

using namespace molt;

extern "C" molt_status molt_token_logprobs_fwd_noalloc(const uint16_t* hidden, const uint16_t* W,
                                                       const int32_t* tokens, const uint8_t* mask, int64_t T,
                                                       int64_t H, int64_t V, float* logp_out,
                                                       float* entropy_out, cudaStream_t stream) {
  if (T < 0 || V < 1 || H < 1) return noalloc_fail(MOLT_ERR_INVALID_ARG, "sizes must satisfy T >= 0, H >= 1, V >= 1");
  if (H % 64 != 0 || H > 65536) return noalloc_fail(MOLT_ERR_UNSUPPORTED_SHAPE, "H must be a multiple of 64, at most 65536");
  if (T > kNoAllocMaxRows)
    return noalloc_fail(MOLT_ERR_UNSUPPORTED_SHAPE,
                        "molt_token_logprobs_fwd_noalloc handles at most " + std::to_string(kNoAllocMaxRows) +
                            " tokens per call (got " + std::to_string(T) + "); split the batch");
  if (V >= (int64_t(1) << 31)) return noalloc_fail(MOLT_ERR_UNSUPPORTED_SHAPE, "V must be below 2^31");
  if (T == 0) return MOLT_OK;
  if (!hidden || !W || !tokens || !logp_out) return noalloc_fail(MOLT_ERR_INVALID_ARG, "null pointer");
  if ((reinterpret_cast<uintptr_t>(hidden) & 15u) || (reinterpret_cast<uintptr_t>(W) & 15u))
    return noalloc_fail(MOLT_ERR_INVALID_ARG, "hidden and W must be 16-byte aligned");

  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess || dev < 0 || dev >= 64) return noalloc_fail(MOLT_ERR_CUDA, "cudaGetDevice failed");
  // set-up per device, with that device current: the device address of the
  // scratch array (the host-side symbol is only a stand-in)
  unsigned char* scratch = nullptr;
  {
    std::lock_guard<std::mutex> lk(g_noalloc_mu);
    if (g_noalloc_addr[dev] == nullptr) {
      void* p = nullptr;
      e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
      if (e != cudaSuccess || p == nullptr) {
        cudaGetLastError();
        return noalloc_fail(MOLT_ERR_CUDA, std::string("cudaGetSymbolAddress(scratch): ") + cudaGetErrorString(e));
      }
      g_noalloc_addr[dev] = static_cast<unsigned char*>(p);
    }
    scratch = g_noalloc_addr[dev];
  }
  molt_status st;
  unsigned* status_word = device_status_word(&st);
  if (!status_word) return st;
  const int n_sm = device_sm_count();

  const int64_t Tcap = ((T + kTileM - 1) / kTileM) * kTileM;
  const int n_vt = static_cast<int>((V + kFwdBN - 1) / kFwdBN);
  int S = static_cast<int>((16 * static_cast<int64_t>(n_sm) * kTileM + Tcap - 1) / Tcap);
  if (S < 1) S = 1;
  if (S > kNoAllocMaxSplits) S = kNoAllocMaxSplits;
  if (S > n_vt) S = n_vt;

  int32_t* counts = reinterpret_cast<int32_t*>(scratch);
  float4* part = reinterpret_cast<float4*>(scratch + kCountsBytes);
  float* zx = reinterpret_cast<float*>(scratch + kCountsBytes + kPartBytes);

  CUtensorMap tm_h, tm_w;
  MOLT_TRY_STATUS(encode_tmap_2d(&tm_h, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, hidden, T, H, kBK, kTileM));
  MOLT_TRY_STATUS(encode_tmap_2d(&tm_w, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, W, V, H, kBK, kFwdBN));

  noalloc_init_kernel<<<static_cast<int>((T + 255) / 256), 256, 0, stream>>>(static_cast<int>(T), counts, zx);
  if ((e = cudaGetLastError()) != cudaSuccess) return noalloc_fail(MOLT_ERR_CUDA, cudaGetErrorString(e));
  note_launches(1);
  FwdArgs fa{};
  fa.tok_p = tokens;
  fa.counts = counts;
  fa.rows_cap = static_cast<int>(Tcap);
  fa.V = static_cast<int>(V);
  fa.H = static_cast<int>(H);
  fa.n_split = S;
  fa.n_vtiles = n_vt;
  fa.part = part;
  fa.zx = zx;
  fa.err = status_word;
  timing_event(1, false, stream);
  if ((e = launch_lmhead_fwd(tm_h, tm_w, fa, n_sm, stream)) != cudaSuccess)
    return noalloc_fail(MOLT_ERR_CUDA, cudaGetErrorString(e));
  note_launches(1);
  timing_event(1, true, stream);
  timing_event(2, false, stream);
  noalloc_merge_kernel<<<static_cast<int>((T + 127) / 128), 128, 0, stream>>>(
      static_cast<int>(T), static_cast<int>(V), S, static_cast<int>(Tcap), tokens, mask, part, zx, logp_out,
      entropy_out, status_word);
  if ((e = cudaGetLastError()) != cudaSuccess) return noalloc_fail(MOLT_ERR_CUDA, cudaGetErrorString(e));
  note_launches(1);
  timing_event(2, true, stream);
  return MOLT_OK;
}
