// Forward pass of the LM head with a fused online log-softmax (Sec. 4.5: the
// actor's recomputed log-probabilities of the generated tokens, plus entropy).
//
// z = h W^T is never written to global memory.  Each work unit is one tile of
// 128 packed token rows times one contiguous split of the vocabulary.  For
// every 256-column vocab tile of the split, the tensor cores accumulate the
// 128 x 256 fp32 logit tile in TMEM (K = H in 64-element steps fed by TMA), and
// the epilogue warps fold it into per-row running statistics:
//   m = running max, s = sum exp(z - m), q = sum exp(z - m) (z - m)
// and pick the target logit z[x].  The split's (m, s, q) go to a small
// workspace; a row-level merge kernel combines the splits into
//   lse = m + log s,  logp = z[x] - lse,  entropy = log s - q / s.
//
// Roles (192 threads, one CTA per SM, persistent over units):
//   warp 0      TMA producer (one lane): h tile [128 x 64] + W tile [256 x 64]
//               per stage, 128-byte swizzle, 4-stage ring
//   warp 1      MMA issuer (one lane): tcgen05.mma kind::f16, M=128 N=256 K=16,
//               double-buffered accumulators (2 x 256 TMEM columns)
//   warps 2-5   epilogue: each thread owns one TMEM lane = one token row
#include <atomic>
#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

#include "molt_internal.cuh"
#include "ptx.cuh"

namespace molt {
namespace {

constexpr int kStages = 4;
constexpr int kABytes = kTileM * kBK * 2;        // 16 KB
constexpr int kBBytes = kFwdBN * kBK * 2;        // 32 KB
constexpr int kStageBytes = kABytes + kBBytes;   // 48 KB
constexpr int kThreads = 192;
constexpr int kSmemBytes = kStages * kStageBytes + 1024;
constexpr uint32_t kIdesc = idesc_bf16_f32(kTileM, kFwdBN, false, false);
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

__device__ __forceinline__ void split_range(int s, int S, int n_vt, int& vt0, int& vt1) {
  vt0 = static_cast<int>(static_cast<int64_t>(s) * n_vt / S);
  vt1 = static_cast<int>(static_cast<int64_t>(s + 1) * n_vt / S);
}

// fold 32 logits (all columns valid) into the running (m, s, q2) of one row;
// q2 is kept in log2 units: q2 = sum e * (z - m) * log2(e)
__device__ __forceinline__ void fold_full(const float (&v)[32], float& m, float& s, float& q2) {
  float cmax = v[0];
#pragma unroll
  for (int j = 1; j < 32; ++j) cmax = fmaxf(cmax, v[j]);
  if (cmax > m) {
    if (m != -INFINITY) {
      const float d2 = (m - cmax) * kLog2e;
      const float sc = ex2_approx(d2);
      q2 = sc * fmaf(d2, s, q2);
      s *= sc;
    }
    m = cmax;
  }
  const float mL = m * kLog2e;
  float s0 = 0.f, s1 = 0.f, q0 = 0.f, q1 = 0.f;
#pragma unroll
  for (int j = 0; j < 32; j += 2) {
    const float y0 = fmaf(v[j], kLog2e, -mL);
    const float y1 = fmaf(v[j + 1], kLog2e, -mL);
    const float e0 = ex2_approx(y0);
    const float e1 = ex2_approx(y1);
    s0 += e0;
    s1 += e1;
    q0 = fmaf(e0, y0, q0);
    q1 = fmaf(e1, y1, q1);
  }
  s += s0 + s1;
  q2 += q0 + q1;
}

// same for a chunk where only the first `nv` (1..31) columns are valid
__device__ __forceinline__ void fold_partial(const float (&v)[32], int nv, float& m, float& s, float& q2) {
  float cmax = v[0];
#pragma unroll
  for (int j = 1; j < 32; ++j)
    if (j < nv) cmax = fmaxf(cmax, v[j]);
  if (cmax > m) {
    if (m != -INFINITY) {
      const float d2 = (m - cmax) * kLog2e;
      const float sc = ex2_approx(d2);
      q2 = sc * fmaf(d2, s, q2);
      s *= sc;
    }
    m = cmax;
  }
  const float mL = m * kLog2e;
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    if (j < nv) {
      const float y = fmaf(v[j], kLog2e, -mL);
      const float e = ex2_approx(y);
      s += e;
      q2 = fmaf(e, y, q2);
    }
  }
}

__global__ void __launch_bounds__(kThreads, 1)
    lmhead_fwd_kernel(const __grid_constant__ CUtensorMap tm_h, const __grid_constant__ CUtensorMap tm_w,
                      const FwdArgs a) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[kStages];
  __shared__ __align__(8) uint64_t empty_bar[kStages];
  __shared__ __align__(8) uint64_t accf_bar[2];
  __shared__ __align__(8) uint64_t acce_bar[2];
  __shared__ __align__(8) uint64_t done_bar;
  __shared__ uint32_t tmem_base_sh;
  __shared__ int abort_sh;

  const uint32_t smem0 = (smem_u32(smem_raw) + 1023u) & ~1023u;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  volatile int* abort_flag = &abort_sh;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(smem_u32(&full_bar[s]), 1);
      mbar_init(smem_u32(&empty_bar[s]), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(smem_u32(&accf_bar[b]), 1);
      mbar_init(smem_u32(&acce_bar[b]), 128);
    }
    mbar_init(smem_u32(&done_bar), 1);
    abort_sh = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&tmem_base_sh), 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = tmem_base_sh;

  const int n_rows = a.counts[0];
  const int n_mt = (n_rows + kTileM - 1) / kTileM;
  const int S = a.n_split;
  const int n_units = n_mt * S;
  const int kblocks = a.H / kBK;

  if (warp == 0) {
    if (lane == 0) {
      prefetch_tmap(&tm_h);
      prefetch_tmap(&tm_w);
      uint32_t it = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < n_units && ok; u += gridDim.x) {
        const int mt = u / S, s = u - mt * S;
        int vt0, vt1;
        split_range(s, S, a.n_vtiles, vt0, vt1);
        for (int vt = vt0; vt < vt1 && ok; ++vt) {
          for (int kb = 0; kb < kblocks; ++kb) {
            const uint32_t st = it % kStages, ph = (it / kStages) & 1u;
            if (!mbar_wait(smem_u32(&empty_bar[st]), ph ^ 1u, abort_flag, a.err)) {
              ok = false;
              break;
            }
            const uint32_t sa = smem0 + st * kStageBytes;
            const uint32_t fb = smem_u32(&full_bar[st]);
            mbar_arrive_expect_tx(fb, kStageBytes);
            tma_load_2d(sa, &tm_h, fb, kb * kBK, mt * kTileM);
            tma_load_2d(sa + kABytes, &tm_w, fb, kb * kBK, vt * kFwdBN);
            ++it;
          }
        }
      }
      // exit path: every issued copy must land before the CTA's smem goes away
      const uint32_t first = it > (uint32_t)kStages ? it - kStages : 0u;
      for (uint32_t j = first; j < it; ++j)
        mbar_wait_drain(smem_u32(&full_bar[j % kStages]), (j / kStages) & 1u, a.err);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      uint32_t it = 0, acc_it = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < n_units && ok; u += gridDim.x) {
        const int mt = u / S, s = u - mt * S;
        (void)mt;
        int vt0, vt1;
        split_range(s, S, a.n_vtiles, vt0, vt1);
        for (int vt = vt0; vt < vt1 && ok; ++vt) {
          const uint32_t buf = acc_it & 1u, aph = (acc_it >> 1) & 1u;
          if (!mbar_wait(smem_u32(&acce_bar[buf]), aph ^ 1u, abort_flag, a.err)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d = tmem_base + buf * kFwdBN;
          for (int kb = 0; kb < kblocks; ++kb) {
            const uint32_t st = it % kStages, ph = (it / kStages) & 1u;
            if (!mbar_wait(smem_u32(&full_bar[st]), ph, abort_flag, a.err)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t sa = smem0 + st * kStageBytes;
            const uint64_t ad = sdesc_sw128(sa, 16, 1024);
            const uint64_t bd = sdesc_sw128(sa + kABytes, 16, 1024);
#pragma unroll
            for (int k = 0; k < kBK / 16; ++k)
              umma_bf16(d, ad + 2u * k, bd + 2u * k, kIdesc, (kb | k) != 0 ? 1u : 0u);
            umma_commit(smem_u32(&empty_bar[st]));
            ++it;
          }
          if (!ok) break;
          umma_commit(smem_u32(&accf_bar[buf]));
          ++acc_it;
        }
      }
      umma_commit(smem_u32(&done_bar));
      mbar_wait_drain(smem_u32(&done_bar), 0, a.err);
    }
  } else {
    // epilogue: warp w may read TMEM lanes [32 (w % 4), 32 (w % 4) + 32)
    const int q = warp & 3;
    const int r_in_tile = q * 32 + lane;
    uint32_t acc_it = 0;
    bool ok = true;
    for (int u = blockIdx.x; u < n_units && ok; u += gridDim.x) {
      const int mt = u / S, s = u - mt * S;
      int vt0, vt1;
      split_range(s, S, a.n_vtiles, vt0, vt1);
      const int row = mt * kTileM + r_in_tile;
      const bool valid = row < n_rows;
      const int x = valid ? a.tok_p[row] : -1;
      float m = -INFINITY, ssum = 0.f, q2 = 0.f, zxv = 0.f;
      bool found = false;
      for (int vt = vt0; vt < vt1; ++vt) {
        const uint32_t buf = acc_it & 1u, aph = (acc_it >> 1) & 1u;
        if (!mbar_wait(smem_u32(&accf_bar[buf]), aph, abort_flag, a.err)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const int col0 = vt * kFwdBN;
        const int ncols = min(kFwdBN, a.V - col0);
        const int lx = x - col0;
        const uint32_t taddr = tmem_base + (static_cast<uint32_t>(q * 32) << 16) + buf * kFwdBN;
#pragma unroll 1
        for (int c0 = 0; c0 < kFwdBN; c0 += 32) {
          if (c0 >= ncols) break;
          float v[32];
          tmem_ld32(taddr + c0, v);
          const int lxc = lx - c0;
          if (static_cast<unsigned>(lxc) < 32u) {
#pragma unroll
            for (int j = 0; j < 32; ++j)
              if (j == lxc) zxv = v[j];
            found = true;
          }
          if (c0 + 32 <= ncols)
            fold_full(v, m, ssum, q2);
          else
            fold_partial(v, ncols - c0, m, ssum, q2);
        }
        tc_fence_before();
        mbar_arrive(smem_u32(&acce_bar[buf]));
        ++acc_it;
      }
      if (!ok) break;
      if (valid) {
        a.part[static_cast<int64_t>(s) * a.rows_cap + row] = make_float4(m, ssum, q2 * kLn2, 0.f);
        if (found) a.zx[row] = zxv;
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) {
    __syncwarp();
    tmem_dealloc(tmem_base, 512);
  }
}

}  // namespace

cudaError_t launch_lmhead_fwd(const CUtensorMap& tm_h, const CUtensorMap& tm_w, const FwdArgs& a, int grid,
                              cudaStream_t s) {
  // the shared-memory attribute is per device: set it on each device once
  static std::atomic<unsigned long long> attr_set{0};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const unsigned long long bit = 1ull << (dev & 63);
  if ((attr_set.load(std::memory_order_acquire) & bit) == 0) {
    e = cudaFuncSetAttribute(lmhead_fwd_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
    if (e != cudaSuccess) return e;
    attr_set.fetch_or(bit, std::memory_order_release);
  }
  lmhead_fwd_kernel<<<grid, kThreads, kSmemBytes, s>>>(tm_h, tm_w, a);
  return cudaGetLastError();
}

}  // namespace molt
