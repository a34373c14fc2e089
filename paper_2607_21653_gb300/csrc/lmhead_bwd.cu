// Backward pass of the fused LM-head + clipped-surrogate loss (Sec. 4.5, Eq. 2).
//
//   g_tv = coef_t (softmax(z_t)_v - [v == x_t]),  coef_t = m_t c_t / D
//          (+ ecoef_t softmax(z_t)_v (z_tv - mu_t) with an entropy bonus)
//   dH_t = sum_v g_tv W_v          dW_v = sum_t g_tv h_t
//
// Neither the logits nor g touch global memory.  A work unit is one 128-row
// tile of active tokens times one 256-column vocab chunk j (chunks counted from
// vc_begin, so the kernel can take a slice of the vocabulary while the cluster
// kernel takes the rest):
//   job Z    z = h_tile W_j^T on the tensor cores (M=128, N=256, K=H) into TMEM;
//            the epilogue turns it into g (bf16) and stores it in shared memory
//            in the 128-byte-swizzled K-major layout
//   job dH   for each 256-wide slice of H: acc = g [128 x 256] * W_j[:, slice]
//            (A = g, K-major; B = W rows, MN-major), drained into the fp32
//            dhidden accumulator with TMA reduce-add
//   job dW   for each 128-wide slice of H and each half of the vocab chunk:
//            acc = g^T [128 x 128] * h_tile[:, slice] (A = the same g buffer
//            read MN-major, B = h rows, MN-major), drained into dW with TMA
//            reduce-add
// Tiles whose rows all have coef = 0 (masked or clipped) are skipped: their
// contribution is exactly zero.
//
// Roles (192 threads, one CTA per SM, persistent):
//   warp 0    TMA producer, 3-stage ring of 48 KB
//   warp 1    MMA issuer; TMEM holds two 256-column accumulators in a ring
//   warps 2-5 epilogue: g computation and the reduce-add drains
#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

#include "molt_internal.cuh"
#include "ptx.cuh"

namespace molt {
namespace {

constexpr int kStages = 3;
constexpr int kStageBytes = 48 * 1024;
constexpr int kZABytes = kTileM * kBK * 2;        // h tile [128 x 64]   16 KB
constexpr int kGSub = kTileM * kBK * 2;           // g sub-tile [128 x 64] 16 KB
constexpr int kGBytes = 4 * kGSub;                // g tile [128 x 256]  64 KB
constexpr int kBoxBytes = 32 * 32 * 4;            // fp32 [32 x 32] reduce box
constexpr int kThreads = 192;
constexpr int kSmemBytes = 1024 + kStages * kStageBytes + kGBytes + 4 * kBoxBytes;
constexpr uint32_t kIdescZ = idesc_bf16_f32(kTileM, kBwdBV, false, false);
constexpr float kLog2e = 1.4426950408889634f;

struct Unit {
  int tile;
  int vc;
};

// Raster: active tiles in groups of `group`; inside a group consecutive units
// walk the group's tiles for one vocab chunk before moving to the next chunk,
// so concurrently running CTAs share W chunks and dhidden rows in L2.
__device__ __forceinline__ Unit unit_of(int u, int n_tiles, int n_vc, int group) {
  const int per_group = group * n_vc;
  const int g = u / per_group;
  const int r = u - g * per_group;
  const int g_tiles = min(group, n_tiles - g * group);
  const int vc = r / g_tiles;
  return {g * group + (r - vc * g_tiles), vc};
}

__device__ __forceinline__ void write_box(uint32_t box, int lane, const float (&v)[32]) {
  const uint32_t rowp = box + lane * 128;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const uint32_t pos = static_cast<uint32_t>(i ^ (lane & 7));
    st_shared_v4(rowp + pos * 16, __float_as_uint(v[4 * i]), __float_as_uint(v[4 * i + 1]),
                 __float_as_uint(v[4 * i + 2]), __float_as_uint(v[4 * i + 3]));
  }
}

template <bool kEnt>
__global__ void __launch_bounds__(kThreads, 1)
    lmhead_bwd_kernel(const __grid_constant__ CUtensorMap tm_h, const __grid_constant__ CUtensorMap tm_wz,
                      const __grid_constant__ CUtensorMap tm_wn, const __grid_constant__ CUtensorMap tm_dh,
                      const __grid_constant__ CUtensorMap tm_dw, const BwdArgs a) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[kStages];
  __shared__ __align__(8) uint64_t empty_bar[kStages];
  __shared__ __align__(8) uint64_t accf_bar[2];
  __shared__ __align__(8) uint64_t acce_bar[2];
  __shared__ __align__(8) uint64_t gready_bar;
  __shared__ __align__(8) uint64_t done_bar;
  __shared__ uint32_t tmem_base_sh;
  __shared__ int abort_sh;

  const uint32_t smem0 = (smem_u32(smem_raw) + 1023u) & ~1023u;
  const uint32_t g_base = smem0 + kStages * kStageBytes;
  const uint32_t box_base = g_base + kGBytes;
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
    mbar_init(smem_u32(&gready_bar), 128);
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

  const int n_tiles = a.counts[1];
  const int n_vc = a.n_vchunks;
  const int n_units = n_tiles * n_vc;
  const int H = a.H, V = a.V;
  const int kblocks = H / kBK;
  const int nH = (H + 255) / 256;
  const int nW = (H + 127) / 128;

  if (warp == 0) {
    if (lane == 0) {
      prefetch_tmap(&tm_h);
      prefetch_tmap(&tm_wz);
      prefetch_tmap(&tm_wn);
      uint32_t it = 0;
      bool ok = true;
      auto next_stage = [&](uint32_t bytes, uint32_t& sa, uint32_t& fb) -> bool {
        const uint32_t st = it % kStages, ph = (it / kStages) & 1u;
        if (!mbar_wait(smem_u32(&empty_bar[st]), ph ^ 1u, abort_flag, a.err)) return false;
        sa = smem0 + st * kStageBytes;
        fb = smem_u32(&full_bar[st]);
        mbar_arrive_expect_tx(fb, bytes);
        ++it;
        return true;
      };
      for (int u = blockIdx.x; u < n_units && ok; u += gridDim.x) {
        const Unit un = unit_of(u, n_tiles, n_vc, a.tile_group);
        const int row0 = a.tile_list[un.tile] * kTileM;
        const int v0 = (a.vc_begin + un.vc) * kBwdBV;
        const int n_kb4 = min(4, (V - v0 + 63) / 64);
        uint32_t sa, fb;
        for (int kb = 0; kb < kblocks && ok; ++kb) {
          if (!(ok = next_stage(kZABytes + kBwdBV * kBK * 2, sa, fb))) break;
          tma_load_2d(sa, &tm_h, fb, kb * kBK, row0);
          tma_load_2d(sa + kZABytes, &tm_wz, fb, kb * kBK, v0);
        }
        for (int nc = 0; nc < nH && ok; ++nc) {
          const int nbox = min(256, H - nc * 256) / 64;
          for (int kb4 = 0; kb4 < n_kb4 && ok; ++kb4) {
            if (!(ok = next_stage(nbox * 64 * 64 * 2, sa, fb))) break;
            for (int q = 0; q < nbox; ++q) tma_load_2d(sa + q * 8192, &tm_wn, fb, nc * 256 + q * 64, v0 + kb4 * 64);
          }
        }
        for (int nc = 0; nc < nW && ok; ++nc) {
          const int nbox = min(128, H - nc * 128) / 64;
          if (!(ok = next_stage(nbox * kTileM * 64 * 2, sa, fb))) break;
          for (int q = 0; q < nbox; ++q) tma_load_2d(sa + q * 16384, &tm_h, fb, nc * 128 + q * 64, row0);
        }
      }
      const uint32_t first = it > (uint32_t)kStages ? it - kStages : 0u;
      for (uint32_t j = first; j < it; ++j)
        mbar_wait_drain(smem_u32(&full_bar[j % kStages]), (j / kStages) & 1u, a.err);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      uint32_t it = 0, jj = 0, unit_it = 0;
      bool ok = true;
      auto wait_stage = [&](uint32_t& sa) -> bool {
        const uint32_t st = it % kStages, ph = (it / kStages) & 1u;
        if (!mbar_wait(smem_u32(&full_bar[st]), ph, abort_flag, a.err)) return false;
        tc_fence_after();
        sa = smem0 + st * kStageBytes;
        return true;
      };
      auto release_stage = [&]() {
        umma_commit(smem_u32(&empty_bar[it % kStages]));
        ++it;
      };
      auto acquire_acc = [&](uint32_t& d) -> bool {
        const uint32_t buf = jj & 1u, aph = (jj >> 1) & 1u;
        if (!mbar_wait(smem_u32(&acce_bar[buf]), aph ^ 1u, abort_flag, a.err)) return false;
        tc_fence_after();
        d = tmem_base + buf * 256;
        return true;
      };
      auto publish_acc = [&]() {
        umma_commit(smem_u32(&accf_bar[jj & 1u]));
        ++jj;
      };
      for (int u = blockIdx.x; u < n_units && ok; u += gridDim.x) {
        const Unit un = unit_of(u, n_tiles, n_vc, a.tile_group);
        const int v0 = (a.vc_begin + un.vc) * kBwdBV;
        const int n_kb4 = min(4, (V - v0 + 63) / 64);
        const int n_mh = (V - v0 > 128) ? 2 : 1;
        uint32_t d, sa;
        // job Z
        if (!(ok = acquire_acc(d))) break;
        for (int kb = 0; kb < kblocks && ok; ++kb) {
          if (!(ok = wait_stage(sa))) break;
          const uint64_t ad = sdesc_sw128(sa, 16, 1024);
          const uint64_t bd = sdesc_sw128(sa + kZABytes, 16, 1024);
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k) umma_bf16(d, ad + 2u * k, bd + 2u * k, kIdescZ, (kb | k) != 0 ? 1u : 0u);
          release_stage();
        }
        if (!ok) break;
        publish_acc();
        // g must be in shared memory before the products that read it
        if (!(ok = mbar_wait(smem_u32(&gready_bar), unit_it & 1u, abort_flag, a.err))) break;
        tc_fence_after();
        // jobs dH
        for (int nc = 0; nc < nH && ok; ++nc) {
          const int ncols = min(256, H - nc * 256);
          const uint32_t idesc = idesc_bf16_f32(kTileM, ncols, false, true);
          if (!(ok = acquire_acc(d))) break;
          for (int kb4 = 0; kb4 < n_kb4 && ok; ++kb4) {
            if (!(ok = wait_stage(sa))) break;
            const uint64_t ad = sdesc_sw128(g_base + kb4 * kGSub, 16, 1024);
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              const uint64_t bd = sdesc_sw128(sa + k * 2048, 8192, 1024);
              umma_bf16(d, ad + 2u * k, bd, idesc, (kb4 | k) != 0 ? 1u : 0u);
            }
            release_stage();
          }
          if (!ok) break;
          publish_acc();
        }
        // jobs dW
        for (int nc = 0; nc < nW && ok; ++nc) {
          const int ncols = min(128, H - nc * 128);
          const uint32_t idesc = idesc_bf16_f32(kTileM, ncols, true, true);
          if (!(ok = acquire_acc(d))) break;
          if (!(ok = wait_stage(sa))) break;
          for (int mh = 0; mh < n_mh; ++mh) {
#pragma unroll
            for (int k = 0; k < kTileM / 16; ++k) {
              const uint64_t ad = sdesc_sw128(g_base + 2 * mh * kGSub + k * 2048, kGSub, 1024);
              const uint64_t bd = sdesc_sw128(sa + k * 2048, 16384, 1024);
              umma_bf16(d + mh * 128, ad, bd, idesc, k != 0 ? 1u : 0u);
            }
          }
          release_stage();
          publish_acc();
        }
        ++unit_it;
      }
      umma_commit(smem_u32(&done_bar));
      mbar_wait_drain(smem_u32(&done_bar), 0, a.err);
    }
  } else {
    const int q = warp & 3;
    const int r = q * 32 + lane;        // row of the tile = TMEM lane
    const uint32_t box = box_base + (warp - 2) * kBoxBytes;
    const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
    uint32_t jj = 0;
    bool ok = true;
    auto acquire_full = [&](uint32_t& taddr) -> bool {
      const uint32_t buf = jj & 1u, aph = (jj >> 1) & 1u;
      if (!mbar_wait(smem_u32(&accf_bar[buf]), aph, abort_flag, a.err)) return false;
      tc_fence_after();
      taddr = tmem_base + lane_off + buf * 256;
      return true;
    };
    auto release = [&]() {
      tc_fence_before();
      mbar_arrive(smem_u32(&acce_bar[jj & 1u]));
      ++jj;
    };
    // one [32 x 32] fp32 slab of this warp's rows -> reduce-add into global
    auto drain_slab = [&](const CUtensorMap* map, uint32_t taddr, int x, int y, bool issue) {
      float v[32];
      tmem_ld32(taddr, v);
      if (lane == 0) bulk_wait_group_read<0>();
      __syncwarp();
      write_box(box, lane, v);
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0 && issue) {
        tma_reduce_add_2d(map, box, x, y);
        bulk_commit_group();
      }
    };
    for (int u = blockIdx.x; u < n_units && ok; u += gridDim.x) {
      const Unit un = unit_of(u, n_tiles, n_vc, a.tile_group);
      const int row0 = a.tile_list[un.tile] * kTileM;
      const int v0 = (a.vc_begin + un.vc) * kBwdBV;
      const int n_mh = (V - v0 > 128) ? 2 : 1;
      const int row = row0 + r;
      const float coef = a.coef[row];
      float ecoef = 0.f, mu = 0.f;
      if constexpr (kEnt) {
        ecoef = a.ecoef[row];
        mu = a.mu[row];
      }
      const bool live = kEnt ? (coef != 0.f || ecoef != 0.f) : (coef != 0.f);
      const float lseL = live ? a.lse[row] * kLog2e : 0.f;
      const int lx = a.tok_p[row] - v0;
      uint32_t taddr;
      // job Z -> g in shared memory
      if (!(ok = acquire_full(taddr))) break;
#pragma unroll 1
      for (int c0 = 0; c0 < kBwdBV; c0 += 32) {
        float v[32];
        tmem_ld32(taddr + c0, v);
        uint32_t w[16];
        if (live) {
          const int lxc = lx - c0;
          const int nvalid = V - v0 - c0;
#pragma unroll
          for (int j = 0; j < 32; j += 2) {
            float g0, g1;
            if constexpr (kEnt) {   // p (coef + ecoef (z - mu)): the entropy-bonus term
              g0 = fmaf(ecoef, v[j] - mu, coef) * ex2_approx(fmaf(v[j], kLog2e, -lseL));
              g1 = fmaf(ecoef, v[j + 1] - mu, coef) * ex2_approx(fmaf(v[j + 1], kLog2e, -lseL));
            } else {
              g0 = coef * ex2_approx(fmaf(v[j], kLog2e, -lseL));
              g1 = coef * ex2_approx(fmaf(v[j + 1], kLog2e, -lseL));
            }
            if (j == lxc) g0 -= coef;
            if (j + 1 == lxc) g1 -= coef;
            if (j >= nvalid) g0 = 0.f;
            if (j + 1 >= nvalid) g1 = 0.f;
            w[j / 2] = pack_bf16x2(g0, g1);
          }
        } else {
#pragma unroll
          for (int j = 0; j < 16; ++j) w[j] = 0u;
        }
        const uint32_t rowp = g_base + (c0 / 64) * kGSub + r * 128;
        const int cc0 = (c0 & 63) / 8;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const uint32_t pos = static_cast<uint32_t>((cc0 + i) ^ (r & 7));
          st_shared_v4(rowp + pos * 16, w[4 * i], w[4 * i + 1], w[4 * i + 2], w[4 * i + 3]);
        }
      }
      fence_proxy_async_smem();
      release();
      mbar_arrive(smem_u32(&gready_bar));
      // jobs dH
      for (int nc = 0; nc < nH && ok; ++nc) {
        if (!(ok = acquire_full(taddr))) break;
        const int ncols = min(256, H - nc * 256);
        for (int c0 = 0; c0 < ncols; c0 += 32) drain_slab(&tm_dh, taddr + c0, nc * 256 + c0, row0 + q * 32, true);
        release();
      }
      // jobs dW
      for (int nc = 0; nc < nW && ok; ++nc) {
        if (!(ok = acquire_full(taddr))) break;
        const int ncols = min(128, H - nc * 128);
        for (int mh = 0; mh < n_mh; ++mh) {
          const int vrow = v0 + mh * 128 + q * 32;
          for (int c0 = 0; c0 < ncols; c0 += 32)
            drain_slab(&tm_dw, taddr + mh * 128 + c0, nc * 128 + c0, vrow, vrow < V);
        }
        release();
      }
    }
    if (lane == 0) bulk_wait_group<0>();
    __syncwarp();
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

cudaError_t launch_lmhead_bwd(const CUtensorMap& tm_h, const CUtensorMap& tm_w_z, const CUtensorMap& tm_w_n,
                              const CUtensorMap& tm_dh, const CUtensorMap& tm_dw, const BwdArgs& a, int grid,
                              cudaStream_t s) {
  const bool ent = a.ecoef != nullptr;
  cudaError_t e = ent ? cudaFuncSetAttribute(lmhead_bwd_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             kSmemBytes)
                      : cudaFuncSetAttribute(lmhead_bwd_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             kSmemBytes);
  if (e != cudaSuccess) return e;
  if (ent)
    lmhead_bwd_kernel<true><<<grid, kThreads, kSmemBytes, s>>>(tm_h, tm_w_z, tm_w_n, tm_dh, tm_dw, a);
  else
    lmhead_bwd_kernel<false><<<grid, kThreads, kSmemBytes, s>>>(tm_h, tm_w_z, tm_w_n, tm_dh, tm_dw, a);
  return cudaGetLastError();
}

}  // namespace molt
