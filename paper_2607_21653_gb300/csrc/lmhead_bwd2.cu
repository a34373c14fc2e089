// Backward pass of the fused LM-head + clipped-surrogate loss on CTA pairs
// (tcgen05 cta_group::2), used when H is a multiple of 256.
//
//   g_tv = coef_t (softmax(z_t)_v - [v == x_t]),  coef_t = m_t c_t / D   (Eq. 2)
//          (+ ecoef_t softmax(z_t)_v (z_tv - mu_t) with an entropy bonus)
//   dH_t = sum_v g_tv W_v          dW_v = sum_t g_tv h_t
//
// A pair unit is 256 active token rows (two 128-row tiles, one per CTA) times a
// 256-column vocab chunk.  Compared with one CTA per 128 x 256 unit this halves
// the operand bytes each SM loads (each CTA stages half of every B operand) and
// doubles the reduction depth of dW (256 tokens), so each SM drains
// 4 B x H x (128 + 128) of partial products per unit instead of
// 4 B x H x (128 + 256): the reduce-add traffic to L2 that bounds the
// single-CTA kernel drops by a third per flop.
//
//   job Z   z = h W_j^T: pair MMA M=256 (tokens; CTA r holds its 128 rows),
//           N=256 (vocab; CTA r stages W rows v0 + 128 r ...), K=H.  Each CTA's
//           TMEM holds its 128 tokens x 256 vocab.
//   g       each CTA turns its z rows into g (bf16) and stores them twice in the
//           128-byte swizzle: GH = own tokens x 256 vocab (K-major A of dH) and
//           GW = all 256 tokens x 128 vocab of one half (MN-major A of dW).  The
//           GW rows for the peer's vocab half are written into the peer's
//           shared memory (distributed shared memory).
//   job dH  per 128 columns of H: pair MMA M=256 tokens, N=128, K=256 vocab;
//           B = W_j rows, MN-major, CTA r staging columns 64 r .. 64 r + 63.
//   job dW  per 128 columns of H: pair MMA M=256 vocab (CTA r: half r),
//           N=128, K=256 tokens; B = h rows of both tiles, MN-major.
// Partial products drain through swizzled 32 x 32 fp32 boxes with TMA
// reduce-add into the fp32 dhidden accumulator and dW.
//
// Schedule.  Each SM can push only ~25 B/clock of reduce-adds to L2, and a
// unit's drains (4 B x H x 256 per CTA) take longer than its products, so the
// drain path must never idle.  TMEM holds one 256-column Z buffer and a ring of
// two 128-column job accumulators; the MMA issuer interleaves the K-blocks of
// the NEXT unit's Z between the current unit's dH/dW jobs (H/64 of each, one
// after the other), so the next logits accumulate while the epilogue drains.
//
// Roles per CTA (192 threads): warp 0 TMA producer (both CTAs load their
// halves; bytes complete on the even CTA's barrier), warp 1 MMA issuer (even
// CTA only) and TMEM owner, warps 2-5 epilogue.
#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

#include "molt_internal.cuh"
#include "ptx.cuh"

namespace molt {
namespace {

constexpr int kStages = 2;
constexpr int kStageBytes = 32 * 1024;
constexpr int kSub = kTileM * kBK * 2;            // [128 rows x 64] bf16 sub-tile, 16 KB
constexpr int kOffGH = kStages * kStageBytes;     // 64 KB
constexpr int kOffGW = kOffGH + 4 * kSub;         // 128 KB
constexpr int kGWBlock = 2 * kSub;                // [256 rows x 64] bf16, 32 KB
constexpr int kOffBox = kOffGW + 2 * kGWBlock;    // 192 KB
constexpr int kBoxBytes = 32 * 32 * 4;
constexpr int kBoxesPerWarp = 2;
constexpr int kThreads = 192;
constexpr int kSmemBytes = 1024 + kOffBox + 4 * kBoxesPerWarp * kBoxBytes;
constexpr uint32_t kIdescZ = idesc_bf16_f32(256, 256, false, false);
constexpr uint32_t kIdescH = idesc_bf16_f32(256, 128, false, true);
constexpr uint32_t kIdescW = idesc_bf16_f32(256, 128, true, true);
constexpr uint32_t kZCol = 0;      // TMEM columns [0, 256): Z buffer
constexpr uint32_t kAccCol = 256;  // [256, 384), [384, 512): job accumulators
constexpr uint32_t kStageTx = 2u * kStageBytes;   // bytes both CTAs load per stage
constexpr float kLog2e = 1.4426950408889634f;

struct PairUnit {
  int tp;   // tile pair index
  int vc;   // vocab chunk
};

// raster: tile pairs in groups of `group`; inside a group consecutive units walk
// the group's pairs for one vocab chunk, then move to the next chunk
__device__ __forceinline__ PairUnit pair_unit_of(int u, int n_tp, int n_vc, int group) {
  const int per_group = group * n_vc;
  const int g = u / per_group;
  const int r = u - g * per_group;
  const int g_pairs = min(group, n_tp - g * group);
  const int vc = r / g_pairs;
  return {g * group + (r - vc * g_pairs), vc};
}

__device__ __forceinline__ void write_box32(uint32_t box, int lane, const float (&v)[32]) {
  const uint32_t rowp = box + lane * 128;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const uint32_t pos = static_cast<uint32_t>(i ^ (lane & 7));
    st_shared_v4(rowp + pos * 16, __float_as_uint(v[4 * i]), __float_as_uint(v[4 * i + 1]),
                 __float_as_uint(v[4 * i + 2]), __float_as_uint(v[4 * i + 3]));
  }
}

template <bool kEnt>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    lmhead_bwd_pair_kernel(const __grid_constant__ CUtensorMap tm_h, const __grid_constant__ CUtensorMap tm_wz,
                           const __grid_constant__ CUtensorMap tm_wn, const __grid_constant__ CUtensorMap tm_dh,
                           const __grid_constant__ CUtensorMap tm_dw, const BwdArgs a) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[kStages];    // even CTA: both CTAs' bytes land here
  __shared__ __align__(8) uint64_t empty_bar[kStages];   // both CTAs, committed by the even CTA
  __shared__ __align__(8) uint64_t accf_bar[2];          // both CTAs: job accumulator full
  __shared__ __align__(8) uint64_t acce_bar[2];          // even CTA: 256 epilogue arrivals
  __shared__ __align__(8) uint64_t zfull_bar;            // both CTAs: Z buffer complete
  __shared__ __align__(8) uint64_t gready_bar;           // even CTA: g written, Z buffer read (256)
  __shared__ __align__(8) uint64_t done_bar;
  __shared__ uint32_t tmem_base_sh;
  __shared__ int abort_sh;

  const uint32_t smem0 = (smem_u32(smem_raw) + 1023u) & ~1023u;
  const uint32_t gh_base = smem0 + kOffGH;
  const uint32_t gw_base = smem0 + kOffGW;
  const uint32_t box_base = smem0 + kOffBox;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const uint32_t peer = rank ^ 1u;
  const bool leader = rank == 0;
  volatile int* abort_flag = &abort_sh;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(smem_u32(&full_bar[s]), 1);
      mbar_init(smem_u32(&empty_bar[s]), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(smem_u32(&accf_bar[b]), 1);
      mbar_init(smem_u32(&acce_bar[b]), 256);
    }
    mbar_init(smem_u32(&zfull_bar), 1);
    mbar_init(smem_u32(&gready_bar), 256);
    mbar_init(smem_u32(&done_bar), 1);
    abort_sh = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc_pair(smem_u32(&tmem_base_sh), 512);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();   // both CTAs' barriers exist before any remote arrival
  tc_fence_after();
  const uint32_t tmem_base = tmem_base_sh;

  const int n_tiles = a.counts[1];
  const int n_tp = (n_tiles + 1) / 2;
  const int n_vc = a.n_vchunks;
  const int n_units = n_tp * n_vc;
  const int H = a.H, V = a.V;
  const int nZ = H / kBK;        // Z K-blocks per unit
  const int nJ = H / kBK;        // jobs per unit: H/128 dH jobs, then H/128 dW jobs
  const int nJH = H / 128;
  const int pair = blockIdx.x >> 1, n_pairs = gridDim.x >> 1;

  if (warp == 0) {
    if (lane == 0) {
      prefetch_tmap(&tm_h);
      prefetch_tmap(&tm_wz);
      prefetch_tmap(&tm_wn);
      uint32_t full_leader[kStages];
      for (int s = 0; s < kStages; ++s) full_leader[s] = mapa_shared(smem_u32(&full_bar[s]), 0);
      uint32_t it = 0;
      bool ok = true;
      // wait for a free stage; the even CTA announces both CTAs' bytes
      auto next_stage = [&](uint32_t& sa, uint32_t& fb) -> bool {
        const uint32_t st = it % kStages, ph = (it / kStages) & 1u;
        if (!mbar_wait(smem_u32(&empty_bar[st]), ph ^ 1u, abort_flag, a.err)) return false;
        sa = smem0 + st * kStageBytes;
        fb = full_leader[st];
        if (leader) mbar_arrive_expect_tx(smem_u32(&full_bar[st]), kStageTx);
        ++it;
        return true;
      };
      auto rows_of = [&](int u, int& ta, int& tb, int& v0) {
        const PairUnit un = pair_unit_of(u, n_tp, n_vc, a.tile_group);
        ta = a.tile_list[2 * un.tp];
        tb = (2 * un.tp + 1 < n_tiles) ? a.tile_list[2 * un.tp + 1] : ta;
        v0 = un.vc * 256;
      };
      auto load_z = [&](int kb, int own_row0, int v0) -> bool {
        uint32_t sa, fb;
        if (!next_stage(sa, fb)) return false;
        tma_load_2d_pair(sa, &tm_h, fb, kb * kBK, own_row0);
        tma_load_2d_pair(sa + kSub, &tm_wz, fb, kb * kBK, v0 + static_cast<int>(rank) * 128);
        return true;
      };
      int u = pair;
      if (u < n_units) {
        int ta, tb, v0;
        rows_of(u, ta, tb, v0);
        for (int kb = 0; kb < nZ && ok; ++kb) ok = load_z(kb, (rank ? tb : ta) * kTileM, v0);
      }
      for (; u < n_units && ok; u += n_pairs) {
        int ta, tb, v0;
        rows_of(u, ta, tb, v0);
        const int un_next = u + n_pairs;
        int nta = 0, ntb = 0, nv0 = 0;
        if (un_next < n_units) rows_of(un_next, nta, ntb, nv0);
        for (int i = 0; i < nJ && ok; ++i) {
          uint32_t sa, fb;
          if (!(ok = next_stage(sa, fb))) break;
          if (i < nJH) {   // dH job: W rows v0 .. v0+255, this CTA's 64 of 128 columns
            const int x = i * 128 + static_cast<int>(rank) * 64;
            for (int vb = 0; vb < 4; ++vb) tma_load_2d_pair(sa + vb * 8192, &tm_wn, fb, x, v0 + vb * 64);
          } else {         // dW job: h rows of both tiles, this CTA's 64 of 128 columns
            const int x = (i - nJH) * 128 + static_cast<int>(rank) * 64;
            tma_load_2d_pair(sa, &tm_h, fb, x, ta * kTileM);
            tma_load_2d_pair(sa + 16384, &tm_h, fb, x, tb * kTileM);
          }
          if (un_next < n_units) ok = load_z(i, (rank ? ntb : nta) * kTileM, nv0);
        }
      }
      if (leader) {
        // every copy of both CTAs completes on these barriers: wait for the
        // last issued stages before the pair may exit
        const uint32_t first = it > (uint32_t)kStages ? it - kStages : 0u;
        for (uint32_t j = first; j < it; ++j)
          mbar_wait_drain(smem_u32(&full_bar[j % kStages]), (j / kStages) & 1u, a.err);
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && leader) {
      uint32_t it = 0, jj = 0, unit_it = 0;
      bool ok = true;
      auto wait_stage = [&](uint32_t& sa) -> bool {
        const uint32_t st = it % kStages, ph = (it / kStages) & 1u;
        if (!mbar_wait_cluster(smem_u32(&full_bar[st]), ph, abort_flag, a.err)) return false;
        tc_fence_after();
        sa = smem0 + st * kStageBytes;
        return true;
      };
      auto release_stage = [&]() {
        umma_commit_pair_mc(smem_u32(&empty_bar[it % kStages]), 3);
        ++it;
      };
      // one Z K-block into the Z buffer
      auto z_block = [&](int kb) -> bool {
        uint32_t sa;
        if (!wait_stage(sa)) return false;
        const uint64_t ad = sdesc_sw128(sa, 16, 1024);
        const uint64_t bd = sdesc_sw128(sa + kSub, 16, 1024);
#pragma unroll
        for (int k = 0; k < kBK / 16; ++k)
          umma_bf16_pair(tmem_base + kZCol, ad + 2u * k, bd + 2u * k, kIdescZ, (kb | k) != 0 ? 1u : 0u);
        release_stage();
        if (kb == nZ - 1) umma_commit_pair_mc(smem_u32(&zfull_bar), 3);
        return true;
      };
      int u = pair;
      if (u < n_units)
        for (int kb = 0; kb < nZ && ok; ++kb) ok = z_block(kb);
      for (; u < n_units && ok; u += n_pairs) {
        const bool has_next = u + n_pairs < n_units;
        // g of this unit in shared memory, and the Z buffer free again
        if (!(ok = mbar_wait_cluster(smem_u32(&gready_bar), unit_it & 1u, abort_flag, a.err))) break;
        tc_fence_after();
        for (int i = 0; i < nJ && ok; ++i) {
          const uint32_t buf = jj & 1u, aph = (jj >> 1) & 1u;
          if (!(ok = mbar_wait_cluster(smem_u32(&acce_bar[buf]), aph ^ 1u, abort_flag, a.err))) break;
          tc_fence_after();
          const uint32_t d = tmem_base + kAccCol + buf * 128;
          uint32_t sa;
          if (!(ok = wait_stage(sa))) break;
          if (i < nJH) {
            // dH: A = g (own tokens x 256 vocab, K-major), B = W rows (MN-major)
#pragma unroll
            for (int k = 0; k < 16; ++k) {
              const int vb = k >> 2, kk = k & 3;
              const uint64_t ad = sdesc_sw128(gh_base + vb * kSub, 16, 1024) + 2u * kk;
              const uint64_t bd = sdesc_sw128(sa + vb * 8192 + kk * 2048, 8192, 1024);
              umma_bf16_pair(d, ad, bd, kIdescH, k != 0 ? 1u : 0u);
            }
          } else {
            // dW: A = g^T (this CTA's 128 vocab x 256 tokens, MN-major), B = h rows (MN-major)
#pragma unroll
            for (int k = 0; k < 16; ++k) {
              const int tt = k >> 3, kk = k & 7;
              const uint64_t ad = sdesc_sw128(gw_base + (tt * 8 + kk) * 2048, kGWBlock, 1024);
              const uint64_t bd = sdesc_sw128(sa + tt * 16384 + kk * 2048, 16384, 1024);
              umma_bf16_pair(d, ad, bd, kIdescW, k != 0 ? 1u : 0u);
            }
          }
          release_stage();
          umma_commit_pair_mc(smem_u32(&accf_bar[buf]), 3);
          ++jj;
          if (has_next) ok = z_block(i);
        }
        ++unit_it;
      }
      umma_commit_pair_mc(smem_u32(&done_bar), 1);
      mbar_wait_drain(smem_u32(&done_bar), 0, a.err);
    }
  } else {
    const int q = warp & 3;
    const int r_in = q * 32 + lane;                       // own row = TMEM lane
    const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
    const uint32_t box0 = box_base + (warp - 2) * kBoxesPerWarp * kBoxBytes;
    const uint32_t acce_leader0 = mapa_shared(smem_u32(&acce_bar[0]), 0);
    const uint32_t acce_leader1 = mapa_shared(smem_u32(&acce_bar[1]), 0);
    const uint32_t gready_leader = mapa_shared(smem_u32(&gready_bar), 0);
    const uint32_t gw_peer = mapa_shared(gw_base, peer);
    uint32_t jj = 0, nbox = 0, unit_it = 0;
    bool ok = true;
    // one [32 x 32] fp32 slab of this warp's rows -> reduce-add into global
    auto drain_slab = [&](const CUtensorMap* map, uint32_t taddr, int x, int y, bool issue) {
      float v[32];
      tmem_ld32(taddr, v);
      const uint32_t box = box0 + (nbox & (kBoxesPerWarp - 1)) * kBoxBytes;
      if (lane == 0) bulk_wait_group_read<kBoxesPerWarp - 1>();
      __syncwarp();
      write_box32(box, lane, v);
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0 && issue) tma_reduce_add_2d(map, box, x, y);
      if (lane == 0) bulk_commit_group();
      ++nbox;
    };
    for (int u = pair; u < n_units && ok; u += n_pairs) {
      const PairUnit un = pair_unit_of(u, n_tp, n_vc, a.tile_group);
      const int ta = a.tile_list[2 * un.tp];
      const bool b_null = (2 * un.tp + 1 >= n_tiles);
      const int tb = b_null ? ta : a.tile_list[2 * un.tp + 1];
      const bool own_null = rank && b_null;              // odd CTA without a tile: g rows are 0
      const int own_row0 = (rank ? tb : ta) * kTileM;
      const int v0 = un.vc * 256;
      const int row = own_row0 + r_in;
      const float coef = own_null ? 0.f : a.coef[row];
      float ecoef = 0.f, mu = 0.f;
      if constexpr (kEnt) {
        if (!own_null) {
          ecoef = a.ecoef[row];
          mu = a.mu[row];
        }
      }
      const bool live = kEnt ? (coef != 0.f || ecoef != 0.f) : (coef != 0.f);
      const float lseL = live ? a.lse[row] * kLog2e : 0.f;
      const int lx = a.tok_p[row] - v0;
      const int R = static_cast<int>(rank) * 128 + r_in;   // row of this token in GW
      // Z buffer -> g in GH (own tokens x 256 vocab) and GW (this / the peer CTA)
      if (!(ok = mbar_wait(smem_u32(&zfull_bar), unit_it & 1u, abort_flag, a.err))) break;
      tc_fence_after();
      const uint32_t zaddr = tmem_base + lane_off + kZCol;
#pragma unroll 1
      for (int c0 = 0; c0 < 256; c0 += 32) {
        float v[32];
        tmem_ld32(zaddr + c0, v);
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
        const int c = c0 >> 6;                  // vocab 64-chunk 0..3
        const int cc0 = (c0 & 63) >> 3;         // first 16-byte chunk in the row
        const uint32_t gh_row = gh_base + c * kSub + r_in * 128;
        const uint32_t gw_off = static_cast<uint32_t>((c & 1) * kGWBlock + R * 128);
        const bool local_half = (c >> 1) == static_cast<int>(rank);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const uint32_t pos = static_cast<uint32_t>(((cc0 + i) ^ (r_in & 7)) * 16);
          st_shared_v4(gh_row + pos, w[4 * i], w[4 * i + 1], w[4 * i + 2], w[4 * i + 3]);
          if (local_half)
            st_shared_v4(gw_base + gw_off + pos, w[4 * i], w[4 * i + 1], w[4 * i + 2], w[4 * i + 3]);
          else
            st_shared_cluster_v4(gw_peer + gw_off + pos, w[4 * i], w[4 * i + 1], w[4 * i + 2], w[4 * i + 3]);
        }
      }
      fence_proxy_async_cluster();
      tc_fence_before();
      mbar_arrive_cluster(gready_leader);
      // jobs: dH for 128 columns of H at a time, then dW
      const int vrow = v0 + static_cast<int>(rank) * 128 + q * 32;
      for (int i = 0; i < nJ && ok; ++i) {
        const uint32_t buf = jj & 1u, aph = (jj >> 1) & 1u;
        if (!(ok = mbar_wait(smem_u32(&accf_bar[buf]), aph, abort_flag, a.err))) break;
        tc_fence_after();
        const uint32_t taddr = tmem_base + lane_off + kAccCol + buf * 128;
        if (i < nJH) {
          for (int c0 = 0; c0 < 128; c0 += 32)
            drain_slab(&tm_dh, taddr + c0, i * 128 + c0, own_row0 + q * 32, !own_null);
        } else {
          for (int c0 = 0; c0 < 128; c0 += 32)
            drain_slab(&tm_dw, taddr + c0, (i - nJH) * 128 + c0, vrow, vrow < V);
        }
        // the accumulator was read with tcgen05.ld + wait::ld; a relaxed arrive
        // after the tcgen05 fence is enough to hand it back to the MMA issuer
        tc_fence_before();
        mbar_arrive_cluster_relaxed(buf ? acce_leader1 : acce_leader0);
        ++jj;
      }
      ++unit_it;
    }
    if (lane == 0) bulk_wait_group<0>();
    __syncwarp();
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync_all();   // no CTA leaves while its peer may still touch its memory
  tc_fence_after();
  if (warp == 1) {
    __syncwarp();
    tmem_dealloc_pair(tmem_base, 512);
  }
}

}  // namespace

int lmhead_bwd_pair_max_clusters(int n_sm) {
  static int cached = -1;
  if (cached >= 0) return cached;
  cudaError_t e =
      cudaFuncSetAttribute(lmhead_bwd_pair_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
  if (e != cudaSuccess) return 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(n_sm, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = kSmemBytes;
  int n = 0;
  e = cudaOccupancyMaxActiveClusters(&n, lmhead_bwd_pair_kernel<false>, &cfg);
  if (e != cudaSuccess) {
    cudaGetLastError();
    n = n_sm / 2;
  }
  cached = n;
  return n;
}

cudaError_t launch_lmhead_bwd_pair(const CUtensorMap& tm_h, const CUtensorMap& tm_w_z128, const CUtensorMap& tm_w_n,
                                   const CUtensorMap& tm_dh, const CUtensorMap& tm_dw, const BwdArgs& a, int n_sm,
                                   cudaStream_t s) {
  const bool ent = a.ecoef != nullptr;
  cudaError_t e = ent ? cudaFuncSetAttribute(lmhead_bwd_pair_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             kSmemBytes)
                      : cudaFuncSetAttribute(lmhead_bwd_pair_kernel<false>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
  if (e != cudaSuccess) return e;
  int clusters = lmhead_bwd_pair_max_clusters(n_sm);
  if (clusters > n_sm / 2) clusters = n_sm / 2;
  if (clusters < 1) clusters = 1;
  if (ent)
    lmhead_bwd_pair_kernel<true><<<2 * clusters, kThreads, kSmemBytes, s>>>(tm_h, tm_w_z128, tm_w_n, tm_dh, tm_dw, a);
  else
    lmhead_bwd_pair_kernel<false><<<2 * clusters, kThreads, kSmemBytes, s>>>(tm_h, tm_w_z128, tm_w_n, tm_dh, tm_dw, a);
  return cudaGetLastError();
}

}  // namespace molt
