// Backward pass of the fused LM-head + policy loss on clusters of four CTAs
// (two tcgen05 CTA pairs), used when H is a multiple of 128.
//
//   g_tv = coef_t (softmax(z_t)_v - [v == x_t]),  coef_t = m_t c_t / D   (Eq. 2)
//          (+ ecoef_t softmax(z_t)_v (z_tv - mu_t) with an entropy bonus)
//   dH_t = sum_v g_tv W_v          dW_v = sum_t g_tv h_t
//
// Why clusters of four.  The products of a unit are partial sums over its
// slice of the reduction dimension (vocab for dH, tokens for dW), so every unit
// drains H-wide fp32 rows into global memory with reduce-adds.  Those drains,
// together with the operand loads, go through each SM's request path to L2,
// which moves about 32 B per clock; with 256 x 256 units that path, not the
// tensor cores, was the limit.  A unit of Tu tokens x Vu vocab drains 4 H (Tu + Vu) bytes
// for 6 Tu Vu H flops, so larger units drain less per flop.  The on-chip state
// that has to grow with the unit is g, which is small (bf16, no H dimension):
// here a unit is 512 tokens x 512 vocab on four CTAs, twice as deep in both
// reductions as a 256 x 256 unit on one CTA pair, which halves the drain bytes
// per flop.  The price is moving g between the CTAs through distributed shared
// memory (96 KB per CTA per unit, against 4 MB of drains).
//
// Layout of a unit.  CTA k (cluster rank k = 0..3) owns token tile k of the
// unit's four 128-row tiles and vocab quarter k (columns v0 + 128 k ...).  Pair
// p = k / 2 (CTAs 2p, 2p+1) computes, on the tensor cores of both its SMs:
//   Z      z = h W^T for its two token tiles x all 512 vocab, as two pair MMAs
//          of M = 256 tokens, N = 256 vocab (Z_a: vocab 0..255, Z_b: 256..511),
//          K = H.  Each CTA's TMEM receives its 128 tokens x 256 vocab.
//   g      each CTA turns z into g (bf16): into TMEM (its 128 tokens x 512 vocab,
//          256 columns, the A operand of dH) and into the GW buffers of all four
//          CTAs: the GW of CTA q holds g of all 512 tokens x vocab quarter q
//          (MN-major A operand of dW), filled by every CTA for its own tokens.
//   dH     per 256 columns of H: pair MMA M = 256 tokens, N = 256, K = 512 vocab;
//          A = g from TMEM, B = W rows (MN-major), CTA r staging columns
//          128 r .. 128 r + 127.
//   dW     per 256 columns of H: pair MMA M = 256 vocab (the pair's two
//          quarters), N = 256, K = 512 tokens; A = GW, B = h rows of all four
//          tiles (MN-major).
// Partial products drain through swizzled 32 x 32 fp32 boxes with TMA
// reduce-add into the fp32 dhidden accumulator and dW.
//
// TMEM (512 columns per CTA): [0, 256) g; [256, 512) the job accumulator.  Z_a
// accumulates over [0, 256) and is converted to g in place (column c of z ->
// column c / 2 of g), so Z_a of the next unit is computed while the current dW
// products run; Z_b accumulates over the accumulator's columns once they are
// idle and is converted into g columns [128, 256) after Z_a's conversion has
// read them.  The job products are N = 256 because a pair MMA of N = 128 takes about
// 1.6x its ideal clocks and one of N = 256 its ideal 128; that leaves room for a
// single accumulator, which eight epilogue warps copy to registers (128 columns
// each) and hand back before draining it.  During the dW products the next
// unit's Z_a stages fill the MMA issuer's wait for that hand-back.
//
// Operands stream through a ring of four 16 KB stages.  Every stage is a round
// trip (the MMA frees it, the producer refills it from L2), and the ring's
// bytes in flight over that latency set the rate at which operands arrive, so
// the ring is cut fine: a logit stage holds K = 32 of h and W in the 64-byte
// swizzle, a dH stage 64 vocab rows x 128 columns of W, a dW stage 64 token
// rows x 128 columns of h.  The MMA issuer waits for operand stages about a
// quarter of the time, yet no unit on the way is saturated: each SM's
// interface to the crossbar is the busiest (about two thirds, mostly the
// reduce-add payload at one cycle per 32-byte sector, the load requests at one
// cycle each), which caps the kernel near 70 % of the tensor roofline, and the
// rest is the latency of the unit's chain of dependencies.  More stages (a
// fifth one paid for with smaller drain boxes, six with the drains issued from
// registers) and multicasting the operands both pairs load did not make it
// faster.
//
// Roles per CTA (320 threads): warp 0 TMA producer (each CTA loads its half of
// every operand; bytes complete on the pair leader's barrier), warp 1 MMA issuer
// (pair leaders only) and TMEM owner, warps 2-9 epilogue, two per TMEM lane
// quarter (warp w reads lanes 32 (w % 4) .. 32 (w % 4) + 31, column half
// (w - 2) / 4).
#include <atomic>
#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

#include "molt_internal.cuh"
#include "ptx.cuh"

namespace molt {
namespace {

constexpr int kStages = 4;
constexpr int kStageBytes = 16 * 1024;
constexpr int kSub = kTileM * kBK * 2;            // [128 rows x 64] bf16 sub-tile, 16 KB
constexpr int kZK = 32;                           // K per logit stage (64-byte swizzle rows)
constexpr int kOffGW = kStages * kStageBytes;     // 64 KB (1024-aligned)
constexpr int kGWBlock = 4 * kSub;                // [512 token rows x 64 vocab] bf16, 64 KB
constexpr int kOffBox = kOffGW + 2 * kGWBlock;    // 192 KB
constexpr int kBoxBytes = 32 * 32 * 4;
constexpr int kEpiWarps = 8;                      // two per TMEM lane quarter
constexpr int kBoxesPerWarp = 1;
constexpr int kThreads = 64 + 32 * kEpiWarps;
constexpr int kEpiThreads = 32 * kEpiWarps;
constexpr int kSmemBytes = 1024 + kOffBox + kEpiWarps * kBoxesPerWarp * kBoxBytes;
constexpr uint32_t kIdescZ = idesc_bf16_f32(256, 256, false, false);
constexpr uint32_t kIdescH = idesc_bf16_f32(256, 256, false, true);   // A from TMEM
constexpr uint32_t kIdescW = idesc_bf16_f32(256, 256, true, true);
constexpr uint32_t kIdescH128 = idesc_bf16_f32(256, 128, false, true);   // the last job when H % 256 == 128
constexpr uint32_t kIdescW128 = idesc_bf16_f32(256, 128, true, true);
constexpr uint32_t kGCol = 0;       // g: 128 tokens x 512 vocab as bf16 pairs
constexpr uint32_t kZaCol = 0;      // Z of vocab 0..255
constexpr uint32_t kZbCol = 256;    // Z of vocab 256..511 (over the idle accumulator)
constexpr uint32_t kAccCol = 256;   // one 256-column job accumulator
constexpr uint32_t kStageTx = 2u * kStageBytes;   // bytes both CTAs of a pair load per stage
constexpr float kLog2e = 1.4426950408889634f;

struct QuadUnit {
  int tq;   // token-tile quad
  int vp;   // 512-column vocab block
};

// raster: tile quads in groups of `group`; inside a group consecutive units walk
// the group's quads for one vocab block, then move to the next block
__device__ __forceinline__ QuadUnit quad_unit_of(int u, int n_tq, int n_vp, int group) {
  const int per_group = group * n_vp;
  const int g = u / per_group;
  const int r = u - g * per_group;
  const int g_q = min(group, n_tq - g * group);
  const int vp = r / g_q;
  return {g * group + (r - vp * g_q), vp};
}

// The units one cluster processes, in order.  Raster schedule: unit u = quad,
// quad + n_quads, ... of quad_unit_of.  Deterministic schedule (det > 0 = the
// number of clusters, a multiple of 4): cluster c takes quad slot s = c % 4 of
// every group of four token quads and the vocab blocks m, m + det / 4, ... with
// m = c / 4; it walks the groups in order and, inside a group, its blocks in
// order.  The four clusters of a class then work on the same vocab block, one
// quad each, and the det / 4 classes of a slot on consecutive blocks of one
// quad, as in the raster with groups of four quads; the reduce-adds into a dW
// row take turns in quad order, those into a dhidden row in block order (see
// the epilogue).
struct UnitSeq {
  int n_tq, n_vp, n_q, group, det;
  int u;                     // raster position
  int g, b, slot, m, n_m;    // deterministic: group, vocab block, quad slot, class, classes
  __device__ __forceinline__ void init(int quad, int n_quads, int ntq, int nvp, int grp, int ndet) {
    n_tq = ntq;
    n_vp = nvp;
    n_q = n_quads;
    group = grp;
    det = ndet;
    u = quad;
    slot = quad & 3;
    m = quad >> 2;
    n_m = ndet >> 2;
    g = 0;
    b = m;
    settle();
  }
  __device__ __forceinline__ void settle() {   // skip groups without a quad in this slot
    if (det > 0)
      while (4 * g < n_tq && (4 * g + slot >= n_tq || b >= n_vp)) {
        ++g;
        b = m;
      }
  }
  __device__ __forceinline__ bool valid() const {
    return det > 0 ? (4 * g + slot < n_tq && b < n_vp) : (u < n_tq * n_vp);
  }
  __device__ __forceinline__ QuadUnit cur() const {
    return det > 0 ? QuadUnit{4 * g + slot, b} : quad_unit_of(u, n_tq, n_vp, group);
  }
  __device__ __forceinline__ void advance() {
    if (det == 0) {
      u += n_q;
      return;
    }
    b += n_m;
    if (b >= n_vp) {
      ++g;
      b = m;
    }
    settle();
  }
};

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
__global__ void __cluster_dims__(4, 1, 1) __launch_bounds__(kThreads, 1)
    lmhead_bwd_quad_kernel(const __grid_constant__ CUtensorMap tm_hz, const __grid_constant__ CUtensorMap tm_wz,
                           const __grid_constant__ CUtensorMap tm_h, const __grid_constant__ CUtensorMap tm_wn,
                           const __grid_constant__ CUtensorMap tm_dh, const __grid_constant__ CUtensorMap tm_dw,
                           const BwdArgs a) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[kStages];   // pair leader: both CTAs' bytes land here
  __shared__ __align__(8) uint64_t empty_bar[kStages];  // both CTAs of the pair
  __shared__ __align__(8) uint64_t accf_bar;            // both CTAs of the pair: accumulator full
  __shared__ __align__(8) uint64_t acce_bar;            // pair leader: one arrival per epilogue warp of the pair (copied out)
  __shared__ __align__(8) uint64_t zfa_bar;             // every CTA: Z_a done in both pairs (2 commits)
  __shared__ __align__(8) uint64_t zfb_bar;             // every CTA: Z_b done in both pairs (2 commits)
  __shared__ __align__(8) uint64_t zfo_bar;             // every CTA: Z_b done in its own pair (1 commit)
  __shared__ __align__(8) uint64_t tb_bar;              // pair leader: Z_b read, g_b in TMEM (both CTAs' epilogues)
  __shared__ __align__(8) uint64_t gw_bar;              // pair leader: both GW buffers of the pair full (all 4 CTAs)
  __shared__ __align__(8) uint64_t dhd_bar;             // pair leader: this unit's dH products done
  __shared__ __align__(8) uint64_t done_bar;
  __shared__ __align__(8) uint64_t qsync_bar[4];        // the two epilogue warps of each lane quarter
  __shared__ uint32_t tmem_base_sh;
  __shared__ int abort_sh;

  const uint32_t smem0 = (smem_u32(smem_raw) + 1023u) & ~1023u;
  const uint32_t gw_base = smem0 + kOffGW;
  const uint32_t box_base = smem0 + kOffBox;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();   // token tile and vocab quarter of this CTA
  const uint32_t prank = rank & 1u;          // rank inside the pair
  const uint32_t lead = rank & ~1u;          // the pair leader's rank
  const bool leader = prank == 0;
  const uint16_t pair_mask = static_cast<uint16_t>(3u << lead);
  volatile int* abort_flag = &abort_sh;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(smem_u32(&full_bar[s]), 1);
      mbar_init(smem_u32(&empty_bar[s]), 1);
    }
    mbar_init(smem_u32(&accf_bar), 1);
    mbar_init(smem_u32(&acce_bar), 2 * kEpiWarps);
    mbar_init(smem_u32(&zfa_bar), 2);
    mbar_init(smem_u32(&zfb_bar), 2);
    mbar_init(smem_u32(&zfo_bar), 1);
    mbar_init(smem_u32(&tb_bar), 2 * kEpiThreads);
    mbar_init(smem_u32(&gw_bar), 4 * kEpiThreads);
    mbar_init(smem_u32(&dhd_bar), 1);
    mbar_init(smem_u32(&done_bar), 1);
    for (int i = 0; i < 4; ++i) mbar_init(smem_u32(&qsync_bar[i]), 64);
    abort_sh = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc_pair(smem_u32(&tmem_base_sh), 512);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();   // every CTA's barriers exist before any remote arrival
  tc_fence_after();
  const uint32_t tmem_base = tmem_base_sh;

  const int n_tiles = a.counts[1];
  const int n_tq = (n_tiles + 3) / 4;
  const int n_vp = (a.V + 511) / 512;
  const int H = a.H, V = a.V;
  const int nZ = H / kZK;        // logit stages per vocab half (4 per dW job)
  const int nJ = (H + 255) / 256;   // dH jobs = dW jobs per unit
  // columns of H job j covers: 256, except a last job of 128 when H % 256 == 128
  auto job_w = [&](int j) -> int { return (H & 255) != 0 && j == nJ - 1 ? 128 : 256; };
  const int quad = blockIdx.x >> 2, n_quads = gridDim.x >> 2;

  // token tile k of unit tq (a missing tile reads tile 0's rows; its g is 0)
  auto tile_of = [&](int tq, int k) -> int {
    const int i = 4 * tq + k;
    return a.tile_list[i < n_tiles ? i : 4 * tq];
  };

  if (warp == 0) {
    if (lane == 0) {
      prefetch_tmap(&tm_hz);
      prefetch_tmap(&tm_wz);
      prefetch_tmap(&tm_h);
      prefetch_tmap(&tm_wn);
      uint32_t full_leader[kStages];
      for (int s = 0; s < kStages; ++s) full_leader[s] = mapa_shared(smem_u32(&full_bar[s]), lead);
      uint32_t it = 0;
      bool ok = true;
      auto next_stage = [&](uint32_t& sa, uint32_t& fb, uint32_t tx = kStageTx) -> bool {
        const uint32_t st = it % kStages, ph = (it / kStages) & 1u;
        if (!mbar_wait(smem_u32(&empty_bar[st]), ph ^ 1u, abort_flag, a.err)) return false;
        sa = smem0 + st * kStageBytes;
        fb = full_leader[st];
        if (leader) mbar_arrive_expect_tx(smem_u32(&full_bar[st]), tx);
        ++it;
        return true;
      };
      // one logit stage: K = 32 of the own token rows and of this CTA's 128 of
      // the half's 256 vocab rows
      auto load_z = [&](int kb, int own_row0, int vrow0) -> bool {
        uint32_t sa, fb;
        if (!next_stage(sa, fb)) return false;
        tma_load_2d_pair(sa, &tm_hz, fb, kb * kZK, own_row0);
        tma_load_2d_pair(sa + kStageBytes / 2, &tm_wz, fb, kb * kZK, vrow0 + static_cast<int>(prank) * 128);
        return true;
      };
      UnitSeq seq;
      seq.init(quad, n_quads, n_tq, n_vp, a.tile_group, a.det_clusters);
      if (seq.valid()) {
        const QuadUnit un = seq.cur();
        const int own_row0 = tile_of(un.tq, static_cast<int>(rank)) * kTileM;
        for (int kb = 0; kb < nZ && ok; ++kb) ok = load_z(kb, own_row0, un.vp * 512);
      }
      for (; seq.valid() && ok; seq.advance()) {
        const QuadUnit un = seq.cur();
        const int v0 = un.vp * 512;
        const int own_row0 = tile_of(un.tq, static_cast<int>(rank)) * kTileM;
        int t4[4];
        for (int k = 0; k < 4; ++k) t4[k] = tile_of(un.tq, k) * kTileM;
        UnitSeq nseq = seq;
        nseq.advance();
        const bool has_next = nseq.valid();
        int n_row0 = 0, n_v0 = 0;
        if (has_next) {
          const QuadUnit nu = nseq.cur();
          n_row0 = tile_of(nu.tq, static_cast<int>(rank)) * kTileM;
          n_v0 = nu.vp * 512;
        }
        // Z_b of this unit
        for (int kb = 0; kb < nZ && ok; ++kb) ok = load_z(kb, own_row0, v0 + 256);
        // dH jobs: W rows of the unit's 512 vocab, 64 per stage, this CTA's 128
        // of the job's 256 columns
        for (int i = 0; i < nJ && ok; ++i) {
          const int w = job_w(i);
          const int x = i * 256 + static_cast<int>(prank) * (w / 2);
          for (int st = 0; st < 8 && ok; ++st) {
            uint32_t sa, fb;
            if (!(ok = next_stage(sa, fb, w == 256 ? kStageTx : kStageTx / 2))) break;
            tma_load_2d_pair(sa, &tm_wn, fb, x, v0 + st * 64);
            if (w == 256) tma_load_2d_pair(sa + 8192, &tm_wn, fb, x + 64, v0 + st * 64);
          }
        }
        // dW jobs: h rows of the four tiles, 64 per stage, this CTA's 128 of the
        // job's 256 columns; the next unit's Z_a stages in between
        for (int j = 0; j < nJ && ok; ++j) {
          const int w = job_w(j);
          const int x = j * 256 + static_cast<int>(prank) * (w / 2);
          for (int st = 0; st < 8 && ok; ++st) {
            uint32_t sa, fb;
            if (!(ok = next_stage(sa, fb, w == 256 ? kStageTx : kStageTx / 2))) break;
            const int row = t4[st >> 1] + (st & 1) * 64;
            tma_load_2d_pair(sa, &tm_h, fb, x, row);
            if (w == 256) tma_load_2d_pair(sa + 8192, &tm_h, fb, x + 64, row);
          }
          if (has_next)
            for (int kb = 8 * j; kb < 8 * j + 8 && kb < nZ && ok; ++kb) ok = load_z(kb, n_row0, n_v0);
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
        // the copies' complete_tx makes both CTAs' bytes visible to the MMAs
        // issued after the phase flips; a CTA-scope wait is enough
        if (!mbar_wait(smem_u32(&full_bar[st]), ph, abort_flag, a.err)) return false;
        tc_fence_after();
        sa = smem0 + st * kStageBytes;
        return true;
      };
      auto release_stage = [&]() {
        umma_commit_pair_mc(smem_u32(&empty_bar[it % kStages]), pair_mask);
        ++it;
      };
      // one logit stage into the TMEM columns at zcol; the last one signals
      // every CTA of the cluster through `bar`
      auto z_block = [&](int kb, uint32_t zcol, uint32_t bar) -> bool {
        uint32_t sa;
        if (!wait_stage(sa)) return false;
        const uint64_t ad = sdesc_sw64(sa);
        const uint64_t bd = sdesc_sw64(sa + kStageBytes / 2);
#pragma unroll
        for (int k = 0; k < kZK / 16; ++k)
          umma_bf16_pair(tmem_base + zcol, ad + 2u * k, bd + 2u * k, kIdescZ, (kb | k) != 0 ? 1u : 0u);
        release_stage();
        if (kb == nZ - 1) umma_commit_pair_mc(bar, 0xF);
        return true;
      };
      // wait until the accumulator may be written by job index j (job j - 1
      // copied out by both CTAs' epilogues)
      auto acc_free = [&](uint32_t j) -> bool {
        if (!mbar_wait(smem_u32(&acce_bar), (j & 1u) ^ 1u, abort_flag, a.err)) return false;
        tc_fence_after();
        return true;
      };
      UnitSeq seq;
      seq.init(quad, n_quads, n_tq, n_vp, a.tile_group, a.det_clusters);
      if (seq.valid())
        for (int kb = 0; kb < nZ && ok; ++kb) ok = z_block(kb, kZaCol, smem_u32(&zfa_bar));
      for (; seq.valid() && ok; seq.advance()) {
        UnitSeq nseq = seq;
        nseq.advance();
        const bool has_next = nseq.valid();
        // Z_b over [256, 512) once the accumulator is idle (its conversion
        // writes g columns [128, 256) after Z_a's has read them)
        if (!(ok = acc_free(jj))) break;
        for (int kb = 0; kb < nZ && ok; ++kb) ok = z_block(kb, kZbCol, smem_u32(&zfb_bar));
        if (!ok) break;
        umma_commit_pair_mc(smem_u32(&zfo_bar), pair_mask);
        // dH: A = g from TMEM (K = 512 vocab), B = W rows (MN-major)
        if (!(ok = mbar_wait_cluster(smem_u32(&tb_bar), unit_it & 1u, abort_flag, a.err))) break;
        tc_fence_after();
        for (int i = 0; i < nJ && ok; ++i) {
          if (!(ok = acc_free(jj))) break;
          const uint32_t d = tmem_base + kAccCol;
          const uint32_t idesc = job_w(i) == 256 ? kIdescH : kIdescH128;
          for (int st = 0; st < 8 && ok; ++st) {   // 64 vocab rows x 128 columns per stage
            uint32_t sa;
            if (!(ok = wait_stage(sa))) break;
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              const uint64_t bd = sdesc_sw128(sa + k * 2048, 8192, 1024);
              umma_bf16_pair_ta(d, tmem_base + kGCol + 8u * static_cast<uint32_t>(st * 4 + k), bd, idesc,
                                (st | k) != 0 ? 1u : 0u);
            }
            release_stage();
          }
          umma_commit_pair_mc(smem_u32(&accf_bar), pair_mask);
          ++jj;
        }
        if (!ok) break;
        umma_commit_pair_mc(smem_u32(&dhd_bar), static_cast<uint16_t>(1u << rank));
        // dW: A = g^T of the pair's two vocab quarters over 512 tokens (GW),
        // B = h rows; the next unit's Z_a K-blocks in between
        if (!(ok = mbar_wait_cluster(smem_u32(&gw_bar), unit_it & 1u, abort_flag, a.err))) break;
        tc_fence_after();
        for (int j = 0; j < nJ && ok; ++j) {
          if (!(ok = acc_free(jj))) break;
          const uint32_t d = tmem_base + kAccCol;
          const uint32_t idesc = job_w(j) == 256 ? kIdescW : kIdescW128;
          for (int st = 0; st < 8 && ok; ++st) {   // 64 token rows x 128 columns per stage
            uint32_t sa;
            if (!(ok = wait_stage(sa))) break;
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              const uint64_t ad = sdesc_sw128(gw_base + (st * 4 + k) * 2048, kGWBlock, 1024);
              const uint64_t bd = sdesc_sw128(sa + k * 2048, 8192, 1024);
              umma_bf16_pair(d, ad, bd, idesc, (st | k) != 0 ? 1u : 0u);
            }
            release_stage();
          }
          umma_commit_pair_mc(smem_u32(&accf_bar), pair_mask);
          ++jj;
          if (has_next && ok) {
            if (j == 0) {   // the dH products have read g: Z_a may overwrite it
              if (!(ok = mbar_wait(smem_u32(&dhd_bar), unit_it & 1u, abort_flag, a.err))) break;
              tc_fence_after();
            }
            for (int kb = 8 * j; kb < 8 * j + 8 && kb < nZ && ok; ++kb) ok = z_block(kb, kZaCol, smem_u32(&zfa_bar));
          }
        }
        if (ok && !has_next) ok = mbar_wait(smem_u32(&dhd_bar), unit_it & 1u, abort_flag, a.err);
        ++unit_it;
      }
      umma_commit_pair_mc(smem_u32(&done_bar), static_cast<uint16_t>(1u << rank));
      mbar_wait_drain(smem_u32(&done_bar), 0, a.err);
    }
  } else {
    const int q = warp & 3;
    const int hf = (warp - 2) >> 2;                       // column half of every TMEM read
    const int r_in = q * 32 + lane;                       // own row = TMEM lane
    const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
    const uint32_t box0 = box_base + (warp - 2) * kBoxesPerWarp * kBoxBytes;
    // the two warps that share this lane quarter meet here (bounded wait; the
    // tcgen05 fences order one warp's TMEM reads before the other's writes)
    uint32_t qsync_it = 0;
    auto pair_warps_sync = [&]() -> bool {
      tc_fence_before();
      mbar_arrive(smem_u32(&qsync_bar[q]));
      const bool w = mbar_wait(smem_u32(&qsync_bar[q]), qsync_it & 1u, abort_flag, a.err);
      ++qsync_it;
      tc_fence_after();
      return w;
    };
    const uint32_t acce_lead = mapa_shared(smem_u32(&acce_bar), lead);
    const uint32_t tb_lead = mapa_shared(smem_u32(&tb_bar), lead);
    const uint32_t gw_lead0 = mapa_shared(smem_u32(&gw_bar), 0);
    const uint32_t gw_lead1 = mapa_shared(smem_u32(&gw_bar), 2);
    // this thread's token row inside every GW buffer (K index of dW)
    const uint32_t gw_row = (rank * 128u + static_cast<uint32_t>(r_in)) * 128u;
    uint32_t jj = 0, nbox = 0, unit_it = 0;
    bool ok = true;

    // g for vocab columns vc0 .. vc0+31 of the unit (packed in w) -> the GW
    // buffer of the CTA that owns those columns
    auto store_gw32 = [&](const uint32_t (&w)[16], int vc0) {
      const int owner = vc0 >> 7;                 // vocab quarter -> CTA
      const int cq = vc0 & 127;
      const uint32_t off = static_cast<uint32_t>((cq >> 6) * kGWBlock) + gw_row;
      const int cc0 = (cq & 63) >> 3;             // first 16-byte chunk in the row
      const uint32_t dst = mapa_shared(gw_base, static_cast<uint32_t>(owner)) + off;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const uint32_t pos = static_cast<uint32_t>(((cc0 + i) ^ (r_in & 7)) * 16);
        if (owner == static_cast<int>(rank))
          st_shared_v4(gw_base + off + pos, w[4 * i], w[4 * i + 1], w[4 * i + 2], w[4 * i + 3]);
        else
          st_shared_cluster_v4(dst + pos, w[4 * i], w[4 * i + 1], w[4 * i + 2], w[4 * i + 3]);
      }
    };
    // z (32 columns at zaddr) -> g for vocab columns vc0 .. vc0+31 of the unit,
    // packed into w (stored to TMEM by the caller), and into GW if to_gw
    auto convert32 = [&](uint32_t zaddr, uint32_t (&w)[16], int vc0, float coef, float ecoef, float mu, float lseL,
                         int lx, int nvalid, bool live, bool to_gw) {
      float v[32];
      tmem_ld32(zaddr, v);
      if (live) {
        const int lxc = lx - vc0;
        const int nv = nvalid - vc0;
#pragma unroll
        for (int j = 0; j < 32; j += 2) {
          float g0, g1;
          if constexpr (kEnt) {
            g0 = fmaf(ecoef, v[j] - mu, coef) * ex2_approx(fmaf(v[j], kLog2e, -lseL));
            g1 = fmaf(ecoef, v[j + 1] - mu, coef) * ex2_approx(fmaf(v[j + 1], kLog2e, -lseL));
          } else {
            g0 = coef * ex2_approx(fmaf(v[j], kLog2e, -lseL));
            g1 = coef * ex2_approx(fmaf(v[j + 1], kLog2e, -lseL));
          }
          if (j == lxc) g0 -= coef;
          if (j + 1 == lxc) g1 -= coef;
          if (j >= nv) g0 = 0.f;
          if (j + 1 >= nv) g1 = 0.f;
          w[j / 2] = pack_bf16x2(g0, g1);
        }
      } else {
#pragma unroll
        for (int j = 0; j < 16; ++j) w[j] = 0u;
      }
      if (to_gw) store_gw32(w, vc0);
    };
    // one logit half (256 columns of z at zcol, vocab vc_base ..): this warp
    // converts its 128 columns; both warps of the lane quarter read all their z
    // before either writes g over it (in place: column c -> c / 2)
    auto convert_half = [&](uint32_t zrow, uint32_t zcol, uint32_t gcol, int vc_base, float coef, float ecoef,
                            float mu, float lseL, int lx, int nvalid, bool live, uint32_t (&w)[4][16],
                            bool to_gw) -> bool {
#pragma unroll
      for (int c = 0; c < 4; ++c)
        convert32(zrow + zcol + hf * 128 + 32 * c, w[c], vc_base + hf * 128 + 32 * c, coef, ecoef, mu, lseL, lx,
                  nvalid, live, to_gw);
      if (!pair_warps_sync()) return false;
#pragma unroll
      for (int c = 0; c < 4; ++c) tmem_st16(zrow + gcol + hf * 64 + 16 * c, w[c]);
      return true;
    };
    // one [32 x 32] fp32 slab of this warp's rows -> reduce-add into global
    auto drain_slab = [&](const CUtensorMap* map, const float (&v)[32], int x, int y, bool issue) {
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
    // Deterministic schedule: the reduce-adds into each [32 x 128] slab of an
    // accumulator take turns.  The slabs of a quad's dhidden rows receive their
    // contributions in vocab-block order, those of a block's dW rows in
    // token-quad order, each from the warp of the same role in another cluster
    // (the same rows and columns).  A turn counter per slab counts the
    // contributions that have completed: a warp waits until it equals its own
    // position (block or quad index), drains, and raises it once its
    // reduce-adds have completed, at its next drain or the end of the unit, so
    // that it does not wait for them in between.
    uint32_t* pend = nullptr;   // counter to raise, and its new value
    uint32_t pend_val = 0;
    auto release_turn = [&]() {
      if (pend != nullptr) {
        if (lane == 0) {
          bulk_wait_group<0>();
          fence_proxy_async_global();
          st_release_gpu(pend, pend_val);
        }
        __syncwarp();
        pend = nullptr;
      }
    };
    auto take_turn = [&](uint32_t* turn, uint32_t pos) -> bool {
      int good = 1;
      if (lane == 0) {
        good = turn_wait(turn, pos, abort_flag, a.det_abort, a.err) ? 1 : 0;
        fence_proxy_async_global();
      }
      return __shfl_sync(0xffffffffu, good, 0) != 0;
    };
    // one job: copy the accumulator to registers, hand it back, then drain it
    // (this warp's 128 of its 256 columns); `turn` (deterministic schedule) is
    // the slab's counter and `pos` this contribution's place in its order
    auto drain_job256 = [&](const CUtensorMap* map, int x0, int y, bool issue, uint32_t* turn, uint32_t pos) -> bool {
      if (!mbar_wait(smem_u32(&accf_bar), jj & 1u, abort_flag, a.err)) return false;
      tc_fence_after();
      const uint32_t taddr = tmem_base + lane_off + kAccCol + hf * 128;
      float v0[32], v1[32], v2[32], v3[32];
      tmem_ld32(taddr, v0);
      tmem_ld32(taddr + 32, v1);
      tmem_ld32(taddr + 64, v2);
      tmem_ld32(taddr + 96, v3);
      // every lane's TMEM reads are complete (wait::ld) and fenced; one
      // arrival per warp hands the accumulator back
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster_relaxed(acce_lead);
      ++jj;
      release_turn();
      if (turn != nullptr && !take_turn(turn, pos)) return false;
      const int xh = x0 + hf * 128;
      drain_slab(map, v0, xh, y, issue);
      drain_slab(map, v1, xh + 32, y, issue);
      drain_slab(map, v2, xh + 64, y, issue);
      drain_slab(map, v3, xh + 96, y, issue);
      if (turn != nullptr) {
        pend = turn;
        pend_val = pos + 1;
      }
      return true;
    };
    // the same for a 128-column last job (H % 256 == 128): 64 columns per warp
    auto drain_job128 = [&](const CUtensorMap* map, int x0, int y, bool issue, uint32_t* turn, uint32_t pos) -> bool {
      if (!mbar_wait(smem_u32(&accf_bar), jj & 1u, abort_flag, a.err)) return false;
      tc_fence_after();
      const uint32_t taddr = tmem_base + lane_off + kAccCol + hf * 64;
      float v0[32], v1[32];
      tmem_ld32(taddr, v0);
      tmem_ld32(taddr + 32, v1);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster_relaxed(acce_lead);
      ++jj;
      release_turn();
      if (turn != nullptr && !take_turn(turn, pos)) return false;
      const int xh = x0 + hf * 64;
      drain_slab(map, v0, xh, y, issue);
      drain_slab(map, v1, xh + 32, y, issue);
      if (turn != nullptr) {
        pend = turn;
        pend_val = pos + 1;
      }
      return true;
    };
    auto drain_job = [&](const CUtensorMap* map, int x0, int y, bool issue, int w, uint32_t* turn,
                         uint32_t pos) -> bool {
      return w == 256 ? drain_job256(map, x0, y, issue, turn, pos) : drain_job128(map, x0, y, issue, turn, pos);
    };
    // this warp's slab counters (deterministic schedule): [unit, job, CTA, warp]
    const bool det = a.det_clusters > 0;
    const int slab = static_cast<int>(rank) * 8 + (warp - 2);
    auto turn_of = [&](uint32_t* base, int unit, int job) -> uint32_t* {
      return det ? base + (static_cast<size_t>(unit) * nJ + job) * 32 + slab : nullptr;
    };

    UnitSeq seq;
    seq.init(quad, n_quads, n_tq, n_vp, a.tile_group, a.det_clusters);
    for (; seq.valid() && ok; seq.advance()) {
      const QuadUnit un = seq.cur();
      const bool own_null = 4 * un.tq + static_cast<int>(rank) >= n_tiles;
      const int own_row0 = tile_of(un.tq, static_cast<int>(rank)) * kTileM;
      const int v0 = un.vp * 512;
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
      const int nvalid = V - v0;
      const uint32_t zrow = tmem_base + lane_off;
      // Z_a -> g of vocab 0..255: TMEM columns [0, 128), GW of CTAs 0 and 1
      if (!(ok = mbar_wait_cluster(smem_u32(&zfa_bar), unit_it & 1u, abort_flag, a.err))) break;
      tc_fence_after();
      uint32_t w[4][16];
      if (!(ok = convert_half(zrow, kZaCol, kGCol, 0, coef, ecoef, mu, lseL, lx, nvalid, live, w, true))) break;
      fence_proxy_async_cluster();
      tc_fence_before();
      mbar_arrive_cluster(gw_lead0);
      // Z_b -> g of vocab 256..511: TMEM columns [128, 256) as soon as this
      // pair's Z_b is done; GW of CTAs 2 and 3 once both pairs' are
      if (!(ok = mbar_wait_cluster(smem_u32(&zfo_bar), unit_it & 1u, abort_flag, a.err))) break;
      tc_fence_after();
      if (!(ok = convert_half(zrow, kZbCol, kGCol + 128, 256, coef, ecoef, mu, lseL, lx, nvalid, live, w, false)))
        break;
      // the dH products need only g in TMEM and Z_b read out: a relaxed
      // arrival after the TMEM fence; the GW stores follow, released on gw_bar
      tc_fence_before();
      mbar_arrive_cluster_relaxed(tb_lead);
      if (!(ok = mbar_wait_cluster(smem_u32(&zfb_bar), unit_it & 1u, abort_flag, a.err))) break;
#pragma unroll
      for (int c = 0; c < 4; ++c) store_gw32(w[c], 256 + hf * 128 + 32 * c);
      fence_proxy_async_cluster();
      mbar_arrive_cluster(gw_lead1);
      // dH jobs: this CTA's 128 token rows, 256 columns of H each (in turn
      // after the quad's earlier vocab blocks)
      const int dh_row = own_row0 + q * 32;
      for (int i = 0; i < nJ && ok; ++i)
        ok = drain_job(&tm_dh, i * 256, dh_row, !own_null, job_w(i), turn_of(a.det_dh_turns, un.tq, i),
                       static_cast<uint32_t>(un.vp));
      // dW jobs: this CTA's 128 vocab rows (its quarter), 256 columns of H
      // each (in turn after the block's earlier token quads)
      const int vrow = v0 + static_cast<int>(rank) * 128 + q * 32;
      for (int j = 0; j < nJ && ok; ++j)
        ok = drain_job(&tm_dw, j * 256, vrow, vrow < V, job_w(j), turn_of(a.det_dw_turns, un.vp, j),
                       static_cast<uint32_t>(un.tq));
      // the unit's last dW slab: the next quad's warp is waiting for it
      release_turn();
      ++unit_it;
    }
    release_turn();
    if (lane == 0) bulk_wait_group<0>();
    __syncwarp();
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync_all();   // no CTA leaves while another may still touch its memory
  tc_fence_after();
  if (warp == 1) {
    __syncwarp();
    tmem_dealloc_pair(tmem_base, 512);
  }
}

}  // namespace

int lmhead_bwd_quad_max_clusters(int n_sm) {
  // per device: the number of 4-CTA clusters that fit at this kernel's
  // shared-memory size (cached as value + 1; 0 = not queried yet)
  static std::atomic<int> cache[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  const int c = cache[dev & 63].load(std::memory_order_acquire);
  if (c > 0) return c - 1;
  cudaError_t e =
      cudaFuncSetAttribute(lmhead_bwd_quad_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
  if (e != cudaSuccess) return 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(n_sm / 4 * 4, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = kSmemBytes;
  int n = 0;
  e = cudaOccupancyMaxActiveClusters(&n, lmhead_bwd_quad_kernel<false>, &cfg);
  if (e != cudaSuccess) {
    cudaGetLastError();
    n = n_sm / 4;
  }
  cache[dev & 63].store(n + 1, std::memory_order_release);
  return n;
}

int lmhead_bwd_quad_det_clusters(int n_sm) { return lmhead_bwd_quad_clusters(n_sm) / 4 * 4; }

int lmhead_bwd_quad_clusters(int n_sm) {
  int clusters = lmhead_bwd_quad_max_clusters(n_sm);
  if (clusters > n_sm / 4) clusters = n_sm / 4;
  if (clusters < 1) clusters = 1;
  return clusters;
}

cudaError_t launch_lmhead_bwd_quad(const CUtensorMap& tm_hz, const CUtensorMap& tm_wz, const CUtensorMap& tm_h,
                                   const CUtensorMap& tm_w_n, const CUtensorMap& tm_dh, const CUtensorMap& tm_dw,
                                   const BwdArgs& a, int n_sm, cudaStream_t s) {
  const bool ent = a.ecoef != nullptr;
  cudaError_t e = ent ? cudaFuncSetAttribute(lmhead_bwd_quad_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             kSmemBytes)
                      : cudaFuncSetAttribute(lmhead_bwd_quad_kernel<false>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
  if (e != cudaSuccess) return e;
  int clusters = lmhead_bwd_quad_clusters(n_sm);
  if (a.det_clusters > 0) {
    if (a.det_clusters > clusters || a.det_clusters % 4 != 0) return cudaErrorInvalidValue;
    clusters = a.det_clusters;
  }
  if (ent)
    lmhead_bwd_quad_kernel<true>
        <<<4 * clusters, kThreads, kSmemBytes, s>>>(tm_hz, tm_wz, tm_h, tm_w_n, tm_dh, tm_dw, a);
  else
    lmhead_bwd_quad_kernel<false>
        <<<4 * clusters, kThreads, kSmemBytes, s>>>(tm_hz, tm_wz, tm_h, tm_w_n, tm_dh, tm_dw, a);
  return cudaGetLastError();
}

}  // namespace molt
