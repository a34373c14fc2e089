// Row-level kernels of the policy-update path: GRPO advantages, advantage
// broadcast, mask count, active-row compaction, packed gathers, the split-vocab
// merge with the clipped surrogate, the fixed-order loss reduction and the
// dhidden cast.  None of these is a contraction; they are launch- or HBM-bound.
#include <cstdint>
#include <cuda_runtime.h>

#include "molt_internal.cuh"
#include "ptx.cuh"

namespace molt {
namespace {

constexpr float kLog2e = 1.4426950408889634f;

// ---------------------------------------------------------------------------
// Advantage estimators (Sec. 4.5: GRPO, a group-mean baseline, Dr. GRPO, RLOO,
// REINFORCE++; Sec. 4.2: one reward per rollout).  One warp per response index;
// the warp whose index starts a run of equal ids processes that group (for
// REINFORCE++, gid == nullptr and warp 0 normalises the whole batch).  Lanes
// load the rewards coalesced, 32 at a time, and fold them with shuffles in
// index order, so the fp64 sums run in the same order as a sequential loop.
// Explicit _rn intrinsics keep the compiler from contracting a multiply and an
// add into an FMA.
// ---------------------------------------------------------------------------
__global__ void group_adv_kernel(const float* __restrict__ r, const int32_t* __restrict__ gid, int n, double eps,
                                 int est, float* __restrict__ out, unsigned* err) {
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (warp >= n) return;
  int start = warp, end = n;
  if (gid == nullptr) {
    if (warp != 0) return;
  } else {
    const int g = gid[start];
    if (start > 0) {
      const int gp = gid[start - 1];
      if (gp == g) return;
      if (gp > g && lane == 0) atomicOr(err, kDevErrUnsortedGroups);
    }
    // end of the run
    for (int base = start;; base += 32) {
      const int j = base + lane;
      const bool same = (j < n) && (gid[j] == g);
      const unsigned m = __ballot_sync(0xffffffffu, same);
      if (m == 0xffffffffu) {
        end = base + 32;
        continue;
      }
      end = base + __ffs(~m) - 1;
      break;
    }
  }
  const int cnt = end - start;
  if (cnt == 1) {
    if (lane == 0) out[start] = 0.0f;
    return;
  }
  double s = 0.0;
  for (int base = start; base < end; base += 32) {
    const int j = base + lane;
    const double v = (j < end) ? static_cast<double>(r[j]) : 0.0;
    const int k = min(32, end - base);
    for (int i = 0; i < k; ++i) {
      const double vi = __shfl_sync(0xffffffffu, v, i);
      s = __dadd_rn(s, vi);
    }
  }
  s = __shfl_sync(0xffffffffu, s, 0);
  if (est == kAdvRloo) {
    // leave-one-out baseline (sum - r_j) / (n - 1)
    for (int base = start; base < end; base += 32) {
      const int j = base + lane;
      if (j < end) {
        const double rj = static_cast<double>(r[j]);
        const double b = __ddiv_rn(__dsub_rn(s, rj), static_cast<double>(cnt - 1));
        out[j] = __double2float_rn(__dsub_rn(rj, b));
      }
    }
    return;
  }
  const double mean = __ddiv_rn(s, static_cast<double>(cnt));
  if (est == kAdvGroupMean || est == kAdvDrGrpo) {
    for (int base = start; base < end; base += 32) {
      const int j = base + lane;
      if (j < end) out[j] = __double2float_rn(__dsub_rn(static_cast<double>(r[j]), mean));
    }
    return;
  }
  double ss = 0.0;
  for (int base = start; base < end; base += 32) {
    const int j = base + lane;
    const double d = (j < end) ? __dsub_rn(static_cast<double>(r[j]), mean) : 0.0;
    const double d2 = __dmul_rn(d, d);
    const int k = min(32, end - base);
    for (int i = 0; i < k; ++i) ss = __dadd_rn(ss, __shfl_sync(0xffffffffu, d2, i));
  }
  ss = __shfl_sync(0xffffffffu, ss, 0);
  const double sd = __dsqrt_rn(__ddiv_rn(ss, static_cast<double>(cnt - 1)));
  const double den = __dadd_rn(sd, eps);
  for (int base = start; base < end; base += 32) {
    const int j = base + lane;
    if (j < end) {
      const double d = __dsub_rn(static_cast<double>(r[j]), mean);
      out[j] = __double2float_rn(__ddiv_rn(d, den));
    }
  }
}

__global__ void broadcast_kernel(const float* __restrict__ adv, const int32_t* __restrict__ rot, int n_resp, int T,
                                 float* __restrict__ out) {
  for (int t = blockIdx.x * blockDim.x + threadIdx.x; t < T; t += gridDim.x * blockDim.x) {
    const int k = rot[t];
    out[t] = (k >= 0 && k < n_resp) ? adv[k] : 0.0f;
  }
}

// sum of a uint8 mask: 16 bytes per load, per-block total, one atomic per block
__global__ void mask_count_kernel(const uint8_t* __restrict__ mask, int64_t T,
                                  unsigned long long* __restrict__ out) {
  unsigned long long c = 0;
  const int64_t nvec = T / 16;
  const uint4* m4 = reinterpret_cast<const uint4*>(mask);
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < nvec; i += (int64_t)gridDim.x * blockDim.x) {
    const uint4 v = m4[i];
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) c += (w[q] & 0xFFu ? 1 : 0) + (w[q] & 0xFF00u ? 1 : 0) +
                                     (w[q] & 0xFF0000u ? 1 : 0) + (w[q] & 0xFF000000u ? 1 : 0);
  }
  for (int64_t i = nvec * 16 + blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < T;
       i += (int64_t)gridDim.x * blockDim.x)
    c += mask[i] ? 1 : 0;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
  __shared__ unsigned long long sh[32];
  if ((threadIdx.x & 31) == 0) sh[threadIdx.x >> 5] = c;
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned long long tot = 0;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) tot += sh[w];
    if (tot) atomicAdd(out, tot);
  }
}

// block-wide exclusive scan of one int per thread (blockDim.x = 1024)
__device__ int block_exclusive_scan(int v, int* total) {
  __shared__ int wsum[32];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) wsum[w] = x;
  __syncthreads();
  if (w == 0) {
    int s = (lane < (int)(blockDim.x >> 5)) ? wsum[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, s, o);
      if (lane >= o) s += y;
    }
    wsum[lane] = s;
  }
  __syncthreads();
  const int before = (w > 0 ? wsum[w - 1] : 0) + x - v;
  if (total) *total = wsum[(blockDim.x >> 5) - 1];
  __syncthreads();
  return before;
}

// order-preserving list of active rows (mask != 0): one block, each thread a
// contiguous chunk
__global__ void __launch_bounds__(1024) compact_kernel(const uint8_t* __restrict__ mask, int T,
                                                       int32_t* __restrict__ row_map, int32_t* __restrict__ pos,
                                                       int32_t* __restrict__ counts) {
  const int per = (T + blockDim.x - 1) / blockDim.x;
  const int b = threadIdx.x * per, e = min(T, b + per);
  int c = 0;
  for (int t = b; t < e; ++t) c += (mask == nullptr || mask[t]) ? 1 : 0;
  int total;
  int k = block_exclusive_scan(c, &total);
  for (int t = b; t < e; ++t) {
    if (mask == nullptr || mask[t]) {
      row_map[k] = t;
      pos[t] = k++;
    } else {
      pos[t] = -1;
    }
  }
  if (threadIdx.x == 0) {
    counts[0] = total;
    counts[1] = 0;
    counts[2] = 0;
  }
}

// packed copies of the active rows; rows in [n, round_up(n,128)) are zeroed so
// that the last tile holds finite values
__global__ void gather_kernel(const uint16_t* __restrict__ hidden, const int32_t* __restrict__ tokens,
                              const float* __restrict__ b, const float* __restrict__ adv, int tok_shift, int Tcap,
                              int H,
                              const int32_t* __restrict__ row_map, const int32_t* __restrict__ counts,
                              uint16_t* __restrict__ h_p, int32_t* __restrict__ tok_p, float* __restrict__ b_p,
                              float* __restrict__ adv_p) {
  const int n = counts[0];
  const int nz = min(Tcap, ((n + kTileM - 1) / kTileM) * kTileM);
  const int vpr = H / 8;   // 16-byte vectors per row
  const int64_t total = (int64_t)nz * vpr;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const int k = (int)(i / vpr), v = (int)(i - (int64_t)k * vpr);
    uint4 val = make_uint4(0, 0, 0, 0);
    if (k < n) {
      const int t = row_map[k];
      val = reinterpret_cast<const uint4*>(hidden + (int64_t)t * H)[v];
      if (v == 0) {
        tok_p[k] = tokens[t] - tok_shift;
        if (b_p) b_p[k] = b[t];
        if (adv_p) adv_p[k] = adv[t];
      }
    } else if (v == 0) {
      tok_p[k] = 0;
      if (b_p) b_p[k] = 0.f;
      if (adv_p) adv_p[k] = 0.f;
    }
    reinterpret_cast<uint4*>(h_p + (int64_t)k * H)[v] = val;
  }
}

// deterministic 128-thread block sum (fixed tree)
template <typename T>
__device__ T block128_sum(T v, T* sh) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  if ((threadIdx.x & 31) == 0) sh[threadIdx.x >> 5] = v;
  __syncthreads();
  T r = (sh[0] + sh[1]) + (sh[2] + sh[3]);
  __syncthreads();
  return r;
}
__device__ double block128_max(double v, double* sh) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmax(v, __shfl_xor_sync(0xffffffffu, v, o));
  if ((threadIdx.x & 31) == 0) sh[threadIdx.x >> 5] = v;
  __syncthreads();
  double r = fmax(fmax(sh[0], sh[1]), fmax(sh[2], sh[3]));
  __syncthreads();
  return r;
}

// Eq. 2 terms of one active row (Sec. 4.5: ratio against the behaviour
// log-prob, PPO clipped surrogate with asymmetric bounds, m c / D).
struct RowLoss {
  float tl, coef, ratio;
  int clip_lo_hit, clip_hi_hit;
  double alr;
};
__device__ __forceinline__ RowLoss surrogate_row(float logp, float b, float A, float clip_lo, float clip_hi,
                                                 double D) {
  RowLoss r;
  r.ratio = expf(logp - b);
  const float lo = 1.0f - clip_lo, hi = 1.0f + clip_hi;
  const bool clipped = (A > 0.f && r.ratio > hi) || (A < 0.f && r.ratio < lo);
  const float rc = fminf(fmaxf(r.ratio, lo), hi);
  r.tl = clipped ? -(rc * A) : -(r.ratio * A);
  const float c = clipped ? 0.f : r.ratio * A;
  r.coef = (D > 0.0) ? static_cast<float>(static_cast<double>(c) / D) : 0.f;
  r.clip_lo_hit = (clipped && A < 0.f) ? 1 : 0;
  r.clip_hi_hit = (clipped && A > 0.f) ? 1 : 0;
  r.alr = fabs(static_cast<double>(logp) - static_cast<double>(b));
  return r;
}

// the tile's fixed-tree partial sums (loss, ratio, entropy, max |log ratio|,
// clip counts) and its activity flag; every thread of the 128-thread block
// calls it
__device__ void tile_partials(bool act, const RowLoss& rl, float ent, double* __restrict__ red,
                              int32_t* __restrict__ tile_flag) {
  __shared__ double shd[4];
  __shared__ long long shl[4];
  const int any = __syncthreads_or(act && rl.coef != 0.f);
  double* r = red + (int64_t)blockIdx.x * kRedSlots;
  const double s_loss = block128_sum<double>(act ? (double)rl.tl : 0.0, shd);
  const double s_ratio = block128_sum<double>(act ? (double)rl.ratio : 0.0, shd);
  const double s_ent = block128_sum<double>(act ? (double)ent : 0.0, shd);
  const double m_alr = block128_max(act ? rl.alr : 0.0, shd);
  const long long c_lo = block128_sum<long long>(act ? rl.clip_lo_hit : 0, shl);
  const long long c_hi = block128_sum<long long>(act ? rl.clip_hi_hit : 0, shl);
  if (threadIdx.x == 0) {
    tile_flag[blockIdx.x] = any ? 1 : 0;
    r[0] = s_loss;
    r[1] = s_ratio;
    r[2] = s_ent;
    r[3] = m_alr;
    r[4] = static_cast<double>(c_lo);
    r[5] = static_cast<double>(c_hi);
    r[6] = 0.0;
    r[7] = 0.0;
  }
}

// One block of 128 threads per packed tile: merge the per-split online
// softmax partials of each row into lse, logp and entropy; in loss mode also
// the ratio, the clipped surrogate (Sec. 4.5, PPO form), the Eq. 2 coefficient
// m c / D, per-tile partial sums and the tile's activity flag.
__global__ void __launch_bounds__(128) merge_kernel(
    int loss_mode, int Tcap, int V, int n_split, double denom, float clip_lo, float clip_hi,
    const int32_t* __restrict__ counts, const int32_t* __restrict__ row_map, const int32_t* __restrict__ tok_p,
    const float* __restrict__ b_p, const float* __restrict__ adv_p, const float4* __restrict__ part,
    const float* __restrict__ zx, float* __restrict__ lse_o, float* __restrict__ coef_o,
    int32_t* __restrict__ tile_flag, double* __restrict__ red, float* __restrict__ logp_out,
    float* __restrict__ ent_out, float* __restrict__ tokloss_out, float* __restrict__ lp_p,
    float* __restrict__ ent_p, unsigned* err) {
  const int n = counts[0];
  const int n_tiles = (n + kTileM - 1) / kTileM;
  if ((int)blockIdx.x >= n_tiles) return;
  const int k = blockIdx.x * kTileM + threadIdx.x;
  const bool act = k < n;
  const double D = denom > 0.0 ? denom : static_cast<double>(n);
  float logp = 0.f, ent = 0.f;
  RowLoss rl{0.f, 0.f, 0.f, 0, 0, 0.0};
  if (act) {
    float M = -INFINITY;
    for (int s = 0; s < n_split; ++s) M = fmaxf(M, part[(int64_t)s * Tcap + k].x);
    float S = 0.f, Q = 0.f;
    for (int s = 0; s < n_split; ++s) {
      const float4 p = part[(int64_t)s * Tcap + k];
      if (p.y > 0.f) {
        const float d = p.x - M;
        const float f = ex2_approx(d * kLog2e);
        S += f * p.y;
        Q += f * (p.z + d * p.y);
      }
    }
    const float logS = logf(S);
    const float lse = M + logS;
    const int x = tok_p[k];
    if (x < 0 || x >= V) atomicOr(err, kDevErrTokenRange);
    logp = zx[k] - lse;
    ent = logS - Q / S;
    lse_o[k] = lse;
    if (loss_mode) rl = surrogate_row(logp, b_p[k], adv_p[k], clip_lo, clip_hi, D);
    const int t = row_map[k];
    if (logp_out) logp_out[t] = logp;
    if (ent_out) ent_out[t] = ent;
    if (tokloss_out) tokloss_out[t] = rl.tl;
    if (lp_p) lp_p[k] = logp;
    if (ent_p) ent_p[k] = ent;
  }
  if (!loss_mode) return;
  if (k < Tcap) coef_o[k] = rl.coef;
  tile_partials(act, rl, ent, red, tile_flag);
}

// ---------------------------------------------------------------------------
// Vocabulary-parallel pieces: the LM head split into vocabulary shards (one per
// tensor-parallel rank).  Each shard reduces its own columns to per-row
// statistics; the statistics of all shards, exchanged by the caller, merge into
// the row's lse, logp and entropy exactly as the forward's own vocab splits do.
// ---------------------------------------------------------------------------

// Statistics of one shard per original row: the forward's split partials
// combined in split order into (M, S, Q, z_x): M the shard's max logit, S =
// sum exp(z - M), Q = sum exp(z - M) (z - M), z_x the target logit if the
// target lies in the shard (tok_p holds the shard-local token) and -inf
// otherwise.  Masked rows get the empty statistics (-inf, 0, 0, -inf).
__global__ void vp_local_kernel(int T, int Tcap, int V_s, int n_split, const int32_t* __restrict__ pos,
                                const int32_t* __restrict__ tok_p, const float4* __restrict__ part,
                                const float* __restrict__ zx, float4* __restrict__ out) {
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= T) return;
  const int k = pos[t];
  if (k < 0) {
    out[t] = make_float4(-INFINITY, 0.f, 0.f, -INFINITY);
    return;
  }
  float M = -INFINITY;
  for (int s = 0; s < n_split; ++s) M = fmaxf(M, part[(int64_t)s * Tcap + k].x);
  float S = 0.f, Q = 0.f;
  for (int s = 0; s < n_split; ++s) {
    const float4 p = part[(int64_t)s * Tcap + k];
    if (p.y > 0.f) {
      const float d = p.x - M;
      const float f = ex2_approx(d * kLog2e);
      S += f * p.y;
      Q += f * (p.z + d * p.y);
    }
  }
  const int xl = tok_p[k];
  out[t] = make_float4(M, S, Q, (xl >= 0 && xl < V_s) ? zx[k] : -INFINITY);
}

// One block of 128 threads per packed tile of active rows: merge the shards'
// statistics of each row (parts [n_shards, T], shard order fixed) into lse,
// logp and entropy, then the Eq. 2 terms as merge_kernel does.  A row whose
// target lies in no shard raises the token-range flag.  Per-row outputs go to
// the original row order (lse and m c / D for the shards' backward).
__global__ void __launch_bounds__(128) vp_merge_kernel(
    int T, int n_shards, double denom, float clip_lo, float clip_hi, const int32_t* __restrict__ counts,
    const int32_t* __restrict__ row_map, const float4* __restrict__ parts, const float* __restrict__ b,
    const float* __restrict__ adv, float* __restrict__ coef_p, int32_t* __restrict__ tile_flag,
    double* __restrict__ red, float* __restrict__ lse_out, float* __restrict__ coef_out,
    float* __restrict__ logp_out, float* __restrict__ ent_out, float* __restrict__ tokloss_out, unsigned* err) {
  const int n = counts[0];
  const int n_tiles = (n + kTileM - 1) / kTileM;
  if ((int)blockIdx.x >= n_tiles) return;
  const int k = blockIdx.x * kTileM + threadIdx.x;
  const bool act = k < n;
  const double D = denom > 0.0 ? denom : static_cast<double>(n);
  float ent = 0.f;
  RowLoss rl{0.f, 0.f, 0.f, 0, 0, 0.0};
  if (act) {
    const int t = row_map[k];
    float M = -INFINITY, zxv = -INFINITY;
    for (int s = 0; s < n_shards; ++s) {
      const float4 p = parts[(int64_t)s * T + t];
      M = fmaxf(M, p.x);
      zxv = fmaxf(zxv, p.w);
    }
    float S = 0.f, Q = 0.f;
    for (int s = 0; s < n_shards; ++s) {
      const float4 p = parts[(int64_t)s * T + t];
      if (p.y > 0.f) {
        const float d = p.x - M;
        const float f = ex2_approx(d * kLog2e);
        S += f * p.y;
        Q += f * (p.z + d * p.y);
      }
    }
    if (zxv == -INFINITY) atomicOr(err, kDevErrTokenRange);
    const float logS = logf(S);
    const float lse = M + logS;
    const float logp = zxv == -INFINITY ? 0.f : zxv - lse;
    ent = logS - Q / S;
    rl = surrogate_row(logp, b[t], adv[t], clip_lo, clip_hi, D);
    lse_out[t] = lse;
    coef_out[t] = rl.coef;
    if (logp_out) logp_out[t] = logp;
    if (ent_out) ent_out[t] = ent;
    if (tokloss_out) tokloss_out[t] = rl.tl;
  }
  if (k < ((n + kTileM - 1) / kTileM) * kTileM) coef_p[k] = rl.coef;
  tile_partials(act, rl, ent, red, tile_flag);
}

// The rows of one shard's backward: those with a gradient coefficient (coef
// from vp_merge_kernel, original order; masked and clipped rows have 0), in
// order.  One block; as finalize_kernel's list.
__global__ void __launch_bounds__(1024) vp_live_kernel(int T, const float* __restrict__ coef,
                                                       int32_t* __restrict__ counts, int32_t* __restrict__ tile_list,
                                                       int32_t* __restrict__ live_map,
                                                       int32_t* __restrict__ live_of) {
  const int per = (T + blockDim.x - 1) / blockDim.x;
  const int t0 = threadIdx.x * per, t1 = min(T, t0 + per);
  int c = 0;
  for (int t = t0; t < t1; ++t) c += coef[t] != 0.f ? 1 : 0;
  int total;
  int j = block_exclusive_scan(c, &total);
  for (int t = t0; t < t1; ++t) {
    if (coef[t] != 0.f) {
      live_map[j] = t;
      live_of[t] = j++;
    } else {
      live_of[t] = -1;
    }
  }
  const int n_lt = (total + kTileM - 1) / kTileM;
  for (int b = threadIdx.x; b < n_lt; b += blockDim.x) tile_list[b] = b;
  if (threadIdx.x == 0) {
    counts[0] = total;
    counts[1] = n_lt;
    counts[2] = 0;
    counts[3] = total;
  }
}

// one shard's dhidden contribution in the original row order, fp32: the
// accumulator row of t's backward row, 0 for rows without a gradient
__global__ void vp_dh_out_kernel(const float* __restrict__ dh32, const int32_t* __restrict__ live_of, int T, int H,
                                 float* __restrict__ out) {
  const int vpr = H / 4;
  const int64_t total = (int64_t)T * vpr;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const int t = (int)(i / vpr), v = (int)(i - (int64_t)t * vpr);
    const int j = live_of[t];
    float4 o = make_float4(0.f, 0.f, 0.f, 0.f);
    if (j >= 0) o = reinterpret_cast<const float4*>(dh32 + (int64_t)j * H)[v];
    reinterpret_cast<float4*>(out + (int64_t)t * H)[v] = o;
  }
}

// ---------------------------------------------------------------------------
// Extended objective (Sec. 4.5: KL control, rejection rules).
// ---------------------------------------------------------------------------

// Sequence gate.  Thread i checks that the ids do not decrease at token i; warp
// w owns packed rows [32 w, 32 w + 32) and handles every sequence that starts
// there: it walks the sequence 32 packed rows at a time (packing keeps the
// original order, so a sequence is a run of packed rows), sums logp - b in
// fp64 with a fixed shuffle tree, and writes the gate weight of every row.
// Reject when exp(mean) lies outside [lo, hi].
__global__ void __launch_bounds__(256) seq_gate_kernel(int T, const int32_t* __restrict__ seq,
                                                       const int32_t* __restrict__ counts,
                                                       const int32_t* __restrict__ row_map,
                                                       const float* __restrict__ lp_p, const float* __restrict__ b_p,
                                                       double lo, double hi, uint8_t* __restrict__ gate_p,
                                                       int32_t* __restrict__ n_rej, unsigned* err) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  const int lane = threadIdx.x & 31;
  if (i < T && i > 0 && seq[i] < seq[i - 1]) atomicOr(err, kDevErrUnsortedGroups);
  const int n = counts[0];
  const int base = i - lane;
  if (base >= n) return;   // whole warp leaves together
  const int k = base + lane;
  const int sid = (k < n) ? seq[row_map[k]] : 0;
  const bool start = (k < n) && (k == 0 || seq[row_map[k - 1]] != sid);
  unsigned starts = __ballot_sync(0xffffffffu, start);
  while (starts) {
    const int s0 = base + __ffs(starts) - 1;
    starts &= starts - 1;
    const int sid0 = __shfl_sync(0xffffffffu, sid, s0 - base);
    double acc = 0.0;
    int len = 0;
    for (int w0 = s0;; w0 += 32) {
      const int kk = w0 + lane;
      const bool in = kk < n && seq[row_map[kk]] == sid0;
      const unsigned m = __ballot_sync(0xffffffffu, in);
      const int run = (m == 0xffffffffu) ? 32 : __ffs(~m) - 1;   // leading rows of this sequence
      double v = (lane < run) ? static_cast<double>(lp_p[kk]) - static_cast<double>(b_p[kk]) : 0.0;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
      acc += v;
      len += run;
      if (run < 32) break;
    }
    const double g = exp(acc / static_cast<double>(len));
    const uint8_t keep = (g < lo || g > hi) ? 0 : 1;
    for (int j = s0 + lane; j < s0 + len; j += 32) gate_p[j] = keep;
    if (lane == 0 && !keep) atomicAdd(n_rej, 1);
  }
}

// One block of 128 threads per packed tile: the per-token loss of the extended
// objective and the two backward coefficients
//   coef  = m w (c + kl_coef (e^r - 1)) / D      on (p - onehot)
//   ecoef = m w entropy_coef / D                 on p (z - mu),  mu = lse - H
__global__ void __launch_bounds__(128) loss_rows_ex_kernel(
    int Tcap, double denom, float clip_lo, float clip_hi, LossEx ex, const int32_t* __restrict__ counts,
    const int32_t* __restrict__ row_map, const float* __restrict__ b_p, const float* __restrict__ adv_p,
    const float* __restrict__ lp_p, const float* __restrict__ ent_p, const float* __restrict__ lse,
    const uint8_t* __restrict__ gate_p, float* __restrict__ coef_o, float* __restrict__ ecoef_o,
    float* __restrict__ mu_o, int32_t* __restrict__ tile_flag, double* __restrict__ red,
    float* __restrict__ tokloss_out) {
  __shared__ double shd[4];
  __shared__ long long shl[4];
  const int n = counts[0];
  const int n_tiles = (n + kTileM - 1) / kTileM;
  if ((int)blockIdx.x >= n_tiles) return;
  const int k = blockIdx.x * kTileM + threadIdx.x;
  const bool act = k < n;
  const double D = denom > 0.0 ? denom : static_cast<double>(n);
  float coef = 0.f, ecoef = 0.f, mu = 0.f, tl = 0.f, ratio = 0.f, ent = 0.f, kl = 0.f;
  int clip_lo_hit = 0, clip_hi_hit = 0, rejected = 0;
  double alr = 0.0;
  if (act) {
    const float logp = lp_p[k], b = b_p[k], A = adv_p[k];
    ent = ent_p[k];
    ratio = expf(logp - b);
    const float lo = 1.0f - clip_lo, hi = 1.0f + clip_hi;
    const bool clipped = (A > 0.f && ratio > hi) || (A < 0.f && ratio < lo);
    const float rc = fminf(fmaxf(ratio, lo), hi);
    const float l_pg = clipped ? -(rc * A) : -(ratio * A);
    const float c = clipped ? 0.f : ratio * A;
    float c_kl = 0.f;
    if (ex.kl_coef != 0.f) {
      const float r = ex.ref_logp[row_map[k]] - logp;
      const float em1 = expm1f(r);
      kl = em1 - r;             // e^r - r - 1 without cancellation near r = 0
      c_kl = ex.kl_coef * em1;
    }
    const bool keep = gate_p == nullptr || gate_p[k] != 0;
    if (keep) {
      tl = l_pg + ex.kl_coef * kl - ex.entropy_coef * ent;
      coef = (D > 0.0) ? static_cast<float>(static_cast<double>(c + c_kl) / D) : 0.f;
      ecoef = (D > 0.0) ? static_cast<float>(static_cast<double>(ex.entropy_coef) / D) : 0.f;
      clip_lo_hit = (clipped && A < 0.f) ? 1 : 0;
      clip_hi_hit = (clipped && A > 0.f) ? 1 : 0;
    } else {
      kl = 0.f;
      rejected = 1;
    }
    mu = lse[k] - ent;
    alr = fabs(static_cast<double>(logp) - static_cast<double>(b));
    if (tokloss_out) tokloss_out[row_map[k]] = tl;
  }
  if (k < Tcap) {
    coef_o[k] = coef;
    ecoef_o[k] = ecoef;
    mu_o[k] = mu;
  }
  const int any = __syncthreads_or(coef != 0.f || ecoef != 0.f);
  double* rr = red + (int64_t)blockIdx.x * kRedSlots;
  const double s_loss = block128_sum<double>(act ? (double)tl : 0.0, shd);
  const double s_ratio = block128_sum<double>(act ? (double)ratio : 0.0, shd);
  const double s_ent = block128_sum<double>(act ? (double)ent : 0.0, shd);
  const double m_alr = block128_max(alr, shd);
  const long long c_lo = block128_sum<long long>(clip_lo_hit, shl);
  const long long c_hi = block128_sum<long long>(clip_hi_hit, shl);
  const double s_kl = block128_sum<double>(act ? (double)kl : 0.0, shd);
  const long long c_rej = block128_sum<long long>(rejected, shl);
  if (threadIdx.x == 0) {
    tile_flag[blockIdx.x] = any ? 1 : 0;
    rr[0] = s_loss;
    rr[1] = s_ratio;
    rr[2] = s_ent;
    rr[3] = m_alr;
    rr[4] = static_cast<double>(c_lo);
    rr[5] = static_cast<double>(c_hi);
    rr[6] = s_kl;
    rr[7] = static_cast<double>(c_rej);
  }
}

struct StatsDev {
  double denom, loss, sum_ratio, sum_entropy, max_abs_log_ratio;
  long long n_active, n_clip_low, n_clip_high, n_grad_rows;
};
struct StatsExDev {
  StatsDev base;
  double sum_kl;
  long long n_tokens_rejected, n_seq_rejected;
};
constexpr int kFinSlots = 8;

// fixed-order reduction of the per-tile partials, the loss scalar and the
// stats; then the order-preserving list of the packed rows whose gradient
// coefficient is nonzero (coef, or ecoef with an entropy bonus): the rows the
// backward processes, packed again by live_gather_kernel into whole tiles
__global__ void __launch_bounds__(1024) finalize_kernel(double denom, int32_t* __restrict__ counts,
                                                        int32_t* __restrict__ tile_list,
                                                        const double* __restrict__ red, float* __restrict__ loss_out,
                                                        StatsDev* __restrict__ stats, StatsExDev* __restrict__ stats_ex,
                                                        const float* __restrict__ coef,
                                                        const float* __restrict__ ecoef,
                                                        int32_t* __restrict__ live_map,
                                                        int32_t* __restrict__ live_of, unsigned* err) {
  __shared__ double sh[kFinSlots][32];
  const int n = counts[0];
  const int n_tiles = (n + kTileM - 1) / kTileM;
  double a[kFinSlots] = {0, 0, 0, 0, 0, 0, 0, 0};
  for (int b = threadIdx.x; b < n_tiles; b += blockDim.x) {
    const double* r = red + (int64_t)b * kRedSlots;
#pragma unroll
    for (int q = 0; q < kFinSlots; ++q) a[q] = (q == 3) ? fmax(a[q], r[q]) : a[q] + r[q];
  }
  // fixed shuffle tree inside each warp, then warp 0 over the 32 warp results
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
#pragma unroll
    for (int q = 0; q < kFinSlots; ++q) {
      const double y = __shfl_xor_sync(0xffffffffu, a[q], o);
      a[q] = (q == 3) ? fmax(a[q], y) : a[q] + y;
    }
  }
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  if (lane == 0)
    for (int q = 0; q < kFinSlots; ++q) sh[q][w] = a[q];
  __syncthreads();
  if (w == 0) {
    for (int q = 0; q < kFinSlots; ++q) a[q] = sh[q][lane];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
#pragma unroll
      for (int q = 0; q < kFinSlots; ++q) {
        const double y = __shfl_xor_sync(0xffffffffu, a[q], o);
        a[q] = (q == 3) ? fmax(a[q], y) : a[q] + y;
      }
    }
    if (lane == 0)
      for (int q = 0; q < kFinSlots; ++q) sh[q][0] = a[q];
  }
  __syncthreads();
  const double D = denom > 0.0 ? denom : static_cast<double>(n);
  if (threadIdx.x == 0) {
    if (!(D > 0.0)) atomicOr(err, kDevErrZeroDenom);
    const double loss = D > 0.0 ? sh[0][0] / D : 0.0;
    if (loss_out) *loss_out = static_cast<float>(loss);
    if (stats) {
      stats->denom = D;
      stats->loss = loss;
      stats->sum_ratio = sh[1][0];
      stats->sum_entropy = sh[2][0];
      stats->max_abs_log_ratio = sh[3][0];
      stats->n_active = n;
      stats->n_clip_low = static_cast<long long>(sh[4][0]);
      stats->n_clip_high = static_cast<long long>(sh[5][0]);
    }
    if (stats_ex) {
      StatsDev& b = stats_ex->base;
      b.denom = D;
      b.loss = loss;
      b.sum_ratio = sh[1][0];
      b.sum_entropy = sh[2][0];
      b.max_abs_log_ratio = sh[3][0];
      b.n_active = n;
      b.n_clip_low = static_cast<long long>(sh[4][0]);
      b.n_clip_high = static_cast<long long>(sh[5][0]);
      stats_ex->sum_kl = sh[6][0];
      stats_ex->n_tokens_rejected = static_cast<long long>(sh[7][0]);
      stats_ex->n_seq_rejected = counts[2];
    }
  }
  // compact the rows with a gradient (order preserving)
  auto live = [&](int k) { return coef[k] != 0.f || (ecoef != nullptr && ecoef[k] != 0.f); };
  const int per = (n + blockDim.x - 1) / blockDim.x;
  const int k0 = threadIdx.x * per, k1 = min(n, k0 + per);
  int c = 0;
  for (int k = k0; k < k1; ++k) c += live(k) ? 1 : 0;
  int total;
  int j = block_exclusive_scan(c, &total);
  for (int k = k0; k < k1; ++k) {
    if (live(k)) {
      live_map[j] = k;
      live_of[k] = j++;
    } else {
      live_of[k] = -1;
    }
  }
  const int n_lt = (total + kTileM - 1) / kTileM;
  for (int b = threadIdx.x; b < n_lt; b += blockDim.x) tile_list[b] = b;
  if (threadIdx.x == 0) {
    counts[1] = n_lt;
    counts[3] = total;
    if (stats) stats->n_grad_rows = total;
    if (stats_ex) stats_ex->base.n_grad_rows = total;
  }
}

// packed copies of the rows with a gradient (live_map from finalize_kernel):
// hidden row, token, lse, m c / D and, with an entropy bonus, its coefficient
// and mu; rows in [n_live, round_up(n_live, 128)) are zeroed so that the last
// tile holds finite values and no gradient
__global__ void live_gather_kernel(int H, int tok_shift, const int32_t* __restrict__ counts,
                                   const int32_t* __restrict__ live_map,
                                   const uint16_t* __restrict__ h_p, const int32_t* __restrict__ tok_p,
                                   const float* __restrict__ lse, const float* __restrict__ coef,
                                   const float* __restrict__ ecoef, const float* __restrict__ mu,
                                   uint16_t* __restrict__ h_l, int32_t* __restrict__ tok_l,
                                   float* __restrict__ lse_l, float* __restrict__ coef_l,
                                   float* __restrict__ ecoef_l, float* __restrict__ mu_l) {
  const int n = counts[3];
  const int nz = ((n + kTileM - 1) / kTileM) * kTileM;
  const int vpr = H / 8;   // 16-byte vectors per row
  const int64_t total = (int64_t)nz * vpr;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const int j = (int)(i / vpr), v = (int)(i - (int64_t)j * vpr);
    uint4 val = make_uint4(0, 0, 0, 0);
    if (j < n) {
      const int k = live_map[j];
      val = reinterpret_cast<const uint4*>(h_p + (int64_t)k * H)[v];
      if (v == 0) {
        tok_l[j] = tok_p[k] - tok_shift;
        lse_l[j] = lse[k];
        coef_l[j] = coef[k];
        if (ecoef) {
          ecoef_l[j] = ecoef[k];
          mu_l[j] = mu[k];
        }
      }
    } else if (v == 0) {
      tok_l[j] = 0;
      lse_l[j] = 0.f;
      coef_l[j] = 0.f;
      if (ecoef) {
        ecoef_l[j] = 0.f;
        mu_l[j] = 0.f;
      }
    }
    reinterpret_cast<uint4*>(h_l + (int64_t)j * H)[v] = val;
  }
}

// dhidden_out[t] = bf16(dh32[live_of[pos[t]]]) for rows with a gradient, 0 for
// masked rows and rows whose gradient coefficient is 0
__global__ void cast_dh_kernel(const float* __restrict__ dh32, const int32_t* __restrict__ pos,
                               const int32_t* __restrict__ live_of, int T, int H, uint16_t* __restrict__ out) {
  const int vpr = H / 8;
  const int64_t total = (int64_t)T * vpr;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const int t = (int)(i / vpr), v = (int)(i - (int64_t)t * vpr);
    const int kp = pos[t];
    const int k = kp >= 0 ? live_of[kp] : -1;
    uint4 o = make_uint4(0, 0, 0, 0);
    if (k >= 0) {
      const float4* src = reinterpret_cast<const float4*>(dh32 + (int64_t)k * H) + 2 * v;
      const float4 a = src[0], c = src[1];
      o.x = pack_bf16x2(a.x, a.y);
      o.y = pack_bf16x2(a.z, a.w);
      o.z = pack_bf16x2(c.x, c.y);
      o.w = pack_bf16x2(c.z, c.w);
    }
    reinterpret_cast<uint4*>(out + (int64_t)t * H)[v] = o;
  }
}

}  // namespace

// words[0]: the call's abort word, words[1]: a counter nothing raises,
// words[2]: 1 if the wait returned true, 2 if it gave up
__global__ void wait_selftest_kernel(uint32_t* words, unsigned* err) {
  __shared__ int abort_sh;
  if (threadIdx.x == 0) {
    abort_sh = 0;
    volatile int* abort_flag = &abort_sh;
    words[2] = turn_wait(words + 1, 1u, abort_flag, words, err) ? 1u : 2u;
  }
}

cudaError_t launch_wait_selftest(uint32_t* words, unsigned* err, cudaStream_t s) {
  wait_selftest_kernel<<<1, 32, 0, s>>>(words, err);
  return cudaGetLastError();
}

cudaError_t launch_group_advantages(const float* rewards, const int32_t* gids, int n, double eps, float* out,
                                    unsigned* err, cudaStream_t s) {
  return launch_advantages(rewards, gids, n, kAdvGrpo, eps, out, err, s);
}

cudaError_t launch_advantages(const float* rewards, const int32_t* gids, int n, int estimator, double eps,
                              float* out, unsigned* err, cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  if (estimator == kAdvReinforcePP) {
    // one warp over the whole batch; zero everything first so a batch of one gives 0
    cudaError_t e = cudaMemsetAsync(out, 0, sizeof(float) * n, s);
    if (e != cudaSuccess) return e;
    group_adv_kernel<<<1, 32, 0, s>>>(rewards, nullptr, n, eps, estimator, out, err);
    return cudaGetLastError();
  }
  const int threads = 256;
  const int blocks = (int)(((int64_t)n * 32 + threads - 1) / threads);
  group_adv_kernel<<<blocks, threads, 0, s>>>(rewards, gids, n, eps, estimator, out, err);
  return cudaGetLastError();
}

cudaError_t launch_broadcast(const float* adv, const int32_t* rot, int n_resp, int T, float* out, cudaStream_t s) {
  if (T <= 0) return cudaSuccess;
  const int blocks = min((T + 255) / 256, 4096);
  broadcast_kernel<<<blocks, 256, 0, s>>>(adv, rot, n_resp, T, out);
  return cudaGetLastError();
}

cudaError_t launch_mask_count(const uint8_t* mask, int64_t T, int64_t* out, cudaStream_t s) {
  cudaError_t e = cudaMemsetAsync(out, 0, sizeof(int64_t), s);
  if (e != cudaSuccess || T <= 0) return e;
  const int64_t nb = (T / 16 + 255) / 256 + 1;
  const int blocks = (int)(nb < 1024 ? nb : 1024);
  mask_count_kernel<<<blocks, 256, 0, s>>>(mask, T, reinterpret_cast<unsigned long long*>(out));
  return cudaGetLastError();
}

cudaError_t launch_compact(const uint8_t* mask, int T, const Workspace& ws, cudaStream_t s) {
  compact_kernel<<<1, 1024, 0, s>>>(mask, T, ws.row_map, ws.pos_of_row, ws.counts);
  return cudaGetLastError();
}

cudaError_t launch_gather(const uint16_t* hidden, const int32_t* tokens, const float* b, const float* adv, int T,
                          int Tcap, int H, const Workspace& ws, int n_sm, cudaStream_t s, int tok_shift) {
  (void)T;
  gather_kernel<<<n_sm * 8, 256, 0, s>>>(hidden, tokens, b, adv, tok_shift, Tcap, H, ws.row_map, ws.counts, ws.h_p,
                                         ws.tok_p, b ? ws.b_p : nullptr, adv ? ws.adv_p : nullptr);
  return cudaGetLastError();
}

cudaError_t launch_merge(bool loss_mode, int Tcap, int V, int n_split, double denom, float clip_lo, float clip_hi,
                         const Workspace& ws, float* logp_out, float* ent_out, float* tokloss_out, unsigned* err,
                         cudaStream_t s) {
  const int blocks = Tcap / kTileM;
  merge_kernel<<<blocks, kTileM, 0, s>>>(loss_mode ? 1 : 0, Tcap, V, n_split, denom, clip_lo, clip_hi, ws.counts,
                                          ws.row_map, ws.tok_p, ws.b_p, ws.adv_p, ws.part, ws.zx, ws.lse, ws.coef,
                                          ws.tile_flag, ws.red, logp_out, ent_out, tokloss_out, nullptr, nullptr,
                                          err);
  return cudaGetLastError();
}

cudaError_t launch_merge_stats_ex(int Tcap, int V, int n_split, const Workspace& ws, float* logp_out, float* ent_out,
                                  unsigned* err, cudaStream_t s) {
  const int blocks = Tcap / kTileM;
  if (blocks == 0) return cudaSuccess;
  merge_kernel<<<blocks, kTileM, 0, s>>>(0, Tcap, V, n_split, 0.0, 0.f, 0.f, ws.counts, ws.row_map, ws.tok_p, ws.b_p,
                                          ws.adv_p, ws.part, ws.zx, ws.lse, ws.coef, ws.tile_flag, ws.red, logp_out,
                                          ent_out, nullptr, ws.lp_p, ws.ent_p, err);
  return cudaGetLastError();
}

cudaError_t launch_seq_gate(int T, int Tcap, const LossEx& ex, const Workspace& ws, unsigned* err, cudaStream_t s) {
  const int blocks = (Tcap + 255) / 256;
  if (blocks == 0 || ex.seq == nullptr) return cudaSuccess;
  seq_gate_kernel<<<blocks, 256, 0, s>>>(T, ex.seq, ws.counts, ws.row_map, ws.lp_p, ws.b_p, ex.gate_lo, ex.gate_hi,
                                         ws.gate_p, ws.counts + 2, err);
  return cudaGetLastError();
}

cudaError_t launch_loss_rows_ex(int Tcap, double denom, float clip_lo, float clip_hi, const LossEx& ex,
                                const Workspace& ws, float* tokloss_out, cudaStream_t s) {
  const int blocks = Tcap / kTileM;
  if (blocks == 0) return cudaSuccess;
  loss_rows_ex_kernel<<<blocks, kTileM, 0, s>>>(Tcap, denom, clip_lo, clip_hi, ex, ws.counts, ws.row_map, ws.b_p,
                                                 ws.adv_p, ws.lp_p, ws.ent_p, ws.lse,
                                                 ex.seq ? ws.gate_p : nullptr, ws.coef, ws.ecoef, ws.mu,
                                                 ws.tile_flag, ws.red, tokloss_out);
  return cudaGetLastError();
}

cudaError_t launch_finalize(int Tcap, double denom, bool with_ecoef, const Workspace& ws, float* loss_out,
                            void* stats_out, void* stats_ex_out, unsigned* err, cudaStream_t s) {
  (void)Tcap;
  finalize_kernel<<<1, 1024, 0, s>>>(denom, ws.counts, ws.tile_list, ws.red, loss_out,
                                     reinterpret_cast<StatsDev*>(stats_out),
                                     reinterpret_cast<StatsExDev*>(stats_ex_out), ws.coef,
                                     with_ecoef ? ws.ecoef : nullptr, ws.live_map, ws.live_of, err);
  return cudaGetLastError();
}

cudaError_t launch_live_gather(int H, bool with_ecoef, const Workspace& ws, int n_sm, cudaStream_t s) {
  live_gather_kernel<<<n_sm * 8, 256, 0, s>>>(H, 0, ws.counts, ws.live_map, ws.h_p, ws.tok_p, ws.lse, ws.coef,
                                              with_ecoef ? ws.ecoef : nullptr, ws.mu, ws.h_l, ws.tok_l, ws.lse_l,
                                              ws.coef_l, ws.ecoef_l, ws.mu_l);
  return cudaGetLastError();
}

cudaError_t launch_vp_local(int T, int Tcap, int V_s, int n_split, const Workspace& ws, float4* out,
                            cudaStream_t s) {
  if (T <= 0) return cudaSuccess;
  vp_local_kernel<<<(T + 255) / 256, 256, 0, s>>>(T, Tcap, V_s, n_split, ws.pos_of_row, ws.tok_p, ws.part, ws.zx,
                                                   out);
  return cudaGetLastError();
}

cudaError_t launch_vp_merge(int T, int Tcap, int n_shards, double denom, float clip_lo, float clip_hi,
                            const float4* parts, const float* b, const float* adv, const Workspace& ws,
                            float* lse_out, float* coef_out, float* logp_out, float* ent_out, float* tokloss_out,
                            unsigned* err, cudaStream_t s) {
  const int blocks = Tcap / kTileM;
  if (blocks == 0) return cudaSuccess;
  vp_merge_kernel<<<blocks, kTileM, 0, s>>>(T, n_shards, denom, clip_lo, clip_hi, ws.counts, ws.row_map, parts, b,
                                            adv, ws.coef, ws.tile_flag, ws.red, lse_out, coef_out, logp_out,
                                            ent_out, tokloss_out, err);
  return cudaGetLastError();
}

cudaError_t launch_vp_live(int T, const float* coef, const Workspace& ws, cudaStream_t s) {
  vp_live_kernel<<<1, 1024, 0, s>>>(T, coef, ws.counts, ws.tile_list, ws.live_map, ws.live_of);
  return cudaGetLastError();
}

cudaError_t launch_vp_gather(const uint16_t* hidden, const int32_t* tokens, const float* lse, const float* coef,
                             int tok_shift, int H, const Workspace& ws, int n_sm, cudaStream_t s) {
  live_gather_kernel<<<n_sm * 8, 256, 0, s>>>(H, tok_shift, ws.counts, ws.live_map, hidden, tokens, lse, coef,
                                              nullptr, nullptr, ws.h_l, ws.tok_l, ws.lse_l, ws.coef_l, ws.ecoef_l,
                                              ws.mu_l);
  return cudaGetLastError();
}

cudaError_t launch_vp_dh_out(const Workspace& ws, int T, int H, float* out, int n_sm, cudaStream_t s) {
  if (T <= 0) return cudaSuccess;
  vp_dh_out_kernel<<<n_sm * 8, 256, 0, s>>>(ws.dh32, ws.live_of, T, H, out);
  return cudaGetLastError();
}

cudaError_t launch_cast_dh(const Workspace& ws, int T, int H, uint16_t* dh_out, int n_sm, cudaStream_t s) {
  if (T <= 0) return cudaSuccess;
  cast_dh_kernel<<<n_sm * 8, 256, 0, s>>>(ws.dh32, ws.pos_of_row, ws.live_of, T, H, dh_out);
  return cudaGetLastError();
}

}  // namespace molt
