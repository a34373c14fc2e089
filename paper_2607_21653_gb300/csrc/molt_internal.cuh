// Internal launch interface between the C-ABI layer (api.cu) and the kernels.
#pragma once

#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>
#include <string>

#include "../../include/molt.h"

namespace molt {

constexpr int kTileM = 128;   // token rows per tile (TMEM lanes)
constexpr int kFwdBN = 256;   // vocab columns per forward MMA tile
constexpr int kBwdBV = 256;   // vocab columns per backward unit
constexpr int kBK = 64;       // K elements per 128-byte swizzled row

// Device pointers into one call's workspace (all regions 256-byte aligned).
struct Workspace {
  int32_t* counts;      // [0] active rows n, [1] backward tiles, [2] rejected sequences,
                        // [3] rows with a gradient (the backward's rows)
  int32_t* row_map;     // [T]    packed row -> original row
  int32_t* pos_of_row;  // [T]    original row -> packed row or -1
  int32_t* tok_p;       // [Tcap] packed tokens
  float* b_p;           // [Tcap] packed behaviour log-probs
  float* adv_p;         // [Tcap] packed advantages
  uint16_t* h_p;        // [Tcap, H] packed hidden rows (bf16 bits), rows >= n zeroed
  float4* part;         // [S, Tcap] per-split (max, sum exp, sum exp*(z-max), -)
  float* zx;            // [Tcap] target logit
  float* lse;           // [Tcap]
  float* coef;          // [Tcap] m c / D
  int32_t* tile_flag;   // [Tcap/128]
  int32_t* tile_list;   // [Tcap/128]
  double* red;          // [n_tiles * kRedSlots] per-tile partial sums
  float* dh32;          // [Tcap, H] fp32 dhidden accumulator, by backward row (loss call only)
  // rows with a nonzero gradient coefficient, packed again (loss call only)
  int32_t* live_map;    // [Tcap] backward row -> packed row
  int32_t* live_of;     // [Tcap] packed row -> backward row or -1
  uint16_t* h_l;        // [Tcap, H] their hidden rows (bf16 bits), rows >= n_live zeroed
  int32_t* tok_l;       // [Tcap] their tokens
  float* lse_l;         // [Tcap]
  float* coef_l;        // [Tcap] m c / D
  float* ecoef_l;       // [Tcap] entropy-bonus coefficient (extended objective)
  float* mu_l;          // [Tcap]
  uint32_t* turns;      // deterministic schedule: abort word + turn counters, or nullptr
  // extended objective (loss call only)
  float* lp_p;          // [Tcap] packed log-probs
  float* ent_p;         // [Tcap] packed entropies
  float* ecoef;         // [Tcap] m w entropy_coef / D
  float* mu;            // [Tcap] sum_v p_v z_v = lse - entropy
  uint8_t* gate_p;      // [Tcap] sequence-gate weight per packed row
};
constexpr int kRedSlots = 8;

// advantage estimators (values of molt_adv_estimator)
constexpr int kAdvGrpo = 0, kAdvGroupMean = 1, kAdvDrGrpo = 2, kAdvRloo = 3, kAdvReinforcePP = 4;

struct FwdArgs {
  const int32_t* tok_p;
  const int32_t* counts;
  int rows_cap;
  int V, H;
  int n_split;
  int n_vtiles;
  float4* part;
  float* zx;
  unsigned* err;
};

struct BwdArgs {
  const int32_t* tok_p;
  const float* lse;
  const float* coef;
  const int32_t* counts;     // counts[1] = backward tiles
  const int32_t* tile_list;
  int V, H;
  int n_vchunks;
  int vc_begin;              // single-CTA backward: first 256-column vocab chunk of its range
  int tile_group;            // token tiles per raster group
  const float* ecoef;        // entropy-bonus coefficient per row, or nullptr
  const float* mu;           // sum_v p_v z_v per row (with ecoef)
  float* dh32;               // [Tcap, H] fp32 dhidden accumulator
  float* dW;                 // [V, H] fp32 dW
  int det_clusters;          // 0: raster schedule; > 0: deterministic schedule on this many
                             // clusters (a multiple of 4), reduce-adds taking turns
  uint32_t* det_abort;       // deterministic: set once any turn wait gives up (zeroed per call)
  uint32_t* det_dh_turns;    // deterministic: [token quads, H jobs, 32] counters, blocks done
  uint32_t* det_dw_turns;    // deterministic: [vocab blocks, H jobs, 32] counters, quads done
  unsigned* err;
};

// options of the extended objective as the row kernels see them
struct LossEx {
  float kl_coef;
  float entropy_coef;
  const float* ref_logp;     // [T] original order
  const int32_t* seq;        // [T] original order, or nullptr
  double gate_lo, gate_hi;
};

// api.cu: shared host helpers
void set_last_error(const std::string& msg);
// benchmark timing hook (molt_set_timing_events): record the calling thread's
// start (stop = false) or stop event of kernel group k on stream s, if set
void timing_event(int k, bool stop, cudaStream_t s);
unsigned* device_status_word(molt_status* st);   // current device's status word
int device_sm_count();                           // current device's SM count
molt_status encode_tmap_2d(CUtensorMap* m, CUtensorMapDataType dt, int elem_bytes, const void* base, uint64_t rows,
                           uint64_t cols, uint32_t box_cols, uint32_t box_rows);

// rows.cu
// one bounded turn wait on a counter nothing raises (words: 3 zeroed uint32)
cudaError_t launch_wait_selftest(uint32_t* words, unsigned* err, cudaStream_t s);
cudaError_t launch_group_advantages(const float* rewards, const int32_t* gids, int n, double eps, float* out,
                                    unsigned* err, cudaStream_t s);
cudaError_t launch_advantages(const float* rewards, const int32_t* gids, int n, int estimator, double eps,
                              float* out, unsigned* err, cudaStream_t s);
cudaError_t launch_broadcast(const float* adv, const int32_t* rot, int n_resp, int T, float* out, cudaStream_t s);
cudaError_t launch_mask_count(const uint8_t* mask, int64_t T, int64_t* out, cudaStream_t s);
cudaError_t launch_compact(const uint8_t* mask, int T, const Workspace& ws, cudaStream_t s);
// tok_shift is subtracted from every token (a vocabulary shard's first column)
cudaError_t launch_gather(const uint16_t* hidden, const int32_t* tokens, const float* b, const float* adv, int T,
                          int Tcap, int H, const Workspace& ws, int n_sm, cudaStream_t s, int tok_shift = 0);
cudaError_t launch_merge(bool loss_mode, int Tcap, int V, int n_split, double denom, float clip_lo, float clip_hi,
                         const Workspace& ws, float* logp_out, float* ent_out, float* tokloss_out, unsigned* err,
                         cudaStream_t s);
cudaError_t launch_finalize(int Tcap, double denom, bool with_ecoef, const Workspace& ws, float* loss_out,
                            void* stats_out, void* stats_ex_out, unsigned* err, cudaStream_t s);
// the rows with a gradient (finalize's list) packed into whole tiles for the backward
cudaError_t launch_live_gather(int H, bool with_ecoef, const Workspace& ws, int n_sm, cudaStream_t s);
// extended objective: packed stats -> sequence gate -> loss rows
cudaError_t launch_merge_stats_ex(int Tcap, int V, int n_split, const Workspace& ws, float* logp_out, float* ent_out,
                                  unsigned* err, cudaStream_t s);
cudaError_t launch_seq_gate(int T, int Tcap, const LossEx& ex, const Workspace& ws, unsigned* err, cudaStream_t s);
cudaError_t launch_loss_rows_ex(int Tcap, double denom, float clip_lo, float clip_hi, const LossEx& ex,
                                const Workspace& ws, float* tokloss_out, cudaStream_t s);
// dhidden_out[t] = bf16(the fp32 accumulator row of t)
cudaError_t launch_cast_dh(const Workspace& ws, int T, int H, uint16_t* dh_out, int n_sm, cudaStream_t s);
// vocabulary shards: one shard's per-row statistics (original order) from the
// forward's split partials; the merge of all shards' statistics with the Eq. 2
// terms; the rows of a shard's backward (coef != 0) and their packing; the
// shard's dhidden contribution in the original order (fp32)
cudaError_t launch_vp_local(int T, int Tcap, int V_s, int n_split, const Workspace& ws, float4* out, cudaStream_t s);
cudaError_t launch_vp_merge(int T, int Tcap, int n_shards, double denom, float clip_lo, float clip_hi,
                            const float4* parts, const float* b, const float* adv, const Workspace& ws,
                            float* lse_out, float* coef_out, float* logp_out, float* ent_out, float* tokloss_out,
                            unsigned* err, cudaStream_t s);
cudaError_t launch_vp_live(int T, const float* coef, const Workspace& ws, cudaStream_t s);
cudaError_t launch_vp_gather(const uint16_t* hidden, const int32_t* tokens, const float* lse, const float* coef,
                             int tok_shift, int H, const Workspace& ws, int n_sm, cudaStream_t s);
cudaError_t launch_vp_dh_out(const Workspace& ws, int T, int H, float* out, int n_sm, cudaStream_t s);

// lmhead_fwd.cu
cudaError_t launch_lmhead_fwd(const CUtensorMap& tm_h, const CUtensorMap& tm_w, const FwdArgs& a, int grid,
                              cudaStream_t s);
// lmhead_bwd4.cu (clusters of two CTA pairs; H % 128 == 0)
int lmhead_bwd_quad_clusters(int n_sm);       // clusters one raster launch runs
int lmhead_bwd_quad_det_clusters(int n_sm);   // clusters of the deterministic schedule (multiple of 4)
// host: count kernels the library enqueued (molt_kernel_launches)
void note_launches(int n);

cudaError_t launch_lmhead_bwd_quad(const CUtensorMap& tm_hz, const CUtensorMap& tm_wz, const CUtensorMap& tm_h,
                                   const CUtensorMap& tm_w_n, const CUtensorMap& tm_dh, const CUtensorMap& tm_dw,
                                   const BwdArgs& a, int n_sm, cudaStream_t s);
// lmhead_bwd.cu
cudaError_t launch_lmhead_bwd(const CUtensorMap& tm_h, const CUtensorMap& tm_w_z, const CUtensorMap& tm_w_n,
                              const CUtensorMap& tm_dh, const CUtensorMap& tm_dw, const BwdArgs& a, int grid,
                              cudaStream_t s);

}  // namespace molt
