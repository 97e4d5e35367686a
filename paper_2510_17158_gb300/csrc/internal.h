// Host-side interface between the C ABI (api.cu) and the kernel translation units.
#pragma once

#include <cstddef>
#include <cstdint>
#include <functional>
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

namespace grpo {

struct WsHeader;

// Packed rows: the scored tokens of all sequences, in order, numbered 0 .. N-1 (then padded to a
// multiple of 128). The GEMMs run 128-row tiles over packed rows; the dz scratch, the dH
// accumulator and the forward partials are indexed by packed row.
constexpr int kTileRows = 128;
// Vocabulary tile (N of the forward and dz GEMMs) and hidden tile (N of the dH / dW GEMMs).
constexpr int kTileN = 256;
// Vocabulary tiles merged on chip by one forward work unit before it writes partial statistics
// (a strip). One tile per unit: CTAs that read the same W tile then start and finish it together
// (longer strips let them drift apart and re-read W from HBM: 8-tile strips ran the forward
// GEMM 6-9 % slower at the 2 x 16, T = 16384, d = 5120 workload), at the price of 16 bytes of
// statistics per token and 256 vocabulary columns for the merge to read back.
#ifndef GRPO_FWD_TILES_PER_STRIP
#define GRPO_FWD_TILES_PER_STRIP 1
#endif
constexpr int kFwdTilesPerStrip = GRPO_FWD_TILES_PER_STRIP;

// FWD_KL / DZ_KL: the forward / dz roles with a second product z_ref = W_ref h_ref (the frozen
// reference model) in the other half of tensor memory, for Eq. 1's exact KL term.
enum GemmRole : int {
  ROLE_FWD = 0, ROLE_DZ = 1, ROLE_DH = 2, ROLE_DW = 3, ROLE_FWD_KL = 4, ROLE_DZ_KL = 5
};

// Arguments of the tcgen05 GEMM kernels (one struct for the four roles).
struct GemmArgs {
  int S, T, d, V;
  const int32_t* row_pos;   // [rows_cap] packed row -> position (-1 for padding rows)
  WsHeader* hdr;            // num_tiles, status word
  const int32_t* tokens;    // [S*T]
  const uint8_t* mask;      // [S*T]
  long long rows_cap;       // packed-row capacity: S*T rounded up to a multiple of 128
  // vocabulary chunk (DZ / DH / DW)
  int vc0, vc_len, dz_pitch;
  // FWD: partial statistics per (strip, tile row) and the target logit per position
  float4* partials;
  int num_strips;
  float* zy;
  // DZ: per-position coefficient g and log-normaliser, bf16 dz scratch [rows_cap, dz_pitch]
  const float* g;
  const float* lse;
  __nv_bfloat16* dz;
  // DH: output (H's dtype), f32 accumulator in tile space, mode (0 single chunk, 1 first,
  //     2 middle, 3 last)
  __nv_bfloat16* dH;
  float* dH_acc;
  int dh_mode;
  // DW: f32 [V, d]
  float* dW;
  // test hook: nonzero makes CTA 0's producer leave its first stage unfilled
  int inject_stall;
  // vocabulary-parallel shard: W holds global rows v_offset .. v_offset + V - 1 (0 otherwise)
  int v_offset;
  // DH: write the final dH in f32 (a shard's partial sum) instead of H's dtype
  int dh_f32;
  // FWD_KL: second set of per-(strip, row) statistics (sum e^{z-m} z_ref, m_ref, s_ref, 0)
  float4* partials2;
  // DZ_KL: per-position log-normaliser of the reference, exact KL, and its coefficient beta*w
  const float* lse_ref;
  const float* kl;
  const float* c;
  // progress window (0 = off): producers wait at every `win_check`-th k-block until the CTAs of
  // the launch are on average within `win_lag` checkpoints of them (counters in hdr)
  int win_check, win_lag;
};

// Fills the progress-window fields of `a` from the process-wide setting (grpo_set_gemm_window).
void gemm_window_config(GemmArgs& a);

// Kernel accounting of the C ABI (grpo_timing_*): runs `launch` (which enqueues one kernel of
// kind `kernel_id`, a GRPO_K_* value, on `st`), counts it and, with timing on, brackets it with
// events on `st`. Returns GRPO_OK or GRPO_ERR_CUDA (GRPO_ERR_INVALID_ARG for a bad id).
int counted_launch(int kernel_id, cudaStream_t st, const std::function<cudaError_t()>& launch);
// Current value of the grpo_debug_inject_stall test hook (nonzero = on).
int debug_inject_stall();

// Launches (all asynchronous on `st`; return the cudaError_t of the launch).
cudaError_t launch_mask_scan(const uint8_t* mask, int S, int T, int32_t* counts,
                             cudaStream_t st);
// Token packing: counts -> seq_base [S+1] (prefix), header (num_tiles = packed rows / 128,
// total_valid), row_pos [rows_cap] (packed row -> position, -1 for padding) and pos_row [S*T]
// (position -> packed row, -1 if unscored).
cudaError_t launch_pack(const uint8_t* mask, const int32_t* counts, int S, int T,
                        long long rows_cap, int32_t* seq_base, int32_t* row_pos, int32_t* pos_row,
                        WsHeader* hdr, cudaStream_t st);
// Hp [packed rows, d] = H rows at row_pos (bf16), zero for padding rows.
cudaError_t launch_gather_rows(const void* H, int d, const int32_t* row_pos, const WsHeader* hdr,
                               long long rows_cap, void* Hp, cudaStream_t st);
cudaError_t launch_group_adv(const float* rewards, const int32_t* go, int num_groups, int S,
                             int std_mode, float std_eps, float* adv, WsHeader* hdr,
                             cudaStream_t st);
cudaError_t launch_fwd_merge(const float4* partials, long long rows_cap, int num_strips,
                             const float* zy, const int32_t* pos_row,
                             const int32_t* tokens, const uint8_t* mask, int S, int T, int V,
                             float* logp, float* lse, float* entropy, int32_t* argmax,
                             WsHeader* hdr, cudaStream_t st);
// mode 0 GRPO (per-token KL estimator), 1 SFT, 2 GRPO with the exact KL (reads kl, writes
// c = beta * w per position).
cudaError_t launch_loss_tokens(const uint8_t* mask, const float* logp, const float* old_logp,
                               const float* ref_logp, const float* adv,
                               const int32_t* valid_count, int S, int T, float eps_low,
                               float eps_high, float beta, int agg, double norm, int mode,
                               const WsHeader* hdr, float* g, float* seq_loss, cudaStream_t st,
                               const float* kl = nullptr, float* c = nullptr);
cudaError_t launch_fwd_merge_kl(const float4* partials, const float4* partials2,
                                long long rows_cap, int num_strips, const float* zy,
                                const int32_t* pos_row, const int32_t* tokens,
                                const uint8_t* mask, int S, int T, int V, float* logp, float* lse,
                                float* entropy, int32_t* argmax, float* lse_ref, float* kl,
                                WsHeader* hdr, cudaStream_t st);
cudaError_t launch_rewards(const uint8_t* correct, const float* t_base, const float* t_new,
                           const int32_t* used, const int32_t* avail, int n, float lambda_tools,
                           float* r, cudaStream_t st);
cudaError_t launch_loss_final(const float* seq_loss, int S, int agg, double norm,
                              const WsHeader* hdr, float* loss_out, cudaStream_t st);
cudaError_t launch_dh_zero_masked(const uint8_t* mask, int S, int T, int d, void* dH,
                                  int elem_bytes, cudaStream_t st);
cudaError_t launch_shard_stats(const float4* partials, long long rows_cap, int num_strips,
                               const float* zy_ws, const int32_t* pos_row,
                               const int32_t* tokens, const uint8_t* mask, int S, int T,
                               int V_shard, int v_offset, float4* stats, float* zy_out,
                               cudaStream_t st);
cudaError_t launch_merge_shards(const float4* stats, const float* zy, int P,
                                const int32_t* tokens, const uint8_t* mask, int S, int T,
                                int V_total, float* logp, float* lse, float* entropy,
                                int32_t* argmax, WsHeader* hdr, cudaStream_t st);
cudaError_t launch_f32_fwd(const float* H, const float* W, const int32_t* tokens,
                           const uint8_t* mask, int S, int T, int d, int V, float* logp,
                           float* lse, float* entropy, int32_t* argmax, WsHeader* hdr,
                           cudaStream_t st);
cudaError_t launch_f32_dh(const float* H, const float* W, const int32_t* tokens,
                          const uint8_t* mask, const float* lse, const float* g, int S, int T,
                          int d, int V, float* dH, cudaStream_t st);
cudaError_t launch_f32_dw(const float* H, const float* W, const int32_t* tokens,
                          const uint8_t* mask, const float* lse, const float* g, int S, int T,
                          int d, int V, float* dW, cudaStream_t st);

// Tensor-core tile mode that GEMM role `role` (ROLE_*) runs in (the process-wide choice made
// through grpo_set_tile_mode / grpo_set_role_tile_mode): 0 single CTA, 128 x 256 tiles
// (cta_group::1); 1 CTA pair, 256 x 256 tiles (cta_group::2); 2 CTA pair, 256 x 512 tiles.
int gemm_role_tile_mode(int role);

// tcgen05 GEMM launches. `grid` = persistent CTAs.
size_t gemm_smem_bytes();
// CTAs per cluster of a tile mode (1 or 2), 256-column tiles per work unit (1, or 2 in mode 2)
// and the rows of the K-major B box each CTA loads (256, or 128 in the pair modes: the pair
// splits B by rows). A boxes are always 128 rows (K-major) or 64 x 64 (MN-major).
int gemm_cluster_size(int tile_mode);
int gemm_col_tiles_per_unit(int tile_mode);
int gemm_b_box_rows(int tile_mode);
// Clusters of a tile mode that can be resident at once (cudaOccupancyMaxActiveClusters, cached
// per device), at most one per `cluster size` SMs.
int gemm_max_clusters(int tile_mode);
// Persistent grid for `row_tiles` x `col_tiles` output tiles of 128 x 256: one CTA per SM, or in
// the pair modes as many pairs as can be resident, each taking 2 consecutive row tiles (and, in
// mode 2, 2 consecutive column tiles) per unit; never more CTAs than units need.
int gemm_grid(long long row_tiles, long long col_tiles, int tile_mode);
// tile_mode 1, 2: pair kernels; `grid` must be even and the K-major B map's box
// gemm_b_box_rows(tile_mode) rows. A forward unit in mode 2 needs one-tile strips.
// mapA2 / mapB2 (H_ref, W_ref) are read by the KL roles only (single-CTA tiles).
cudaError_t launch_gemm(int role, const CUtensorMap& mapA, const CUtensorMap& mapB,
                        const GemmArgs& args, int grid, int tile_mode, cudaStream_t st,
                        const CUtensorMap* mapA2 = nullptr, const CUtensorMap* mapB2 = nullptr);

}  // namespace grpo
