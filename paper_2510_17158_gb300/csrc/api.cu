// C ABI of the GRPO library: argument checks, workspace layout, TMA descriptors and the launch
// sequence of each entry point (declared and documented in include/grpo.h).
#include <cudaTypedefs.h>

#include <atomic>
#include <cstring>
#include <mutex>
#include <vector>

#include "../../include/grpo.h"
#include "common.cuh"
#include "internal.h"

using namespace grpo;

namespace {

// ------------------------------------------------------------------------------------------
// kernel accounting
// ------------------------------------------------------------------------------------------
const char* const kKernelNames[GRPO_K_COUNT] = {
    "mask_scan",       "pack_tokens",  "group_adv",   "fwd_gemm_tc",  "fwd_merge",
    "loss_tokens",     "loss_final",   "bwd_dz_gemm_tc", "bwd_dh_gemm_tc", "bwd_dw_gemm_tc",
    "dh_zero_unscored", "f32_fwd",     "f32_dh",      "f32_dw",      "rewards",
    "shard_stats",     "merge_shards", "gather_rows"};

struct EventPair {
  cudaEvent_t a, b;
};

std::mutex g_mu;
std::atomic<int> g_timing{0};
std::atomic<int> g_inject_stall{0};
// Tensor-core tile mode (GRPO_TILE_*) of each LM-head GEMM role, GRPO_ROLE_FWD .. GRPO_ROLE_DW.
// The forward product and the dz recompute (K = d, a short reduction per tile) keep single-CTA
// tiles, whose two accumulators overlap each tile's epilogue with the next tile's MMAs. dH and
// dW (K = vocabulary / tokens: thousands of k-blocks per tile) take the 256 x 512 CTA-pair
// tiles, which stage half of a single-CTA tile's operand bytes per flop.
constexpr int kRoleDefault[4] = {GRPO_TILE_SINGLE, GRPO_TILE_SINGLE, GRPO_TILE_CTA_PAIR_WIDE,
                                 GRPO_TILE_CTA_PAIR_WIDE};
std::atomic<int> g_role_mode[4] = {{kRoleDefault[0]}, {kRoleDefault[1]}, {kRoleDefault[2]},
                                   {kRoleDefault[3]}};
// GEMM progress window of the long-K roles (checkpoint spacing, lag): by default a barrier every
// 256 k-blocks of dH and dW (lag 1), which keeps the CTA pairs that share a dz or W tile within
// the L2's reuse window (dH and dW 296 -> 265-267 ms at 2 x 16 completions, T = 16384,
// d = 5120, V = 151936; a barrier at every work unit's start: 267-268 ms, 10 % more DRAM bytes).
std::atomic<int> g_win_check{GRPO_GEMM_WINDOW_DEFAULT_CHECK}, g_win_lag{GRPO_GEMM_WINDOW_DEFAULT_LAG};
std::atomic<long long> g_launches[GRPO_K_COUNT];
std::vector<EventPair> g_pending[GRPO_K_COUNT];
double g_total_ms[GRPO_K_COUNT];
std::vector<EventPair> g_free_events;

bool take_events(EventPair* p) {
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_free_events.empty()) {
    *p = g_free_events.back();
    g_free_events.pop_back();
    return true;
  }
  if (cudaEventCreate(&p->a) != cudaSuccess) return false;
  if (cudaEventCreate(&p->b) != cudaSuccess) {
    cudaEventDestroy(p->a);
    return false;
  }
  return true;
}

// Runs `launch` (which enqueues one kernel on `st` and returns its cudaError_t), counting it
// and, with timing on, bracketing it with events.
template <class F>
int counted(int kid, cudaStream_t st, F&& launch) {
  EventPair ev{};
  const bool timed = g_timing.load() != 0 && take_events(&ev);
  if (timed) cudaEventRecord(ev.a, st);
  const cudaError_t e = launch();
  if (timed) {
    cudaEventRecord(ev.b, st);
    std::lock_guard<std::mutex> lk(g_mu);
    g_pending[kid].push_back(ev);
  }
  g_launches[kid].fetch_add(1);
  return e == cudaSuccess ? GRPO_OK : GRPO_ERR_CUDA;
}

}  // namespace

namespace grpo {
int counted_launch(int kernel_id, cudaStream_t st, const std::function<cudaError_t()>& launch) {
  if (kernel_id < 0 || kernel_id >= GRPO_K_COUNT) return GRPO_ERR_INVALID_ARG;
  return counted(kernel_id, st, launch);
}

int debug_inject_stall() { return g_inject_stall.load(); }
}  // namespace grpo

namespace {

#define GRPO_TRY(x)             \
  do {                          \
    const int _st = (x);        \
    if (_st != GRPO_OK) return _st; \
  } while (0)

// ------------------------------------------------------------------------------------------
// workspace layout
// ------------------------------------------------------------------------------------------
size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

struct Layout {
  int max_tiles;        // packed-row tiles of the worst case (every position scored)
  long long rows_cap;   // packed-row capacity: S*T rounded up to a multiple of 128
  int num_strips;
  int v_round;          // V rounded up to a multiple of 256
  size_t seq_base, row_pos, pos_row, counts, zy, partials, partials2, g, cvec, seq_loss, hp, hrp;
  size_t fixed_end;     // end of the regions that do not depend on the vocabulary chunk
};

// `kl`: the exact-KL entry points' layout, with the reference model's packed hidden states and
// forward statistics; the other entry points leave those two regions out (10 GB at 2 x 16
// completions of T = 16384, d = 5120, V = 151936).
Layout make_layout(int S, int T, int d, int V, int dtype, bool kl = false) {
  Layout L{};
  const size_t P = static_cast<size_t>(S) * T;
  L.rows_cap = static_cast<long long>((P + kTileRows - 1) / kTileRows) * kTileRows;
  L.max_tiles = static_cast<int>(L.rows_cap / kTileRows);
  const int nvt = (V + kTileN - 1) / kTileN;
  L.num_strips = (nvt + kFwdTilesPerStrip - 1) / kFwdTilesPerStrip;
  L.v_round = nvt * kTileN;
  const bool bf16 = dtype == GRPO_BF16;
  size_t off = sizeof(WsHeader);
  L.seq_base = off;       off = align256(off + sizeof(int32_t) * (S + 1));
  L.row_pos = off;        off = align256(off + sizeof(int32_t) * L.rows_cap);
  L.pos_row = off;        off = align256(off + sizeof(int32_t) * P);
  L.counts = off;         off = align256(off + sizeof(int32_t) * S);
  L.zy = off;             off = align256(off + sizeof(float) * P);
  L.partials = off;
  if (bf16) off = align256(off + sizeof(float4) * L.num_strips * L.rows_cap);
  L.partials2 = off;      // exact-KL forward only
  if (bf16 && kl) off = align256(off + sizeof(float4) * L.num_strips * L.rows_cap);
  L.g = off;              off = align256(off + sizeof(float) * P);
  L.cvec = off;           off = align256(off + sizeof(float) * P);
  L.seq_loss = off;       off = align256(off + sizeof(float) * S);
  L.hp = off;             // packed hidden states (bf16 path)
  if (bf16) off = align256(off + static_cast<size_t>(L.rows_cap) * d * 2);
  L.hrp = off;            // packed reference hidden states (exact-KL path)
  if (bf16 && kl) off = align256(off + static_cast<size_t>(L.rows_cap) * d * 2);
  L.fixed_end = off;
  return L;
}

// Bytes of the chunk-dependent regions (f32 dH accumulator when chunked + bf16 dz scratch).
size_t chunk_bytes(const Layout& L, int d, int vc) {
  const size_t dz = align256(static_cast<size_t>(L.rows_cap) * vc * 2);
  if (vc >= L.v_round) return dz;
  return align256(static_cast<size_t>(L.rows_cap) * d * 4) + dz;
}

bool shape_ok(int S, int T, int d, int V) {
  return S > 0 && T > 0 && d > 0 && V > 0 &&
         static_cast<long long>(S) * T < (1ll << 31) && V < (1 << 30);
}

int check_dtype_shape(int dtype, int d) {
  if (dtype == GRPO_BF16) return (d % 64 == 0) ? GRPO_OK : GRPO_ERR_UNSUPPORTED;
  if (dtype == GRPO_F32) return (d <= 4096) ? GRPO_OK : GRPO_ERR_UNSUPPORTED;
  return GRPO_ERR_INVALID_ARG;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// ------------------------------------------------------------------------------------------
// TMA descriptors (driver entry point fetched through the runtime, no -lcuda needed)
// ------------------------------------------------------------------------------------------
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

#ifndef GRPO_TMA_L2_PROMOTION
#define GRPO_TMA_L2_PROMOTION CU_TENSOR_MAP_L2_PROMOTION_L2_256B
#endif

// 2-D bf16 tensor [outer, inner] (inner contiguous, row pitch `pitch_elems`), box
// [box_outer, 64], 128-byte swizzle, out-of-range elements read as zero.
bool make_map(CUtensorMap* map, const void* base, uint64_t inner, uint64_t outer,
              uint64_t pitch_elems, uint32_t box_outer) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {pitch_elems * 2};
  cuuint32_t box[2] = {64, box_outer};
  cuuint32_t es[2] = {1, 1};
  const CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims,
                        strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, GRPO_TMA_L2_PROMOTION,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}


struct Views {
  WsHeader* hdr;
  int32_t* seq_base;
  int32_t* row_pos;
  int32_t* pos_row;
  int32_t* counts;
  float* zy;
  float4* partials;
  float4* partials2;
  float* g;
  float* cvec;
  float* seq_loss;
  void* hp;
  void* hrp;
};

Views views(void* ws, const Layout& L) {
  char* b = static_cast<char*>(ws);
  Views v;
  v.hdr = reinterpret_cast<WsHeader*>(b);
  v.seq_base = reinterpret_cast<int32_t*>(b + L.seq_base);
  v.row_pos = reinterpret_cast<int32_t*>(b + L.row_pos);
  v.pos_row = reinterpret_cast<int32_t*>(b + L.pos_row);
  v.counts = reinterpret_cast<int32_t*>(b + L.counts);
  v.zy = reinterpret_cast<float*>(b + L.zy);
  v.partials = reinterpret_cast<float4*>(b + L.partials);
  v.partials2 = reinterpret_cast<float4*>(b + L.partials2);
  v.g = reinterpret_cast<float*>(b + L.g);
  v.cvec = reinterpret_cast<float*>(b + L.cvec);
  v.seq_loss = reinterpret_cast<float*>(b + L.seq_loss);
  v.hp = b + L.hp;
  v.hrp = b + L.hrp;
  return v;
}

// Packs the scored tokens: counts from the mask, packed-row maps, and H gathered into Hp.
int pack_tokens(const uint8_t* mask, int S, int T, int d, const void* H, const Layout& L,
                const Views& v, int32_t* counts_out, cudaStream_t st);

GemmArgs base_args(const Layout& L, const Views& v, int S, int T, int d, int V,
                   const int32_t* tokens, const uint8_t* mask) {
  GemmArgs a;
  std::memset(&a, 0, sizeof(a));
  a.S = S;
  a.T = T;
  a.d = d;
  a.V = V;
  a.row_pos = v.row_pos;
  a.hdr = v.hdr;
  a.tokens = tokens;
  a.mask = mask;
  a.rows_cap = L.rows_cap;
  a.num_strips = L.num_strips;
  a.inject_stall = g_inject_stall.load();
  gemm_window_config(a);
  return a;
}

int pack_tokens(const uint8_t* mask, int S, int T, int d, const void* H, const Layout& L,
                const Views& v, int32_t* counts_out, cudaStream_t st) {
  GRPO_TRY(counted(GRPO_K_MASK_SCAN, st,
                   [&] { return launch_mask_scan(mask, S, T, counts_out, st); }));
  GRPO_TRY(counted(GRPO_K_PACK, st, [&] {
    return launch_pack(mask, counts_out, S, T, L.rows_cap, v.seq_base, v.row_pos, v.pos_row,
                       v.hdr, st);
  }));
  if (!H) return GRPO_OK;
  return counted(GRPO_K_GATHER, st, [&] {
    return launch_gather_rows(H, d, v.row_pos, v.hdr, L.rows_cap, v.hp, st);
  });
}

}  // namespace

// ==========================================================================================
// C ABI
// ==========================================================================================
extern "C" {

const char* grpo_status_string(int status) {
  switch (status) {
    case GRPO_OK: return "ok";
    case GRPO_ERR_INVALID_ARG: return "invalid argument";
    case GRPO_ERR_UNSUPPORTED: return "unsupported shape or dtype";
    case GRPO_ERR_CUDA: return "CUDA runtime or launch error";
    case GRPO_ERR_WORKSPACE: return "workspace too small or misaligned";
    case GRPO_ERR_TOKEN_RANGE: return "token id outside [0, V) at a scored position";
    case GRPO_ERR_TIMEOUT: return "a bounded wait inside a kernel ran out";
    case GRPO_ERR_GROUPS: return "group offsets do not rise from 0 to S";
    default: return "unknown status";
  }
}

const char* grpo_kernel_name(int32_t kernel_id) {
  if (kernel_id < 0 || kernel_id >= GRPO_K_COUNT) return "unknown";
  return kKernelNames[kernel_id];
}

}  // extern "C"

namespace {
size_t workspace_bytes(int32_t S, int32_t T, int32_t d, int32_t V, int32_t dtype,
                       int32_t vocab_chunk, bool kl) {
  if (!shape_ok(S, T, d, V) || check_dtype_shape(dtype, d) == GRPO_ERR_INVALID_ARG) return 0;
  if (kl && dtype != GRPO_BF16) return 0;
  const Layout L = make_layout(S, T, d, V, dtype, kl);
  if (dtype != GRPO_BF16) return L.fixed_end;
  int vc = L.v_round;
  if (vocab_chunk > 0) {
    vc = ((vocab_chunk + kTileN - 1) / kTileN) * kTileN;
    if (vc > L.v_round) vc = L.v_round;
  }
  return L.fixed_end + chunk_bytes(L, d, vc);
}
}  // namespace

extern "C" {

size_t grpo_workspace_bytes(int32_t S, int32_t T, int32_t d, int32_t V, int32_t dtype,
                            int32_t vocab_chunk) {
  return workspace_bytes(S, T, d, V, dtype, vocab_chunk, false);
}

size_t grpo_workspace_bytes_kl(int32_t S, int32_t T, int32_t d, int32_t V, int32_t dtype,
                               int32_t vocab_chunk) {
  return workspace_bytes(S, T, d, V, dtype, vocab_chunk, true);
}

int grpo_workspace_init(void* workspace, size_t workspace_bytes, grpo_stream_t stream) {
  if (!workspace || workspace_bytes < sizeof(WsHeader)) return GRPO_ERR_WORKSPACE;
  if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0) return GRPO_ERR_WORKSPACE;
  return cudaMemsetAsync(workspace, 0, sizeof(WsHeader), reinterpret_cast<cudaStream_t>(stream)) ==
                 cudaSuccess
             ? GRPO_OK
             : GRPO_ERR_CUDA;
}

int group_advantages(const float* rewards, const int32_t* group_offsets, int32_t num_groups,
                     int32_t num_seqs, int32_t std_mode, float std_eps, float* adv_out,
                     void* workspace, size_t workspace_bytes, grpo_stream_t stream) {
  if (!rewards || !group_offsets || !adv_out) return GRPO_ERR_INVALID_ARG;
  if (num_groups <= 0 || num_seqs <= 0) return GRPO_ERR_INVALID_ARG;
  if (std_mode != GRPO_STD_UNBIASED && std_mode != GRPO_STD_POPULATION) return GRPO_ERR_INVALID_ARG;
  if (!(std_eps >= 0.f)) return GRPO_ERR_INVALID_ARG;
  if (!workspace || workspace_bytes < sizeof(WsHeader) ||
      (reinterpret_cast<uintptr_t>(workspace) & 255u) != 0)
    return GRPO_ERR_WORKSPACE;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  WsHeader* hdr = static_cast<WsHeader*>(workspace);
  return counted(GRPO_K_GROUP_ADV, st, [&] {
    return launch_group_adv(rewards, group_offsets, num_groups, num_seqs, std_mode, std_eps,
                            adv_out, hdr, st);
  });
}

int grpo_score_fwd(const void* H, const void* W, int32_t dtype, const int32_t* tokens,
                   const uint8_t* mask, int32_t S, int32_t T, int32_t d, int32_t V, float* logp,
                   float* lse, float* entropy, int32_t* argmax, int32_t* valid_count,
                   void* workspace, size_t workspace_bytes, grpo_stream_t stream) {
  if (!H || !W || !tokens || !mask || !logp || !lse || !entropy || !argmax || !valid_count)
    return GRPO_ERR_INVALID_ARG;
  if (!shape_ok(S, T, d, V)) return GRPO_ERR_INVALID_ARG;
  GRPO_TRY(check_dtype_shape(dtype, d));
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255u) != 0) return GRPO_ERR_WORKSPACE;
  const Layout L = make_layout(S, T, d, V, dtype);
  if (workspace_bytes < L.fixed_end) return GRPO_ERR_WORKSPACE;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const Views v = views(workspace, L);

  if (dtype == GRPO_F32) {
    GRPO_TRY(counted(GRPO_K_MASK_SCAN, st,
                     [&] { return launch_mask_scan(mask, S, T, valid_count, st); }));
    return counted(GRPO_K_F32_FWD, st, [&] {
      return launch_f32_fwd(static_cast<const float*>(H), static_cast<const float*>(W), tokens,
                            mask, S, T, d, V, logp, lse, entropy, argmax, v.hdr, st);
    });
  }
  if (!aligned16(H) || !aligned16(W)) return GRPO_ERR_INVALID_ARG;
  GRPO_TRY(pack_tokens(mask, S, T, d, H, L, v, valid_count, st));
  const int tm = gemm_role_tile_mode(ROLE_FWD);
  CUtensorMap mapH, mapW;
  if (!make_map(&mapH, v.hp, d, L.rows_cap, d, kTileRows) ||
      !make_map(&mapW, W, d, V, d, gemm_b_box_rows(tm)))
    return GRPO_ERR_CUDA;
  GemmArgs a = base_args(L, v, S, T, d, V, tokens, mask);
  a.partials = v.partials;
  a.zy = v.zy;
  const int grid = gemm_grid(L.max_tiles, L.num_strips, tm);
  GRPO_TRY(counted(GRPO_K_FWD_GEMM, st,
                   [&] { return launch_gemm(ROLE_FWD, mapH, mapW, a, grid, tm, st); }));
  return counted(GRPO_K_FWD_MERGE, st, [&] {
    return launch_fwd_merge(v.partials, L.rows_cap, L.num_strips, v.zy, v.pos_row, tokens,
                            mask, S, T, V, logp, lse, entropy, argmax, v.hdr, st);
  });
}

}  // extern "C"

namespace {

// Shared by grpo_loss_bwd (mode 0) and grpo_sft_loss_bwd (mode 1): the per-token loss kernel
// differs, the recompute + dz + dH + dW GEMMs are the same.
int loss_bwd_impl(int mode, const void* H, const void* W, int32_t dtype, const int32_t* tokens,
                  const uint8_t* mask, int32_t S, int32_t T, int32_t d, int32_t V,
                  const float* logp, const float* lse, const float* old_logp,
                  const float* ref_logp, const float* adv, const int32_t* valid_count,
                  float eps_low, float eps_high, float beta, int32_t agg, double norm,
                  float* loss_out, void* dH, float* dW, void* workspace, size_t workspace_bytes,
                  grpo_stream_t stream, int32_t v_offset = 0, bool dh_f32 = false,
                  const void* H_ref = nullptr, const void* W_ref = nullptr,
                  const float* lse_ref = nullptr, const float* kl = nullptr) {
  if (!H || !W || !tokens || !mask || !logp || !lse || !valid_count || !loss_out || !dH || !dW)
    return GRPO_ERR_INVALID_ARG;
  if (mode != 1 && (!old_logp || !adv)) return GRPO_ERR_INVALID_ARG;
  if (mode == 0 && !ref_logp && beta != 0.f) return GRPO_ERR_INVALID_ARG;
  if (mode == 1) {   // the distillation loss reads none of these
    old_logp = logp;
    ref_logp = logp;
    adv = logp;
    beta = 0.f;
  }
  if (mode == 2) {   // exact KL: the reference model's hidden states and head replace ref_logp
    if (!H_ref || !W_ref || !lse_ref || !kl) return GRPO_ERR_INVALID_ARG;
    if (dtype != GRPO_BF16) return GRPO_ERR_UNSUPPORTED;
    if (!aligned16(H_ref) || !aligned16(W_ref)) return GRPO_ERR_INVALID_ARG;
    ref_logp = logp;
  }
  if (!shape_ok(S, T, d, V)) return GRPO_ERR_INVALID_ARG;
  GRPO_TRY(check_dtype_shape(dtype, d));
  if (agg != GRPO_AGG_SEQ_MEAN && agg != GRPO_AGG_TOKEN_MEAN) return GRPO_ERR_INVALID_ARG;
  if (!(eps_low >= 0.f) || !(eps_high >= 0.f) || !(beta >= 0.f) || !(norm >= 0.0))
    return GRPO_ERR_INVALID_ARG;
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255u) != 0) return GRPO_ERR_WORKSPACE;
  const Layout L = make_layout(S, T, d, V, dtype, mode == 2);
  if (workspace_bytes < L.fixed_end) return GRPO_ERR_WORKSPACE;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const Views v = views(workspace, L);
  // ref_logp is not read when beta == 0; pass a valid pointer anyway.
  const float* ref = ref_logp ? ref_logp : logp;

  // counts from the mask and the packed-row maps (also Sum n for token_mean); H is gathered
  // below, on the tensor-core path only
  GRPO_TRY(pack_tokens(mask, S, T, d, nullptr, L, v, v.counts, st));
  GRPO_TRY(counted(GRPO_K_LOSS_TOKENS, st, [&] {
    return launch_loss_tokens(mask, logp, old_logp, ref, adv, valid_count, S, T, eps_low,
                              eps_high, beta, agg, norm, mode, v.hdr, v.g, v.seq_loss, st, kl,
                              v.cvec);
  }));
  GRPO_TRY(counted(GRPO_K_LOSS_FINAL, st, [&] {
    return launch_loss_final(v.seq_loss, S, agg, norm, v.hdr, loss_out, st);
  }));

  if (dtype == GRPO_F32) {
    GRPO_TRY(counted(GRPO_K_F32_DH, st, [&] {
      return launch_f32_dh(static_cast<const float*>(H), static_cast<const float*>(W), tokens,
                           mask, lse, v.g, S, T, d, V, static_cast<float*>(dH), st);
    }));
    return counted(GRPO_K_F32_DW, st, [&] {
      return launch_f32_dw(static_cast<const float*>(H), static_cast<const float*>(W), tokens,
                           mask, lse, v.g, S, T, d, V, dW, st);
    });
  }

  if (!aligned16(H) || !aligned16(W) || !aligned16(dH) || !aligned16(dW))
    return GRPO_ERR_INVALID_ARG;
  // Vocabulary chunk: the whole vocabulary if the workspace holds it, else the largest
  // multiple of 256 that fits next to the f32 dH accumulator.
  const size_t avail = workspace_bytes - L.fixed_end;
  int vc;
  if (avail >= chunk_bytes(L, d, L.v_round)) {
    vc = L.v_round;
  } else {
    const size_t acc = align256(static_cast<size_t>(L.rows_cap) * d * 4);
    if (avail < acc) return GRPO_ERR_WORKSPACE;
    const size_t per_col = static_cast<size_t>(L.rows_cap) * 2;
    long long cols = static_cast<long long>((avail - acc - 256) / per_col);
    vc = static_cast<int>((cols / kTileN) * kTileN);
    if (vc < kTileN) return GRPO_ERR_WORKSPACE;
  }
  const int nchunks = (V + vc - 1) / vc;
  char* wsb = static_cast<char*>(workspace);
  float* dH_acc = nullptr;
  __nv_bfloat16* dz;
  if (nchunks == 1) {
    dz = reinterpret_cast<__nv_bfloat16*>(wsb + L.fixed_end);
  } else {
    dH_acc = reinterpret_cast<float*>(wsb + L.fixed_end);
    dz = reinterpret_cast<__nv_bfloat16*>(wsb + L.fixed_end +
                                          align256(static_cast<size_t>(L.rows_cap) * d * 4));
  }
  GRPO_TRY(counted(GRPO_K_GATHER, st, [&] {
    return launch_gather_rows(H, d, v.row_pos, v.hdr, L.rows_cap, v.hp, st);
  }));
  if (mode == 2) {
    GRPO_TRY(counted(GRPO_K_GATHER, st, [&] {
      return launch_gather_rows(H_ref, d, v.row_pos, v.hdr, L.rows_cap, v.hrp, st);
    }));
  }
  // exact-KL roles: single-CTA tiles
  const int tm = mode == 2 ? 0 : gemm_role_tile_mode(ROLE_DZ);
  const int tm_dh = gemm_role_tile_mode(ROLE_DH), tm_dw = gemm_role_tile_mode(ROLE_DW);
  CUtensorMap mapHk, mapWk, mapDzK, mapWmn, mapDzMn, mapHmn, mapHrk, mapWrk, mapDzSt;
  if (mode == 2 && (!make_map(&mapHrk, v.hrp, d, L.rows_cap, d, kTileRows) ||
                    !make_map(&mapWrk, W_ref, d, V, d, kTileN)))
    return GRPO_ERR_CUDA;
  if (!make_map(&mapHk, v.hp, d, L.rows_cap, d, kTileRows) ||
      !make_map(&mapWk, W, d, V, d, gemm_b_box_rows(tm)) ||
      !make_map(&mapDzK, dz, vc, L.rows_cap, vc, kTileRows) ||
      !make_map(&mapWmn, W, d, V, d, 64) || !make_map(&mapDzMn, dz, vc, L.rows_cap, vc, 64) ||
      !make_map(&mapHmn, v.hp, d, L.rows_cap, d, 64) ||
      // single-CTA dz tiles store 32-row x 64-column boxes of dz through this map
      !make_map(&mapDzSt, dz, vc, L.rows_cap, vc, 32))
    return GRPO_ERR_CUDA;

  GemmArgs a = base_args(L, v, S, T, d, V, tokens, mask);
  a.v_offset = v_offset;
  a.dh_f32 = dh_f32 ? 1 : 0;
  a.g = v.g;
  a.lse = lse;
  a.c = v.cvec;
  a.lse_ref = lse_ref;
  a.kl = kl;
  a.dz = dz;
  a.dz_pitch = vc;
  a.dH = static_cast<__nv_bfloat16*>(dH);
  a.dH_acc = dH_acc;
  a.dW = dW;
  const long long dtiles = (d + kTileN - 1) / kTileN;   // output column tiles of dH and dW
  for (int c = 0; c < nchunks; ++c) {
    a.vc0 = c * vc;
    a.vc_len = (V - a.vc0) < vc ? (V - a.vc0) : vc;
    a.dh_mode = nchunks == 1 ? 0 : (c == 0 ? 1 : (c == nchunks - 1 ? 3 : 2));
    const long long vt = (a.vc_len + kTileN - 1) / kTileN;
    GRPO_TRY(counted(GRPO_K_BWD_DZ_GEMM, st, [&] {
      if (mode == 2)
        return launch_gemm(ROLE_DZ_KL, mapHk, mapWk, a, gemm_grid(L.max_tiles, vt, 0), 0, st,
                           &mapHrk, &mapWrk);
      return launch_gemm(ROLE_DZ, mapHk, mapWk, a, gemm_grid(L.max_tiles, vt, tm), tm, st,
                         &mapDzSt);
    }));
    GRPO_TRY(counted(GRPO_K_BWD_DH_GEMM, st, [&] {
      return launch_gemm(ROLE_DH, mapDzK, mapWmn, a, gemm_grid(L.max_tiles, dtiles, tm_dh),
                         tm_dh, st);
    }));
    const long long vm = (a.vc_len + kTileRows - 1) / kTileRows;
    GRPO_TRY(counted(GRPO_K_BWD_DW_GEMM, st, [&] {
      return launch_gemm(ROLE_DW, mapDzMn, mapHmn, a, gemm_grid(vm, dtiles, tm_dw), tm_dw,
                         st);
    }));
  }
  return counted(GRPO_K_DH_ZERO, st, [&] {
    return launch_dh_zero_masked(mask, S, T, d, dH, dh_f32 ? 4 : 2, st);
  });
}

}  // namespace

extern "C" {

int grpo_loss_bwd(const void* H, const void* W, int32_t dtype, const int32_t* tokens,
                  const uint8_t* mask, int32_t S, int32_t T, int32_t d, int32_t V,
                  const float* logp, const float* lse, const float* old_logp,
                  const float* ref_logp, const float* adv, const int32_t* valid_count,
                  float eps_low, float eps_high, float beta, int32_t agg, double norm,
                  float* loss_out, void* dH, float* dW, void* workspace, size_t workspace_bytes,
                  grpo_stream_t stream) {
  return loss_bwd_impl(0, H, W, dtype, tokens, mask, S, T, d, V, logp, lse, old_logp, ref_logp,
                       adv, valid_count, eps_low, eps_high, beta, agg, norm, loss_out, dH, dW,
                       workspace, workspace_bytes, stream);
}

int grpo_sft_loss_bwd(const void* H, const void* W, int32_t dtype, const int32_t* tokens,
                      const uint8_t* mask, int32_t S, int32_t T, int32_t d, int32_t V,
                      const float* logp, const float* lse, const int32_t* valid_count,
                      int32_t agg, double norm, float* loss_out, void* dH, float* dW,
                      void* workspace, size_t workspace_bytes, grpo_stream_t stream) {
  return loss_bwd_impl(1, H, W, dtype, tokens, mask, S, T, d, V, logp, lse, nullptr, nullptr,
                       nullptr, valid_count, 0.f, 0.f, 0.f, agg, norm, loss_out, dH, dW, workspace,
                       workspace_bytes, stream);
}

int grpo_score_fwd_kl(const void* H, const void* W, const void* H_ref, const void* W_ref,
                      int32_t dtype, const int32_t* tokens, const uint8_t* mask, int32_t S,
                      int32_t T, int32_t d, int32_t V, float* logp, float* lse, float* entropy,
                      int32_t* argmax, int32_t* valid_count, float* lse_ref, float* kl,
                      void* workspace, size_t workspace_bytes, grpo_stream_t stream) {
  if (!H || !W || !H_ref || !W_ref || !tokens || !mask || !logp || !lse || !entropy || !argmax ||
      !valid_count || !lse_ref || !kl)
    return GRPO_ERR_INVALID_ARG;
  if (!shape_ok(S, T, d, V)) return GRPO_ERR_INVALID_ARG;
  if (dtype != GRPO_BF16) return GRPO_ERR_UNSUPPORTED;
  GRPO_TRY(check_dtype_shape(dtype, d));
  if (!aligned16(H) || !aligned16(W) || !aligned16(H_ref) || !aligned16(W_ref))
    return GRPO_ERR_INVALID_ARG;
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255u) != 0) return GRPO_ERR_WORKSPACE;
  const Layout L = make_layout(S, T, d, V, dtype, true);
  if (workspace_bytes < L.fixed_end) return GRPO_ERR_WORKSPACE;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const Views v = views(workspace, L);
  GRPO_TRY(pack_tokens(mask, S, T, d, H, L, v, valid_count, st));
  GRPO_TRY(counted(GRPO_K_GATHER, st, [&] {
    return launch_gather_rows(H_ref, d, v.row_pos, v.hdr, L.rows_cap, v.hrp, st);
  }));
  CUtensorMap mapH, mapW, mapHr, mapWr;
  if (!make_map(&mapH, v.hp, d, L.rows_cap, d, kTileRows) ||
      !make_map(&mapW, W, d, V, d, kTileN) ||
      !make_map(&mapHr, v.hrp, d, L.rows_cap, d, kTileRows) ||
      !make_map(&mapWr, W_ref, d, V, d, kTileN))
    return GRPO_ERR_CUDA;
  GemmArgs a = base_args(L, v, S, T, d, V, tokens, mask);
  a.partials = v.partials;
  a.partials2 = v.partials2;
  a.zy = v.zy;
  GRPO_TRY(counted(GRPO_K_FWD_GEMM, st, [&] {
    return launch_gemm(ROLE_FWD_KL, mapH, mapW, a, gemm_grid(L.max_tiles, L.num_strips, 0),
                       false, st, &mapHr, &mapWr);
  }));
  return counted(GRPO_K_FWD_MERGE, st, [&] {
    return launch_fwd_merge_kl(v.partials, v.partials2, L.rows_cap, L.num_strips, v.zy,
                               v.pos_row, tokens, mask, S, T, V, logp, lse, entropy, argmax,
                               lse_ref, kl, v.hdr, st);
  });
}

int grpo_loss_bwd_kl(const void* H, const void* W, const void* H_ref, const void* W_ref,
                     int32_t dtype, const int32_t* tokens, const uint8_t* mask, int32_t S,
                     int32_t T, int32_t d, int32_t V, const float* logp, const float* lse,
                     const float* lse_ref, const float* kl, const float* old_logp,
                     const float* adv, const int32_t* valid_count, float eps_low, float eps_high,
                     float beta, int32_t agg, double norm, float* loss_out, void* dH, float* dW,
                     void* workspace, size_t workspace_bytes, grpo_stream_t stream) {
  return loss_bwd_impl(2, H, W, dtype, tokens, mask, S, T, d, V, logp, lse, old_logp, logp, adv,
                       valid_count, eps_low, eps_high, beta, agg, norm, loss_out, dH, dW,
                       workspace, workspace_bytes, stream, 0, false, H_ref, W_ref, lse_ref, kl);
}

int grpo_score_fwd_shard(const void* H, const void* W_shard, int32_t dtype,
                         const int32_t* tokens, const uint8_t* mask, int32_t S, int32_t T,
                         int32_t d, int32_t V_shard, int32_t v_offset, int32_t V_total,
                         float* stats, float* zy, void* workspace, size_t workspace_bytes,
                         grpo_stream_t stream) {
  if (!H || !W_shard || !tokens || !mask || !stats || !zy) return GRPO_ERR_INVALID_ARG;
  if (!shape_ok(S, T, d, V_shard) || v_offset < 0 || V_total <= 0 ||
      static_cast<long long>(v_offset) + V_shard > V_total)
    return GRPO_ERR_INVALID_ARG;
  if (dtype != GRPO_BF16) return GRPO_ERR_UNSUPPORTED;
  GRPO_TRY(check_dtype_shape(dtype, d));
  if (!aligned16(H) || !aligned16(W_shard) || !aligned16(stats)) return GRPO_ERR_INVALID_ARG;
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255u) != 0) return GRPO_ERR_WORKSPACE;
  const Layout L = make_layout(S, T, d, V_shard, dtype);
  if (workspace_bytes < L.fixed_end) return GRPO_ERR_WORKSPACE;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const Views v = views(workspace, L);
  GRPO_TRY(pack_tokens(mask, S, T, d, H, L, v, v.counts, st));
  const int tm = gemm_role_tile_mode(ROLE_FWD);
  CUtensorMap mapH, mapW;
  if (!make_map(&mapH, v.hp, d, L.rows_cap, d, kTileRows) ||
      !make_map(&mapW, W_shard, d, V_shard, d, gemm_b_box_rows(tm)))
    return GRPO_ERR_CUDA;
  GemmArgs a = base_args(L, v, S, T, d, V_shard, tokens, mask);
  a.v_offset = v_offset;
  a.partials = v.partials;
  a.zy = v.zy;
  GRPO_TRY(counted(GRPO_K_FWD_GEMM, st, [&] {
    return launch_gemm(ROLE_FWD, mapH, mapW, a, gemm_grid(L.max_tiles, L.num_strips, tm), tm, st);
  }));
  return counted(GRPO_K_SHARD_STATS, st, [&] {
    return launch_shard_stats(v.partials, L.rows_cap, L.num_strips, v.zy, v.pos_row, tokens,
                              mask, S, T, V_shard, v_offset, reinterpret_cast<float4*>(stats), zy,
                              st);
  });
}

int grpo_merge_shard_stats(const float* stats, const float* zy, int32_t num_shards,
                           const int32_t* tokens, const uint8_t* mask, int32_t S, int32_t T,
                           int32_t V_total, float* logp, float* lse, float* entropy,
                           int32_t* argmax, int32_t* valid_count, void* workspace,
                           size_t workspace_bytes, grpo_stream_t stream) {
  if (!stats || !zy || !tokens || !mask || !logp || !lse || !entropy || !argmax || !valid_count)
    return GRPO_ERR_INVALID_ARG;
  if (num_shards <= 0 || S <= 0 || T <= 0 || V_total <= 0 ||
      static_cast<long long>(S) * T >= (1ll << 31))
    return GRPO_ERR_INVALID_ARG;
  if (!aligned16(stats)) return GRPO_ERR_INVALID_ARG;
  if (!workspace || workspace_bytes < sizeof(WsHeader) ||
      (reinterpret_cast<uintptr_t>(workspace) & 255u) != 0)
    return GRPO_ERR_WORKSPACE;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  WsHeader* hdr = static_cast<WsHeader*>(workspace);
  GRPO_TRY(counted(GRPO_K_MASK_SCAN, st,
                   [&] { return launch_mask_scan(mask, S, T, valid_count, st); }));
  return counted(GRPO_K_MERGE_SHARDS, st, [&] {
    return launch_merge_shards(reinterpret_cast<const float4*>(stats), zy, num_shards, tokens,
                               mask, S, T, V_total, logp, lse, entropy, argmax, hdr, st);
  });
}

int grpo_loss_bwd_shard(const void* H, const void* W_shard, int32_t dtype,
                        const int32_t* tokens, const uint8_t* mask, int32_t S, int32_t T,
                        int32_t d, int32_t V_shard, int32_t v_offset, int32_t V_total,
                        const float* logp, const float* lse, const float* old_logp,
                        const float* ref_logp, const float* adv, const int32_t* valid_count,
                        float eps_low, float eps_high, float beta, int32_t agg, double norm,
                        float* loss_out, float* dH_partial, float* dW_shard, void* workspace,
                        size_t workspace_bytes, grpo_stream_t stream) {
  if (v_offset < 0 || V_total <= 0 || V_shard <= 0 ||
      static_cast<long long>(v_offset) + V_shard > V_total)
    return GRPO_ERR_INVALID_ARG;
  if (dtype != GRPO_BF16) return GRPO_ERR_UNSUPPORTED;
  return loss_bwd_impl(0, H, W_shard, dtype, tokens, mask, S, T, d, V_shard, logp, lse, old_logp,
                       ref_logp, adv, valid_count, eps_low, eps_high, beta, agg, norm, loss_out,
                       dH_partial, dW_shard, workspace, workspace_bytes, stream, v_offset, true);
}

int grpo_rewards(const uint8_t* correct, const float* t_base, const float* t_new,
                 const int32_t* tools_used, const int32_t* tools_avail, int32_t n,
                 float lambda_tools, float* r_out, grpo_stream_t stream) {
  if (!correct || !t_base || !t_new || !tools_used || !tools_avail || !r_out || n <= 0)
    return GRPO_ERR_INVALID_ARG;
  if (!(lambda_tools >= 0.f)) return GRPO_ERR_INVALID_ARG;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  return counted(GRPO_K_REWARDS, st, [&] {
    return launch_rewards(correct, t_base, t_new, tools_used, tools_avail, n, lambda_tools,
                          r_out, st);
  });
}

int grpo_last_device_error(void* workspace, int32_t* where_out, grpo_stream_t stream) {
  if (!workspace) return GRPO_ERR_WORKSPACE;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  int32_t word[2] = {0, 0};
  if (cudaMemcpyAsync(word, workspace, sizeof(word), cudaMemcpyDeviceToHost, st) != cudaSuccess)
    return GRPO_ERR_CUDA;
  if (cudaStreamSynchronize(st) != cudaSuccess) return GRPO_ERR_CUDA;
  if (cudaMemsetAsync(workspace, 0, sizeof(word), st) != cudaSuccess) return GRPO_ERR_CUDA;
  if (cudaStreamSynchronize(st) != cudaSuccess) return GRPO_ERR_CUDA;
  if (where_out) *where_out = word[1];
  return word[0];
}

int grpo_timing_enable(int32_t enable) {
  g_timing.store(enable ? 1 : 0);
  return GRPO_OK;
}

int grpo_timing_reset(void) {
  std::lock_guard<std::mutex> lk(g_mu);
  for (int k = 0; k < GRPO_K_COUNT; ++k) {
    for (auto& p : g_pending[k]) g_free_events.push_back(p);
    g_pending[k].clear();
    g_total_ms[k] = 0.0;
    g_launches[k].store(0);
  }
  return GRPO_OK;
}

int grpo_timing_read(int32_t kernel_id, int64_t* launches, double* total_ms) {
  if (kernel_id < 0 || kernel_id >= GRPO_K_COUNT) return GRPO_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> lk(g_mu);
  for (auto& p : g_pending[kernel_id]) {
    if (cudaEventSynchronize(p.b) != cudaSuccess) return GRPO_ERR_CUDA;
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, p.a, p.b) != cudaSuccess) return GRPO_ERR_CUDA;
    g_total_ms[kernel_id] += ms;
    g_free_events.push_back(p);
  }
  g_pending[kernel_id].clear();
  if (launches) *launches = g_launches[kernel_id].load();
  if (total_ms) *total_ms = g_total_ms[kernel_id];
  return GRPO_OK;
}

/* Test hook, not part of the documented ABI: while set, the first CTA of every tensor-core
 * GEMM leaves its first pipeline stage unfilled, so its MMA warp's bounded wait runs out and the
 * kernel records GRPO_ERR_TIMEOUT and exits. */
int grpo_debug_inject_stall(int32_t on) {
  g_inject_stall.store(on ? 1 : 0);
  return GRPO_OK;
}

int grpo_set_tile_mode(int32_t mode) {
  if (mode < GRPO_TILE_DEFAULT || mode > GRPO_TILE_CTA_PAIR_WIDE) return GRPO_ERR_INVALID_ARG;
  for (int r = GRPO_ROLE_FWD; r <= GRPO_ROLE_DW; ++r)
    g_role_mode[r].store(mode == GRPO_TILE_DEFAULT ? kRoleDefault[r] : mode);
  return GRPO_OK;
}

int grpo_set_cta_pair(int32_t on) {
  return grpo_set_tile_mode(on ? GRPO_TILE_CTA_PAIR : GRPO_TILE_SINGLE);
}

int grpo_get_tile_mode(void) {
  const int m = g_role_mode[GRPO_ROLE_FWD].load();
  for (int r = GRPO_ROLE_DZ; r <= GRPO_ROLE_DW; ++r)
    if (g_role_mode[r].load() != m) return GRPO_TILE_DEFAULT;   // roles differ
  return m;
}

int grpo_set_role_tile_mode(int32_t role, int32_t mode) {
  if (role < GRPO_ROLE_FWD || role > GRPO_ROLE_DW) return GRPO_ERR_INVALID_ARG;
  if (mode < GRPO_TILE_DEFAULT || mode > GRPO_TILE_CTA_PAIR_WIDE) return GRPO_ERR_INVALID_ARG;
  g_role_mode[role].store(mode == GRPO_TILE_DEFAULT ? kRoleDefault[role] : mode);
  return GRPO_OK;
}

int grpo_get_role_tile_mode(int32_t role) {
  if (role < GRPO_ROLE_FWD || role > GRPO_ROLE_DW) return GRPO_ERR_INVALID_ARG;
  return gemm_role_tile_mode(role);
}

int grpo_set_gemm_window(int32_t check_kblocks, int32_t lag) {
  if (lag < 0 || (check_kblocks != 0 && lag == 0)) return GRPO_ERR_INVALID_ARG;
  g_win_check.store(check_kblocks);
  g_win_lag.store(check_kblocks != 0 ? lag : 0);
  return GRPO_OK;
}

}  // extern "C"

namespace grpo {
void gemm_window_config(GemmArgs& a) {
  a.win_check = g_win_check.load();
  a.win_lag = g_win_lag.load();
}

int gemm_role_tile_mode(int role) {
  // the exact-KL roles always run single-CTA tiles
  return (role >= ROLE_FWD && role <= ROLE_DW) ? g_role_mode[role].load() : GRPO_TILE_SINGLE;
}
}  // namespace grpo
