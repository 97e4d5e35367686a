// grpo_score_fwd_static: the forward scoring pass with its scratch in a fixed, library-owned
// device array instead of a caller-provided workspace, for callers that cannot allocate device
// memory at all -- for example a plugin whose host framework owns every device allocation and
// forbids extensions from making their own, or a latency-critical section where an allocation
// (which can synchronise the device) is not allowed. The caller still provides every input and
// output buffer.
//
// The scratch is one file-scope __device__ array of kStaticScratchBytes (64 MiB). Every GPU on
// which this library is loaded keeps that array until the process exits. In host code the
// array's name is only a host-side stand-in, so its device address is looked up with
// cudaGetSymbolAddress, with the device current, on the first call made on that device, and
// cached. A call made while its stream is not being captured looks the address up again (cheap,
// allocates nothing), so a context torn down and re-created (cudaDeviceReset) never leaves a
// stale address behind; a call made during stream capture uses the cached address, which is why
// the first call on a device must come before any capture.
#include <cudaTypedefs.h>

#include <cstring>
#include <mutex>

#include "../../include/grpo.h"
#include "common.cuh"
#include "internal.h"

using namespace grpo;

namespace {

constexpr size_t kStaticScratchBytes = size_t(64) << 20;
static_assert(kStaticScratchBytes == GRPO_STATIC_SCRATCH_BYTES, "keep grpo.h in step");

__device__ __align__(256) unsigned char g_fwd_scratch[kStaticScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void* g_dev_ptr[kMaxDevices];  // device address of g_fwd_scratch, per device

int scratch_address(cudaStream_t st, void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return GRPO_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return GRPO_ERR_UNSUPPORTED;
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(st, &cap) != cudaSuccess) return GRPO_ERR_CUDA;
  std::lock_guard<std::mutex> lk(g_mu);
  if (g_dev_ptr[dev] == nullptr || cap == cudaStreamCaptureStatusNone) {
    if (cap != cudaStreamCaptureStatusNone) return GRPO_ERR_CUDA;   // first call inside a capture
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_fwd_scratch) != cudaSuccess || p == nullptr)
      return GRPO_ERR_CUDA;
    g_dev_ptr[dev] = p;
  }
  *out = g_dev_ptr[dev];
  return GRPO_OK;
}

size_t up256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

struct StaticLayout {
  int max_tiles, num_strips;
  long long rows_cap;
  size_t seq_base, row_pos, pos_row, zy, partials, hp, end;
};

StaticLayout static_layout(int S, int T, int d, int V, int dtype) {
  StaticLayout L{};
  const size_t P = static_cast<size_t>(S) * T;
  L.rows_cap = static_cast<long long>((P + kTileRows - 1) / kTileRows) * kTileRows;
  L.max_tiles = static_cast<int>(L.rows_cap / kTileRows);
  const int nvt = (V + kTileN - 1) / kTileN;
  L.num_strips = (nvt + kFwdTilesPerStrip - 1) / kFwdTilesPerStrip;
  size_t off = sizeof(WsHeader);
  L.seq_base = off;      off = up256(off + sizeof(int32_t) * (S + 1));
  L.row_pos = off;       off = up256(off + sizeof(int32_t) * L.rows_cap);
  L.pos_row = off;       off = up256(off + sizeof(int32_t) * P);
  L.zy = off;            off = up256(off + sizeof(float) * P);
  L.partials = off;
  if (dtype == GRPO_BF16) off = up256(off + sizeof(float4) * L.num_strips * L.rows_cap);
  L.hp = off;
  if (dtype == GRPO_BF16) off = up256(off + static_cast<size_t>(L.rows_cap) * d * 2);
  L.end = off;
  return L;
}

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
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

bool bf16_map(CUtensorMap* map, const void* base, uint64_t inner, uint64_t outer,
              uint32_t box_outer) {
  auto fn = tensor_map_encoder();
  if (!fn) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {inner * 2};
  cuuint32_t box[2] = {64, box_outer};
  cuuint32_t es[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
            es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int ok_or_cuda(cudaError_t e) { return e == cudaSuccess ? GRPO_OK : GRPO_ERR_CUDA; }

}  // namespace

extern "C" int grpo_score_fwd_static(const void* H, const void* W, int32_t dtype,
                                     const int32_t* tokens, const uint8_t* mask, int32_t S,
                                     int32_t T, int32_t d, int32_t V, float* logp, float* lse,
                                     float* entropy, int32_t* argmax, int32_t* valid_count,
                                     int32_t* status_out, grpo_stream_t stream) {
  if (!H || !W || !tokens || !mask || !logp || !lse || !entropy || !argmax || !valid_count)
    return GRPO_ERR_INVALID_ARG;
  if (S <= 0 || T <= 0 || d <= 0 || V <= 0 || static_cast<long long>(S) * T >= (1ll << 31) ||
      V >= (1 << 30))
    return GRPO_ERR_INVALID_ARG;
  if (dtype == GRPO_BF16) {
    if (d % 64 != 0) return GRPO_ERR_UNSUPPORTED;
    if ((reinterpret_cast<uintptr_t>(H) & 15u) || (reinterpret_cast<uintptr_t>(W) & 15u))
      return GRPO_ERR_INVALID_ARG;
  } else if (dtype == GRPO_F32) {
    if (d > 4096) return GRPO_ERR_UNSUPPORTED;
  } else {
    return GRPO_ERR_INVALID_ARG;
  }
  const StaticLayout L = static_layout(S, T, d, V, dtype);
  if (L.end > kStaticScratchBytes) return GRPO_ERR_WORKSPACE;  // batch too large for the array

  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  void* base = nullptr;
  const int st_addr = scratch_address(st, &base);
  if (st_addr != GRPO_OK) return st_addr;
  char* b = static_cast<char*>(base);
  WsHeader* hdr = reinterpret_cast<WsHeader*>(b);
  int32_t* seq_base = reinterpret_cast<int32_t*>(b + L.seq_base);
  int32_t* row_pos = reinterpret_cast<int32_t*>(b + L.row_pos);
  int32_t* pos_row = reinterpret_cast<int32_t*>(b + L.pos_row);
  float* zy = reinterpret_cast<float*>(b + L.zy);
  float4* partials = reinterpret_cast<float4*>(b + L.partials);
  void* hp = b + L.hp;

  // The array keeps the previous call's contents: the status word must start at zero. Every
  // other region used below is fully written before it is read within this call.
  int rc = ok_or_cuda(cudaMemsetAsync(hdr, 0, sizeof(WsHeader), st));
  if (rc != GRPO_OK) return rc;
  rc = counted_launch(GRPO_K_MASK_SCAN, st,
                      [&] { return launch_mask_scan(mask, S, T, valid_count, st); });
  if (rc != GRPO_OK) return rc;
  if (dtype == GRPO_F32) {
    rc = counted_launch(GRPO_K_F32_FWD, st, [&] {
      return launch_f32_fwd(static_cast<const float*>(H), static_cast<const float*>(W), tokens,
                            mask, S, T, d, V, logp, lse, entropy, argmax, hdr, st);
    });
  } else {
    rc = counted_launch(GRPO_K_PACK, st, [&] {
      return launch_pack(mask, valid_count, S, T, L.rows_cap, seq_base, row_pos, pos_row, hdr,
                         st);
    });
    if (rc != GRPO_OK) return rc;
    rc = counted_launch(GRPO_K_GATHER, st, [&] {
      return launch_gather_rows(H, d, row_pos, hdr, L.rows_cap, hp, st);
    });
    if (rc != GRPO_OK) return rc;
    const int tm = gemm_role_tile_mode(ROLE_FWD);
    CUtensorMap mapH, mapW;
    if (!bf16_map(&mapH, hp, d, static_cast<uint64_t>(L.rows_cap), kTileRows) ||
        !bf16_map(&mapW, W, d, V, gemm_b_box_rows(tm)))
      return GRPO_ERR_CUDA;
    GemmArgs a;
    std::memset(&a, 0, sizeof(a));
    a.S = S;
    a.T = T;
    a.d = d;
    a.V = V;
    a.row_pos = row_pos;
    a.hdr = hdr;
    a.tokens = tokens;
    a.mask = mask;
    a.rows_cap = L.rows_cap;
    a.num_strips = L.num_strips;
    a.partials = partials;
    a.zy = zy;
    a.inject_stall = debug_inject_stall();
    gemm_window_config(a);
    const int grid = gemm_grid(L.max_tiles, L.num_strips, tm);
    rc = counted_launch(GRPO_K_FWD_GEMM, st,
                        [&] { return launch_gemm(ROLE_FWD, mapH, mapW, a, grid, tm, st); });
    if (rc != GRPO_OK) return rc;
    rc = counted_launch(GRPO_K_FWD_MERGE, st, [&] {
      return launch_fwd_merge(partials, L.rows_cap, L.num_strips, zy, pos_row, tokens, mask, S,
                              T, V, logp, lse, entropy, argmax, hdr, st);
    });
  }
  if (rc != GRPO_OK) return rc;
  if (status_out)
    rc = ok_or_cuda(cudaMemcpyAsync(status_out, &hdr->status, sizeof(int32_t),
                                    cudaMemcpyDeviceToDevice, st));
  return rc;
}
