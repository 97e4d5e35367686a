// Persistent, warp-specialised tcgen05 GEMM for the four LM-head contractions of the GRPO path.
//
//   role FWD : z = H W^T per 128-token x 256-vocab tile (K = d), reduced on chip to the
//              running max / sum e^{z-m} / sum e^{z-m} z / argmax / target logit of each token
//              over a strip of 8 vocabulary tiles (Eq. 1's log pi: log-softmax at the sampled
//              token, plus entropy and argmax). The logits never leave the SM.
//   role DZ  : the same product recomputed, turned in registers into
//              dz = g_t (onehot(y_t) - exp(z - lse_t)) and stored as bf16 (one vocab chunk).
//   role DH  : dH = dz W (K = vocabulary chunk), f32 accumulation, written in H's dtype.
//   role DW  : dW = dz^T H (K = tokens), f32.
//
// Block = 6 warps: warp 0 issues TMA loads into a 4-stage shared-memory ring, warp 1 issues
// tcgen05.mma (M=128, N=256, K=16, bf16 in, f32 accumulate in tensor memory), warps 2-5 read
// the accumulator back with tcgen05.ld (one TMEM lane = one output row per thread) and run the
// role's epilogue. Two 256-column accumulators in TMEM let the epilogue of one tile overlap the
// MMAs of the next. Every wait is bounded (see mbar_wait_bounded).
#include <cfloat>

#include "common.cuh"
#include "internal.h"

namespace grpo {
namespace {

constexpr int BM = kTileRows;  // 128
constexpr int BN = kTileN;     // 256
constexpr int BK = 64;         // one 128-byte swizzle row of bf16
constexpr int STAGES = 4;
constexpr uint32_t A_STAGE = BM * BK * 2;  // 16 KB
constexpr uint32_t B_STAGE = BN * BK * 2;  // 32 KB
constexpr uint32_t STAGE_TX = A_STAGE + B_STAGE;
constexpr uint32_t BOX_MN = 64 * 64 * 2;   // one 64 x 64 bf16 box (MN-major operands)
constexpr uint32_t TMEM_COLS = 512;        // two 128 x 256 f32 accumulators
constexpr int NUM_THREADS = 192;
constexpr int GROUP_M = 16;                // raster: 16 row tiles share each column sweep
constexpr size_t SMEM_BYTES = size_t(STAGES) * STAGE_TX + 1024 + 256;

struct Dims {
  int num_m, num_n, num_kb;
};

template <int ROLE>
__device__ __forceinline__ Dims role_dims(const GemmArgs& a, int num_tiles) {
  Dims d;
  if (ROLE == ROLE_FWD) {
    d.num_m = num_tiles;
    d.num_n = a.num_strips;
    d.num_kb = a.d / BK;
  } else if (ROLE == ROLE_DZ) {
    d.num_m = num_tiles;
    d.num_n = (a.vc_len + BN - 1) / BN;
    d.num_kb = a.d / BK;
  } else if (ROLE == ROLE_DH) {
    d.num_m = num_tiles;
    d.num_n = a.d / BN;
    d.num_kb = (a.vc_len + BK - 1) / BK;
  } else {
    d.num_m = (a.vc_len + BM - 1) / BM;
    d.num_n = a.d / BN;
    d.num_kb = num_tiles * (BM / BK);
  }
  return d;
}

// Grouped raster: consecutive units walk GROUP_M row tiles before moving to the next column
// tile, so the CTAs resident at one time share a small set of A and B tiles in L2.
__device__ __forceinline__ void decode_unit(int u, int num_m, int num_n, int& m, int& n) {
  const int per_group = GROUP_M * num_n;
  const int grp = u / per_group;
  const int first_m = grp * GROUP_M;
  const int gm = min(GROUP_M, num_m - first_m);
  const int within = u - grp * per_group;
  m = first_m + within % gm;
  n = within / gm;
}

template <int ROLE>
__device__ __forceinline__ int acc_tiles_of_unit(const GemmArgs& a, int n) {
  if (ROLE == ROLE_FWD) {
    const int nvt = (a.V + BN - 1) / BN;
    return min(kFwdTilesPerStrip, nvt - n * kFwdTilesPerStrip);
  }
  return 1;
}

// ------------------------------------------------------------------------------------------
// producer: one thread
// ------------------------------------------------------------------------------------------
template <int ROLE>
__device__ void run_producer(const CUtensorMap* mapA, const CUtensorMap* mapB, const GemmArgs& a,
                             const Dims& dm, uint8_t* sA, uint8_t* sB, uint64_t* full,
                             uint64_t* empty, volatile int* abort_flag) {
  const int num_units = dm.num_m * dm.num_n;
  const bool stall = (a.inject_stall != 0) && blockIdx.x == 0;
  uint32_t stage = 0, phase = 0;
  long long issued = 0;
  bool ok = true;
  for (int u = blockIdx.x; u < num_units && ok; u += gridDim.x) {
    int m, n;
    decode_unit(u, dm.num_m, dm.num_n, m, n);
    const int nacc = acc_tiles_of_unit<ROLE>(a, n);
    int hrow = 0;
    if (ROLE == ROLE_FWD || ROLE == ROLE_DZ) {
      const int2 tl = a.tiles[m];
      hrow = tl.x * a.T + tl.y;
    }
    for (int t = 0; t < nacc && ok; ++t) {
      for (int kb = 0; kb < dm.num_kb; ++kb) {
        if (!mbar_wait_bounded(&empty[stage], phase ^ 1u, abort_flag, a.hdr,
                               WHERE_GEMM_BASE + ROLE * 16 + 1)) {
          ok = false;
          break;
        }
        const uint32_t dA = smem_u32(sA + stage * A_STAGE);
        const uint32_t dB = smem_u32(sB + stage * B_STAGE);
        if (stall && issued == 0) {
          // test hook: leave stage 0 unfilled so that the MMA warp's bounded wait runs out
        } else {
          mbar_arrive_expect_tx(&full[stage], STAGE_TX);
          if (ROLE == ROLE_FWD || ROLE == ROLE_DZ) {
            const int vt = (ROLE == ROLE_FWD) ? n * kFwdTilesPerStrip + t : a.vc0 / BN + n;
            tma_load_2d(dA, mapA, &full[stage], kb * BK, hrow);
            tma_load_2d(dB, mapB, &full[stage], kb * BK, vt * BN);
          } else if (ROLE == ROLE_DH) {
            tma_load_2d(dA, mapA, &full[stage], kb * BK, m * BM);
#pragma unroll
            for (int j = 0; j < BN / 64; ++j)
              tma_load_2d(dB + j * BOX_MN, mapB, &full[stage], n * BN + j * 64, a.vc0 + kb * BK);
          } else {  // ROLE_DW
#pragma unroll
            for (int j = 0; j < BM / 64; ++j)
              tma_load_2d(dA + j * BOX_MN, mapA, &full[stage], m * BM + j * 64, kb * BK);
            const int2 tl = a.tiles[kb >> 1];
            const int row = tl.x * a.T + tl.y + (kb & 1) * BK;
#pragma unroll
            for (int j = 0; j < BN / 64; ++j)
              tma_load_2d(dB + j * BOX_MN, mapB, &full[stage], n * BN + j * 64, row);
          }
        }
        ++issued;
        if (++stage == STAGES) {
          stage = 0;
          phase ^= 1u;
        }
      }
    }
  }
  if (!ok) {
    // Aborted: let the copies already in flight land before the CTA exits (bounded).
    const long long back = issued < STAGES ? issued : STAGES;
    for (long long i = 1; i <= back; ++i) {
      const long long it = issued - i;
      if (stall && it == 0) continue;
      const uint32_t s = static_cast<uint32_t>(it % STAGES);
      const uint32_t ph = static_cast<uint32_t>((it / STAGES) & 1);
      mbar_wait_drain(&full[s], ph, 100000000ull);
    }
  }
}

// ------------------------------------------------------------------------------------------
// MMA issuer: one thread
// ------------------------------------------------------------------------------------------
template <int ROLE>
__device__ void run_mma(const GemmArgs& a, const Dims& dm, uint8_t* sA, uint8_t* sB,
                        uint64_t* full, uint64_t* empty, uint64_t* accf, uint64_t* acce,
                        uint64_t* drain, uint32_t tmem_base, volatile int* abort_flag) {
  constexpr bool A_MN = (ROLE == ROLE_DW);
  constexpr bool B_MN = (ROLE == ROLE_DH || ROLE == ROLE_DW);
  constexpr uint32_t idesc = idesc_bf16_f32(BM, BN, A_MN, B_MN);
  const int num_units = dm.num_m * dm.num_n;
  uint32_t stage = 0, phase = 0, buf = 0, bphase = 0;
  bool ok = true;
  for (int u = blockIdx.x; u < num_units && ok; u += gridDim.x) {
    int m, n;
    decode_unit(u, dm.num_m, dm.num_n, m, n);
    const int nacc = acc_tiles_of_unit<ROLE>(a, n);
    for (int t = 0; t < nacc && ok; ++t) {
      if (!mbar_wait_bounded(&acce[buf], bphase ^ 1u, abort_flag, a.hdr,
                             WHERE_GEMM_BASE + ROLE * 16 + 2)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t d_tmem = tmem_base + buf * BN;
      for (int kb = 0; kb < dm.num_kb; ++kb) {
        if (!mbar_wait_bounded(&full[stage], phase, abort_flag, a.hdr,
                               WHERE_GEMM_BASE + ROLE * 16 + 3)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t a0 = smem_u32(sA + stage * A_STAGE);
        const uint32_t b0 = smem_u32(sB + stage * B_STAGE);
#pragma unroll
        for (int k = 0; k < BK / 16; ++k) {
          const uint64_t ad = A_MN ? sdesc_sw128(a0 + k * 2048, BOX_MN, 1024)
                                   : sdesc_sw128(a0 + k * 32, 16, 1024);
          const uint64_t bd = B_MN ? sdesc_sw128(b0 + k * 2048, BOX_MN, 1024)
                                   : sdesc_sw128(b0 + k * 32, 16, 1024);
          umma_bf16(d_tmem, ad, bd, idesc, (kb | k) != 0 ? 1u : 0u);
        }
        umma_commit(&empty[stage]);  // frees the smem stage once these MMAs have read it
        if (++stage == STAGES) {
          stage = 0;
          phase ^= 1u;
        }
      }
      if (!ok) break;
      umma_commit(&accf[buf]);       // accumulator ready for the epilogue
      buf ^= 1u;
      if (buf == 0) bphase ^= 1u;
    }
  }
  // Make sure no MMA is still writing tensor memory when it is released.
  umma_commit(drain);
  mbar_wait_drain(drain, 0, 200000000ull);
}

// ------------------------------------------------------------------------------------------
// epilogues: warps 2..5, thread = one accumulator row (TMEM lane)
// ------------------------------------------------------------------------------------------
__device__ __forceinline__ bool epi_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                         WsHeader* hdr, int32_t where) {
  const bool ok = mbar_wait_bounded(bar, parity, abort_flag, hdr, where);
  return __all_sync(0xffffffffu, ok);
}

__device__ __forceinline__ void epi_release(uint64_t* bar, int lane) {
  tc_fence_before();
  __syncwarp();
  if (lane == 0) mbar_arrive(bar);
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 p = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&p);
}

template <int ROLE>
__device__ void run_epilogue(const GemmArgs& a, const Dims& dm, uint64_t* accf, uint64_t* acce,
                             uint32_t tmem_base, volatile int* abort_flag) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int q = warp & 3;               // TMEM lane quadrant this warp may access
  const int r = q * 32 + lane;          // accumulator row of this thread
  const uint32_t t_row = tmem_base + (static_cast<uint32_t>(q * 32) << 16);
  const int num_units = dm.num_m * dm.num_n;
  const int32_t where = WHERE_GEMM_BASE + ROLE * 16 + 4;
  uint32_t buf = 0, bphase = 0;
  for (int u = blockIdx.x; u < num_units; u += gridDim.x) {
    int m, n;
    decode_unit(u, dm.num_m, dm.num_n, m, n);

    if (ROLE == ROLE_FWD) {
      const int2 tl = a.tiles[m];
      const bool rv = tl.y + r < a.T;
      const long long pos = static_cast<long long>(tl.x) * a.T + tl.y + r;
      const int y = (rv && a.mask[pos] != 0) ? a.tokens[pos] : -1;
      float rm = -INFINITY, rs = 0.f, ru = 0.f, zyv = 0.f;
      int ri = 0;
      bool found = false;
      const int nacc = acc_tiles_of_unit<ROLE>(a, n);
      for (int t = 0; t < nacc; ++t) {
        if (!epi_wait(&accf[buf], bphase, abort_flag, a.hdr, where)) return;
        tc_fence_after();
        const int vbase = (n * kFwdTilesPerStrip + t) * BN;
        for (int c = 0; c < BN / 32; ++c) {
          const int v0 = vbase + c * 32;
          if (v0 >= a.V) break;  // uniform across the warp
          float x[32];
          tmem_load_32cols(t_row + buf * BN + c * 32, x);
          const int nvalid = a.V - v0;
          if (nvalid < 32) {
#pragma unroll
            for (int j = 0; j < 32; ++j)
              if (j >= nvalid) x[j] = -1.0e30f;  // columns past the vocabulary
          }
          float cm = x[0];
          int ci = 0;
#pragma unroll
          for (int j = 1; j < 32; ++j) {
            if (x[j] > cm) {
              cm = x[j];
              ci = j;
            }
          }
          if (cm > rm) {  // strictly greater: earlier (lower) index wins ties
            const float sc = ex2_approx((rm - cm) * kLog2e);
            rs *= sc;
            ru *= sc;
            rm = cm;
            ri = v0 + ci;
          }
          const float ml = rm * kLog2e;
          float ps = 0.f, pu = 0.f;
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            const float e = ex2_approx(fmaf(x[j], kLog2e, -ml));
            ps += e;
            pu = fmaf(e, x[j], pu);
          }
          rs += ps;
          ru += pu;
          const int rel = y - v0;
          if (rel >= 0 && rel < 32) {
            float zt = x[0];
#pragma unroll
            for (int j = 1; j < 32; ++j)
              if (j == rel) zt = x[j];
            zyv = zt;
            found = true;
          }
        }
        epi_release(&acce[buf], lane);
        buf ^= 1u;
        if (buf == 0) bphase ^= 1u;
      }
      a.partials[static_cast<long long>(n) * a.rows_cap + static_cast<long long>(m) * BM + r] =
          make_float4(rm, rs, ru, __int_as_float(ri));
      if (found) a.zy[pos] = zyv;

    } else if (ROLE == ROLE_DZ) {
      const int2 tl = a.tiles[m];
      const bool rv = tl.y + r < a.T;
      const long long pos = static_cast<long long>(tl.x) * a.T + tl.y + r;
      const bool act = rv && a.mask[pos] != 0;
      const float gt = act ? a.g[pos] : 0.f;
      const float ll = act ? a.lse[pos] * kLog2e : 0.f;
      const int y = act ? a.tokens[pos] : -1;
      if (!epi_wait(&accf[buf], bphase, abort_flag, a.hdr, where)) return;
      tc_fence_after();
      __nv_bfloat16* dst_row =
          a.dz + (static_cast<size_t>(m) * BM + r) * static_cast<size_t>(a.dz_pitch);
      for (int c = 0; c < BN / 32; ++c) {
        const int vloc = n * BN + c * 32;
        const int v0 = a.vc0 + vloc;
        float x[32];
        tmem_load_32cols(t_row + buf * BN + c * 32, x);
        uint32_t pk[16];
        if (act) {
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            const int va = v0 + 2 * j, vb = va + 1;
            const float pa = ex2_approx(fmaf(x[2 * j], kLog2e, -ll));
            const float pb = ex2_approx(fmaf(x[2 * j + 1], kLog2e, -ll));
            const float da = va < a.V ? gt * ((va == y ? 1.f : 0.f) - pa) : 0.f;
            const float db = vb < a.V ? gt * ((vb == y ? 1.f : 0.f) - pb) : 0.f;
            pk[j] = pack_bf16x2(da, db);
          }
        } else {
#pragma unroll
          for (int j = 0; j < 16; ++j) pk[j] = 0u;
        }
        uint4* dst = reinterpret_cast<uint4*>(dst_row + vloc);
#pragma unroll
        for (int j = 0; j < 4; ++j)
          dst[j] = make_uint4(pk[4 * j], pk[4 * j + 1], pk[4 * j + 2], pk[4 * j + 3]);
      }
      epi_release(&acce[buf], lane);
      buf ^= 1u;
      if (buf == 0) bphase ^= 1u;

    } else if (ROLE == ROLE_DH) {
      const int2 tl = a.tiles[m];
      const bool rv = tl.y + r < a.T;
      const long long pos = static_cast<long long>(tl.x) * a.T + tl.y + r;
      if (!epi_wait(&accf[buf], bphase, abort_flag, a.hdr, where)) return;
      tc_fence_after();
      for (int c = 0; c < BN / 32; ++c) {
        const int col = n * BN + c * 32;
        float x[32];
        tmem_load_32cols(t_row + buf * BN + c * 32, x);
        if (!rv) continue;
        float* acc_row = a.dH_acc + (static_cast<size_t>(m) * BM + r) * a.d + col;
        if (a.dh_mode == 2 || a.dh_mode == 3) {
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const float4 p = reinterpret_cast<const float4*>(acc_row)[j];
            x[4 * j] += p.x;
            x[4 * j + 1] += p.y;
            x[4 * j + 2] += p.z;
            x[4 * j + 3] += p.w;
          }
        }
        if (a.dh_mode == 1 || a.dh_mode == 2) {
#pragma unroll
          for (int j = 0; j < 8; ++j)
            reinterpret_cast<float4*>(acc_row)[j] =
                make_float4(x[4 * j], x[4 * j + 1], x[4 * j + 2], x[4 * j + 3]);
        } else {
          uint4* dst = reinterpret_cast<uint4*>(a.dH + pos * a.d + col);
#pragma unroll
          for (int j = 0; j < 4; ++j)
            dst[j] = make_uint4(pack_bf16x2(x[8 * j], x[8 * j + 1]),
                                pack_bf16x2(x[8 * j + 2], x[8 * j + 3]),
                                pack_bf16x2(x[8 * j + 4], x[8 * j + 5]),
                                pack_bf16x2(x[8 * j + 6], x[8 * j + 7]));
        }
      }
      epi_release(&acce[buf], lane);
      buf ^= 1u;
      if (buf == 0) bphase ^= 1u;

    } else {  // ROLE_DW
      const int vrow = m * BM + r;
      const bool rv = vrow < a.vc_len;
      // No scored token at all (K = 0): no MMA ran, the accumulator holds nothing -> dW = 0.
      const bool empty_k = dm.num_kb == 0;
      if (!epi_wait(&accf[buf], bphase, abort_flag, a.hdr, where)) return;
      tc_fence_after();
      float* dst_row = a.dW + static_cast<size_t>(a.vc0 + vrow) * a.d + n * BN;
      for (int c = 0; c < BN / 32; ++c) {
        float x[32];
        tmem_load_32cols(t_row + buf * BN + c * 32, x);
        if (!rv) continue;
        if (empty_k) {
#pragma unroll
          for (int j = 0; j < 32; ++j) x[j] = 0.f;
        }
        float4* dst = reinterpret_cast<float4*>(dst_row + c * 32);
#pragma unroll
        for (int j = 0; j < 8; ++j)
          dst[j] = make_float4(x[4 * j], x[4 * j + 1], x[4 * j + 2], x[4 * j + 3]);
      }
      epi_release(&acce[buf], lane);
      buf ^= 1u;
      if (buf == 0) bphase ^= 1u;
    }
  }
}

// ------------------------------------------------------------------------------------------
// kernel
// ------------------------------------------------------------------------------------------
template <int ROLE>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    tc_gemm(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapB,
            const __grid_constant__ GemmArgs args) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + STAGES * A_STAGE;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sB + STAGES * B_STAGE);
  uint64_t* full = bars;
  uint64_t* empty = bars + STAGES;
  uint64_t* accf = bars + 2 * STAGES;
  uint64_t* acce = accf + 2;
  uint64_t* drain = acce + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&accf[b], 1);
      mbar_init(&acce[b], 4);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_barrier_init();
    fence_proxy_async_smem();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&mapA);
    tma_prefetch_desc(&mapB);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const Dims dm = role_dims<ROLE>(args, args.hdr->num_tiles);

  if (warp == 0) {
    if (lane == 0) run_producer<ROLE>(&mapA, &mapB, args, dm, sA, sB, full, empty, abort_flag);
  } else if (warp == 1) {
    if (lane == 0)
      run_mma<ROLE>(args, dm, sA, sB, full, empty, accf, acce, drain, tmem_base, abort_flag);
  } else {
    run_epilogue<ROLE>(args, dm, accf, acce, tmem_base, abort_flag);
  }
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem_base, TMEM_COLS);
}

template <int ROLE>
cudaError_t launch_role(const CUtensorMap& mapA, const CUtensorMap& mapB, const GemmArgs& args,
                        int grid, cudaStream_t st) {
  cudaError_t e = cudaFuncSetAttribute(tc_gemm<ROLE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(SMEM_BYTES));
  if (e != cudaSuccess) return e;
  tc_gemm<ROLE><<<grid, NUM_THREADS, SMEM_BYTES, st>>>(mapA, mapB, args);
  return cudaGetLastError();
}

}  // namespace

size_t gemm_smem_bytes() { return SMEM_BYTES; }

cudaError_t launch_gemm(int role, const CUtensorMap& mapA, const CUtensorMap& mapB,
                        const GemmArgs& args, int grid, cudaStream_t st) {
  switch (role) {
    case ROLE_FWD: return launch_role<ROLE_FWD>(mapA, mapB, args, grid, st);
    case ROLE_DZ: return launch_role<ROLE_DZ>(mapA, mapB, args, grid, st);
    case ROLE_DH: return launch_role<ROLE_DH>(mapA, mapB, args, grid, st);
    case ROLE_DW: return launch_role<ROLE_DW>(mapA, mapB, args, grid, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace grpo
