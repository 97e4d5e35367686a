// Persistent, warp-specialised tcgen05 GEMM for the four LM-head contractions of the GRPO path.
//
//   role FWD : z = H W^T per 128-token x 256-vocab tile (K = d), reduced on chip to the
//              max / sum e^{z-m} / sum e^{z-m} z / argmax / target logit of each token over the
//              tile's strip of vocabulary columns (Eq. 1's log pi: log-softmax at the sampled
//              token, plus entropy and argmax). The logits never leave the SM.
//   role DZ  : the same product recomputed, turned in registers into
//              dz = g_t (onehot(y_t) - exp(z - lse_t)) and stored as bf16 (one vocab chunk).
//   role DH  : dH = dz W (K = vocabulary chunk), f32 accumulation, written in H's dtype.
//   role DW  : dW = dz^T H (K = tokens), f32.
//
// Block = 6 warps: warp 0 issues TMA loads into a shared-memory ring, warp 1 issues tcgen05.mma
// (bf16 in, f32 accumulate in tensor memory), warps 2-5 read the accumulator back with
// tcgen05.ld (one TMEM lane = one output row per thread) and run the role's epilogue.
// Tile modes (see Cfg): one CTA per 128 x 256 tile (cta_group::1) with two TMEM accumulators so
// that the epilogue of one tile overlaps the MMAs of the next; a CTA pair per 256 x 256 tile
// (cta_group::2, two accumulators); or, for the long-K roles DH and DW, a CTA pair per 256 x 512
// tile (cta_group::2, two N = 256 MMAs per k-step into one 512-column accumulator). Every TMA
// load lands in the issuing CTA's own shared memory (the pair modes count both CTAs' bytes on
// the leader's barrier). Every wait is bounded (see mbar_wait_bounded).
#include <cfloat>

#include "common.cuh"
#include <atomic>

#include "internal.h"

namespace grpo {
namespace {

constexpr int BM = kTileRows;  // 128 accumulator rows per CTA
constexpr int BN = kTileN;     // 256
constexpr int BK = 64;         // one 128-byte swizzle row of bf16
constexpr uint32_t BOX_MN = 64 * 64 * 2;   // one 64 x 64 bf16 box (MN-major operands)
constexpr uint32_t TMEM_COLS = 512;        // two 128 x 256 f32 accumulators
constexpr int NUM_THREADS = 192;          // 6 warps (modes 0, 1); mode 2: Cfg<2>::THREADS
// Raster groups: row tiles that consecutive work units walk before moving to the next column
// unit, per role. Measured on a power-capped GB300 at 2 x 16 completions, T = 16384, d = 5120,
// V = 151936 (the GEMM's time against the neighbouring values): forward 32 (16: +0-2 %,
// 48: +8 %, 64: +14 %: the group's H rows no longer stay in L2), dz recompute 32 (16: +1.5 %,
// 48: +9 %, 64: +12 %), dH and dW 32 (24, 48: +0.5-1 %; 64: +1 %, with 20-24 % more DRAM
// bytes). A wave of 76 CTA-pair units covers g/2 row units x 152/g column units, so larger
// groups re-read the row operand (dz) more often and smaller ones the column operand (W, Hp).
#ifndef GRPO_GROUP_M_FWD
#define GRPO_GROUP_M_FWD 32
#endif
#ifndef GRPO_GROUP_M_DZ
#define GRPO_GROUP_M_DZ 32
#endif
#ifndef GRPO_GROUP_M_DH
#define GRPO_GROUP_M_DH 32
#endif
#ifndef GRPO_GROUP_M_DW
#define GRPO_GROUP_M_DW 32
#endif
template <int ROLE>
constexpr int group_rows() {
  return ROLE == ROLE_FWD || ROLE == ROLE_FWD_KL ? GRPO_GROUP_M_FWD
         : ROLE == ROLE_DZ || ROLE == ROLE_DZ_KL ? GRPO_GROUP_M_DZ
         : ROLE == ROLE_DH                       ? GRPO_GROUP_M_DH
                                                 : GRPO_GROUP_M_DW;
}

// Tile modes (MODE template parameter):
//   0 single CTA : one CTA computes a 128 x 256 tile (tcgen05 cta_group::1, M = 128); two
//                  256-column accumulators in TMEM.
//   1 CTA pair   : a cluster of 2 CTAs on one TPC computes a 256 x 256 tile with cta_group::2
//                  (M = 256): each CTA stages its 128 rows of A and half (128 rows) of B, and the
//                  pair's tensor cores read both halves of B, so per-SM operand traffic per flop
//                  is 2/3 of mode 0's and the ring can be 6 deep. Two accumulators.
//   2 wide pair  : the CTA pair computes a 256 x 512 tile: per k-step two N = 256 MMAs write the
//                  two 256-column halves of one 512-column accumulator. Each CTA stages 128 rows
//                  of A and 2 x 128 rows of B per k-block (48 KB), i.e. half of mode 0's operand
//                  bytes per flop; eight epilogue warps each read one half. The epilogue does not
//                  overlap the next tile's MMAs, which is negligible for the long-K roles DH and
//                  DW (thousands of k-blocks per tile against one epilogue) that this mode is
//                  made for; a forward or dz unit is two vocabulary tiles.
template <int MODE>
struct Cfg {
  static constexpr bool PAIR = MODE != 0;                   // cta_group::2 on a 2-CTA cluster
  static constexpr int CL = PAIR ? 2 : 1;                   // CTAs per cluster
  static constexpr int NT = MODE == 2 ? 2 : 1;              // 256-column MMAs per k-step
  static constexpr int ACC_BUFS = MODE == 2 ? 1 : 2;        // accumulators in TMEM
  // epilogue warps: 4 (one per TMEM lane quadrant), or 8 in mode 2 (two per quadrant, each
  // reading one 256-column half of the single accumulator, which halves the time the next
  // tile's MMAs wait for it)
  static constexpr int EPI_WARPS = MODE == 2 ? 8 : 4;
  static constexpr int THREADS = (2 + EPI_WARPS) * 32;
  static constexpr int STAGES = MODE == 1 ? 6 : 4;
  static constexpr uint32_t A_STAGE = BM * BK * 2;          // 16 KB
  static constexpr uint32_t B_HALF_ROWS = PAIR ? BN / 2 : BN;   // B rows per MMA staged here
  static constexpr uint32_t B_ROWS = NT * B_HALF_ROWS;      // B rows staged here per k-block
  static constexpr uint32_t B_HALF_STAGE = B_HALF_ROWS * BK * 2;
  static constexpr uint32_t B_STAGE = B_ROWS * BK * 2;      // 32, 16 or 32 KB
  static constexpr uint32_t STAGE_TX = A_STAGE + B_STAGE;   // bytes landing per CTA
  static constexpr size_t SMEM = size_t(STAGES) * STAGE_TX + 1024 + 256;
};
// Shared-memory staging of the dz tile for its TMA stores (single-CTA dz only): per epilogue warp
// two buffers of 32 rows x 64 bf16 columns (4 KB, rows of 128 bytes in the 128-byte swizzle), so
// that a warp fills one while the TMA engine reads the other.
template <int ROLE, int MODE>
struct OutStage {
  static constexpr bool on = MODE == 0 && ROLE == ROLE_DZ;
  static constexpr uint32_t BUF = 32 * 64 * 2;
  static constexpr uint32_t BYTES = on ? 4 * 2 * BUF : 0;
};
template <int ROLE, int MODE>
constexpr size_t smem_bytes() {
  return Cfg<MODE>::SMEM + OutStage<ROLE, MODE>::BYTES;
}
constexpr size_t smax(size_t a, size_t b) { return a > b ? a : b; }
constexpr size_t SMEM_BYTES =
    smax(smem_bytes<ROLE_DZ, 0>(), smax(Cfg<0>::SMEM, smax(Cfg<1>::SMEM, Cfg<2>::SMEM)));
static_assert(SMEM_BYTES <= 227 * 1024, "shared memory per CTA");

struct Dims {
  int num_m, num_n, num_kb;
};

template <int ROLE>
__device__ __forceinline__ Dims role_dims(const GemmArgs& a, int num_tiles) {
  Dims d;
  if (ROLE == ROLE_FWD || ROLE == ROLE_FWD_KL) {
    d.num_m = num_tiles;
    d.num_n = a.num_strips;
    d.num_kb = (ROLE == ROLE_FWD_KL ? 2 : 1) * (a.d / BK);   // KL: policy, then reference
  } else if (ROLE == ROLE_DZ || ROLE == ROLE_DZ_KL) {
    d.num_m = num_tiles;
    d.num_n = (a.vc_len + BN - 1) / BN;
    d.num_kb = (ROLE == ROLE_DZ_KL ? 2 : 1) * (a.d / BK);
  } else if (ROLE == ROLE_DH) {   // d % 64 == 0: the last column tile may be partial
    d.num_m = num_tiles;
    d.num_n = (a.d + BN - 1) / BN;
    d.num_kb = (a.vc_len + BK - 1) / BK;
  } else {
    d.num_m = (a.vc_len + BM - 1) / BM;
    d.num_n = (a.d + BN - 1) / BN;
    d.num_kb = num_tiles * (BM / BK);
  }
  return d;
}

// Grouped raster: consecutive units walk `group` row units before moving to the next column
// tile, so the CTAs resident at one time share a small set of A and B tiles in L2.
__device__ __forceinline__ void decode_unit(int u, int num_m, int num_n, int group, int& m,
                                            int& n) {
  const int per_group = group * num_n;
  const int grp = u / per_group;
  const int first_m = grp * group;
  const int gm = min(group, num_m - first_m);
  const int within = u - grp * per_group;
  m = first_m + within % gm;
  n = within / gm;
}

// Roles whose tile holds two products (policy z in TMEM columns 0-255, reference z_ref in
// 256-511): one accumulator buffer instead of two.
template <int ROLE>
struct Dual {
  static constexpr bool value = (ROLE == ROLE_FWD_KL || ROLE == ROLE_DZ_KL);
};

template <int ROLE>
__device__ __forceinline__ int acc_tiles_of_unit(const GemmArgs& a, int n) {
  if (ROLE == ROLE_FWD || ROLE == ROLE_FWD_KL) {
    const int nvt = (a.V + BN - 1) / BN;
    return min(kFwdTilesPerStrip, nvt - n * kFwdTilesPerStrip);
  }
  return 1;
}

// Work layout shared by the three roles of a CTA. In the pair modes a unit is the 2 consecutive
// row tiles of a pair (2*mu + rank for CTA `rank`) with one column unit of NT 256-column tiles,
// and units are strided over the resident pairs.
template <int ROLE, int MODE>
struct Sched {
  int rank;        // CTA rank in the cluster (pair modes: 0 = leader, issues the MMAs); 0 in mode 0
  int group;       // row units per raster group
  int first, step; // unit loop: u = first; u < num_units; u += step
  int num_mu, num_nu, num_units;

  __device__ __forceinline__ Sched(const Dims& dm) {
    constexpr int CL = Cfg<MODE>::CL;
    constexpr int NT = Cfg<MODE>::NT;
    rank = CL > 1 ? static_cast<int>(cluster_ctarank()) : 0;
    first = static_cast<int>(blockIdx.x) / CL;
    step = static_cast<int>(gridDim.x) / CL;
    num_mu = (dm.num_m + CL - 1) / CL;
    num_nu = (dm.num_n + NT - 1) / NT;
    group = group_rows<ROLE>() / CL > 0 ? group_rows<ROLE>() / CL : 1;   // in row units
    num_units = num_mu * num_nu;
  }
  // Unit u -> the row tile m this CTA stages (always a valid tile), the column unit n, and
  // whether this CTA stores its result (false for the second CTA of a pair past the last row
  // tile, which stages a copy of its leader's rows so that the pair's MMAs read valid data).
  __device__ __forceinline__ void decode(int u, const Dims& dm, int& m, int& n, bool& ok) const {
    constexpr int CL = Cfg<MODE>::CL;
    int mu;
    decode_unit(u, num_mu, num_nu, group, mu, n);
    m = CL * mu + rank;
    ok = m < dm.num_m;
    if (!ok) m = CL * mu;
  }
};

// ------------------------------------------------------------------------------------------
// producer: one thread per CTA
// ------------------------------------------------------------------------------------------
// Progress window. CTAs that read the same operand tile at the same k-block (a row tile of A
// shared by the CTAs working on its other column tiles, or a column tile of B shared by the
// CTAs on other row tiles) find it in L2 only if they read it within a few tens of microseconds
// of one another: the L2 turns over that fast under these kernels' traffic. Over the thousands
// of k-blocks of a long-K unit, and over the successive units a CTA takes in turn, CTAs
// otherwise drift apart by more than that. So at every checkpoint the producer of each CTA
// counts itself in and waits until the CTAs of the launch have, on average, reached `lag`
// checkpoints behind it. Checkpoints fall every `check` k-blocks (check > 0) or at the start of
// every -check-th work unit (check < 0: with lag 1, a barrier between the waves of units, so
// the drift never outlasts one unit and no wait falls inside one). The slowest CTA never waits,
// so the window cannot deadlock. It is a hint: a wait that runs past its bound switches the
// window off for this CTA, and a CTA that leaves adds 2^40 so that no one waits for it.
struct ProgressWindow {
  unsigned long long* arrivals;
  uint32_t* exited;
  unsigned long long grid;
  int check, lag;
  bool on;
  // `long_k`: the window applies to the long-K roles (dH, dW) only; the forward and dz GEMMs,
  // whose units are one short tile, never wait (a barrier there costs 3-4 % and saves nothing).
  __device__ __forceinline__ ProgressWindow(const GemmArgs& a, bool long_k)
      : arrivals(&a.hdr->win_arrivals), exited(&a.hdr->win_exited), grid(gridDim.x),
        check(a.win_check), lag(a.win_lag), on(long_k && a.win_check != 0 && a.win_lag > 0) {}
  // Checkpoint number c reached: count in, then wait for the launch's average.
  __device__ __forceinline__ void arrive_and_wait(long long c) {
    atomicAdd(arrivals, 1ull);
    if (c < lag) return;
    const unsigned long long target = grid * static_cast<unsigned long long>(c - lag + 1);
    const uint64_t t0 = global_timer_ns();
    while (ld_relaxed_u64(arrivals) < target) {
      if (global_timer_ns() - t0 > 500000ull) {   // 0.5 ms: give up the window
        on = false;
        return;
      }
      __nanosleep(64);
    }
  }
  // Before issuing k-block number `kblocks_issued` (counted over the whole launch).
  __device__ __forceinline__ void at(long long kblocks_issued) {
    if (!on || check <= 0 || kblocks_issued == 0 || kblocks_issued % check != 0) return;
    arrive_and_wait(kblocks_issued / check);
  }
  // Before the first k-block of this CTA's work unit number `units_started` (0, 1, ...).
  __device__ __forceinline__ void at_unit(long long units_started) {
    if (!on || check >= 0 || units_started == 0 || units_started % (-check) != 0) return;
    arrive_and_wait(units_started / (-check));
  }
  __device__ __forceinline__ void leave() {
    atomicAdd(arrivals, 1ull << 40);
    __threadfence();
    if (atomicAdd(exited, 1u) == static_cast<uint32_t>(grid - 1)) {   // last CTA: reset
      atomicExch(arrivals, 0ull);
      atomicExch(exited, 0u);
    }
  }
};

template <int ROLE, int MODE>
__device__ void run_producer(const CUtensorMap* mapA, const CUtensorMap* mapB,
                             const CUtensorMap* mapA2, const CUtensorMap* mapB2, const GemmArgs& a,
                             const Dims& dm, const Sched<ROLE, MODE>& sc, uint8_t* sA, uint8_t* sB,
                             uint64_t* full, uint64_t* empty, volatile int* abort_flag) {
  using C = Cfg<MODE>;
  constexpr bool PAIR = C::PAIR;
  constexpr int NT = C::NT;
  // pair modes: only the leader's barriers count (both CTAs' bytes); mode 0: every CTA's own
  const bool leader = !PAIR || sc.rank == 0;
  const bool stall = (a.inject_stall != 0) && blockIdx.x == 0;   // CTA 0 is a leader
  constexpr int B_BOXES = static_cast<int>(C::B_HALF_ROWS) / 64;  // MN-major B boxes per MMA
  // first B row (N) of this CTA's share of each 256-column MMA: the pair splits B by rows
  const int b_row0 = PAIR ? sc.rank * static_cast<int>(C::B_HALF_ROWS) : 0;
  uint32_t stage = 0, phase = 0;
  long long issued = 0;
  bool ok = true;
  ProgressWindow win(a, ROLE == ROLE_DH || ROLE == ROLE_DW);
  long long units_started = 0;
  for (int u = sc.first; u < sc.num_units && ok; u += sc.step) {
    int m_load, n;
    bool m_ok;
    sc.decode(u, dm, m_load, n, m_ok);
    win.at_unit(units_started++);
    const int nacc = acc_tiles_of_unit<ROLE>(a, n);
    const int hrow = m_load * BM;   // first packed row of the tile (FWD / DZ / KL A operand)
    // The boxes of k-block kbi of accumulator tile ti: fa / fb(smem offset, map, x, y) for each
    // box of A / B this CTA loads.
    auto boxes = [&](int ti, int kbi, auto&& fa, auto&& fb) {
      if (ROLE == ROLE_FWD || ROLE == ROLE_DZ) {
        fa(0u, mapA, kbi * BK, hrow);
#pragma unroll
        for (int h = 0; h < NT; ++h) {   // wide pair: vocabulary tiles 2n and 2n+1
          const int vt = (ROLE == ROLE_FWD) ? (n * NT + h) * kFwdTilesPerStrip + ti
                                            : a.vc0 / BN + n * NT + h;
          fb(h * C::B_HALF_STAGE, mapB, kbi * BK, vt * BN + b_row0);
        }
      } else if (Dual<ROLE>::value) {
        // k-blocks 0 .. nk-1: policy (H, W); nk .. 2nk-1: reference (H_ref, W_ref)
        const int nk = dm.num_kb / 2;
        const bool second = kbi >= nk;
        const int kk = second ? kbi - nk : kbi;
        const int vt = (ROLE == ROLE_FWD_KL) ? n * kFwdTilesPerStrip + ti : a.vc0 / BN + n;
        fa(0u, second ? mapA2 : mapA, kk * BK, hrow);
        fb(0u, second ? mapB2 : mapB, kk * BK, vt * BN + b_row0);
      } else if (ROLE == ROLE_DH) {
        fa(0u, mapA, kbi * BK, m_load * BM);
#pragma unroll
        for (int h = 0; h < NT; ++h)
#pragma unroll
          for (int j = 0; j < B_BOXES; ++j)
            fb((h * B_BOXES + j) * BOX_MN, mapB, (n * NT + h) * BN + b_row0 + j * 64,
               a.vc0 + kbi * BK);
      } else {  // ROLE_DW: K runs over packed rows
#pragma unroll
        for (int j = 0; j < BM / 64; ++j)
          fa(j * BOX_MN, mapA, m_load * BM + j * 64, kbi * BK);
#pragma unroll
        for (int h = 0; h < NT; ++h)
#pragma unroll
          for (int j = 0; j < B_BOXES; ++j)
            fb((h * B_BOXES + j) * BOX_MN, mapB, (n * NT + h) * BN + b_row0 + j * 64, kbi * BK);
      }
    };
    for (int t = 0; t < nacc && ok; ++t) {
      for (int kb = 0; kb < dm.num_kb; ++kb) {
        win.at(issued);
        if (!mbar_wait_bounded(&empty[stage], phase ^ 1u, abort_flag, a.hdr,
                               WHERE_GEMM_BASE + ROLE * 16 + 1)) {
          ok = false;
          break;
        }
        const uint32_t dA = smem_u32(sA + stage * C::A_STAGE);
        const uint32_t dB = smem_u32(sB + stage * C::B_STAGE);
        // pair modes: completion of both CTAs' copies is counted on the leader's barrier
        const uint32_t bar = PAIR ? mapa_shared(smem_u32(&full[stage]), 0)
                                  : smem_u32(&full[stage]);
        auto load_a = [&](uint32_t off, const CUtensorMap* map, int x, int y) {
          if (PAIR) {
            tma_load_2d_pair(dA + off, map, bar, x, y);
          } else {
            tma_load_2d(dA + off, map, &full[stage], x, y);
          }
        };
        auto load_b = [&](uint32_t off, const CUtensorMap* map, int x, int y) {
          if (PAIR) {
            tma_load_2d_pair(dB + off, map, bar, x, y);
          } else {
            tma_load_2d(dB + off, map, &full[stage], x, y);
          }
        };
        if (stall && issued == 0) {
          // test hook: leave stage 0 unfilled so that the MMA warp's bounded wait runs out
        } else {
          if (leader) mbar_arrive_expect_tx(&full[stage], PAIR ? 2 * C::STAGE_TX : C::STAGE_TX);
          boxes(t, kb, load_a, load_b);
        }
        ++issued;
        if (++stage == C::STAGES) {
          stage = 0;
          phase ^= 1u;
        }
      }
    }
  }
  if (ok && PAIR) {
    // Pair modes: the leader's MMAs release this CTA's stages by remote arrivals. Wait until
    // every stage has been released for the last time, so that none of them lands after this
    // CTA has left.
    for (int i = 0; i < C::STAGES; ++i) {
      if (!mbar_wait_bounded(&empty[stage], phase ^ 1u, abort_flag, a.hdr,
                             WHERE_GEMM_BASE + ROLE * 16 + 1))
        break;
      if (++stage == C::STAGES) {
        stage = 0;
        phase ^= 1u;
      }
    }
  }
  win.leave();
  if (!ok && leader) {
    // Aborted: let the copies already in flight land before the CTA exits (bounded). In the
    // pair modes the leader's barriers also count the peer's copies; the peer waits for the
    // leader at the final cluster barrier.
    const long long back = issued < C::STAGES ? issued : C::STAGES;
    for (long long i = 1; i <= back; ++i) {
      const long long it = issued - i;
      if (stall && it == 0) continue;
      const uint32_t s = static_cast<uint32_t>(it % C::STAGES);
      const uint32_t ph = static_cast<uint32_t>((it / C::STAGES) & 1);
      mbar_wait_drain(&full[s], ph, 100000000ull);
    }
  }
}

// ------------------------------------------------------------------------------------------
// MMA issuer: one thread (of the leader CTA in the pair modes)
// ------------------------------------------------------------------------------------------
// Roles and modes with one accumulator buffer: the exact-KL roles (policy and reference
// products in the two TMEM halves) and the wide pair mode (one 512-column tile).
template <int ROLE, int MODE>
struct OneBuf {
  static constexpr bool value = Dual<ROLE>::value || Cfg<MODE>::ACC_BUFS == 1;
};

template <int ROLE, int MODE>
__device__ void run_mma(const GemmArgs& a, const Dims& dm, const Sched<ROLE, MODE>& sc, uint8_t* sA,
                        uint8_t* sB, uint64_t* full, uint64_t* empty, uint64_t* accf,
                        uint64_t* acce, uint64_t* drain, uint32_t tmem_base,
                        volatile int* abort_flag) {
  using C = Cfg<MODE>;
  constexpr bool PAIR = C::PAIR;
  constexpr int NT = C::NT;
  if (PAIR && sc.rank != 0) return;
  constexpr bool A_MN = (ROLE == ROLE_DW);
  constexpr bool B_MN = (ROLE == ROLE_DH || ROLE == ROLE_DW);
  constexpr uint32_t idesc = idesc_bf16_f32(PAIR ? 2 * BM : BM, BN, A_MN, B_MN);
  uint32_t stage = 0, phase = 0, buf = 0, bphase = 0;
  bool ok = true;
  for (int u = sc.first; u < sc.num_units && ok; u += sc.step) {
    int m_load, n;
    bool m_ok;
    sc.decode(u, dm, m_load, n, m_ok);
    const int nacc = acc_tiles_of_unit<ROLE>(a, n);
    for (int t = 0; t < nacc && ok; ++t) {
      if (!mbar_wait_bounded(&acce[buf], bphase ^ 1u, abort_flag, a.hdr,
                             WHERE_GEMM_BASE + ROLE * 16 + 2)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t d_tmem = tmem_base + buf * BN;
      const int nk = Dual<ROLE>::value ? dm.num_kb / 2 : dm.num_kb;
      for (int kb = 0; kb < dm.num_kb; ++kb) {
        if (!mbar_wait_bounded(&full[stage], phase, abort_flag, a.hdr,
                               WHERE_GEMM_BASE + ROLE * 16 + 3)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t a0 = smem_u32(sA + stage * C::A_STAGE);
        const uint32_t b0 = smem_u32(sB + stage * C::B_STAGE);
        // dual roles: the reference product goes to the other TMEM half, accumulating afresh
        const bool second = Dual<ROLE>::value && kb >= nk;
        const uint32_t dst = second ? d_tmem + BN : d_tmem;
        const int kr = second ? kb - nk : kb;
#pragma unroll
        for (int k = 0; k < BK / 16; ++k) {
          const uint64_t ad = A_MN ? sdesc_sw128(a0 + k * 2048, BOX_MN, 1024)
                                   : sdesc_sw128(a0 + k * 32, 16, 1024);
#pragma unroll
          for (int h = 0; h < NT; ++h) {   // wide pair: column halves 0-255 and 256-511
            const uint32_t bh = b0 + h * C::B_HALF_STAGE;
            const uint64_t bd = B_MN ? sdesc_sw128(bh + k * 2048, BOX_MN, 1024)
                                     : sdesc_sw128(bh + k * 32, 16, 1024);
            if (PAIR) {
              umma_bf16_pair(dst + h * BN, ad, bd, idesc, (kr | k) != 0 ? 1u : 0u);
            } else {
              umma_bf16(dst, ad, bd, idesc, (kr | k) != 0 ? 1u : 0u);
            }
          }
        }
        // frees the smem stage once these MMAs have read it (pair modes: in both CTAs)
        if (PAIR) {
          umma_commit_pair(&empty[stage], 0x3);
        } else {
          umma_commit(&empty[stage]);
        }
        if (++stage == C::STAGES) {
          stage = 0;
          phase ^= 1u;
        }
      }
      if (!ok) break;
      if (PAIR) {                      // accumulator ready for both CTAs' epilogues
        umma_commit_pair(&accf[buf], 0x3);
      } else {
        umma_commit(&accf[buf]);
      }
      if (OneBuf<ROLE, MODE>::value) {  // one buffer spanning all of TMEM
        bphase ^= 1u;
      } else {
        buf ^= 1u;
        if (buf == 0) bphase ^= 1u;
      }
    }
  }
  // Make sure no MMA is still writing tensor memory when it is released.
  if (PAIR) {
    umma_commit_pair(drain, 0x1);
  } else {
    umma_commit(drain);
  }
  mbar_wait_drain(drain, 0, 200000000ull);
}

// ------------------------------------------------------------------------------------------
// epilogues: warps 2..5, thread = one accumulator row (TMEM lane)
// ------------------------------------------------------------------------------------------
#ifndef GRPO_EPI_SLEEP_NS
#define GRPO_EPI_SLEEP_NS 20000
#endif
// Epilogue warps wait for a whole tile's MMAs (tens of microseconds to milliseconds): they sleep
// in hardware between checks rather than keep four schedulers busy polling.
__device__ __forceinline__ bool epi_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                         WsHeader* hdr, int32_t where) {
  const bool ok = mbar_wait_bounded(bar, parity, abort_flag, hdr, where, GRPO_EPI_SLEEP_NS);
  return __all_sync(0xffffffffu, ok);
}

// Tells the MMA issuer that this warp has read accumulator `bar`'s buffer; in the pair modes
// the barrier lives in the leader CTA and counts the epilogue warps of both CTAs.
template <int MODE>
__device__ __forceinline__ void epi_release(uint64_t* bar, int lane, int rank) {
  constexpr bool PAIR = Cfg<MODE>::PAIR;
  tc_fence_before();
  __syncwarp();
  if (lane == 0) {
    if (PAIR && rank != 0) {
      mbar_arrive_cluster(mapa_shared(smem_u32(bar), 0));
    } else {
      mbar_arrive(bar);
    }
  }
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 p = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&p);
}

// Next accumulator buffer and the parity of its barriers.
template <int ROLE, int MODE>
__device__ __forceinline__ void advance_buf(uint32_t& buf, uint32_t& bphase) {
  if (OneBuf<ROLE, MODE>::value) {
    bphase ^= 1u;
  } else {
    buf ^= 1u;
    if (buf == 0) bphase ^= 1u;
  }
}

template <int ROLE, int MODE>
__device__ void run_epilogue_tiles(const GemmArgs& a, const Dims& dm, const Sched<ROLE, MODE>& sc,
                                   uint64_t* accf, uint64_t* acce, uint32_t tmem_base,
                                   volatile int* abort_flag, uint8_t* s_out,
                                   const CUtensorMap* map_out) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int q = warp & 3;               // TMEM lane quadrant this warp may access
  const int r = q * 32 + lane;          // accumulator row of this thread
  const uint32_t t_row = tmem_base + (static_cast<uint32_t>(q * 32) << 16);
  const int32_t where = WHERE_GEMM_BASE + ROLE * 16 + 4;
  constexpr int NT = Cfg<MODE>::NT;   // 256-column halves of the accumulator tile
  // columns of the accumulator tile this warp reads: all of them with 4 epilogue warps, one
  // 256-column half (h = 0 for warps 2-5, 1 for warps 6-9) with 8
  constexpr int CW = NT * BN / (Cfg<MODE>::EPI_WARPS / 4);
  const int h = (warp - 2) / 4;
  const int col0 = h * CW;
  uint32_t buf = 0, bphase = 0;
  uint32_t ob = 0;                    // dz staging buffer this warp fills next (TMA-store path)
  for (int u = sc.first; u < sc.num_units; u += sc.step) {
    int m_load, n;
    bool m_ok;   // this CTA stores the tile (false: a pair's second CTA past the last tile)
    sc.decode(u, dm, m_load, n, m_ok);

    if (ROLE == ROLE_FWD) {
      const int prow = a.row_pos[static_cast<long long>(m_load) * BM + r];  // position or -1
      const bool rv = m_ok && prow >= 0;
      const long long pos = rv ? prow : 0;
      // sampled token as a column of this W (a vocabulary shard's rows start at v_offset)
      const int y = (rv && a.mask[pos] != 0) ? a.tokens[pos] - a.v_offset : -1;
      float rm = -INFINITY, rs = 0.f, ru = 0.f, zyv = 0.f;
      int ri = 0;
      bool found = false;
      const int nacc = acc_tiles_of_unit<ROLE>(a, n);
      for (int t = 0; t < nacc; ++t) {
        if (!epi_wait(&accf[buf], bphase, abort_flag, a.hdr, where)) return;
        tc_fence_after();
        const int vbase = (n * NT * kFwdTilesPerStrip + t) * BN + col0;
        for (int c = 0; c < CW / 32; ++c) {
          const int v0 = vbase + c * 32;
          if (v0 >= a.V) break;  // uniform across the warp
          float x[32];
          tmem_load_32cols(t_row + buf * BN + col0 + c * 32, x);
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
            const float scl = ex2_approx((rm - cm) * kLog2e);
            rs *= scl;
            ru *= scl;
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
        epi_release<MODE>(&acce[buf], lane, sc.rank);
        advance_buf<ROLE, MODE>(buf, bphase);
      }
      const int strip = n * NT + h;   // this warp's strip of vocabulary columns
      if (m_ok && strip < a.num_strips)
        a.partials[static_cast<long long>(strip) * a.rows_cap +
                   static_cast<long long>(m_load) * BM + r] =
            make_float4(rm, rs, ru, __int_as_float(ri));
      if (found) a.zy[pos] = zyv;

    } else if (ROLE == ROLE_FWD_KL) {
      // policy z in columns 0-255, reference z_ref in 256-511 of the one buffer
      const int prow = a.row_pos[static_cast<long long>(m_load) * BM + r];  // position or -1
      const bool rv = m_ok && prow >= 0;
      const long long pos = rv ? prow : 0;
      const int y = (rv && a.mask[pos] != 0) ? a.tokens[pos] : -1;
      float rm = -INFINITY, rs = 0.f, ru = 0.f, rc = 0.f, zyv = 0.f;
      float qm = -INFINITY, qs = 0.f;
      int ri = 0;
      bool found = false;
      const int nacc = acc_tiles_of_unit<ROLE>(a, n);
      for (int t = 0; t < nacc; ++t) {
        if (!epi_wait(&accf[0], bphase, abort_flag, a.hdr, where)) return;
        tc_fence_after();
        const int vbase = (n * kFwdTilesPerStrip + t) * BN;
        for (int c = 0; c < BN / 32; ++c) {
          const int v0 = vbase + c * 32;
          if (v0 >= a.V) break;
          float x[32], xr[32];
          tmem_load_32cols(t_row + c * 32, x);
          tmem_load_32cols(t_row + BN + c * 32, xr);
          const int nvalid = a.V - v0;
          if (nvalid < 32) {
#pragma unroll
            for (int j = 0; j < 32; ++j)
              if (j >= nvalid) {
                x[j] = -1.0e30f;
                xr[j] = -1.0e30f;
              }
          }
          float cm = x[0], cq = xr[0];
          int ci = 0;
#pragma unroll
          for (int j = 1; j < 32; ++j) {
            if (x[j] > cm) {
              cm = x[j];
              ci = j;
            }
            cq = fmaxf(cq, xr[j]);
          }
          if (cm > rm) {
            const float scl = ex2_approx((rm - cm) * kLog2e);
            rs *= scl;
            ru *= scl;
            rc *= scl;
            rm = cm;
            ri = v0 + ci;
          }
          if (cq > qm) {
            qs *= ex2_approx((qm - cq) * kLog2e);
            qm = cq;
          }
          const float ml = rm * kLog2e, ql = qm * kLog2e;
          float ps = 0.f, pu = 0.f, pc = 0.f, qq = 0.f;
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            const float e = ex2_approx(fmaf(x[j], kLog2e, -ml));
            ps += e;
            pu = fmaf(e, x[j], pu);
            pc = fmaf(e, xr[j], pc);
            qq += ex2_approx(fmaf(xr[j], kLog2e, -ql));
          }
          rs += ps;
          ru += pu;
          rc += pc;
          qs += qq;
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
        epi_release<MODE>(&acce[0], lane, sc.rank);
        bphase ^= 1u;
      }
      if (m_ok) {
        const long long at = static_cast<long long>(n) * a.rows_cap +
                             static_cast<long long>(m_load) * BM + r;
        a.partials[at] = make_float4(rm, rs, ru, __int_as_float(ri));
        a.partials2[at] = make_float4(rc, qm, qs, 0.f);
      }
      if (found) a.zy[pos] = zyv;

    } else if (ROLE == ROLE_DZ_KL) {
      // dz = g (onehot - p) + c p (log p - log q - KL), p from z, q from z_ref
      const int prow = a.row_pos[static_cast<long long>(m_load) * BM + r];  // position or -1
      const bool rv = m_ok && prow >= 0;
      const long long pos = rv ? prow : 0;
      const bool act = rv && a.mask[pos] != 0;
      const float gt = act ? a.g[pos] : 0.f;
      const float ct = act ? a.c[pos] : 0.f;
      const float lse = act ? a.lse[pos] : 0.f;
      const float lser = act ? a.lse_ref[pos] : 0.f;
      const float klt = act ? a.kl[pos] : 0.f;
      const int y = act ? a.tokens[pos] : -1;
      if (!epi_wait(&accf[0], bphase, abort_flag, a.hdr, where)) return;
      tc_fence_after();
      __nv_bfloat16* dst_row =
          a.dz + (static_cast<size_t>(m_load) * BM + r) * static_cast<size_t>(a.dz_pitch);
      for (int c = 0; c < BN / 32; ++c) {
        const int vloc = n * BN + c * 32;
        const int v0 = a.vc0 + vloc;
        float x[32], xr[32];
        tmem_load_32cols(t_row + c * 32, x);
        tmem_load_32cols(t_row + BN + c * 32, xr);
        if (!m_ok) continue;
        uint32_t pk[16];
        if (act) {
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            float dv[2];
#pragma unroll
            for (int e = 0; e < 2; ++e) {
              const int v = v0 + 2 * j + e;
              const float lp = x[2 * j + e] - lse;              // log p
              const float p = ex2_approx(lp * kLog2e);
              const float lq = xr[2 * j + e] - lser;            // log q
              const float val = gt * ((v == y ? 1.f : 0.f) - p) + ct * p * (lp - lq - klt);
              dv[e] = v < a.V ? val : 0.f;
            }
            pk[j] = pack_bf16x2(dv[0], dv[1]);
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
      epi_release<MODE>(&acce[0], lane, sc.rank);
      bphase ^= 1u;

    } else if (ROLE == ROLE_DZ) {
      const int prow = a.row_pos[static_cast<long long>(m_load) * BM + r];  // position or -1
      const bool rv = m_ok && prow >= 0;
      const long long pos = rv ? prow : 0;
      const bool act = rv && a.mask[pos] != 0;
      const float gt = act ? a.g[pos] : 0.f;
      const float ll = act ? a.lse[pos] * kLog2e : 0.f;
      const int y = act ? a.tokens[pos] - a.v_offset : -1;
      if (!epi_wait(&accf[buf], bphase, abort_flag, a.hdr, where)) return;
      tc_fence_after();
      // dz of 32 consecutive columns of this row, bf16 pairs, from accumulator columns c*32..
      // (c counts 32-column chunks from this warp's first column)
      auto dz_chunk = [&](int c, uint32_t (&pk)[16]) {
        const int v0 = a.vc0 + n * NT * BN + col0 + c * 32;
        float x[32];
        tmem_load_32cols(t_row + buf * BN + col0 + c * 32, x);
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
      };
      if constexpr (OutStage<ROLE, MODE>::on) {
        // 64 columns at a time: the warp's 32 rows go to a 4 KB staging buffer (row = lane,
        // 16-byte chunk j stored at chunk j ^ (row % 8): the 128-byte swizzle of the store's
        // tensor map), then one TMA store writes them as full 128-byte row segments.
        for (int c2 = 0; c2 < BN / 64; ++c2) {
          uint32_t lo[16], hi[16];
          dz_chunk(2 * c2, lo);
          dz_chunk(2 * c2 + 1, hi);
          uint8_t* stage = s_out + (q * 2 + ob) * OutStage<ROLE, MODE>::BUF;
          if (lane == 0) bulk_wait_group_read<1>();   // this buffer's previous store has read it
          __syncwarp();
          uint8_t* row = stage + lane * 128;
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const uint32_t* p = j < 4 ? &lo[4 * j] : &hi[4 * (j - 4)];
            *reinterpret_cast<uint4*>(row + ((j ^ (lane & 7)) << 4)) =
                make_uint4(p[0], p[1], p[2], p[3]);
          }
          fence_proxy_async_smem();   // make the writes visible to the TMA engine
          __syncwarp();
          if (lane == 0 && m_ok) {
            tma_store_2d(map_out, smem_u32(stage), n * BN + c2 * 64, m_load * BM + q * 32);
            bulk_commit_group();
          }
          ob ^= 1u;
        }
      } else {
        __nv_bfloat16* dst_row =
            a.dz + (static_cast<size_t>(m_load) * BM + r) * static_cast<size_t>(a.dz_pitch);
        for (int c = 0; c < CW / 32; ++c) {
          const int vloc = n * NT * BN + col0 + c * 32;
          uint32_t pk[16];
          dz_chunk(c, pk);
          // a wide unit's second tile may lie past the scratch row (odd tile count)
          if (!m_ok || vloc >= a.dz_pitch) continue;
          uint4* dst = reinterpret_cast<uint4*>(dst_row + vloc);
#pragma unroll
          for (int j = 0; j < 4; ++j)
            dst[j] = make_uint4(pk[4 * j], pk[4 * j + 1], pk[4 * j + 2], pk[4 * j + 3]);
        }
      }
      epi_release<MODE>(&acce[buf], lane, sc.rank);
      advance_buf<ROLE, MODE>(buf, bphase);

    } else if (ROLE == ROLE_DH) {
      const int prow = a.row_pos[static_cast<long long>(m_load) * BM + r];  // position or -1
      const bool rv = m_ok && prow >= 0;
      const long long pos = rv ? prow : 0;
      if (!epi_wait(&accf[buf], bphase, abort_flag, a.hdr, where)) return;
      tc_fence_after();
      for (int c = 0; c < CW / 32; ++c) {
        const int col = n * NT * BN + col0 + c * 32;
        float x[32];
        tmem_load_32cols(t_row + buf * BN + col0 + c * 32, x);
        if (!rv || col >= a.d) continue;   // columns past d (a partial last tile) hold zeros
        float* acc_row = a.dH_acc + (static_cast<size_t>(m_load) * BM + r) * a.d + col;
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
        } else if (a.dh_f32) {
          float4* dst = reinterpret_cast<float4*>(reinterpret_cast<float*>(a.dH) + pos * a.d + col);
#pragma unroll
          for (int j = 0; j < 8; ++j)
            dst[j] = make_float4(x[4 * j], x[4 * j + 1], x[4 * j + 2], x[4 * j + 3]);
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
      epi_release<MODE>(&acce[buf], lane, sc.rank);
      advance_buf<ROLE, MODE>(buf, bphase);

    } else {  // ROLE_DW
      const int vrow = m_load * BM + r;
      const bool rv = m_ok && vrow < a.vc_len;
      // No scored token at all (K = 0): no MMA ran, the accumulator holds nothing -> dW = 0.
      const bool empty_k = dm.num_kb == 0;
      if (!epi_wait(&accf[buf], bphase, abort_flag, a.hdr, where)) return;
      tc_fence_after();
      float* dst_row = a.dW + static_cast<size_t>(a.vc0 + vrow) * a.d + n * NT * BN + col0;
      for (int c = 0; c < CW / 32; ++c) {
        float x[32];
        tmem_load_32cols(t_row + buf * BN + col0 + c * 32, x);
        if (!rv || n * NT * BN + col0 + c * 32 >= a.d) continue;   // columns past d
        if (empty_k) {
#pragma unroll
          for (int j = 0; j < 32; ++j) x[j] = 0.f;
        }
        float4* dst = reinterpret_cast<float4*>(dst_row + c * 32);
#pragma unroll
        for (int j = 0; j < 8; ++j)
          dst[j] = make_float4(x[4 * j], x[4 * j + 1], x[4 * j + 2], x[4 * j + 3]);
      }
      epi_release<MODE>(&acce[buf], lane, sc.rank);
      advance_buf<ROLE, MODE>(buf, bphase);
    }
  }
}

template <int ROLE, int MODE>
__device__ void run_epilogue(const GemmArgs& a, const Dims& dm, const Sched<ROLE, MODE>& sc,
                             uint64_t* accf, uint64_t* acce, uint32_t tmem_base,
                             volatile int* abort_flag, uint8_t* s_out,
                             const CUtensorMap* map_out) {
  run_epilogue_tiles<ROLE, MODE>(a, dm, sc, accf, acce, tmem_base, abort_flag, s_out, map_out);
  // TMA-store path: the issuing lane's stores must have written global memory (and finished
  // reading the staging buffers) before the CTA leaves
  if (OutStage<ROLE, MODE>::on && (threadIdx.x & 31) == 0) bulk_wait_group_all();
}

// ------------------------------------------------------------------------------------------
// kernel body (every tile mode) and one kernel per mode
// ------------------------------------------------------------------------------------------
template <int ROLE, int MODE>
__device__ __forceinline__ void gemm_body(const CUtensorMap* mapA, const CUtensorMap* mapB,
                                          const CUtensorMap* mapA2, const CUtensorMap* mapB2,
                                          const GemmArgs& args) {
  using C = Cfg<MODE>;
  constexpr bool PAIR = C::PAIR;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + C::STAGES * C::A_STAGE;
  uint8_t* sOut = sB + C::STAGES * C::B_STAGE;   // dz staging (OutStage), 1024-byte aligned
  uint64_t* bars = reinterpret_cast<uint64_t*>(sOut + OutStage<ROLE, MODE>::BYTES);
  uint64_t* full = bars;
  uint64_t* empty = bars + C::STAGES;
  uint64_t* accf = bars + 2 * C::STAGES;
  uint64_t* acce = accf + 2;
  uint64_t* drain = acce + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&accf[b], 1);
      mbar_init(&acce[b], (PAIR ? 2 : 1) * C::EPI_WARPS);  // epilogue warps of one or both CTAs
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_barrier_init();
    fence_proxy_async_smem();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(mapA);
    tma_prefetch_desc(mapB);
    if (Dual<ROLE>::value) {
      tma_prefetch_desc(mapA2);
      tma_prefetch_desc(mapB2);
    }
    if (OutStage<ROLE, MODE>::on) tma_prefetch_desc(mapA2);   // the dz store map
  }
  if (warp == 1) {
    if (PAIR) {
      tmem_alloc_pair(tmem_slot, TMEM_COLS);
      tmem_relinquish_pair();
    } else {
      tmem_alloc(tmem_slot, TMEM_COLS);
      tmem_relinquish();
    }
  }
  tc_fence_before();
  if (PAIR) {
    cluster_sync_all();  // barriers of both CTAs initialised before any cross-CTA traffic
  } else {
    __syncthreads();
  }
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const Dims dm = role_dims<ROLE>(args, args.hdr->num_tiles);
  const Sched<ROLE, MODE> sc(dm);

  if (warp == 0) {
    if (lane == 0)
      run_producer<ROLE, MODE>(mapA, mapB, mapA2, mapB2, args, dm, sc, sA, sB, full, empty,
                               abort_flag);
  } else if (warp == 1) {
    if (lane == 0)
      run_mma<ROLE, MODE>(args, dm, sc, sA, sB, full, empty, accf, acce, drain, tmem_base,
                          abort_flag);
  } else {
    run_epilogue<ROLE, MODE>(args, dm, sc, accf, acce, tmem_base, abort_flag, sOut, mapA2);
  }
  __syncwarp();
  tc_fence_before();
  if (PAIR) {
    cluster_sync_all();  // no CTA leaves while its peer may still signal or write into it
  } else {
    __syncthreads();
  }
  tc_fence_after();
  if (warp == 1) {
    if (PAIR) {
      tmem_dealloc_pair(tmem_base, TMEM_COLS);
    } else {
      tmem_dealloc(tmem_base, TMEM_COLS);
    }
  }
}

template <int ROLE>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    tc_gemm(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapB,
            const __grid_constant__ CUtensorMap mapA2, const __grid_constant__ CUtensorMap mapB2,
            const __grid_constant__ GemmArgs args) {
  gemm_body<ROLE, 0>(&mapA, &mapB, &mapA2, &mapB2, args);
}

// MODE 1 (256 x 256 tiles) or 2 (256 x 512 tiles) on CTA pairs.
template <int ROLE, int MODE>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(Cfg<MODE>::THREADS, 1)
    tc_gemm_pair(const __grid_constant__ CUtensorMap mapA,
                 const __grid_constant__ CUtensorMap mapB, const __grid_constant__ GemmArgs args) {
  gemm_body<ROLE, MODE>(&mapA, &mapB, &mapA, &mapB, args);
}

template <class Kernel, class... Args>
cudaError_t launch_with_smem(Kernel kernel, size_t smem, int grid, int threads, cudaStream_t st,
                             Args&&... args) {
  cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  kernel<<<grid, threads, smem, st>>>(args...);
  return cudaGetLastError();
}

template <int ROLE>
cudaError_t launch_role(const CUtensorMap& mapA, const CUtensorMap& mapB, const GemmArgs& args,
                        int grid, int mode, cudaStream_t st, const CUtensorMap& mapA2,
                        const CUtensorMap& mapB2) {
  if constexpr (!Dual<ROLE>::value) {       // exact-KL roles: single-CTA tiles only
    if (mode == 1)
      return launch_with_smem(tc_gemm_pair<ROLE, 1>, smem_bytes<ROLE, 1>(), grid,
                              Cfg<1>::THREADS, st, mapA, mapB, args);
    // wide pair: a forward unit is two 256-column strips (one-tile strips only)
    if constexpr (ROLE != ROLE_FWD || kFwdTilesPerStrip == 1) {
      if (mode == 2)
        return launch_with_smem(tc_gemm_pair<ROLE, 2>, smem_bytes<ROLE, 2>(), grid,
                                Cfg<2>::THREADS, st, mapA, mapB, args);
    }
  }
  if (mode != 0) return cudaErrorInvalidValue;
  return launch_with_smem(tc_gemm<ROLE>, smem_bytes<ROLE, 0>(), grid, Cfg<0>::THREADS, st, mapA,
                          mapB, mapA2, mapB2, args);
}

}  // namespace

size_t gemm_smem_bytes() { return SMEM_BYTES; }

int gemm_cluster_size(int tile_mode) { return tile_mode != 0 ? 2 : 1; }

int gemm_col_tiles_per_unit(int tile_mode) { return tile_mode == 2 ? 2 : 1; }

int gemm_b_box_rows(int tile_mode) { return tile_mode == 0 ? BN : BN / 2; }

namespace {
template <typename Kernel>
int query_active_clusters(Kernel kernel, size_t smem, int cl, int threads) {
  if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(smem)) != cudaSuccess)
    return 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(cl), 1, 1);
  cfg.blockDim = dim3(static_cast<unsigned>(threads), 1, 1);
  cfg.dynamicSmemBytes = smem;
  int n = 0;   // the kernels fix their cluster shape at compile time: no attribute here
  if (cudaOccupancyMaxActiveClusters(&n, reinterpret_cast<const void*>(kernel), &cfg) !=
      cudaSuccess) {
    (void)cudaGetLastError();
    return 0;
  }
  return n;
}

constexpr int kMaxDevices = 64;
std::atomic<int> g_active_clusters[kMaxDevices][3];   // 0 = not queried yet
}  // namespace

int gemm_max_clusters(int tile_mode) {
  const int cl = gemm_cluster_size(tile_mode);
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return 1;
  int cap = sms / cl > 0 ? sms / cl : 1;
  if (cl == 1 || dev < 0 || dev >= kMaxDevices || tile_mode < 0 || tile_mode > 2) return cap;
  int known = g_active_clusters[dev][tile_mode].load();
  if (known == 0) {
    int n = 0;
    if (tile_mode == 1)
      n = query_active_clusters(tc_gemm_pair<ROLE_FWD, 1>, Cfg<1>::SMEM, cl, Cfg<1>::THREADS);
    if (tile_mode == 2)
      n = query_active_clusters(tc_gemm_pair<ROLE_DW, 2>, Cfg<2>::SMEM, cl, Cfg<2>::THREADS);
    known = n > 0 ? n : cap;   // a failed query falls back to one cluster per `cl` SMs
    g_active_clusters[dev][tile_mode].store(known);
  }
  return known < cap ? known : cap;
}

int gemm_grid(long long row_tiles, long long col_tiles, int tile_mode) {
  const long long cl = gemm_cluster_size(tile_mode);
  const long long nt = gemm_col_tiles_per_unit(tile_mode);
  const long long cap = gemm_max_clusters(tile_mode);
  const long long units = ((row_tiles + cl - 1) / cl) * ((col_tiles + nt - 1) / nt);
  return static_cast<int>(cl * (units < cap ? (units > 0 ? units : 1) : cap));
}

cudaError_t launch_gemm(int role, const CUtensorMap& mapA, const CUtensorMap& mapB,
                        const GemmArgs& args, int grid, int mode, cudaStream_t st,
                        const CUtensorMap* mapA2, const CUtensorMap* mapB2) {
  const CUtensorMap& a2 = mapA2 ? *mapA2 : mapA;
  const CUtensorMap& b2 = mapB2 ? *mapB2 : mapB;
  switch (role) {
    case ROLE_FWD: return launch_role<ROLE_FWD>(mapA, mapB, args, grid, mode, st, a2, b2);
    case ROLE_DZ:   // single-CTA tiles store dz through mapA2 (the dz scratch, 64 x 32 boxes)
      if (mode == 0 && !mapA2) return cudaErrorInvalidValue;
      return launch_role<ROLE_DZ>(mapA, mapB, args, grid, mode, st, a2, b2);
    case ROLE_DH: return launch_role<ROLE_DH>(mapA, mapB, args, grid, mode, st, a2, b2);
    case ROLE_DW: return launch_role<ROLE_DW>(mapA, mapB, args, grid, mode, st, a2, b2);
    case ROLE_FWD_KL:
      if (!mapA2 || !mapB2 || mode != 0) return cudaErrorInvalidValue;
      return launch_role<ROLE_FWD_KL>(mapA, mapB, args, grid, 0, st, a2, b2);
    case ROLE_DZ_KL:
      if (!mapA2 || !mapB2 || mode != 0) return cudaErrorInvalidValue;
      return launch_role<ROLE_DZ_KL>(mapA, mapB, args, grid, 0, st, a2, b2);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace grpo
