// Reduction and bookkeeping kernels of the GRPO path, plus the f32 CUDA-core path for small
// problems: valid-token counts and the packed token rows, group-relative advantages (Eq. 1's
// w(x): rewards normalised within each group, Alg. 1), the merge of per-strip softmax statistics into
// logp / lse / entropy / argmax, and the per-token clipped surrogate + KL loss with its
// coefficient g_t = dL/dlogp_t (Sec. 6.1, Eq. 1). All reductions use a fixed order, so results
// are bitwise reproducible run to run.
#include <cfloat>
#include <cmath>

#include "common.cuh"
#include "internal.h"

namespace grpo {

namespace {

constexpr unsigned kFull = 0xffffffffu;

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
  return v;
}

// ------------------------------------------------------------------------------------------
// Valid counts n_i of every sequence (one warp per sequence).
// ------------------------------------------------------------------------------------------
__global__ void k_mask_scan(const uint8_t* __restrict__ mask, int S, int T,
                            int32_t* __restrict__ counts) {
  const int warps = blockDim.x / 32;
  const int i = blockIdx.x * warps + threadIdx.x / 32;
  const int lane = threadIdx.x & 31;
  if (i >= S) return;
  const uint8_t* row = mask + static_cast<size_t>(i) * T;
  int cnt = 0;
  for (int t = lane; t < T; t += 32) cnt += (row[t] != 0);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) cnt += __shfl_xor_sync(kFull, cnt, o);
  if (lane == 0) counts[i] = cnt;
}

// ------------------------------------------------------------------------------------------
// Token packing. The scored tokens of all sequences, in order, become consecutive "packed rows"
// (sequence i's tokens start at seq_base[i] = n_0 + ... + n_{i-1}); the GEMMs run 128-row tiles
// over packed rows, so no tile row is spent on padding or on masked (tool-result) tokens.
// k_seq_scan: exclusive prefix of the counts (one block of 1024, chunks of 1024 carried), total
// and tile count into the header, and row_pos = -1 for the padding rows of the last tile.
// ------------------------------------------------------------------------------------------
__global__ void k_seq_scan(const int32_t* __restrict__ counts, int S, long long rows_cap,
                           int32_t* __restrict__ seq_base, int32_t* __restrict__ row_pos,
                           WsHeader* hdr) {
  __shared__ long long warp_tot[32];
  __shared__ long long carry;
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  if (tid == 0) carry = 0;
  __syncthreads();
  for (int base = 0; base < S; base += 1024) {
    const int i = base + tid;
    const long long n = (i < S) ? counts[i] : 0;
    long long x = n;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const long long y = __shfl_up_sync(kFull, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) warp_tot[wid] = x;
    __syncthreads();
    if (wid == 0) {
      const long long w = warp_tot[lane];
      long long xs = w;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const long long y = __shfl_up_sync(kFull, xs, o);
        if (lane >= o) xs += y;
      }
      warp_tot[lane] = xs - w;
    }
    __syncthreads();
    const long long excl = carry + warp_tot[wid] + x - n;
    if (i < S) seq_base[i] = static_cast<int32_t>(excl);
    __syncthreads();
    if (tid == 1023) carry = excl + n;
    __syncthreads();
  }
  const long long total = carry;
  const long long padded = (total + kTileRows - 1) / kTileRows * kTileRows;
  for (long long r = total + tid; r < padded && r < rows_cap; r += blockDim.x) row_pos[r] = -1;
  if (tid == 0) {
    seq_base[S] = static_cast<int32_t>(total);
    hdr->num_tiles = static_cast<int32_t>(padded / kTileRows);
    hdr->total_valid = total;
  }
}

// One block per sequence: ranks of the scored positions (block-wide scan over T), and the two
// maps packed row -> position (row_pos) and position -> packed row (pos_row, -1 if unscored).
constexpr int kPackThreads = 256;

__global__ void __launch_bounds__(kPackThreads)
    k_pack(const uint8_t* __restrict__ mask, int S, int T, const int32_t* __restrict__ seq_base,
           int32_t* __restrict__ row_pos, int32_t* __restrict__ pos_row) {
  __shared__ int warp_tot[kPackThreads / 32];
  const int i = blockIdx.x;
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  const int chunk = (T + kPackThreads - 1) / kPackThreads;
  const int t0 = min(T, tid * chunk), t1 = min(T, t0 + chunk);
  const size_t rowb = static_cast<size_t>(i) * T;
  int n = 0;
  for (int t = t0; t < t1; ++t) n += (mask[rowb + t] != 0);
  int x = n;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(kFull, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_tot[wid] = x;
  __syncthreads();
  if (wid == 0) {
    const int w = lane < kPackThreads / 32 ? warp_tot[lane] : 0;
    int xs = w;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(kFull, xs, o);
      if (lane >= o) xs += y;
    }
    if (lane < kPackThreads / 32) warp_tot[lane] = xs - w;
  }
  __syncthreads();
  int r = seq_base[i] + warp_tot[wid] + x - n;
  for (int t = t0; t < t1; ++t) {
    const size_t pos = rowb + t;
    if (mask[pos] != 0) {
      row_pos[r] = static_cast<int32_t>(pos);
      pos_row[pos] = r;
      ++r;
    } else {
      pos_row[pos] = -1;
    }
  }
}

// Hp[r, :] = H[row_pos[r], :] for the packed rows of the current batch (zero for padding rows).
__global__ void k_gather_rows(const uint4* __restrict__ H, int vec_per_row,
                              const int32_t* __restrict__ row_pos, const WsHeader* hdr,
                              uint4* __restrict__ Hp) {
  const long long rows = static_cast<long long>(hdr->num_tiles) * kTileRows;
  for (long long r = blockIdx.x; r < rows; r += gridDim.x) {
    const int pos = row_pos[r];
    uint4* dst = Hp + r * vec_per_row;
    if (pos >= 0) {
      const uint4* src = H + static_cast<long long>(pos) * vec_per_row;
      for (int k = threadIdx.x; k < vec_per_row; k += blockDim.x) dst[k] = src[k];
    } else {
      for (int k = threadIdx.x; k < vec_per_row; k += blockDim.x) dst[k] = make_uint4(0, 0, 0, 0);
    }
  }
}

// dH rows of unscored positions are zero (scored rows are written by the dH GEMM).
__global__ void k_dh_zero_masked(const uint8_t* __restrict__ mask, long long P, int vec_per_row,
                                 uint4* __restrict__ dH) {
  for (long long pos = blockIdx.x; pos < P; pos += gridDim.x) {
    if (mask[pos] != 0) continue;
    uint4* p = dH + pos * vec_per_row;
    for (int k = threadIdx.x; k < vec_per_row; k += blockDim.x) p[k] = make_uint4(0, 0, 0, 0);
  }
}

// ------------------------------------------------------------------------------------------
// Group advantages: one warp per group; mean and std in f32 with a fixed summation order.
// ------------------------------------------------------------------------------------------
__global__ void k_group_adv(const float* __restrict__ r, const int32_t* __restrict__ go,
                            int num_groups, int S, int std_mode, float std_eps,
                            float* __restrict__ adv, WsHeader* hdr) {
  const int g = blockIdx.x;
  const int lane = threadIdx.x;
  if (g >= num_groups) return;
  const int lo = go[g], hi = go[g + 1];
  bool bad = lo < 0 || hi < lo || hi > S;
  if (g == 0 && lo != 0) bad = true;
  if (g == num_groups - 1 && hi != S) bad = true;
  if (bad) {
    if (lane == 0) record_error(hdr, ST_GROUPS, WHERE_GROUP_OFFSETS);
    const int a = max(lo, 0), b = min(max(hi, a), S);
    for (int i = a + lane; i < b; i += 32) adv[i] = __int_as_float(0x7fc00000);
    return;
  }
  const int G = hi - lo;
  if (G <= 0) return;
  float s = 0.f;
  bool same = true;
  const float r0 = r[lo];
  for (int i = lo + lane; i < hi; i += 32) {
    const float v = r[i];
    s += v;
    same &= (__float_as_uint(v) == __float_as_uint(r0));
  }
  same = __all_sync(kFull, same);
  const float mu = warp_sum(s) / static_cast<float>(G);
  float q = 0.f;
  for (int i = lo + lane; i < hi; i += 32) {
    const float dv = r[i] - mu;
    q = fmaf(dv, dv, q);
  }
  q = warp_sum(q);
  const int dof = (std_mode == 0) ? G - 1 : G;
  const bool degenerate = (G == 1) || same;
  const float sigma = dof > 0 ? sqrtf(q / static_cast<float>(dof)) : 0.f;
  for (int i = lo + lane; i < hi; i += 32) {
    adv[i] = degenerate ? 0.f : (r[i] - mu) / (sigma + std_eps);
  }
}

// ------------------------------------------------------------------------------------------
// Merge of per-strip statistics (max m, sum s = sum e^{z-m}, u = sum e^{z-m} z, argmax) into
// lse, logp, entropy, argmax; one thread per position, one pass over the strips in vocabulary
// order with the running sums rescaled whenever the running maximum rises (so ties keep the
// lowest index).
// ------------------------------------------------------------------------------------------
struct StripMerge {
  float M = -INFINITY, S = 0.f, U = 0.f;
  int idx = 0;
  // Adds strip statistics p = (m, s, u, argmax bits); returns the factor e^{m - M} that scales
  // quantities summed with e^{z - m} weights into the running maximum's frame.
  __device__ __forceinline__ float add(const float4 p) {
    if (p.x > M) {
      const float r = ex2_approx((M - p.x) * kLog2e);   // 0 on the first strip (M = -inf)
      S = fmaf(S, r, p.y);
      U = fmaf(U, r, p.z);
      M = p.x;
      idx = __float_as_int(p.w);
      rescale = r;
      return 1.f;
    }
    const float sc = ex2_approx((p.x - M) * kLog2e);
    S = fmaf(p.y, sc, S);
    U = fmaf(p.z, sc, U);
    rescale = 1.f;
    return sc;
  }
  float rescale = 1.f;   // factor the running sums were multiplied by in the last add()
};

// Strips are read in batches of kMergeBatch independent loads before they are merged, in the
// same vocabulary order: each thread then keeps that many loads in flight, which is what keeps
// HBM busy when there are few positions (one load at a time leaves small batches latency bound).
constexpr int kMergeBatch = 8;

__device__ __forceinline__ void merge_strips(const float4* __restrict__ partials,
                                             long long rows_cap, int num_strips, long long row,
                                             StripMerge& mg) {
  int j = 0;
  for (; j + kMergeBatch <= num_strips; j += kMergeBatch) {
    float4 p[kMergeBatch];
#pragma unroll
    for (int k = 0; k < kMergeBatch; ++k)
      p[k] = partials[static_cast<long long>(j + k) * rows_cap + row];
#pragma unroll
    for (int k = 0; k < kMergeBatch; ++k) mg.add(p[k]);
  }
  for (; j < num_strips; ++j) mg.add(partials[static_cast<long long>(j) * rows_cap + row]);
}

__global__ void k_fwd_merge(const float4* __restrict__ partials, long long rows_cap,
                            int num_strips, const float* __restrict__ zy,
                            const int32_t* __restrict__ pos_row,
                            const int32_t* __restrict__ tokens, const uint8_t* __restrict__ mask,
                            int S, int T, int V, float* __restrict__ logp,
                            float* __restrict__ lse_out, float* __restrict__ entropy,
                            int32_t* __restrict__ argmax, WsHeader* hdr) {
  const long long pos = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (pos >= static_cast<long long>(S) * T) return;
  if (mask[pos] == 0) {
    logp[pos] = 0.f;
    lse_out[pos] = 0.f;
    entropy[pos] = 0.f;
    argmax[pos] = -1;
    return;
  }
  const long long row = pos_row[pos];   // packed row of this scored position
  StripMerge mg;
  merge_strips(partials, rows_cap, num_strips, row, mg);
  const float M = mg.M, Ssum = mg.S, U = mg.U;
  const int idx = mg.idx;
  const float lse = M + logf(Ssum);
  const int y = tokens[pos];
  float lp;
  if (y < 0 || y >= V) {
    record_error(hdr, ST_TOKEN_RANGE, WHERE_MERGE_TOKEN);
    lp = __int_as_float(0x7fc00000);
  } else {
    lp = zy[pos] - lse;
  }
  logp[pos] = lp;
  lse_out[pos] = lse;
  entropy[pos] = lse - U / Ssum;
  argmax[pos] = idx;
}

// Merge for the exact-KL forward: also combines sum e^{z-m} z_ref and the reference model's
// (m_ref, s_ref) into lse_ref and KL_t = E_p[z] - lse - E_p[z_ref] + lse_ref.
__global__ void k_fwd_merge_kl(const float4* __restrict__ partials,
                               const float4* __restrict__ partials2, long long rows_cap,
                               int num_strips, const float* __restrict__ zy,
                               const int32_t* __restrict__ pos_row,
                               const int32_t* __restrict__ tokens,
                               const uint8_t* __restrict__ mask, int S, int T, int V,
                               float* __restrict__ logp, float* __restrict__ lse_out,
                               float* __restrict__ entropy, int32_t* __restrict__ argmax,
                               float* __restrict__ lse_ref, float* __restrict__ kl,
                               WsHeader* hdr) {
  const long long pos = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (pos >= static_cast<long long>(S) * T) return;
  if (mask[pos] == 0) {
    logp[pos] = 0.f;
    lse_out[pos] = 0.f;
    entropy[pos] = 0.f;
    argmax[pos] = -1;
    lse_ref[pos] = 0.f;
    kl[pos] = 0.f;
    return;
  }
  const long long row = pos_row[pos];   // packed row of this scored position
  StripMerge mg;                        // policy: (m, s, u, argmax)
  float C = 0.f;                        // sum e^{z-M} z_ref in the policy's frame
  float Mr = -INFINITY, Sr = 0.f;       // reference: running max and sum e^{z_ref - Mr}
  auto add = [&](const float4 p, const float4 q) {
    const float sc = mg.add(p);
    C = fmaf(C, mg.rescale, q.x * sc);
    if (q.y > Mr) {
      Sr = fmaf(Sr, ex2_approx((Mr - q.y) * kLog2e), q.z);
      Mr = q.y;
    } else {
      Sr = fmaf(q.z, ex2_approx((q.y - Mr) * kLog2e), Sr);
    }
  };
  int j = 0;
  for (; j + kMergeBatch <= num_strips; j += kMergeBatch) {   // batched loads, as merge_strips
    float4 p[kMergeBatch], q[kMergeBatch];
#pragma unroll
    for (int k = 0; k < kMergeBatch; ++k) {
      p[k] = partials[static_cast<long long>(j + k) * rows_cap + row];
      q[k] = partials2[static_cast<long long>(j + k) * rows_cap + row];
    }
#pragma unroll
    for (int k = 0; k < kMergeBatch; ++k) add(p[k], q[k]);
  }
  for (; j < num_strips; ++j)
    add(partials[static_cast<long long>(j) * rows_cap + row],
        partials2[static_cast<long long>(j) * rows_cap + row]);
  const float M = mg.M, Ssum = mg.S, U = mg.U;
  const int idx = mg.idx;
  const float lse = M + logf(Ssum);
  const float lser = Mr + logf(Sr);
  const int y = tokens[pos];
  float lp;
  if (y < 0 || y >= V) {
    record_error(hdr, ST_TOKEN_RANGE, WHERE_MERGE_TOKEN);
    lp = __int_as_float(0x7fc00000);
  } else {
    lp = zy[pos] - lse;
  }
  logp[pos] = lp;
  lse_out[pos] = lse;
  entropy[pos] = lse - U / Ssum;
  argmax[pos] = idx;
  lse_ref[pos] = lser;
  kl[pos] = fmaxf(0.f, (U - C) / Ssum - lse + lser);   // >= 0; rounding can dip below 0
}

// ------------------------------------------------------------------------------------------
// Per-token loss terms and g_t = dL/dlogp_t; one block per sequence, fixed-order block sum.
// ------------------------------------------------------------------------------------------
constexpr int kLossThreads = 256;

__device__ __forceinline__ float block_sum_fixed(float v, float* sh) {
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  v = warp_sum(v);
  if (lane == 0) sh[wid] = v;
  __syncthreads();
  float tot = 0.f;
  if (tid == 0) {
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) tot += sh[w];
  }
  __syncthreads();
  return tot;  // valid in thread 0
}

// mode 0: GRPO clipped surrogate + KL (Sec. 6.1, Eq. 1); mode 1: distillation token
// cross-entropy l_t = -logp_t (Sec. 6.2).
__global__ void __launch_bounds__(kLossThreads)
    k_loss_tokens(const uint8_t* __restrict__ mask, const float* __restrict__ logp,
                  const float* __restrict__ old_logp, const float* __restrict__ ref_logp,
                  const float* __restrict__ adv, const int32_t* __restrict__ valid_count, int S,
                  int T, float eps_low, float eps_high, float beta, int agg, double norm,
                  int mode, const WsHeader* hdr, float* __restrict__ g,
                  float* __restrict__ seq_loss, const float* __restrict__ kl,
                  float* __restrict__ cvec) {
  __shared__ float sh[32];
  const int i = blockIdx.x;
  const float A = mode != 1 ? adv[i] : 0.f;
  const int n_i = valid_count[i];
  float w;
  if (agg == 0) {
    const double Sn = norm > 0 ? norm : static_cast<double>(S);
    w = n_i > 0 ? static_cast<float>(1.0 / (Sn * n_i)) : 0.f;
  } else {
    const double Nn = norm > 0 ? norm : static_cast<double>(hdr->total_valid);
    w = Nn > 0 ? static_cast<float>(1.0 / Nn) : 0.f;
  }
  const float lo = 1.f - eps_low, hi = 1.f + eps_high;
  float acc = 0.f;
  const size_t base = static_cast<size_t>(i) * T;
  for (int t = threadIdx.x; t < T; t += kLossThreads) {
    const size_t pos = base + t;
    float gt = 0.f;
    if (mask[pos] != 0 && mode == 1) {
      acc -= logp[pos];
      gt = -w;
    } else if (mask[pos] != 0) {
      const float lp = logp[pos];
      const float rho = expf(lp - old_logp[pos]);
      const float unclipped = rho * A;
      const float clipped = fminf(fmaxf(rho, lo), hi) * A;
      const float surr = fminf(unclipped, clipped);
      float ell = -surr;
      float dell = 0.f;
      const bool active = (A >= 0.f) ? (rho <= hi) : (rho >= lo);
      if (active) dell = -A * rho;
      if (mode == 2) {
        // exact KL (Eq. 1): its gradient enters dz directly with coefficient beta * w
        ell = fmaf(beta, kl[pos], ell);
        cvec[pos] = beta * w;
      } else if (beta != 0.f) {
        const float delta = ref_logp[pos] - lp;
        const float ed = expf(delta);
        ell = fmaf(beta, ed - delta - 1.f, ell);
        dell = fmaf(beta, 1.f - ed, dell);
      }
      acc += ell;
      gt = w * dell;
    } else if (mode == 2) {
      cvec[pos] = 0.f;
    }
    g[pos] = gt;
  }
  const float tot = block_sum_fixed(acc, sh);
  if (threadIdx.x == 0) seq_loss[i] = tot * w;
}

// Eqs. 2-4: r = r_perf + r_tools, r_perf = -2 (incorrect), -1 (correct, t > t_base),
// else min(10, t_base / t - 1); r_tools = lambda * used / avail (NaN if the counts are invalid).
__global__ void k_rewards(const uint8_t* __restrict__ correct, const float* __restrict__ t_base,
                          const float* __restrict__ t_new, const int32_t* __restrict__ used,
                          const int32_t* __restrict__ avail, int n, float lambda_tools,
                          float* __restrict__ r) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  float rp;
  if (correct[i] == 0) {
    rp = -2.f;
  } else if (t_new[i] > t_base[i]) {
    rp = -1.f;
  } else {
    rp = fminf(10.f, t_base[i] / t_new[i] - 1.f);
  }
  const int u = used[i], a = avail[i];
  const float rt = (a > 0 && u >= 0 && u <= a)
                       ? lambda_tools * static_cast<float>(u) / static_cast<float>(a)
                       : __int_as_float(0x7fc00000);
  r[i] = rp + rt;
}

__global__ void k_loss_final(const float* __restrict__ seq_loss, int S, float* loss_out) {
  __shared__ float sh[32];
  float acc = 0.f;
  for (int i = threadIdx.x; i < S; i += blockDim.x) acc += seq_loss[i];
  const float tot = block_sum_fixed(acc, sh);
  if (threadIdx.x == 0) *loss_out = tot;
}

// ------------------------------------------------------------------------------------------
// Vocabulary-parallel scoring: statistics of one shard per position, and the merge of the
// statistics of all shards.
// ------------------------------------------------------------------------------------------
__global__ void k_shard_stats(const float4* __restrict__ partials, long long rows_cap,
                              int num_strips, const float* __restrict__ zy_ws,
                              const int32_t* __restrict__ pos_row,
                              const int32_t* __restrict__ tokens,
                              const uint8_t* __restrict__ mask, int S, int T, int V_shard,
                              int v_offset, float4* __restrict__ stats,
                              float* __restrict__ zy_out) {
  const long long pos = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (pos >= static_cast<long long>(S) * T) return;
  if (mask[pos] == 0) {
    stats[pos] = make_float4(-INFINITY, 0.f, 0.f, __int_as_float(-1));
    zy_out[pos] = -INFINITY;
    return;
  }
  const long long row = pos_row[pos];   // packed row of this scored position
  StripMerge mg;
  merge_strips(partials, rows_cap, num_strips, row, mg);
  stats[pos] = make_float4(mg.M, mg.S, mg.U, __int_as_float(mg.idx + v_offset));
  const int yl = tokens[pos] - v_offset;
  zy_out[pos] = (yl >= 0 && yl < V_shard) ? zy_ws[pos] : -INFINITY;
}

__global__ void k_merge_shards(const float4* __restrict__ stats, const float* __restrict__ zy,
                               int P, const int32_t* __restrict__ tokens,
                               const uint8_t* __restrict__ mask, int S, int T, int V_total,
                               float* __restrict__ logp, float* __restrict__ lse_out,
                               float* __restrict__ entropy, int32_t* __restrict__ argmax,
                               WsHeader* hdr) {
  const long long n = static_cast<long long>(S) * T;
  const long long pos = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (pos >= n) return;
  if (mask[pos] == 0) {
    logp[pos] = 0.f;
    lse_out[pos] = 0.f;
    entropy[pos] = 0.f;
    argmax[pos] = -1;
    return;
  }
  float M = -INFINITY, zyv = -INFINITY;
  int idx = 0x7fffffff;
  for (int p = 0; p < P; ++p) {
    const float4 s = stats[p * n + pos];
    const int ip = __float_as_int(s.w);
    if (s.x > M || (s.x == M && ip < idx)) {  // lowest global index among the maxima
      M = s.x;
      idx = ip;
    }
    zyv = fmaxf(zyv, zy[p * n + pos]);
  }
  float Ssum = 0.f, U = 0.f;
  for (int p = 0; p < P; ++p) {
    const float4 s = stats[p * n + pos];
    const float sc = ex2_approx((s.x - M) * kLog2e);
    Ssum = fmaf(s.y, sc, Ssum);
    U = fmaf(s.z, sc, U);
  }
  const float lse = M + logf(Ssum);
  const int y = tokens[pos];
  float lp = zyv - lse;
  if (y < 0 || y >= V_total) {
    record_error(hdr, ST_TOKEN_RANGE, WHERE_MERGE_TOKEN);
    lp = __int_as_float(0x7fc00000);
  }
  logp[pos] = lp;
  lse_out[pos] = lse;
  entropy[pos] = lse - U / Ssum;
  argmax[pos] = idx;
}

// ------------------------------------------------------------------------------------------
// f32 path (CUDA cores, exact f32 arithmetic, small problems): one block per position.
// ------------------------------------------------------------------------------------------
constexpr int kF32Threads = 128;

struct SoftStat {
  float m, s, u, zy;
  int idx;
};

__global__ void __launch_bounds__(kF32Threads)
    k_f32_fwd(const float* __restrict__ H, const float* __restrict__ W,
              const int32_t* __restrict__ tokens, const uint8_t* __restrict__ mask, int S, int T,
              int d, int V, float* __restrict__ logp, float* __restrict__ lse_out,
              float* __restrict__ entropy, int32_t* __restrict__ argmax, WsHeader* hdr) {
  extern __shared__ float smem[];
  float* h = smem;                                  // [d]
  __shared__ float sm_m[kF32Threads], sm_s[kF32Threads], sm_u[kF32Threads];
  __shared__ int sm_i[kF32Threads];
  __shared__ float sm_zy;
  const long long pos = blockIdx.x;
  const int tid = threadIdx.x;
  if (mask[pos] == 0) {
    if (tid == 0) {
      logp[pos] = 0.f;
      lse_out[pos] = 0.f;
      entropy[pos] = 0.f;
      argmax[pos] = -1;
    }
    return;
  }
  for (int k = tid; k < d; k += kF32Threads) h[k] = H[pos * d + k];
  if (tid == 0) sm_zy = __int_as_float(0x7fc00000);
  __syncthreads();
  const int y = tokens[pos];
  float m = -INFINITY, s = 0.f, u = 0.f;
  int idx = 0x7fffffff;
  for (int v = tid; v < V; v += kF32Threads) {
    const float* wr = W + static_cast<size_t>(v) * d;
    float z = 0.f;
    for (int k = 0; k < d; ++k) z = fmaf(wr[k], h[k], z);
    if (v == y) sm_zy = z;
    if (z > m) {
      const float sc = expf(m - z);
      s *= sc;
      u *= sc;
      m = z;
      idx = v;
    }
    const float e = expf(z - m);
    s += e;
    u = fmaf(e, z, u);
  }
  sm_m[tid] = m;
  sm_s[tid] = s;
  sm_u[tid] = u;
  sm_i[tid] = idx;
  __syncthreads();
  if (tid == 0) {
    float M = -INFINITY;
    int I = 0x7fffffff;
    for (int j = 0; j < kF32Threads; ++j) {
      if (sm_m[j] > M || (sm_m[j] == M && sm_i[j] < I)) {
        M = sm_m[j];
        I = sm_i[j];
      }
    }
    float Ss = 0.f, U = 0.f;
    for (int j = 0; j < kF32Threads; ++j) {
      if (sm_m[j] == -INFINITY) continue;
      const float sc = expf(sm_m[j] - M);
      Ss = fmaf(sm_s[j], sc, Ss);
      U = fmaf(sm_u[j], sc, U);
    }
    const float l = M + logf(Ss);
    if (y < 0 || y >= V) {
      record_error(hdr, ST_TOKEN_RANGE, WHERE_MERGE_TOKEN);
    }
    logp[pos] = sm_zy - l;
    lse_out[pos] = l;
    entropy[pos] = l - U / Ss;
    argmax[pos] = I;
  }
}

constexpr int kF32VChunk = 2048;

__global__ void __launch_bounds__(kF32Threads)
    k_f32_dh(const float* __restrict__ H, const float* __restrict__ W,
             const int32_t* __restrict__ tokens, const uint8_t* __restrict__ mask,
             const float* __restrict__ lse, const float* __restrict__ g, int S, int T, int d,
             int V, float* __restrict__ dH) {
  extern __shared__ float smem[];
  float* h = smem;               // [d]
  float* dz = smem + d;          // [kF32VChunk]
  const long long pos = blockIdx.x;
  const int tid = threadIdx.x;
  float* out = dH + pos * d;
  if (mask[pos] == 0) {
    for (int k = tid; k < d; k += kF32Threads) out[k] = 0.f;
    return;
  }
  for (int k = tid; k < d; k += kF32Threads) h[k] = H[pos * d + k];
  const int y = tokens[pos];
  const float gt = g[pos], l = lse[pos];
  // each thread owns hidden indices k = tid, tid + 128, ...; at most 32 per thread here
  float acc[32];
#pragma unroll
  for (int j = 0; j < 32; ++j) acc[j] = 0.f;
  for (int v0 = 0; v0 < V; v0 += kF32VChunk) {
    const int v1 = min(V, v0 + kF32VChunk);
    __syncthreads();
    for (int v = v0 + tid; v < v1; v += kF32Threads) {
      const float* wr = W + static_cast<size_t>(v) * d;
      float z = 0.f;
      for (int k = 0; k < d; ++k) z = fmaf(wr[k], h[k], z);
      const float p = expf(z - l);
      dz[v - v0] = gt * ((v == y ? 1.f : 0.f) - p);
    }
    __syncthreads();
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      const int k = tid + j * kF32Threads;
      if (k < d) {
        float a = acc[j];
        for (int v = v0; v < v1; ++v) a = fmaf(dz[v - v0], W[static_cast<size_t>(v) * d + k], a);
        acc[j] = a;
      }
    }
  }
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    const int k = tid + j * kF32Threads;
    if (k < d) out[k] = acc[j];
  }
}

__global__ void __launch_bounds__(kF32Threads)
    k_f32_dw(const float* __restrict__ H, const float* __restrict__ W,
             const int32_t* __restrict__ tokens, const uint8_t* __restrict__ mask,
             const float* __restrict__ lse, const float* __restrict__ g, int S, int T, int d,
             int V, float* __restrict__ dW) {
  extern __shared__ float smem[];
  float* w = smem;                     // [d]
  __shared__ float dzc[kF32Threads];
  const int v = blockIdx.x;
  const int tid = threadIdx.x;
  for (int k = tid; k < d; k += kF32Threads) w[k] = W[static_cast<size_t>(v) * d + k];
  float acc[32];
#pragma unroll
  for (int j = 0; j < 32; ++j) acc[j] = 0.f;
  const long long P = static_cast<long long>(S) * T;
  for (long long p0 = 0; p0 < P; p0 += kF32Threads) {
    __syncthreads();
    const long long pos = p0 + tid;
    float dzv = 0.f;
    if (pos < P && mask[pos] != 0) {
      const float* hr = H + pos * d;
      float z = 0.f;
      for (int k = 0; k < d; ++k) z = fmaf(w[k], hr[k], z);
      const float pr = expf(z - lse[pos]);
      dzv = g[pos] * ((tokens[pos] == v ? 1.f : 0.f) - pr);
    }
    dzc[tid] = dzv;
    __syncthreads();
    const long long rem = P - p0;
    const int cnt = rem < kF32Threads ? static_cast<int>(rem) : kF32Threads;
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      const int k = tid + j * kF32Threads;
      if (k < d) {
        float a = acc[j];
        for (int q = 0; q < cnt; ++q) {
          const float c = dzc[q];
          if (c != 0.f) a = fmaf(c, H[(p0 + q) * d + k], a);
        }
        acc[j] = a;
      }
    }
  }
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    const int k = tid + j * kF32Threads;
    if (k < d) dW[static_cast<size_t>(v) * d + k] = acc[j];
  }
}

}  // namespace

// ------------------------------------------------------------------------------------------
// launches
// ------------------------------------------------------------------------------------------
cudaError_t launch_mask_scan(const uint8_t* mask, int S, int T, int32_t* counts,
                             cudaStream_t st) {
  const int warps = 8;
  k_mask_scan<<<(S + warps - 1) / warps, warps * 32, 0, st>>>(mask, S, T, counts);
  return cudaGetLastError();
}

cudaError_t launch_pack(const uint8_t* mask, const int32_t* counts, int S, int T,
                        long long rows_cap, int32_t* seq_base, int32_t* row_pos, int32_t* pos_row,
                        WsHeader* hdr, cudaStream_t st) {
  k_seq_scan<<<1, 1024, 0, st>>>(counts, S, rows_cap, seq_base, row_pos, hdr);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  k_pack<<<S, kPackThreads, 0, st>>>(mask, S, T, seq_base, row_pos, pos_row);
  return cudaGetLastError();
}

cudaError_t launch_gather_rows(const void* H, int d, const int32_t* row_pos, const WsHeader* hdr,
                               long long rows_cap, void* Hp, cudaStream_t st) {
  const int vec = d * 2 / 16;                 // bf16 rows, d % 64 == 0
  const long long blocks = rows_cap < 8192 ? (rows_cap > 0 ? rows_cap : 1) : 8192;
  k_gather_rows<<<static_cast<unsigned>(blocks), 128, 0, st>>>(
      static_cast<const uint4*>(H), vec, row_pos, hdr, static_cast<uint4*>(Hp));
  return cudaGetLastError();
}

cudaError_t launch_dh_zero_masked(const uint8_t* mask, int S, int T, int d, void* dH,
                                  int elem_bytes, cudaStream_t st) {
  const long long P = static_cast<long long>(S) * T;
  const int vec = d * elem_bytes / 16;
  const long long blocks = P < 16384 ? (P > 0 ? P : 1) : 16384;
  k_dh_zero_masked<<<static_cast<unsigned>(blocks), 128, 0, st>>>(mask, P, vec,
                                                                  static_cast<uint4*>(dH));
  return cudaGetLastError();
}

cudaError_t launch_group_adv(const float* rewards, const int32_t* go, int num_groups, int S,
                             int std_mode, float std_eps, float* adv, WsHeader* hdr,
                             cudaStream_t st) {
  k_group_adv<<<num_groups, 32, 0, st>>>(rewards, go, num_groups, S, std_mode, std_eps, adv, hdr);
  return cudaGetLastError();
}

cudaError_t launch_fwd_merge(const float4* partials, long long rows_cap, int num_strips,
                             const float* zy, const int32_t* pos_row,
                             const int32_t* tokens, const uint8_t* mask, int S, int T, int V,
                             float* logp, float* lse, float* entropy, int32_t* argmax,
                             WsHeader* hdr, cudaStream_t st) {
  const long long P = static_cast<long long>(S) * T;
  const int threads = 256;
  k_fwd_merge<<<static_cast<unsigned>((P + threads - 1) / threads), threads, 0, st>>>(
      partials, rows_cap, num_strips, zy, pos_row, tokens, mask, S, T, V, logp, lse,
      entropy, argmax, hdr);
  return cudaGetLastError();
}

cudaError_t launch_loss_tokens(const uint8_t* mask, const float* logp, const float* old_logp,
                               const float* ref_logp, const float* adv,
                               const int32_t* valid_count, int S, int T, float eps_low,
                               float eps_high, float beta, int agg, double norm, int mode,
                               const WsHeader* hdr, float* g, float* seq_loss, cudaStream_t st,
                               const float* kl, float* c) {
  k_loss_tokens<<<S, kLossThreads, 0, st>>>(mask, logp, old_logp, ref_logp, adv, valid_count, S,
                                            T, eps_low, eps_high, beta, agg, norm, mode, hdr, g,
                                            seq_loss, kl, c);
  return cudaGetLastError();
}

cudaError_t launch_fwd_merge_kl(const float4* partials, const float4* partials2,
                                long long rows_cap, int num_strips, const float* zy,
                                const int32_t* pos_row, const int32_t* tokens,
                                const uint8_t* mask, int S, int T, int V, float* logp, float* lse,
                                float* entropy, int32_t* argmax, float* lse_ref, float* kl,
                                WsHeader* hdr, cudaStream_t st) {
  const long long P = static_cast<long long>(S) * T;
  k_fwd_merge_kl<<<static_cast<unsigned>((P + 255) / 256), 256, 0, st>>>(
      partials, partials2, rows_cap, num_strips, zy, pos_row, tokens, mask, S, T, V, logp,
      lse, entropy, argmax, lse_ref, kl, hdr);
  return cudaGetLastError();
}

cudaError_t launch_rewards(const uint8_t* correct, const float* t_base, const float* t_new,
                           const int32_t* used, const int32_t* avail, int n, float lambda_tools,
                           float* r, cudaStream_t st) {
  k_rewards<<<(n + 255) / 256, 256, 0, st>>>(correct, t_base, t_new, used, avail, n,
                                             lambda_tools, r);
  return cudaGetLastError();
}

cudaError_t launch_loss_final(const float* seq_loss, int S, int agg, double norm,
                              const WsHeader* hdr, float* loss_out, cudaStream_t st) {
  (void)agg;
  (void)norm;
  (void)hdr;
  k_loss_final<<<1, 1024, 0, st>>>(seq_loss, S, loss_out);
  return cudaGetLastError();
}

cudaError_t launch_shard_stats(const float4* partials, long long rows_cap, int num_strips,
                               const float* zy_ws, const int32_t* pos_row,
                               const int32_t* tokens, const uint8_t* mask, int S, int T,
                               int V_shard, int v_offset, float4* stats, float* zy_out,
                               cudaStream_t st) {
  const long long P = static_cast<long long>(S) * T;
  k_shard_stats<<<static_cast<unsigned>((P + 255) / 256), 256, 0, st>>>(
      partials, rows_cap, num_strips, zy_ws, pos_row, tokens, mask, S, T, V_shard,
      v_offset, stats, zy_out);
  return cudaGetLastError();
}

cudaError_t launch_merge_shards(const float4* stats, const float* zy, int P,
                                const int32_t* tokens, const uint8_t* mask, int S, int T,
                                int V_total, float* logp, float* lse, float* entropy,
                                int32_t* argmax, WsHeader* hdr, cudaStream_t st) {
  const long long n = static_cast<long long>(S) * T;
  k_merge_shards<<<static_cast<unsigned>((n + 255) / 256), 256, 0, st>>>(
      stats, zy, P, tokens, mask, S, T, V_total, logp, lse, entropy, argmax, hdr);
  return cudaGetLastError();
}

cudaError_t launch_f32_fwd(const float* H, const float* W, const int32_t* tokens,
                           const uint8_t* mask, int S, int T, int d, int V, float* logp,
                           float* lse, float* entropy, int32_t* argmax, WsHeader* hdr,
                           cudaStream_t st) {
  const long long P = static_cast<long long>(S) * T;
  k_f32_fwd<<<static_cast<unsigned>(P), kF32Threads, d * sizeof(float), st>>>(
      H, W, tokens, mask, S, T, d, V, logp, lse, entropy, argmax, hdr);
  return cudaGetLastError();
}

cudaError_t launch_f32_dh(const float* H, const float* W, const int32_t* tokens,
                          const uint8_t* mask, const float* lse, const float* g, int S, int T,
                          int d, int V, float* dH, cudaStream_t st) {
  const long long P = static_cast<long long>(S) * T;
  const size_t sm = (static_cast<size_t>(d) + kF32VChunk) * sizeof(float);
  k_f32_dh<<<static_cast<unsigned>(P), kF32Threads, sm, st>>>(H, W, tokens, mask, lse, g, S, T,
                                                              d, V, dH);
  return cudaGetLastError();
}

cudaError_t launch_f32_dw(const float* H, const float* W, const int32_t* tokens,
                          const uint8_t* mask, const float* lse, const float* g, int S, int T,
                          int d, int V, float* dW, cudaStream_t st) {
  k_f32_dw<<<V, kF32Threads, d * sizeof(float), st>>>(H, W, tokens, mask, lse, g, S, T, d, V, dW);
  return cudaGetLastError();
}

}  // namespace grpo
