// Router (fp32 logits, top-k, softmax over the selected experts, histogram),
// the standalone histogram, and the router backward.
//
// Routing indicator E[i,j,l] and per-expert token number: Sec. 3.2, Eq. 1 and
// Algorithm 1 Step 1 of the LAEP paper. Pruned experts receive no token
// (Sec. 4, Table 5): their logit is -inf before the top-k.
#include <math.h>

#include "common.cuh"
#include "tc_ptx.cuh"
#include "tmap.cuh"

MOE_DEV_ERR_DECL

namespace {

constexpr int kRouteThreads = 256;
int padded_experts(int E) { return E <= 64 ? 64 : (E <= 128 ? 128 : (E <= 192 ? 192 : 256)); }

__global__ void zero_i32_kernel(int32_t *p, int n) {
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) p[i] = 0;
}

// ---- logits on the tensor cores ----------------------------------------------
// The fp32 router weight is split into three bf16 terms, W = W_hi + W_mid + W_lo,
// each the bf16 rounding of what the earlier terms leave (the bf16x3 scheme of
// Henry, Tang and Heinecke, "Leveraging the bfloat16 artificial intelligence
// datatype for higher-precision computations", 2019). Three 8-bit significands
// cover the 24 of a normal fp32 weight, every bf16 x bf16 product is exact in
// fp32, and the three MMAs of each k-step accumulate into one fp32 accumulator
// in tensor memory, so the logits carry fp32 accumulation error only.
//
// One CTA = one 128-token tile x one range of k-blocks (a split of the
// reduction over d when there are fewer tiles than CTA slots). Warp 0 issues the
// TMA loads (x tile + the three weight terms per k-block), warp 1 owns TMEM and
// issues the MMAs, then all four warps read the accumulator (one TMEM lane
// quarter each) and write the partial logits partial[split][t][0..NP). The same
// kernel computes the router weight gradient with the roles changed (see
// route_tc_kernel): 128-feature tiles of x^T, the reduction over tokens.
constexpr int kRtBM = 128;       // tokens per tile (TMEM lanes)
constexpr int kRtBK = 64;        // k-block: 64 bf16 = one 128-byte swizzle row
constexpr int kRtThreads = 128;
constexpr int kRtSms = 152;           // SMs of a GB300: the splits aim to fill them
constexpr int kRtSmemPerSm = 233472;  // shared memory per SM (228 KB)
constexpr int kRtMaxSplits = 8;
constexpr uint32_t kRtABytes = kRtBM * kRtBK * 2;
constexpr int kRtMaxSmem = 232448;  // opt-in dynamic shared memory per CTA
constexpr uint64_t kRtWaitNs = 2000000000ull;

struct RouteTcParams {
  int M;             // output rows: tokens (logits) or d_model (router weight gradient)
  int MT;            // 128-row tiles per CTA (1 or 2); tile m's accumulator at TMEM column 256*m
  int kb_per_split;  // k-blocks of one split
  int nkb;           // k-blocks of the reduction (over d, or over the padded tokens)
  int NP;            // MMA N: experts rounded up to 16
  int NE;            // row stride of the partial logits
  int stages;        // shared-memory ring depth
  uint32_t tmem_cols;
  float *partial;
};

// Experts rounded up to the MMA's N granularity, and the matching TMEM allocation.
int route_tc_np(int E) { return (E + 15) / 16 * 16; }
// 128-row tiles per CTA: two above 96 experts (up to 192), where the three weight terms of a
// k-block (3 x NP x 128 bytes) outweigh the 16 KB x tile: two x tiles share each weight stage,
// halving the L2 reads of the weight terms per FLOP; one CTA per SM either way.
int route_tc_mt(int NP) { return (NP > 96 && NP <= 192) ? 2 : 1; }
uint32_t route_tc_tmem_cols(int NP, int MT) {
  if (MT == 2) return 512u;
  return NP <= 32 ? 32u : (NP <= 64 ? 64u : (NP <= 128 ? 128u : 256u));
}
uint32_t route_tc_stage_bytes(int NP, int MT = 1) {
  return uint32_t(MT) * kRtABytes + 3u * uint32_t(NP) * 128u;
}
size_t route_tc_smem(int NP, int stages, int MT = 1) {
  return 1024 + size_t(stages) * route_tc_stage_bytes(NP, MT) + size_t(2 * stages + 1) * 8 + 16;
}
// Two CTAs per SM with a ring of at least two stages each where that fits (more
// independent x streams per SM: measured faster than one CTA with a deeper ring), else
// one CTA per SM with the deepest ring that fits.
bool route_tc_two_per_sm(int NP) {
  return 2 * (route_tc_smem(NP, 2) + 1024) <= size_t(kRtSmemPerSm);
}
int route_tc_stages(int NP) {
  int st = 2;
  if (route_tc_two_per_sm(NP)) {
    while (st < 8 && 2 * (route_tc_smem(NP, st + 1) + 1024) <= size_t(kRtSmemPerSm)) ++st;
  } else {
    st = int((kRtMaxSmem - 2048) / route_tc_stage_bytes(NP, route_tc_mt(NP)));
  }
  return std::min(8, st);
}
// Splits of the reduction: enough CTAs to fill the SMs' CTA slots when the M rows (tokens
// for the logits, d_model for the weight gradient) give few tiles. A function of
// (M, K, NP) alone, so the workspace size is too. K > 0.
void route_tc_split(int M, int K, int NP, int *splits, int *kb_per_split) {
  const int rows = kRtBM * route_tc_mt(NP);
  const int tiles = std::max(1, (M + rows - 1) / rows);
  const int nkb = (K + kRtBK - 1) / kRtBK;
  const int target = kRtSms * (route_tc_two_per_sm(NP) ? 2 : 1);
  int s = std::max(1, std::min({target / tiles, kRtMaxSplits, nkb}));
  const int per = (nkb + s - 1) / s;
  *kb_per_split = per;
  *splits = (nkb + per - 1) / per;  // every split gets at least one k-block
}

// Router weight gradient: tokens padded to one k-block, and the row stride of its
// partial sums (the epilogue writes 32 columns at a time).
int route_tokens_padded(int T) { return (T + kRtBK - 1) / kRtBK * kRtBK; }
int route_dw_stride(int E) { return (route_tc_np(E) + 31) / 32 * 32; }

// W [d, E] fp32 -> W3 [3][NP][d] bf16 (hi, mid, lo; rows e >= E are zero), by
// 32 x 32 tiles transposed through shared memory.
__global__ void route_split_w_kernel(const float *__restrict__ w, int d, int E, int NP,
                                     uint16_t *__restrict__ w3) {
  __shared__ float tile[32][33];
  const int k0 = blockIdx.x * 32, e0 = blockIdx.y * 32;
  const int tx = threadIdx.x, ty = threadIdx.y;
  for (int i = ty; i < 32; i += 8) {
    const int k = k0 + i, e = e0 + tx;
    tile[i][tx] = (k < d && e < E) ? w[size_t(k) * E + e] : 0.f;
  }
  __syncthreads();
  for (int i = ty; i < 32; i += 8) {
    const int e = e0 + i, k = k0 + tx;
    if (e < NP && k < d) {
      const float v = tile[tx][i];
      const __nv_bfloat16 hi = __float2bfloat16_rn(v);
      const float r1 = v - __bfloat162float(hi);
      const __nv_bfloat16 mid = __float2bfloat16_rn(r1);
      const float r2 = r1 - __bfloat162float(mid);
      const __nv_bfloat16 lo = __float2bfloat16_rn(r2);
      const size_t plane = size_t(NP) * d, at = size_t(e) * d + k;
      w3[at] = __bfloat16_as_ushort(hi);
      w3[plane + at] = __bfloat16_as_ushort(mid);
      w3[2 * plane + at] = __bfloat16_as_ushort(lo);
    }
  }
}

// DW = false: the logits, partial[split][t][e] = x[t, k-range] . W3[e, k-range].
// DW = true: the router weight gradient, partial[split][i][e] = sum over the split's
// tokens t of x[t, i] * dZ[t, e] (A = x^T, read MN-major from x itself as two 64 x 64
// boxes per k-block; B = dZ's three bf16 terms, K-major [3][NP][T padded to 64]).
template <bool DW>
__global__ void __launch_bounds__(kRtThreads, 1)
    route_tc_kernel(const __grid_constant__ CUtensorMap tmX,
                    const __grid_constant__ CUtensorMap tmW, const RouteTcParams p) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = tc::smem_u32(smem_raw);
  const uint32_t pad = (1024u - (raw & 1023u)) & 1023u;
  const uint32_t b_bytes = uint32_t(p.NP) * 128u;
  const uint32_t a_bytes = uint32_t(p.MT) * kRtABytes;  // the CTA's x tiles of a k-block
  const uint32_t stage_bytes = a_bytes + 3u * b_bytes;
  const int S = p.stages;
  const uint32_t s0 = raw + pad;
  uint64_t *bars = reinterpret_cast<uint64_t *>(smem_raw + pad + size_t(S) * stage_bytes);
  int *misc = reinterpret_cast<int *>(bars + 2 * S + 1);
  volatile int *abort_flag = misc + 1;
  volatile int no_abort = 0;
  const uint32_t bar0 = tc::smem_u32(bars);
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (S + s); };
  const uint32_t done_bar = bar0 + 8u * (2 * S);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int mt = blockIdx.x, split = blockIdx.y;
  const int kb0 = split * p.kb_per_split, nk = min(p.nkb, kb0 + p.kb_per_split) - kb0;
  // Each tile starts its k-loop at its own offset, so that the CTAs do not all read
  // the same weight tile from L2 at the same time (the order is fixed per tile).
  const int rot = nk > 0 ? int((mt * 7u) % uint32_t(nk)) : 0;
  const uint32_t idesc = tc::idesc_bf16_f32(kRtBM, p.NP, DW, false);

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      tc::mbar_init(full_bar(s), 1);
      tc::mbar_init(empty_bar(s), 1);
    }
    tc::mbar_init(done_bar, 1);
    tc::fence_mbar_init();
    misc[1] = 0;
  }
  if (warp == 0 && lane == 0) {
    tc::tma_prefetch_desc(&tmX);
    tc::tma_prefetch_desc(&tmW);
  }
  if (warp == 1) {
    tc::tmem_alloc(tc::smem_u32(misc), p.tmem_cols);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem_base = static_cast<uint32_t>(misc[0]);

  if (warp == 0 && lane == 0) {
    // ---- TMA producer ----
    uint32_t it = 0;
    for (; int(it) < nk; ++it) {
      const int kb = kb0 + (int(it) + rot) % nk;
      const int s = it % S;
      const uint32_t ph = (it / S) & 1u;
      if (!tc::mbar_wait(empty_bar(s), ph ^ 1u, kRtWaitNs, abort_flag)) {
        dev_flag(&g_dev_err, MOE_DEV_WAIT_TIMEOUT);
        *abort_flag = 1;
        break;
      }
      tc::mbar_arrive_expect_tx(full_bar(s), stage_bytes);
      const uint32_t dst = s0 + s * stage_bytes;
      const int k0 = kb * kRtBK;
      for (int m = 0; m < p.MT; ++m) {
        const int row0 = (mt * p.MT + m) * kRtBM;
        const uint32_t am = dst + uint32_t(m) * kRtABytes;
        if (DW) {  // x^T: features row0 .. +127 (two 64-wide boxes) x tokens k0 .. k0+63
          tc::tma_load_2d(am, &tmX, full_bar(s), row0, k0);
          tc::tma_load_2d(am + 64 * 128, &tmX, full_bar(s), row0 + 64, k0);
        } else {
          tc::tma_load_2d(am, &tmX, full_bar(s), k0, row0);
        }
      }
#pragma unroll
      for (int j = 0; j < 3; ++j)
        tc::tma_load_2d(dst + a_bytes + j * b_bytes, &tmW, full_bar(s), k0, j * p.NP);
    }
    // every issued load lands before the CTA may exit (also after an abort)
    for (int s = 0; s < S; ++s) {
      if (it > uint32_t(s)) {
        const uint32_t n = (it - 1 - s) / S;
        if (!tc::mbar_wait(full_bar(s), n & 1u, kRtWaitNs, &no_abort))
          dev_flag(&g_dev_err, MOE_DEV_WAIT_TIMEOUT);
      }
    }
  } else if (warp == 1 && lane == 0) {
    // ---- MMA issuer ----
    uint32_t it = 0;
    bool issued = false;
    for (; int(it) < nk; ++it) {
      const int s = it % S;
      const uint32_t ph = (it / S) & 1u;
      if (!tc::mbar_wait(full_bar(s), ph, kRtWaitNs, abort_flag)) {
        dev_flag(&g_dev_err, MOE_DEV_WAIT_TIMEOUT);
        *abort_flag = 1;
        break;
      }
      tc::fence_after_sync();
      const uint32_t a_s = s0 + s * stage_bytes, b_s = a_s + a_bytes;
      for (int m = 0; m < p.MT; ++m) {
        const uint32_t am = a_s + uint32_t(m) * kRtABytes;
#pragma unroll
        for (int kk = 0; kk < kRtBK / 16; ++kk) {
          const uint64_t ad = DW ? tc::smem_desc_sw128(am + kk * 2048, 8192, 1024)
                                 : tc::smem_desc_sw128(am + kk * 32, 16, 1024);
#pragma unroll
          for (int j = 0; j < 3; ++j) {
            const uint64_t bd = tc::smem_desc_sw128(b_s + j * b_bytes + kk * 32, 16, 1024);
            tc::mma_bf16(tmem_base + uint32_t(m) * 256u, ad, bd, idesc,
                         (it != 0 || kk != 0 || j != 0) ? 1u : 0u);
          }
        }
      }
      tc::mma_commit(empty_bar(s));
      issued = true;
    }
    if (issued) tc::mma_commit(done_bar);
    else *abort_flag = 1;  // nothing to wait for: the epilogue must not wait either
  }
  __syncwarp();

  // ---- epilogue: TMEM lane quarter `warp` -> 32 output rows x NP partial sums ----
  int ok = 0;
  if (lane == 0) {
    ok = tc::mbar_wait(done_bar, 0, kRtWaitNs, abort_flag) ? 1 : 0;
    if (!ok && !*abort_flag) {
      dev_flag(&g_dev_err, MOE_DEV_WAIT_TIMEOUT);
      *abort_flag = 1;
    }
  }
  ok = __shfl_sync(0xffffffffu, ok, 0);
  if (ok) {
    tc::fence_after_sync();
    for (int m = 0; m < p.MT; ++m) {
      const int t = (mt * p.MT + m) * kRtBM + warp * 32 + lane;
      float *dst = p.partial + (size_t(split) * p.M + t) * p.NE;
      for (int c0 = 0; c0 < p.NP; c0 += 32) {
        uint32_t r[32];
        tc::tmem_ld_32x32b_x32(tmem_base + (uint32_t(warp * 32) << 16) + uint32_t(m) * 256u +
                                   uint32_t(c0),
                               r);
        tc::tmem_ld_wait();
        if (t < p.M) {
#pragma unroll
          for (int q = 0; q < 8; ++q)
            stg_v4(dst + c0 + 4 * q, make_uint4(r[4 * q], r[4 * q + 1], r[4 * q + 2], r[4 * q + 3]));
        }
      }
    }
  }
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem_base, p.tmem_cols);
  }
}

// One warp per token: logits = sum of the split
// partials (fixed order) + bias, pruned experts -inf, k rounds of a warp arg-max
// (ties to the lower index), softmax over the selected logits, per-expert
// histogram (shared per block, then one global add per expert and block).
template <int NE>
__global__ void __launch_bounds__(kRouteThreads, 4) route_topk_kernel(
    const float *__restrict__ partial, int splits, const float *__restrict__ logits_in,
    const float *__restrict__ bias, const uint8_t *__restrict__ active_mask, int T, int E, int k,
    float *__restrict__ logits_out, int32_t *__restrict__ topk_idx, float *__restrict__ topk_gate,
    int32_t *__restrict__ counts) {
  constexpr int TK = NE / 32;  // logits per lane
  __shared__ int hist[NE];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (int e = tid; e < NE; e += kRouteThreads) hist[e] = 0;
  __syncthreads();
  for (int t = blockIdx.x * (kRouteThreads / 32) + warp; t < T;
       t += gridDim.x * (kRouteThreads / 32)) {
    float v[TK];
#pragma unroll
    for (int j = 0; j < TK; ++j) {
      const int e = lane + 32 * j;
      float z = 0.f;
      if (logits_in != nullptr) {
        z = e < E ? logits_in[size_t(t) * E + e] : 0.f;
      } else {
        for (int y = 0; y < splits; ++y) z += partial[(size_t(y) * T + t) * NE + e];
        if (bias != nullptr && e < E) z += bias[e];
      }
      if (e >= E || (active_mask != nullptr && active_mask[e] == 0)) z = -INFINITY;
      v[j] = z;
      if (logits_out != nullptr && e < E) logits_out[size_t(t) * E + e] = z;
    }
    // Order-preserving unsigned keys of the logits (a larger float gives a larger key,
    // -0 is taken as +0 so that equal logits tie; 0 marks an expert that cannot be
    // selected). Each round takes the warp maximum of the keys with one redux and the
    // lowest expert holding it with a second: a lane offers expert 32 j + lane for its
    // lowest slot j holding its own maximum, when that equals the warp's. (One ballot per
    // slot and round before: ~1,200 warp instructions per token at 192 experts, top-8.)
    unsigned key[TK];
#pragma unroll
    for (int j = 0; j < TK; ++j) {
      const unsigned u = __float_as_uint(v[j] == 0.f ? 0.f : v[j]);
      key[j] = (lane + 32 * j < E) ? ((u & 0x80000000u) ? ~u : (u | 0x80000000u)) : 0u;
    }
    float sel_v[8];
    int sel_e[8];
#pragma unroll
    for (int s = 0; s < 8; ++s) {
      if (s >= k) break;
      unsigned best = 0;
      int bj = 0;
#pragma unroll
      for (int j = 0; j < TK; ++j)
        if (key[j] > best) {  // strict: the lowest slot keeps a tie
          best = key[j];
          bj = j;
        }
      const unsigned m = __reduce_max_sync(0xffffffffu, best);
      const int be = int(__reduce_min_sync(0xffffffffu, best == m ? unsigned(32 * bj + lane) : ~0u));
#pragma unroll
      for (int j = 0; j < TK; ++j)
        if (32 * j + lane == be) key[j] = 0u;
      sel_v[s] = __uint_as_float((m & 0x80000000u) ? (m & 0x7fffffffu) : ~m);
      sel_e[s] = be;
    }
    // softmax over the selected logits (renormalised top-k), fp32
    const float zmax = sel_v[0];
    float den = 0.f, ex[8];
    bool too_few = false;
#pragma unroll
    for (int s = 0; s < 8; ++s) {
      if (s < k) {
        ex[s] = expf(sel_v[s] - zmax);
        den += ex[s];
        if (sel_v[s] == -INFINITY) too_few = true;
      }
    }
    if (lane == 0 && too_few) dev_flag(&g_dev_err, MOE_DEV_TOO_FEW_LIVE);
#pragma unroll
    for (int s = 0; s < 8; ++s) {
      if (s < k && lane == s) {
        topk_idx[size_t(t) * k + s] = sel_e[s];
        topk_gate[size_t(t) * k + s] = ex[s] / den;
        if (sel_e[s] >= 0 && sel_e[s] < E) atomicAdd(&hist[sel_e[s]], 1);
      }
    }
  }
  __syncthreads();
  if (counts != nullptr)
    for (int e = tid; e < E; e += kRouteThreads)
      if (hist[e]) atomicAdd(&counts[e], hist[e]);
}

__global__ void load_stats_kernel(const int32_t *__restrict__ topk_idx, int64_t A, int E,
                                  int32_t *__restrict__ counts) {
  __shared__ int hist[256];
  for (int e = threadIdx.x; e < E; e += blockDim.x) hist[e] = 0;
  __syncthreads();
  for (int64_t a = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; a < A;
       a += int64_t(gridDim.x) * blockDim.x) {
    const int e = topk_idx[a];
    if (e >= 0 && e < E)
      atomicAdd(&hist[e], 1);
    else
      dev_flag(&g_dev_err, MOE_DEV_BAD_EXPERT);
  }
  __syncthreads();
  for (int e = threadIdx.x; e < E; e += blockDim.x)
    if (hist[e]) atomicAdd(&counts[e], hist[e]);
}

// ---- router backward -------------------------------------------------------

// Softmax backward over the selected k, d_logits[t,j] = g_j (dg_j - sum_i g_i dg_i),
// and dZ (the [T, E] logit gradient, zero off the selected experts) as three bf16
// terms, K-major for the tensor cores: dz3[s][e][t] for e < NP, t < Tp (tokens padded
// to 64; the padding is zero). One thread per token and 16 experts (blockIdx.y); the
// y = 0 blocks also write d_logits.
constexpr int kDzExperts = 16;
__global__ void route_bwd_dz_kernel(const int32_t *__restrict__ topk_idx,
                                    const float *__restrict__ gate, const float *__restrict__ dgate,
                                    int T, int Tp, int k, int NP, float *__restrict__ d_logits,
                                    uint16_t *__restrict__ dz3) {
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= Tp) return;
  float g[8], dg[8], s = 0.f;
  int ei[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    g[j] = 0.f;
    dg[j] = 0.f;
    ei[j] = -1;
    if (j < k && t < T) {
      g[j] = gate[size_t(t) * k + j];
      dg[j] = dgate[size_t(t) * k + j];
      ei[j] = topk_idx[size_t(t) * k + j];
      s = fmaf(g[j], dg[j], s);
    }
  }
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    g[j] = g[j] * (dg[j] - s);
    if (blockIdx.y == 0 && j < k && t < T) d_logits[size_t(t) * k + j] = g[j];
  }
  const size_t plane = size_t(NP) * Tp;
  const int e0 = blockIdx.y * kDzExperts;
  for (int e = e0; e < min(NP, e0 + kDzExperts); ++e) {
    float v = 0.f;
#pragma unroll
    for (int j = 0; j < 8; ++j)
      if (ei[j] == e) v = g[j];  // the k selected experts of a token are distinct
    const __nv_bfloat16 hi = __float2bfloat16_rn(v);
    const float r1 = v - __bfloat162float(hi);
    const __nv_bfloat16 mid = __float2bfloat16_rn(r1);
    const float r2 = r1 - __bfloat162float(mid);
    const __nv_bfloat16 lo = __float2bfloat16_rn(r2);
    const size_t at = size_t(e) * Tp + t;
    dz3[at] = __bfloat16_as_ushort(hi);
    dz3[plane + at] = __bfloat16_as_ushort(mid);
    dz3[2 * plane + at] = __bfloat16_as_ushort(lo);
  }
}

// dw_router[i, e] = sum over the splits, in order, of partial[split][i][e].
__global__ void route_dw_reduce_kernel(const float *__restrict__ partial, int splits, int d,
                                       int E, int NE, float *__restrict__ dw_router) {
  const int n = d * E;
  for (int idx = blockIdx.x * blockDim.x + threadIdx.x; idx < n; idx += gridDim.x * blockDim.x) {
    const int i = idx / E, e = idx - i * E;
    float acc = 0.f;
    for (int y = 0; y < splits; ++y) acc += partial[(size_t(y) * d + i) * NE + e];
    dw_router[idx] = acc;
  }
}

__global__ void zero_f32_kernel(float *p, int n) {
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) p[i] = 0.f;
}

// Tensor-core logits: splits W into its three bf16 terms (w3), then one CTA per
// (token tile, split). Returns the number of partial planes written in *splits.
int launch_route_tc(const uint16_t *x, const float *w, int T, int d, int E, int NE, uint16_t *w3,
                    float *partial, int *splits_out, cudaStream_t s) {
  const int NP = route_tc_np(E), MT = route_tc_mt(NP);
  const int stages = route_tc_stages(NP);
  const size_t smem = route_tc_smem(NP, stages, MT);
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(route_tc_kernel<false>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, kRtMaxSmem);
    if (e != cudaSuccess) return moe::cuda_status(e, "moe_route: set smem attribute");
    attr_set = true;
  }
  dim3 sgrid((d + 31) / 32, (NP + 31) / 32);
  MOE_LAUNCH("route_split_w", s, route_split_w_kernel<<<sgrid, dim3(32, 8), 0, s>>>(w, d, E, NP, w3));
  if (int st = moe::launch_status("moe_route: split router weight")) return st;
  CUtensorMap mx, mw;
  int st;
  if ((st = moe::make_map(&mx, x, uint64_t(T), uint64_t(d), kRtBK, kRtBM, "router x"))) return st;
  if ((st = moe::make_map(&mw, w3, uint64_t(3 * NP), uint64_t(d), kRtBK, uint32_t(NP), "router w")))
    return st;
  int splits = 1, per = 1;
  route_tc_split(T, d, route_tc_np(E), &splits, &per);
  RouteTcParams p;
  p.M = T;
  p.MT = MT;
  p.kb_per_split = per;
  p.nkb = (d + kRtBK - 1) / kRtBK;
  p.NP = NP;
  p.NE = NE;
  p.stages = stages;
  p.tmem_cols = route_tc_tmem_cols(NP, MT);
  p.partial = partial;
  dim3 grid((T + kRtBM * MT - 1) / (kRtBM * MT), splits);
  MOE_LAUNCH("route_logits", s, route_tc_kernel<false><<<grid, kRtThreads, smem, s>>>(mx, mw, p));
  *splits_out = splits;
  return moe::launch_status("moe_route: logits");
}

template <int NE>
int launch_route(const uint16_t *x, const float *w, const float *b, const uint8_t *mask, int T,
                 int d, int E, int k, const float *lin, float *lout, int32_t *idx, float *gate,
                 int32_t *counts, float *partial, uint16_t *w3, cudaStream_t s) {
  int splits = 0;
  if (lin == nullptr)
    if (int st = launch_route_tc(x, w, T, d, E, NE, w3, partial, &splits, s)) return st;
  // one warp per token, grid-stride over the tokens; four blocks per SM, so that each
  // block's shared histogram sums ~100 tokens' assignments before its global atomics (one
  // block per 8 tokens sent 512k atomics to the counters at T=65536, top-8; the heaviest
  // expert's counter took ~60k of them one after another)
  const int grid2 = int(std::min<int64_t>((int64_t(T) + kRouteThreads / 32 - 1) / (kRouteThreads / 32),
                                          int64_t(moe::num_sms()) * 4));
  MOE_LAUNCH("route_topk", s, route_topk_kernel<NE><<<grid2, kRouteThreads, 0, s>>>(
                                  partial, splits, lin, b, mask, T, E, k, lout, idx, gate, counts));
  return moe::launch_status("moe_route: top-k");
}

}  // namespace

namespace moe {
MOE_DEV_ERR_DEFINE_READER(route_dev_error)

size_t route_partial_bytes(int T, int d, int E) {
  if (T <= 0) return 0;
  int splits = 1, per = 1;
  route_tc_split(T, d, route_tc_np(E), &splits, &per);
  return size_t(splits) * size_t(T) * size_t(padded_experts(E)) * 4;
}
size_t route_w3_bytes(int d, int E) { return size_t(3) * route_tc_np(E) * size_t(d) * 2; }
size_t route_dz3_bytes(int T, int E) {
  return size_t(3) * route_tc_np(E) * size_t(route_tokens_padded(T)) * 2;
}
size_t route_dw_partial_bytes(int T, int d, int E) {
  if (T <= 0) return 0;
  int splits = 1, per = 1;
  route_tc_split(d, route_tokens_padded(T), route_tc_np(E), &splits, &per);
  return size_t(splits) * size_t(d) * size_t(route_dw_stride(E)) * 4;
}
}  // namespace moe

extern "C" {

int moe_route(const uint16_t *x, const float *w_router, const float *bias,
              const uint8_t *active_mask, int T, int d, int E, int k, const float *logits_in,
              float *logits_out, int32_t *topk_idx, float *topk_gate, int32_t *counts, void *ws,
              size_t ws_bytes, moe_stream_t stream) {
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (E < 1 || E > 256) return moe::set_error(MOE_ERR_UNSUPPORTED, "moe_route: E=%d not in [1,256]", E);
  if (k < 1 || k > 8 || k > E) return moe::set_error(MOE_ERR_UNSUPPORTED, "moe_route: k=%d", k);
  if (T < 0 || d <= 0 || d % 8) return moe::set_error(MOE_ERR_ARG, "moe_route: T=%d d=%d", T, d);
  if (T > 0 && (!topk_idx || !topk_gate)) return moe::set_error(MOE_ERR_ARG, "moe_route: null output");
  if (T > 0 && !logits_in && (!x || !w_router))
    return moe::set_error(MOE_ERR_ARG, "moe_route: null x/w_router");
  if (x && !moe::aligned16(x)) return moe::set_error(MOE_ERR_ARG, "moe_route: x not 16-byte aligned");
  float *partial = nullptr;
  uint16_t *w3 = nullptr;
  if (!logits_in && T > 0) {
    const moe::WsLayout L = moe::ws_layout(T, d, E, k, 0);
    if (!ws || ws_bytes < L.total) return moe::set_error(MOE_ERR_WORKSPACE, "moe_route: workspace");
    if (!moe::aligned16(ws)) return moe::set_error(MOE_ERR_ARG, "moe_route: ws alignment");
    partial = reinterpret_cast<float *>(static_cast<char *>(ws) + L.route_partial);
    w3 = reinterpret_cast<uint16_t *>(static_cast<char *>(ws) + L.route_w3);
  }
  if (counts) {
    MOE_LAUNCH("zero_counts", s, zero_i32_kernel<<<1, 256, 0, s>>>(counts, E));
    if (int st = moe::launch_status("moe_route: zero counts")) return st;
  }
  if (T == 0) return MOE_OK;
  switch (padded_experts(E)) {
    case 64: return launch_route<64>(x, w_router, bias, active_mask, T, d, E, k, logits_in, logits_out, topk_idx, topk_gate, counts, partial, w3, s);
    case 128: return launch_route<128>(x, w_router, bias, active_mask, T, d, E, k, logits_in, logits_out, topk_idx, topk_gate, counts, partial, w3, s);
    case 192: return launch_route<192>(x, w_router, bias, active_mask, T, d, E, k, logits_in, logits_out, topk_idx, topk_gate, counts, partial, w3, s);
    default: return launch_route<256>(x, w_router, bias, active_mask, T, d, E, k, logits_in, logits_out, topk_idx, topk_gate, counts, partial, w3, s);
  }
}

int moe_load_stats(const int32_t *topk_idx, int T, int k, int E, int32_t *counts, int accumulate,
                   moe_stream_t stream) {
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (E < 1 || E > 256 || k < 1 || T < 0) return moe::set_error(MOE_ERR_ARG, "moe_load_stats: sizes");
  if (!counts || (T > 0 && !topk_idx)) return moe::set_error(MOE_ERR_ARG, "moe_load_stats: null");
  if (!accumulate) {
    MOE_LAUNCH("zero_counts", s, zero_i32_kernel<<<1, 256, 0, s>>>(counts, E));
    if (int st = moe::launch_status("moe_load_stats: zero")) return st;
  }
  const int64_t A = int64_t(T) * k;
  if (A == 0) return MOE_OK;
  const int grid = int(std::min<int64_t>((A + 255) / 256, int64_t(moe::num_sms()) * 4));
  MOE_LAUNCH("load_stats", s, load_stats_kernel<<<grid, 256, 0, s>>>(topk_idx, A, E, counts));
  return moe::launch_status("moe_load_stats: launch");
}

}  // extern "C"

namespace {
// Weight-gradient launch on the tensor cores: partial[split][i][e] over the split's tokens.
int launch_route_dw(const uint16_t *x, const uint16_t *dz3, int T, int d, int E, float *partial,
                    int *splits_out, cudaStream_t s) {
  const int NP = route_tc_np(E), Tp = route_tokens_padded(T), MT = route_tc_mt(NP);
  const int stages = route_tc_stages(NP);
  const size_t smem = route_tc_smem(NP, stages, MT);
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(route_tc_kernel<true>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, kRtMaxSmem);
    if (e != cudaSuccess) return moe::cuda_status(e, "moe_route_bwd: set smem attribute");
    attr_set = true;
  }
  CUtensorMap mx, mz;
  int st;
  // x [T, d] read as 64 features x 64 tokens boxes (features contiguous: MN-major A)
  if ((st = moe::make_map(&mx, x, uint64_t(T), uint64_t(d), 64, kRtBK, "router bwd x"))) return st;
  if ((st = moe::make_map(&mz, dz3, uint64_t(3 * NP), uint64_t(Tp), kRtBK, uint32_t(NP), "router bwd dz")))
    return st;
  int splits = 1, per = 1;
  route_tc_split(d, Tp, NP, &splits, &per);
  RouteTcParams p;
  p.M = d;
  p.MT = MT;
  p.kb_per_split = per;
  p.nkb = Tp / kRtBK;
  p.NP = NP;
  p.NE = route_dw_stride(E);
  p.stages = stages;
  p.tmem_cols = route_tc_tmem_cols(NP, MT);
  p.partial = partial;
  dim3 grid((d + kRtBM * MT - 1) / (kRtBM * MT), splits);
  MOE_LAUNCH("route_bwd_dw", s, route_tc_kernel<true><<<grid, kRtThreads, smem, s>>>(mx, mz, p));
  *splits_out = splits;
  return moe::launch_status("moe_route_bwd: weight gradient");
}
}  // namespace

extern "C" {

int moe_route_bwd(const uint16_t *x, const int32_t *topk_idx, const float *topk_gate,
                  const float *d_gate, int T, int d, int E, int k, float *d_logits,
                  float *dw_router, void *ws, size_t ws_bytes, moe_stream_t stream) {
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (E < 1 || E > 256 || k < 1 || k > 8 || k > E || T < 0 || d <= 0 || d % 8)
    return moe::set_error(MOE_ERR_ARG, "moe_route_bwd: sizes");
  if (!dw_router || (T > 0 && (!x || !topk_idx || !topk_gate || !d_gate || !d_logits || !ws)))
    return moe::set_error(MOE_ERR_ARG, "moe_route_bwd: null pointer");
  if ((x && !moe::aligned16(x)) || (ws && !moe::aligned16(ws)))
    return moe::set_error(MOE_ERR_ARG, "moe_route_bwd: alignment");
  if (T == 0) {
    const int n = d * E;
    MOE_LAUNCH("zero_dw_router", s, zero_f32_kernel<<<std::min((n + 255) / 256, 1024), 256, 0, s>>>(dw_router, n));
    return moe::launch_status("moe_route_bwd: zero");
  }
  const moe::WsLayout L = moe::ws_layout(T, d, E, k, 0);
  if (ws_bytes < L.total) return moe::set_error(MOE_ERR_WORKSPACE, "moe_route_bwd: workspace");
  uint16_t *dz3 = reinterpret_cast<uint16_t *>(static_cast<char *>(ws) + L.route_dz3);
  float *partial = reinterpret_cast<float *>(static_cast<char *>(ws) + L.route_dw_partial);
  const int NP = route_tc_np(E), Tp = route_tokens_padded(T);
  dim3 zgrid((Tp + 255) / 256, (NP + kDzExperts - 1) / kDzExperts);
  MOE_LAUNCH("route_bwd_dz", s, route_bwd_dz_kernel<<<zgrid, 256, 0, s>>>(
                                    topk_idx, topk_gate, d_gate, T, Tp, k, NP, d_logits, dz3));
  if (int st = moe::launch_status("moe_route_bwd: dz")) return st;
  int splits = 0;
  if (int st = launch_route_dw(x, dz3, T, d, E, partial, &splits, s)) return st;
  const int n = d * E;
  MOE_LAUNCH("route_bwd_reduce", s, route_dw_reduce_kernel<<<std::min((n + 255) / 256, 4 * moe::num_sms()), 256, 0, s>>>(
                                        partial, splits, d, E, route_dw_stride(E), dw_router));
  return moe::launch_status("moe_route_bwd: reduce");
}

}  // extern "C"
