// Router (fp32 logits, top-k, softmax over the selected experts, histogram),
// the standalone histogram, and the router backward.
//
// Routing indicator E[i,j,l] and per-expert token number: Sec. 3.2, Eq. 1 and
// Algorithm 1 Step 1 of the LAEP paper. Pruned experts receive no token
// (Sec. 4, Table 5): their logit is -inf before the top-k.
#include <math.h>

#include "common.cuh"

MOE_DEV_ERR_DECL

namespace {

constexpr int kRouteThreads = 256;
constexpr int kRouteBK = 16;            // reduction chunk of the logit contraction
constexpr int kRouteTargetCtas = 304;   // split the reduction until about this many CTAs

// Logits kernel shape for the padded expert count NE (multiple of 64). Thread
// (eg, tg) owns 8 tokens (tg*8 ..) and 8 experts {j*4*EG + eg*4 + q : j < 2,
// q < 4}: per k it reads 8 x values and 8 W values as float4s (0.5-1 byte of
// shared memory per FFMA; the float4 reads of one W row are contiguous across
// eg) and keeps 64 accumulators, so two CTAs fit on an SM (<= 128 registers).
template <int NE> struct RouteShape {
  static constexpr int EG = NE / 8;                       // threads along the experts
  static constexpr int THREADS = NE == 192 ? 384 : 256;
  static constexpr int TN = 8;                            // experts per thread
  static constexpr int TG = THREADS / EG;                 // threads along the tokens
  static constexpr int TM = 8;                            // tokens per thread
  static constexpr int BM = TG * TM;                      // tokens per CTA
  static constexpr int MIN_BLOCKS = NE == 192 ? 1 : 2;
  static constexpr size_t kStage = size_t(kRouteBK) * BM * 4 + size_t(kRouteBK) * NE * 4;
  static constexpr size_t kSmem = 2 * kStage;
};

// Reduction split so that T/BM token tiles give about kRouteTargetCtas CTAs (at
// most 8, never more CTAs than that target); fixed by (T, NE) alone, so the
// workspace size is too.
template <int NE> int route_splits(int T, int d) {
  const int tiles = (T + RouteShape<NE>::BM - 1) / RouteShape<NE>::BM;
  const int chunks = (d + kRouteBK - 1) / kRouteBK;
  const int s = kRouteTargetCtas / std::max(tiles, 1);
  return std::max(1, std::min({s, 8, chunks}));
}
int padded_experts(int E) { return E <= 64 ? 64 : (E <= 128 ? 128 : (E <= 192 ? 192 : 256)); }

__device__ __forceinline__ bool better(float v, int e, float bv, int be) {
  return v > bv || (v == bv && e < be);
}

__global__ void zero_i32_kernel(int32_t *p, int n) {
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) p[i] = 0;
}

// partial[split][t][e] = sum over this split's k range of x[t,k] * W_r[k,e]
// (fp32 FFMA, x converted from bf16 exactly; columns e >= E are zero). The next
// k-chunk is loaded into registers while the current one is multiplied.
template <int NE>
__global__ void __launch_bounds__(RouteShape<NE>::THREADS, RouteShape<NE>::MIN_BLOCKS)
    route_logits_kernel(
    const uint16_t *__restrict__ x, const float *__restrict__ w_router, int T, int d, int E,
    int k_per_split, float *__restrict__ partial) {
  using S = RouteShape<NE>;
  constexpr int TM = S::TM, TN = S::TN, EG = S::EG, BM = S::BM, BK = kRouteBK, NT = S::THREADS;
  constexpr int XN = BM * BK / 8;             // 16-byte x loads per chunk
  constexpr int XV = (XN + NT - 1) / NT;      // ... per thread
  constexpr int WV = BK * NE / NT;            // W values per thread per chunk
  extern __shared__ __align__(16) float smem[];
  const int tid = threadIdx.x;
  const int eg = tid % EG, tg = tid / EG;
  const int t0 = blockIdx.x * BM;
  const int kb = blockIdx.y * k_per_split, ke = min(d, kb + k_per_split);

  float acc[TM][TN];
#pragma unroll
  for (int i = 0; i < TM; ++i)
#pragma unroll
    for (int j = 0; j < TN; ++j) acc[i][j] = 0.f;
  float xr[XV][8], wr[WV];
  auto load_chunk = [&](int k0) {
#pragma unroll
    for (int i = 0; i < XV; ++i) {
      const int v = tid + i * NT;
      const int row = v / (BK / 8), col = (v % (BK / 8)) * 8;
      if (v < XN && t0 + row < T && k0 + col < ke) {
        unpack8(ldg_nc_v4(x + size_t(t0 + row) * d + k0 + col), xr[i]);
      } else {
#pragma unroll
        for (int q = 0; q < 8; ++q) xr[i][q] = 0.f;
      }
    }
#pragma unroll
    for (int i = 0; i < WV; ++i) {
      const int v = tid + i * NT;
      const int kk = v / NE, e = v % NE;
      wr[i] = (e < E && k0 + kk < ke) ? __ldg(w_router + size_t(k0 + kk) * E + e) : 0.f;
    }
  };
  auto store_chunk = [&](int buf) {
    float *Xs = smem + buf * (S::kStage / 4);  // [BK][BM]
    float *Ws = Xs + BK * BM;                  // [BK][NE]
#pragma unroll
    for (int i = 0; i < XV; ++i) {
      const int v = tid + i * NT;
      const int row = v / (BK / 8), col = (v % (BK / 8)) * 8;
      if (v < XN) {
#pragma unroll
        for (int q = 0; q < 8; ++q) Xs[(col + q) * BM + row] = xr[i][q];
      }
    }
#pragma unroll
    for (int i = 0; i < WV; ++i) Ws[tid + i * NT] = wr[i];
  };
  const int nchunks = (ke - kb + BK - 1) / BK;
  if (nchunks > 0) {
    load_chunk(kb);
    store_chunk(0);
  }
  __syncthreads();
  for (int ch = 0; ch < nchunks; ++ch) {
    if (ch + 1 < nchunks) load_chunk(kb + (ch + 1) * BK);
    const float *Xs = smem + (ch & 1) * (S::kStage / 4);
    const float *Ws = Xs + BK * BM;
#pragma unroll
    for (int kk = 0; kk < BK; ++kk) {
      const float4 x0 = *reinterpret_cast<const float4 *>(&Xs[kk * BM + tg * TM]);
      const float4 x1 = *reinterpret_cast<const float4 *>(&Xs[kk * BM + tg * TM + 4]);
      const float xs[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
#pragma unroll
      for (int j4 = 0; j4 < TN / 4; ++j4) {
        const float4 wv = *reinterpret_cast<const float4 *>(&Ws[kk * NE + j4 * 4 * EG + eg * 4]);
        const float ws[4] = {wv.x, wv.y, wv.z, wv.w};
#pragma unroll
        for (int i = 0; i < TM; ++i)
#pragma unroll
          for (int q = 0; q < 4; ++q) acc[i][j4 * 4 + q] = fmaf(xs[i], ws[q], acc[i][j4 * 4 + q]);
      }
    }
    if (ch + 1 < nchunks) store_chunk((ch + 1) & 1);
    __syncthreads();
  }
  float *out = partial + size_t(blockIdx.y) * T * NE;
#pragma unroll
  for (int i = 0; i < TM; ++i) {
    const int t = t0 + tg * TM + i;
    if (t >= T) break;
#pragma unroll
    for (int j4 = 0; j4 < TN / 4; ++j4)
      *reinterpret_cast<float4 *>(out + size_t(t) * NE + j4 * 4 * EG + eg * 4) =
          make_float4(acc[i][j4 * 4], acc[i][j4 * 4 + 1], acc[i][j4 * 4 + 2], acc[i][j4 * 4 + 3]);
  }
}

// One warp per token: logits = sum of the split partials (fixed order) + bias,
// pruned experts -inf, k rounds of a warp arg-max (ties to the lower index),
// softmax over the selected logits, per-expert histogram.
template <int NE>
__global__ void __launch_bounds__(kRouteThreads) route_topk_kernel(
    const float *__restrict__ partial, int splits, const float *__restrict__ logits_in,
    const float *__restrict__ bias, const uint8_t *__restrict__ active_mask, int T, int E, int k,
    float *__restrict__ logits_out, int32_t *__restrict__ topk_idx, float *__restrict__ topk_gate,
    int32_t *__restrict__ counts) {
  constexpr int TK = NE / 32;  // logits per lane
  __shared__ int hist[NE];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (int e = tid; e < NE; e += kRouteThreads) hist[e] = 0;
  __syncthreads();
  const int t = blockIdx.x * (kRouteThreads / 32) + warp;
  if (t < T) {
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
    unsigned taken = 0;
    float sel_v[8];
    int sel_e[8];
#pragma unroll
    for (int s = 0; s < 8; ++s) {
      if (s >= k) break;
      float bv = -INFINITY;
      int be = 0x7fffffff;
#pragma unroll
      for (int j = 0; j < TK; ++j) {
        const int e = lane + 32 * j;
        if (e < E && !((taken >> j) & 1u) && better(v[j], e, bv, be)) { bv = v[j]; be = e; }
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) {
        const float ov = __shfl_xor_sync(0xffffffffu, bv, off);
        const int oe = __shfl_xor_sync(0xffffffffu, be, off);
        if (better(ov, oe, bv, be)) { bv = ov; be = oe; }
      }
      if ((be & 31) == lane) taken |= 1u << (be >> 5);
      sel_v[s] = bv;
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

// d_logits[t,j] = g_j (dg_j - sum_i g_i dg_i); also scattered to the grouped rows.
__global__ void route_bwd_dz_kernel(const float *__restrict__ gate, const float *__restrict__ dgate,
                                    const int32_t *__restrict__ row_of_assignment, int T, int k,
                                    int64_t rows_cap, float *__restrict__ d_logits,
                                    float *__restrict__ dz_perm) {
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= T) return;
  float g[8], dg[8], s = 0.f;
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    if (j < k) {
      g[j] = gate[size_t(t) * k + j];
      dg[j] = dgate[size_t(t) * k + j];
      s = fmaf(g[j], dg[j], s);
    }
  }
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    if (j < k) {
      const float dz = g[j] * (dg[j] - s);
      d_logits[size_t(t) * k + j] = dz;
      const int r = row_of_assignment[size_t(t) * k + j];
      if (r >= 0 && r < rows_cap) dz_perm[r] = dz;
    }
  }
}

// One CTA per 128-row tile of the grouped layout: partial[tile, :] =
// sum over the tile's real rows of dz_perm[r] * x_perm[r, :].
__global__ void __launch_bounds__(256) route_bwd_partial_kernel(
    const uint16_t *__restrict__ x_perm, const float *__restrict__ dz_perm,
    const int32_t *__restrict__ group_offsets, const int32_t *__restrict__ group_counts, int E,
    int d, float *__restrict__ partial) {
  const int tile = blockIdx.x;
  const int row0 = tile * moe::kGroupPad;
  if (row0 >= group_offsets[E]) return;
  // group containing row0: last e with group_offsets[e] <= row0
  int lo = 0, hi = E - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (group_offsets[mid] <= row0) lo = mid; else hi = mid - 1;
  }
  const int e = lo;
  const int row_end = min(row0 + moe::kGroupPad, group_offsets[e] + group_counts[e]);
  for (int c8 = threadIdx.x; c8 < d / 8; c8 += blockDim.x) {
    float acc[8];
#pragma unroll
    for (int q = 0; q < 8; ++q) acc[q] = 0.f;
    for (int r = row0; r < row_end; ++r) {
      const float w = dz_perm[r];
      float f[8];
      unpack8(ldg_nc_v4(x_perm + size_t(r) * d + c8 * 8), f);
#pragma unroll
      for (int q = 0; q < 8; ++q) acc[q] = fmaf(w, f[q], acc[q]);
    }
    float4 *dst = reinterpret_cast<float4 *>(partial + size_t(tile) * d + c8 * 8);
    dst[0] = make_float4(acc[0], acc[1], acc[2], acc[3]);
    dst[1] = make_float4(acc[4], acc[5], acc[6], acc[7]);
  }
}

// dw_router[i, e] = sum over the tiles of group e of partial[tile, i]
__global__ void route_bwd_reduce_kernel(const float *__restrict__ partial,
                                        const int32_t *__restrict__ group_offsets, int E, int d,
                                        float *__restrict__ dw_router) {
  const int e = blockIdx.y;
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= d) return;
  const int tb = group_offsets[e] / moe::kGroupPad, te = group_offsets[e + 1] / moe::kGroupPad;
  float s = 0.f;
  for (int tile = tb; tile < te; ++tile) s += partial[size_t(tile) * d + i];
  dw_router[size_t(i) * E + e] = s;
}

template <int NE>
int launch_route(const uint16_t *x, const float *w, const float *b, const uint8_t *mask, int T,
                 int d, int E, int k, const float *lin, float *lout, int32_t *idx, float *gate,
                 int32_t *counts, float *partial, cudaStream_t s) {
  using S = RouteShape<NE>;
  int splits = 0;
  if (lin == nullptr) {
    static bool attr_set = false;
    if (!attr_set) {
      cudaError_t e = cudaFuncSetAttribute(route_logits_kernel<NE>,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, int(S::kSmem));
      if (e != cudaSuccess) return moe::cuda_status(e, "moe_route: set smem attribute");
      attr_set = true;
    }
    splits = route_splits<NE>(T, d);
    const int chunks = (d + kRouteBK - 1) / kRouteBK;
    const int k_per_split = ((chunks + splits - 1) / splits) * kRouteBK;
    dim3 grid((T + S::BM - 1) / S::BM, splits);
    MOE_LAUNCH("route_logits", s, route_logits_kernel<NE><<<grid, S::THREADS, S::kSmem, s>>>(
                                      x, w, T, d, E, k_per_split, partial));
    if (int st = moe::launch_status("moe_route: logits")) return st;
  }
  const int grid2 = (T + kRouteThreads / 32 - 1) / (kRouteThreads / 32);
  MOE_LAUNCH("route_topk", s, route_topk_kernel<NE><<<grid2, kRouteThreads, 0, s>>>(
                                  partial, splits, lin, b, mask, T, E, k, lout, idx, gate, counts));
  return moe::launch_status("moe_route: top-k");
}

}  // namespace

namespace moe {
MOE_DEV_ERR_DEFINE_READER(route_dev_error)

size_t route_partial_bytes(int T, int d, int E) {
  if (T <= 0) return 0;
  const int NE = padded_experts(E);
  int splits = 1;
  switch (NE) {
    case 64: splits = route_splits<64>(T, d); break;
    case 128: splits = route_splits<128>(T, d); break;
    case 192: splits = route_splits<192>(T, d); break;
    default: splits = route_splits<256>(T, d); break;
  }
  return size_t(splits) * size_t(T) * size_t(NE) * 4;
}
}

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
  if (!logits_in && T > 0) {
    const moe::WsLayout L = moe::ws_layout(T, d, E, k, 0);
    if (!ws || ws_bytes < L.total) return moe::set_error(MOE_ERR_WORKSPACE, "moe_route: workspace");
    if (!moe::aligned16(ws)) return moe::set_error(MOE_ERR_ARG, "moe_route: ws alignment");
    partial = reinterpret_cast<float *>(static_cast<char *>(ws) + L.route_partial);
  }
  if (counts) {
    MOE_LAUNCH("zero_counts", s, zero_i32_kernel<<<1, 256, 0, s>>>(counts, E));
    if (int st = moe::launch_status("moe_route: zero counts")) return st;
  }
  if (T == 0) return MOE_OK;
  switch (padded_experts(E)) {
    case 64: return launch_route<64>(x, w_router, bias, active_mask, T, d, E, k, logits_in, logits_out, topk_idx, topk_gate, counts, partial, s);
    case 128: return launch_route<128>(x, w_router, bias, active_mask, T, d, E, k, logits_in, logits_out, topk_idx, topk_gate, counts, partial, s);
    case 192: return launch_route<192>(x, w_router, bias, active_mask, T, d, E, k, logits_in, logits_out, topk_idx, topk_gate, counts, partial, s);
    default: return launch_route<256>(x, w_router, bias, active_mask, T, d, E, k, logits_in, logits_out, topk_idx, topk_gate, counts, partial, s);
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

int moe_route_bwd(const uint16_t *x_perm, const int32_t *topk_idx, const float *topk_gate,
                  const float *d_gate, const int32_t *row_of_assignment,
                  const int32_t *group_offsets, const int32_t *group_counts, int T, int d, int E,
                  int k, int64_t rows_cap, float *d_logits, float *dw_router, void *ws,
                  size_t ws_bytes, moe_stream_t stream) {
  (void)topk_idx;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (E < 1 || E > 256 || k < 1 || k > 8 || T < 0 || d <= 0 || d % 8)
    return moe::set_error(MOE_ERR_ARG, "moe_route_bwd: sizes");
  if (!x_perm || !group_offsets || !group_counts || !dw_router || !ws ||
      (T > 0 && (!topk_gate || !d_gate || !row_of_assignment || !d_logits)))
    return moe::set_error(MOE_ERR_ARG, "moe_route_bwd: null pointer");
  if (rows_cap < moe_perm_rows_max(T, k, E))
    return moe::set_error(MOE_ERR_ARG, "moe_route_bwd: rows_cap too small");
  if (!moe::aligned16(x_perm) || !moe::aligned16(ws))
    return moe::set_error(MOE_ERR_ARG, "moe_route_bwd: alignment");
  const moe::WsLayout L = moe::ws_layout(T, d, E, k, 0);
  if (ws_bytes < L.total) return moe::set_error(MOE_ERR_WORKSPACE, "moe_route_bwd: workspace");
  float *dz_perm = reinterpret_cast<float *>(static_cast<char *>(ws) + L.dz_perm);
  float *partial = reinterpret_cast<float *>(static_cast<char *>(ws) + L.rb_partial);
  if (T > 0) {
    MOE_LAUNCH("route_bwd_dz", s, route_bwd_dz_kernel<<<(T + 255) / 256, 256, 0, s>>>(topk_gate, d_gate, row_of_assignment, T, k,
                                                        rows_cap, d_logits, dz_perm));
    if (int st = moe::launch_status("moe_route_bwd: dz")) return st;
    const int tiles = int(rows_cap / moe::kGroupPad);
    MOE_LAUNCH("route_bwd_partial", s, route_bwd_partial_kernel<<<tiles, 256, 0, s>>>(x_perm, dz_perm, group_offsets, group_counts, E,
                                                   d, partial));
    if (int st = moe::launch_status("moe_route_bwd: partial")) return st;
  }
  dim3 grid((d + 255) / 256, E);
  MOE_LAUNCH("route_bwd_reduce", s, route_bwd_reduce_kernel<<<grid, 256, 0, s>>>(partial, group_offsets, E, d, dw_router));
  return moe::launch_status("moe_route_bwd: reduce");
}

}  // extern "C"
