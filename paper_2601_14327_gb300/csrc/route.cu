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
constexpr int kBM = 64;  // tokens per CTA

// Padded expert count NE (multiple of 64). 16 x 16 threads: thread (tx, ty) owns
// tokens ty*4 .. ty*4+3 and experts j*64 + tx*4 + q (j < NE/64, q < 4), so the
// shared-memory reads of one row of W are contiguous float4s across tx.
template <int NE> struct RouteShape {
  static constexpr int BK = NE <= 128 ? 32 : 16;  // reduction chunk (registers stage one)
  static constexpr int TN = NE / 16;   // experts per thread
  static constexpr int TM = 4;         // tokens per thread
  static constexpr int LDL = NE + 1;   // logits row stride in shared memory
  static constexpr size_t kStage = size_t(BK) * kBM * 4 + size_t(BK) * NE * 4;
  static constexpr size_t kGemmSmem = 2 * kStage;
  static constexpr size_t kLogitSmem = size_t(kBM) * LDL * 4;
  static constexpr size_t kSmem = (kGemmSmem > kLogitSmem ? kGemmSmem : kLogitSmem) + NE * 4;
};

__device__ __forceinline__ bool better(float v, int e, float bv, int be) {
  return v > bv || (v == bv && e < be);
}

__global__ void zero_i32_kernel(int32_t *p, int n) {
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) p[i] = 0;
}

// One CTA: 64 tokens x all experts. Logits by FFMA in fp32 (x converted from
// bf16 exactly) with the next k-chunk prefetched into registers while the
// current one is multiplied; then one warp per token runs k rounds of a warp
// arg-max over the logits row.
template <int NE>
__global__ void __launch_bounds__(kRouteThreads) route_kernel(
    const uint16_t *__restrict__ x, const float *__restrict__ w_router,
    const float *__restrict__ bias, const uint8_t *__restrict__ active_mask, int T, int d, int E,
    int k, const float *__restrict__ logits_in, float *__restrict__ logits_out,
    int32_t *__restrict__ topk_idx, float *__restrict__ topk_gate, int32_t *__restrict__ counts) {
  using S = RouteShape<NE>;
  constexpr int TM = S::TM, TN = S::TN, LDL = S::LDL, BM = kBM, kBK = S::BK;
  constexpr int WPT = kBK * NE / kRouteThreads;  // W elements each thread stages per chunk
  extern __shared__ __align__(16) float smem[];
  float *Ls = smem;  // [BM][LDL] (reuses the staging buffers)
  int *hist = reinterpret_cast<int *>(
      smem + (S::kGemmSmem > S::kLogitSmem ? S::kGemmSmem : S::kLogitSmem) / 4);

  const int tid = threadIdx.x;
  const int t0 = blockIdx.x * BM;
  for (int e = tid; e < NE; e += kRouteThreads) hist[e] = 0;

  if (logits_in == nullptr) {
    const int tx = tid & 15, ty = tid >> 4;
    float acc[TM][TN];
#pragma unroll
    for (int i = 0; i < TM; ++i)
#pragma unroll
      for (int j = 0; j < TN; ++j) acc[i][j] = 0.f;
    // register staging of one chunk: x (threads 0..127: one row, 8 columns) and W
    float xr[8];
    float wr[WPT];
    constexpr int XSEG = kBK / 8;  // 16-byte segments of x per row and chunk
    const int xrow = tid / XSEG, xcol = (tid % XSEG) * 8;
    auto load_chunk = [&](int k0) {
      if (tid < BM * kBK / 8) {
        if (t0 + xrow < T && k0 + xcol < d) {
          unpack8(ldg_nc_v4(x + size_t(t0 + xrow) * d + k0 + xcol), xr);
        } else {
#pragma unroll
          for (int q = 0; q < 8; ++q) xr[q] = 0.f;
        }
      }
#pragma unroll
      for (int i = 0; i < WPT; ++i) {
        const int v = tid + i * kRouteThreads;
        const int kk = v / NE, e = v % NE;
        wr[i] = (e < E && k0 + kk < d) ? __ldg(w_router + size_t(k0 + kk) * E + e) : 0.f;
      }
    };
    auto store_chunk = [&](int buf) {
      float *Xs = smem + buf * (S::kStage / 4);  // [kBK][BM]
      float *Ws = Xs + kBK * BM;                 // [kBK][NE]
      if (tid < BM * kBK / 8) {
#pragma unroll
        for (int q = 0; q < 8; ++q) Xs[(xcol + q) * BM + xrow] = xr[q];
      }
#pragma unroll
      for (int i = 0; i < WPT; ++i) Ws[tid + i * kRouteThreads] = wr[i];
    };
    const int nchunks = (d + kBK - 1) / kBK;
    load_chunk(0);
    store_chunk(0);
    __syncthreads();
    for (int ch = 0; ch < nchunks; ++ch) {
      if (ch + 1 < nchunks) load_chunk((ch + 1) * kBK);
      const float *Xs = smem + (ch & 1) * (S::kStage / 4);
      const float *Ws = Xs + kBK * BM;
#pragma unroll
      for (int kk = 0; kk < kBK; ++kk) {
        const float4 xv = *reinterpret_cast<const float4 *>(&Xs[kk * BM + ty * TM]);
        const float xs[4] = {xv.x, xv.y, xv.z, xv.w};
#pragma unroll
        for (int j4 = 0; j4 < NE / 64; ++j4) {
          const float4 wv = *reinterpret_cast<const float4 *>(&Ws[kk * NE + j4 * 64 + tx * 4]);
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
#pragma unroll
    for (int j = 0; j < TN; ++j) {
      const int e = (j >> 2) * 64 + tx * 4 + (j & 3);
      const float b = (bias != nullptr && e < E) ? bias[e] : 0.f;
#pragma unroll
      for (int i = 0; i < TM; ++i) Ls[(ty * TM + i) * LDL + e] = acc[i][j] + b;
    }
  } else {
    for (int v = tid; v < BM * NE; v += kRouteThreads) {
      const int r = v / NE, e = v % NE;
      Ls[r * LDL + e] = (t0 + r < T && e < E) ? logits_in[size_t(t0 + r) * E + e] : 0.f;
    }
  }
  __syncthreads();
  // Pruned experts and padding columns can never win.
  for (int v = tid; v < BM * NE; v += kRouteThreads) {
    const int r = v / NE, e = v % NE;
    if (e >= E || (active_mask != nullptr && active_mask[e] == 0)) Ls[r * LDL + e] = -INFINITY;
  }
  __syncthreads();
  if (logits_out != nullptr) {
    for (int v = tid; v < BM * E; v += kRouteThreads) {
      const int r = v / E, e = v % E;
      if (t0 + r < T) logits_out[size_t(t0 + r) * E + e] = Ls[r * LDL + e];
    }
  }

  // Top-k per token: warp w handles tokens w, w+8, ...
  const int tx = tid & 31, ty = tid >> 5;
  for (int m = ty; m < BM; m += 8) {
    const int t = t0 + m;
    if (t >= T) break;
    constexpr int TK = NE / 32;  // logits per lane
    float v[TK];
    unsigned taken = 0;
#pragma unroll
    for (int j = 0; j < TK; ++j) v[j] = Ls[m * LDL + tx + 32 * j];
    float sel_v[8];
    int sel_e[8];
#pragma unroll
    for (int s = 0; s < 8; ++s) {
      if (s >= k) break;
      float bv = -INFINITY;
      int be = 0x7fffffff;
#pragma unroll
      for (int j = 0; j < TK; ++j) {
        const int e = tx + 32 * j;
        if (e < E && !((taken >> j) & 1u) && better(v[j], e, bv, be)) { bv = v[j]; be = e; }
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) {
        const float ov = __shfl_xor_sync(0xffffffffu, bv, off);
        const int oe = __shfl_xor_sync(0xffffffffu, be, off);
        if (better(ov, oe, bv, be)) { bv = ov; be = oe; }
      }
      if ((be & 31) == tx) taken |= 1u << (be >> 5);
      sel_v[s] = bv;
      sel_e[s] = be;
    }
    // softmax over the selected logits (renormalised top-k), fp32
    const float zmax = sel_v[0];
    float den = 0.f, ex[8];
#pragma unroll
    for (int s = 0; s < 8; ++s) {
      if (s < k) { ex[s] = expf(sel_v[s] - zmax); den += ex[s]; }
    }
    bool too_few = false;
#pragma unroll
    for (int s = 0; s < 8; ++s)
      if (s < k && sel_v[s] == -INFINITY) too_few = true;
    if (tx == 0 && too_few) dev_flag(&g_dev_err, MOE_DEV_TOO_FEW_LIVE);
#pragma unroll
    for (int s = 0; s < 8; ++s) {
      if (s < k && tx == s) {
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
                 int32_t *counts, cudaStream_t s) {
  using S = RouteShape<NE>;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(route_kernel<NE>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, int(S::kSmem));
    if (e != cudaSuccess) return moe::cuda_status(e, "moe_route: set smem attribute");
    attr_set = true;
  }
  const int grid = (T + kBM - 1) / kBM;
  MOE_LAUNCH("route", s, route_kernel<NE><<<grid, kRouteThreads, S::kSmem, s>>>(x, w, b, mask, T, d, E, k, lin, lout,
                                                        idx, gate, counts));
  return moe::launch_status("moe_route: launch");
}

}  // namespace

namespace moe {
MOE_DEV_ERR_DEFINE_READER(route_dev_error)
}

extern "C" {

int moe_route(const uint16_t *x, const float *w_router, const float *bias,
              const uint8_t *active_mask, int T, int d, int E, int k, const float *logits_in,
              float *logits_out, int32_t *topk_idx, float *topk_gate, int32_t *counts,
              moe_stream_t stream) {
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (E < 1 || E > 256) return moe::set_error(MOE_ERR_UNSUPPORTED, "moe_route: E=%d not in [1,256]", E);
  if (k < 1 || k > 8 || k > E) return moe::set_error(MOE_ERR_UNSUPPORTED, "moe_route: k=%d", k);
  if (T < 0 || d <= 0 || d % 8) return moe::set_error(MOE_ERR_ARG, "moe_route: T=%d d=%d", T, d);
  if (!topk_idx || !topk_gate) return moe::set_error(MOE_ERR_ARG, "moe_route: null output");
  if (!logits_in && (!x || !w_router)) return moe::set_error(MOE_ERR_ARG, "moe_route: null x/w_router");
  if (x && !moe::aligned16(x)) return moe::set_error(MOE_ERR_ARG, "moe_route: x not 16-byte aligned");
  if (counts) {
    MOE_LAUNCH("zero_counts", s, zero_i32_kernel<<<1, 256, 0, s>>>(counts, E));
    if (int st = moe::launch_status("moe_route: zero counts")) return st;
  }
  if (T == 0) return MOE_OK;
  if (E <= 64) return launch_route<64>(x, w_router, bias, active_mask, T, d, E, k, logits_in, logits_out, topk_idx, topk_gate, counts, s);
  if (E <= 128) return launch_route<128>(x, w_router, bias, active_mask, T, d, E, k, logits_in, logits_out, topk_idx, topk_gate, counts, s);
  if (E <= 192) return launch_route<192>(x, w_router, bias, active_mask, T, d, E, k, logits_in, logits_out, topk_idx, topk_gate, counts, s);
  return launch_route<256>(x, w_router, bias, active_mask, T, d, E, k, logits_in, logits_out, topk_idx, topk_gate, counts, s);
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
  if (!x_perm || !topk_gate || !d_gate || !row_of_assignment || !group_offsets ||
      !group_counts || !d_logits || !dw_router || !ws)
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
