// Dispatch and combine: the data movement around the grouped expert FFN.
//
// moe_permute is a stable counting sort of the T*k assignments by expert
// (order inside a group: token, then slot), so the grouped layout is
// deterministic and bit-exact. Groups start at multiples of 128 rows so that
// every 128-row GEMM tile belongs to one expert; padding rows are zero.
#include <cuda.h>

#include <mutex>

#include "common.cuh"

MOE_DEV_ERR_DECL

namespace {

constexpr int kChunk = moe::kPermChunk;  // assignments per block
constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kPerWarp = kChunk / kWarps;  // 512 assignments per warp

// Block histograms: hist[e * nblk + b] = #{a in chunk b : idx[a] == e}.
__global__ void __launch_bounds__(kThreads) perm_hist_kernel(const int32_t *__restrict__ idx,
                                                             int64_t A, int E, int nblk,
                                                             int32_t *__restrict__ hist) {
  __shared__ int sh[256];
  for (int e = threadIdx.x; e < E; e += kThreads) sh[e] = 0;
  __syncthreads();
  const int64_t a0 = int64_t(blockIdx.x) * kChunk;
  const int64_t a1 = min(A, a0 + kChunk);
  for (int64_t a = a0 + threadIdx.x; a < a1; a += kThreads) {
    const int e = idx[a];
    if (e >= 0 && e < E) atomicAdd(&sh[e], 1);
    else dev_flag(&g_dev_err, MOE_DEV_BAD_EXPERT);
  }
  __syncthreads();
  for (int e = threadIdx.x; e < E; e += kThreads) hist[size_t(e) * nblk + blockIdx.x] = sh[e];
}

// One CTA of 1024 threads: per-expert exclusive scan over blocks (in place),
// group counts, and the padded group offsets.
__global__ void __launch_bounds__(1024) perm_scan_kernel(
    int32_t *__restrict__ hist, int E, int nblk, const int32_t *__restrict__ counts_check,
    int64_t rows_cap, int32_t *__restrict__ group_offsets, int32_t *__restrict__ group_counts) {
  __shared__ int s_cnt[256];
  __shared__ int s_pad[257];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int e = warp; e < E; e += 32) {
    int running = 0;
    int32_t *h = hist + size_t(e) * nblk;
    for (int base = 0; base < nblk; base += 32) {
      const int v = (base + lane < nblk) ? h[base + lane] : 0;
      int incl = v;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const int o = __shfl_up_sync(0xffffffffu, incl, off);
        if (lane >= off) incl += o;
      }
      if (base + lane < nblk) h[base + lane] = running + incl - v;
      running += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (lane == 0) s_cnt[e] = running;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int acc = 0;
    for (int e = 0; e < E; ++e) {
      s_pad[e] = acc;
      acc += (s_cnt[e] + moe::kGroupPad - 1) / moe::kGroupPad * moe::kGroupPad;
    }
    s_pad[E] = acc;
    if (int64_t(acc) > rows_cap) dev_flag(&g_dev_err, MOE_DEV_ROWS_OVERFLOW);
  }
  __syncthreads();
  for (int e = threadIdx.x; e <= E; e += blockDim.x) group_offsets[e] = s_pad[e];
  for (int e = threadIdx.x; e < E; e += blockDim.x) {
    group_counts[e] = s_cnt[e];
    if (counts_check != nullptr && counts_check[e] != s_cnt[e])
      dev_flag(&g_dev_err, MOE_DEV_COUNT_MISMATCH);
  }
}

// Row of every assignment: group start + rank among the earlier assignments
// of the same expert. Warps walk consecutive sub-chunks in order; inside a
// 32-wide step, lanes with equal experts are ranked by lane order.
__global__ void __launch_bounds__(kThreads) perm_rank_kernel(
    const int32_t *__restrict__ idx, int64_t A, int E, int nblk,
    const int32_t *__restrict__ hist_prefix, const int32_t *__restrict__ group_offsets,
    int64_t rows_cap, int32_t *__restrict__ row_of_assignment, int k,
    int32_t *__restrict__ token_of_row) {
  __shared__ int wh[kWarps][256];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int i = threadIdx.x; i < kWarps * 256; i += kThreads) (&wh[0][0])[i] = 0;
  __syncthreads();
  const int64_t a0 = int64_t(blockIdx.x) * kChunk + int64_t(warp) * kPerWarp;
  for (int s = 0; s < kPerWarp; s += 32) {
    const int64_t a = a0 + s + lane;
    if (a < A) {
      const int e = idx[a];
      if (e >= 0 && e < E) atomicAdd(&wh[warp][e], 1);
    }
  }
  __syncthreads();
  const bool overflow = group_offsets[E] > rows_cap;
  for (int e = threadIdx.x; e < E; e += kThreads) {
    int running = group_offsets[e] + hist_prefix[size_t(e) * nblk + blockIdx.x];
#pragma unroll
    for (int w = 0; w < kWarps; ++w) {
      const int c = wh[w][e];
      wh[w][e] = running;
      running += c;
    }
  }
  __syncthreads();
  const unsigned lt = (1u << lane) - 1u;
  for (int s = 0; s < kPerWarp; s += 32) {
    const int64_t a = a0 + s + lane;
    int e = -1;
    if (a < A) {
      e = idx[a];
      if (e < 0 || e >= E) e = -1;
    }
    const unsigned peers = __match_any_sync(0xffffffffu, e);
    const int rank = __popc(peers & lt);
    const int leader = __ffs(peers) - 1;
    int row = -1;
    if (e >= 0) row = wh[warp][e] + rank;
    __syncwarp();
    if (e >= 0 && lane == leader) wh[warp][e] += __popc(peers);
    __syncwarp();
    if (a < A) row_of_assignment[a] = (e >= 0 && !overflow) ? row : -1;
    if (token_of_row != nullptr && a < A && e >= 0 && !overflow) token_of_row[row] = int(a / k);
  }
}

// Pad rows of every group read token 0 (their products are multiplied by zero
// downstream: the pad rows of d_out_perm and of the router's d_logits are zero).
__global__ void __launch_bounds__(kThreads) pad_token_kernel(const int32_t *__restrict__ group_offsets,
                                                             const int32_t *__restrict__ group_counts,
                                                             int E, int64_t rows_cap,
                                                             int32_t *__restrict__ token_of_row) {
  const int e = blockIdx.x;
  const int r0 = group_offsets[e] + group_counts[e];
  const int r1 = int(min((long long)group_offsets[e + 1], (long long)rows_cap));
  for (int r = r0 + threadIdx.x; r < r1; r += kThreads) token_of_row[r] = 0;
}

// One warp per token: read x[t,:] once, write it to its k grouped rows.
__global__ void __launch_bounds__(kThreads) perm_gather_kernel(
    const uint16_t *__restrict__ x, const int32_t *__restrict__ row_of_assignment, int T, int d,
    int k, int64_t rows_cap, uint16_t *__restrict__ x_perm) {
  const int warp = (blockIdx.x * kThreads + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (warp >= T) return;
  const int t = warp;
  int my_row = (lane < k) ? row_of_assignment[size_t(t) * k + lane] : -1;
  int rows[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) rows[j] = __shfl_sync(0xffffffffu, my_row, j);
  const int nv = d / 8;
  const uint16_t *src = x + size_t(t) * d;
  // four 16-byte loads in flight per lane before their stores
  for (int c0 = lane; c0 < nv; c0 += 128) {
    uint4 v[4];
#pragma unroll
    for (int u = 0; u < 4; ++u)
      if (c0 + 32 * u < nv) v[u] = ldg_nc_v4(src + (c0 + 32 * u) * 8);
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int c = c0 + 32 * u;
      if (c >= nv) break;
#pragma unroll
      for (int j = 0; j < 8; ++j)
        if (j < k && rows[j] >= 0 && rows[j] < rows_cap) stg_v4(x_perm + size_t(rows[j]) * d + c * 8, v[u]);
    }
  }
}

// Zero the padding rows [group_offsets[e] + group_counts[e], group_offsets[e+1]);
// blockIdx.x = expert, blockIdx.y splits that expert's padding rows.
__global__ void __launch_bounds__(kThreads) pad_zero_kernel(const int32_t *__restrict__ group_offsets,
                                                            const int32_t *__restrict__ group_counts,
                                                            int E, int d, int64_t rows_cap,
                                                            uint16_t *__restrict__ buf) {
  const int e = blockIdx.x;
  const int r0 = group_offsets[e] + group_counts[e];
  const int r1 = int(min((long long)group_offsets[e + 1], (long long)rows_cap));
  const int nv = d / 8;
  const uint4 z = make_uint4(0, 0, 0, 0);
  const int64_t n = int64_t(r1 - r0) * nv;
  for (int64_t i = int64_t(blockIdx.y) * kThreads + threadIdx.x; i < n;
       i += int64_t(gridDim.y) * kThreads) {
    const int64_t r = r0 + i / nv, c = i % nv;
    stg_v4(buf + size_t(r) * d + c * 8, z);
  }
}

constexpr int kPadSplit = 8;  // blocks per expert in pad_zero_kernel

// y[t] = sum_j g[t,j] * out_perm[row(t,j)]  (fp32 sum, one bf16 rounding)
__global__ void __launch_bounds__(kThreads) combine_kernel(
    const uint16_t *__restrict__ out_perm, const int32_t *__restrict__ row_of_assignment,
    const float *__restrict__ gate, int T, int d, int k, uint16_t *__restrict__ y) {
  const int warp = (blockIdx.x * kThreads + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (warp >= T) return;
  const int t = warp;
  int my_row = (lane < k) ? row_of_assignment[size_t(t) * k + lane] : -1;
  float my_g = (lane < k) ? gate[size_t(t) * k + lane] : 0.f;
  int rows[8];
  float g[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    rows[j] = __shfl_sync(0xffffffffu, my_row, j);
    g[j] = __shfl_sync(0xffffffffu, my_g, j);
  }
  const int nv = d / 8;
  for (int c = lane; c < nv; c += 32) {
    uint4 v[8];
#pragma unroll
    for (int j = 0; j < 8; ++j)
      if (j < k && rows[j] >= 0) v[j] = ldg_nc_v4(out_perm + size_t(rows[j]) * d + c * 8);
    float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      if (j < k && rows[j] >= 0) {
        float f[8];
        unpack8(v[j], f);
#pragma unroll
        for (int q = 0; q < 8; ++q) acc[q] = fmaf(g[j], f[q], acc[q]);
      }
    }
    stg_v4(y + size_t(t) * d + c * 8, pack8(acc));
  }
}

// d_out_perm[row(t,j)] = g[t,j] * dy[t];  d_gate[t,j] = <dy[t], out_perm[row(t,j)]>
// DOUT: d_out_perm rows = g * dy[t]; DGATE: d_gate = <dy[t], out_perm rows>. The two
// halves can run as separate launches (DGATE alone reads out_perm and writes nothing
// large; DOUT alone never reads out_perm).
template <bool DOUT, bool DGATE>
__global__ void __launch_bounds__(kThreads) combine_bwd_kernel(
    const uint16_t *__restrict__ dy, const uint16_t *__restrict__ out_perm,
    const int32_t *__restrict__ row_of_assignment, const float *__restrict__ gate, int T, int d,
    int k, int64_t rows_cap, uint16_t *__restrict__ d_out_perm, float *__restrict__ d_gate) {
  const int warp = (blockIdx.x * kThreads + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (warp >= T) return;
  const int t = warp;
  int my_row = (lane < k) ? row_of_assignment[size_t(t) * k + lane] : -1;
  float my_g = (lane < k) ? gate[size_t(t) * k + lane] : 0.f;
  int rows[8];
  float g[8], dot[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    rows[j] = __shfl_sync(0xffffffffu, my_row, j);
    if (rows[j] >= rows_cap) rows[j] = -1;
    g[j] = __shfl_sync(0xffffffffu, my_g, j);
    dot[j] = 0.f;
  }
  const int nv = d / 8;
  for (int c = lane; c < nv; c += 32) {
    float fd[8];
    unpack8(ldg_nc_v4(dy + size_t(t) * d + c * 8), fd);
    uint4 v[8];
    if (DGATE) {
#pragma unroll
      for (int j = 0; j < 8; ++j)
        if (j < k && rows[j] >= 0) v[j] = ldg_nc_v4(out_perm + size_t(rows[j]) * d + c * 8);
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      if (j < k && rows[j] >= 0) {
        if (DGATE) {
          float f[8];
          unpack8(v[j], f);
#pragma unroll
          for (int q = 0; q < 8; ++q) dot[j] = fmaf(fd[q], f[q], dot[j]);
        }
        if (DOUT) {
          float o[8];
#pragma unroll
          for (int q = 0; q < 8; ++q) o[q] = g[j] * fd[q];
          stg_v4(d_out_perm + size_t(rows[j]) * d + c * 8, pack8(o));
        }
      }
    }
  }
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    if (DGATE && j < k) {
      float s = dot[j];
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
      if (lane == 0) d_gate[size_t(t) * k + j] = s;
    }
  }
}

// w_t[e, i] = w[i, e]
__global__ void transpose_router_kernel(const float *__restrict__ w, int d, int E,
                                        float *__restrict__ w_t) {
  __shared__ float tile[32][33];
  const int i0 = blockIdx.x * 32, e0 = blockIdx.y * 32;
  for (int r = threadIdx.y; r < 32; r += blockDim.y) {
    const int i = i0 + r, e = e0 + threadIdx.x;
    tile[r][threadIdx.x] = (i < d && e < E) ? w[size_t(i) * E + e] : 0.f;
  }
  __syncthreads();
  for (int r = threadIdx.y; r < 32; r += blockDim.y) {
    const int e = e0 + r, i = i0 + threadIdx.x;
    if (e < E && i < d) w_t[size_t(e) * d + i] = tile[threadIdx.x][r];
  }
}

// dx[t] = sum_j dx_perm[row(t,j)] + sum_j d_logits[t,j] * w_t[e_j]
__global__ void __launch_bounds__(kThreads) permute_bwd_kernel(
    const uint16_t *__restrict__ dx_perm, const int32_t *__restrict__ row_of_assignment,
    const int32_t *__restrict__ topk_idx, const float *__restrict__ d_logits,
    const float *__restrict__ w_t, int T, int d, int E, int k, uint16_t *__restrict__ dx) {
  const int warp = (blockIdx.x * kThreads + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (warp >= T) return;
  const int t = warp;
  const bool router = (d_logits != nullptr && w_t != nullptr);
  int my_row = (lane < k) ? row_of_assignment[size_t(t) * k + lane] : -1;
  int my_e = (lane < k && router) ? topk_idx[size_t(t) * k + lane] : -1;
  float my_dz = (lane < k && router) ? d_logits[size_t(t) * k + lane] : 0.f;
  int rows[8], ex[8];
  float dz[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    rows[j] = __shfl_sync(0xffffffffu, my_row, j);
    ex[j] = __shfl_sync(0xffffffffu, my_e, j);
    if (ex[j] >= E) ex[j] = -1;
    dz[j] = __shfl_sync(0xffffffffu, my_dz, j);
  }
  const int nv = d / 8;
  for (int c = lane; c < nv; c += 32) {
    uint4 v[8];
#pragma unroll
    for (int j = 0; j < 8; ++j)
      if (j < k && rows[j] >= 0) v[j] = ldg_nc_v4(dx_perm + size_t(rows[j]) * d + c * 8);
    float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      if (j < k && rows[j] >= 0) {
        float f[8];
        unpack8(v[j], f);
#pragma unroll
        for (int q = 0; q < 8; ++q) acc[q] += f[q];
      }
    }
    if (router) {
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        if (j < k && ex[j] >= 0) {
          const float4 *wp = reinterpret_cast<const float4 *>(w_t + size_t(ex[j]) * d + c * 8);
          const float4 w0 = __ldg(wp), w1 = __ldg(wp + 1);
          acc[0] = fmaf(dz[j], w0.x, acc[0]); acc[1] = fmaf(dz[j], w0.y, acc[1]);
          acc[2] = fmaf(dz[j], w0.z, acc[2]); acc[3] = fmaf(dz[j], w0.w, acc[3]);
          acc[4] = fmaf(dz[j], w1.x, acc[4]); acc[5] = fmaf(dz[j], w1.y, acc[5]);
          acc[6] = fmaf(dz[j], w1.z, acc[6]); acc[7] = fmaf(dz[j], w1.w, acc[7]);
        }
      }
    }
    stg_v4(dx + size_t(t) * d + c * 8, pack8(acc));
  }
}

int warp_grid(int T) { return (T + kWarps - 1) / kWarps; }

}  // namespace

namespace moe {
MOE_DEV_ERR_DEFINE_READER(permute_dev_error)
}

extern "C" {

int moe_permute(const uint16_t *x, const int32_t *topk_idx, const int32_t *counts, int T, int d,
                int E, int k, int64_t rows_cap, int32_t *group_offsets, int32_t *group_counts,
                int32_t *row_of_assignment, uint16_t *x_perm, void *ws, size_t ws_bytes,
                moe_stream_t stream) {
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (E < 1 || E > 256 || k < 1 || k > 8 || T < 0 || d <= 0 || d % 8)
    return moe::set_error(MOE_ERR_ARG, "moe_permute: sizes T=%d d=%d E=%d k=%d", T, d, E, k);
  if (!group_offsets || !group_counts || !ws || (T > 0 && (!x || !topk_idx || !row_of_assignment || !x_perm)))
    return moe::set_error(MOE_ERR_ARG, "moe_permute: null pointer");
  if (rows_cap < moe_perm_rows_max(T, k, E))
    return moe::set_error(MOE_ERR_ARG, "moe_permute: rows_cap %lld < %lld", (long long)rows_cap,
                          (long long)moe_perm_rows_max(T, k, E));
  if (rows_cap >= (int64_t(1) << 31)) return moe::set_error(MOE_ERR_UNSUPPORTED, "moe_permute: rows_cap >= 2^31");
  if ((x && !moe::aligned16(x)) || (x_perm && !moe::aligned16(x_perm)))
    return moe::set_error(MOE_ERR_ARG, "moe_permute: x/x_perm not 16-byte aligned");
  const moe::WsLayout L = moe::ws_layout(T, d, E, k, 0);
  if (ws_bytes < L.total) return moe::set_error(MOE_ERR_WORKSPACE, "moe_permute: workspace");
  const int64_t A = int64_t(T) * k;
  const int nblk = int(std::max<int64_t>(1, (A + kChunk - 1) / kChunk));
  int32_t *hist = reinterpret_cast<int32_t *>(static_cast<char *>(ws) + L.perm_hist);
  MOE_LAUNCH("perm_hist", s, perm_hist_kernel<<<nblk, kThreads, 0, s>>>(topk_idx, A, E, nblk, hist));
  if (int st = moe::launch_status("moe_permute: hist")) return st;
  MOE_LAUNCH("perm_scan", s, perm_scan_kernel<<<1, 1024, 0, s>>>(hist, E, nblk, counts, rows_cap, group_offsets, group_counts));
  if (int st = moe::launch_status("moe_permute: scan")) return st;
  if (A > 0) {
    MOE_LAUNCH("perm_rank", s, perm_rank_kernel<<<nblk, kThreads, 0, s>>>(topk_idx, A, E, nblk, hist, group_offsets, rows_cap,
                                               row_of_assignment, k, nullptr));
    if (int st = moe::launch_status("moe_permute: rank")) return st;
    MOE_LAUNCH("perm_gather", s, perm_gather_kernel<<<warp_grid(T), kThreads, 0, s>>>(x, row_of_assignment, T, d, k, rows_cap,
                                                         x_perm));
    if (int st = moe::launch_status("moe_permute: gather")) return st;
  }
  MOE_LAUNCH("pad_zero", s, pad_zero_kernel<<<dim3(E, kPadSplit), kThreads, 0, s>>>(group_offsets, group_counts, E, d, rows_cap, x_perm));
  return moe::launch_status("moe_permute: pad");
}

int moe_permute_map(const int32_t *topk_idx, const int32_t *counts, int T, int E, int k,
                    int64_t rows_cap, int32_t *group_offsets, int32_t *group_counts,
                    int32_t *row_of_assignment, int32_t *token_of_row, void *ws, size_t ws_bytes,
                    moe_stream_t stream) {
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (E < 1 || E > 256 || k < 1 || k > 8 || T < 0)
    return moe::set_error(MOE_ERR_ARG, "moe_permute_map: sizes T=%d E=%d k=%d", T, E, k);
  if (!group_offsets || !group_counts || !ws || !token_of_row ||
      (T > 0 && (!topk_idx || !row_of_assignment)))
    return moe::set_error(MOE_ERR_ARG, "moe_permute_map: null pointer");
  if (rows_cap < moe_perm_rows_max(T, k, E))
    return moe::set_error(MOE_ERR_ARG, "moe_permute_map: rows_cap %lld < %lld", (long long)rows_cap,
                          (long long)moe_perm_rows_max(T, k, E));
  if (rows_cap >= (int64_t(1) << 31))
    return moe::set_error(MOE_ERR_UNSUPPORTED, "moe_permute_map: rows_cap >= 2^31");
  const moe::WsLayout L = moe::ws_layout(T, 8, E, k, 0);
  if (ws_bytes < L.perm_hist + size_t(E) * std::max<int64_t>(1, (int64_t(T) * k + kChunk - 1) / kChunk) * 4)
    return moe::set_error(MOE_ERR_WORKSPACE, "moe_permute_map: workspace");
  const int64_t A = int64_t(T) * k;
  const int nblk = int(std::max<int64_t>(1, (A + kChunk - 1) / kChunk));
  int32_t *hist = reinterpret_cast<int32_t *>(static_cast<char *>(ws) + L.perm_hist);
  MOE_LAUNCH("perm_hist", s, perm_hist_kernel<<<nblk, kThreads, 0, s>>>(topk_idx, A, E, nblk, hist));
  if (int st = moe::launch_status("moe_permute_map: hist")) return st;
  MOE_LAUNCH("perm_scan", s, perm_scan_kernel<<<1, 1024, 0, s>>>(hist, E, nblk, counts, rows_cap, group_offsets, group_counts));
  if (int st = moe::launch_status("moe_permute_map: scan")) return st;
  if (A > 0) {
    MOE_LAUNCH("perm_rank", s, perm_rank_kernel<<<nblk, kThreads, 0, s>>>(topk_idx, A, E, nblk, hist, group_offsets, rows_cap,
                                               row_of_assignment, k, token_of_row));
    if (int st = moe::launch_status("moe_permute_map: rank")) return st;
  }
  MOE_LAUNCH("pad_token", s, pad_token_kernel<<<E, kThreads, 0, s>>>(group_offsets, group_counts, E, rows_cap, token_of_row));
  return moe::launch_status("moe_permute_map: pad");
}

int moe_unpermute_combine(const uint16_t *out_perm, const int32_t *row_of_assignment,
                          const float *topk_gate, int T, int d, int k, uint16_t *y,
                          moe_stream_t stream) {
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (k < 1 || k > 8 || T < 0 || d <= 0 || d % 8) return moe::set_error(MOE_ERR_ARG, "moe_unpermute_combine: sizes");
  if (T == 0) return MOE_OK;
  if (!out_perm || !row_of_assignment || !topk_gate || !y)
    return moe::set_error(MOE_ERR_ARG, "moe_unpermute_combine: null pointer");
  if (!moe::aligned16(out_perm) || !moe::aligned16(y))
    return moe::set_error(MOE_ERR_ARG, "moe_unpermute_combine: alignment");
  MOE_LAUNCH("combine", s, combine_kernel<<<warp_grid(T), kThreads, 0, s>>>(out_perm, row_of_assignment, topk_gate, T, d, k, y));
  return moe::launch_status("moe_unpermute_combine: launch");
}

int moe_unpermute_combine_bwd(const uint16_t *dy, const uint16_t *out_perm,
                              const int32_t *row_of_assignment, const float *topk_gate,
                              const int32_t *group_offsets, const int32_t *group_counts, int T,
                              int d, int E, int k, uint16_t *d_out_perm, float *d_gate,
                              moe_stream_t stream) {
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (E < 1 || E > 256 || k < 1 || k > 8 || T < 0 || d <= 0 || d % 8)
    return moe::set_error(MOE_ERR_ARG, "moe_unpermute_combine_bwd: sizes");
  if (!d_out_perm && !d_gate && T > 0)  // (with no tokens d_gate is empty and may be NULL)
    return moe::set_error(MOE_ERR_ARG, "moe_unpermute_combine_bwd: no output requested");
  if ((d_out_perm && (!group_offsets || !group_counts)) ||
      (T > 0 && (!dy || !row_of_assignment || !topk_gate || (d_gate && !out_perm))))
    return moe::set_error(MOE_ERR_ARG, "moe_unpermute_combine_bwd: null pointer");
  if ((d_out_perm && !moe::aligned16(d_out_perm)) || (dy && !moe::aligned16(dy)) ||
      (out_perm && !moe::aligned16(out_perm)))
    return moe::set_error(MOE_ERR_ARG, "moe_unpermute_combine_bwd: alignment");
  const int64_t rows_cap = moe_perm_rows_max(T, k, E);
  if (T > 0) {
    const int grid = warp_grid(T);
    if (d_out_perm && d_gate) {
      MOE_LAUNCH("combine_bwd", s, (combine_bwd_kernel<true, true><<<grid, kThreads, 0, s>>>(
                                       dy, out_perm, row_of_assignment, topk_gate, T, d, k,
                                       rows_cap, d_out_perm, d_gate)));
    } else if (d_out_perm) {
      MOE_LAUNCH("combine_bwd_dout", s, (combine_bwd_kernel<true, false><<<grid, kThreads, 0, s>>>(
                                            dy, out_perm, row_of_assignment, topk_gate, T, d, k,
                                            rows_cap, d_out_perm, d_gate)));
    } else {
      MOE_LAUNCH("combine_bwd_dgate", s, (combine_bwd_kernel<false, true><<<grid, kThreads, 0, s>>>(
                                             dy, out_perm, row_of_assignment, topk_gate, T, d, k,
                                             rows_cap, d_out_perm, d_gate)));
    }
    if (int st = moe::launch_status("moe_unpermute_combine_bwd: launch")) return st;
  }
  if (!d_out_perm) return MOE_OK;
  MOE_LAUNCH("pad_zero", s, pad_zero_kernel<<<dim3(E, kPadSplit), kThreads, 0, s>>>(group_offsets, group_counts, E, d, rows_cap, d_out_perm));
  return moe::launch_status("moe_unpermute_combine_bwd: pad");
}

int moe_permute_bwd(const uint16_t *dx_perm, const int32_t *row_of_assignment,
                    const int32_t *topk_idx, const float *d_logits, const float *w_router, int T,
                    int d, int E, int k, uint16_t *dx, void *ws, size_t ws_bytes,
                    moe_stream_t stream) {
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (E < 1 || E > 256 || k < 1 || k > 8 || T < 0 || d <= 0 || d % 8)
    return moe::set_error(MOE_ERR_ARG, "moe_permute_bwd: sizes");
  if (T == 0) return MOE_OK;
  if (!dx_perm || !row_of_assignment || !dx) return moe::set_error(MOE_ERR_ARG, "moe_permute_bwd: null pointer");
  if ((d_logits == nullptr) != (w_router == nullptr))
    return moe::set_error(MOE_ERR_ARG, "moe_permute_bwd: d_logits and w_router go together");
  if (!moe::aligned16(dx_perm) || !moe::aligned16(dx)) return moe::set_error(MOE_ERR_ARG, "moe_permute_bwd: alignment");
  float *w_t = nullptr;
  if (w_router) {
    if (!topk_idx || !ws) return moe::set_error(MOE_ERR_ARG, "moe_permute_bwd: router term needs topk_idx and ws");
    const moe::WsLayout L = moe::ws_layout(T, d, E, k, 0);
    if (ws_bytes < L.total) return moe::set_error(MOE_ERR_WORKSPACE, "moe_permute_bwd: workspace");
    if (!moe::aligned16(ws)) return moe::set_error(MOE_ERR_ARG, "moe_permute_bwd: ws alignment");
    w_t = reinterpret_cast<float *>(static_cast<char *>(ws) + L.w_router_t);
    dim3 grid((d + 31) / 32, (E + 31) / 32), block(32, 8);
    MOE_LAUNCH("transpose_router", s, transpose_router_kernel<<<grid, block, 0, s>>>(w_router, d, E, w_t));
    if (int st = moe::launch_status("moe_permute_bwd: transpose")) return st;
  }
  MOE_LAUNCH("permute_bwd", s, permute_bwd_kernel<<<warp_grid(T), kThreads, 0, s>>>(dx_perm, row_of_assignment, topk_idx,
                                                       d_logits, w_t, T, d, E, k, dx));
  return moe::launch_status("moe_permute_bwd: launch");
}

}  // extern "C"

// ---------------------------------------------------------------------------
// moe_permute_noalloc: moe_permute for callers that cannot allocate device
// memory (no cudaMalloc and no caller workspace), e.g. an inference engine's
// plugin, whose device memory the engine planned and owns before execution
// and which receives only its input and output buffers. The
// per-block histograms live in a fixed array compiled into the library
// instead of the caller's workspace.
//
// The array holds kNoAllocScratchInts int32 entries (256 KiB). A call needs
// E * ceil(T*k / 4096) of them, so 256 experts fit with up to 1,048,576
// assignments (T*k). Every GPU that loads the library keeps the array until
// the process exits. All calls share it: calls whose kernels overlap on the
// GPU (different streams, or different host threads) race on it and must be
// serialized by the caller. Nothing in it has to start at zero: every entry a
// call reads was written earlier in the same call.
constexpr int kNoAllocScratchInts = 65536;
static __device__ __align__(256) int32_t g_perm_noalloc_scratch[kNoAllocScratchInts];

namespace {
typedef CUresult (*CtxGetCurrentFn)(CUcontext *);
typedef CUresult (*CtxGetIdFn)(CUcontext, unsigned long long *);

// Unique id of the calling thread's current CUDA context (0: none is current yet).
// Ids are never reused, so a context created after cudaDeviceReset, or another
// context of the same device, has an id of its own.
int current_context_id(unsigned long long *id) {
  static CtxGetCurrentFn get_current = nullptr;
  static CtxGetIdFn get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<CtxGetCurrentFn>(p);
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<CtxGetIdFn>(p);
  });
  if (!get_current || !get_id)
    return moe::set_error(MOE_ERR_CUDA, "moe_permute_noalloc: cuCtxGetCurrent/cuCtxGetId unavailable");
  CUcontext ctx = nullptr;
  if (get_current(&ctx) != CUDA_SUCCESS)
    return moe::set_error(MOE_ERR_CUDA, "moe_permute_noalloc: cuCtxGetCurrent failed");
  *id = 0;
  if (ctx && get_id(ctx, id) != CUDA_SUCCESS)
    return moe::set_error(MOE_ERR_CUDA, "moe_permute_noalloc: cuCtxGetId failed");
  return MOE_OK;
}

// Device address of the array in the current context. Host code cannot use the
// array's name as a device pointer, and the address belongs to the context that
// loaded the library's module: it is looked up once per context (keyed by the
// context's unique id) and cached; another context of the same device, or the new
// primary context after cudaDeviceReset, gets a lookup of its own.
int noalloc_scratch(int32_t **out) {
  constexpr int kSlots = 64;
  static std::mutex mu;
  static unsigned long long ids[kSlots] = {0};
  static int32_t *addr[kSlots] = {nullptr};
  static int next = 0;
  unsigned long long id = 0;
  if (int st = current_context_id(&id)) return st;
  std::lock_guard<std::mutex> g(mu);
  if (id != 0) {
    for (int i = 0; i < kSlots; ++i)
      if (ids[i] == id) {
        *out = addr[i];
        return MOE_OK;
      }
  }
  void *p = nullptr;  // the runtime makes the primary context current if none is
  cudaError_t e = cudaGetSymbolAddress(&p, g_perm_noalloc_scratch);
  if (e != cudaSuccess) return moe::cuda_status(e, "moe_permute_noalloc: cudaGetSymbolAddress");
  if (id == 0 && (current_context_id(&id) != MOE_OK || id == 0))
    return moe::set_error(MOE_ERR_CUDA, "moe_permute_noalloc: no current context");
  ids[next] = id;  // oldest entry replaced when all slots are taken
  addr[next] = static_cast<int32_t *>(p);
  next = (next + 1) % kSlots;
  *out = static_cast<int32_t *>(p);
  return MOE_OK;
}
}  // namespace

extern "C" int moe_permute_noalloc(const uint16_t *x, const int32_t *topk_idx,
                                   const int32_t *counts, int T, int d, int E, int k,
                                   int64_t rows_cap, int32_t *group_offsets,
                                   int32_t *group_counts, int32_t *row_of_assignment,
                                   uint16_t *x_perm, moe_stream_t stream) {
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (E < 1 || E > 256 || k < 1 || k > 8 || T < 0 || d <= 0 || d % 8)
    return moe::set_error(MOE_ERR_ARG, "moe_permute_noalloc: sizes T=%d d=%d E=%d k=%d", T, d, E, k);
  const int64_t A = int64_t(T) * k;
  const int64_t nblk64 = std::max<int64_t>(1, (A + kChunk - 1) / kChunk);
  if (int64_t(E) * nblk64 > kNoAllocScratchInts)
    return moe::set_error(MOE_ERR_UNSUPPORTED,
                          "moe_permute_noalloc: E * ceil(T*k/%d) = %lld exceeds the built-in "
                          "scratch of %d entries (use moe_permute with a workspace)",
                          kChunk, (long long)(int64_t(E) * nblk64), kNoAllocScratchInts);
  if (!group_offsets || !group_counts || (T > 0 && (!x || !topk_idx || !row_of_assignment || !x_perm)))
    return moe::set_error(MOE_ERR_ARG, "moe_permute_noalloc: null pointer");
  if (rows_cap < moe_perm_rows_max(T, k, E))
    return moe::set_error(MOE_ERR_ARG, "moe_permute_noalloc: rows_cap %lld < %lld",
                          (long long)rows_cap, (long long)moe_perm_rows_max(T, k, E));
  if (rows_cap >= (int64_t(1) << 31))
    return moe::set_error(MOE_ERR_UNSUPPORTED, "moe_permute_noalloc: rows_cap >= 2^31");
  if ((x && !moe::aligned16(x)) || (x_perm && !moe::aligned16(x_perm)))
    return moe::set_error(MOE_ERR_ARG, "moe_permute_noalloc: x/x_perm not 16-byte aligned");
  int32_t *hist = nullptr;
  if (int st = noalloc_scratch(&hist)) return st;
  const int nblk = int(nblk64);
  MOE_LAUNCH("perm_hist", s, perm_hist_kernel<<<nblk, kThreads, 0, s>>>(topk_idx, A, E, nblk, hist));
  if (int st = moe::launch_status("moe_permute_noalloc: hist")) return st;
  MOE_LAUNCH("perm_scan", s, perm_scan_kernel<<<1, 1024, 0, s>>>(hist, E, nblk, counts, rows_cap,
                                                                  group_offsets, group_counts));
  if (int st = moe::launch_status("moe_permute_noalloc: scan")) return st;
  if (A > 0) {
    MOE_LAUNCH("perm_rank", s, perm_rank_kernel<<<nblk, kThreads, 0, s>>>(
                                   topk_idx, A, E, nblk, hist, group_offsets, rows_cap,
                                   row_of_assignment, k, nullptr));
    if (int st = moe::launch_status("moe_permute_noalloc: rank")) return st;
    MOE_LAUNCH("perm_gather", s, perm_gather_kernel<<<warp_grid(T), kThreads, 0, s>>>(
                                     x, row_of_assignment, T, d, k, rows_cap, x_perm));
    if (int st = moe::launch_status("moe_permute_noalloc: gather")) return st;
  }
  MOE_LAUNCH("pad_zero", s, pad_zero_kernel<<<dim3(E, kPadSplit), kThreads, 0, s>>>(group_offsets, group_counts, E,
                                                                    d, rows_cap, x_perm));
  return moe::launch_status("moe_permute_noalloc: pad");
}
