// Grouped SwiGLU expert FFN on the 5th-generation tensor cores (sm_103a):
// TMA-fed shared-memory ring -> tcgen05.mma (one issuing thread) -> fp32
// accumulators in tensor memory (double-buffered) -> epilogue warps.
//
// Three matrices per expert (gate, up, down; Table A1 of the LAEP paper). The
// groups are the per-expert row ranges of the grouped layout, padded to 128
// rows, so every 128-row tile belongs to one expert. A persistent grid walks
// a tile list built on the device from group_offsets: no host round trip on
// the expert loads, and empty groups produce no tile. In the weight-gradient
// GEMMs (reduction over a group's rows, so tile cost ~ group size) the
// experts are ordered heaviest first, the longest-processing-time order that
// Algorithm 2's greedy balancing also uses; experts without rows get no tile: the
// epilogue warps store their zero gradients up front, while the first tiles' MMAs
// run (CTA-pair kernel; the one-SM kernel stores them as tiles at the end).
//
// Warps: 0 issues TMA loads, 1 owns TMEM and issues the MMAs, 2..9 are the epilogue
// (two per TMEM lane quarter, each taking half of the tile's columns).
//
// Six GEMM shapes share one kernel template:
//   kGateUp      [A|B] = X W_gu^T        (A: K-major rows, B: K-major weights)
//                epilogue: H = silu(A)*B, keeps A and B (32-row blocked) for the backward
//   kDown        O = H W_down^T
//   kDgradDown   dH = dO W_down           (B is MN-major)
//                epilogue: dA = dH*B*silu'(A), dB = dH*silu(A)
//   kDgradGateUp dX = [dA|dB] W_gu        (B is MN-major)
//   kWgradDown   dW_down[e] = dO_e^T H_e  (A and B MN-major; K = group rows)
//   kWgradGateUp dW_gu[e] = [dA|dB]_e^T X_e
#include <cuda.h>
#include <stdlib.h>

#include "common.cuh"
#include "tc_ptx.cuh"
#include "tmap.cuh"

MOE_DEV_ERR_DECL

namespace {

enum Mode : int {
  kGateUp = 0,
  kDown = 1,
  kDgradDown = 2,
  kDgradGateUp = 3,
  kWgradDown = 4,
  kWgradGateUp = 5
};

const char *const kGemmName[] = {"gemm_gate_up",       "gemm_down",
                                 "gemm_dgrad_down",    "gemm_dgrad_gate_up",
                                 "gemm_wgrad_down",    "gemm_wgrad_gate_up"};

constexpr int BM = 128;   // tile rows (TMEM lanes)
constexpr int BK = 64;    // k-block: 64 bf16 = one 128-byte swizzle row
constexpr int UMMA_K = 16;
constexpr int kEpiWarps = 8;   // two epilogue warps per TMEM lane quarter, each half the columns
constexpr int kThreads = 64 + 32 * kEpiWarps;  // warp 0 TMA, warp 1 MMA + TMEM owner, epilogue
constexpr uint64_t kWaitLimitNs = 2000000000ull;

template <int MODE> struct Traits {
  static constexpr bool A_MN = (MODE == kWgradDown || MODE == kWgradGateUp);
  static constexpr bool B_MN = (MODE != kGateUp && MODE != kDown);
  static constexpr bool WGRAD = (MODE == kWgradDown || MODE == kWgradGateUp);
};

// In-place scan by one warp of s[1..n] (n <= 256): afterwards s[i] = s[1] + ... + s[i] and
// s[0] = 0. With the count of list position j stored at s[j + 1], s[i] is then the first
// tile (or unit) of position i and s[n] the total.
__device__ __forceinline__ void warp_prefix_counts(int *s, int n, int lane) {
  const int c = (n + 31) >> 5;
  const int lo = lane * c + 1, hi = min(n, lo + c - 1);
  int sum = 0;
  for (int i = lo; i <= hi; ++i) {
    sum += s[i];
    s[i] = sum;
  }
  int incl = sum;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int v = __shfl_up_sync(0xffffffffu, incl, off);
    if (lane >= off) incl += v;
  }
  const int excl = incl - sum;
  for (int i = lo; i <= hi; ++i) s[i] += excl;
  if (lane == 0) s[0] = 0;
}

template <int BN> struct Shape {
  static constexpr int STAGES = BN == 256 ? 4 : 6;
  static constexpr uint32_t A_BYTES = BM * BK * 2;
  static constexpr uint32_t B_BYTES = BN * BK * 2;
  static constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int NBARS = 2 * STAGES + 5;
  static constexpr size_t SMEM = 1024 + size_t(STAGES) * STAGE_BYTES + NBARS * 8 +
                                 (4 + 257 + 256 + 257 + 256) * 4 + 1024 + kEpiWarps * 2048;
  static constexpr uint32_t TMEM_COLS = 2 * BN;
};

struct GemmParams {
  const int32_t *group_offsets;  // [E+1], padded group starts (device)
  int E, d, F;
  int n_tiles;     // output column tiles
  int m_tiles_w;   // weight-gradient modes: row tiles of one expert's output
  int nkb;         // k-blocks per tile (activation modes)
  uint16_t *out;   // primary output
  uint16_t *out2;  // kGateUp: pre-activations [A|B] (32-row blocked, see ab_block_index)
  const uint16_t *aux;  // kDgradDown: saved pre-activations [rows, 2F]
  // Gathered operand (kGateUp: A, kWgradGateUp: B): grouped row r reads row
  // token_of_row[r] of x [T, d] instead of row r of X_perm (nullptr: X_perm).
  const int32_t *token_of_row;
  // kDown with the combine in the epilogue (nullptr: no combine): for every real
  // grouped row r, y_acc[row_token[r], cols] += row_gate[r] * O[r, cols] in fp32
  // (row_token[r] < 0 on padding rows). out == nullptr then skips the O store.
  float *y_acc;
  const int32_t *row_token;
  const float *row_gate;
  // kDgradGateUp with the router's term of the input gradient (nullptr: without):
  // dX[r, :] += row_dz[r] * W_r[:, e] for every grouped row r of expert e, with
  // row_dz [rows] the router logit gradient of the row's assignment (0 on padding rows)
  // and w_router [d, E] fp32.
  const float *row_dz;
  const float *w_router;
  // kDgradDown with the gate gradient (nullptr: without): for every grouped row r,
  // gate_partial[r * gate_stride + nt * 2 + half] = sum over the tile's column half of
  // dH[r, f] * H[r, f], H = silu(A) * B recomputed from the saved pre-activations; the
  // row's sum over its partials is g * <dy, O> (dH = g * dy W_down).
  float *gate_partial;
  int gate_stride;
  // Weight-gradient modes: experts with active_mask[e] == 0 (pruned by LAEP) get no tile
  // and no store; their gradient buffers are left as they are (nullptr: all experts live).
  const uint8_t *active_mask;
  // CTA-pair kernel: tile counter of the dynamic schedule (zero at launch, 4 bytes of the
  // caller's workspace); dynamic = 0 walks the list with a fixed stride instead.
  int *sched_ctr;
  int dynamic;
  // Activation GEMMs split between two launches (0: no split): 1 = the CTA-pair kernel
  // takes each group's whole pairs of 128-row blocks only, 2 = the one-SM kernel takes the
  // last block of each group with an odd number of blocks only.
  int rows_split;
};

struct Tile {
  int e, goff, mt, nt, nkb;
};

__device__ __forceinline__ void fail(volatile int *abort_flag) {
  dev_flag(&g_dev_err, MOE_DEV_WAIT_TIMEOUT);
  *abort_flag = 1;
}

// sigmoid(a) = 1 / (1 + e^-a) with the fast reciprocal-based divide (2 ulp; the
// results are rounded to bf16). For very negative a, e^-a overflows to +inf and
// the quotient is 0, the limit of the function.
__device__ __forceinline__ float sigmoid_f(float a) { return __fdividef(1.f, 1.f + __expf(-a)); }
__device__ __forceinline__ float silu_f(float a) { return a * sigmoid_f(a); }

// Saved pre-activations [A|B] are stored in 32-row blocks: element (r, c) of the
// [rows, 2F] matrix lives at ((r/32)*(2F/8) + c/8)*256 + (r%32)*8 + c%8, so the
// 32 rows a warp owns in the epilogue touch 512 contiguous bytes per 8 columns
// (one coalesced warp access in the forward's store and the backward's load).
__device__ __forceinline__ size_t ab_block_index(size_t row, int col, int F) {
  return ((row >> 5) * size_t(2 * F / 8) + size_t(col >> 3)) * 256 + (row & 31) * 8 + (col & 7);
}

// Epilogue of one accumulator tile for the 32 rows and the column half (`half`) this
// warp owns: reads the fp32
// accumulator from tensor memory at `tb` (lane base and column base included) and
// writes the mode's outputs. `row` = row of this thread in the grouped layout
// (activation modes), `out_row` = row in the expert's weight-gradient matrix.
// Output staging: each epilogue warp owns a 2 KB shared-memory buffer that holds
// one 32-row x 32-column bf16 chunk in the 64-byte-swizzle layout of a TMA tile
// (row r, 16-byte chunk c at r*64 + ((c ^ ((r >> 1) & 3)) * 16): conflict-free
// when every lane writes its own row); one lane then issues a TMA tensor store.
constexpr uint32_t kStageBytes = 32 * 64;

__device__ __forceinline__ void st_shared_v4(uint32_t addr, const uint4 &v) {
  asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};" ::"r"(addr), "r"(v.x), "r"(v.y), "r"(v.z),
               "r"(v.w)
               : "memory");
}

// Writes this lane's 32 bf16 values (row `lane` of the chunk) to the staging
// buffer and stores the chunk at (col, trow) of tensor map `tm`.
__device__ __forceinline__ void stage_and_store(const CUtensorMap *tm, uint32_t stage, int lane,
                                                const uint4 (&v)[4], int col, int trow) {
  if (lane == 0) tc::bulk_wait_read0();  // the previous chunk has left the buffer
  __syncwarp();
  const uint32_t rowbase = stage + uint32_t(lane) * 64u;
  const uint32_t sw = (uint32_t(lane) >> 1) & 3u;
#pragma unroll
  for (uint32_t c = 0; c < 4; ++c) st_shared_v4(rowbase + ((c ^ sw) << 4), v[c]);
  tc::fence_proxy_async_smem();
  __syncwarp();
  if (lane == 0) {
    tc::tma_store_2d(tm, stage, col, trow);
    tc::bulk_commit();
  }
}

__device__ __forceinline__ void pack32(const uint32_t (&r)[32], uint4 (&v)[4]) {
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    v[q].x = pack_bf16x2(__uint_as_float(r[q * 8 + 0]), __uint_as_float(r[q * 8 + 1]));
    v[q].y = pack_bf16x2(__uint_as_float(r[q * 8 + 2]), __uint_as_float(r[q * 8 + 3]));
    v[q].z = pack_bf16x2(__uint_as_float(r[q * 8 + 4]), __uint_as_float(r[q * 8 + 5]));
    v[q].w = pack_bf16x2(__uint_as_float(r[q * 8 + 6]), __uint_as_float(r[q * 8 + 7]));
  }
}

template <int MODE, int BN>
__device__ __forceinline__ void epilogue_tile(const GemmParams &p, const CUtensorMap *tmO,
                                              uint32_t stage, int lane, uint32_t tb, size_t row,
                                              int out_row, int e, int nt, int half) {
  using Tr = Traits<MODE>;
  if (MODE == kGateUp) {
    const int F = p.F;
    const int trow = int(row) - lane;
#pragma unroll 1
    for (int c = half * 64; c < half * 64 + 64; c += 32) {
      uint32_t ra[32], rb[32];
      tc::tmem_ld_32x32b_x32(tb + c, ra);
      tc::tmem_ld_32x32b_x32(tb + 128 + c, rb);
      tc::tmem_ld_wait();
      uint4 vh[4];
#pragma unroll
      for (int v = 0; v < 4; ++v) {
        float fa[8], fb[8], fh[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          fa[i] = __uint_as_float(ra[v * 8 + i]);
          fb[i] = __uint_as_float(rb[v * 8 + i]);
          fh[i] = silu_f(fa[i]) * fb[i];
        }
        const int col = nt * 128 + c + v * 8;
        vh[v] = pack8(fh);
        stg_v4(p.out2 + ab_block_index(row, col, F), pack8(fa));
        stg_v4(p.out2 + ab_block_index(row, F + col, F), pack8(fb));
      }
      stage_and_store(tmO, stage, lane, vh, nt * 128 + c, trow);
    }
  } else if (MODE == kDgradDown) {
    const int F = p.F;
    const int f0 = nt * BN;
    const int trow = int(row) - lane;
    float gsum = 0.f;  // this row's sum of dH * H over the warp's columns
#pragma unroll 1
    for (int c = half * (BN / 2); c < (half + 1) * (BN / 2); c += 32) {
      uint4 va[4], vb[4];
#pragma unroll
      for (int v = 0; v < 4; ++v) {
        va[v] = ldg_nc_v4(p.aux + ab_block_index(row, f0 + c + v * 8, F));
        vb[v] = ldg_nc_v4(p.aux + ab_block_index(row, F + f0 + c + v * 8, F));
      }
      uint32_t r[32];
      tc::tmem_ld_32x32b_x32(tb + c, r);
      tc::tmem_ld_wait();
      uint4 vda[4], vdb[4];
#pragma unroll
      for (int v = 0; v < 4; ++v) {
        float fa[8], fb[8], da[8], db[8];
        unpack8(va[v], fa);
        unpack8(vb[v], fb);
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const float dh = __uint_as_float(r[v * 8 + i]);
          const float sg = sigmoid_f(fa[i]);
          da[i] = dh * fb[i] * (sg * (1.f + fa[i] * (1.f - sg)));
          db[i] = dh * fa[i] * sg;
          gsum = fmaf(db[i], fb[i], gsum);  // dh * silu(a) * b = dH * H
        }
        vda[v] = pack8(da);
        vdb[v] = pack8(db);
      }
      stage_and_store(tmO, stage, lane, vda, f0 + c, trow);
      stage_and_store(tmO, stage, lane, vdb, F + f0 + c, trow);
    }
    if (p.gate_partial != nullptr) p.gate_partial[row * p.gate_stride + nt * 2 + half] = gsum;
  } else {
    int trow;
    if (Tr::WGRAD) {
      const int M_out = p.m_tiles_w * BM;
      trow = e * M_out + out_row - lane;
    } else {
      trow = int(row) - lane;
    }
    // combine: this lane's row goes to token `tok` with weight `g` (tok < 0: padding)
    int tok = -1;
    float g = 0.f;
    if (MODE == kDown && p.y_acc != nullptr) {
      tok = p.row_token[row];
      g = p.row_gate[row];
    }
    // dX with the router's term: this lane's row gets dz * W_r[col, e] added (dz = 0 on
    // padding rows); the W_r values of a 32-column chunk are loaded one per lane.
    float dz = 0.f;
    const bool router = MODE == kDgradGateUp && p.row_dz != nullptr;
    if (router) dz = p.row_dz[row];
#pragma unroll 1
    for (int c = half * (BN / 2); c < (half + 1) * (BN / 2); c += 32) {
      uint32_t r[32];
      float w = 0.f;
      if (router) w = __ldg(p.w_router + size_t(nt * BN + c + lane) * p.E + e);
      tc::tmem_ld_32x32b_x32(tb + c, r);
      tc::tmem_ld_wait();
      if (router) {
#pragma unroll
        for (int v = 0; v < 32; ++v)
          r[v] = __float_as_uint(fmaf(dz, __shfl_sync(0xffffffffu, w, v), __uint_as_float(r[v])));
      }
      if (MODE == kDown && tok >= 0) {
        float4 *dst = reinterpret_cast<float4 *>(p.y_acc + size_t(tok) * p.d + nt * BN + c);
#pragma unroll
        for (int q = 0; q < 8; ++q)
          atomicAdd(dst + q, make_float4(g * __uint_as_float(r[4 * q]), g * __uint_as_float(r[4 * q + 1]),
                                         g * __uint_as_float(r[4 * q + 2]), g * __uint_as_float(r[4 * q + 3])));
      }
      if (MODE != kDown || p.out != nullptr) {
        uint4 v[4];
        pack32(r, v);
        stage_and_store(tmO, stage, lane, v, nt * BN + c, trow);
      }
    }
  }
}

// Zeroes this warp's 2 KB staging chunk (after its earlier stores have read it).
__device__ __forceinline__ void zero_fill_stage(uint32_t stage, int lane) {
  if (lane == 0) tc::bulk_wait_read0();
  __syncwarp();
  const uint4 z = make_uint4(0, 0, 0, 0);
#pragma unroll
  for (uint32_t c = 0; c < 4; ++c) st_shared_v4(stage + uint32_t(lane) * 64u + c * 16u, z);
  tc::fence_proxy_async_smem();
  __syncwarp();
}
// One lane: stores the staging chunk to every 32-column chunk of this warp's column
// half of output tile (trow, nt), as one bulk group.
template <int BN>
__device__ __forceinline__ void store_chunks_from(const CUtensorMap *tmO, uint32_t stage, int trow,
                                                  int nt, int half) {
  for (int c = half * (BN / 2); c < (half + 1) * (BN / 2); c += 32)
    tc::tma_store_2d(tmO, stage, nt * BN + c, trow);
  tc::bulk_commit();
}

// Zero weight gradient of an expert without rows: this warp's 32 rows and column half.
template <int BN>
__device__ __forceinline__ void zero_tile_store(const CUtensorMap *tmO, uint32_t stage, int lane,
                                                int trow, int nt, int half) {
  if (lane == 0) tc::bulk_wait_read0();
  __syncwarp();
  const uint4 z = make_uint4(0, 0, 0, 0);
#pragma unroll
  for (uint32_t c = 0; c < 4; ++c) st_shared_v4(stage + uint32_t(lane) * 64u + c * 16u, z);
  tc::fence_proxy_async_smem();
  __syncwarp();
  if (lane == 0) {
    for (int c = half * (BN / 2); c < (half + 1) * (BN / 2); c += 32)
      tc::tma_store_2d(tmO, stage, nt * BN + c, trow);
    tc::bulk_commit();
  }
}

template <int MODE, int BN>
__global__ void __launch_bounds__(kThreads, 1)
    grouped_gemm_kernel(const __grid_constant__ CUtensorMap tmA,
                        const __grid_constant__ CUtensorMap tmB,
                        const __grid_constant__ CUtensorMap tmO, const GemmParams p) {
  using Tr = Traits<MODE>;
  using Sh = Shape<BN>;
  constexpr int STAGES = Sh::STAGES;
  constexpr uint32_t IDESC = tc::idesc_bf16_f32(BM, BN, Tr::A_MN, Tr::B_MN);

  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = tc::smem_u32(smem_raw);
  const uint32_t pad = (1024u - (raw & 1023u)) & 1023u;
  uint8_t *smem = smem_raw + pad;
  const uint32_t sA0 = raw + pad;
  const uint32_t sB0 = sA0 + STAGES * Sh::A_BYTES;
  uint64_t *bars = reinterpret_cast<uint64_t *>(smem + STAGES * Sh::STAGE_BYTES);
  int *misc = reinterpret_cast<int *>(bars + Sh::NBARS);
  int *s_goff = misc + 4;          // [E+1]
  int *s_order = s_goff + 257;     // [E]   experts in schedule order
  int *s_prefix = s_order + 256;   // [E+1] first tile of each scheduled expert
  int *s_key = s_prefix + 257;     // [E]   rows of each expert, -1 when pruned
  const uint32_t stage_base =
      (tc::smem_u32(s_key + 256) + 1023u) & ~1023u;  // epilogue staging, 2 KB per warp
  volatile int *abort_flag = misc + 1;
  volatile int no_abort = 0;

  const uint32_t bar0 = tc::smem_u32(bars);
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (STAGES + s); };
  auto tfull_bar = [&](int a) { return bar0 + 8u * (2 * STAGES + a); };
  auto tempty_bar = [&](int a) { return bar0 + 8u * (2 * STAGES + 2 + a); };
  const uint32_t drain_bar = bar0 + 8u * (2 * STAGES + 4);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int E = p.E;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      tc::mbar_init(full_bar(s), 1);
      tc::mbar_init(empty_bar(s), 1);
    }
    for (int a = 0; a < 2; ++a) {
      tc::mbar_init(tfull_bar(a), 1);
      tc::mbar_init(tempty_bar(a), kEpiWarps);
    }
    tc::mbar_init(drain_bar, 1);
    tc::fence_mbar_init();
    misc[1] = 0;
  }
  if (warp == 0 && lane == 0) {
    tc::tma_prefetch_desc(&tmA);
    tc::tma_prefetch_desc(&tmB);
    tc::tma_prefetch_desc(&tmO);
  }
  if (warp == 1) {
    tc::tmem_alloc(tc::smem_u32(misc), Sh::TMEM_COLS);
    tc::tmem_relinquish();
  }
  // ---- tile schedule, built from the device-resident group offsets ----
  // Weight gradients: experts heaviest first (ties to the lower id), pruned experts
  // (active_mask 0) last with no tile, live experts without rows with tiles of zero
  // k-blocks (their zero gradient). Activation GEMMs: expert order.
  for (int e = threadIdx.x; e <= E; e += kThreads) s_goff[e] = p.group_offsets[e];
  __syncthreads();
  for (int e = threadIdx.x; e < E; e += kThreads) {
    const int rows = s_goff[e + 1] - s_goff[e];
    s_key[e] = (Tr::WGRAD && p.active_mask != nullptr && p.active_mask[e] == 0) ? -1 : rows;
  }
  __syncthreads();
  for (int e = threadIdx.x; e < E; e += kThreads) {
    if (!Tr::WGRAD) {  // equal-cost tiles: expert order, the grouped layout's memory order
      s_order[e] = e;
      continue;
    }
    const int ce = s_key[e];
    int r = 0;
    for (int q = 0; q < E; ++q) {
      const int cq = s_key[q];
      r += (cq > ce) || (cq == ce && q < e);
    }
    s_order[r] = e;
  }
  __syncthreads();
  for (int i = threadIdx.x; i < E; i += kThreads) {  // tiles of list position i
    const int key = s_key[s_order[i]];
    const int mt = p.rows_split == 2 ? (key / BM) & 1 : key / BM;  // odd last block only
    s_prefix[i + 1] = key < 0 ? 0 : Tr::WGRAD ? p.m_tiles_w * p.n_tiles : mt * p.n_tiles;
  }
  __syncthreads();
  if (warp == 0) warp_prefix_counts(s_prefix, E, lane);
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem_base = static_cast<uint32_t>(misc[0]);
  const int total = s_prefix[E];

  auto decode = [&](int tile) {
    int lo = 0, hi = E - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (s_prefix[mid] <= tile) lo = mid; else hi = mid - 1;
    }
    Tile t;
    const int local = tile - s_prefix[lo];
    t.e = s_order[lo];
    t.goff = s_goff[t.e];
    if (!Tr::WGRAD && p.rows_split == 2) {  // the group's last (odd) block, every N tile
      t.mt = (s_goff[t.e + 1] - t.goff) / BM - 1;
      t.nt = local;
    } else {
      t.mt = local / p.n_tiles;
      t.nt = local - t.mt * p.n_tiles;
    }
    t.nkb = Tr::WGRAD ? (s_goff[t.e + 1] - t.goff) / BK : p.nkb;
    return t;
  };

  if (warp == 0) {
    // ===================== TMA producer (one thread) =====================
    if (lane == 0) {
      uint32_t it = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < total && ok; tile += gridDim.x) {
        const Tile t = decode(tile);
        for (int kb = 0; kb < t.nkb; ++kb, ++it) {
          const int s = it % STAGES;
          const uint32_t ph = (it / STAGES) & 1u;
          if (!tc::mbar_wait(empty_bar(s), ph ^ 1u, kWaitLimitNs, abort_flag)) { fail(abort_flag); ok = false; break; }
          tc::mbar_arrive_expect_tx(full_bar(s), Sh::STAGE_BYTES);
          const uint32_t a_dst = sA0 + s * Sh::A_BYTES, b_dst = sB0 + s * Sh::B_BYTES;
          const uint32_t fb = full_bar(s);
          const int k0 = kb * BK;
          if (MODE == kGateUp) {
            const int row0 = t.goff + t.mt * BM;
            tc::tma_load_2d(a_dst, &tmA, fb, k0, row0);
            const int wrow = t.e * 2 * p.F + t.nt * 128;
            tc::tma_load_2d(b_dst, &tmB, fb, k0, wrow);
            tc::tma_load_2d(b_dst + 128 * 128, &tmB, fb, k0, wrow + p.F);
          } else if (MODE == kDown) {
            const int row0 = t.goff + t.mt * BM;
            tc::tma_load_2d(a_dst, &tmA, fb, k0, row0);
#pragma unroll
            for (int i = 0; i < BN / 128; ++i)
              tc::tma_load_2d(b_dst + i * 128 * 128, &tmB, fb, k0, t.e * p.d + t.nt * BN + i * 128);
          } else if (MODE == kDgradDown || MODE == kDgradGateUp) {
            const int row0 = t.goff + t.mt * BM;
            tc::tma_load_2d(a_dst, &tmA, fb, k0, row0);
            const int krow = (MODE == kDgradDown ? t.e * p.d : t.e * 2 * p.F) + k0;
#pragma unroll
            for (int i = 0; i < BN / 64; ++i)
              tc::tma_load_2d(b_dst + i * 64 * 128, &tmB, fb, t.nt * BN + i * 64, krow);
          } else {  // weight gradients: both operands MN-major, K = group rows
            const int krow = t.goff + k0;
#pragma unroll
            for (int i = 0; i < BM / 64; ++i)
              tc::tma_load_2d(a_dst + i * 64 * 128, &tmA, fb, t.mt * BM + i * 64, krow);
#pragma unroll
            for (int i = 0; i < BN / 64; ++i)
              tc::tma_load_2d(b_dst + i * 64 * 128, &tmB, fb, t.nt * BN + i * 64, krow);
          }
        }
      }
      // Drain: every issued load has landed before the CTA may exit (also
      // after an abort, so this wait ignores the abort flag).
      for (int s = 0; s < STAGES; ++s) {
        if (it > uint32_t(s)) {
          const uint32_t n = (it - 1 - s) / STAGES;
          if (!tc::mbar_wait(full_bar(s), n & 1u, kWaitLimitNs, &no_abort)) fail(abort_flag);
        }
      }
    }
  } else if (warp == 1) {
    // ===================== MMA issuer (one thread) =====================
    if (lane == 0) {
      uint32_t it = 0, tcount = 0;
      bool ok = true, issued = false;
      for (int tile = blockIdx.x; tile < total && ok; tile += gridDim.x) {
        const Tile t = decode(tile);
        if (t.nkb == 0) continue;
        const uint32_t a = tcount & 1u, aph = (tcount >> 1) & 1u;
        if (!tc::mbar_wait(tempty_bar(a), aph ^ 1u, kWaitLimitNs, abort_flag)) { fail(abort_flag); break; }
        tc::fence_after_sync();
        const uint32_t d_tmem = tmem_base + a * BN;
        for (int kb = 0; kb < t.nkb; ++kb, ++it) {
          const int s = it % STAGES;
          const uint32_t ph = (it / STAGES) & 1u;
          if (!tc::mbar_wait(full_bar(s), ph, kWaitLimitNs, abort_flag)) { fail(abort_flag); ok = false; break; }
          tc::fence_after_sync();
          const uint32_t a_s = sA0 + s * Sh::A_BYTES, b_s = sB0 + s * Sh::B_BYTES;
#pragma unroll
          for (int kk = 0; kk < BK / UMMA_K; ++kk) {
            const uint64_t ad = Tr::A_MN ? tc::smem_desc_sw128(a_s + kk * 2048, 8192, 1024)
                                         : tc::smem_desc_sw128(a_s + kk * 32, 16, 1024);
            const uint64_t bd = Tr::B_MN ? tc::smem_desc_sw128(b_s + kk * 2048, 8192, 1024)
                                         : tc::smem_desc_sw128(b_s + kk * 32, 16, 1024);
            tc::mma_bf16(d_tmem, ad, bd, IDESC, (kb | kk) != 0);
          }
          tc::mma_commit(empty_bar(s));  // frees the stage once these MMAs finish
          issued = true;
        }
        if (!ok) break;
        tc::mma_commit(tfull_bar(a));  // accumulator ready for the epilogue
        ++tcount;
      }
      if (issued) {  // all issued MMAs complete before TMEM is released
        tc::mma_commit(drain_bar);
        if (!tc::mbar_wait(drain_bar, 0, kWaitLimitNs, &no_abort)) fail(abort_flag);
      }
    }
  } else {
    // ===================== epilogue (warps 2..9) =====================
    const int q = warp & 3;  // TMEM lane quarter this warp may access
    const int half = (warp - 2) / 4;  // column half this warp handles
    const uint32_t stage = stage_base + uint32_t(warp - 2) * kStageBytes;
    const int r_in_tile = q * 32 + lane;
    uint32_t tcount = 0;
    for (int tile = blockIdx.x; tile < total; tile += gridDim.x) {
      const Tile t = decode(tile);
      if (Tr::WGRAD && t.nkb == 0) {
        // empty group: its weight gradient is exactly zero
        const int M_out = p.m_tiles_w * BM;
        zero_tile_store<BN>(&tmO, stage, lane, t.e * M_out + t.mt * BM + q * 32, t.nt, half);
        continue;
      }
      const uint32_t a = tcount & 1u, aph = (tcount >> 1) & 1u;
      const bool ok = tc::mbar_wait(tfull_bar(a), aph, kWaitLimitNs, abort_flag);
      __syncwarp();
      if (!ok) { fail(abort_flag); break; }
      tc::fence_after_sync();
      const uint32_t tb = tmem_base + (uint32_t(q * 32) << 16) + a * BN;

      epilogue_tile<MODE, BN>(p, &tmO, stage, lane, tb,
                              size_t(t.goff) + size_t(t.mt) * BM + r_in_tile,
                              t.mt * BM + r_in_tile, t.e, t.nt, half);
      tc::fence_before_sync();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(tempty_bar(a));
      ++tcount;
    }
    if (lane == 0) tc::bulk_wait0();  // this warp's output stores are complete
    __syncwarp();
  }

  tc::fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem_base, Sh::TMEM_COLS);
  }
}


// ============================================================================
// CTA-pair variant (cta_group::2): a cluster of two CTAs on two SMs computes a
// 256 x BN tile. Each CTA stages its own 128 rows of A and half of B (BN/2 rows)
// per k-block; one thread of the even CTA issues M=256 MMAs that read both CTAs'
// shared memory and write each CTA's 128 accumulator rows into its own TMEM.
// Per SM this moves 32 KB per 64-deep k-block instead of 48 KB through shared
// memory and L2; the ring holds 3 stages of 128-deep k-blocks (BN 256) or 4
// (BN 128), and 6 or 8 64-deep stages in the gathered-operand variant.
// Synchronization: both CTAs' loads complete on the even CTA's `full` barrier
// (it expects both CTAs' bytes); the MMA commit arrives on the `empty` and
// `tfull` barriers of both CTAs; both CTAs' epilogue warps arrive on the even
// CTA's `tempty` barrier. Tiles whose odd row block lies past the group (a group
// with an odd number of 128-row blocks) are computed on a zero-filled A box and not
// stored; on 2^18 or more grouped rows the activation GEMMs leave those blocks to the
// one-SM kernel (see run_gemm_out).
// ============================================================================
// KB = k-block depth of one ring stage: 128 (two 64-wide swizzle blocks of each
// operand, K-half h at h * 16 KB of A and h * BNH * 128 bytes of B), or 64 for the
// gathered-operand variant. Deeper stages halve the barrier waits, descriptor setup and
// commits per FLOP (measured -2.5% to -4.4% cycles per k-block) at the same bytes in flight.
// Claim hand-off ring of the CTA-pair kernel: the even CTA's producer claims units (a
// tile, or several tiles of a light expert) and publishes each one in a slot of both
// CTAs' rings; the odd CTA's producer and the MMA issuer read it there. A slot is
// rewritten kRing units later, which the load ring's STAGES (< kRing) bound: a producer
// can run at most STAGES k-blocks, hence STAGES units, ahead of the MMAs that need the
// other readers' progress.
constexpr int kRing = 16;
// Row pairs per block of the weight-gradient tile order (see tile_in).
constexpr int kWgradBlock = 8;

template <int BN, int KB> struct PairShape {
  static constexpr int BNH = BN / 2;  // B rows staged by each CTA
  static constexpr int STAGES = KB == 128 ? (BN == 256 ? 3 : 4) : (BN == 256 ? 6 : 8);
  static_assert(STAGES + 1 < kRing, "the tile ring must outlast the load ring");
  static constexpr uint32_t A_BYTES = BM * KB * 2;
  static constexpr uint32_t B_BYTES = BNH * KB * 2;
  static constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
  // full/empty per stage, tfull/tempty per accumulator, drain, tile ring, epilogue tile
  static constexpr int NBARS = 2 * STAGES + 5 + kRing + 2;
  static constexpr size_t SMEM = 1024 + size_t(STAGES) * STAGE_BYTES + NBARS * 8 +
                                 (4 + 257 + 256 + 257 + 256 + kRing + 2) * 4 + 1024 + kEpiWarps * 2048;
  static constexpr uint32_t TMEM_COLS = 2 * BN;
};

struct PairTile {
  int e, goff, mp, nt, nkb, mtiles;
};

// A claim unit: tiles lt0 .. lt0 + cnt - 1 (in the expert's tile order) of expert e.
struct PairUnit {
  int e, goff, nkb, mtiles, lt0, cnt;
};

// Tiles of one claim unit of the dynamic weight-gradient schedule, from the expert's
// k-blocks per tile: light experts' tiles (one to seven 128-row k-blocks) are claimed,
// published to the pair and handed to the epilogue warps several at a time, about eight
// k-blocks of work per claim. Each hand-off costs the single producer and MMA-issuer
// threads ~2,000 cycles (a cluster-scope release and arrive), which one tile of one
// k-block (~1,000 cycles of MMA) could not hide.
__host__ __device__ constexpr int unit_tiles(int nkb) {
  return nkb >= 8 ? 1 : nkb >= 4 ? 2 : nkb >= 2 ? 4 : 8;
}

__device__ __forceinline__ int4 ld_rows4(const int32_t *p) {
  return __ldg(reinterpret_cast<const int4 *>(p));
}

// GATHER (kGateUp, kWgradGateUp): the X_perm operand is read from x through
// token_of_row with 4-row TMA gathers, so X_perm is never materialized. The whole
// producer warp issues them, one gather of 4 rows per lane and k-block: the 128
// A rows of the tile (kGateUp), or 2 x 64 k-rows of B (kWgradGateUp, whose row
// indices change every k-block and are loaded one k-block ahead). Measured on
// GB300 at T=16384, d=4096, 48 live experts: both GEMMs take ~3.3x as long as with
// X_perm tile loads (each k-block needs 32 gathers of 4 x 128 bytes where one tile
// load moves 128 rows; the per-instruction cost of the gathers sets the pace).
template <int MODE, int BN, bool GATHER>
__global__ void __launch_bounds__(kThreads, 1)
    grouped_gemm_pair_kernel(const __grid_constant__ CUtensorMap tmA,
                             const __grid_constant__ CUtensorMap tmB,
                             const __grid_constant__ CUtensorMap tmO, const GemmParams p) {
  using Tr = Traits<MODE>;
  constexpr int KB = GATHER ? 64 : 128;
  using Sh = PairShape<BN, KB>;
  constexpr int STAGES = Sh::STAGES;
  constexpr int BNH = Sh::BNH;
  constexpr uint32_t IDESC = tc::idesc_bf16_f32(2 * BM, BN, Tr::A_MN, Tr::B_MN);

  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = tc::smem_u32(smem_raw);
  const uint32_t pad = (1024u - (raw & 1023u)) & 1023u;
  uint8_t *smem = smem_raw + pad;
  const uint32_t sA0 = raw + pad;
  const uint32_t sB0 = sA0 + STAGES * Sh::A_BYTES;
  uint64_t *bars = reinterpret_cast<uint64_t *>(smem + STAGES * Sh::STAGE_BYTES);
  int *misc = reinterpret_cast<int *>(bars + Sh::NBARS);
  int *s_goff = misc + 4;
  int *s_order = s_goff + 257;
  int *s_prefix = s_order + 256;
  int *s_key = s_prefix + 257;            // [E] rows of each expert, -1 when pruned (wgrad)
  volatile int *s_ring = s_key + 256;     // [kRing] unit hand-off (see kRing)
  volatile int *s_epi = s_ring + kRing;   // [2] unit of each parity of the unit count, for the epilogue
  const uint32_t stage_base =
      (tc::smem_u32(const_cast<int *>(s_epi + 2)) + 1023u) & ~1023u;  // epilogue staging, 2 KB per warp
  volatile int *abort_flag = misc + 1;
  volatile int no_abort = 0;

  const uint32_t bar0 = tc::smem_u32(bars);
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (STAGES + s); };
  auto tfull_bar = [&](int a) { return bar0 + 8u * (2 * STAGES + a); };
  auto tempty_bar = [&](int a) { return bar0 + 8u * (2 * STAGES + 2 + a); };
  const uint32_t drain_bar = bar0 + 8u * (2 * STAGES + 4);
  auto ring_bar = [&](int r) { return bar0 + 8u * (2 * STAGES + 5 + r); };
  auto epi_bar = [&](int a) { return bar0 + 8u * (2 * STAGES + 5 + kRing + a); };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int E = p.E;
  const uint32_t rank = tc::cluster_ctarank();
  const bool leader = rank == 0;
  const int cluster = int(tc::cluster_id_x());
  const int nclusters = int(tc::cluster_count_x());

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      tc::mbar_init(full_bar(s), 1);
      tc::mbar_init(empty_bar(s), 1);
    }
    for (int a = 0; a < 2; ++a) {
      tc::mbar_init(tfull_bar(a), 1);
      tc::mbar_init(tempty_bar(a), 2 * kEpiWarps);  // the epilogue warps of both CTAs
      tc::mbar_init(epi_bar(a), 1);                 // the even CTA's MMA issuer
    }
    for (int r = 0; r < kRing; ++r) tc::mbar_init(ring_bar(r), 1);  // the even CTA's producer
    tc::mbar_init(drain_bar, 1);
    tc::fence_mbar_init();
    misc[1] = 0;
    misc[2] = 0;  // live experts without rows (weight gradients)
    misc[3] = 0;  // pruned experts
  }
  if (warp == 0 && lane == 0) {
    tc::tma_prefetch_desc(&tmA);
    tc::tma_prefetch_desc(&tmB);
    tc::tma_prefetch_desc(&tmO);
  }
  if (warp == 1) {
    tc::tmem_alloc_pair(tc::smem_u32(misc), Sh::TMEM_COLS);
    tc::tmem_relinquish_pair();
  }
  // ---- tile list: identical in both CTAs of every pair ----
  // Weight gradients (a tile costs as much as its expert has rows): experts in descending
  // order of rows (ties to the lower id), the longest-processing-time order of Algorithm
  // 2's greedy balancing; a pair that runs out of work claims the next tile of this list,
  // i.e. the heaviest tile left goes to the least-loaded pair. Pruned experts (active_mask
  // 0) come last and get nothing; live experts without rows come before them and get no
  // tile either (their zero gradients are stored by the epilogue warps up front, while the
  // first tiles' MMAs run). Activation GEMMs (every tile costs the same): expert order,
  // which follows the grouped layout in memory (measured 1-2% faster than heaviest first).
  for (int e = threadIdx.x; e <= E; e += kThreads) s_goff[e] = p.group_offsets[e];
  __syncthreads();
  for (int e = threadIdx.x; e < E; e += kThreads) {
    const int rows = s_goff[e + 1] - s_goff[e];
    s_key[e] = (Tr::WGRAD && p.active_mask != nullptr && p.active_mask[e] == 0) ? -1 : rows;
  }
  __syncthreads();
  for (int e = threadIdx.x; e < E; e += kThreads) {
    if (!Tr::WGRAD) {  // equal-cost tiles: expert order, the grouped layout's memory order
      s_order[e] = e;
      continue;
    }
    const int ce = s_key[e];
    int r = 0;
    for (int q = 0; q < E; ++q) {
      const int cq = s_key[q];
      r += (cq > ce) || (cq == ce && q < e);
    }
    s_order[r] = e;
  }
  __syncthreads();
  const bool dyn = Tr::WGRAD && p.dynamic;
  // claim units of list position i (tiles, or groups of light experts' tiles when dyn) at
  // s_prefix[i + 1], then one warp's scan; measured before as a loop of one thread over the
  // experts, ~9.5 us per launch (36 us in the weight gradients, with the mask read from
  // global memory by the sort)
  for (int i = threadIdx.x; i < E; i += kThreads) {
    const int key = s_key[s_order[i]];
    int units = 0;
    if (Tr::WGRAD && key <= 0) {
      atomicAdd(&misc[key < 0 ? 3 : 2], 1);  // pruned / live without rows: no tile
    } else {
      const int mt = Tr::WGRAD ? p.m_tiles_w : key / BM;
      // pairs of row blocks; with rows_split == 1 a last odd block is left to the one-SM kernel
      const int tiles = ((p.rows_split == 1 ? mt : mt + 1) / 2) * p.n_tiles;
      const int g = dyn ? unit_tiles(key / KB) : 1;
      units = (tiles + g - 1) / g;
    }
    s_prefix[i + 1] = units;
  }
  __syncthreads();
  if (warp == 0) warp_prefix_counts(s_prefix, E, lane);
  tc::fence_before_sync();
  __syncthreads();
  tc::cluster_sync();  // barriers of both CTAs initialized before any remote use
  tc::fence_after_sync();
  const uint32_t tmem_base = static_cast<uint32_t>(misc[0]);
  const int total = s_prefix[E];

  // Every role of a pair sees the pair's tiles in increasing order (a fixed stride, or
  // claims from a counter that only grows), so the expert of the next tile is found by
  // walking forward from the previous one: a step or two of shared-memory reads per
  // tile instead of a binary search over all experts (measured ~1,100 cycles per tile,
  // which one-k-block tiles of light experts could not hide).
  int cursor = 0;
  auto decode_unit = [&](int unit) {
    int lo = s_prefix[cursor] <= unit ? cursor : 0;
    while (lo + 1 < E && s_prefix[lo + 1] <= unit) ++lo;
    cursor = lo;
    PairUnit u;
    u.e = s_order[lo];
    u.goff = s_goff[u.e];
    const int rows = s_goff[u.e + 1] - u.goff;
    u.nkb = Tr::WGRAD ? rows / KB : p.nkb / (KB / BK);
    u.mtiles = Tr::WGRAD ? p.m_tiles_w : rows / BM;
    const int g = dyn ? unit_tiles(u.nkb) : 1;
    u.lt0 = (unit - s_prefix[lo]) * g;
    u.cnt = min(g, ((p.rows_split == 1 ? u.mtiles : u.mtiles + 1) / 2) * p.n_tiles - u.lt0);
    return u;
  };
  // Tile j of a unit: the expert's tile lt0 + j as (row pair, column tile).
  auto tile_in = [&](const PairUnit &u, int j) {
    PairTile t;
    const int local = u.lt0 + j;
    t.e = u.e;
    t.goff = u.goff;
    t.nkb = u.nkb;
    t.mtiles = u.mtiles;
    if (Tr::WGRAD && p.n_tiles > kWgradBlock) {
      // Weight gradients with many column tiles: an expert's (row pair, column) tiles in
      // blocks of kWgradBlock row pairs, column by column inside a block, so that the
      // tiles the pairs run at the same time (consecutive in the list) share few operand
      // panels: about kWgradBlock row panels and 76 / kWgradBlock column panels per wave
      // instead of 3 row and 28 column panels (dW_gate_up at d_model = 7168). The pairs
      // of a wave move through the reduction (the expert's rows) together, and each
      // panel slice they share is read from DRAM once: measured at d_model = 7168,
      // 65,536 rows over 8 experts, dW_gate_up read 3.8 GB instead of 6.9 GB and ran
      // 8% faster. With few column tiles (dW_down: 8) the rows-first order already
      // shares as few panels and stays.
      const int MP = (p.m_tiles_w + 1) / 2;
      const int blk = local / (kWgradBlock * p.n_tiles);
      const int rem = local - blk * kWgradBlock * p.n_tiles;
      const int bh = min(kWgradBlock, MP - blk * kWgradBlock);
      t.nt = rem / bh;
      t.mp = blk * kWgradBlock + (rem - t.nt * bh);
    } else {
      t.mp = local / p.n_tiles;
      t.nt = local - t.mp * p.n_tiles;
    }
    return t;
  };

  // ---- claim units. The weight gradients' tiles differ in cost (K = the expert's rows):
  // there the even CTA's producer takes unit number n of this pair, the pair's index for
  // n = 0, then the next unclaimed unit of the list (an atomic counter shared by all
  // pairs), -1 once the list is exhausted. It writes the unit into slot n % kRing of both
  // CTAs' rings and arrives on the slots' barriers before it issues the unit's loads; the
  // odd CTA's producer and the MMA issuer wait there, and the MMA issuer passes each unit
  // on to both CTAs' epilogue warps through s_epi[n % 2] and epi_bar[n % 2] once the
  // accumulator buffer of the unit's first tile is free. The activation GEMMs' tiles all
  // cost the same (and with p.dynamic == 0 the weight gradients' too): a unit is one tile,
  // and every role of a pair computes its unit numbers itself, cluster, cluster +
  // nclusters, ..., with no hand-off.
  auto static_unit = [&](uint32_t n) -> int {
    const int unit = cluster + int(n) * nclusters;
    return unit < total ? unit : -1;
  };
  const uint32_t ring_peer = tc::mapa(tc::smem_u32(const_cast<int *>(s_ring)), 1);
  const uint32_t ring_bar_peer = tc::mapa(ring_bar(0), 1);
  int claimed = cluster;  // even CTA's producer: the unit it publishes next
  // Returns this pair's unit number n (-1: no more), or -2 after a failed wait.
  auto next_unit = [&](uint32_t n) -> int {
    if (!dyn) return static_unit(n);
    const int slot = int(n % kRing);
    if (leader) {
      const int v = claimed < total ? claimed : -1;
      s_ring[slot] = v;
      tc::st_cluster_u32(ring_peer + 4u * slot, v);
      tc::mbar_arrive(ring_bar(slot));
      tc::mbar_arrive_cluster(ring_bar_peer + 8u * slot);
      if (v >= 0) claimed = nclusters + atomicAdd(p.sched_ctr, 1);
      return v;
    }
    if (!tc::mbar_wait_cluster(ring_bar(slot), (n / kRing) & 1u, kWaitLimitNs, abort_flag)) {
      fail(abort_flag);
      return -2;
    }
    return s_ring[slot];
  };

  if (warp == 0 && GATHER) {
    // ============ TMA producer, gathered operand (the whole warp in each CTA) ============
    const uint32_t full_leader = tc::mapa(full_bar(0), 0);
    const int box = lane >> 4, grp = lane & 15;  // kWgradGateUp: B box and 4-row group
    uint32_t it = 0;
    bool ok = true;
    for (uint32_t n = 0; ok; ++n) {
      int unit = 0;
      if (lane == 0) unit = next_unit(n);
      unit = __shfl_sync(0xffffffffu, unit, 0);
      if (unit < 0) break;
      const PairUnit u = decode_unit(unit);
      for (int j = 0; j < u.cnt && ok; ++j) {
        const PairTile t = tile_in(u, j);
        const int mt = 2 * t.mp + int(rank);
        int4 rows4 = make_int4(0, 0, 0, 0), nxt = make_int4(0, 0, 0, 0);
        // kGateUp: this lane's 4 rows of the tile (token 0 for the row block past an
        // odd group end, which is computed but not stored)
        if (MODE == kGateUp && mt < t.mtiles) rows4 = ld_rows4(p.token_of_row + t.goff + mt * BM + 4 * lane);
        if (MODE == kWgradGateUp && t.nkb > 0) nxt = ld_rows4(p.token_of_row + t.goff + 4 * grp);
        for (int kb = 0; kb < t.nkb; ++kb, ++it) {
          const int s = it % STAGES;
          const uint32_t ph = (it / STAGES) & 1u;
          if (MODE == kWgradGateUp) {
            rows4 = nxt;
            if (kb + 1 < t.nkb) nxt = ld_rows4(p.token_of_row + t.goff + (kb + 1) * BK + 4 * grp);
          }
          int w_ok = 1;
          if (lane == 0) w_ok = tc::mbar_wait(empty_bar(s), ph ^ 1u, kWaitLimitNs, abort_flag) ? 1 : 0;
          w_ok = __shfl_sync(0xffffffffu, w_ok, 0);
          if (!w_ok) {
            if (lane == 0) fail(abort_flag);
            ok = false;
            break;
          }
          const uint32_t a_dst = sA0 + s * Sh::A_BYTES, b_dst = sB0 + s * Sh::B_BYTES;
          const uint32_t fb = full_leader + 8u * s;
          const int k0 = kb * BK;
          if (lane == 0) {
            if (leader) tc::mbar_arrive_expect_tx(full_bar(s), 2 * Sh::STAGE_BYTES);
            if (MODE == kGateUp) {  // even CTA: gate rows, odd CTA: up rows
              tc::tma_load_2d_pair(b_dst, &tmB, fb, k0, t.e * 2 * p.F + int(rank) * p.F + t.nt * 128);
            } else {  // A = [dA | dB] of the group, MN-major
              const int krow = t.goff + k0;
#pragma unroll
              for (int i = 0; i < BM / 64; ++i)
                tc::tma_load_2d_pair(a_dst + i * 64 * 128, &tmA, fb, mt * BM + i * 64, krow);
            }
          }
          if (MODE == kGateUp) {
            tc::tma_gather4_pair(a_dst + uint32_t(lane) * 512u, &tmA, fb, k0, rows4.x, rows4.y,
                                 rows4.z, rows4.w);
          } else if (box < BNH / 64) {
            tc::tma_gather4_pair(b_dst + uint32_t(box) * 64u * 128u + uint32_t(grp) * 512u, &tmB, fb,
                                 t.nt * BN + int(rank) * BNH + box * 64, rows4.x, rows4.y, rows4.z,
                                 rows4.w);
          }
        }
      }
    }
    // Drain (even CTA): its full barriers count the loads of both CTAs.
    if (leader && lane == 0) {
      for (int s = 0; s < STAGES; ++s) {
        if (it > uint32_t(s)) {
          const uint32_t n = (it - 1 - s) / STAGES;
          if (!tc::mbar_wait(full_bar(s), n & 1u, kWaitLimitNs, &no_abort)) fail(abort_flag);
        }
      }
    }
  } else if (warp == 0) {
    // ============ TMA producer (one thread in each CTA) ============
    if (lane == 0) {
      const uint32_t full_leader = tc::mapa(full_bar(0), 0);
      uint32_t it = 0;
      bool ok = true;
      for (uint32_t n = 0; ok; ++n) {
        const int unit = next_unit(n);
        if (unit < 0) break;
        const PairUnit u = decode_unit(unit);
        for (int j = 0; j < u.cnt && ok; ++j) {
          const PairTile t = tile_in(u, j);
          const int mt = 2 * t.mp + int(rank);  // this CTA's 128-row block
          for (int kb = 0; kb < t.nkb; ++kb, ++it) {
            const int s = it % STAGES;
            const uint32_t ph = (it / STAGES) & 1u;
            if (!tc::mbar_wait(empty_bar(s), ph ^ 1u, kWaitLimitNs, abort_flag)) { fail(abort_flag); ok = false; break; }
            if (leader) tc::mbar_arrive_expect_tx(full_bar(s), 2 * Sh::STAGE_BYTES);
            const uint32_t a_dst = sA0 + s * Sh::A_BYTES, b_dst = sB0 + s * Sh::B_BYTES;
            const uint32_t fb = full_leader + 8u * s;
            const int k0 = kb * KB;
            // K-major operands: one box per 64-deep K half (the 128-byte swizzle row), half h
            // at h * rows * 128 bytes. MN-major operands: one box of 64 columns x KB k-rows per
            // 64 columns, column block i at i * KB * 128 bytes (half as many loads).
            if (Tr::A_MN) {  // weight gradients: [dA|dB] or dO of the group, K = group rows
#pragma unroll
              for (int i = 0; i < BM / 64; ++i)
                tc::tma_load_2d_pair(a_dst + i * (KB * 128), &tmA, fb, mt * BM + i * 64, t.goff + k0);
            } else {
              // A row block past the expert's last one (the odd CTA of a pair tile over an
              // odd number of blocks): a box wholly above the tensor, which TMA fills with
              // zeros without reading memory, instead of the next expert's rows
              const int arow = mt < t.mtiles ? t.goff + mt * BM : -2 * BM;
#pragma unroll
              for (int h = 0; h < KB / 64; ++h)
                tc::tma_load_2d_pair(a_dst + h * (BM * 128), &tmA, fb, k0 + h * 64, arow);
            }
            if (Tr::B_MN) {
              const int krow = (MODE == kDgradDown ? t.e * p.d : MODE == kDgradGateUp ? t.e * 2 * p.F : t.goff) + k0;
#pragma unroll
              for (int i = 0; i < BNH / 64; ++i)
                tc::tma_load_2d_pair(b_dst + i * (KB * 128), &tmB, fb, t.nt * BN + int(rank) * BNH + i * 64, krow);
            } else {
              // kGateUp: even CTA gate rows, odd CTA up rows; kDown: rows of W_down
              const int brow = MODE == kGateUp ? t.e * 2 * p.F + int(rank) * p.F + t.nt * 128
                                               : t.e * p.d + t.nt * BN + int(rank) * BNH;
#pragma unroll
              for (int h = 0; h < KB / 64; ++h)
                tc::tma_load_2d_pair(b_dst + h * (BNH * 128), &tmB, fb, k0 + h * 64, brow);
            }
          }
        }
      }
      // Drain (even CTA): its full barriers count the loads of both CTAs.
      if (leader) {
        for (int s = 0; s < STAGES; ++s) {
          if (it > uint32_t(s)) {
            const uint32_t n = (it - 1 - s) / STAGES;
            if (!tc::mbar_wait(full_bar(s), n & 1u, kWaitLimitNs, &no_abort)) fail(abort_flag);
          }
        }
      }
    }
  } else if (warp == 1) {
    // ============ MMA issuer (one thread of the even CTA) ============
    if (leader && lane == 0) {
      const uint32_t epi_peer = tc::mapa(tc::smem_u32(const_cast<int *>(s_epi)), 1);
      const uint32_t epi_bar_peer = tc::mapa(epi_bar(0), 1);
      uint32_t it = 0;
      bool ok = true, issued = false;
      uint32_t nt_done = 0;  // tiles issued: tile i accumulates in buffer i % 2
      for (uint32_t n = 0; ok; ++n) {
        int unit;
        if (dyn) {
          const int slot = int(n % kRing);
          if (!tc::mbar_wait(ring_bar(slot), (n / kRing) & 1u, kWaitLimitNs, abort_flag)) { fail(abort_flag); break; }
          unit = s_ring[slot];
        } else {
          unit = static_unit(n);
          if (unit < 0) break;
        }
        // The buffer of the unit's first tile is free: the epilogue warps are done with
        // tile nt_done - 2, hence have read the unit that slot n % 2 held before.
        {
          const uint32_t a = nt_done & 1u, aph = (nt_done >> 1) & 1u;
          if (!tc::mbar_wait(tempty_bar(a), aph ^ 1u, kWaitLimitNs, abort_flag)) { fail(abort_flag); break; }
        }
        if (dyn) {
          // the epilogue warps of both CTAs learn the unit (-1: no more units)
          const uint32_t e_slot = n & 1u;
          s_epi[e_slot] = unit;
          tc::st_cluster_u32(epi_peer + 4u * e_slot, unit);
          tc::mbar_arrive(epi_bar(e_slot));
          tc::mbar_arrive_cluster(epi_bar_peer + 8u * e_slot);
        }
        if (unit < 0) break;
        tc::fence_after_sync();
        const PairUnit u = decode_unit(unit);
        for (int j = 0; j < u.cnt && ok; ++j, ++nt_done) {
          const uint32_t a = nt_done & 1u, aph = (nt_done >> 1) & 1u;
          if (j > 0) {
            if (!tc::mbar_wait(tempty_bar(a), aph ^ 1u, kWaitLimitNs, abort_flag)) { fail(abort_flag); ok = false; break; }
            tc::fence_after_sync();
          }
          const PairTile t = tile_in(u, j);
          const uint32_t d_tmem = tmem_base + a * BN;
          for (int kb = 0; kb < t.nkb; ++kb, ++it) {
            const int s = it % STAGES;
            const uint32_t ph = (it / STAGES) & 1u;
            if (!tc::mbar_wait(full_bar(s), ph, kWaitLimitNs, abort_flag)) { fail(abort_flag); ok = false; break; }
            tc::fence_after_sync();
            const uint32_t a_s = sA0 + s * Sh::A_BYTES, b_s = sB0 + s * Sh::B_BYTES;
#pragma unroll
            for (int kk = 0; kk < KB / UMMA_K; ++kk) {
              // K-major: K-half kk / 4 of the stage, 16-wide step kk % 4 inside it (32 bytes
              // along the swizzled row). MN-major: k-rows 16 kk .. 16 kk + 15 of every
              // 64-column block (2 KB each), blocks KB * 128 bytes apart.
              const uint32_t ha = uint32_t(kk >> 2) * (BM * 128), hb = uint32_t(kk >> 2) * (BNH * 128);
              const int q = kk & 3;
              const uint64_t ad = Tr::A_MN ? tc::smem_desc_sw128(a_s + kk * 2048, KB * 128, 1024)
                                           : tc::smem_desc_sw128(a_s + ha + q * 32, 16, 1024);
              const uint64_t bd = Tr::B_MN ? tc::smem_desc_sw128(b_s + kk * 2048, KB * 128, 1024)
                                           : tc::smem_desc_sw128(b_s + hb + q * 32, 16, 1024);
              tc::mma_bf16_pair(d_tmem, ad, bd, IDESC, (kb | kk) != 0);
            }
            tc::mma_commit_pair_mc(empty_bar(s), 0x3);  // frees the stage in both CTAs
            issued = true;
          }
          if (!ok) break;
          tc::mma_commit_pair_mc(tfull_bar(a), 0x3);  // both halves of the accumulator ready
        }
      }
      if (issued) {
        tc::mma_commit_pair(drain_bar);
        if (!tc::mbar_wait(drain_bar, 0, kWaitLimitNs, &no_abort)) fail(abort_flag);
      }
    }
  } else {
    // ============ epilogue (warps 2..9 of each CTA) ============
    const int q = warp & 3;
    const int half = (warp - 2) / 4;
    const uint32_t stage = stage_base + uint32_t(warp - 2) * kStageBytes;
    const int r_in_tile = q * 32 + lane;
    const uint32_t tempty_leader = tc::mapa(tempty_bar(0), 0);
    if (Tr::WGRAD) {
      // Live experts without rows: their weight gradient is exactly zero. Units of 128
      // rows x BN columns, spread over all CTAs; every store reads the same zeroed chunk.
      const int n_empty = misc[2], n_pruned = misc[3];
      const int per_e = p.m_tiles_w * p.n_tiles;
      const int units = n_empty * per_e;
      if (int(blockIdx.x) < units) {
        const int M_out = p.m_tiles_w * BM;
        zero_fill_stage(stage, lane);
        for (int u = int(blockIdx.x); u < units; u += int(gridDim.x)) {
          const int e = s_order[E - n_pruned - n_empty + u / per_e];
          const int rem = u % per_e;
          const int mb = rem / p.n_tiles, nt = rem - mb * p.n_tiles;
          if (lane == 0) store_chunks_from<BN>(&tmO, stage, e * M_out + mb * BM + q * 32, nt, half);
        }
      }
    }
    uint32_t nt_done = 0;  // tiles finished: tile i is in accumulator buffer i % 2
    bool ok = true;
    for (uint32_t n = 0; ok; ++n) {
      int unit;
      if (dyn) {
        const uint32_t e_slot = n & 1u;
        ok = tc::mbar_wait_cluster(epi_bar(e_slot), (n >> 1) & 1u, kWaitLimitNs, abort_flag);
        __syncwarp();
        if (!ok) { fail(abort_flag); break; }
        unit = s_epi[e_slot];
      } else {
        unit = static_unit(n);
      }
      if (unit < 0) break;
      const PairUnit u = decode_unit(unit);
      for (int j = 0; j < u.cnt; ++j, ++nt_done) {
        const uint32_t a = nt_done & 1u, aph = (nt_done >> 1) & 1u;
        const PairTile t = tile_in(u, j);
        const int mt = 2 * t.mp + int(rank);
        const bool mine = mt < t.mtiles;  // this CTA's row block exists
        ok = tc::mbar_wait(tfull_bar(a), aph, kWaitLimitNs, abort_flag);
        __syncwarp();
        if (!ok) { fail(abort_flag); break; }
        tc::fence_after_sync();
        const uint32_t tb = tmem_base + (uint32_t(q * 32) << 16) + a * BN;
        if (Tr::WGRAD) {
          // Weight gradients: the whole column half into registers with one wait, the
          // accumulator back to the MMA issuer, then the stores. A light expert's tile
          // (one or two k-blocks) takes less MMA time than its epilogue, which sets the pace
          // there: measured ~4,600 cycles per tile with a load and a wait per 32 columns.
          uint32_t r[BN / 2];
          if (mine) {
#pragma unroll
            for (int c = 0; c < BN / 2; c += 32)
              tc::tmem_ld_32x32b_x32(tb + half * (BN / 2) + c, *reinterpret_cast<uint32_t(*)[32]>(&r[c]));
            tc::tmem_ld_wait();
          }
          tc::fence_before_sync();
          __syncwarp();
          if (lane == 0) tc::mbar_arrive_cluster(tempty_leader + 8u * a);
          if (mine) {
            const int trow = t.e * (p.m_tiles_w * BM) + mt * BM + q * 32;
#pragma unroll
            for (int c = 0; c < BN / 2; c += 32) {
              uint4 v[4];
              pack32(*reinterpret_cast<const uint32_t(*)[32]>(&r[c]), v);
              stage_and_store(&tmO, stage, lane, v, t.nt * BN + half * (BN / 2) + c, trow);
            }
          }
          continue;
        }
        if (mine) {
          epilogue_tile<MODE, BN>(p, &tmO, stage, lane, tb,
                                  size_t(t.goff) + size_t(mt) * BM + r_in_tile,
                                  mt * BM + r_in_tile, t.e, t.nt, half);
        }
        tc::fence_before_sync();
        __syncwarp();
        if (lane == 0) tc::mbar_arrive_cluster(tempty_leader + 8u * a);
      }
    }
    if (lane == 0) tc::bulk_wait0();  // this warp's output stores are complete
    __syncwarp();
  }

  tc::fence_before_sync();
  __syncthreads();
  tc::cluster_sync();  // no CTA leaves while its peer may still signal it
  if (warp == 1) {
    tc::fence_after_sync();
    tc::tmem_dealloc_pair(tmem_base, Sh::TMEM_COLS);
  }
}

// ------------------------------------------------------------------ host side

using moe::make_map;

// The CTA-pair kernel runs every shape; MOE_GEMM_1SM=1 selects the one-SM kernel
// instead (kept for A/B measurements of the two forms).
template <int MODE> bool use_pair() {
  static int v = -1;
  if (v < 0) {
    const char *e = getenv("MOE_GEMM_1SM");
    v = (e && e[0] == '1') ? 0 : 1;
  }
  return v == 1;
}

// The CTA pairs claim tiles from a shared counter (Algorithm 2's greedy, online);
// MOE_GEMM_STATIC=1 gives every pair a fixed stride of the list instead (for A/B runs).
bool sched_dynamic() {
  static int v = -1;
  if (v < 0) {
    const char *e = getenv("MOE_GEMM_STATIC");
    v = (e && e[0] == '1') ? 0 : 1;
  }
  return v == 1;
}

// Points p at the tile counter in the first bytes of the caller's workspace.
int use_sched_ws(GemmParams &p, void *ws, size_t ws_bytes, const char *fn) {
  if (!ws || !moe::aligned16(ws) || ws_bytes < moe::kGemmSchedBytes)
    return moe::set_error(MOE_ERR_WORKSPACE,
                          "%s: workspace of at least %zu bytes, 16-byte aligned, needed", fn,
                          moe::kGemmSchedBytes);
  p.sched_ctr = static_cast<int *>(ws);
  p.dynamic = sched_dynamic() ? 1 : 0;
  return MOE_OK;
}

template <int MODE, int BN>
int launch_one(const CUtensorMap &a, const CUtensorMap &b, const CUtensorMap &o,
               const GemmParams &p, cudaStream_t s, const char *what) {
  using Sh = Shape<BN>;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(grouped_gemm_kernel<MODE, BN>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, int(Sh::SMEM));
    if (e != cudaSuccess) return moe::cuda_status(e, what);
    attr = true;
  }
  MOE_LAUNCH(kGemmName[MODE], s, grouped_gemm_kernel<MODE, BN><<<moe::num_sms(), kThreads, Sh::SMEM, s>>>(a, b, o, p));
  return moe::launch_status(what);
}

template <int MODE, int BN, bool GATHER>
int launch_pair(const CUtensorMap &a, const CUtensorMap &b, const CUtensorMap &o,
                const GemmParams &p, cudaStream_t s, const char *what) {
  using Sh = PairShape<BN, GATHER ? 64 : 128>;
  auto kern = grouped_gemm_pair_kernel<MODE, BN, GATHER>;
  cudaLaunchAttribute at[2];
  at[0].id = cudaLaunchAttributeClusterDimension;
  at[0].val.clusterDim.x = 2;
  at[0].val.clusterDim.y = 1;
  at[0].val.clusterDim.z = 1;
  // the highest scheduling priority: a kernel launched beside it on another stream
  // does not take the SMs its persistent CTA pairs are waiting for
  static int prio = [] {
    int least = 0, greatest = 0;
    cudaDeviceGetStreamPriorityRange(&least, &greatest);
    return greatest;
  }();
  at[1].id = cudaLaunchAttributePriority;
  at[1].val.priority = prio;
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = Sh::SMEM;
  cfg.stream = s;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  static int nclusters = 0;
  if (!nclusters) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, int(Sh::SMEM));
    if (e != cudaSuccess) return moe::cuda_status(e, what);
    cfg.gridDim = dim3(2 * (moe::num_sms() / 2));
    int n = 0;
    e = cudaOccupancyMaxActiveClusters(&n, kern, &cfg);
    if (e != cudaSuccess) return moe::cuda_status(e, what);
    if (n <= 0) return moe::set_error(MOE_ERR_CUDA, "%s: no co-resident CTA pair fits", what);
    nclusters = n;
  }
  cfg.gridDim = dim3(2 * nclusters);
  cfg.numAttrs = 2;
  if (p.dynamic) {  // the tile counter starts at zero for every launch
    cudaError_t e = cudaMemsetAsync(p.sched_ctr, 0, sizeof(int), s);
    if (e != cudaSuccess) return moe::cuda_status(e, what);
  }
  MOE_LAUNCH(kGemmName[MODE], s, cudaLaunchKernelEx(&cfg, kern, a, b, o, p));
  return moe::launch_status(what);
}

// Row-block split of the activation GEMMs (see run_gemm_out): on when the grouped layout
// has at least 2^18 rows. Measured on GB300 (same box, split on / off): T=65536,
// d_model=7168, 171 live experts 94.5-95.0 / 95.2-95.4 ms per layer step; T=32768 and
// T=16384 at d_model=4096 unchanged (the second launch costs what the half tiles save).
// MOE_GEMM_SPLIT=0 turns it off (A/B runs).
bool split_rows(uint64_t rows) {
  static int on = -1;
  if (on < 0) {
    const char *e = getenv("MOE_GEMM_SPLIT");
    on = (e != nullptr && e[0] == '0') ? 0 : 1;
  }
  return on && rows >= (uint64_t(1) << 18);
}

// Builds the tensor maps for one GEMM and launches it. A: [a_rows, a_cols] row-major
// bf16; B likewise. N = output columns (for kGateUp: 2F, in tiles of 128 gate + 128 up).
// The output p.out is [o_rows, o_cols] row-major bf16.
template <int MODE>
int run_gemm_out(int N, const void *a_base, uint64_t a_rows, uint64_t a_cols, const void *b_base,
                 uint64_t b_rows, uint64_t b_cols, const void *o_base, uint64_t o_rows,
                 uint64_t o_cols, GemmParams p, cudaStream_t s, const char *what);

template <int MODE>
int run_gemm(int N, const void *a_base, uint64_t a_rows, uint64_t a_cols, const void *b_base,
             uint64_t b_rows, uint64_t b_cols, uint64_t o_rows, uint64_t o_cols, GemmParams p,
             cudaStream_t s, const char *what) {
  return run_gemm_out<MODE>(N, a_base, a_rows, a_cols, b_base, b_rows, b_cols, p.out, o_rows,
                            o_cols, p, s, what);
}

// As run_gemm, with the output tensor map built over o_base (p.out may be nullptr when
// the epilogue stores no output tile).
template <int MODE>
int run_gemm_out(int N, const void *a_base, uint64_t a_rows, uint64_t a_cols, const void *b_base,
                 uint64_t b_rows, uint64_t b_cols, const void *o_base, uint64_t o_rows,
                 uint64_t o_cols, GemmParams p, cudaStream_t s, const char *what) {
  using Tr = Traits<MODE>;
  const bool pair = use_pair<MODE>();
  if (!Tr::WGRAD) p.dynamic = 0;  // equal-cost tiles: fixed stride, no counter to reset
  const int BN = (MODE == kGateUp || N % 256 == 0) ? 256 : 128;
  p.n_tiles = (MODE == kGateUp) ? N / 256 : N / BN;
  const bool gather = p.token_of_row != nullptr;
  if (gather && MODE != kGateUp && MODE != kWgradGateUp)
    return moe::set_error(MOE_ERR_UNSUPPORTED, "%s: no gathered operand in this GEMM", what);
  if (gather && !pair)
    return moe::set_error(MOE_ERR_UNSUPPORTED, "%s: the gathered operand needs the CTA-pair kernel", what);
  // the gathered operand's map is over x [T, d] with a one-row box (4-row gathers)
  const bool gather_a = gather && MODE == kGateUp, gather_b = gather && MODE == kWgradGateUp;
  CUtensorMap ma, mb;
  int st;
  // MN-major boxes: 64 columns x one ring stage of k-rows (128 in the CTA-pair kernel
  // without gathers, BK = 64 in the others)
  const uint32_t mn_rows = pair && !gather ? 128u : uint32_t(BK);
  if ((st = gather_a  ? make_map(&ma, a_base, a_rows, a_cols, BK, 1, what)
            : Tr::A_MN ? make_map(&ma, a_base, a_rows, a_cols, 64, mn_rows, what)
                       : make_map(&ma, a_base, a_rows, a_cols, BK, BM, what)))
    return st;
  const uint32_t b_box_rows = pair ? uint32_t(BN / 2) : 128u;
  if ((st = gather_b  ? make_map(&mb, b_base, b_rows, b_cols, 64, 1, what)
            : Tr::B_MN ? make_map(&mb, b_base, b_rows, b_cols, 64, mn_rows, what)
                       : make_map(&mb, b_base, b_rows, b_cols, BK, b_box_rows, what)))
    return st;
  CUtensorMap mo;  // the epilogue's output, in 32 x 32 chunks
  if ((st = make_map(&mo, o_base, o_rows, o_cols, 32, 32, what, CU_TENSOR_MAP_SWIZZLE_64B))) return st;
  if (pair) {
    if constexpr (MODE == kGateUp || MODE == kWgradGateUp) {
      if (gather)
        return BN == 256 ? launch_pair<MODE, 256, true>(ma, mb, mo, p, s, what)
                         : launch_pair<MODE, 128, true>(ma, mb, mo, p, s, what);
    }
    if (Tr::WGRAD || !split_rows(a_rows))
      return BN == 256 ? launch_pair<MODE, 256, false>(ma, mb, mo, p, s, what)
                       : launch_pair<MODE, 128, false>(ma, mb, mo, p, s, what);
    // Activation GEMMs on many rows: a group's last block of an odd number of 128-row
    // blocks would be half of a 256-row pair tile whose other half is computed and dropped;
    // the one-SM kernel (128-row tiles) takes those blocks in a second launch.
    GemmParams q = p;
    q.rows_split = 1;
    if ((st = BN == 256 ? launch_pair<MODE, 256, false>(ma, mb, mo, q, s, what)
                        : launch_pair<MODE, 128, false>(ma, mb, mo, q, s, what)))
      return st;
    CUtensorMap mb1;  // the one-SM kernel's B boxes
    if ((st = Tr::B_MN ? make_map(&mb1, b_base, b_rows, b_cols, 64, BK, what)
                       : make_map(&mb1, b_base, b_rows, b_cols, BK, 128, what)))
      return st;
    q.rows_split = 2;
    return BN == 256 ? launch_one<MODE, 256>(ma, mb1, mo, q, s, what)
                     : launch_one<MODE, 128>(ma, mb1, mo, q, s, what);
  }
  return BN == 256 ? launch_one<MODE, 256>(ma, mb, mo, p, s, what)
                   : launch_one<MODE, 128>(ma, mb, mo, p, s, what);
}

int check_common(int E, int d, int F, int64_t rows_cap, const char *fn) {
  if (E < 1 || E > 256) return moe::set_error(MOE_ERR_UNSUPPORTED, "%s: E=%d not in [1,256]", fn, E);
  if (d <= 0 || F <= 0 || d % 128 || F % 128)
    return moe::set_error(MOE_ERR_UNSUPPORTED, "%s: d=%d F=%d must be multiples of 128", fn, d, F);
  if (rows_cap < BM || rows_cap >= (int64_t(1) << 31))
    return moe::set_error(MOE_ERR_ARG, "%s: rows_cap=%lld", fn, (long long)rows_cap);
  if (int64_t(E) * 2 * F >= (int64_t(1) << 31) || int64_t(E) * d >= (int64_t(1) << 31))
    return moe::set_error(MOE_ERR_UNSUPPORTED, "%s: weight rows exceed 2^31", fn);
  return MOE_OK;
}

// Self-test of the bounded pipeline wait of the tensor-core kernels: one thread
// initializes an mbarrier that nothing will ever arrive on and waits for its first
// phase with the same bounded wait; after limit_ns it gives up, records
// MOE_DEV_WAIT_TIMEOUT and returns, leaving the context usable.
__global__ void wait_timeout_selftest_kernel(uint64_t limit_ns) {
  __shared__ uint64_t bar;
  __shared__ int abort_word;
  const uint32_t b = tc::smem_u32(&bar);
  tc::mbar_init(b, 1);
  tc::fence_mbar_init();
  abort_word = 0;
  if (!tc::mbar_wait(b, 0, limit_ns, &abort_word)) dev_flag(&g_dev_err, MOE_DEV_WAIT_TIMEOUT);
}

// ---- combine in the down GEMM's epilogue: helpers ----
// row_token[r] = -1 for every grouped row (padding rows keep it).
__global__ void combine_rows_fill_kernel(int32_t *__restrict__ row_token, int64_t R) {
  for (int64_t r = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; r < R;
       r += int64_t(gridDim.x) * blockDim.x)
    row_token[r] = -1;
}
// The row of assignment a = t*k + j gets token t and weight topk_gate[a].
__global__ void combine_rows_scatter_kernel(const int32_t *__restrict__ row_of_assignment,
                                            const float *__restrict__ topk_gate, int64_t A, int k,
                                            int64_t R, int32_t *__restrict__ row_token,
                                            float *__restrict__ row_gate) {
  for (int64_t a = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; a < A;
       a += int64_t(gridDim.x) * blockDim.x) {
    const int32_t r = row_of_assignment[a];
    if (r >= 0 && r < R) {
      row_token[r] = int32_t(a / k);
      row_gate[r] = topk_gate[a];
    } else {
      dev_flag(&g_dev_err, MOE_DEV_ROWS_OVERFLOW);
    }
  }
}
// The router's logit gradient of every assignment (softmax over the k selected experts:
// dz_j = g_j (dg_j - sum_i g_i dg_i), summed in slot order with fused multiply-adds, as
// moe_route_bwd computes it) written to the assignment's grouped row. Padding rows keep
// the zeros the caller wrote first.
__global__ void router_row_dz_kernel(const float *__restrict__ topk_gate,
                                     const float *__restrict__ d_gate,
                                     const int32_t *__restrict__ row_of_assignment, int T, int k,
                                     int64_t R, float *__restrict__ row_dz) {
  for (int t = blockIdx.x * blockDim.x + threadIdx.x; t < T; t += gridDim.x * blockDim.x) {
    float g[8], dg[8], s = 0.f;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      g[j] = 0.f;
      dg[j] = 0.f;
      if (j < k) {
        g[j] = topk_gate[size_t(t) * k + j];
        dg[j] = d_gate[size_t(t) * k + j];
        s = fmaf(g[j], dg[j], s);
      }
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      if (j < k) {
        const int32_t r = row_of_assignment[size_t(t) * k + j];
        if (r >= 0 && r < R) row_dz[r] = g[j] * (dg[j] - s);
        else dev_flag(&g_dev_err, MOE_DEV_ROWS_OVERFLOW);
      }
    }
  }
}
// d_gate[t, j] = <dy[t], O[row(t, j)]> from the dH GEMM's per-row partial sums of dH * H
// (summed in a fixed order), which equal g[t, j] * <dy[t], O[row]>; divided by the gate
// (positive for every selected expert; 0 is written for a zero gate).
__global__ void gate_from_rows_kernel(const float *__restrict__ partial, int stride,
                                      const float *__restrict__ topk_gate,
                                      const int32_t *__restrict__ row_of_assignment, int64_t A,
                                      int64_t R, float *__restrict__ d_gate) {
  for (int64_t a = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; a < A;
       a += int64_t(gridDim.x) * blockDim.x) {
    const int32_t r = row_of_assignment[a];
    if (r < 0 || r >= R) {
      dev_flag(&g_dev_err, MOE_DEV_ROWS_OVERFLOW);
      continue;
    }
    float s = 0.f;
    for (int i = 0; i < stride; ++i) s += partial[size_t(r) * stride + i];
    const float g = topk_gate[a];
    d_gate[a] = g > 0.f ? s / g : 0.f;
  }
}
__global__ void zero_f32x4_kernel(float4 *__restrict__ p, int64_t n4) {
  for (int64_t i = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; i < n4;
       i += int64_t(gridDim.x) * blockDim.x)
    p[i] = make_float4(0.f, 0.f, 0.f, 0.f);
}
// y = bf16(y_acc), 8 elements per thread (n8 = T*d/8).
__global__ void f32_to_bf16_kernel(const float4 *__restrict__ src, uint4 *__restrict__ dst,
                                   int64_t n8) {
  for (int64_t i = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; i < n8;
       i += int64_t(gridDim.x) * blockDim.x) {
    const float4 a = src[2 * i], b = src[2 * i + 1];
    dst[i] = make_uint4(pack_bf16x2(a.x, a.y), pack_bf16x2(a.z, a.w), pack_bf16x2(b.x, b.y),
                        pack_bf16x2(b.z, b.w));
  }
}
int grid_for(int64_t n) {
  return int(std::max<int64_t>(1, std::min<int64_t>((n + 255) / 256, int64_t(moe::num_sms()) * 8)));
}

}  // namespace

namespace moe {
MOE_DEV_ERR_DEFINE_READER(gemm_dev_error)
}

extern "C" {

int moe_selftest_wait_timeout(int64_t limit_ns, moe_stream_t stream) {
  if (limit_ns < 1000000 || limit_ns > 2000000000)
    return moe::set_error(MOE_ERR_ARG, "moe_selftest_wait_timeout: limit_ns %lld not in [1e6, 2e9]",
                          (long long)limit_ns);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  MOE_LAUNCH("selftest_wait_timeout", s,
             wait_timeout_selftest_kernel<<<1, 1, 0, s>>>(uint64_t(limit_ns)));
  return moe::launch_status("moe_selftest_wait_timeout");
}

int moe_grouped_ffn_fwd(const uint16_t *x_perm, const int32_t *group_offsets, int E, int d, int F,
                        int64_t rows_cap, const uint16_t *w_gate_up, const uint16_t *w_down,
                        uint16_t *ab_saved, uint16_t *h, uint16_t *out_perm, void *ws,
                        size_t ws_bytes, moe_stream_t stream) {
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (int st = check_common(E, d, F, rows_cap, "moe_grouped_ffn_fwd")) return st;
  const void *ptrs[] = {x_perm, group_offsets, w_gate_up, w_down, ab_saved, h, out_perm};
  for (const void *q : ptrs)
    if (!q || !moe::aligned16(q)) return moe::set_error(MOE_ERR_ARG, "moe_grouped_ffn_fwd: null or unaligned pointer");
  const uint64_t R = uint64_t(rows_cap);
  GemmParams p{};
  if (int st = use_sched_ws(p, ws, ws_bytes, "moe_grouped_ffn_fwd")) return st;
  p.group_offsets = group_offsets;
  p.E = E; p.d = d; p.F = F;
  // [A | B] = X W_gate_up^T, H = silu(A) * B
  p.nkb = d / BK;
  p.out = h;
  p.out2 = ab_saved;
  if (int st = run_gemm<kGateUp>(2 * F, x_perm, R, d, w_gate_up, uint64_t(E) * 2 * F, d, R, F, p,
                                 s, "moe_grouped_ffn_fwd: gate/up GEMM"))
    return st;
  // O = H W_down^T
  GemmParams q{};
  use_sched_ws(q, ws, ws_bytes, "moe_grouped_ffn_fwd");
  q.group_offsets = group_offsets;
  q.E = E; q.d = d; q.F = F;
  q.nkb = F / BK;
  q.out = out_perm;
  return run_gemm<kDown>(d, h, R, F, w_down, uint64_t(E) * d, F, R, d, q, s,
                         "moe_grouped_ffn_fwd: down GEMM");
}

int moe_grouped_ffn_fwd_combine(const uint16_t *x_perm, const int32_t *group_offsets, int E, int d,
                                int F, int64_t rows_cap, const uint16_t *w_gate_up,
                                const uint16_t *w_down, const int32_t *row_of_assignment,
                                const float *topk_gate, int T, int k, uint16_t *ab_saved,
                                uint16_t *h, uint16_t *out_perm, float *y_acc, uint16_t *y,
                                void *ws, size_t ws_bytes, moe_stream_t stream) {
  const char *fn = "moe_grouped_ffn_fwd_combine";
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (int st = check_common(E, d, F, rows_cap, fn)) return st;
  if (T < 0 || k < 1 || k > 8 || k > E) return moe::set_error(MOE_ERR_ARG, "%s: T=%d k=%d", fn, T, k);
  if (rows_cap < moe_perm_rows_max(T, k, E)) return moe::set_error(MOE_ERR_ARG, "%s: rows_cap too small", fn);
  const void *ptrs[] = {x_perm, group_offsets, w_gate_up, w_down, ab_saved, h, ws};
  for (const void *q : ptrs)
    if (!q || !moe::aligned16(q)) return moe::set_error(MOE_ERR_ARG, "%s: null or unaligned pointer", fn);
  if (out_perm && !moe::aligned16(out_perm)) return moe::set_error(MOE_ERR_ARG, "%s: unaligned out_perm", fn);
  if (T > 0 && (!row_of_assignment || !topk_gate || !y_acc || !y || !moe::aligned16(y_acc) ||
                !moe::aligned16(y)))
    return moe::set_error(MOE_ERR_ARG, "%s: null or unaligned combine argument", fn);
  const moe::WsLayout L = moe::ws_layout(T, d, E, k, F);
  if (ws_bytes < L.total) return moe::set_error(MOE_ERR_WORKSPACE, "%s: workspace", fn);
  const uint64_t R = uint64_t(rows_cap);
  const int64_t Rr = moe_perm_rows_max(T, k, E);  // rows the layout can use
  int32_t *row_token = reinterpret_cast<int32_t *>(static_cast<char *>(ws) + L.combine_rows);
  float *row_gate = reinterpret_cast<float *>(row_token + Rr);
  GemmParams p{};
  if (int st = use_sched_ws(p, ws, ws_bytes, fn)) return st;
  p.group_offsets = group_offsets;
  p.E = E; p.d = d; p.F = F;
  p.nkb = d / BK;
  p.out = h;
  p.out2 = ab_saved;
  if (int st = run_gemm<kGateUp>(2 * F, x_perm, R, d, w_gate_up, uint64_t(E) * 2 * F, d, R, F, p,
                                 s, "moe_grouped_ffn_fwd_combine: gate/up GEMM"))
    return st;
  const int64_t A = int64_t(T) * k, n = int64_t(T) * d;
  if (T > 0) {
    MOE_LAUNCH("combine_rows_fill", s, combine_rows_fill_kernel<<<grid_for(Rr), 256, 0, s>>>(row_token, Rr));
    if (int st = moe::launch_status("moe_grouped_ffn_fwd_combine: row fill")) return st;
    MOE_LAUNCH("combine_rows_scatter", s, combine_rows_scatter_kernel<<<grid_for(A), 256, 0, s>>>(
                                              row_of_assignment, topk_gate, A, k, Rr, row_token, row_gate));
    if (int st = moe::launch_status("moe_grouped_ffn_fwd_combine: row scatter")) return st;
    MOE_LAUNCH("zero_y_acc", s, zero_f32x4_kernel<<<grid_for(n / 4), 256, 0, s>>>(
                                    reinterpret_cast<float4 *>(y_acc), n / 4));
    if (int st = moe::launch_status("moe_grouped_ffn_fwd_combine: zero")) return st;
  }
  // O = H W_down^T, combined into y_acc by the epilogue (O itself stored only if asked)
  GemmParams q{};
  use_sched_ws(q, ws, ws_bytes, fn);
  q.group_offsets = group_offsets;
  q.E = E; q.d = d; q.F = F;
  q.nkb = F / BK;
  q.out = out_perm;
  if (T > 0) {
    q.y_acc = y_acc;
    q.row_token = row_token;
    q.row_gate = row_gate;
  }
  // without out_perm the output map is built over h (never stored to)
  void *o_base = out_perm ? static_cast<void *>(out_perm) : static_cast<void *>(h);
  const uint64_t o_cols = out_perm ? uint64_t(d) : uint64_t(F);
  if (int st = run_gemm_out<kDown>(d, h, R, F, w_down, uint64_t(E) * d, F, o_base, R, o_cols, q, s,
                                   "moe_grouped_ffn_fwd_combine: down GEMM"))
    return st;
  if (T == 0) return MOE_OK;
  MOE_LAUNCH("combine_y_bf16", s, f32_to_bf16_kernel<<<grid_for(n / 8), 256, 0, s>>>(
                                      reinterpret_cast<const float4 *>(y_acc), reinterpret_cast<uint4 *>(y), n / 8));
  return moe::launch_status("moe_grouped_ffn_fwd_combine: bf16 output");
}

int moe_grouped_ffn_fwd_gather(const uint16_t *x, const int32_t *token_of_row, int T,
                               const int32_t *group_offsets, int E, int d, int F,
                               int64_t rows_cap, const uint16_t *w_gate_up,
                               const uint16_t *w_down, uint16_t *ab_saved, uint16_t *h,
                               uint16_t *out_perm, void *ws, size_t ws_bytes, moe_stream_t stream) {
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (int st = check_common(E, d, F, rows_cap, "moe_grouped_ffn_fwd_gather")) return st;
  if (T < 0) return moe::set_error(MOE_ERR_ARG, "moe_grouped_ffn_fwd_gather: T=%d", T);
  const void *ptrs[] = {token_of_row, group_offsets, w_gate_up, w_down, ab_saved, h, out_perm};
  for (const void *q : ptrs)
    if (!q || !moe::aligned16(q))
      return moe::set_error(MOE_ERR_ARG, "moe_grouped_ffn_fwd_gather: null or unaligned pointer");
  if (T > 0 && (!x || !moe::aligned16(x)))
    return moe::set_error(MOE_ERR_ARG, "moe_grouped_ffn_fwd_gather: null or unaligned x");
  const uint64_t R = uint64_t(rows_cap);
  GemmParams p{};
  if (int st = use_sched_ws(p, ws, ws_bytes, "moe_grouped_ffn_fwd_gather")) return st;
  p.group_offsets = group_offsets;
  p.E = E; p.d = d; p.F = F;
  p.nkb = d / BK;
  p.out = h;
  p.out2 = ab_saved;
  p.token_of_row = token_of_row;
  // no tokens: no tile reads x; the map needs some valid base
  const void *xa = T > 0 ? static_cast<const void *>(x) : static_cast<const void *>(h);
  if (int st = run_gemm<kGateUp>(2 * F, xa, uint64_t(std::max(T, 1)), d, w_gate_up,
                                 uint64_t(E) * 2 * F, d, R, F, p, s,
                                 "moe_grouped_ffn_fwd_gather: gate/up GEMM"))
    return st;
  GemmParams q{};
  use_sched_ws(q, ws, ws_bytes, "moe_grouped_ffn_fwd_gather");
  q.group_offsets = group_offsets;
  q.E = E; q.d = d; q.F = F;
  q.nkb = F / BK;
  q.out = out_perm;
  return run_gemm<kDown>(d, h, R, F, w_down, uint64_t(E) * d, F, R, d, q, s,
                         "moe_grouped_ffn_fwd_gather: down GEMM");
}

int moe_grouped_ffn_bwd_dgrad(const uint16_t *d_out_perm, const uint16_t *ab_saved,
                              const int32_t *group_offsets, int E, int d, int F, int64_t rows_cap,
                              const uint16_t *w_gate_up, const uint16_t *w_down,
                              const float *topk_gate, const float *d_gate,
                              const int32_t *row_of_assignment, const float *w_router, int T,
                              int k, float *d_gate_out, uint16_t *d_ab, uint16_t *dx_perm,
                              void *ws, size_t ws_bytes, moe_stream_t stream) {
  const char *fn = "moe_grouped_ffn_bwd_dgrad";
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (int st = check_common(E, d, F, rows_cap, fn)) return st;
  const void *ptrs[] = {d_out_perm, ab_saved, group_offsets, w_gate_up, w_down, d_ab, dx_perm};
  for (const void *q : ptrs)
    if (!q || !moe::aligned16(q)) return moe::set_error(MOE_ERR_ARG, "%s: null or unaligned pointer", fn);
  const uint64_t R = uint64_t(rows_cap);
  int st;
  GemmParams p{};
  if ((st = use_sched_ws(p, ws, ws_bytes, fn))) return st;
  // d_gate_out: the gate gradient from the dH GEMM's epilogue; w_router: the router's term
  // of the input gradient, added in the dX GEMM's epilogue (from d_gate_out, or d_gate)
  const bool router = w_router != nullptr, gate = d_gate_out != nullptr;
  if (!router && d_gate)
    return moe::set_error(MOE_ERR_ARG, "%s: d_gate without w_router", fn);
  if (d_gate && gate)
    return moe::set_error(MOE_ERR_ARG, "%s: d_gate is either an input or computed here", fn);
  if (!router && !gate && (topk_gate || row_of_assignment))
    return moe::set_error(MOE_ERR_ARG, "%s: routing arguments without a router term or d_gate_out", fn);
  int64_t Rr = 0;
  moe::WsLayout L{};
  if (router || gate) {
    if (T < 0 || k < 1 || k > 8 || k > E) return moe::set_error(MOE_ERR_ARG, "%s: T=%d k=%d", fn, T, k);
    if (T > 0 && (!topk_gate || !row_of_assignment || (router && !gate && !d_gate)))
      return moe::set_error(MOE_ERR_ARG, "%s: the router term needs topk_gate, d_gate (or "
                            "d_gate_out) and row_of_assignment; d_gate_out needs topk_gate and "
                            "row_of_assignment", fn);
    Rr = moe_perm_rows_max(T, k, E);
    if (rows_cap < Rr) return moe::set_error(MOE_ERR_ARG, "%s: rows_cap too small", fn);
    L = moe::ws_layout(T, d, E, k, F);
    if (ws_bytes < L.total) return moe::set_error(MOE_ERR_WORKSPACE, "%s: workspace", fn);
  }
  p.group_offsets = group_offsets;
  p.E = E; p.d = d; p.F = F;
  // dH = dO W_down, fused SwiGLU backward -> [dA | dB] (and the rows' dH * H sums)
  p.nkb = d / BK;
  p.out = d_ab;
  p.aux = ab_saved;
  if (gate) {
    p.gate_partial = reinterpret_cast<float *>(static_cast<char *>(ws) + L.gate_partial);
    p.gate_stride = 2 * (F / (F % 256 == 0 ? 256 : 128));  // column halves of the N tiles
  }
  if ((st = run_gemm<kDgradDown>(F, d_out_perm, R, d, w_down, uint64_t(E) * d, F, R, 2 * F, p,
                                 s, "moe_grouped_ffn_bwd: dH GEMM")))
    return st;
  p.gate_partial = nullptr;
  const int64_t A = int64_t(T) * k;
  if (gate && A > 0) {
    MOE_LAUNCH("gate_from_rows", s, gate_from_rows_kernel<<<grid_for(A), 256, 0, s>>>(
                                        reinterpret_cast<const float *>(static_cast<char *>(ws) + L.gate_partial),
                                        2 * (F / (F % 256 == 0 ? 256 : 128)), topk_gate,
                                        row_of_assignment, A, Rr, d_gate_out));
    if ((st = moe::launch_status("moe_grouped_ffn_bwd_dgrad: gate gradient"))) return st;
  }
  if (router) {
    float *row_dz = reinterpret_cast<float *>(static_cast<char *>(ws) + L.row_dz);
    cudaError_t e = cudaMemsetAsync(row_dz, 0, size_t(Rr) * 4, s);
    if (e != cudaSuccess) return moe::cuda_status(e, "moe_grouped_ffn_bwd_dgrad: zero row_dz");
    if (T > 0) {
      MOE_LAUNCH("router_row_dz", s, router_row_dz_kernel<<<grid_for(T), 256, 0, s>>>(
                                         topk_gate, gate ? d_gate_out : d_gate, row_of_assignment,
                                         T, k, Rr, row_dz));
      if ((st = moe::launch_status("moe_grouped_ffn_bwd_dgrad: router rows"))) return st;
    }
    p.row_dz = row_dz;
    p.w_router = w_router;
  }
  // dX = [dA | dB] W_gate_up
  p.nkb = 2 * F / BK;
  p.out = dx_perm;
  p.aux = nullptr;
  return run_gemm<kDgradGateUp>(d, d_ab, R, 2 * F, w_gate_up, uint64_t(E) * 2 * F, d, R, d, p,
                                s, "moe_grouped_ffn_bwd: dX GEMM");
}

int moe_grouped_ffn_bwd_wgrad(const uint16_t *d_out_perm, const uint16_t *x_perm,
                              const uint16_t *h, const uint16_t *d_ab,
                              const int32_t *group_offsets, const uint8_t *active_mask, int E,
                              int d, int F, int64_t rows_cap, uint16_t *dw_gate_up,
                              uint16_t *dw_down, void *ws, size_t ws_bytes, moe_stream_t stream) {
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (int st = check_common(E, d, F, rows_cap, "moe_grouped_ffn_bwd_wgrad")) return st;
  const void *ptrs[] = {d_out_perm, x_perm, h, d_ab, group_offsets, dw_gate_up, dw_down};
  for (const void *q : ptrs)
    if (!q || !moe::aligned16(q)) return moe::set_error(MOE_ERR_ARG, "moe_grouped_ffn_bwd_wgrad: null or unaligned pointer");
  const uint64_t R = uint64_t(rows_cap);
  int st;
  GemmParams p{};
  if ((st = use_sched_ws(p, ws, ws_bytes, "moe_grouped_ffn_bwd_wgrad"))) return st;
  p.group_offsets = group_offsets;
  p.active_mask = active_mask;
  p.E = E; p.d = d; p.F = F;
  // dW_down[e] = dO_e^T H_e   ([d, F])
  p.nkb = 0;
  p.m_tiles_w = d / BM;
  p.out = dw_down;
  if ((st = run_gemm<kWgradDown>(F, d_out_perm, R, d, h, R, F, uint64_t(E) * d, F, p, s,
                                 "moe_grouped_ffn_bwd: dW_down GEMM")))
    return st;
  // dW_gate_up[e] = [dA | dB]_e^T X_e   ([2F, d])
  p.m_tiles_w = 2 * F / BM;
  p.out = dw_gate_up;
  return run_gemm<kWgradGateUp>(d, d_ab, R, 2 * F, x_perm, R, d, uint64_t(E) * 2 * F, d, p, s,
                                "moe_grouped_ffn_bwd: dW_gate_up GEMM");
}

int moe_grouped_ffn_bwd_wgrad_gather(const uint16_t *d_out_perm, const uint16_t *x,
                                     const int32_t *token_of_row, int T, const uint16_t *h,
                                     const uint16_t *d_ab, const int32_t *group_offsets,
                                     const uint8_t *active_mask, int E, int d, int F,
                                     int64_t rows_cap, uint16_t *dw_gate_up, uint16_t *dw_down,
                                     void *ws, size_t ws_bytes, moe_stream_t stream) {
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (int st = check_common(E, d, F, rows_cap, "moe_grouped_ffn_bwd_wgrad_gather")) return st;
  if (T < 0) return moe::set_error(MOE_ERR_ARG, "moe_grouped_ffn_bwd_wgrad_gather: T=%d", T);
  const void *ptrs[] = {d_out_perm, token_of_row, h, d_ab, group_offsets, dw_gate_up, dw_down};
  for (const void *q : ptrs)
    if (!q || !moe::aligned16(q))
      return moe::set_error(MOE_ERR_ARG, "moe_grouped_ffn_bwd_wgrad_gather: null or unaligned pointer");
  if (T > 0 && (!x || !moe::aligned16(x)))
    return moe::set_error(MOE_ERR_ARG, "moe_grouped_ffn_bwd_wgrad_gather: null or unaligned x");
  const uint64_t R = uint64_t(rows_cap);
  int st;
  GemmParams p{};
  if ((st = use_sched_ws(p, ws, ws_bytes, "moe_grouped_ffn_bwd_wgrad_gather"))) return st;
  p.group_offsets = group_offsets;
  p.active_mask = active_mask;
  p.E = E; p.d = d; p.F = F;
  p.nkb = 0;
  p.m_tiles_w = d / BM;
  p.out = dw_down;
  if ((st = run_gemm<kWgradDown>(F, d_out_perm, R, d, h, R, F, uint64_t(E) * d, F, p, s,
                                 "moe_grouped_ffn_bwd_wgrad_gather: dW_down GEMM")))
    return st;
  p.m_tiles_w = 2 * F / BM;
  p.out = dw_gate_up;
  p.token_of_row = token_of_row;
  const void *xb = T > 0 ? static_cast<const void *>(x) : static_cast<const void *>(dw_gate_up);
  return run_gemm<kWgradGateUp>(d, d_ab, R, 2 * F, xb, uint64_t(std::max(T, 1)), d,
                                uint64_t(E) * 2 * F, d, p, s,
                                "moe_grouped_ffn_bwd_wgrad_gather: dW_gate_up GEMM");
}

int moe_grouped_ffn_bwd(const uint16_t *d_out_perm, const uint16_t *x_perm,
                        const uint16_t *ab_saved, const uint16_t *h, const int32_t *group_offsets,
                        const uint8_t *active_mask, int E, int d, int F, int64_t rows_cap,
                        const uint16_t *w_gate_up, const uint16_t *w_down,
                        const float *topk_gate, const float *d_gate,
                        const int32_t *row_of_assignment, const float *w_router, int T, int k,
                        float *d_gate_out, uint16_t *d_ab, uint16_t *dx_perm,
                        uint16_t *dw_gate_up, uint16_t *dw_down, void *ws, size_t ws_bytes,
                        moe_stream_t stream) {
  if (int st = moe_grouped_ffn_bwd_dgrad(d_out_perm, ab_saved, group_offsets, E, d, F, rows_cap,
                                         w_gate_up, w_down, topk_gate, d_gate, row_of_assignment,
                                         w_router, T, k, d_gate_out, d_ab, dx_perm, ws, ws_bytes,
                                         stream))
    return st;
  return moe_grouped_ffn_bwd_wgrad(d_out_perm, x_perm, h, d_ab, group_offsets, active_mask, E, d,
                                   F, rows_cap, dw_gate_up, dw_down, ws, ws_bytes, stream);
}

}  // extern "C"

namespace moe {
namespace {
typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                  const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                  const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static bool tried = false;
  if (!tried) {
    tried = true;
    void *ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(ptr);
  }
  return fn;
}

}  // namespace

int make_map(CUtensorMap *m, const void *base, uint64_t rows, uint64_t cols, uint32_t box_cols,
             uint32_t box_rows, const char *what, CUtensorMapSwizzle swizzle) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return moe::set_error(MOE_ERR_CUDA, "cuTensorMapEncodeTiled unavailable");
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {box_cols, box_rows};
  cuuint32_t es[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides,
                  box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return moe::set_error(MOE_ERR_CUDA, "tensor map for %s: CUresult %d", what, int(r));
  return MOE_OK;
}
}  // namespace moe
