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
// Algorithm 2's greedy balancing also uses.
//
// Six GEMM shapes share one kernel template:
//   kGateUp      [A|B] = X W_gu^T        (A: K-major rows, B: K-major weights)
//                epilogue: H = silu(A)*B, keeps A and B for the backward
//   kDown        O = H W_down^T
//   kDgradDown   dH = dO W_down           (B is MN-major)
//                epilogue: dA = dH*B*silu'(A), dB = dH*silu(A)
//   kDgradGateUp dX = [dA|dB] W_gu        (B is MN-major)
//   kWgradDown   dW_down[e] = dO_e^T H_e  (A and B MN-major; K = group rows)
//   kWgradGateUp dW_gu[e] = [dA|dB]_e^T X_e
#include <cuda.h>

#include "common.cuh"
#include "tc_ptx.cuh"

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
constexpr int kThreads = 192;  // warp 0 TMA, warp 1 MMA + TMEM owner, warps 2-5 epilogue
constexpr uint64_t kWaitLimitNs = 2000000000ull;

template <int MODE> struct Traits {
  static constexpr bool A_MN = (MODE == kWgradDown || MODE == kWgradGateUp);
  static constexpr bool B_MN = (MODE != kGateUp && MODE != kDown);
  static constexpr bool WGRAD = (MODE == kWgradDown || MODE == kWgradGateUp);
};

template <int BN> struct Shape {
  static constexpr int STAGES = BN == 256 ? 4 : 6;
  static constexpr uint32_t A_BYTES = BM * BK * 2;
  static constexpr uint32_t B_BYTES = BN * BK * 2;
  static constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int NBARS = 2 * STAGES + 5;
  static constexpr size_t SMEM = 1024 + size_t(STAGES) * STAGE_BYTES + NBARS * 8 +
                                 (4 + 257 + 256 + 257) * 4;
  static constexpr uint32_t TMEM_COLS = 2 * BN;
};

struct GemmParams {
  const int32_t *group_offsets;  // [E+1], padded group starts (device)
  int E, d, F;
  int n_tiles;     // output column tiles
  int m_tiles_w;   // weight-gradient modes: row tiles of one expert's output
  int nkb;         // k-blocks per tile (activation modes)
  uint16_t *out;   // primary output
  uint16_t *out2;  // kGateUp: pre-activations [rows, 2F]
  const uint16_t *aux;  // kDgradDown: saved pre-activations [rows, 2F]
};

struct Tile {
  int e, goff, mt, nt, nkb;
};

__device__ __forceinline__ void fail(volatile int *abort_flag) {
  dev_flag(&g_dev_err, MOE_DEV_WAIT_TIMEOUT);
  *abort_flag = 1;
}

__device__ __forceinline__ void store_row_bf16(uint16_t *dst, const uint32_t (&r)[32]) {
#pragma unroll
  for (int v = 0; v < 4; ++v) {
    uint4 o;
    o.x = pack_bf16x2(__uint_as_float(r[v * 8 + 0]), __uint_as_float(r[v * 8 + 1]));
    o.y = pack_bf16x2(__uint_as_float(r[v * 8 + 2]), __uint_as_float(r[v * 8 + 3]));
    o.z = pack_bf16x2(__uint_as_float(r[v * 8 + 4]), __uint_as_float(r[v * 8 + 5]));
    o.w = pack_bf16x2(__uint_as_float(r[v * 8 + 6]), __uint_as_float(r[v * 8 + 7]));
    stg_v4(dst + v * 8, o);
  }
}

__device__ __forceinline__ float silu_f(float a) { return a / (1.f + __expf(-a)); }

template <int MODE, int BN>
__global__ void __launch_bounds__(kThreads, 1)
    grouped_gemm_kernel(const __grid_constant__ CUtensorMap tmA,
                        const __grid_constant__ CUtensorMap tmB, const GemmParams p) {
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
      tc::mbar_init(tempty_bar(a), 4);
    }
    tc::mbar_init(drain_bar, 1);
    tc::fence_mbar_init();
    misc[1] = 0;
  }
  if (warp == 0 && lane == 0) {
    tc::tma_prefetch_desc(&tmA);
    tc::tma_prefetch_desc(&tmB);
  }
  if (warp == 1) {
    tc::tmem_alloc(tc::smem_u32(misc), Sh::TMEM_COLS);
    tc::tmem_relinquish();
  }
  // ---- tile schedule, built from the device-resident group offsets ----
  for (int e = threadIdx.x; e <= E; e += kThreads) s_goff[e] = p.group_offsets[e];
  __syncthreads();
  if (Tr::WGRAD) {
    for (int e = threadIdx.x; e < E; e += kThreads) {
      const int ce = s_goff[e + 1] - s_goff[e];
      int r = 0;
      for (int q = 0; q < E; ++q) {
        const int cq = s_goff[q + 1] - s_goff[q];
        r += (cq > ce) || (cq == ce && q < e);
      }
      s_order[r] = e;
    }
  } else {
    for (int e = threadIdx.x; e < E; e += kThreads) s_order[e] = e;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int acc = 0;
    for (int i = 0; i < E; ++i) {
      s_prefix[i] = acc;
      const int e = s_order[i];
      const int rows = s_goff[e + 1] - s_goff[e];
      acc += Tr::WGRAD ? p.m_tiles_w * p.n_tiles : (rows / BM) * p.n_tiles;
    }
    s_prefix[E] = acc;
  }
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
    t.mt = local / p.n_tiles;
    t.nt = local - t.mt * p.n_tiles;
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
    // ===================== epilogue (warps 2..5) =====================
    const int q = warp & 3;  // TMEM lane quarter this warp may access
    const int r_in_tile = q * 32 + lane;
    uint32_t tcount = 0;
    for (int tile = blockIdx.x; tile < total; tile += gridDim.x) {
      const Tile t = decode(tile);
      if (Tr::WGRAD && t.nkb == 0) {
        // empty group: its weight gradient is exactly zero
        const int M_out = p.m_tiles_w * BM, N_out = p.n_tiles * BN;
        uint16_t *o = p.out + (size_t(t.e) * M_out + t.mt * BM + r_in_tile) * N_out + t.nt * BN;
        const uint4 z = make_uint4(0, 0, 0, 0);
#pragma unroll 4
        for (int c = 0; c < BN; c += 8) stg_v4(o + c, z);
        continue;
      }
      const uint32_t a = tcount & 1u, aph = (tcount >> 1) & 1u;
      const bool ok = tc::mbar_wait(tfull_bar(a), aph, kWaitLimitNs, abort_flag);
      __syncwarp();
      if (!ok) { fail(abort_flag); break; }
      tc::fence_after_sync();
      const uint32_t tb = tmem_base + (uint32_t(q * 32) << 16) + a * BN;

      if (MODE == kGateUp) {
        const int F = p.F;
        const size_t row = size_t(t.goff) + t.mt * BM + r_in_tile;
        uint16_t *hrow = p.out + row * F + t.nt * 128;
        uint16_t *arow = p.out2 + row * 2 * F + t.nt * 128;
        uint16_t *brow = arow + F;
#pragma unroll 1
        for (int c = 0; c < 128; c += 32) {
          uint32_t ra[32], rb[32];
          tc::tmem_ld_32x32b_x32(tb + c, ra);
          tc::tmem_ld_32x32b_x32(tb + 128 + c, rb);
          tc::tmem_ld_wait();
#pragma unroll
          for (int v = 0; v < 4; ++v) {
            float fa[8], fb[8], fh[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) {
              fa[i] = __uint_as_float(ra[v * 8 + i]);
              fb[i] = __uint_as_float(rb[v * 8 + i]);
              fh[i] = silu_f(fa[i]) * fb[i];
            }
            stg_v4(hrow + c + v * 8, pack8(fh));
            stg_v4(arow + c + v * 8, pack8(fa));
            stg_v4(brow + c + v * 8, pack8(fb));
          }
        }
      } else if (MODE == kDgradDown) {
        const int F = p.F;
        const size_t row = size_t(t.goff) + t.mt * BM + r_in_tile;
        const int f0 = t.nt * BN;
        const uint16_t *arow = p.aux + row * 2 * F + f0;
        const uint16_t *brow = arow + F;
        uint16_t *darow = p.out + row * 2 * F + f0;
        uint16_t *dbrow = darow + F;
#pragma unroll 1
        for (int c = 0; c < BN; c += 32) {
          uint4 va[4], vb[4];
#pragma unroll
          for (int v = 0; v < 4; ++v) {
            va[v] = ldg_nc_v4(arow + c + v * 8);
            vb[v] = ldg_nc_v4(brow + c + v * 8);
          }
          uint32_t r[32];
          tc::tmem_ld_32x32b_x32(tb + c, r);
          tc::tmem_ld_wait();
#pragma unroll
          for (int v = 0; v < 4; ++v) {
            float fa[8], fb[8], da[8], db[8];
            unpack8(va[v], fa);
            unpack8(vb[v], fb);
#pragma unroll
            for (int i = 0; i < 8; ++i) {
              const float dh = __uint_as_float(r[v * 8 + i]);
              const float sg = 1.f / (1.f + __expf(-fa[i]));
              da[i] = dh * fb[i] * (sg * (1.f + fa[i] * (1.f - sg)));
              db[i] = dh * fa[i] * sg;
            }
            stg_v4(darow + c + v * 8, pack8(da));
            stg_v4(dbrow + c + v * 8, pack8(db));
          }
        }
      } else {
        uint16_t *orow;
        if (Tr::WGRAD) {
          const int M_out = p.m_tiles_w * BM, N_out = p.n_tiles * BN;
          orow = p.out + (size_t(t.e) * M_out + t.mt * BM + r_in_tile) * N_out + t.nt * BN;
        } else {
          const size_t row = size_t(t.goff) + t.mt * BM + r_in_tile;
          orow = p.out + row * p.d + t.nt * BN;
        }
#pragma unroll 1
        for (int c = 0; c < BN; c += 32) {
          uint32_t r[32];
          tc::tmem_ld_32x32b_x32(tb + c, r);
          tc::tmem_ld_wait();
          store_row_bf16(orow + c, r);
        }
      }
      tc::fence_before_sync();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(tempty_bar(a));
      ++tcount;
    }
  }

  tc::fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem_base, Sh::TMEM_COLS);
  }
}

// ------------------------------------------------------------------ host side

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

// bf16 row-major [rows, cols]; box = box_cols (inner) x box_rows; 128-byte swizzle.
int make_map(CUtensorMap *m, const void *base, uint64_t rows, uint64_t cols, uint32_t box_cols,
             uint32_t box_rows, const char *what) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return moe::set_error(MOE_ERR_CUDA, "cuTensorMapEncodeTiled unavailable");
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {box_cols, box_rows};
  cuuint32_t es[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides,
                  box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return moe::set_error(MOE_ERR_CUDA, "tensor map for %s: CUresult %d", what, int(r));
  return MOE_OK;
}
int map_kmajor(CUtensorMap *m, const void *base, uint64_t rows, uint64_t cols, const char *w) {
  return make_map(m, base, rows, cols, BK, BM, w);
}
int map_mnmajor(CUtensorMap *m, const void *base, uint64_t rows, uint64_t cols, const char *w) {
  return make_map(m, base, rows, cols, 64, BK, w);
}

template <int MODE, int BN>
int launch(const CUtensorMap &a, const CUtensorMap &b, const GemmParams &p, cudaStream_t s,
           const char *what) {
  using Sh = Shape<BN>;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(grouped_gemm_kernel<MODE, BN>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, int(Sh::SMEM));
    if (e != cudaSuccess) return moe::cuda_status(e, what);
    attr = true;
  }
  MOE_LAUNCH(kGemmName[MODE], s, grouped_gemm_kernel<MODE, BN><<<moe::num_sms(), kThreads, Sh::SMEM, s>>>(a, b, p));
  return moe::launch_status(what);
}

template <int MODE>
int launch_bn(int N, const CUtensorMap &a, const CUtensorMap &b, GemmParams p, cudaStream_t s,
              const char *what) {
  if (N % 256 == 0) {
    p.n_tiles = N / 256;
    return launch<MODE, 256>(a, b, p, s, what);
  }
  p.n_tiles = N / 128;
  return launch<MODE, 128>(a, b, p, s, what);
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

}  // namespace

namespace moe {
MOE_DEV_ERR_DEFINE_READER(gemm_dev_error)
}

extern "C" {

int moe_grouped_ffn_fwd(const uint16_t *x_perm, const int32_t *group_offsets, int E, int d, int F,
                        int64_t rows_cap, const uint16_t *w_gate_up, const uint16_t *w_down,
                        uint16_t *ab_saved, uint16_t *h, uint16_t *out_perm, void *ws,
                        size_t ws_bytes, moe_stream_t stream) {
  (void)ws;
  (void)ws_bytes;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (int st = check_common(E, d, F, rows_cap, "moe_grouped_ffn_fwd")) return st;
  const void *ptrs[] = {x_perm, group_offsets, w_gate_up, w_down, ab_saved, h, out_perm};
  for (const void *q : ptrs)
    if (!q || !moe::aligned16(q)) return moe::set_error(MOE_ERR_ARG, "moe_grouped_ffn_fwd: null or unaligned pointer");
  CUtensorMap mX, mWgu, mH, mWd;
  int st;
  if ((st = map_kmajor(&mX, x_perm, rows_cap, d, "x_perm"))) return st;
  if ((st = map_kmajor(&mWgu, w_gate_up, uint64_t(E) * 2 * F, d, "w_gate_up"))) return st;
  if ((st = map_kmajor(&mH, h, rows_cap, F, "h"))) return st;
  if ((st = map_kmajor(&mWd, w_down, uint64_t(E) * d, F, "w_down"))) return st;
  GemmParams p{};
  p.group_offsets = group_offsets;
  p.E = E; p.d = d; p.F = F;
  p.nkb = d / BK;
  p.n_tiles = F / 128;
  p.out = h;
  p.out2 = ab_saved;
  if ((st = launch<kGateUp, 256>(mX, mWgu, p, s, "moe_grouped_ffn_fwd: gate/up GEMM"))) return st;
  GemmParams q{};
  q.group_offsets = group_offsets;
  q.E = E; q.d = d; q.F = F;
  q.nkb = F / BK;
  q.out = out_perm;
  return launch_bn<kDown>(d, mH, mWd, q, s, "moe_grouped_ffn_fwd: down GEMM");
}

int moe_grouped_ffn_bwd(const uint16_t *d_out_perm, const uint16_t *x_perm,
                        const uint16_t *ab_saved, const uint16_t *h, const int32_t *group_offsets,
                        int E, int d, int F, int64_t rows_cap, const uint16_t *w_gate_up,
                        const uint16_t *w_down, uint16_t *d_ab, uint16_t *dx_perm,
                        uint16_t *dw_gate_up, uint16_t *dw_down, void *ws, size_t ws_bytes,
                        moe_stream_t stream) {
  (void)ws;
  (void)ws_bytes;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (int st = check_common(E, d, F, rows_cap, "moe_grouped_ffn_bwd")) return st;
  const void *ptrs[] = {d_out_perm, x_perm, ab_saved, h, group_offsets, w_gate_up, w_down,
                        d_ab, dx_perm, dw_gate_up, dw_down};
  for (const void *q : ptrs)
    if (!q || !moe::aligned16(q)) return moe::set_error(MOE_ERR_ARG, "moe_grouped_ffn_bwd: null or unaligned pointer");
  CUtensorMap mdO_k, mWd_mn, mdAB_k, mWgu_mn, mdO_mn, mH_mn, mdAB_mn, mX_mn;
  int st;
  if ((st = map_kmajor(&mdO_k, d_out_perm, rows_cap, d, "d_out_perm"))) return st;
  if ((st = map_mnmajor(&mWd_mn, w_down, uint64_t(E) * d, F, "w_down"))) return st;
  if ((st = map_kmajor(&mdAB_k, d_ab, rows_cap, 2 * F, "d_ab"))) return st;
  if ((st = map_mnmajor(&mWgu_mn, w_gate_up, uint64_t(E) * 2 * F, d, "w_gate_up"))) return st;
  if ((st = map_mnmajor(&mdO_mn, d_out_perm, rows_cap, d, "d_out_perm"))) return st;
  if ((st = map_mnmajor(&mH_mn, h, rows_cap, F, "h"))) return st;
  if ((st = map_mnmajor(&mdAB_mn, d_ab, rows_cap, 2 * F, "d_ab"))) return st;
  if ((st = map_mnmajor(&mX_mn, x_perm, rows_cap, d, "x_perm"))) return st;

  GemmParams p{};
  p.group_offsets = group_offsets;
  p.E = E; p.d = d; p.F = F;
  // dH = dO W_down, fused SwiGLU backward -> [dA | dB]
  p.nkb = d / BK;
  p.out = d_ab;
  p.aux = ab_saved;
  if ((st = launch_bn<kDgradDown>(F, mdO_k, mWd_mn, p, s, "moe_grouped_ffn_bwd: dH GEMM"))) return st;
  // dX = [dA | dB] W_gate_up
  p.nkb = 2 * F / BK;
  p.out = dx_perm;
  p.aux = nullptr;
  if ((st = launch_bn<kDgradGateUp>(d, mdAB_k, mWgu_mn, p, s, "moe_grouped_ffn_bwd: dX GEMM"))) return st;
  // dW_down[e] = dO_e^T H_e   ([d, F])
  p.nkb = 0;
  p.m_tiles_w = d / BM;
  p.out = dw_down;
  if ((st = launch_bn<kWgradDown>(F, mdO_mn, mH_mn, p, s, "moe_grouped_ffn_bwd: dW_down GEMM"))) return st;
  // dW_gate_up[e] = [dA | dB]_e^T X_e   ([2F, d])
  p.m_tiles_w = 2 * F / BM;
  p.out = dw_gate_up;
  return launch_bn<kWgradGateUp>(d, mdAB_mn, mX_mn, p, s, "moe_grouped_ffn_bwd: dW_gate_up GEMM");
}

}  // extern "C"
