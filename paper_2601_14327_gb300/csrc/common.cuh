// Shared host/device helpers of the MoE/LAEP CUDA library (sm_103a).
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>
#include <stddef.h>

#include <algorithm>

#include <nvtx3/nvToolsExt.h>

#include "../../include/moe_laep.h"

// ---------------------------------------------------------------- host side
namespace moe {

// Records the error text for moe_last_error_string() and returns `code`.
int set_error(int code, const char *fmt, ...);
// Checks a CUDA runtime result; on failure records it and returns MOE_ERR_CUDA.
int cuda_status(cudaError_t e, const char *what);
// Checks for a launch error right after a kernel launch.
int launch_status(const char *what);

inline bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int num_sms();

// The first bytes of every workspace belong to the grouped GEMMs' tile scheduler
// (their entry points know neither T nor k, so the region has a fixed offset and size).
constexpr size_t kGemmSchedBytes = 256;

// Workspace layout shared by the entry points (disjoint regions, 256-byte aligned).
struct WsLayout {
  size_t gemm_sched;    // int32 [1]               grouped GEMM tile counter (offset 0)
  size_t perm_hist;     // int32 [E * nblk]        moe_permute block histograms
  size_t route_dz3;     // bf16  [3, NP, Tp]       moe_route_bwd logit gradient as three bf16 terms
  size_t route_dw_partial; // fp32 [splits, d, NE] moe_route_bwd split-reduction partial sums
  size_t w_router_t;    // fp32  [E, d]            moe_permute_bwd transposed router
  size_t combine_rows;  // int32 + fp32 [rows_cap] moe_grouped_ffn_fwd_combine token and gate of each row
  size_t row_dz;        // fp32  [rows_cap]        moe_grouped_ffn_bwd_dgrad router logit gradient per grouped row
  size_t gate_partial;  // fp32  [rows_cap, F/64]  moe_grouped_ffn_bwd_dgrad per-row dH * H sums (gate gradient)
  size_t route_partial; // fp32  [splits, T, NE]   moe_route split-reduction partial logits
  size_t route_w3;      // bf16  [3, NP, d]        moe_route router weight as three bf16 terms
  size_t total;
};
WsLayout ws_layout(int T, int d, int E, int k, int F);
size_t route_partial_bytes(int T, int d, int E);
size_t route_w3_bytes(int d, int E);
size_t route_dz3_bytes(int T, int E);
size_t route_dw_partial_bytes(int T, int d, int E);
constexpr int kPermChunk = 4096;  // assignments per block in the permutation
constexpr int kGroupPad = 128;    // rows per group are padded to this

// Kernel timing registry (moe_timing_enable / moe_timing_read). When enabled,
// every kernel launch of the library is bracketed by CUDA events recorded on
// the launching stream; otherwise these calls cost a flag test.
cudaEvent_t timing_begin(cudaStream_t s);
void timing_end(const char *name, cudaEvent_t begin, cudaStream_t s);

// Device error words of each translation unit.
int route_dev_error(int clear, int *code);
int permute_dev_error(int clear, int *code);
int gemm_dev_error(int clear, int *code);

}  // namespace moe

// Launches a kernel (the variadic part is the launch statement) under the
// timing registry and inside an NVTX range named after it (a profiler can select
// the library's launches by range; without a tool attached the range costs a
// pointer test).
#define MOE_LAUNCH(name, stream, ...)                        \
  do {                                                       \
    nvtxRangePushA(name);                                    \
    cudaEvent_t moe_ev_ = moe::timing_begin(stream);         \
    __VA_ARGS__;                                             \
    moe::timing_end(name, moe_ev_, stream);                  \
    nvtxRangePop();                                          \
  } while (0)

// -------------------------------------------------------------- device side
#define MOE_DEV_ERR_DECL static __device__ int g_dev_err;
#define MOE_DEV_ERR_DEFINE_READER(fn)                                               \
  int fn(int clear, int *code) {                                                    \
    int v = 0;                                                                      \
    cudaError_t e = cudaMemcpyFromSymbol(&v, g_dev_err, sizeof(int));               \
    if (e != cudaSuccess) return moe::cuda_status(e, "read device error word");     \
    if (clear && v) {                                                               \
      int z = 0;                                                                    \
      e = cudaMemcpyToSymbol(g_dev_err, &z, sizeof(int));                           \
      if (e != cudaSuccess) return moe::cuda_status(e, "clear device error word");  \
    }                                                                               \
    *code = v;                                                                      \
    return MOE_OK;                                                                  \
  }

__device__ __forceinline__ void dev_flag(int *word, int code) { atomicCAS(word, 0, code); }

__device__ __forceinline__ float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xffff0000u); }

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 p = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t *>(&p);
}

// 8 bf16 values (one 16-byte vector) <-> 8 floats
__device__ __forceinline__ void unpack8(const uint4 &v, float (&f)[8]) {
  f[0] = bf16_lo(v.x); f[1] = bf16_hi(v.x);
  f[2] = bf16_lo(v.y); f[3] = bf16_hi(v.y);
  f[4] = bf16_lo(v.z); f[5] = bf16_hi(v.z);
  f[6] = bf16_lo(v.w); f[7] = bf16_hi(v.w);
}
__device__ __forceinline__ uint4 pack8(const float (&f)[8]) {
  uint4 v;
  v.x = pack_bf16x2(f[0], f[1]);
  v.y = pack_bf16x2(f[2], f[3]);
  v.z = pack_bf16x2(f[4], f[5]);
  v.w = pack_bf16x2(f[6], f[7]);
  return v;
}

__device__ __forceinline__ uint4 ldg_nc_v4(const void *p) {
  uint4 v;
  asm volatile("ld.global.nc.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
  return v;
}
__device__ __forceinline__ void stg_v4(void *p, const uint4 &v) {
  asm volatile("st.global.v4.u32 [%0], {%1,%2,%3,%4};" ::"l"(p), "r"(v.x), "r"(v.y), "r"(v.z),
               "r"(v.w)
               : "memory");
}
