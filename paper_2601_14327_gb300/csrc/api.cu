// Host-side entry points: errors, sizes, workspace layout, kernel timing.
#include <stdarg.h>
#include <stdio.h>

#include <algorithm>
#include <map>
#include <mutex>
#include <numeric>
#include <string>
#include <vector>

#include "common.cuh"

namespace moe {

static thread_local char g_err_text[512] = "";

int set_error(int code, const char *fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err_text, sizeof(g_err_text), fmt, ap);
  va_end(ap);
  return code;
}

int cuda_status(cudaError_t e, const char *what) {
  if (e == cudaSuccess) return MOE_OK;
  return set_error(MOE_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

int launch_status(const char *what) { return cuda_status(cudaGetLastError(), what); }

int num_sms() {
  static int cached[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 148;
  if (!cached[dev]) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
      n = 148;
    cached[dev] = n;
  }
  return cached[dev];
}

// ---- kernel timing registry ----
namespace {
struct TimingRec {
  const char *name;
  cudaEvent_t a, b;
};
struct Timing {
  std::mutex mu;
  bool enabled = false;
  std::vector<cudaEvent_t> pool;
  std::vector<TimingRec> recs;
};
Timing &timing() {
  static Timing t;
  return t;
}
cudaEvent_t take_event(Timing &t) {
  if (!t.pool.empty()) {
    cudaEvent_t e = t.pool.back();
    t.pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
  return e;
}
}  // namespace

cudaEvent_t timing_begin(cudaStream_t s) {
  Timing &t = timing();
  if (!t.enabled) return nullptr;
  std::lock_guard<std::mutex> g(t.mu);
  cudaEvent_t e = take_event(t);
  if (e && cudaEventRecord(e, s) != cudaSuccess) {
    t.pool.push_back(e);
    return nullptr;
  }
  return e;
}

void timing_end(const char *name, cudaEvent_t begin, cudaStream_t s) {
  if (!begin) return;
  Timing &t = timing();
  std::lock_guard<std::mutex> g(t.mu);
  cudaEvent_t e = take_event(t);
  if (!e || cudaEventRecord(e, s) != cudaSuccess) {
    t.pool.push_back(begin);
    if (e) t.pool.push_back(e);
    return;
  }
  t.recs.push_back({name, begin, e});
}

static size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

WsLayout ws_layout(int T, int d, int E, int k, int F) {
  (void)F;
  WsLayout w{};
  const int64_t A = int64_t(T) * k;
  const int64_t nblk = std::max<int64_t>(1, (A + kPermChunk - 1) / kPermChunk);
  size_t off = 0;
  w.gemm_sched = off;
  off += kGemmSchedBytes;
  w.perm_hist = off;
  off += align256(size_t(E) * nblk * 4);
  w.route_dz3 = off;
  off += align256(route_dz3_bytes(T, E));
  w.route_dw_partial = off;
  off += align256(route_dw_partial_bytes(T, d, E));
  w.w_router_t = off;
  off += align256(size_t(E) * d * 4);
  w.combine_rows = off;
  off += align256(size_t(moe_perm_rows_max(T, k, E)) * 8);
  w.row_dz = off;
  off += align256(size_t(moe_perm_rows_max(T, k, E)) * 4);
  w.gate_partial = off;
  off += align256(size_t(moe_perm_rows_max(T, k, E)) * size_t(std::max(F, 0) / 64) * 4);
  w.route_partial = off;
  off += align256(route_partial_bytes(T, d, E));
  w.route_w3 = off;
  off += align256(route_w3_bytes(d, E));
  w.total = off;
  return w;
}

}  // namespace moe

extern "C" {

int moe_version(void) { return 100; }

const char *moe_last_error_string(void) { return moe::g_err_text; }

int64_t moe_perm_rows_max(int T, int k, int E) {
  if (T < 0 || k < 0 || E < 0) return 0;
  return int64_t(T) * k + int64_t(moe::kGroupPad) * E;
}

size_t moe_workspace_size(int T, int d, int E, int k, int F) {
  if (T < 0 || d <= 0 || E <= 0 || k <= 0) return 0;
  return moe::ws_layout(T, d, E, k, F).total;
}

int moe_device_error(int *code, int clear) {
  if (!code) return moe::set_error(MOE_ERR_ARG, "moe_device_error: null code");
  int st = moe::cuda_status(cudaDeviceSynchronize(), "moe_device_error: synchronize");
  if (st) return st;
  int c0 = 0, c1 = 0, c2 = 0;
  if ((st = moe::route_dev_error(clear, &c0))) return st;
  if ((st = moe::permute_dev_error(clear, &c1))) return st;
  if ((st = moe::gemm_dev_error(clear, &c2))) return st;
  *code = c0 ? c0 : (c1 ? c1 : c2);
  return MOE_OK;
}

int moe_timing_enable(int enable) {
  moe::Timing &t = moe::timing();
  std::lock_guard<std::mutex> g(t.mu);
  t.enabled = enable != 0;
  return MOE_OK;
}

int moe_timing_read(char *buf, size_t buf_len, int reset) {
  if (!buf || buf_len == 0) return moe::set_error(MOE_ERR_ARG, "moe_timing_read: null buffer");
  moe::Timing &t = moe::timing();
  std::lock_guard<std::mutex> g(t.mu);
  struct Acc {
    long long n = 0;
    double ms = 0;
  };
  std::map<std::string, Acc> acc;
  std::vector<std::string> order;
  for (const auto &r : t.recs) {
    if (cudaEventSynchronize(r.b) != cudaSuccess)
      return moe::set_error(MOE_ERR_CUDA, "moe_timing_read: event synchronize");
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, r.a, r.b) != cudaSuccess)
      return moe::set_error(MOE_ERR_CUDA, "moe_timing_read: elapsed time");
    if (!acc.count(r.name)) order.push_back(r.name);
    acc[r.name].n += 1;
    acc[r.name].ms += ms;
  }
  size_t off = 0;
  buf[0] = 0;
  for (const auto &name : order) {
    const int w = snprintf(buf + off, buf_len - off, "%s %lld %.6f\n", name.c_str(), acc[name].n,
                           acc[name].ms);
    if (w < 0 || size_t(w) >= buf_len - off)
      return moe::set_error(MOE_ERR_ARG, "moe_timing_read: buffer too small");
    off += size_t(w);
  }
  if (reset) {
    for (const auto &r : t.recs) {
      t.pool.push_back(r.a);
      t.pool.push_back(r.b);
    }
    t.recs.clear();
  }
  return MOE_OK;
}

}  // extern "C"
