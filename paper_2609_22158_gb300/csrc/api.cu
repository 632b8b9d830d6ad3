// C ABI of the StepKV compression pass: argument validation, workspace layout, and the order of
// kernel launches.  Every function only enqueues work on the caller's stream.
#include <math.h>
#include <stdio.h>

#include <algorithm>
#include <mutex>
#include <map>
#include <utility>
#include <vector>

#include "common.cuh"
#include "internal.h"

namespace stepkv {

static thread_local char g_last_error[256] = {0};

// Caller-owned CUDA events stepkv_compress records on its stream (stepkv_set_stage_events), per thread.
struct StageEvents {
  cudaEvent_t e[3];
};
static thread_local StageEvents t_stage_events = {{nullptr, nullptr, nullptr}};

void set_last_cuda_error(cudaError_t e) {
  snprintf(g_last_error, sizeof(g_last_error), "%s: %s", cudaGetErrorName(e), cudaGetErrorString(e));
}

cudaError_t device_sm_count(int* n) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  return cudaDeviceGetAttribute(n, cudaDevAttrMultiProcessorCount, dev);
}

// Raise a kernel's dynamic shared-memory limit on the current device.  The limit only ever grows, so a
// launch that needs less than an earlier one keeps working.
cudaError_t ensure_smem_attr(const void* func, int bytes) {
  static std::mutex mu;
  static std::map<std::pair<const void*, int>, int> limit;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(mu);
  auto key = std::make_pair(func, dev);
  auto it = limit.find(key);
  if (it != limit.end() && it->second >= bytes) return cudaSuccess;
  e = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess) limit[key] = bytes;
  return e;
}

// Device-visible address of page-locked host memory (cudaHostAlloc / cudaHostRegister); false for any
// other kind of pointer (device, managed, pageable).
static bool host_pinned_device_ptr(const void* p, void** dev) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  if (a.type != cudaMemoryTypeHost || !a.devicePointer) return false;
  *dev = a.devicePointer;
  return true;
}

// A problem's cache pointers as the kernels see them: host-resident caches translated to their
// device-visible addresses.
struct CachePtrs {
  std::vector<const void*> K, V;
  std::vector<void*> K_out, V_out;
};

static stepkv_status_t resolve_cache_ptrs(const stepkv_problem_t& p, CachePtrs* c) {
  if ((p.kv_location != STEPKV_MEM_DEVICE && p.kv_location != STEPKV_MEM_HOST) ||
      (p.out_location != STEPKV_MEM_DEVICE && p.out_location != STEPKV_MEM_HOST))
    return STEPKV_EINVAL;
  c->K.assign(p.K, p.K + p.L);
  c->V.assign(p.V, p.V + p.L);
  c->K_out.assign(p.K_out, p.K_out + p.L);
  c->V_out.assign(p.V_out, p.V_out + p.L);
  auto tr_in = [](std::vector<const void*>& v) {
    for (auto& x : v) {
      void* d = nullptr;
      if (!host_pinned_device_ptr(x, &d)) return false;
      x = d;
    }
    return true;
  };
  auto tr_out = [](std::vector<void*>& v) {
    for (auto& x : v) {
      void* d = nullptr;
      if (!host_pinned_device_ptr(x, &d)) return false;
      x = d;
    }
    return true;
  };
  if (p.kv_location == STEPKV_MEM_HOST && !(tr_in(c->K) && tr_in(c->V))) return STEPKV_EINVAL;
  if (p.out_location == STEPKV_MEM_HOST && !(tr_out(c->K_out) && tr_out(c->V_out))) return STEPKV_EINVAL;
  return STEPKV_OK;
}

static size_t align256(size_t x) { return (x + 255) & ~size_t(255); }
static bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

static stepkv_status_t check_score_args(int n_layers, const void* const* K, int64_t k_head_stride, const void* const* Q,
                                        int64_t q_head_stride, int Hkv, int Hq, int d, int T, int W) {
  if (n_layers < 1 || n_layers > kMaxSalLayers) return STEPKV_EUNSUPPORTED;
  if (!K || !Q) return STEPKV_EINVAL;
  if (Hkv < 1 || Hq < 1 || Hq % Hkv != 0 || T < 1 || W < 1 || W > T) return STEPKV_EINVAL;
  if (d != 64 && d != 128) return STEPKV_EUNSUPPORTED;
  if (W > 4096) return STEPKV_EUNSUPPORTED;
  if (k_head_stride < (int64_t)T * d || q_head_stride < (int64_t)W * d) return STEPKV_EINVAL;
  if (k_head_stride % 8 || q_head_stride % 8) return STEPKV_EUNSUPPORTED;
  for (int l = 0; l < n_layers; ++l) {
    if (!K[l] || !Q[l]) return STEPKV_EINVAL;
    if (!aligned16(K[l]) || !aligned16(Q[l])) return STEPKV_EUNSUPPORTED;
  }
  return STEPKV_OK;
}

static stepkv_status_t check_select_args(int n_sal, int T, const int32_t* step_id, const uint8_t* prot,
                                         const stepkv_steps_t* steps, const stepkv_params_t* params,
                                         const stepkv_budget_t* budget, const stepkv_select_out_t* out) {
  if (!steps || !params || !budget || !out || !step_id || !prot) return STEPKV_EINVAL;
  if (n_sal < 1 || T < 1) return STEPKV_EINVAL;
  if (T > 262144) return STEPKV_EUNSUPPORTED;
  if (steps->n_steps < 1 || steps->n_steps > 65535) return STEPKV_EINVAL;
  if (!steps->valid || !steps->gain || !steps->red || !steps->reuse_in) return STEPKV_EINVAL;
  if (!out->kept_idx || !out->n_kept || out->kept_cap < 0) return STEPKV_EINVAL;
  if (params->sal_norm != STEPKV_NORM_MAX && params->sal_norm != STEPKV_NORM_NONE) return STEPKV_EINVAL;
  if (params->sal_pool < 1 || params->sal_pool > STEPKV_MAX_POOL || (params->sal_pool & 1) == 0) return STEPKV_EINVAL;
  if (params->sal_pool_mode != STEPKV_POOL_MAX && params->sal_pool_mode != STEPKV_POOL_AVG) return STEPKV_EINVAL;
  if (budget->mode == STEPKV_BUDGET_RATIO) {
    if (budget->ratio_num < 0 || budget->ratio_den < 1) return STEPKV_EINVAL;
  } else if (budget->mode == STEPKV_BUDGET_COUNT) {
    if (budget->count < 0) return STEPKV_EINVAL;
  } else {
    return STEPKV_EINVAL;
  }
  return STEPKV_OK;
}

// In place (every K_out[l] == K_in[l] and V_out[l] == V_in[l], one head stride) is accepted only where
// `inplace` is non-null (the fused pass); it is then reported there.
static stepkv_status_t check_compact_args(int n_layers, const void* const* K_in, const void* const* V_in,
                                          int64_t in_head_stride, int Hkv, int d, int T, const int32_t* kept_idx,
                                          const int32_t* n_kept, int kept_cap, void* const* K_out,
                                          void* const* V_out, int64_t out_head_stride, bool* inplace = nullptr) {
  if (inplace) *inplace = false;
  if (n_layers < 0 || Hkv < 1 || d < 8 || T < 1 || kept_cap < 0) return STEPKV_EINVAL;
  if (!kept_idx || !n_kept) return STEPKV_EINVAL;
  if ((d * 2) % 16 || d > 256) return STEPKV_EUNSUPPORTED;
  // one launch's row items of a trajectory (at most 96 layers x K, V x heads x kept_cap) use 32-bit indices
  if ((int64_t)std::min(n_layers, 96) * 2 * Hkv * std::max(kept_cap, 1) >= ((int64_t)1 << 30))
    return STEPKV_EUNSUPPORTED;
  if (n_layers > 0) {
    if (!K_in || !K_out) return STEPKV_EINVAL;
    if ((V_in == nullptr) != (V_out == nullptr)) return STEPKV_EINVAL;
    if (in_head_stride < (int64_t)T * d || out_head_stride < (int64_t)kept_cap * d) return STEPKV_EINVAL;
    if (in_head_stride % 8 || out_head_stride % 8) return STEPKV_EUNSUPPORTED;
    int same = 0, tensors = 0;
    for (int l = 0; l < n_layers; ++l) {
      if (!K_in[l] || !K_out[l]) return STEPKV_EINVAL;
      if (!aligned16(K_in[l]) || !aligned16(K_out[l])) return STEPKV_EUNSUPPORTED;
      same += K_in[l] == K_out[l];
      ++tensors;
      if (V_in) {
        if (!V_in[l] || !V_out[l]) return STEPKV_EINVAL;
        if (!aligned16(V_in[l]) || !aligned16(V_out[l])) return STEPKV_EUNSUPPORTED;
        same += V_in[l] == V_out[l];
        ++tensors;
      }
    }
    if (same != 0) {
      if (!inplace || same != tensors || in_head_stride != out_head_stride) return STEPKV_EUNSUPPORTED;
      *inplace = true;
    }
  }
  return STEPKV_OK;
}

static size_t score_ws(int n_layers, int Hkv, int Hq, int T, int W, bool need_rows) {
  const int n_rg = score_row_groups(Hkv, Hq, W);
  size_t b = align256(score_partial_bytes(n_layers, Hkv, Hq, W));
  if (need_rows) b += align256((size_t)n_layers * Hkv * n_rg * T * sizeof(float));
  return b;
}

}  // namespace stepkv

using namespace stepkv;

extern "C" {

void stepkv_default_params(stepkv_params_t* p) {
  if (!p) return;
  p->lambda = 0.3f;
  p->w_r = 0.85f;
  p->w_c = 0.15f;
  p->r_min = -1.0f;
  p->r_max = 2.0f;
  p->s_max = 8.0f;
  p->eta = 1.5f;
  p->alpha = 0.2f;
  p->beta = 0.8f;
  p->sal_norm = STEPKV_NORM_MAX;
  p->sal_pool = 1;
  p->sal_pool_mode = STEPKV_POOL_MAX;
}

// T_i from the saliency rows: their mean, each row first pooled over params->sal_pool tokens when
// that is > 1 (the SnapKV-style estimator).
static stepkv_status_t token_saliency_run(const float* sal, int n_sal, int T, const stepkv_params_t& params,
                                          float* Tbuf, cudaStream_t s) {
  if (params.sal_pool > 1)
    return pool_mean_rows_run(sal, n_sal, T, 1.0f / (float)n_sal, T, params.sal_pool / 2,
                              params.sal_pool_mode == STEPKV_POOL_MAX, Tbuf, s);
  return mean_rows_run(sal, n_sal, T, 1.0f / (float)n_sal, T, Tbuf, s);
}

const char* stepkv_status_string(int32_t status) {
  switch (status) {
    case STEPKV_OK: return "ok";
    case STEPKV_EINVAL: return "invalid argument";
    case STEPKV_ECUDA: return "CUDA error";
    case STEPKV_ENOSPACE: return "insufficient space (workspace or kept_cap)";
    case STEPKV_EUNSUPPORTED: return "unsupported shape or alignment";
    case STEPKV_EDATA: return "invalid data (step id or kept index out of range)";
    case STEPKV_ETIMEOUT: return "device-side wait timed out";
    default: return "unknown status";
  }
}

int32_t stepkv_version(void) { return 1000; }

const char* stepkv_last_cuda_error(void) { return g_last_error; }

size_t stepkv_score_workspace_size(int32_t n_layers, int32_t Hkv, int32_t Hq, int32_t T, int32_t W) {
  if (n_layers < 1 || Hkv < 1 || Hq < Hkv || T < 1 || W < 1) return 0;
  return score_ws(n_layers, Hkv, Hq, T, W, score_row_groups(Hkv, Hq, W) > 1);
}

static stepkv_status_t score_entry(int32_t n_layers, const void* const* K, int64_t k_head_stride,
                                   const void* const* Q, int64_t q_head_stride, const float* const* lse, int32_t Hkv,
                                   int32_t Hq, int32_t d, int32_t T, int32_t W, float* sal, void* ws, size_t ws_bytes,
                                   int32_t* dev_status, void* stream) {
  stepkv_status_t st = check_score_args(n_layers, K, k_head_stride, Q, q_head_stride, Hkv, Hq, d, T, W);
  if (st != STEPKV_OK) return st;
  if (lse) {
    for (int l = 0; l < n_layers; ++l)
      if (!lse[l] || (reinterpret_cast<uintptr_t>(lse[l]) & 3u) != 0) return STEPKV_EINVAL;
  }
  if (!sal || !ws) return STEPKV_EINVAL;
  const int n_rg = score_row_groups(Hkv, Hq, W);
  const size_t need = score_ws(n_layers, Hkv, Hq, T, W, n_rg > 1);
  if (ws_bytes < need) return STEPKV_ENOSPACE;
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return STEPKV_EINVAL;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  float2* part = static_cast<float2*>(ws);
  float* rows = sal;
  if (n_rg > 1)
    rows = reinterpret_cast<float*>(static_cast<uint8_t*>(ws) + align256(score_partial_bytes(n_layers, Hkv, Hq, W)));
  st = score_run(n_layers, K, k_head_stride, Q, q_head_stride, Hkv, Hq, d, T, W, rows, T, nullptr, 0, part,
                 dev_status, s, 0, lse);
  if (st != STEPKV_OK) return st;
  if (n_rg > 1) st = score_sum_row_groups(rows, n_layers * Hkv, n_rg, T, sal, s);
  return st;
}

stepkv_status_t stepkv_score(int32_t n_layers, const void* const* K, int64_t k_head_stride, const void* const* Q,
                             int64_t q_head_stride, int32_t Hkv, int32_t Hq, int32_t d, int32_t T, int32_t W,
                             float* sal, void* ws, size_t ws_bytes, int32_t* dev_status, void* stream) {
  return score_entry(n_layers, K, k_head_stride, Q, q_head_stride, nullptr, Hkv, Hq, d, T, W, sal, ws, ws_bytes,
                     dev_status, stream);
}

stepkv_status_t stepkv_score_lse(int32_t n_layers, const void* const* K, int64_t k_head_stride, const void* const* Q,
                                 int64_t q_head_stride, const float* const* lse, int32_t Hkv, int32_t Hq, int32_t d,
                                 int32_t T, int32_t W, float* sal, void* ws, size_t ws_bytes, int32_t* dev_status,
                                 void* stream) {
  if (!lse) return STEPKV_EINVAL;
  return score_entry(n_layers, K, k_head_stride, Q, q_head_stride, lse, Hkv, Hq, d, T, W, sal, ws, ws_bytes,
                     dev_status, stream);
}

stepkv_status_t stepkv_selftest_score_timeout(int32_t n_layers, const void* const* K, int64_t k_head_stride,
                                              const void* const* Q, int64_t q_head_stride, int32_t Hkv, int32_t Hq,
                                              int32_t d, int32_t T, int32_t W, float* sal, void* ws, size_t ws_bytes,
                                              uint64_t wait_limit_ns, int32_t* dev_status, void* stream) {
  stepkv_status_t st = check_score_args(n_layers, K, k_head_stride, Q, q_head_stride, Hkv, Hq, d, T, W);
  if (st != STEPKV_OK) return st;
  if (!sal || !ws || !dev_status) return STEPKV_EINVAL;
  if (wait_limit_ns < 1000 || wait_limit_ns > kWaitLimitNs) return STEPKV_EINVAL;
  if (ws_bytes < score_ws(n_layers, Hkv, Hq, T, W, false)) return STEPKV_ENOSPACE;
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return STEPKV_EINVAL;
  if (score_row_groups(Hkv, Hq, W) != 1) return STEPKV_EUNSUPPORTED;  // G*W <= 256: rows straight into sal
  return score_run(n_layers, K, k_head_stride, Q, q_head_stride, Hkv, Hq, d, T, W, sal, T, nullptr, 0,
                   static_cast<float2*>(ws), dev_status, static_cast<cudaStream_t>(stream), wait_limit_ns);
}

size_t stepkv_select_workspace_size(int32_t n_sal, int32_t T, int32_t n_steps) {
  (void)n_sal;
  if (T < 1 || n_steps < 1) return 0;
  return align256((size_t)T * sizeof(float)) + select_ws_bytes(T, n_steps);
}

stepkv_status_t stepkv_select(const float* sal, int32_t n_sal, int32_t T, const int32_t* step_id,
                              const uint8_t* prot, const stepkv_steps_t* steps, const stepkv_params_t* params,
                              const stepkv_budget_t* budget, const stepkv_select_out_t* out, void* ws,
                              size_t ws_bytes, int32_t* dev_status, void* stream) {
  stepkv_status_t st = check_select_args(n_sal, T, step_id, prot, steps, params, budget, out);
  if (st != STEPKV_OK) return st;
  if (!sal || !ws) return STEPKV_EINVAL;
  if (ws_bytes < stepkv_select_workspace_size(n_sal, T, steps->n_steps)) return STEPKV_ENOSPACE;
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return STEPKV_EINVAL;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  float* Tbuf = static_cast<float*>(ws);
  void* sel_ws = static_cast<uint8_t*>(ws) + align256((size_t)T * sizeof(float));
  st = token_saliency_run(sal, n_sal, T, *params, Tbuf, s);
  if (st != STEPKV_OK) return st;
  return select_run(Tbuf, nullptr, 0.0, T, step_id, prot, *steps, *params, *budget, *out, sel_ws, dev_status, s);
}

// Selection with a fixed device scratch instead of a caller workspace, for callers that cannot
// allocate device memory at call time (fully pre-reserved HBM, no tolerance for the synchronisation
// of cudaFree, no caching allocator).  Not part of the method.  The array below is the only scratch;
// its address is looked up once per device and reused, so calls that overlap on one device race.
// Layout: the mean saliency row (4 B per token), then the step utility, count, fixed-point sum, max
// and kept count (24 B per step), each 256-byte aligned: 1,146,880 bytes at the limits.
static __device__ __align__(256) unsigned char g_select_scratch[(size_t)STEPKV_STATIC_SCRATCH_MAX_T * 4 +
                                                                (size_t)STEPKV_STATIC_SCRATCH_MAX_STEPS * 24];
constexpr int kScratchDevices = 64;
static std::mutex g_scratch_mu;
static void* g_scratch_addr[kScratchDevices];

static stepkv_status_t static_scratch_address(void** addr) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return STEPKV_ECUDA;
  }
  if (dev < 0 || dev >= kScratchDevices) return STEPKV_EUNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (!g_scratch_addr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_select_scratch);
    if (e != cudaSuccess || !p) {
      set_last_cuda_error(e);
      return STEPKV_ECUDA;
    }
    g_scratch_addr[dev] = p;
  }
  *addr = g_scratch_addr[dev];
  return STEPKV_OK;
}

stepkv_status_t stepkv_select_static_scratch(const float* sal, int32_t n_sal, int32_t T, const int32_t* step_id,
                                             const uint8_t* prot, const stepkv_steps_t* steps,
                                             const stepkv_params_t* params, const stepkv_budget_t* budget,
                                             const stepkv_select_out_t* out, int32_t* dev_status, void* stream) {
  stepkv_status_t st = check_select_args(n_sal, T, step_id, prot, steps, params, budget, out);
  if (st != STEPKV_OK) return st;
  if (!sal) return STEPKV_EINVAL;
  if (T > STEPKV_STATIC_SCRATCH_MAX_T || steps->n_steps > STEPKV_STATIC_SCRATCH_MAX_STEPS) return STEPKV_ENOSPACE;
  const size_t t_bytes = align256((size_t)T * sizeof(float));
  if (t_bytes + select_ws_bytes(T, steps->n_steps) > sizeof(g_select_scratch)) return STEPKV_ENOSPACE;
  void* scratch = nullptr;
  st = static_scratch_address(&scratch);
  if (st != STEPKV_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  float* Tbuf = static_cast<float*>(scratch);
  void* sel_ws = static_cast<uint8_t*>(scratch) + t_bytes;
  st = token_saliency_run(sal, n_sal, T, *params, Tbuf, s);
  if (st != STEPKV_OK) return st;
  return select_run(Tbuf, nullptr, 0.0, T, step_id, prot, *steps, *params, *budget, *out, sel_ws, dev_status, s);
}

stepkv_status_t stepkv_compact(int32_t n_layers, const void* const* K_in, const void* const* V_in,
                               int64_t in_head_stride, int32_t Hkv, int32_t d, int32_t T, const int32_t* kept_idx,
                               const int32_t* n_kept, int32_t kept_cap, void* const* K_out, void* const* V_out,
                               int64_t out_head_stride, const int32_t* step_id_in, const int32_t* pos_in,
                               int32_t* step_id_out, int32_t* pos_out, int32_t* dev_status, void* stream) {
  stepkv_status_t st = check_compact_args(n_layers, K_in, V_in, in_head_stride, Hkv, d, T, kept_idx, n_kept, kept_cap,
                                          K_out, V_out, out_head_stride);
  if (st != STEPKV_OK) return st;
  return compact_run(n_layers, K_in, V_in, in_head_stride, Hkv, d, T, kept_idx, n_kept, kept_cap, K_out, V_out,
                     out_head_stride, step_id_in, pos_in, step_id_out, pos_out, dev_status,
                     static_cast<cudaStream_t>(stream));
}

size_t stepkv_decode_workspace_size(int32_t n_layers, int32_t Hkv, int32_t Hq, int32_t d, int32_t n_cap) {
  if (n_layers < 1 || Hkv < 1 || Hq < Hkv || n_cap < 1 || (d != 64 && d != 128)) return 0;
  return decode_ws_bytes(std::min(n_layers, kMaxDecodeLayers), Hkv, Hq, d, n_cap);
}

stepkv_status_t stepkv_decode(int32_t n_layers, const void* const* q, const void* const* K, const void* const* V,
                              int64_t kv_head_stride, int32_t Hkv, int32_t Hq, int32_t d, const int32_t* n_dev,
                              int32_t n_host, int32_t n_cap, float* const* out, void* ws, size_t ws_bytes,
                              int32_t* dev_status, void* stream) {
  if (n_layers < 1 || !q || !K || !V || !out || !ws) return STEPKV_EINVAL;
  if (Hkv < 1 || Hq < 1 || Hq % Hkv != 0 || n_cap < 1) return STEPKV_EINVAL;
  if (d != 64 && d != 128) return STEPKV_EUNSUPPORTED;
  const int G = Hq / Hkv;
  if (G != 1 && G != 2 && G != 4 && G != 5 && G != 8) return STEPKV_EUNSUPPORTED;
  if (kv_head_stride < (int64_t)n_cap * d) return STEPKV_EINVAL;
  if (kv_head_stride % 8) return STEPKV_EUNSUPPORTED;
  if (!n_dev && (n_host < 1 || n_host > n_cap)) return STEPKV_EINVAL;
  if (ws_bytes < stepkv_decode_workspace_size(n_layers, Hkv, Hq, d, n_cap)) return STEPKV_ENOSPACE;
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return STEPKV_EINVAL;
  for (int l = 0; l < n_layers; ++l) {
    if (!q[l] || !K[l] || !V[l] || !out[l]) return STEPKV_EINVAL;
    if (!aligned16(q[l]) || !aligned16(K[l]) || !aligned16(V[l]) || !aligned16(out[l])) return STEPKV_EUNSUPPORTED;
  }
  return decode_run(n_layers, q, K, V, kv_head_stride, Hkv, Hq, d, n_dev, n_host, n_cap, out, ws, dev_status,
                    static_cast<cudaStream_t>(stream));
}

stepkv_status_t stepkv_step_signals(const uint32_t* cues, const int32_t* n_cues, int32_t n_steps, int32_t k0,
                                    float* gain, float* red, float* obs_sim, int32_t* dev_status, void* stream) {
  if (!cues || !n_cues || n_steps < 1 || n_steps > 65535 || k0 < 0 || k0 > n_steps) return STEPKV_EINVAL;
  if (k0 < n_steps && (!gain || !red)) return STEPKV_EINVAL;
  if ((reinterpret_cast<uintptr_t>(cues) & 3u) || (reinterpret_cast<uintptr_t>(n_cues) & 3u)) return STEPKV_EUNSUPPORTED;
  return signals_run(cues, n_cues, n_steps, k0, gain, red, obs_sim, dev_status, static_cast<cudaStream_t>(stream));
}

size_t stepkv_decode_h2o_workspace_size(int32_t n_layers, int32_t Hkv, int32_t Hq, int32_t d, int32_t n_cap) {
  if (stepkv_decode_workspace_size(n_layers, Hkv, Hq, d, n_cap) == 0) return 0;
  return decode_mass_ws_bytes(std::min(n_layers, kMaxDecodeLayers), Hkv, Hq, d, n_cap);
}

stepkv_status_t stepkv_decode_h2o(int32_t n_layers, const void* const* q, const void* const* K, const void* const* V,
                                  int64_t kv_head_stride, int32_t Hkv, int32_t Hq, int32_t d, const int32_t* n_dev,
                                  int32_t n_host, int32_t n_cap, float* const* out, float* const* mass,
                                  int64_t mass_head_stride, void* ws, size_t ws_bytes, int32_t* dev_status,
                                  void* stream) {
  if (!mass || mass_head_stride < n_cap) return STEPKV_EINVAL;
  for (int l = 0; l < n_layers; ++l)
    if (!mass[l]) return STEPKV_EINVAL;
  if (ws_bytes < stepkv_decode_h2o_workspace_size(n_layers, Hkv, Hq, d, n_cap)) return STEPKV_ENOSPACE;
  // every other argument rule is stepkv_decode's
  if (n_layers < 1 || !q || !K || !V || !out || !ws) return STEPKV_EINVAL;
  if (Hkv < 1 || Hq < 1 || Hq % Hkv != 0 || n_cap < 1) return STEPKV_EINVAL;
  if (d != 64 && d != 128) return STEPKV_EUNSUPPORTED;
  const int G = Hq / Hkv;
  if (G != 1 && G != 2 && G != 4 && G != 5 && G != 8) return STEPKV_EUNSUPPORTED;
  if (kv_head_stride < (int64_t)n_cap * d) return STEPKV_EINVAL;
  if (kv_head_stride % 8) return STEPKV_EUNSUPPORTED;
  if (!n_dev && (n_host < 1 || n_host > n_cap)) return STEPKV_EINVAL;
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return STEPKV_EINVAL;
  for (int l = 0; l < n_layers; ++l) {
    if (!q[l] || !K[l] || !V[l] || !out[l]) return STEPKV_EINVAL;
    if (!aligned16(q[l]) || !aligned16(K[l]) || !aligned16(V[l]) || !aligned16(out[l])) return STEPKV_EUNSUPPORTED;
    if ((reinterpret_cast<uintptr_t>(mass[l]) & 3u) != 0) return STEPKV_EUNSUPPORTED;
  }
  return decode_run(n_layers, q, K, V, kv_head_stride, Hkv, Hq, d, n_dev, n_host, n_cap, out, ws, dev_status,
                    static_cast<cudaStream_t>(stream), mass, mass_head_stride);
}

// K of the saliency layers as the score stage reads it (device memory in either cache location).
static const void* const* sal_keys(const stepkv_problem_t& p) {
  const int Ls = std::min(p.n_sal_layers, p.L);
  return p.kv_location == STEPKV_MEM_HOST ? p.K_sal : p.K + (p.L - Ls);
}

// Saliency batches of the fused pass: runs of consecutive trajectories with one head shape (lengths and
// strides may differ), up to kMaxScoreBatch trajectories and kMaxScoreMaps tensor maps each, share one
// launch while the batch's saliency keys total at most kSalBatchBytes.  Each launch has fixed costs (the
// ring's first fill, the change of pass, the exit skew: ~20 us), which a batch pays once; against that,
// the second pass finds fewer of the tiles the first pass read last still in L2 the more keys a launch
// streams.  512 MB is the measured optimum for 16 trajectories of 8K-32K tokens (Llama-3-8B heads:
// 64 MB 2.68 ms, 256 MB 2.58, 512 MB 2.48, 1 GB 2.54, one launch for all 2.82 ms at a 10% budget).
constexpr size_t kSalBatchBytes = 512ull << 20;
struct SalBatch {
  int first, n;
};
static size_t sal_key_bytes(const stepkv_problem_t& p) {
  return (size_t)std::min(p.n_sal_layers, p.L) * p.Hkv * p.T * p.d * 2;
}
static std::vector<SalBatch> saliency_batches(const stepkv_problem_t* probs, int n_traj) {
  std::vector<SalBatch> out;
  auto same = [](const stepkv_problem_t& a, const stepkv_problem_t& b) {
    return std::min(a.n_sal_layers, a.L) == std::min(b.n_sal_layers, b.L) && a.Hkv == b.Hkv && a.Hq == b.Hq &&
           a.d == b.d && a.W == b.W && (a.sal_lse != nullptr) == (b.sal_lse != nullptr);
  };
  for (int i = 0; i < n_traj;) {
    const int Ls = std::max(1, std::min(probs[i].n_sal_layers, probs[i].L));
    int n = 1;
    size_t bytes = sal_key_bytes(probs[i]);
    while (i + n < n_traj && n < kMaxScoreBatch && (n + 1) * Ls <= kMaxScoreMaps && same(probs[i], probs[i + n]) &&
           bytes + sal_key_bytes(probs[i + n]) <= kSalBatchBytes) {
      bytes += sal_key_bytes(probs[i + n]);
      ++n;
    }
    out.push_back(SalBatch{i, n});
    i += n;
  }
  return out;
}

// Workspace of the fused pass: one region of pass-1 partials (the saliency launches run one after
// another and reuse it; sized for the largest batch), then per trajectory its fixed-point token
// saliency T_acc and its selection scratch (all selections run in one batched launch, so these are
// private).
static size_t compress_part_bytes(const stepkv_problem_t& p, int n_batch) {
  const int Ls = std::min(p.n_sal_layers, p.L);
  return align256(score_partial_bytes(Ls, p.Hkv, p.Hq, p.W, n_batch));
}
static size_t compress_traj_bytes(const stepkv_problem_t& p) {
  return align256((size_t)p.T * sizeof(unsigned long long)) + align256(select_ws_bytes(p.T, p.steps.n_steps)) +
         align256(compact_inplace_ws_bytes(p.T));
}
// Saliency rows of one trajectory, for a pooled token saliency (params.sal_pool > 1), which needs every
// (layer, KV head) row before the mean: the row groups' rows, then (when there are several row groups)
// their per-(layer, KV head) sums.  One region, reused trajectory after trajectory.
static size_t compress_rows_bytes(const stepkv_problem_t& p) {
  const int Ls = std::min(p.n_sal_layers, p.L);
  const int n_rg = score_row_groups(p.Hkv, p.Hq, p.W);
  return align256((size_t)Ls * p.Hkv * (n_rg + (n_rg > 1 ? 1 : 0)) * p.T * sizeof(float));
}

size_t stepkv_compress_workspace_size(const stepkv_problem_t* probs, int32_t n_traj) {
  if (!probs || n_traj < 1) return 0;
  size_t part = 0, per = 0, rows = 0;
  for (int i = 0; i < n_traj; ++i) {
    const stepkv_problem_t& p = probs[i];
    if (p.L < 1 || p.Hkv < 1 || p.Hq < p.Hkv || p.T < 1 || p.W < 1 || p.n_sal_layers < 1 || p.steps.n_steps < 1)
      return 0;
    per += compress_traj_bytes(p);
    rows = std::max(rows, compress_rows_bytes(p));
  }
  for (const SalBatch& b : saliency_batches(probs, n_traj))
    part = std::max(part, compress_part_bytes(probs[b.first], b.n));
  return part + per + rows;
}

stepkv_status_t stepkv_compress(const stepkv_problem_t* probs, int32_t n_traj, const stepkv_params_t* params,
                                void* ws, size_t ws_bytes, int32_t* dev_status, void* stream) {
  if (!probs || n_traj < 1 || !params || !ws) return STEPKV_EINVAL;
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return STEPKV_EINVAL;
  // validate everything before enqueueing anything
  std::vector<char> in_place((size_t)n_traj, 0);
  for (int i = 0; i < n_traj; ++i) {
    const stepkv_problem_t& p = probs[i];
    if (p.L < 1 || p.n_sal_layers < 1) return STEPKV_EINVAL;
    const int Ls = std::min(p.n_sal_layers, p.L);
    if (Ls > kMaxSalLayers) return STEPKV_EUNSUPPORTED;
    if (!p.K || !p.Q) return STEPKV_EINVAL;
    if (p.kv_location == STEPKV_MEM_HOST && !p.K_sal) return STEPKV_EINVAL;
    stepkv_status_t st = check_score_args(Ls, sal_keys(p), p.kv_head_stride, p.Q, p.q_head_stride, p.Hkv, p.Hq,
                                          p.d, p.T, p.W);
    if (st != STEPKV_OK) return st;
    st = check_select_args(Ls * p.Hkv, p.T, p.step_id, p.prot, &p.steps, params, &p.budget, &p.sel);
    if (st != STEPKV_OK) return st;
    if (p.sal_lse) {
      for (int l = 0; l < Ls; ++l)
        if (!p.sal_lse[l] || (reinterpret_cast<uintptr_t>(p.sal_lse[l]) & 3u) != 0) return STEPKV_EINVAL;
    }
    bool inplace = false;
    st = check_compact_args(p.L, p.K, p.V, p.kv_head_stride, p.Hkv, p.d, p.T, p.sel.kept_idx, p.sel.n_kept,
                            p.sel.kept_cap, p.K_out, p.V_out, p.out_head_stride, &inplace);
    if (st != STEPKV_OK) return st;
    if (inplace && p.kv_location != p.out_location) return STEPKV_EINVAL;
    in_place[i] = inplace ? 1 : 0;
  }
  // cache pointers as the kernels see them (host-resident caches: checked and translated here)
  std::vector<CachePtrs> caches((size_t)n_traj);
  for (int i = 0; i < n_traj; ++i) {
    stepkv_status_t st = resolve_cache_ptrs(probs[i], &caches[i]);
    if (st != STEPKV_OK) return st;
  }
  if (ws_bytes < stepkv_compress_workspace_size(probs, n_traj)) return STEPKV_ENOSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const std::vector<SalBatch> batches = saliency_batches(probs, n_traj);
  size_t part_bytes = 0;
  for (const SalBatch& b : batches) part_bytes = std::max(part_bytes, compress_part_bytes(probs[b.first], b.n));
  float2* part = reinterpret_cast<float2*>(ws);
  uint8_t* w = static_cast<uint8_t*>(ws) + part_bytes;
  std::vector<SelectSpec> specs((size_t)n_traj);
  std::vector<void*> plan_ws((size_t)n_traj);
  std::vector<ScoreTrajSpec> sal((size_t)n_traj);
  // a pooled token saliency (SnapKV-style) needs every (layer, KV head) row before the mean, so the
  // saliency stage writes rows per trajectory and a pooling launch forms T; the fixed-point token sums of
  // the fused saliency pass are not used then (their region holds the float T instead)
  const bool pooled = params->sal_pool > 1;
  std::vector<float*> t_float((size_t)n_traj);
  for (int i = 0; i < n_traj; ++i) {
    const stepkv_problem_t& p = probs[i];
    const int Ls = std::min(p.n_sal_layers, p.L);
    unsigned long long* t_acc = reinterpret_cast<unsigned long long*>(w);
    void* sel_ws = w + align256((size_t)p.T * sizeof(unsigned long long));
    plan_ws[i] = static_cast<uint8_t*>(sel_ws) + align256(select_ws_bytes(p.T, p.steps.n_steps));
    w += compress_traj_bytes(p);
    const int n_pairs = Ls * p.Hkv;
    const int shift = score_acc_shift(n_pairs, p.W);
    sal[i] = ScoreTrajSpec{sal_keys(p), p.Q, p.T, t_acc, p.kv_head_stride, p.q_head_stride, p.sal_lse};
    t_float[i] = reinterpret_cast<float*>(t_acc);
    specs[i] = pooled ? SelectSpec{t_float[i], nullptr, 0.0, p.T, p.step_id, p.prot, p.steps, *params, p.budget,
                                   p.sel, sel_ws, dev_status}
                      : SelectSpec{nullptr, t_acc, ldexp(1.0, -shift) / (double)n_pairs, p.T, p.step_id, p.prot,
                                   p.steps, *params, p.budget, p.sel, sel_ws, dev_status};
    if (in_place[i]) {  // the selection also writes the hole-filling plan and the in-place rows' metadata
      specs[i].plan = static_cast<int32_t*>(plan_ws[i]);
      specs[i].pos_in = p.pos_in;
      specs[i].step_id_out = p.step_id_out;
      specs[i].pos_out = p.pos_out;
    }
  }
  float* rows_ws = reinterpret_cast<float*>(w);  // compress_rows_bytes of the largest trajectory
  // optional stage timing (profiling): caller-owned events recorded on the stream of this call
  const StageEvents ev = t_stage_events;
  if (ev.e[0]) {
    const cudaError_t er = cudaEventRecord(ev.e[0], s);
    if (er != cudaSuccess) { set_last_cuda_error(er); return STEPKV_ECUDA; }
  }
  // stage 1: one cooperative launch per saliency batch (pooled: per trajectory, rows then the pooled mean)
  for (const SalBatch& b : (pooled ? std::vector<SalBatch>{} : batches)) {
    const stepkv_problem_t& p = probs[b.first];
    const int Ls = std::min(p.n_sal_layers, p.L);
    stepkv_status_t st = score_run_batch(Ls, &sal[b.first], b.n, p.Hkv, p.Hq, p.d, p.W, nullptr, 0,
                                         score_acc_shift(Ls * p.Hkv, p.W), part, dev_status, s);
    if (st != STEPKV_OK) return st;
  }
  for (int i = 0; pooled && i < n_traj; ++i) {
    const stepkv_problem_t& p = probs[i];
    const int Ls = std::min(p.n_sal_layers, p.L);
    const int n_pairs = Ls * p.Hkv, n_rg = score_row_groups(p.Hkv, p.Hq, p.W);
    float* sal_rows = n_rg > 1 ? rows_ws + (size_t)n_pairs * n_rg * p.T : rows_ws;
    stepkv_status_t st = score_run(Ls, sal_keys(p), p.kv_head_stride, p.Q, p.q_head_stride, p.Hkv, p.Hq, p.d, p.T,
                                   p.W, rows_ws, p.T, nullptr, 0, part, dev_status, s, 0, p.sal_lse);
    if (st == STEPKV_OK && n_rg > 1) st = score_sum_row_groups(rows_ws, n_pairs, n_rg, p.T, sal_rows, s);
    if (st == STEPKV_OK)
      st = pool_mean_rows_run(sal_rows, n_pairs, p.T, 1.0f / (float)n_pairs, p.T, params->sal_pool / 2,
                              params->sal_pool_mode == STEPKV_POOL_MAX, t_float[i], s);
    if (st != STEPKV_OK) return st;
  }
  // stages 2-4 for all trajectories in one launch (one cluster per trajectory)
  stepkv_status_t st = select_run_batch(specs.data(), n_traj, s);
  if (st != STEPKV_OK) return st;
  if (ev.e[1]) {
    const cudaError_t er = cudaEventRecord(ev.e[1], s);  // the compaction is launched plainly after it
    if (er != cudaSuccess) { set_last_cuda_error(er); return STEPKV_ECUDA; }
  }
  // stage 5: in place by hole filling where the outputs are the inputs (one move launch per trajectory,
  // following the plan its selection wrote), the rest out of place, sharing launches
  std::vector<CompactSpec> outs;
  for (int i = 0; i < n_traj; ++i) {
    const stepkv_problem_t& p = probs[i];
    const CachePtrs& c = caches[i];
    if (in_place[i]) {
      st = compact_inplace_run(p.L, c.K_out.data(), c.V_out.data(), p.kv_head_stride, p.Hkv, p.d, p.T,
                               p.sel.kept_idx, p.sel.n_kept, p.sel.kept_cap, p.step_id, p.pos_in, p.step_id_out,
                               p.pos_out, plan_ws[i], dev_status, s);
      if (st != STEPKV_OK) return st;
      continue;
    }
    outs.push_back(CompactSpec{p.L, c.K.data(), c.V.data(), p.kv_head_stride, p.Hkv, p.d, p.T, p.sel.kept_idx,
                               p.sel.n_kept, p.sel.kept_cap, c.K_out.data(), c.V_out.data(), p.out_head_stride,
                               p.step_id, p.pos_in, p.step_id_out, p.pos_out});
  }
  if (!outs.empty()) {
    st = compact_run_batch(outs.data(), (int)outs.size(), dev_status, s);
    if (st != STEPKV_OK) return st;
  }
  if (ev.e[2]) {
    const cudaError_t er = cudaEventRecord(ev.e[2], s);
    if (er != cudaSuccess) { set_last_cuda_error(er); return STEPKV_ECUDA; }
  }
  return STEPKV_OK;
}

void stepkv_set_stage_events(void* before, void* after_select, void* after) {
  t_stage_events = StageEvents{{static_cast<cudaEvent_t>(before), static_cast<cudaEvent_t>(after_select),
                                static_cast<cudaEvent_t>(after)}};
}

}  // extern "C"
