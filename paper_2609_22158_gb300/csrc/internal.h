// Host-side internals shared by the StepKV translation units (not part of the C ABI).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>
#include <string.h>

#include <utility>

#include "../../include/stepkv.h"

namespace stepkv {

constexpr int kMaxSalLayers = 8;        // saliency layers per score launch (tensor maps in kernel params)
constexpr int kMaxScoreBatch = 16;      // trajectories per saliency launch
constexpr int kMaxScoreMaps = 48;       // trajectories x saliency layers per saliency launch
constexpr int kMaxGrid = 1024;          // upper bound on the persistent score grid (partial-slot sizing)
constexpr int kMaxCompactLayers = 256;  // layers per compaction launch (pointer tables in kernel params)

void set_last_cuda_error(cudaError_t e);
cudaError_t device_sm_count(int* n);
cudaError_t ensure_smem_attr(const void* func, int bytes);

// Kernel launch on `stream`.  Ordinary stream order unless `pdl` is set: then the launch carries the
// programmatic-stream-serialization attribute, so the kernel may start while the preceding kernel
// finishes and must execute griddepcontrol.wait (pdl_wait) before reading anything that kernel wrote.
// Only the selection kernel uses it.  Measured on GB300 with the 32K workload, the compaction kernel
// ran ~25% slower when launched with the attribute (178 us vs 140 us), so it is launched plainly.
// Every kernel executes griddepcontrol.launch_dependents, a no-op when the next launch is ordinary.
template <typename... KArgs, typename... Args>
cudaError_t launch_kernel(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                          Args&&... args) {
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof(cfg));
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cfg.attrs = nullptr;
  cfg.numAttrs = 0;
  return cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...);
}

template <typename... KArgs, typename A0>
cudaError_t launch_kernel(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream, A0&& a0,
                          bool pdl) {
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof(cfg));
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, std::forward<A0>(a0));
}

template <typename... KArgs, typename A0>
cudaError_t launch_cluster(void (*kern)(KArgs...), dim3 grid, dim3 block, int cluster_x, size_t smem,
                           cudaStream_t stream, A0&& a0, bool pdl = false) {
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof(cfg));
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = cluster_x;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kern, std::forward<A0>(a0));
}

// ---- decode attention (decode.cu)
constexpr int kMaxDecodeLayers = 64;  // layers per launch (pointer arrays travel in the kernel parameters)
size_t decode_ws_bytes(int n_layers, int Hkv, int Hq, int d, int n_cap);
size_t decode_mass_ws_bytes(int n_layers, int Hkv, int Hq, int d, int n_cap);
// With mass (per layer [Hkv][mass_stride] fp32), each call also adds every key's group-mean softmax mass.
stepkv_status_t decode_run(int n_layers, const void* const* q, const void* const* K, const void* const* V,
                           int64_t head_stride, int Hkv, int Hq, int d, const int32_t* n_dev, int n_host, int n_cap,
                           float* const* out, void* ws, int32_t* status, cudaStream_t stream,
                           float* const* mass = nullptr, int64_t mass_stride = 0);

// ---- step signals from evidence cues (signals.cu)
stepkv_status_t signals_run(const uint32_t* cues, const int32_t* n_cues, int n_steps, int k0, float* gain, float* red,
                            float* obs_sim, int32_t* status, cudaStream_t stream);

// ---- score (score.cu)
int score_row_groups(int Hkv, int Hq, int W);
size_t score_partial_bytes(int n_layers, int Hkv, int Hq, int W, int n_traj = 1);
int score_acc_shift(int n_pairs, int W);
// Pass 2 either writes rows (row pair*n_rg + rg of rows_out, stride out_stride, pair = layer*Hkv + h) or,
// when t_acc is non-null, adds every contribution to the per-token fixed-point sum t_acc[T] (scale
// 2^acc_shift; the first launch zeroes it).
// One trajectory of a batched saliency launch (per-layer device pointers, tokens, accumulator).
struct ScoreTrajSpec {
  const void* const* K;
  const void* const* Q;
  int T;
  unsigned long long* t_acc;
  int64_t k_head_stride, q_head_stride;
  const float* const* lse = nullptr;  // per layer [Hq][W] natural-log row log-sum-exp (skips pass 1), or NULL
};
// Saliency of n_traj trajectories of one head shape in one cooperative launch (n_traj <= kMaxScoreBatch,
// n_traj * n_layers <= kMaxScoreMaps); rows output only for n_traj == 1.
stepkv_status_t score_run_batch(int n_layers, const ScoreTrajSpec* trajs, int n_traj, int Hkv, int Hq, int d,
                                int W, float* rows_out,
                                int64_t out_stride, int acc_shift, float2* part, int32_t* status, cudaStream_t stream,
                                unsigned long long selftest_wait_ns = 0);
stepkv_status_t score_run(int n_layers, const void* const* K, int64_t k_head_stride, const void* const* Q,
                          int64_t q_head_stride, int Hkv, int Hq, int d, int T, int W, float* rows_out,
                          int64_t out_stride, unsigned long long* t_acc, int acc_shift, float2* part, int32_t* status,
                          cudaStream_t stream, unsigned long long selftest_wait_ns = 0,
                          const float* const* lse = nullptr);
stepkv_status_t score_sum_row_groups(const float* rows, int n_pairs, int n_rg, int T, float* sal, cudaStream_t stream);

// ---- select (select.cu)
size_t select_ws_bytes(int T, int n_steps);
// Token saliency comes either as floats T_in[T] or as fixed-point sums t_acc[T] with T_i = t_acc * acc_to_T.
struct SelectSpec {
  const float* T_in;
  const unsigned long long* t_acc;
  double acc_to_T;
  int T;
  const int32_t* step_id;
  const uint8_t* prot;
  stepkv_steps_t steps;
  stepkv_params_t params;
  stepkv_budget_t budget;
  stepkv_select_out_t out;
  void* ws;          // select_ws_bytes(T, n_steps), 256-byte aligned, private to this trajectory
  int32_t* status;
  // in-place compaction: the selection also writes the hole-filling plan (compact_inplace_ws_bytes(T))
  // and the step id / position of the rows retained in place
  int32_t* plan = nullptr;
  const int32_t* pos_in = nullptr;
  int32_t* step_id_out = nullptr;
  int32_t* pos_out = nullptr;
};
// Independent trajectories in as few launches as possible (one cluster each).
stepkv_status_t select_run_batch(const SelectSpec* specs, int n, cudaStream_t stream);
stepkv_status_t select_run(const float* T_in, const unsigned long long* t_acc, double acc_to_T, int T,
                           const int32_t* step_id, const uint8_t* prot, const stepkv_steps_t& steps,
                           const stepkv_params_t& params, const stepkv_budget_t& budget,
                           const stepkv_select_out_t& out, void* ws, int32_t* status, cudaStream_t stream);
// T_out[j] = inv_div * sum_r rows[r * row_stride + j] (fixed order over r).
stepkv_status_t mean_rows_run(const float* rows, int n_rows, int64_t row_stride, float inv_div, int T, float* T_out,
                              cudaStream_t stream);
// The same mean after a token-axis pooling of each row over [j - h, j + h] clipped to [0, T): the
// maximum (is_max) or the mean of the in-range values.
stepkv_status_t pool_mean_rows_run(const float* rows, int n_rows, int64_t row_stride, float inv_div, int T, int h,
                                   bool is_max, float* T_out, cudaStream_t stream);

// ---- compact (compact.cu)
// One out-of-place compaction (as stepkv_compact's arguments).
struct CompactSpec {
  int n_layers;
  const void* const* K_in;
  const void* const* V_in;
  int64_t in_head_stride;
  int Hkv, d, T;
  const int32_t* kept_idx;
  const int32_t* n_kept;
  int kept_cap;
  void* const* K_out;
  void* const* V_out;
  int64_t out_head_stride;
  const int32_t* step_id_in;
  const int32_t* pos_in;
  int32_t* step_id_out;
  int32_t* pos_out;
};
// Several compactions, sharing launches where they fit.
stepkv_status_t compact_run_batch(const CompactSpec* specs, int n, int32_t* status, cudaStream_t stream);
stepkv_status_t compact_run(int n_layers, const void* const* K_in, const void* const* V_in, int64_t in_head_stride,
                            int Hkv, int d, int T, const int32_t* kept_idx, const int32_t* n_kept, int kept_cap,
                            void* const* K_out, void* const* V_out, int64_t out_head_stride,
                            const int32_t* step_id_in, const int32_t* pos_in, int32_t* step_id_out,
                            int32_t* pos_out, int32_t* status, cudaStream_t stream);

// In place (K_out == K): hole filling, following the plan the selection kernel wrote into ws
// (compact_inplace_ws_bytes(T), SelectSpec::plan); the move kernel also writes the step id / position of
// every filled hole.
size_t compact_inplace_ws_bytes(int T);
stepkv_status_t compact_inplace_run(int n_layers, void* const* K, void* const* V, int64_t head_stride, int Hkv, int d,
                                    int T, const int32_t* kept_idx, const int32_t* n_kept, int kept_cap,
                                    const int32_t* step_id_in, const int32_t* pos_in, int32_t* step_id_out,
                                    int32_t* pos_out, void* ws, int32_t* status, cudaStream_t stream);

}  // namespace stepkv
