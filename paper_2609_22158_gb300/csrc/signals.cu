// Step signals from evidence cues (Sec. 4.1 "New-step Scoring" and "Previous-step Updating"): each step's
// Thought, Action and Observation fields are represented by up to 64 evidence cues (sorted, distinct
// 32-bit ids), and sim(a, b) is the overlap similarity of two cue sets, |A n B| / |A u B| (0 when both
// are empty).  For every target step k in [k0, n_steps):
//   gain_k = 1 - max_{u<k} sim(Th_k || Obs_k, Th_u || Obs_u)   (gain = 1 for the first step)
//   red_k  = max_{u<k} sim(Act_k, Act_u)                        (red = 0 for the first step)
// where a concatenation of fields is the union of their cues; and for the newest step t = n_steps - 1
//   obs_sim[k] = sim(Obs_t, Obs_k), k < t                      (Eq. 3's input; obs_sim[t] = 0).
//
// The work is O(t x 128) comparisons per target step: one CTA per target step (plus one for obs_sim),
// eight warps over the earlier steps, every set-membership test a binary search in a sorted cue list, and
// the maxima reduced in a fixed order (deterministic).  A count outside [0, 64] or a cue list that is not
// strictly increasing sets STEPKV_EDATA and the values that depend on it are not written.
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace stepkv {

constexpr int kSigThreads = 256;
constexpr int kSigWarps = kSigThreads / 32;

struct SignalArgs {
  const uint32_t* cues;  // [n_steps][3][STEPKV_MAX_CUES]
  const int32_t* n_cues; // [n_steps][3]
  int n_steps;
  int k0;
  float* gain;           // [n_steps] (entries k >= k0 written) or NULL
  float* red;
  float* obs_sim;        // [n_steps] or NULL
  int32_t* status;
};

__device__ __forceinline__ const uint32_t* field(const SignalArgs& a, int k, int f) {
  return a.cues + ((size_t)k * 3 + f) * STEPKV_MAX_CUES;
}
__device__ __forceinline__ int field_n(const SignalArgs& a, int k, int f) {
  const int n = a.n_cues[k * 3 + f];
  return n < 0 ? 0 : (n > STEPKV_MAX_CUES ? STEPKV_MAX_CUES : n);
}

// true when x is in the sorted list p[0..n)
__device__ __forceinline__ bool contains(const uint32_t* p, int n, uint32_t x) {
  int lo = 0, hi = n;
  while (lo < hi) {
    const int mid = (lo + hi) >> 1;
    const uint32_t v = __ldg(p + mid);
    if (v < x) lo = mid + 1;
    else hi = mid;
  }
  return lo < n && __ldg(p + lo) == x;
}

// Warp-wide: number of distinct cues of A1 u A2 that lie in B1 u B2, and |A1 u A2| (B2 / A2 may be empty).
__device__ __forceinline__ void union_overlap(const uint32_t* a1, int na1, const uint32_t* a2, int na2,
                                              const uint32_t* b1, int nb1, const uint32_t* b2, int nb2,
                                              int lane, int& inter, int& size) {
  int ci = 0, cs = 0;
  for (int i = lane; i < na1 + na2; i += 32) {
    const bool first = i < na1;
    const uint32_t x = first ? __ldg(a1 + i) : __ldg(a2 + i - na1);
    if (!first && contains(a1, na1, x)) continue;  // already counted as a cue of the first field
    ++cs;
    if (contains(b1, nb1, x) || contains(b2, nb2, x)) ++ci;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    ci += __shfl_xor_sync(0xffffffffu, ci, o);
    cs += __shfl_xor_sync(0xffffffffu, cs, o);
  }
  inter = ci;
  size = cs;
}

__device__ __forceinline__ float jaccard(int inter, int na, int nb) {
  const int uni = na + nb - inter;
  return uni > 0 ? (float)inter / (float)uni : 0.f;
}

// Every field's count must lie in [0, 64] and its cue list be strictly increasing (sorted, distinct).
__device__ bool lists_ok(const SignalArgs& a, int k, int lane) {
  bool ok = true;
  for (int f = 0; f < 3; ++f) {
    const int raw = a.n_cues[k * 3 + f];
    ok &= raw >= 0 && raw <= STEPKV_MAX_CUES;
    const uint32_t* p = field(a, k, f);
    const int n = field_n(a, k, f);
    for (int i = lane + 1; i < n; i += 32) ok &= __ldg(p + i - 1) < __ldg(p + i);
  }
  return __all_sync(0xffffffffu, ok);
}

__global__ void __launch_bounds__(kSigThreads) step_signals_kernel(const __grid_constant__ SignalArgs a) {
  __shared__ float s_g[kSigWarps], s_r[kSigWarps];
  __shared__ int s_bad;
  pdl_wait();
  pdl_launch_dependents();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_targets = a.n_steps - a.k0;
  if (threadIdx.x == 0) s_bad = 0;
  __syncthreads();
  if ((int)blockIdx.x < n_targets) {
    // ---- gain / red of target step k against every earlier step
    const int k = a.k0 + blockIdx.x;
    if (warp == 0 && !lists_ok(a, k, lane) && lane == 0) s_bad = 1;
    const uint32_t *th = field(a, k, 0), *ac = field(a, k, 1), *ob = field(a, k, 2);
    const int nth = field_n(a, k, 0), nac = field_n(a, k, 1), nob = field_n(a, k, 2);
    float best_g = 0.f, best_r = 0.f;
    for (int u = warp; u < k; u += kSigWarps) {
      if (!lists_ok(a, u, lane)) {
        if (lane == 0) s_bad = 1;
        continue;
      }
      const uint32_t *th2 = field(a, u, 0), *ac2 = field(a, u, 1), *ob2 = field(a, u, 2);
      const int nth2 = field_n(a, u, 0), nac2 = field_n(a, u, 1), nob2 = field_n(a, u, 2);
      int inter, sa, unused, sb;
      union_overlap(th, nth, ob, nob, th2, nth2, ob2, nob2, lane, inter, sa);  // |X n Y|, |X|
      union_overlap(th2, nth2, ob2, nob2, th2, 0, ob2, 0, lane, unused, sb);   // |Y|
      best_g = fmaxf(best_g, jaccard(inter, sa, sb));
      int ia, na;
      union_overlap(ac, nac, ac, 0, ac2, nac2, ac2, 0, lane, ia, na);          // |Act_k n Act_u|
      best_r = fmaxf(best_r, jaccard(ia, na, nac2));
    }
    if (lane == 0) {
      s_g[warp] = best_g;
      s_r[warp] = best_r;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      float g = 0.f, r = 0.f;
      for (int w = 0; w < kSigWarps; ++w) {
        g = fmaxf(g, s_g[w]);
        r = fmaxf(r, s_r[w]);
      }
      if (s_bad) {
        record_status(a.status, STEPKV_EDATA);
      } else {
        if (a.gain) a.gain[k] = 1.f - g;
        if (a.red) a.red[k] = r;
      }
    }
  } else {
    // ---- obs_sim of the newest step t against every earlier step
    const int t = a.n_steps - 1;
    if (warp == 0 && !lists_ok(a, t, lane) && lane == 0) s_bad = 1;
    const uint32_t* ob = field(a, t, 2);
    const int nob = field_n(a, t, 2);
    for (int k = warp; k < t; k += kSigWarps) {
      const uint32_t* ob2 = field(a, k, 2);
      const int nob2 = field_n(a, k, 2);
      if (!lists_ok(a, k, lane)) {
        if (lane == 0) s_bad = 1;
        continue;
      }
      int inter, na;
      union_overlap(ob, nob, ob, 0, ob2, nob2, ob2, 0, lane, inter, na);
      if (lane == 0) a.obs_sim[k] = jaccard(inter, na, nob2);
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      if (s_bad) record_status(a.status, STEPKV_EDATA);
      a.obs_sim[t] = 0.f;
    }
  }
}

stepkv_status_t signals_run(const uint32_t* cues, const int32_t* n_cues, int n_steps, int k0, float* gain, float* red,
                            float* obs_sim, int32_t* status, cudaStream_t stream) {
  SignalArgs a;
  memset(&a, 0, sizeof(a));
  a.cues = cues;
  a.n_cues = n_cues;
  a.n_steps = n_steps;
  a.k0 = k0;
  a.gain = gain;
  a.red = red;
  a.obs_sim = obs_sim;
  a.status = status;
  const int blocks = (n_steps - k0) + (obs_sim != nullptr ? 1 : 0);
  if (blocks == 0) return STEPKV_OK;
  const cudaError_t e = launch_kernel(step_signals_kernel, dim3(blocks), dim3(kSigThreads), 0, stream, a);
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return STEPKV_ECUDA;
  }
  return STEPKV_OK;
}

}  // namespace stepkv
