// Stages 2-4 -- step reduction, score fusion and global top-B selection.
//   T_i   = mean of the saliency rows (layers x KV heads), normalised by its maximum over prunable
//           tokens (appendix "Combination with token-level importance": H_i in [0, H_max]);
//   r_k   = valid_k + gain_k - lambda red_k                                  (Eq. 2)
//   c_k  <- c_k + min(1, eta sim(Obs_t, Obs_k)) for k < t, c_t = 0            (Eq. 3, Alg. 1 Phases 1-2)
//   S_k   = clip(w_r clip(r_k, r_min, r_max) + w_c log(1 + c_k), 0, S_max)    (Eq. 4)
//   P_i   = alpha T_i + beta S_{s(i)}                                        (Eq. 5)
//   K     = top B_t prunable tokens by (P desc, index asc), B_t from Eq. 1   (Alg. 1 Phase 3)
//
// GB300 design: the tokens live in shared memory (saliency, then the order-preserving 32-bit key of P,
// and a 16-bit step id) -- in one 1024-thread CTA up to 2048 tokens, else in a cluster of 8 CTAs.
// The exact B-th largest key is found by three radix passes (11/11/10 bits) over warp-aggregated
// shared-memory histograms (summed across the cluster through distributed shared memory); retained
// slots are written in ascending order by warp ballot + prefix counts.  Per-step statistics use
// integer atomics only (fixed-point sums), so every output is bit-reproducible run to run.
#include <cooperative_groups.h>
#include <math.h>

#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace cg = cooperative_groups;

namespace stepkv {

// Two shapes of the same algorithm: one 1024-thread CTA for short trajectories (no cluster barriers),
// else a cluster of 8 CTAs of 512 threads whose histograms and counts meet through distributed shared
// memory.  Measured on GB300 at T = 32768: one CTA 78 us, 8-CTA cluster 31 us, 16-CTA cluster 35 us
// (the token loops shrink with more SMs, the cluster barriers and DSMEM gathers grow).
constexpr int kSelSingleMaxT = 2048;
constexpr int kSelClusterCtas = 8;

struct SelectArgs {
  const float* T_in;                  // token saliency as floats, or
  const unsigned long long* t_acc;    // as fixed-point sums: T_i = t_acc[i] * acc_to_T
  float acc_to_T;
  int T;
  int chunk;                          // tokens per CTA
  int s_in_smem;                      // S_k kept in shared memory (all CTAs compute all steps)
  const int32_t* step_id;
  const uint8_t* prot;
  stepkv_steps_t steps;
  stepkv_params_t prm;
  stepkv_budget_t budget;
  stepkv_select_out_t out;
  float* S;                           // [n_steps] step utilities (workspace)
  int32_t* acc_cnt;                   // [n_steps] workspace accumulators (zeroed here)
  unsigned long long* acc_sum;
  uint32_t* acc_max;
  int32_t* acc_kept;
  int32_t* status;
  // In-place compaction by hole filling (NULL plan: none).  The write pass also lays out the plan the move
  // kernel follows: plan[0] = number of holes H (slots below n_kept that are not retained), plan[1 + j] =
  // the j-th hole in slot order; the j-th mover is kept_idx[n_kept - H + j].  Rows retained in place get
  // their step id / position here; the move kernel writes those of the filled holes.
  int32_t* plan;
  const int32_t* pos_in;
  int32_t* step_id_out;
  int32_t* pos_out;
};

// Exchange block shared by the cluster (read remotely through DSMEM).
struct SelShared {
  float loc_max;
  int loc_N;
  int loc_err;
  int loc_keep_base;   // protected + strictly-greater count
  int loc_eq;          // ties at the threshold key
  int pad[3];
};

// Several independent trajectories in one launch: cluster (or CTA) c selects for trajectory c, so the
// latency-bound passes of different trajectories run side by side on different SMs.
constexpr int kMaxSelBatch = 16;
struct SelectBatch {
  SelectArgs t[kMaxSelBatch];
};
static_assert(sizeof(SelectBatch) <= 32000, "kernel parameter space");

// Inclusive suffix sum over the warp: lane l gets v[l] + v[l + 1] + ... + v[31].
__device__ __forceinline__ int warp_suffix_sum(int v, int lane) {
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_down_sync(0xffffffffu, v, o);
    if (lane + o < 32) v += y;
  }
  return v;
}

template <int NT>
__device__ __forceinline__ int block_reduce_sum_int(int v, int* scratch) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  __syncthreads();
  if (lane == 0) scratch[warp] = v;
  __syncthreads();
  int t = 0;
  for (int w = 0; w < NT / 32; ++w) t += scratch[w];
  return t;
}

template <int NT>
__device__ __forceinline__ float block_reduce_max(float v, float* scratch) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  __syncthreads();
  if (lane == 0) scratch[warp] = v;
  __syncthreads();
  float t = -INFINITY;
  for (int w = 0; w < NT / 32; ++w) t = fmaxf(t, scratch[w]);
  return t;
}

// In-place exclusive prefix of arr[0..n) with starting value `init` (block-wide, fixed order).
template <int NT>
__device__ __forceinline__ void block_scan_array(int* arr, int n, int init, int* scratch) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int per = (n + NT - 1) / NT;
  const int lo = min(n, (int)threadIdx.x * per), hi = min(n, lo + per);
  int mine = 0;
  for (int i = lo; i < hi; ++i) mine += arr[i];
  int x = mine;
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  __syncthreads();
  if (lane == 31) scratch[warp] = x;
  __syncthreads();
  int run = init + x - mine;
  for (int w = 0; w < warp; ++w) run += scratch[w];
  for (int i = lo; i < hi; ++i) {
    const int c = arr[i];
    arr[i] = run;
    run += c;
  }
  __syncthreads();
}

// One step-statistics contribution per warp when the warp's (consecutive) tokens share one step, else
// one per lane.  Integer atomics only: the totals do not depend on the order of arrival.
__device__ __forceinline__ void step_stat_add(bool act, int sid, unsigned long long fx, uint32_t mx_bits, int32_t* cnt,
                                              unsigned long long* sum, uint32_t* mx) {
  const unsigned am = __ballot_sync(0xffffffffu, act);
  if (!am) return;
  const int lane = threadIdx.x & 31;
  const int sid0 = __shfl_sync(0xffffffffu, sid, __ffs(am) - 1);
  if (__all_sync(0xffffffffu, !act || sid == sid0)) {
    unsigned long long v = act ? fx : 0ull;
    uint32_t m = act ? mx_bits : 0u;
    for (int o = 16; o > 0; o >>= 1) {
      v += __shfl_xor_sync(0xffffffffu, v, o);
      m = max(m, __shfl_xor_sync(0xffffffffu, m, o));
    }
    if (lane == 0) {
      atomicAdd(&cnt[sid0], __popc(am));
      if (sum) atomicAdd(&sum[sid0], v);
      if (mx) atomicMax(&mx[sid0], m);
    }
  } else if (act) {
    atomicAdd(&cnt[sid], 1);
    if (sum) atomicAdd(&sum[sid], fx);
    if (mx) atomicMax(&mx[sid], mx_bits);
  }
}

// Warp-wide flush of per-lane step statistics (lane: `act`, its step `sid`, count, fixed-point sum,
// max bits): one set of atomics per warp when every active lane holds the same step, else one per
// lane.  Integer atomics only, so the totals do not depend on the order of arrival.
__device__ __forceinline__ void step_stat_flush(bool act, int sid, int cnt_v, unsigned long long sum_v,
                                                uint32_t max_v, int32_t* cnt, unsigned long long* sum,
                                                uint32_t* mx) {
  const unsigned am = __ballot_sync(0xffffffffu, act);
  if (!am) return;
  const int lane = threadIdx.x & 31;
  const int sid0 = __shfl_sync(0xffffffffu, sid, __ffs(am) - 1);
  if (__all_sync(0xffffffffu, !act || sid == sid0)) {
    int c = act ? cnt_v : 0;
    unsigned long long v = act ? sum_v : 0ull;
    uint32_t m = act ? max_v : 0u;
    for (int o = 16; o > 0; o >>= 1) {
      c += __shfl_xor_sync(0xffffffffu, c, o);
      if (sum) v += __shfl_xor_sync(0xffffffffu, v, o);
      if (mx) m = max(m, __shfl_xor_sync(0xffffffffu, m, o));
    }
    if (lane == 0) {
      atomicAdd(&cnt[sid0], c);
      if (sum) atomicAdd(&sum[sid0], v);
      if (mx) atomicMax(&mx[sid0], m);
    }
  } else if (act) {
    atomicAdd(&cnt[sid], cnt_v);
    if (sum) atomicAdd(&sum[sid], sum_v);
    if (mx) atomicMax(&mx[sid], max_v);
  }
}

__device__ __forceinline__ float step_utility(const SelectArgs& a, int k, int t_last, float* c_out) {
  const stepkv_params_t& p = a.prm;
  const float r = a.steps.valid[k] + a.steps.gain[k] - p.lambda * a.steps.red[k];  // Eq. 2
  float c = 0.f;                                                                     // Alg. 1: c_t = 0
  if (k != t_last) {
    c = a.steps.reuse_in[k];
    if (a.steps.obs_sim) c += fminf(1.f, p.eta * a.steps.obs_sim[k]);              // Eq. 3
  }
  *c_out = c;
  const float rc = fminf(fmaxf(r, p.r_min), p.r_max);
  return fminf(fmaxf(p.w_r * rc + p.w_c * log1pf(c), 0.f), p.s_max);               // Eq. 4
}

template <int NC>
struct ClusterOps {
  cg::cluster_group cluster;
  __device__ ClusterOps() : cluster(cg::this_cluster()) {}
  __device__ int rank() const { return (int)cluster.block_rank(); }
  __device__ void sync() { cluster.sync(); }
  template <typename P>
  __device__ P* peer(P* p, int r) { return cluster.map_shared_rank(p, r); }
};
template <>
struct ClusterOps<1> {
  __device__ int rank() const { return 0; }
  __device__ void sync() { __syncthreads(); }
  template <typename P>
  __device__ P* peer(P* p, int) { return p; }
};

template <int NC, int NT>
__global__ void __launch_bounds__(NT, 1) select_kernel(const __grid_constant__ SelectBatch batch) {
  const SelectArgs& a = batch.t[blockIdx.x / NC];
  constexpr int NW = NT / 32;
  constexpr int UNROLL = NT >= 1024 ? 4 : 8;
  ClusterOps<NC> cl;
  const int rank = cl.rank();
  extern __shared__ __align__(16) uint8_t smem_raw[];
  // layout: [chunk] float/uint32 keys | [chunk] u16 step id (0xFFFF = protected) | 2 x 2048 int hist |
  //         SelShared (own) | SelShared[NC] (gathered) | scratch[64] | coarse[2][NC][64] | S_k (when s_in_smem)
  uint32_t* sKey = reinterpret_cast<uint32_t*>(smem_raw);
  float* sT = reinterpret_cast<float*>(smem_raw);
  uint16_t* sSid = reinterpret_cast<uint16_t*>(smem_raw + (size_t)a.chunk * 4);
  int* hist = reinterpret_cast<int*>(smem_raw + (((size_t)a.chunk * 6 + 15) & ~size_t(15)));
  SelShared* ex = reinterpret_cast<SelShared*>(hist + 2 * 2048);
  SelShared* all = ex + 1;
  int* scratch = reinterpret_cast<int*>(all + NC);  // 64 ints
  int* bcast = scratch + 48;                        // radix decision
  int* allc = scratch + 64;                         // [2 passes][NC ranks][64] every CTA's coarse counts
  float* sS = reinterpret_cast<float*>(allc + 2 * NC * 64);

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int T = a.T;
  const int n_steps = a.steps.n_steps;
  const int t_last = n_steps - 1;
  const int base = rank * a.chunk;
  const int len = max(0, min(a.chunk, T - base));
  const bool s_in_smem = a.s_in_smem != 0;
  // per-step statistics are outputs only (they do not enter P): skip them when none is requested
  const bool want_stats = a.out.step_count || a.out.step_sal_sum || a.out.step_sal_max;
  const bool want_kept = a.out.step_kept != nullptr;

  // Launched with programmatic dependent launch: everything up to pdl_wait() reads only the call's
  // inputs (step signals, step ids, mask) and writes only this kernel's workspace and outputs, so it
  // may overlap the tail of the kernel that produces the token saliency.
  pdl_launch_dependents();

  // ---- Phase 1+2 of Algorithm 1 (Eqs. 2-4).  With few steps every CTA keeps all S_k in shared memory
  // (CTA 0 publishes them); otherwise the steps are split over the CTAs through global memory.
  if (s_in_smem) {
    for (int k = tid; k < n_steps; k += NT) {
      float c;
      const float sk = step_utility(a, k, t_last, &c);
      sS[k] = sk;
      if (rank == 0) {
        a.S[k] = sk;
        if (a.out.step_util) a.out.step_util[k] = sk;
        // reuse_out may alias reuse_in, which every CTA reads here: written after barrier (A)
      }
    }
  } else {
    for (int k = rank * NT + tid; k < n_steps; k += NC * NT) {
      float c;
      const float sk = step_utility(a, k, t_last, &c);
      a.S[k] = sk;
      if (a.out.step_util) a.out.step_util[k] = sk;
      if (a.steps.reuse_out) a.steps.reuse_out[k] = c;
    }
  }
  if (a.plan && rank == 0 && tid == 0) a.plan[0] = 0;  // hole count, summed after barrier (B)
  for (int k = rank * NT + tid; k < n_steps; k += NC * NT) {
    a.acc_cnt[k] = 0;
    a.acc_sum[k] = 0ull;
    a.acc_max[k] = 0u;
    a.acc_kept[k] = 0;
  }

  // ---- this CTA's tokens: step ids / protection flags (inputs), then, once the producing kernel has
  // finished, token saliency T_i (loads batched)
  float lmax = -INFINITY;
  int lN = 0, lerr = 0;
  for (int i0 = 0; i0 < len; i0 += NT * UNROLL) {
    uint8_t pv[UNROLL];
    int sv[UNROLL];
#pragma unroll
    for (int u = 0; u < UNROLL; ++u) {
      const int i = i0 + u * NT + tid;
      if (i < len) {
        pv[u] = __ldg(&a.prot[base + i]);
        sv[u] = __ldg(&a.step_id[base + i]);
      }
    }
#pragma unroll
    for (int u = 0; u < UNROLL; ++u) {
      const int i = i0 + u * NT + tid;
      if (i < len) {
        if (!pv[u]) {
          ++lN;
          const bool bad = sv[u] < 0 || sv[u] >= n_steps;
          if (bad) lerr = 1;
          sSid[i] = bad ? 0 : (uint16_t)sv[u];
        } else {
          sSid[i] = 0xFFFFu;
        }
      }
    }
  }
  pdl_wait();  // t_acc / T_in come from the preceding kernel
  for (int i0 = 0; i0 < len; i0 += NT * UNROLL) {
    float tv[UNROLL];
#pragma unroll
    for (int u = 0; u < UNROLL; ++u) {
      const int i = i0 + u * NT + tid;
      if (i < len) {
        const int gi = base + i;
        tv[u] = a.t_acc ? __ull2float_rn(__ldcg(&a.t_acc[gi])) * a.acc_to_T : __ldcg(&a.T_in[gi]);
      }
    }
#pragma unroll
    for (int u = 0; u < UNROLL; ++u) {
      const int i = i0 + u * NT + tid;
      if (i < len) {
        sT[i] = tv[u];
        if (sSid[i] != 0xFFFFu) lmax = fmaxf(lmax, tv[u]);  // this thread wrote sSid[i] above
      }
    }
  }
  {
    // one block reduction for (max T, prunable count, error flag); the histogram area is free here
    for (int o = 16; o > 0; o >>= 1) {
      lmax = fmaxf(lmax, __shfl_xor_sync(0xffffffffu, lmax, o));
      lN += __shfl_xor_sync(0xffffffffu, lN, o);
      lerr |= __shfl_xor_sync(0xffffffffu, lerr, o);
    }
    float* red_max = reinterpret_cast<float*>(hist);
    int* red_n = hist + NW;
    int* red_e = hist + 2 * NW;
    if (lane == 0) {
      red_max[warp] = lmax;
      red_n[warp] = lN;
      red_e[warp] = lerr;
    }
    __syncthreads();
    if (tid == 0) {
      float bm = -INFINITY;
      int bn = 0, be = 0;
      for (int w = 0; w < NW; ++w) {
        bm = fmaxf(bm, red_max[w]);
        bn += red_n[w];
        be |= red_e[w];
      }
      ex->loc_max = bm;
      ex->loc_N = bn;
      ex->loc_err = be;
    }
  }
  cl.sync();  // (A) S_k, zeroed accumulators and per-CTA summaries visible to every CTA
  if (s_in_smem && rank == 0 && a.steps.reuse_out) {
    for (int k = tid; k < n_steps; k += NT) {
      float c;
      step_utility(a, k, t_last, &c);
      a.steps.reuse_out[k] = c;
    }
  }
  if (tid < NC) {
    const int4* rex = reinterpret_cast<const int4*>(cl.peer(ex, tid));
    const int4 v0 = rex[0], v1 = rex[1];
    reinterpret_cast<int4*>(&all[tid])[0] = v0;
    reinterpret_cast<int4*>(&all[tid])[1] = v1;
  }
  __syncthreads();
  float gmax = -INFINITY;
  int N = 0, err = 0;
  for (int r = 0; r < NC; ++r) {
    gmax = fmaxf(gmax, all[r].loc_max);
    N += all[r].loc_N;
    err += all[r].loc_err;
  }
  if (err) {
    if (rank == 0 && tid == 0) {
      record_status(a.status, STEPKV_EDATA);
      *a.out.n_kept = 0;
      if (a.out.n_budget) { a.out.n_budget[0] = N; a.out.n_budget[1] = 0; }
    }
    cl.sync();
    return;
  }
  // ---- budget (Eq. 1): B = max(1, floor(num N / den)) or a count, then |K| = min(B, N)
  int B = 0;
  if (N > 0) {
    if (a.budget.mode == STEPKV_BUDGET_RATIO)
      B = (int)max(1ll, ((long long)a.budget.ratio_num * N) / a.budget.ratio_den);
    else
      B = a.budget.count;
    B = min(B, N);
  }
  const bool norm = a.prm.sal_norm == STEPKV_NORM_MAX && gmax > 0.f && N > 0;
  const float inv_max = norm ? 1.0f / gmax : 1.0f;
  // fixed-point scale for per-step sums of normalised saliency: values <= vmax, at most N terms
  const float vmax = norm ? 1.0f : fmaxf(gmax, 1e-30f);
  int e_max;
  frexpf(vmax, &e_max);                       // vmax < 2^e_max
  const int log2N = 32 - __clz(max(N, 1));    // N < 2^log2N
  const int fx_shift = min(62 - log2N - e_max, 126);  // every partial sum < 2^62
  const float* Sk = s_in_smem ? sS : a.S;

  // Warp w owns the consecutive slots [w*seg, (w+1)*seg) of this CTA in the passes that need slot order
  // or per-step runs (keys and statistics, counts, ordered write); lanes take consecutive slots.
  const int seg = ((len + NW - 1) / NW + 31) & ~31;
  const int s0 = min(len, warp * seg), s1 = min(len, s0 + seg);

  // ---- priorities (Eq. 5), ordered keys and per-step statistics.  A lane accumulates its tokens'
  // statistics while their step does not change (slots of a step are mostly contiguous) and flushes
  // with integer atomics; T_hat is read before its shared-memory slot is overwritten by the key.
  {
    int run_sid = -1, run_c = 0;
    unsigned long long run_s = 0ull;
    uint32_t run_m = 0u;
    for (int i0 = s0; i0 < s1; i0 += 32) {
      const int i = i0 + lane;
      if (i >= s1) break;
      const int gi = base + i;
      const float th = sT[i] * inv_max;
      const int sid = sSid[i];
      uint32_t key = 0u;
      if (sid != 0xFFFF) {
        const float P = fmaf(a.prm.alpha, th, a.prm.beta * Sk[sid]);
        key = float_to_ordered(P);
        if (a.out.priority) a.out.priority[gi] = P;
        if (want_stats) {
          const float thc = fmaxf(th, 0.f);
          if (sid != run_sid) {
            if (run_c) {
              atomicAdd(&a.acc_cnt[run_sid], run_c);
              atomicAdd(&a.acc_sum[run_sid], run_s);
              atomicMax(&a.acc_max[run_sid], run_m);
            }
            run_sid = sid;
            run_c = 0;
            run_s = 0ull;
            run_m = 0u;
          }
          ++run_c;
          run_s += to_fixed(thc, fx_shift);
          run_m = max(run_m, __float_as_uint(thc));
        }
      } else if (a.out.priority) {
        a.out.priority[gi] = -INFINITY;
      }
      if (a.out.token_sal) a.out.token_sal[gi] = th;
      sKey[i] = key;
    }
    step_stat_flush(run_c > 0, run_sid, run_c, run_s, run_m, a.acc_cnt, a.acc_sum, a.acc_max);
  }
  __syncthreads();

  // ---- exact radix select of the B-th largest key among prunable tokens
  uint32_t kth = 0u;
  int need_eq = 0;
  if (B == 0) {
    kth = 0xFFFFFFFFu;
  } else if (B < N) {
    uint32_t prefix = 0u, mask = 0u;
    int remaining = B;
    for (int pass = 0; pass < 3; ++pass) {
      int* h = hist + (pass & 1) * 2048;
      const int nbits = pass < 2 ? 11 : 10;
      const int sh = pass == 0 ? 21 : (pass == 1 ? 10 : 0);
      const int nb = 1 << nbits;
      for (int b = tid; b < nb; b += NT) h[b] = 0;
      __syncthreads();
      // keys of one step share their leading bits, so many lanes hit the same bin: aggregate per warp
      for (int i0 = 0; i0 < len; i0 += NT) {
        const int i = i0 + tid;
        const uint32_t k = i < len ? sKey[i] : 0u;
        const bool hit = i < len && sSid[i] != 0xFFFF && (k & mask) == prefix;
        if (__ballot_sync(0xffffffffu, hit) == 0u) continue;  // after the first pass most keys miss the prefix
        const int bin = hit ? (int)((k >> sh) & (nb - 1)) : -1;
        const unsigned peers = __match_any_sync(0xffffffffu, bin);
        if (hit && (__ffs(peers) - 1) == lane) atomicAdd(&h[bin], __popc(peers));
      }
      __syncthreads();
      // this CTA's coarse counts: sums of 32 consecutive bins (64 coarse bins for 11 bits, 32 for 10),
      // pushed into every CTA's table before the barrier (lane r stores into rank r), so the coarse step
      // below reads them from its own shared memory
      int* ac = allc + (pass & 1) * NC * 64;
      const int ncoarse = nb >> 5;
      for (int c = warp; c < ncoarse; c += NW) {
        int v = h[c * 32 + lane];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
        if (lane < NC) cl.peer(ac, lane)[rank * 64 + c] = v;
      }
      cl.sync();  // every CTA's histogram and coarse counts of this pass are complete
      if (warp == 0) {
        // The digit in two small cluster-wide steps (keys in descending order): first the coarse bin that
        // holds the remaining-th largest key, then the bin within it.  Lane l holds coarse bins l and
        // 32 + l, then fine bin 32 * c* + l.
        int clo = 0, chi = 0;
#pragma unroll
        for (int r = 0; r < NC; ++r) {
          clo += ac[r * 64 + lane];
          if (ncoarse > 32) chi += ac[r * 64 + 32 + lane];
        }
        const int shi = warp_suffix_sum(chi, lane);                                    // keys in bins >= 32 + l
        const int slo = warp_suffix_sum(clo, lane) + __shfl_sync(0xffffffffu, shi, 0);  // keys in bins >= l
        const unsigned mhi = __ballot_sync(0xffffffffu, shi - chi < remaining && remaining <= shi);
        const unsigned mlo = __ballot_sync(0xffffffffu, slo - clo < remaining && remaining <= slo);
        const int lhi = __ffs(mhi) - 1, llo = __ffs(mlo) - 1;
        const int above_hi = __shfl_sync(0xffffffffu, shi - chi, lhi < 0 ? 0 : lhi);
        const int above_lo = __shfl_sync(0xffffffffu, slo - clo, llo < 0 ? 0 : llo);
        bool found = mhi != 0 || mlo != 0;
        const int cstar = mhi ? 32 + lhi : (mlo ? llo : 0);
        const int above_c = mhi ? above_hi : (mlo ? above_lo : 0);
        int f = 0;
#pragma unroll
        for (int r = 0; r < NC; ++r) f += cl.peer(h, r)[cstar * 32 + lane];
        const int sf = warp_suffix_sum(f, lane);
        const unsigned mf = __ballot_sync(0xffffffffu, above_c + sf - f < remaining && remaining <= above_c + sf);
        const int lf = __ffs(mf) - 1;
        found = found && mf != 0;
        const int above_f = __shfl_sync(0xffffffffu, above_c + sf - f, lf < 0 ? 0 : lf);
        if (lane == 0) {
          // the counts always hold the remaining-th key; the guard only keeps every index in range
          if (!found) record_status(a.status, STEPKV_EDATA);
          bcast[0] = found ? cstar * 32 + lf : 0;
          bcast[1] = found ? above_f : 0;
        }
      }
      __syncthreads();
      const int bstar = bcast[0];
      remaining -= bcast[1];
      prefix |= (uint32_t)bstar << sh;
      mask |= (uint32_t)(nb - 1) << sh;
      __syncthreads();
    }
    kth = prefix;
    need_eq = remaining;
  }
  // B == N: kth = 0 keeps every prunable token (all prunable keys are > 0)

  // ---- counts per warp segment: kept for sure (protected or strictly above the threshold) and ties
  int strict_w = 0, eq_w = 0;  // warp-uniform
  for (int i0 = s0; i0 < s1; i0 += 32) {
    const int i = i0 + lane;
    const bool in = i < s1;
    const uint32_t k = in ? sKey[i] : 0u;
    const bool pr = in && sSid[i] == 0xFFFF;
    strict_w += __popc(__ballot_sync(0xffffffffu, in && (pr || k > kth)));
    eq_w += __popc(__ballot_sync(0xffffffffu, in && !pr && k == kth));
  }
  // [NW] each, in the second radix pass's histogram buffer (hist + 2048): peers may still be reading the
  // last pass's buffer (hist[0..]) through DSMEM until barrier (B), but every CTA is done with this one
  int* seg_strict = hist + 2048;
  int* seg_eq = hist + 2048 + NW;
  if (lane == 0) {
    seg_strict[warp] = strict_w;
    seg_eq[warp] = eq_w;
  }
  __syncthreads();
  int strict_before = 0, eq_before = 0, strict_cta = 0, eq_cta = 0;  // exclusive prefixes over warps
  for (int w = 0; w < NW; ++w) {
    const int sw = seg_strict[w], ew = seg_eq[w];
    if (w < warp) {
      strict_before += sw;
      eq_before += ew;
    }
    strict_cta += sw;
    eq_cta += ew;
  }
  if (tid == 0) {
    ex->loc_keep_base = strict_cta;
    ex->loc_eq = eq_cta;
  }
  cl.sync();  // (B)
  if (tid < NC) {
    const int4* rex = reinterpret_cast<const int4*>(cl.peer(ex, tid));
    const int4 v0 = rex[0], v1 = rex[1];
    reinterpret_cast<int4*>(&all[tid])[0] = v0;
    reinterpret_cast<int4*>(&all[tid])[1] = v1;
  }
  __syncthreads();
  // offsets: CTA r keeps its protected + strictly-greater tokens and the ties that fall within the
  // first need_eq ties in slot order
  int out_off = 0, total_kept = 0, ties_before = 0, eq_cum = 0, granted_cta = 0;
  for (int r = 0; r < NC; ++r) {
    const int granted = max(0, min(need_eq - eq_cum, all[r].loc_eq));
    const int kept_r = all[r].loc_keep_base + granted;
    if (r < rank) {
      out_off += kept_r;
      ties_before += all[r].loc_eq;
    }
    if (r == rank) granted_cta = granted;
    total_kept += kept_r;
    eq_cum += all[r].loc_eq;
  }
  const bool overflow = total_kept > a.out.kept_cap;
  if (rank == 0 && tid == 0) {
    *a.out.n_kept = total_kept;
    if (a.out.n_budget) { a.out.n_budget[0] = N; a.out.n_budget[1] = B; }
    if (overflow) record_status(a.status, STEPKV_ENOSPACE);
  }

  // ---- ordered write of the retained slots: a warp walks its segment in slot order with running
  // counts (ballot + popc), starting from its segment's prefix within the CTA and the cluster.
  if (!overflow) {
    int tie_rank = ties_before + eq_before;                                 // cluster-wide tie rank
    int out_pos = out_off + strict_before + min(granted_cta, eq_before);   // next output slot
    int run_sid = -1, run_c = 0;
    int holes = 0;  // in-place plan: holes among this lane's slots
    for (int i0 = s0; i0 < s1; i0 += 32) {
      const int i = i0 + lane;
      const bool in = i < s1;
      const uint32_t k = in ? sKey[i] : 0u;
      const int sid = in ? sSid[i] : 0xFFFF;
      const bool pr = in && sid == 0xFFFF;
      const bool is_eq = in && !pr && k == kth;
      const unsigned lt = (1u << lane) - 1u;
      const unsigned em = __ballot_sync(0xffffffffu, is_eq);
      const bool keep = in && (pr || k > kth || (is_eq && tie_rank + __popc(em & lt) < need_eq));
      const unsigned km = __ballot_sync(0xffffffffu, keep);
      const int kept_before = out_pos + __popc(km & lt);  // retained slots below this one, cluster-wide
      if (keep) a.out.kept_idx[kept_before] = base + i;
      if (a.plan && in && base + i < total_kept) {
        const int gi = base + i;
        if (keep) {  // retained in place
          if (a.step_id_out) a.step_id_out[gi] = __ldg(&a.step_id[gi]);
          if (a.pos_out) a.pos_out[gi] = a.pos_in ? __ldg(&a.pos_in[gi]) : gi;
        } else {     // hole number gi - kept_before, filled by the mover of that number
          a.plan[1 + gi - kept_before] = gi;
          ++holes;
        }
      }
      out_pos += __popc(km);
      tie_rank += __popc(em);
      if (want_kept && keep && !pr) {
        if (sid != run_sid) {
          if (run_c) atomicAdd(&a.acc_kept[run_sid], run_c);
          run_sid = sid;
          run_c = 0;
        }
        ++run_c;
      }
    }
    step_stat_flush(run_c > 0, run_sid, run_c, 0ull, 0u, a.acc_kept, nullptr, nullptr);
    if (a.plan) {
      for (int o = 16; o > 0; o >>= 1) holes += __shfl_xor_sync(0xffffffffu, holes, o);
      if (lane == 0 && holes) atomicAdd(&a.plan[0], holes);
    }
  }
  if (want_stats || want_kept) {
    cl.sync();  // (C) all step accumulators final

    // ---- per-step outputs
    const double fx_unit = ldexp(1.0, -fx_shift);
    for (int k = rank * NT + tid; k < n_steps; k += NC * NT) {
      if (a.out.step_count) a.out.step_count[k] = a.acc_cnt[k];
      if (a.out.step_sal_sum) a.out.step_sal_sum[k] = (float)((double)a.acc_sum[k] * fx_unit);
      if (a.out.step_sal_max) a.out.step_sal_max[k] = __uint_as_float(a.acc_max[k]);
      if (a.out.step_kept) a.out.step_kept[k] = a.acc_kept[k];
    }
  }
  if (NC > 1) cl.sync();  // no CTA exits while another may still read its shared memory
}

// -------------------------------------------------------------------------------------------------
// T_out[j] = inv_div * sum over rows (fixed order): the token-saliency input of stepkv_select when the
// caller supplies per-(layer, head) saliency rows.  Four rows in flight per thread.
__global__ void mean_rows_kernel(const float* __restrict__ rows, int n_rows, int64_t row_stride, float inv_div, int T,
                                 float* __restrict__ T_out) {
  pdl_wait();
  pdl_launch_dependents();
  for (int j = blockIdx.x * blockDim.x + threadIdx.x; j < T; j += gridDim.x * blockDim.x) {
    float s = 0.f;
    int r = 0;
    for (; r + 4 <= n_rows; r += 4) {
      const float a0 = __ldg(&rows[(int64_t)r * row_stride + j]);
      const float a1 = __ldg(&rows[(int64_t)(r + 1) * row_stride + j]);
      const float a2 = __ldg(&rows[(int64_t)(r + 2) * row_stride + j]);
      const float a3 = __ldg(&rows[(int64_t)(r + 3) * row_stride + j]);
      s = (((s + a0) + a1) + a2) + a3;
    }
    for (; r < n_rows; ++r) s += __ldg(&rows[(int64_t)r * row_stride + j]);
    T_out[j] = s * inv_div;
  }
}

// SnapKV-style estimator (Sec. 4.2: T_i from an existing token-level estimator): each row pooled along the
// token axis over the window [j - h, j + h] clipped to [0, T) -- its maximum, or the mean of its in-range
// values -- then T_out[j] = inv_div * the sum over rows in row order.  A CTA takes 256 tokens and stages
// each row's 256 + 2h values (the tile and its halo) in shared memory, one row at a time.
constexpr int kPoolTile = 256;

template <bool IS_MAX>
__global__ void __launch_bounds__(kPoolTile) pool_mean_rows_kernel(const float* __restrict__ rows, int n_rows,
                                                                   int64_t row_stride, float inv_div, int T, int h,
                                                                   float* __restrict__ T_out) {
  extern __shared__ float tile[];  // [kPoolTile + 2h]
  pdl_wait();
  pdl_launch_dependents();
  const int j0 = blockIdx.x * kPoolTile, j = j0 + (int)threadIdx.x;
  const int span = kPoolTile + 2 * h;
  // this token's window as tile indices (tile index x holds token j0 - h + x)
  const int lo = max(0, j - h) - (j0 - h), hi = min(T - 1, j + h) - (j0 - h);
  float acc = 0.f;
  for (int r = 0; r < n_rows; ++r) {
    const float* row = rows + (int64_t)r * row_stride;
    __syncthreads();  // the previous row's tile has been read
    for (int x = (int)threadIdx.x; x < span; x += kPoolTile) {
      const int src = j0 - h + x;
      tile[x] = (src >= 0 && src < T) ? __ldg(row + src) : 0.f;
    }
    __syncthreads();
    if (j < T) {
      float v = tile[lo];
      for (int x = lo + 1; x <= hi; ++x) v = IS_MAX ? fmaxf(v, tile[x]) : v + tile[x];
      if (!IS_MAX) v = v / (float)(hi - lo + 1);
      acc += v;
    }
  }
  if (j < T) T_out[j] = acc * inv_div;
}

stepkv_status_t pool_mean_rows_run(const float* rows, int n_rows, int64_t row_stride, float inv_div, int T, int h,
                                   bool is_max, float* T_out, cudaStream_t stream) {
  const int blocks = (T + kPoolTile - 1) / kPoolTile;
  const size_t smem = (size_t)(kPoolTile + 2 * h) * sizeof(float);
  const cudaError_t e =
      is_max ? launch_kernel(pool_mean_rows_kernel<true>, dim3(blocks), dim3(kPoolTile), smem, stream, rows, n_rows,
                             row_stride, inv_div, T, h, T_out)
             : launch_kernel(pool_mean_rows_kernel<false>, dim3(blocks), dim3(kPoolTile), smem, stream, rows, n_rows,
                             row_stride, inv_div, T, h, T_out);
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return STEPKV_ECUDA;
  }
  return STEPKV_OK;
}

stepkv_status_t mean_rows_run(const float* rows, int n_rows, int64_t row_stride, float inv_div, int T, float* T_out,
                              cudaStream_t stream) {
  const int blocks = std::max(1, std::min((T + 255) / 256, 4096));
  cudaError_t e = launch_kernel(mean_rows_kernel, dim3(blocks), dim3(256), 0, stream, rows, n_rows, row_stride, inv_div,
                             T, T_out);
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return STEPKV_ECUDA;
  }
  return STEPKV_OK;
}

static size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

size_t select_ws_bytes(int T, int n_steps) {
  (void)T;
  const size_t n = (size_t)std::max(n_steps, 1);
  return align256(n * 4) + align256(n * 4) + align256(n * 8) + align256(n * 4) + align256(n * 4);
}

static SelectArgs make_select_args(const SelectSpec& sp) {
  SelectArgs a;
  memset(&a, 0, sizeof(a));
  a.T_in = sp.T_in;
  a.t_acc = sp.t_acc;
  a.acc_to_T = (float)sp.acc_to_T;
  a.T = sp.T;
  a.step_id = sp.step_id;
  a.prot = sp.prot;
  a.steps = sp.steps;
  a.prm = sp.params;
  a.budget = sp.budget;
  a.out = sp.out;
  const size_t n = (size_t)std::max(sp.steps.n_steps, 1);
  uint8_t* w = static_cast<uint8_t*>(sp.ws);
  a.S = reinterpret_cast<float*>(w);
  w += align256(n * 4);
  a.acc_cnt = reinterpret_cast<int32_t*>(w);
  w += align256(n * 4);
  a.acc_sum = reinterpret_cast<unsigned long long*>(w);
  w += align256(n * 8);
  a.acc_max = reinterpret_cast<uint32_t*>(w);
  w += align256(n * 4);
  a.acc_kept = reinterpret_cast<int32_t*>(w);
  a.status = sp.status;
  a.plan = sp.plan;
  a.pos_in = sp.pos_in;
  a.step_id_out = sp.step_id_out;
  a.pos_out = sp.pos_out;
  return a;
}

// Shared memory of one trajectory's CTA: keys + step ids of its chunk, histograms, exchange blocks,
// scratch, and S_k when it fits.
static size_t select_smem(int chunk, int nc, int n_steps, int* s_in_smem) {
  const size_t fixed = (((size_t)chunk * 6 + 15) & ~size_t(15)) + 2 * 2048 * 4 + (1 + nc) * sizeof(SelShared) +
                       (64 + 2 * (size_t)nc * 64) * 4;
  const size_t budget_smem = 232448 - 1024;
  *s_in_smem = fixed + (size_t)n_steps * 4 <= budget_smem ? 1 : 0;
  return fixed + (*s_in_smem ? (size_t)n_steps * 4 : 0);
}

stepkv_status_t select_run_batch(const SelectSpec* specs, int n, cudaStream_t stream) {
  for (int b0 = 0; b0 < n; b0 += kMaxSelBatch) {
    const int nb = std::min(kMaxSelBatch, n - b0);
    int T_max = 0;
    for (int i = 0; i < nb; ++i) T_max = std::max(T_max, specs[b0 + i].T);
    const int nc = T_max <= kSelSingleMaxT ? 1 : kSelClusterCtas;
    SelectBatch batch;
    memset(&batch, 0, sizeof(batch));
    size_t smem = 0;
    for (int i = 0; i < nb; ++i) {
      SelectArgs a = make_select_args(specs[b0 + i]);
      a.chunk = ((a.T + nc - 1) / nc + 15) & ~15;
      smem = std::max(smem, select_smem(a.chunk, nc, a.steps.n_steps, &a.s_in_smem));
      batch.t[i] = a;
    }
    cudaError_t e;
    if (nc == 1) {
      void (*kern)(SelectBatch) = select_kernel<1, 1024>;
      e = ensure_smem_attr(reinterpret_cast<const void*>(kern), (int)smem);
      if (e == cudaSuccess) e = launch_kernel(kern, dim3(nb), dim3(1024), smem, stream, batch, true);
    } else {
      void (*kern)(SelectBatch) = select_kernel<kSelClusterCtas, 512>;
      e = ensure_smem_attr(reinterpret_cast<const void*>(kern), (int)smem);
      if (e == cudaSuccess)
        e = launch_cluster(kern, dim3(kSelClusterCtas * nb), dim3(512), kSelClusterCtas, smem, stream, batch, true);
    }
    if (e != cudaSuccess) {
      set_last_cuda_error(e);
      return STEPKV_ECUDA;
    }
  }
  return STEPKV_OK;
}

stepkv_status_t select_run(const float* T_in, const unsigned long long* t_acc, double acc_to_T, int T,
                           const int32_t* step_id, const uint8_t* prot, const stepkv_steps_t& steps,
                           const stepkv_params_t& params, const stepkv_budget_t& budget,
                           const stepkv_select_out_t& out, void* ws, int32_t* status, cudaStream_t stream) {
  const SelectSpec sp{T_in, t_acc, acc_to_T, T, step_id, prot, steps, params, budget, out, ws, status};
  return select_run_batch(&sp, 1, stream);
}

}  // namespace stepkv
