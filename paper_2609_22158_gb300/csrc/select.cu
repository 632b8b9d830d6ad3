// Stages 2-4 -- step reduction, score fusion and global top-B selection.
//   T_i   = mean of the saliency rows (layers x KV heads), normalised by its maximum over prunable
//           tokens (appendix "Combination with token-level importance": H_i in [0, H_max]);
//   r_k   = valid_k + gain_k - lambda red_k                                  (Eq. 2)
//   c_k  <- c_k + min(1, eta sim(Obs_t, Obs_k)) for k < t, c_t = 0            (Eq. 3, Alg. 1 Phases 1-2)
//   S_k   = clip(w_r clip(r_k, r_min, r_max) + w_c log(1 + c_k), 0, S_max)    (Eq. 4)
//   P_i   = alpha T_i + beta S_{s(i)}                                        (Eq. 5)
//   K     = top B_t prunable tokens by (P desc, index asc), B_t from Eq. 1   (Alg. 1 Phase 3)
//
// GB300 design: one thread-block cluster of 8 CTAs per trajectory.  Each CTA keeps its slice of the
// tokens in shared memory (saliency, then the order-preserving 32-bit key of P); the exact B-th
// largest key is found by three radix passes (11/11/10 bits) whose per-CTA shared-memory histograms
// are summed across the cluster through distributed shared memory; retained slots are written in
// ascending order by warp ballot + prefix counts.  Per-step statistics use integer atomics only
// (fixed-point sums), so every output is bit-reproducible run to run.
#include <cooperative_groups.h>
#include <math.h>

#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace cg = cooperative_groups;

namespace stepkv {

constexpr int kSelCluster = 8;
constexpr int kSelThreads = 512;
constexpr int kSelWarps = kSelThreads / 32;
constexpr int kSelMaxChunk = 32768;  // tokens per CTA held in shared memory (T <= 262144)

struct SelectArgs {
  const float* rows;
  int n_rows;
  int64_t row_stride;
  float inv_div;
  int T;
  int chunk;  // tokens per CTA
  const int32_t* step_id;
  const uint8_t* prot;
  stepkv_steps_t steps;
  stepkv_params_t prm;
  stepkv_budget_t budget;
  stepkv_select_out_t out;
  float* S;                  // [n_steps] step utilities (ws or out.step_util)
  int32_t* acc_cnt;          // [n_steps] ws accumulators (zeroed here)
  unsigned long long* acc_sum;
  uint32_t* acc_max;
  int32_t* acc_kept;
  int32_t* status;
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

__device__ __forceinline__ int block_reduce_sum_int(int v, int* scratch) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  __syncthreads();
  if (lane == 0) scratch[warp] = v;
  __syncthreads();
  int t = 0;
  for (int w = 0; w < kSelWarps; ++w) t += scratch[w];
  return t;
}

__device__ __forceinline__ float block_reduce_max(float v, float* scratch) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  __syncthreads();
  if (lane == 0) scratch[warp] = v;
  __syncthreads();
  float t = -INFINITY;
  for (int w = 0; w < kSelWarps; ++w) t = fmaxf(t, scratch[w]);
  return t;
}

// Exclusive prefix over the block of per-thread counts (thread order); returns the block total.
__device__ __forceinline__ int block_excl_scan(int v, int* excl, int* scratch) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  __syncthreads();
  if (lane == 31) scratch[warp] = x;
  __syncthreads();
  int before = 0, total = 0;
  for (int w = 0; w < kSelWarps; ++w) {
    if (w < warp) before += scratch[w];
    total += scratch[w];
  }
  *excl = before + x - v;
  return total;
}

__global__ void __launch_bounds__(kSelThreads, 1)
    select_kernel(const SelectArgs a) {
  cg::cluster_group cluster = cg::this_cluster();
  const int rank = (int)cluster.block_rank();
  extern __shared__ uint8_t smem_raw[];
  // layout: [chunk] float/uint32 keys | [chunk] u8 flags | 2 x 2048 int hist | SelShared | scratch
  uint32_t* sKey = reinterpret_cast<uint32_t*>(smem_raw);
  float* sT = reinterpret_cast<float*>(smem_raw);
  uint8_t* sProt = smem_raw + (size_t)a.chunk * 4;
  int* hist = reinterpret_cast<int*>(smem_raw + (((size_t)a.chunk * 5 + 15) & ~size_t(15)));
  SelShared* ex = reinterpret_cast<SelShared*>(hist + 2 * 2048);
  int* scratch = reinterpret_cast<int*>(ex + 1);   // kSelWarps ints
  int* bcast = scratch + kSelWarps;                  // 4 ints

  const int tid = threadIdx.x;
  const int T = a.T;
  const int n_steps = a.steps.n_steps;
  const int t_last = n_steps - 1;
  const int base = rank * a.chunk;
  const int len = max(0, min(a.chunk, T - base));

  pdl_wait();
  pdl_launch_dependents();

  // ---- Phase 1+2 of Algorithm 1 (Eqs. 2-4), steps distributed over the cluster; zero accumulators.
  for (int k = rank * kSelThreads + tid; k < n_steps; k += kSelCluster * kSelThreads) {
    const stepkv_params_t& p = a.prm;
    const float r = a.steps.valid[k] + a.steps.gain[k] - p.lambda * a.steps.red[k];
    float c = 0.f;
    if (k != t_last) {
      c = a.steps.reuse_in[k];
      if (a.steps.obs_sim) c += fminf(1.f, p.eta * a.steps.obs_sim[k]);
    }
    const float rc = fminf(fmaxf(r, p.r_min), p.r_max);
    const float s = fminf(fmaxf(p.w_r * rc + p.w_c * log1pf(c), 0.f), p.s_max);
    a.S[k] = s;
    if (a.out.step_util && a.out.step_util != a.S) a.out.step_util[k] = s;
    if (a.steps.reuse_out) a.steps.reuse_out[k] = c;
    a.acc_cnt[k] = 0;
    a.acc_sum[k] = 0ull;
    a.acc_max[k] = 0u;
    a.acc_kept[k] = 0;
  }

  // ---- token saliency T_i (fixed-order sum over rows), prunable max and count, step-id check
  float lmax = -INFINITY;
  int lN = 0, lerr = 0;
  for (int i = tid; i < len; i += kSelThreads) {
    const int gi = base + i;
    float s = 0.f;
    for (int r = 0; r < a.n_rows; ++r) s += __ldg(&a.rows[(int64_t)r * a.row_stride + gi]);
    s *= a.inv_div;
    sT[i] = s;
    const uint8_t pr = a.prot[gi] ? 1 : 0;
    sProt[i] = pr;
    if (!pr) {
      ++lN;
      lmax = fmaxf(lmax, s);
      const int sid = a.step_id[gi];
      if (sid < 0 || sid >= n_steps) lerr = 1;
    }
  }
  {
    const float bm = block_reduce_max(lmax, reinterpret_cast<float*>(scratch));
    const int bn = block_reduce_sum_int(lN, scratch);
    const int be = block_reduce_sum_int(lerr, scratch);
    if (tid == 0) {
      ex->loc_max = bm;
      ex->loc_N = bn;
      ex->loc_err = be;
    }
  }
  cluster.sync();  // (A) S_k and zeroed accumulators visible; per-CTA summaries published
  float gmax = -INFINITY;
  int N = 0, err = 0;
  for (int r = 0; r < kSelCluster; ++r) {
    const SelShared* rex = cluster.map_shared_rank(ex, r);
    gmax = fmaxf(gmax, rex->loc_max);
    N += rex->loc_N;
    err += rex->loc_err;
  }
  if (err) {
    if (rank == 0 && tid == 0) {
      record_status(a.status, STEPKV_EDATA);
      *a.out.n_kept = 0;
      if (a.out.n_budget) { a.out.n_budget[0] = N; a.out.n_budget[1] = 0; }
    }
    cluster.sync();
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
  const int fx_shift = 62 - log2N - e_max;    // every partial sum < 2^62
  const float fx_scale = ldexpf(1.0f, min(fx_shift, 126));

  // ---- priorities and ordered keys; per-step statistics (run-aggregated integer atomics)
  {
    int run_sid = -1, run_cnt = 0;
    unsigned long long run_sum = 0ull;
    uint32_t run_max = 0u;
    auto flush = [&]() {
      if (run_sid >= 0 && run_cnt) {
        atomicAdd(&a.acc_cnt[run_sid], run_cnt);
        atomicAdd(&a.acc_sum[run_sid], run_sum);
        atomicMax(&a.acc_max[run_sid], run_max);
      }
    };
    for (int i = tid; i < len; i += kSelThreads) {
      const int gi = base + i;
      const float th = sT[i] * inv_max;
      if (a.out.token_sal) a.out.token_sal[gi] = th;
      uint32_t key = 0u;
      if (!sProt[i]) {
        const int sid = a.step_id[gi];
        const float P = fmaf(a.prm.alpha, th, a.prm.beta * a.S[sid]);
        key = float_to_ordered(P);
        if (a.out.priority) a.out.priority[gi] = P;
        const float thc = fmaxf(th, 0.f);
        if (sid != run_sid) {
          flush();
          run_sid = sid;
          run_cnt = 0;
          run_sum = 0ull;
          run_max = 0u;
        }
        ++run_cnt;
        run_sum += (unsigned long long)llrintf(thc * fx_scale);
        run_max = max(run_max, __float_as_uint(thc));
      } else if (a.out.priority) {
        a.out.priority[gi] = -INFINITY;
      }
      sKey[i] = key;
    }
    flush();
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
    const int shifts[3] = {21, 10, 0};
    const int nbits[3] = {11, 11, 10};
    for (int pass = 0; pass < 3; ++pass) {
      int* h = hist + (pass & 1) * 2048;
      const int nb = 1 << nbits[pass];
      const int sh = shifts[pass];
      for (int b = tid; b < nb; b += kSelThreads) h[b] = 0;
      __syncthreads();
      for (int i = tid; i < len; i += kSelThreads) {
        const uint32_t k = sKey[i];
        if (!sProt[i] && (k & mask) == prefix) atomicAdd(&h[(k >> sh) & (nb - 1)], 1);
      }
      cluster.sync();  // every CTA's histogram of this pass is complete
      // global histogram; thread t owns bins [t*bpt, (t+1)*bpt)
      const int bpt = nb / kSelThreads;  // 4 or 2
      int cnt[4] = {0, 0, 0, 0};
      for (int r = 0; r < kSelCluster; ++r) {
        const int* rh = cluster.map_shared_rank(h, r);
        for (int q = 0; q < bpt; ++q) cnt[q] += rh[tid * bpt + q];
      }
      int mine = 0;
      for (int q = 0; q < bpt; ++q) mine += cnt[q];
      // suffix sum over threads (bins above mine): scan in reversed thread order
      int excl_rev;
      {
        const int lane = tid & 31, warp = tid >> 5;
        // reversed index: thread 511 first
        int x = mine;
        for (int o = 1; o < 32; o <<= 1) {
          const int y = __shfl_down_sync(0xffffffffu, x, o);
          if (lane + o < 32) x += y;
        }
        __syncthreads();
        if (lane == 0) scratch[warp] = x;  // sum of lanes >= 0 of this warp = warp total
        __syncthreads();
        int after = 0;
        for (int w = warp + 1; w < kSelWarps; ++w) after += scratch[w];
        excl_rev = after + x - mine;  // keys in bins owned by higher threads
      }
      int above = excl_rev;
      for (int q = bpt - 1; q >= 0; --q) {
        if (above < remaining && remaining <= above + cnt[q]) {
          bcast[0] = tid * bpt + q;
          bcast[1] = above;
        }
        above += cnt[q];
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

  // ---- per-CTA counts: protected + strictly greater, ties at the threshold
  {
    int kb = 0, eq = 0;
    for (int i = tid; i < len; i += kSelThreads) {
      if (sProt[i]) ++kb;
      else if (sKey[i] > kth) ++kb;
      else if (sKey[i] == kth) ++eq;
    }
    const int bkb = block_reduce_sum_int(kb, scratch);
    const int beq = block_reduce_sum_int(eq, scratch);
    if (tid == 0) {
      ex->loc_keep_base = bkb;
      ex->loc_eq = beq;
    }
  }
  cluster.sync();  // (B)
  // offsets: CTA r keeps its protected + strictly-greater tokens and the ties that fall within the
  // first need_eq ties in slot order
  int out_off = 0, total_kept = 0, ties_before = 0, eq_cum = 0;
  for (int r = 0; r < kSelCluster; ++r) {
    const SelShared* rex = cluster.map_shared_rank(ex, r);
    const int granted = max(0, min(need_eq - eq_cum, rex->loc_eq));
    const int kept_r = rex->loc_keep_base + granted;
    if (r < rank) {
      out_off += kept_r;
      ties_before += rex->loc_eq;
    }
    total_kept += kept_r;
    eq_cum += rex->loc_eq;
  }
  const bool overflow = total_kept > a.out.kept_cap;
  if (rank == 0 && tid == 0) {
    *a.out.n_kept = total_kept;
    if (a.out.n_budget) { a.out.n_budget[0] = N; a.out.n_budget[1] = B; }
    if (overflow) record_status(a.status, STEPKV_ENOSPACE);
  }

  // ---- ordered write of the retained slots (ballot + prefix per 512-token round)
  if (!overflow) {
    int run_keep = 0, run_eq = 0;
    const int lane = tid & 31, warp = tid >> 5;
    int* wk = scratch;               // kSelWarps kept counts
    int* we = scratch + kSelWarps;   // uses bcast area too (kSelWarps more ints)
    for (int r0 = 0; r0 < len; r0 += kSelThreads) {
      const int i = r0 + tid;
      const bool in = i < len;
      const uint32_t k = in ? sKey[i] : 0u;
      const bool pr = in && sProt[i];
      const bool is_eq = in && !pr && k == kth;
      const unsigned eq_mask = __ballot_sync(0xffffffffu, is_eq);
      const int eq_lane_before = __popc(eq_mask & ((1u << lane) - 1u));
      if (lane == 0) we[warp] = __popc(eq_mask);
      __syncthreads();
      int eq_warp_before = 0, eq_round = 0;
      for (int w = 0; w < kSelWarps; ++w) {
        if (w < warp) eq_warp_before += we[w];
        eq_round += we[w];
      }
      const int eq_rank = ties_before + run_eq + eq_warp_before + eq_lane_before;
      const bool keep = in && (pr || (k > kth) || (is_eq && eq_rank < need_eq));
      const unsigned keep_mask = __ballot_sync(0xffffffffu, keep);
      const int keep_lane_before = __popc(keep_mask & ((1u << lane) - 1u));
      if (lane == 0) wk[warp] = __popc(keep_mask);
      __syncthreads();
      int keep_warp_before = 0, keep_round = 0;
      for (int w = 0; w < kSelWarps; ++w) {
        if (w < warp) keep_warp_before += wk[w];
        keep_round += wk[w];
      }
      if (keep) {
        const int gi = base + i;
        a.out.kept_idx[out_off + run_keep + keep_warp_before + keep_lane_before] = gi;
        if (!pr) atomicAdd(&a.acc_kept[a.step_id[gi]], 1);
      }
      run_keep += keep_round;
      run_eq += eq_round;
      __syncthreads();
    }
  }
  cluster.sync();  // (C) all step accumulators final

  // ---- per-step outputs
  for (int k = rank * kSelThreads + tid; k < n_steps; k += kSelCluster * kSelThreads) {
    if (a.out.step_count) a.out.step_count[k] = a.acc_cnt[k];
    if (a.out.step_sal_sum) a.out.step_sal_sum[k] = (float)((double)a.acc_sum[k] / (double)fx_scale);
    if (a.out.step_sal_max) a.out.step_sal_max[k] = __uint_as_float(a.acc_max[k]);
    if (a.out.step_kept) a.out.step_kept[k] = a.acc_kept[k];
  }
  cluster.sync();  // no CTA exits while another may still read its shared memory
}

// -------------------------------------------------------------------------------------------------
static size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

size_t select_ws_bytes(int T, int n_steps) {
  (void)T;
  const size_t n = (size_t)std::max(n_steps, 1);
  return align256(n * 4) + align256(n * 4) + align256(n * 8) + align256(n * 4) + align256(n * 4);
}

stepkv_status_t select_run(const float* rows, int n_rows, int64_t row_stride, float inv_div, int T,
                           const int32_t* step_id, const uint8_t* prot, const stepkv_steps_t& steps,
                           const stepkv_params_t& params, const stepkv_budget_t& budget,
                           const stepkv_select_out_t& out, void* ws, int32_t* status, cudaStream_t stream) {
  SelectArgs a;
  memset(&a, 0, sizeof(a));
  a.rows = rows;
  a.n_rows = n_rows;
  a.row_stride = row_stride;
  a.inv_div = inv_div;
  a.T = T;
  a.chunk = ((T + kSelCluster - 1) / kSelCluster + 15) & ~15;
  a.step_id = step_id;
  a.prot = prot;
  a.steps = steps;
  a.prm = params;
  a.budget = budget;
  a.out = out;
  const size_t n = (size_t)std::max(steps.n_steps, 1);
  uint8_t* w = static_cast<uint8_t*>(ws);
  a.S = reinterpret_cast<float*>(w);
  w += align256(n * 4);
  a.acc_cnt = reinterpret_cast<int32_t*>(w);
  w += align256(n * 4);
  a.acc_sum = reinterpret_cast<unsigned long long*>(w);
  w += align256(n * 8);
  a.acc_max = reinterpret_cast<uint32_t*>(w);
  w += align256(n * 4);
  a.acc_kept = reinterpret_cast<int32_t*>(w);
  a.status = status;
  const size_t smem = (((size_t)a.chunk * 5 + 15) & ~size_t(15)) + 2 * 2048 * 4 + sizeof(SelShared) + 64 * 4;
  cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(select_kernel), (int)smem);
  if (e == cudaSuccess)
    e = launch_pdl_cluster(select_kernel, dim3(kSelCluster), dim3(kSelThreads), kSelCluster, smem, stream, a);
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return STEPKV_ECUDA;
  }
  return STEPKV_OK;
}

}  // namespace stepkv
