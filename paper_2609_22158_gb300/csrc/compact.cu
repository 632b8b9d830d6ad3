// Stage 5 -- compaction of the retained rows (Eq. 1: C_hat = C_prot || C_traj[K]).
//   out[l][h][r][:] = in[l][h][kept_idx[r]][:]  for every layer, KV head and tensor (K, V)
//
// GB300 design: a pure HBM copy (about 4/5 of the pass's bytes).  The work is the list of row items
// (row set, retained row), row set = (layer, tensor, KV head); a grid of 8 CTAs per SM (4 resident at
// this kernel's registers, so two waves; one wave of 4 measured the same) splits it into equal
// contiguous ranges, so every SM streams the same number of rows.  A row of d bf16 is
// d/8 16-byte vectors handled by d/8 lanes, so a warp moves 32/(d/8) rows per instruction; four such
// groups are loaded before the first store (8 rows, 2 KB per warp in flight at d = 128).  Loads and
// stores are streaming (.cs): the data is touched once.  n_kept is read on the device.
#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace stepkv {

constexpr int kCompactThreads = 256;
constexpr int kCompactCtasPerSm = 8;
constexpr int kCompactUnroll = 4;
constexpr int kCompactLayersPerLaunch = 96;

// The in-place move kernel's arguments: the row sets of up to kCompactLayersPerLaunch layers and the plan
// the selection kernel wrote.
struct CompactMoveArgs {
  uint8_t* dst[2 * kCompactLayersPerLaunch];  // per (layer, tensor): base of [Hkv][rows][d]
  int n_sets;               // n_layers_in_launch * n_tensors * Hkv
  int Hkv;
  int row_bytes;            // d * 2
  int64_t out_head_bytes;
  int T;
  int kept_cap;
  const int32_t* plan;      // plan[0] = holes H, plan[1 + j] = hole j (ascending)
  const int32_t* kept_idx;  // the j-th mover is kept_idx[n_kept - H + j]
  const int32_t* n_kept;
  const int32_t* step_id_in;  // metadata of the filled holes (first launch of a trajectory only)
  const int32_t* pos_in;
  int32_t* step_id_out;
  int32_t* pos_out;
  int meta;
  int32_t* status;
};

__device__ __forceinline__ uint4 ld_stream(const uint4* p) {
  uint4 v;
  asm volatile("ld.global.cs.v4.u32 {%0,%1,%2,%3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
  return v;
}
__device__ __forceinline__ void st_stream(uint4* p, const uint4& v) {
  asm volatile("st.global.cs.v4.u32 [%0], {%1,%2,%3,%4};" ::"l"(p), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w) : "memory");
}

// Out-of-place compaction of up to kCompactMaxTraj trajectories in one launch (one stepkv_compress call's
// trajectories share it, so short ones do not each pay a launch and a tail).  The row items of all
// trajectories form one list, in trajectory order, split into equal contiguous ranges per CTA.
constexpr int kCompactMaxTraj = 16;
constexpr int kCompactMaxTensors = 1024;  // (layer, tensor) entries per launch: 16 trajectories x 32 layers x K, V

struct CompactTraj {
  int tensor0;              // first (layer, tensor) entry of this trajectory in src / dst
  int n_sets;               // its row sets: n_layers * n_tensors * Hkv
  int Hkv;
  int T;
  int kept_cap;
  int gather_meta;          // this launch gathers the trajectory's step_id / pos
  int64_t in_head_bytes;
  int64_t out_head_bytes;
  const int32_t* kept_idx;
  const int32_t* n_kept;
  const int32_t* step_id_in;
  const int32_t* pos_in;
  int32_t* step_id_out;
  int32_t* pos_out;
};

struct CompactBatchArgs {
  const uint8_t* src[kCompactMaxTensors];  // per (trajectory, layer, tensor): base of [Hkv][rows][d]
  uint8_t* dst[kCompactMaxTensors];
  CompactTraj tr[kCompactMaxTraj];
  int n_traj;
  int row_bytes;            // d * 2
  int32_t* status;
};

static_assert(sizeof(CompactBatchArgs) <= 32000, "kernel parameter space");

__global__ void __launch_bounds__(kCompactThreads) compact_kernel(const __grid_constant__ CompactBatchArgs a) {
  pdl_wait();  // kept_idx / n_kept come from the selection kernel
  pdl_launch_dependents();
  __shared__ int s_nk[kCompactMaxTraj];
  __shared__ long long s_off[kCompactMaxTraj + 1];  // first row item of each trajectory
  if (threadIdx.x < a.n_traj) {
    const CompactTraj& t = a.tr[threadIdx.x];
    int nk = *t.n_kept;
    if (nk > t.kept_cap || nk < 0) {
      if (blockIdx.x == 0) record_status(a.status, STEPKV_ENOSPACE);
      nk = 0;
    }
    s_nk[threadIdx.x] = nk;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    long long o = 0;
    for (int b = 0; b < a.n_traj; ++b) {
      s_off[b] = o;
      o += (long long)a.tr[b].n_sets * s_nk[b];
    }
    s_off[a.n_traj] = o;
  }
  __syncthreads();
  for (int b = 0; b < a.n_traj; ++b) {
    const CompactTraj& t = a.tr[b];
    if (!t.gather_meta) continue;
    for (int r = blockIdx.x * kCompactThreads + threadIdx.x; r < s_nk[b]; r += gridDim.x * kCompactThreads) {
      const int s = t.kept_idx[r];
      const bool ok = s >= 0 && s < t.T;
      if (!ok) record_status(a.status, STEPKV_EDATA);
      if (t.step_id_out) t.step_id_out[r] = (ok && t.step_id_in) ? t.step_id_in[s] : -1;
      if (t.pos_out) t.pos_out[r] = ok ? (t.pos_in ? t.pos_in[s] : s) : -1;
    }
  }
  const int64_t total = s_off[a.n_traj];  // row items
  const int64_t per_cta = (total + gridDim.x - 1) / gridDim.x;
  const int64_t lo = blockIdx.x * per_cta;
  const int64_t hi = min(total, lo + per_cta);
  const int vpr = a.row_bytes >> 4;      // lanes per row
  const int rpw = 32 / vpr;              // rows per warp instruction
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int sub_row = lane / vpr, col = lane - sub_row * vpr;
  const bool lane_active = sub_row < rpw;  // d/8 need not divide 32: the spare lanes idle
  const int stride = (kCompactThreads / 32) * rpw * kCompactUnroll;  // items between a thread's iterations
  // The CTA's range, one trajectory segment at a time; within a segment each thread walks its items as
  // (row set, retained row) pairs, advanced by `stride` items per iteration without a division.
  for (int b = 0; b < a.n_traj; ++b) {
    const int64_t seg_lo = max(lo, (int64_t)s_off[b]), seg_hi = min(hi, (int64_t)s_off[b + 1]);
    if (seg_lo >= seg_hi) continue;
    const CompactTraj& t = a.tr[b];
    const int nk = s_nk[b];
    const int i0 = (int)(seg_lo - s_off[b]), i1 = (int)(seg_hi - s_off[b]);  // items of the trajectory
    const int32_t* __restrict__ kidx = t.kept_idx;
    const int Hkv = t.Hkv, T = t.T, tensor0 = t.tensor0;
    const int64_t in_hb = t.in_head_bytes, out_hb = t.out_head_bytes;
    int set[kCompactUnroll], row[kCompactUnroll];
#pragma unroll
    for (int u = 0; u < kCompactUnroll; ++u) {
      const int it = i0 + warp * rpw * kCompactUnroll + u * rpw + sub_row;
      set[u] = it / nk;
      row[u] = it - set[u] * nk;
    }
    for (int base = i0 + warp * rpw * kCompactUnroll; base < i1; base += stride) {
      uint4 buf[kCompactUnroll];
      uint4* dptr[kCompactUnroll];
#pragma unroll
      for (int u = 0; u < kCompactUnroll; ++u) {
        const int it = base + u * rpw + sub_row;
        dptr[u] = nullptr;
        if (lane_active && it < i1) {
          const int s = __ldg(&kidx[row[u]]);
          if (s >= 0 && s < T) {
            const int lt = set[u] / Hkv, h = set[u] - lt * Hkv;
            const uint8_t* src = a.src[tensor0 + lt] + (int64_t)h * in_hb + (int64_t)s * a.row_bytes;
            buf[u] = ld_stream(reinterpret_cast<const uint4*>(src) + col);
            dptr[u] = reinterpret_cast<uint4*>(a.dst[tensor0 + lt] + (int64_t)h * out_hb +
                                               (int64_t)row[u] * a.row_bytes) + col;
          }
        }
      }
#pragma unroll
      for (int u = 0; u < kCompactUnroll; ++u)
        if (dptr[u]) st_stream(dptr[u], buf[u]);
#pragma unroll
      for (int u = 0; u < kCompactUnroll; ++u) {
        row[u] += stride;
        while (row[u] >= nk) {
          row[u] -= nk;
          ++set[u];
        }
      }
    }
  }
}

// -------------------------------------------------------------------------------------------------
// In-place compaction by hole filling.  With the retained slots kept_idx ascending and n = n_kept, the
// slots below n that are retained stay where they are; every slot below n that is not retained (a hole)
// receives one retained row from a slot at or above n (a mover), the j-th hole the j-th mover.  Sources
// (>= n) and destinations (< n) never overlap, so all moves run in parallel.  Rows [0, n) then hold the
// retained set, no longer in slot order; step_id_out / pos_out record each row's step and original
// position.  Only the movers are read and written, instead of every retained row.  The selection kernel
// lays out the plan as it writes kept_idx (the number of a hole is its slot minus the retained slots below
// it, which that pass counts anyway), so the moves need no launch of their own to find it.

__global__ void __launch_bounds__(kCompactThreads) compact_move_kernel(const __grid_constant__ CompactMoveArgs a) {
  pdl_wait();
  pdl_launch_dependents();
  const int n = __ldcg(a.n_kept);
  if (n < 0 || n > a.kept_cap || n > a.T) return;  // the selection has recorded the error; nothing moves
  const int n_moves = __ldcg(a.plan);
  if (n_moves < 0 || n_moves > n) {
    if (blockIdx.x == 0 && threadIdx.x == 0) record_status(a.status, STEPKV_EDATA);
    return;
  }
  const int m0 = n - n_moves;  // the movers are kept_idx[m0 .. n), the retained slots at or above n
  const int32_t* hole = a.plan + 1;
  if (a.meta) {
    for (int j = blockIdx.x * kCompactThreads + threadIdx.x; j < n_moves; j += gridDim.x * kCompactThreads) {
      const int r = __ldcg(&hole[j]), src = __ldcg(&a.kept_idx[m0 + j]);
      if (r < 0 || r >= n || src < n || src >= a.T) {
        record_status(a.status, STEPKV_EDATA);
        continue;
      }
      if (a.step_id_out) a.step_id_out[r] = a.step_id_in ? __ldg(&a.step_id_in[src]) : -1;
      if (a.pos_out) a.pos_out[r] = a.pos_in ? __ldg(&a.pos_in[src]) : src;
    }
  }
  const int64_t total = (int64_t)a.n_sets * n_moves;
  const int64_t per_cta = (total + gridDim.x - 1) / gridDim.x;
  const int64_t lo = blockIdx.x * per_cta;
  const int64_t hi = min(total, lo + per_cta);
  const int vpr = a.row_bytes >> 4;
  const int rpw = 32 / vpr;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int sub_row = lane / vpr, col = lane - sub_row * vpr;
  const bool lane_active = sub_row < rpw;
  const int64_t step = (int64_t)(kCompactThreads / 32) * rpw * kCompactUnroll;
  for (int64_t base = lo + (int64_t)warp * rpw * kCompactUnroll; base < hi; base += step) {
    uint4 buf[kCompactUnroll];
    uint4* dptr[kCompactUnroll];
#pragma unroll
    for (int u = 0; u < kCompactUnroll; ++u) {
      const int64_t ri = base + u * rpw + sub_row;
      dptr[u] = nullptr;
      if (lane_active && ri < hi) {
        const int set = (int)(ri / n_moves);
        const int j = (int)(ri - (int64_t)set * n_moves);
        // written by the selection kernel (programmatic dependent launch): read through L2
        const int src_row = __ldcg(&a.kept_idx[m0 + j]), dst_row = __ldcg(&hole[j]);
        if (src_row >= n && src_row < a.T && dst_row >= 0 && dst_row < n) {
          const int lt = set / a.Hkv, h = set - lt * a.Hkv;
          uint8_t* head = a.dst[lt] + (int64_t)h * a.out_head_bytes;
          buf[u] = ld_stream(reinterpret_cast<const uint4*>(head + (int64_t)src_row * a.row_bytes) + col);
          dptr[u] = reinterpret_cast<uint4*>(head + (int64_t)dst_row * a.row_bytes) + col;
        }
      }
    }
#pragma unroll
    for (int u = 0; u < kCompactUnroll; ++u)
      if (dptr[u]) st_stream(dptr[u], buf[u]);
  }
}

size_t compact_inplace_ws_bytes(int T) { return (size_t)(1 + (size_t)T) * sizeof(int32_t); }

stepkv_status_t compact_inplace_run(int n_layers, void* const* K, void* const* V, int64_t head_stride, int Hkv, int d,
                                    int T, const int32_t* kept_idx, const int32_t* n_kept, int kept_cap,
                                    const int32_t* step_id_in, const int32_t* pos_in, int32_t* step_id_out,
                                    int32_t* pos_out, void* ws, int32_t* status, cudaStream_t stream) {
  static int resident = 0;  // move-kernel CTAs resident per SM (registers bound it): one wave of them
  int n_sm = 0;
  cudaError_t e = device_sm_count(&n_sm);
  if (e == cudaSuccess && resident == 0) {
    int r = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&r, compact_move_kernel, kCompactThreads, 0);
    resident = std::max(1, std::min(r, kCompactCtasPerSm));
  }
  const int n_tensors = V ? 2 : 1;
  for (int l0 = 0; e == cudaSuccess && l0 < std::max(n_layers, 1); l0 += kCompactLayersPerLaunch) {
    const int nl = std::min(kCompactLayersPerLaunch, n_layers - l0);
    if (nl <= 0) break;
    CompactMoveArgs a;
    memset(&a, 0, sizeof(a));
    for (int l = 0; l < nl; ++l) {
      a.dst[l * n_tensors] = static_cast<uint8_t*>(K[l0 + l]);
      if (n_tensors == 2) a.dst[l * 2 + 1] = static_cast<uint8_t*>(V[l0 + l]);
    }
    a.n_sets = nl * n_tensors * Hkv;
    a.Hkv = Hkv;
    a.row_bytes = d * 2;
    a.out_head_bytes = head_stride * 2;
    a.T = T;
    a.kept_cap = kept_cap;
    a.plan = static_cast<const int32_t*>(ws);
    a.kept_idx = kept_idx;
    a.n_kept = n_kept;
    a.step_id_in = step_id_in;
    a.pos_in = pos_in;
    a.step_id_out = step_id_out;
    a.pos_out = pos_out;
    a.meta = l0 == 0;
    a.status = status;
    // moves: at most min(n_kept, T - n_kept) <= T / 2 rows per set
    const int64_t rows_max = (int64_t)a.n_sets * std::max(std::min(kept_cap, T / 2), 1);
    const int64_t want = (rows_max + 31) / 32;
    const int grid = (int)std::max<int64_t>(1, std::min<int64_t>((int64_t)n_sm * resident, want));
    e = launch_kernel(compact_move_kernel, dim3(grid), dim3(kCompactThreads), 0, stream, a, true);
  }
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return STEPKV_ECUDA;
  }
  return STEPKV_OK;
}

// Launches for a list of out-of-place compactions: consecutive ones with one row size share a launch while
// they fit (kCompactMaxTraj trajectories, kCompactMaxTensors (layer, tensor) entries); a trajectory with
// more entries than one launch holds is split by layers over launches of its own.
stepkv_status_t compact_run_batch(const CompactSpec* specs, int n, int32_t* status, cudaStream_t stream) {
  int n_sm = 0;
  cudaError_t e = device_sm_count(&n_sm);
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return STEPKV_ECUDA;
  }
  CompactBatchArgs a;
  int64_t rows_max = 0;
  auto reset = [&]() {
    memset(&a, 0, sizeof(a));
    a.status = status;
    rows_max = 0;
  };
  auto flush = [&]() -> cudaError_t {
    if (a.n_traj == 0) return cudaSuccess;
    const int64_t want = (rows_max + 31) / 32;  // no more CTAs than 32 row items each at full capacity
    const int grid = (int)std::max<int64_t>(1, std::min<int64_t>((int64_t)n_sm * kCompactCtasPerSm, want));
    cudaError_t err = launch_kernel(compact_kernel, dim3(grid), dim3(kCompactThreads), 0, stream, a);
    reset();
    return err;
  };
  int used = 0;  // (layer, tensor) entries in the pending launch
  reset();
  for (int i = 0; i < n && e == cudaSuccess; ++i) {
    const CompactSpec& c = specs[i];
    const int n_tensors = c.V_in ? 2 : 1;
    const int max_layers = kCompactMaxTensors / n_tensors;
    for (int l0 = 0; l0 < std::max(c.n_layers, 1) && e == cudaSuccess; l0 += max_layers) {
      const int nl = std::max(0, std::min(max_layers, c.n_layers - l0));
      if (a.n_traj > 0 && (a.n_traj == kCompactMaxTraj || used + nl * n_tensors > kCompactMaxTensors ||
                           a.row_bytes != c.d * 2)) {
        e = flush();
        used = 0;
        if (e != cudaSuccess) break;
      }
      CompactTraj& t = a.tr[a.n_traj];
      t.tensor0 = used;
      for (int l = 0; l < nl; ++l) {
        a.src[used + l * n_tensors] = static_cast<const uint8_t*>(c.K_in[l0 + l]);
        a.dst[used + l * n_tensors] = static_cast<uint8_t*>(c.K_out[l0 + l]);
        if (n_tensors == 2) {
          a.src[used + l * 2 + 1] = static_cast<const uint8_t*>(c.V_in[l0 + l]);
          a.dst[used + l * 2 + 1] = static_cast<uint8_t*>(c.V_out[l0 + l]);
        }
      }
      used += nl * n_tensors;
      t.n_sets = nl * n_tensors * c.Hkv;
      t.Hkv = c.Hkv;
      t.T = c.T;
      t.kept_cap = c.kept_cap;
      t.gather_meta = l0 == 0;
      t.in_head_bytes = c.in_head_stride * 2;
      t.out_head_bytes = c.out_head_stride * 2;
      t.kept_idx = c.kept_idx;
      t.n_kept = c.n_kept;
      t.step_id_in = c.step_id_in;
      t.pos_in = c.pos_in;
      t.step_id_out = c.step_id_out;
      t.pos_out = c.pos_out;
      a.row_bytes = c.d * 2;
      ++a.n_traj;
      rows_max += (int64_t)std::max(t.n_sets, 1) * std::max(c.kept_cap, 1);
      if (nl < c.n_layers) {  // a split trajectory keeps its launches to itself
        e = flush();
        used = 0;
      }
    }
  }
  if (e == cudaSuccess) e = flush();
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return STEPKV_ECUDA;
  }
  return STEPKV_OK;
}

stepkv_status_t compact_run(int n_layers, const void* const* K_in, const void* const* V_in, int64_t in_head_stride,
                            int Hkv, int d, int T, const int32_t* kept_idx, const int32_t* n_kept, int kept_cap,
                            void* const* K_out, void* const* V_out, int64_t out_head_stride,
                            const int32_t* step_id_in, const int32_t* pos_in, int32_t* step_id_out,
                            int32_t* pos_out, int32_t* status, cudaStream_t stream) {
  const CompactSpec c{n_layers, K_in, V_in, in_head_stride, Hkv, d, T, kept_idx, n_kept, kept_cap,
                      K_out, V_out, out_head_stride, step_id_in, pos_in, step_id_out, pos_out};
  return compact_run_batch(&c, 1, status, stream);
}

}  // namespace stepkv
