// Stage 5 -- compaction of the retained rows (Eq. 1: C_hat = C_prot || C_traj[K]).
//   out[l][h][r][:] = in[l][h][kept_idx[r]][:]  for every layer, KV head and tensor (K, V)
//
// GB300 design: a pure HBM copy (about 4/5 of the pass's bytes).  Each CTA owns a block of 64
// retained rows, keeps their source indices in registers/shared memory, and walks a slice of the
// (layer, tensor, head) row sets.  Each thread moves 16-byte vectors with streaming loads/stores
// (the data is touched once; keep it from evicting the L2-resident score data); four independent
// vectors per thread are in flight before the first store.  n_kept is read on the device.
#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace stepkv {

constexpr int kCompactThreads = 256;
constexpr int kCompactRows = 64;       // retained rows per CTA
constexpr int kCompactSetsPerCta = 16; // (layer, tensor, head) row sets per CTA
constexpr int kCompactLayersPerLaunch = 96;

struct CompactArgs {
  const uint8_t* src[2 * kCompactLayersPerLaunch];  // per (layer, tensor): base of [Hkv][rows][d]
  uint8_t* dst[2 * kCompactLayersPerLaunch];
  int n_sets;               // n_layers_in_launch * n_tensors * Hkv
  int n_tensors;            // 1 (K only) or 2
  int Hkv;
  int row_bytes;            // d * 2
  int64_t in_head_bytes;
  int64_t out_head_bytes;
  int T;
  const int32_t* kept_idx;
  const int32_t* n_kept;
  int kept_cap;
  const int32_t* step_id_in;
  const int32_t* pos_in;
  int32_t* step_id_out;
  int32_t* pos_out;
  int gather_meta;          // this launch also gathers step_id / pos
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

__global__ void __launch_bounds__(kCompactThreads) compact_kernel(const __grid_constant__ CompactArgs a) {
  __shared__ int s_src[kCompactRows];
  pdl_wait();  // kept_idx / n_kept come from the selection kernel
  pdl_launch_dependents();
  const int n_kept = *a.n_kept;
  if (n_kept > a.kept_cap || n_kept < 0) {
    if (blockIdx.x == 0 && blockIdx.y == 0 && threadIdx.x == 0) record_status(a.status, STEPKV_ENOSPACE);
    return;
  }
  const int r0 = blockIdx.x * kCompactRows;
  if (r0 >= n_kept) return;
  const int nr = min(kCompactRows, n_kept - r0);
  if (threadIdx.x < kCompactRows) {
    int s = -1;
    if ((int)threadIdx.x < nr) {
      s = a.kept_idx[r0 + threadIdx.x];
      if (s < 0 || s >= a.T) {
        record_status(a.status, STEPKV_EDATA);
        s = -1;
      }
    }
    s_src[threadIdx.x] = s;
    if (a.gather_meta && blockIdx.y == 0 && (int)threadIdx.x < nr) {
      const int r = r0 + threadIdx.x;
      if (a.step_id_out) a.step_id_out[r] = (s >= 0 && a.step_id_in) ? a.step_id_in[s] : -1;
      if (a.pos_out) a.pos_out[r] = s < 0 ? -1 : (a.pos_in ? a.pos_in[s] : s);
    }
  }
  __syncthreads();
  const int vpr = a.row_bytes >> 4;  // 16-byte vectors per row
  const int nvec = nr * vpr;
  const int set_lo = blockIdx.y * kCompactSetsPerCta;
  const int set_hi = min(a.n_sets, set_lo + kCompactSetsPerCta);
  for (int set = set_lo; set < set_hi; ++set) {
    const int h = set % a.Hkv;
    const int lt = set / a.Hkv;  // layer*n_tensors + tensor
    const uint8_t* src = a.src[lt] + (int64_t)h * a.in_head_bytes;
    uint8_t* dst = a.dst[lt] + (int64_t)h * a.out_head_bytes + (int64_t)r0 * a.row_bytes;
    for (int v0 = threadIdx.x; v0 < nvec; v0 += 4 * kCompactThreads) {
      uint4 buf[4];
      int rr[4], cc[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int v = v0 + u * kCompactThreads;
        rr[u] = v / vpr;
        cc[u] = v - rr[u] * vpr;
        const int s = v < nvec ? s_src[rr[u]] : -1;
        if (s >= 0) buf[u] = ld_stream(reinterpret_cast<const uint4*>(src + (int64_t)s * a.row_bytes) + cc[u]);
        else rr[u] = -1;
      }
#pragma unroll
      for (int u = 0; u < 4; ++u)
        if (rr[u] >= 0) st_stream(reinterpret_cast<uint4*>(dst + (int64_t)rr[u] * a.row_bytes) + cc[u], buf[u]);
    }
  }
}

stepkv_status_t compact_run(int n_layers, const void* const* K_in, const void* const* V_in, int64_t in_head_stride,
                            int Hkv, int d, int T, const int32_t* kept_idx, const int32_t* n_kept, int kept_cap,
                            void* const* K_out, void* const* V_out, int64_t out_head_stride,
                            const int32_t* step_id_in, const int32_t* pos_in, int32_t* step_id_out,
                            int32_t* pos_out, int32_t* status, cudaStream_t stream) {
  const int n_tensors = V_in ? 2 : 1;
  for (int l0 = 0; l0 < std::max(n_layers, 1); l0 += kCompactLayersPerLaunch) {
    const int nl = std::min(kCompactLayersPerLaunch, n_layers - l0);
    CompactArgs a;
    memset(&a, 0, sizeof(a));
    for (int l = 0; l < nl; ++l) {
      a.src[l * n_tensors] = static_cast<const uint8_t*>(K_in[l0 + l]);
      a.dst[l * n_tensors] = static_cast<uint8_t*>(K_out[l0 + l]);
      if (n_tensors == 2) {
        a.src[l * 2 + 1] = static_cast<const uint8_t*>(V_in[l0 + l]);
        a.dst[l * 2 + 1] = static_cast<uint8_t*>(V_out[l0 + l]);
      }
    }
    a.n_sets = std::max(nl, 0) * n_tensors * Hkv;
    a.n_tensors = n_tensors;
    a.Hkv = Hkv;
    a.row_bytes = d * 2;
    a.in_head_bytes = in_head_stride * 2;
    a.out_head_bytes = out_head_stride * 2;
    a.T = T;
    a.kept_idx = kept_idx;
    a.n_kept = n_kept;
    a.kept_cap = kept_cap;
    a.step_id_in = step_id_in;
    a.pos_in = pos_in;
    a.step_id_out = step_id_out;
    a.pos_out = pos_out;
    a.gather_meta = l0 == 0;
    a.status = status;
    const int gx = std::max(1, (kept_cap + kCompactRows - 1) / kCompactRows);
    const int gy = std::max(1, (a.n_sets + kCompactSetsPerCta - 1) / kCompactSetsPerCta);
    cudaError_t e = launch_pdl(compact_kernel, dim3(gx, gy), dim3(kCompactThreads), 0, stream, a);
    if (e != cudaSuccess) {
      set_last_cuda_error(e);
      return STEPKV_ECUDA;
    }
    if (n_layers <= 0) break;
  }
  return STEPKV_OK;
}

}  // namespace stepkv
