// Decode attention over the compacted cache: after a compression boundary the agent keeps decoding,
// and every new token attends to the retained rows C_hat = C_prot || C_traj[K] (Eq. 1).  For each
// layer and query head g (KV head g / G):
//   out[g][:] = sum_{j < n} softmax_j( q[g] . K[g/G][j] / sqrt(d) ) V[g/G][j][:]
//
// GB300 design: HBM-bound (the K and V rows are read once per token, 1.08 GB for 32 layers x 8 heads x
// 8272 rows), so the kernel is built around coalesced 16-byte loads and enough bytes in flight; the
// contraction is 2 x G x d flop per key row and stays on the FP32 pipe.  Split-K: a CTA owns 512 keys of
// one (layer, KV head) pair and all G query heads of its group, so every key row is loaded once for the
// whole group.  d/8 lanes share a key row (8 bf16 each); a warp covers 32/(d/8) keys per step, four steps
// per block, and keeps a running (max, sum, weighted values) per head, rescaled once per block.  A
// second kernel merges the per-split partials of each (pair, head) in split order (deterministic).
// The number of keys may be read on the device (n_kept of a compaction), so no host sync is needed.
//
// Accumulated attention (the H2O-style token saliency, Sec. 4.2: T_i may come from an existing
// token-level importance estimator): with mass rows given, the partial kernel also stores every key's
// logits per head, and the merge runs up to 8 CTAs per (layer, KV head), each over a contiguous share of
// the keys.  Every CTA merges the heads' (m, l) split states in split order into each head's
// log-sum-exp (the first CTA also merges the value rows, in the same order as the plain merge, so the
// outputs are bit-identical).  Then its threads add (1/G) sum_g softmax_j(q_g . k_j / sqrt(d)) to
// mass[j] for each of its keys: one writer per element and call, a fixed order over g, so the result is
// deterministic.
#include <math.h>

#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace stepkv {

constexpr int kDecThreads = 128;
constexpr int kDecWarps = kDecThreads / 32;
constexpr int kDecSplitKeys = 512;
constexpr int kDecBlockSteps = 4;

struct DecodeArgs {
  const uint16_t* q[kMaxDecodeLayers];
  const uint16_t* K[kMaxDecodeLayers];
  const uint16_t* V[kMaxDecodeLayers];
  float* out[kMaxDecodeLayers];
  int64_t head_stride;  // elements
  int Hkv;
  int n_splits;
  const int32_t* n_dev;
  int n_host;
  int n_cap;
  float c;              // log2(e) / sqrt(d)
  float* part;          // [pairs][n_splits][G][d + 4]: m, l, -, -, acc[d]
  float* logits;        // [pairs][n_cap][G] (accumulated-attention mode, else NULL): key logits in log2 units
  float* mass[kMaxDecodeLayers];  // per layer [Hkv][mass_stride]: accumulated attention (+=), or NULL
  int64_t mass_stride;
  int32_t* status;
};

static_assert(sizeof(DecodeArgs) <= 32000, "kernel parameter space");

__device__ __forceinline__ int decode_n(const DecodeArgs& a) {
  const int n = a.n_dev ? *a.n_dev : a.n_host;
  return n;
}

__device__ __forceinline__ void bf16x8_to_f32(const uint4& r, float (&f)[8]) {
  const uint32_t w[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    f[2 * i] = __uint_as_float(w[i] << 16);
    f[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
  }
}

// Merge the state (m2, l2, acc2) into (m, l, acc); -inf marks an empty state.
template <int E>
__device__ __forceinline__ void merge_state(float& m, float& l, float (&acc)[E], float m2, float l2,
                                            const float (&acc2)[E]) {
  const float mn = fmaxf(m, m2);
  if (mn == -INFINITY) return;
  const float a = ex2_approx(m - mn), b = ex2_approx(m2 - mn);
  l = l * a + l2 * b;
#pragma unroll
  for (int e = 0; e < E; ++e) acc[e] = acc[e] * a + acc2[e] * b;
  m = mn;
}

// MASS: the accumulated-attention variant, which also stores every key's logits (a separate
// instantiation, so the plain decode keeps its register budget).
template <int D, int G, bool MASS>
__global__ void __launch_bounds__(kDecThreads) decode_partial_kernel(const __grid_constant__ DecodeArgs a) {
  constexpr int LPK = D / 8;          // lanes per key row
  constexpr int KPS = 32 / LPK;       // keys per warp step
  constexpr int BLK = KPS * kDecBlockSteps;
  __shared__ float s_m[kDecWarps][G], s_l[kDecWarps][G];
  __shared__ float s_acc[kDecWarps][G][D];

  pdl_wait();
  pdl_launch_dependents();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int pair = blockIdx.x / a.n_splits, split = blockIdx.x - pair * a.n_splits;
  const int layer = pair / a.Hkv, h = pair - layer * a.Hkv;
  int n = decode_n(a);
  if (n > a.n_cap) {
    if (threadIdx.x == 0 && blockIdx.x == 0) record_status(a.status, STEPKV_ENOSPACE);
    n = a.n_cap;
  }
  if (n < 1 && threadIdx.x == 0 && blockIdx.x == 0) record_status(a.status, STEPKV_EDATA);
  const int k_begin = split * kDecSplitKeys;
  const int k_end = min(n, k_begin + kDecSplitKeys);
  const int kslot = lane / LPK, hl = lane - kslot * LPK;

  // this lane's 8 elements of every query head of the group, pre-scaled for exp2
  float q[G][8];
#pragma unroll
  for (int g = 0; g < G; ++g) {
    const uint4 r = __ldg(reinterpret_cast<const uint4*>(a.q[layer] + (size_t)(h * G + g) * D) + hl);
    bf16x8_to_f32(r, q[g]);
#pragma unroll
    for (int e = 0; e < 8; ++e) q[g][e] *= a.c;
  }
  // Value accumulators as packed fp32 pairs: a bf16 word holds two neighbouring elements, so a value row
  // converts straight into pairs and every value FMA and rescale is one f32x2 instruction for two elements.
  float m[G], l[G];
  uint64_t accp[G][4];
#pragma unroll
  for (int g = 0; g < G; ++g) {
    m[g] = -INFINITY;
    l[g] = 0.f;
#pragma unroll
    for (int e = 0; e < 4; ++e) accp[g][e] = 0ull;
  }

  const uint16_t* Kh = a.K[layer] + (size_t)h * a.head_stride;
  const uint16_t* Vh = a.V[layer] + (size_t)h * a.head_stride;
  // warp w takes blocks w, w + 4, ... of BLK consecutive keys
  for (int kb = k_begin + warp * BLK; kb < k_end; kb += kDecWarps * BLK) {
    uint4 kr[kDecBlockSteps], vr[kDecBlockSteps];
    bool ok[kDecBlockSteps];
#pragma unroll
    for (int t = 0; t < kDecBlockSteps; ++t) {
      const int j = kb + t * KPS + kslot;
      ok[t] = j < k_end;
      kr[t] = ok[t] ? __ldcs(reinterpret_cast<const uint4*>(Kh + (size_t)j * D) + hl) : make_uint4(0, 0, 0, 0);
      vr[t] = ok[t] ? __ldcs(reinterpret_cast<const uint4*>(Vh + (size_t)j * D) + hl) : make_uint4(0, 0, 0, 0);
    }
    // The warp's next block is fetched into L2 while this one is computed: the loads above wait for
    // DRAM only until the pipeline fills, and the prefetch holds no registers.
    const int kn = kb + kDecWarps * BLK;
    if (lane == 0 && kn < k_end) {
      const uint32_t nbytes = (uint32_t)(min(BLK, k_end - kn) * D * 2);
      bulk_prefetch_l2(Kh + (size_t)kn * D, nbytes);
      bulk_prefetch_l2(Vh + (size_t)kn * D, nbytes);
    }
    float s[kDecBlockSteps][G];
#pragma unroll
    for (int t = 0; t < kDecBlockSteps; ++t) {
      float kf[8];
      bf16x8_to_f32(kr[t], kf);
      float x[G];
#pragma unroll
      for (int g = 0; g < G; ++g) {
        x[g] = 0.f;
#pragma unroll
        for (int e = 0; e < 8; ++e) x[g] = fmaf(q[g][e], kf[e], x[g]);
      }
      if constexpr (G == 4) {
        // reduce-scatter over the LPK lanes of the row (each lane ends with one head's full sum), then
        // broadcast the four sums: 9 shuffles instead of 4 x log2(LPK)
        constexpr int A = LPK / 2, Bx = LPK / 4;
        const bool ba = (hl & A) != 0, bb = (hl & Bx) != 0;
        const float y0 = (ba ? x[2] : x[0]) + __shfl_xor_sync(0xffffffffu, ba ? x[0] : x[2], A);
        const float y1 = (ba ? x[3] : x[1]) + __shfl_xor_sync(0xffffffffu, ba ? x[1] : x[3], A);
        float z = (bb ? y1 : y0) + __shfl_xor_sync(0xffffffffu, bb ? y0 : y1, Bx);
#pragma unroll
        for (int o = Bx / 2; o > 0; o >>= 1) z += __shfl_xor_sync(0xffffffffu, z, o);
        const int base_lane = lane & ~(LPK - 1);
#pragma unroll
        for (int g = 0; g < 4; ++g) {
          const float v = __shfl_sync(0xffffffffu, z, base_lane | (((g >> 1) ? A : 0) | ((g & 1) ? Bx : 0)));
          s[t][g] = ok[t] ? v : -INFINITY;
        }
      } else {
#pragma unroll
        for (int g = 0; g < G; ++g) {
          float v = x[g];
#pragma unroll
          for (int o = LPK / 2; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
          s[t][g] = ok[t] ? v : -INFINITY;
        }
      }
    }
    if (MASS && hl == 0) {
      // every lane of a key row holds the row's logits of all G heads: the first one stores them
#pragma unroll
      for (int t = 0; t < kDecBlockSteps; ++t) {
        const int j = kb + t * KPS + kslot;
        if (ok[t]) {
          float* dst = a.logits + ((size_t)pair * a.n_cap + j) * G;
          if constexpr (G % 4 == 0) {
#pragma unroll
            for (int g = 0; g < G; g += 4)
              *reinterpret_cast<float4*>(dst + g) = make_float4(s[t][g], s[t][g + 1], s[t][g + 2], s[t][g + 3]);
          } else {
#pragma unroll
            for (int g = 0; g < G; ++g) dst[g] = s[t][g];
          }
        }
      }
    }
    // probabilities of the block's keys per head (state rescaled once per block), then one pass over
    // the value rows: each is converted once and accumulated into every head
    float p[kDecBlockSteps][G];
#pragma unroll
    for (int g = 0; g < G; ++g) {
      float mb = m[g];
#pragma unroll
      for (int t = 0; t < kDecBlockSteps; ++t) mb = fmaxf(mb, s[t][g]);
      if (mb == -INFINITY) {
#pragma unroll
        for (int t = 0; t < kDecBlockSteps; ++t) p[t][g] = 0.f;
        continue;
      }
      const float sc = ex2_approx(m[g] - mb);
      l[g] *= sc;
#pragma unroll
      for (int e = 0; e < 4; ++e) accp[g][e] = f2_mul(accp[g][e], f2_pack(sc, sc));
#pragma unroll
      for (int t = 0; t < kDecBlockSteps; ++t) {
        p[t][g] = ex2_approx(s[t][g] - mb);
        l[g] += p[t][g];
      }
      m[g] = mb;
    }
#pragma unroll
    for (int t = 0; t < kDecBlockSteps; ++t) {
      const uint32_t w[4] = {vr[t].x, vr[t].y, vr[t].z, vr[t].w};
      uint64_t vp[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) vp[e] = f2_pack(__uint_as_float(w[e] << 16), __uint_as_float(w[e] & 0xFFFF0000u));
#pragma unroll
      for (int g = 0; g < G; ++g) {
        const uint64_t pp = f2_pack(p[t][g], p[t][g]);
#pragma unroll
        for (int e = 0; e < 4; ++e) accp[g][e] = f2_fma(vp[e], pp, accp[g][e]);
      }
    }
  }
  float acc[G][8];
#pragma unroll
  for (int g = 0; g < G; ++g)
#pragma unroll
    for (int e = 0; e < 4; ++e) f2_unpack(accp[g][e], acc[g][2 * e], acc[g][2 * e + 1]);
  // merge the key slots of the warp (lanes with the same hl), then the warps through shared memory
#pragma unroll
  for (int o = LPK; o < 32; o <<= 1) {
#pragma unroll
    for (int g = 0; g < G; ++g) {
      const float m2 = __shfl_xor_sync(0xffffffffu, m[g], o);
      const float l2 = __shfl_xor_sync(0xffffffffu, l[g], o);
      float acc2[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) acc2[e] = __shfl_xor_sync(0xffffffffu, acc[g][e], o);
      merge_state<8>(m[g], l[g], acc[g], m2, l2, acc2);
    }
  }
  if (kslot == 0) {
#pragma unroll
    for (int g = 0; g < G; ++g) {
      if (hl == 0) {
        s_m[warp][g] = m[g];
        s_l[warp][g] = l[g];
      }
#pragma unroll
      for (int e = 0; e < 8; ++e) s_acc[warp][g][hl * 8 + e] = acc[g][e];
    }
  }
  __syncthreads();
  // thread t < G*D/4: head g = t / (D/4), elements 4*(t % (D/4)) .. +4 -> merge the warps in order
  constexpr int PER = 4;
  for (int t = threadIdx.x; t < G * (D / PER); t += kDecThreads) {
    const int g = t / (D / PER), e0 = (t - g * (D / PER)) * PER;
    float mm = -INFINITY, ll = 0.f, aa[PER] = {0.f, 0.f, 0.f, 0.f};
    for (int w = 0; w < kDecWarps; ++w) {
      float a2[PER];
#pragma unroll
      for (int e = 0; e < PER; ++e) a2[e] = s_acc[w][g][e0 + e];
      merge_state<PER>(mm, ll, aa, s_m[w][g], s_l[w][g], a2);
    }
    float* dst = a.part + ((size_t)(pair * a.n_splits + split) * G + g) * (D + 4);
    if (e0 == 0) {
      dst[0] = mm;
      dst[1] = ll;
    }
    *reinterpret_cast<float4*>(dst + 4 + e0) = make_float4(aa[0], aa[1], aa[2], aa[3]);
  }
}

// One warp per (pair, head): merge the splits in order and write out = acc / l.
template <int D, int G>
__global__ void __launch_bounds__(128) decode_merge_kernel(const __grid_constant__ DecodeArgs a, int n_items) {
  constexpr int PER = D / 32;
  pdl_wait();
  pdl_launch_dependents();
  const int item = blockIdx.x * 4 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (item >= n_items) return;
  const int pair = item / G, g = item - pair * G;
  const int layer = pair / a.Hkv, h = pair - layer * a.Hkv;
  int n = min(decode_n(a), a.n_cap);
  const int used = max(0, min(a.n_splits, (n + kDecSplitKeys - 1) / kDecSplitKeys));
  float mm = -INFINITY, ll = 0.f, aa[PER];
#pragma unroll
  for (int e = 0; e < PER; ++e) aa[e] = 0.f;
  for (int sp = 0; sp < used; ++sp) {
    const float* src = a.part + ((size_t)(pair * a.n_splits + sp) * G + g) * (D + 4);
    float a2[PER];
#pragma unroll
    for (int e = 0; e < PER; ++e) a2[e] = __ldcg(src + 4 + lane * PER + e);
    merge_state<PER>(mm, ll, aa, __ldcg(src), __ldcg(src + 1), a2);
  }
  const float inv = ll > 0.f ? 1.f / ll : 0.f;
  float* o = a.out[layer] + (size_t)(h * G + g) * D + lane * PER;
#pragma unroll
  for (int e = 0; e < PER; ++e) o[e] = aa[e] * inv;
}

// Accumulated-attention merge: one CTA per (layer, KV head).  Warp w merges heads w, w + 4, ... exactly as
// decode_merge_kernel does (bit-identical outputs) and keeps each head's log-sum-exp; then every thread adds
// the group-mean softmax mass of its keys to the pair's mass row.
template <int D, int G>
__global__ void __launch_bounds__(128) decode_merge_mass_kernel(const __grid_constant__ DecodeArgs a, int chunks) {
  constexpr int PER = D / 32;
  __shared__ float s_lse[G];
  pdl_wait();
  pdl_launch_dependents();
  const int pair = blockIdx.x / chunks, chunk = blockIdx.x - pair * chunks;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int layer = pair / a.Hkv, h = pair - layer * a.Hkv;
  const int n = max(0, min(decode_n(a), a.n_cap));
  const int used = max(0, min(a.n_splits, (n + kDecSplitKeys - 1) / kDecSplitKeys));
  for (int g = warp; g < G; g += 4) {
    if (chunk == 0) {
      // the pair's outputs: the splits merged in order, as decode_merge_kernel
      float mm = -INFINITY, ll = 0.f, aa[PER];
#pragma unroll
      for (int e = 0; e < PER; ++e) aa[e] = 0.f;
      for (int sp = 0; sp < used; ++sp) {
        const float* src = a.part + ((size_t)(pair * a.n_splits + sp) * G + g) * (D + 4);
        float a2[PER];
#pragma unroll
        for (int e = 0; e < PER; ++e) a2[e] = __ldcg(src + 4 + lane * PER + e);
        merge_state<PER>(mm, ll, aa, __ldcg(src), __ldcg(src + 1), a2);
      }
      const float inv = ll > 0.f ? 1.f / ll : 0.f;
      float* o = a.out[layer] + (size_t)(h * G + g) * D + lane * PER;
#pragma unroll
      for (int e = 0; e < PER; ++e) o[e] = aa[e] * inv;
      if (lane == 0) s_lse[g] = ll > 0.f ? mm + __log2f(ll) : INFINITY;
    } else if (lane == 0) {
      // the same (m, l) merge without the value rows: the same log-sum-exp in every chunk
      float mm = -INFINITY, ll = 0.f, none[1] = {0.f};
      for (int sp = 0; sp < used; ++sp) {
        const float* src = a.part + ((size_t)(pair * a.n_splits + sp) * G + g) * (D + 4);
        merge_state<1>(mm, ll, none, __ldcg(src), __ldcg(src + 1), none);
      }
      s_lse[g] = ll > 0.f ? mm + __log2f(ll) : INFINITY;
    }
  }
  __syncthreads();
  float lse[G];
#pragma unroll
  for (int g = 0; g < G; ++g) lse[g] = s_lse[g];
  const float inv_G = 1.f / (float)G;
  float* mrow = a.mass[layer] + (size_t)h * a.mass_stride;
  const float* lg = a.logits + (size_t)pair * a.n_cap * G;
  // this chunk's keys (one writer per key: the additions are ordered across calls by the stream)
  const int per = (n + chunks - 1) / chunks;
  const int j0 = chunk * per, j1 = min(n, j0 + per);
  for (int j = j0 + threadIdx.x; j < j1; j += 128) {
    float sum = 0.f;
    if constexpr (G % 4 == 0) {
#pragma unroll
      for (int g4 = 0; g4 < G; g4 += 4) {
        const float4 v = __ldcg(reinterpret_cast<const float4*>(lg + (size_t)j * G + g4));
        sum += ex2_approx(v.x - lse[g4]) + ex2_approx(v.y - lse[g4 + 1]) + ex2_approx(v.z - lse[g4 + 2]) +
               ex2_approx(v.w - lse[g4 + 3]);
      }
    } else {
#pragma unroll
      for (int g = 0; g < G; ++g) sum += ex2_approx(__ldcg(lg + (size_t)j * G + g) - lse[g]);
    }
    mrow[j] += sum * inv_G;
  }
}

size_t decode_ws_bytes(int n_layers, int Hkv, int Hq, int d, int n_cap) {
  const int n_splits = std::max(1, (n_cap + kDecSplitKeys - 1) / kDecSplitKeys);
  return (size_t)n_layers * Hq * n_splits * (d + 4) * sizeof(float);
}

size_t decode_mass_ws_bytes(int n_layers, int Hkv, int Hq, int d, int n_cap) {
  // partials (256-byte aligned), then the key logits of every head
  const size_t part = (decode_ws_bytes(n_layers, Hkv, Hq, d, n_cap) + 255) & ~(size_t)255;
  return part + (size_t)n_layers * Hq * std::max(1, n_cap) * sizeof(float);
}

template <int D, int G>
static cudaError_t decode_launch(const DecodeArgs& a, int pairs, cudaStream_t stream) {
  if (a.logits != nullptr) {
    cudaError_t e = launch_kernel(decode_partial_kernel<D, G, true>, dim3(pairs * a.n_splits), dim3(kDecThreads), 0,
                                  stream, a);
    if (e != cudaSuccess) return e;
    // several CTAs per pair over the keys' mass updates (a pair's ~n keys are too few per SM otherwise)
    const int chunks = std::max(1, std::min(8, (a.n_cap + 1023) / 1024));
    return launch_kernel(decode_merge_mass_kernel<D, G>, dim3(pairs * chunks), dim3(128), 0, stream, a, chunks);
  }
  cudaError_t e = launch_kernel(decode_partial_kernel<D, G, false>, dim3(pairs * a.n_splits), dim3(kDecThreads), 0,
                                stream, a);
  if (e != cudaSuccess) return e;
  const int items = pairs * G;
  return launch_kernel(decode_merge_kernel<D, G>, dim3((items + 3) / 4), dim3(128), 0, stream, a, items);
}

template <int D>
static cudaError_t decode_dispatch_g(const DecodeArgs& a, int G, int pairs, cudaStream_t stream) {
  switch (G) {
    case 1: return decode_launch<D, 1>(a, pairs, stream);
    case 2: return decode_launch<D, 2>(a, pairs, stream);
    case 4: return decode_launch<D, 4>(a, pairs, stream);
    case 5: return decode_launch<D, 5>(a, pairs, stream);
    case 8: return decode_launch<D, 8>(a, pairs, stream);
    default: return cudaErrorInvalidValue;
  }
}

stepkv_status_t decode_run(int n_layers, const void* const* q, const void* const* K, const void* const* V,
                           int64_t head_stride, int Hkv, int Hq, int d, const int32_t* n_dev, int n_host, int n_cap,
                           float* const* out, void* ws, int32_t* status, cudaStream_t stream, float* const* mass,
                           int64_t mass_stride) {
  const int G = Hq / Hkv;
  const int n_splits = std::max(1, (n_cap + kDecSplitKeys - 1) / kDecSplitKeys);
  float* part = static_cast<float*>(ws);
  float* logits = nullptr;
  if (mass != nullptr)
    logits = reinterpret_cast<float*>(static_cast<uint8_t*>(ws) +
                                      ((decode_ws_bytes(n_layers, Hkv, Hq, d, n_cap) + 255) & ~(size_t)255));
  for (int l0 = 0; l0 < n_layers; l0 += kMaxDecodeLayers) {
    const int nl = std::min(kMaxDecodeLayers, n_layers - l0);
    DecodeArgs a;
    memset(&a, 0, sizeof(a));
    for (int l = 0; l < nl; ++l) {
      a.q[l] = static_cast<const uint16_t*>(q[l0 + l]);
      a.K[l] = static_cast<const uint16_t*>(K[l0 + l]);
      a.V[l] = static_cast<const uint16_t*>(V[l0 + l]);
      a.out[l] = out[l0 + l];
      a.mass[l] = mass != nullptr ? mass[l0 + l] : nullptr;
    }
    a.logits = logits;  // the chunk's pairs index their own slice of the logit scratch from 0
    a.mass_stride = mass_stride;
    a.head_stride = head_stride;
    a.Hkv = Hkv;
    a.n_splits = n_splits;
    a.n_dev = n_dev;
    a.n_host = n_host;
    a.n_cap = n_cap;
    a.c = (float)(1.4426950408889634 / sqrt((double)d));
    a.part = part;
    a.status = status;
    const cudaError_t e = d == 128 ? decode_dispatch_g<128>(a, G, nl * Hkv, stream)
                                   : decode_dispatch_g<64>(a, G, nl * Hkv, stream);
    if (e != cudaSuccess) {
      set_last_cuda_error(e);
      return STEPKV_ECUDA;
    }
  }
  return STEPKV_OK;
}

}  // namespace stepkv
