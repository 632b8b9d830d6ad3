// Stage 1 -- token saliency from the observation-window queries (Sec. 4.2 "Token Saliency";
// Table H: last 3 layers).  For layer l, KV head h, key j:
//   A[l,h,j] = (1/G) sum_{g in group(h)} sum_w softmax_{j' <= T-W+w}(q_{g,w} . k_{j'} / sqrt(d))[j]
//
// GB300 design.  The softmax normalises over keys while A sums over query rows, so the two
// reductions run in two tensor-core passes over K, each in the orientation that makes its
// reduction a per-thread loop over TMEM columns:
//   pass 1  S   = Q . K^T  (M = 128 query rows, N = 128 keys): per-row running max m and
//                 Z = sum 2^((s - m) c), c = log2(e)/sqrt(d); one partial (m, Z) per CTA segment;
//   pass 2  S^T = K . Q^T  (M = 128 keys, N = up to 256 query rows): per-key
//                 sum_r 2^(s c - off_r), off_r = m_r c + log2 Z_r combined from the pass-1 partials.
// K tiles are TMA-staged (128-byte swizzle) through an mbarrier ring; one thread issues tcgen05.mma
// into a double-buffered TMEM accumulator (2 x 256 columns); 8 epilogue warps read TMEM with
// tcgen05.ld and spend one MUFU ex2 per logit.  Each CTA (one per SM) owns a contiguous range of key
// tiles, so a (pair, row-group) unit has a few pass-1 partials that pass 2 combines in a fixed order
// (deterministic).  Pairs are launched in groups whose K fits in L2, so pass 2 re-reads K from L2.
#include <math.h>

#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace stepkv {

constexpr int kEpiWarps = 16;   // four warps per TMEM lane quarter
constexpr int kGroupWarps = 8;  // two epilogue groups, one per accumulator buffer (alternate tiles)
constexpr int kThreads = 64 + kEpiWarps * 32;  // warp 0: TMA producer, warp 1: MMA issuer + TMEM owner, rest: epilogue
constexpr int kKeyTile = 128;
constexpr int kMaxRows = 256;   // query rows per row group
constexpr int kTmemCols = 512;  // two accumulator buffers of 256 columns
constexpr int kQChunkBytes = kMaxRows * 128;   // one 64-wide d chunk of the Q staging area
constexpr int kKChunkBytes = kKeyTile * 128;   // one 64-wide d chunk of a K tile

struct ScoreGeom {
  int Hkv, Hq, G, d, T, W;
  int W_pad;         // W rounded up to 8 (each head's block starts on a 1024-byte swizzle atom)
  int split;         // 0: several whole heads per row group; 1: a head's window split over row groups
  int hpr;           // heads per row group (split == 0)
  int rph;           // row groups per head (split == 1)
  int n_rg;          // row groups per (layer, KV head) pair
  int n_tiles;       // ceil(T / 128)
  float c;           // log2(e) / sqrt(d)
  float inv_G;
};

struct ScoreLaunch {
  CUtensorMap tmK[kMaxSalLayers];
  CUtensorMap tmQ[kMaxSalLayers];
  ScoreGeom g;
  int n_layers;
  int pair0;          // first (layer*Hkv + head) pair of this launch
  int n_units;        // units = pairs of this launch x n_rg
  int tpc;            // tiles per CTA (contiguous range)
  float2* part;       // pass-1 partials: slot (unit + cta) x 256 rows
  float* out;         // pass-2 output rows: row (pair*n_rg + rg), stride out_stride (when t_acc == nullptr)
  int64_t out_stride;
  unsigned long long* t_acc;  // pass 2: per-token fixed-point sum over all (pair, row group) (when non-null)
  int acc_shift;      // k: fixed-point scale 2^k of t_acc
  int zero_acc;       // pass 1: zero t_acc[0..T) first (first launch of a compression pass)
  int32_t* status;
};

struct RowGroup {
  int g_first;   // first local query head (0..G-1) of this group
  int n_blk;     // head blocks
  int blk_rows;  // rows per block
  int w0;        // window offset of the block's first row
  int rows;      // n_blk * blk_rows (<= 256)
};

__host__ __device__ inline RowGroup row_group(const ScoreGeom& g, int rg) {
  RowGroup r;
  if (!g.split) {
    r.g_first = rg * g.hpr;
    r.n_blk = min(g.hpr, g.G - r.g_first);
    r.blk_rows = g.W_pad;
    r.w0 = 0;
  } else {
    r.g_first = rg / g.rph;
    r.n_blk = 1;
    r.w0 = (rg % g.rph) * kMaxRows;
    r.blk_rows = min(kMaxRows, g.W_pad - r.w0);
  }
  r.rows = r.n_blk * r.blk_rows;
  return r;
}

template <int PASS, int NCH>
struct ScoreCfg {
  // Pass 1 needs no shared tables, so it affords a fifth K stage (more bytes in flight per SM).
  static constexpr int kStages = PASS == 1 ? (NCH == 2 ? 5 : 10) : (NCH == 2 ? 4 : 8);
  static constexpr int kQBytes = NCH * kQChunkBytes;
  static constexpr int kStageBytes = NCH * kKChunkBytes;
  static constexpr int kOffOff = kQBytes + kStages * kStageBytes;             // pass 2: float sNegOff[2][256]
  static constexpr int kPwOff = kOffOff + (PASS == 2 ? 2 * kMaxRows * 4 : 0); // pass 2: int sPw[2][256]
  static constexpr int kCombOff = kPwOff + (PASS == 2 ? 2 * kMaxRows * 4 : 0);// pass 2: float[2][2][128]
  static constexpr int kBarOff = kCombOff + (PASS == 2 ? 2048 : 0);
  static constexpr int kNumBars = 2 * kStages + 2 + 4 + 2;
  static constexpr int kMiscOff = kBarOff + kNumBars * 8;                 // tmem base, abort flag
  static constexpr int kBytes = kMiscOff + 16;
  static constexpr int kDynSmem = kBytes + 1024;                          // + alignment slack
  static_assert(kDynSmem <= 232448, "shared memory budget");
};

// Pass-1 partial (m, Z) slots: one per (unit, CTA), each with 4 entries per row (one per warp that
// covers part of the row's keys).
constexpr int kPartEntries = 4;

// Bounded barrier among the 8 epilogue warps (an mbarrier with one arrival per warp).  Returns false
// if the CTA aborted or the wait limit passed.
__device__ __forceinline__ bool epi_sync(uint64_t* bar, uint32_t& phase, volatile int* abort_flag) {
  __syncwarp();
  if ((threadIdx.x & 31) == 0) mbar_arrive(bar);
  const bool ok = mbar_wait(bar, phase, abort_flag);
  phase ^= 1;
  __syncwarp();
  return ok;
}

__device__ __forceinline__ bool mbar_wait_drain(uint64_t* bar, uint32_t parity) {
  int zero = 0;
  return mbar_wait(bar, parity, &zero);
}

// Maximum of n consecutive values as a tree of 3-input max instructions (short dependency chain).
template <int N>
__device__ __forceinline__ float tree_max(const float* v) {
  if constexpr (N == 1) {
    return v[0];
  } else if constexpr (N == 2) {
    return fmaxf(v[0], v[1]);
  } else if constexpr (N == 3) {
    return fmax3(v[0], v[1], v[2]);
  } else {
    constexpr int A = N / 3, B = (N - A) / 2;
    return fmax3(tree_max<A>(v), tree_max<B>(v + A), tree_max<N - A - B>(v + A + B));
  }
}

// Pass 1: fold NCHUNK x 32 logits of one query row into its running (m, Z), Z = sum 2^((s - m) c).
template <int NCHUNK>
__device__ __forceinline__ void row_stats_update(const float (&va)[32], const float (&vb)[32], float c, float& m,
                                                 float& Z) {
  float mn = fmaxf(tree_max<32>(va), m);
  if (NCHUNK == 2) mn = fmaxf(mn, tree_max<32>(vb));
  if (mn == -INFINITY) return;
  const float nmc = -mn * c;
  const uint64_t c2 = f2_pack(c, c), b2 = f2_pack(nmc, nmc);
  uint64_t acc2[4] = {0ull, 0ull, 0ull, 0ull};
#pragma unroll
  for (int ch = 0; ch < NCHUNK; ++ch) {
    const float* v = ch == 0 ? va : vb;
#pragma unroll
    for (int i = 0; i < 32; i += 8) {
#pragma unroll
      for (int k2 = 0; k2 < 4; ++k2) {
        float lo, hi;
        f2_unpack(f2_fma(f2_pack(v[i + 2 * k2], v[i + 2 * k2 + 1]), c2, b2), lo, hi);
        acc2[k2] = f2_add(acc2[k2], f2_pack(ex2_approx(lo), ex2_approx(hi)));
      }
    }
  }
  float s0, s1, s2, s3, s4, s5, s6, s7;
  f2_unpack(acc2[0], s0, s1);
  f2_unpack(acc2[1], s2, s3);
  f2_unpack(acc2[2], s4, s5);
  f2_unpack(acc2[3], s6, s7);
  Z = Z * ex2_approx((m - mn) * c) + (((s0 + s1) + (s2 + s3)) + ((s4 + s5) + (s6 + s7)));
  m = mn;
}

// Pass 2: sum over 32 query columns of 2^(s c - off_r) for key j; columns whose causal limit pw_r is
// below j contribute nothing (only tiles that reach into the window need the test).
__device__ __forceinline__ float key_mass(const float (&v)[32], const float* negoff, const int* pw, int j,
                                          bool need_mask, float c) {
  if (!need_mask) {
    const uint64_t c2 = f2_pack(c, c);
    uint64_t acc2[4] = {0ull, 0ull, 0ull, 0ull};
#pragma unroll
    for (int i = 0; i < 32; i += 8) {
#pragma unroll
      for (int k2 = 0; k2 < 4; ++k2) {
        const float2 o = *reinterpret_cast<const float2*>(&negoff[i + 2 * k2]);
        float lo, hi;
        f2_unpack(f2_fma(f2_pack(v[i + 2 * k2], v[i + 2 * k2 + 1]), c2, f2_pack(o.x, o.y)), lo, hi);
        acc2[k2] = f2_add(acc2[k2], f2_pack(ex2_approx(lo), ex2_approx(hi)));
      }
    }
    float t0, t1, t2, t3, t4, t5, t6, t7;
    f2_unpack(acc2[0], t0, t1);
    f2_unpack(acc2[1], t2, t3);
    f2_unpack(acc2[2], t4, t5);
    f2_unpack(acc2[3], t6, t7);
    return ((t0 + t1) + (t2 + t3)) + ((t4 + t5) + (t6 + t7));
  }
  float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
#pragma unroll
  for (int i = 0; i < 32; i += 4) {
    const float4 o = *reinterpret_cast<const float4*>(&negoff[i]);
    const int4 w = *reinterpret_cast<const int4*>(&pw[i]);
    s0 += j <= w.x ? ex2_approx(fmaf(v[i + 0], c, o.x)) : 0.f;
    s1 += j <= w.y ? ex2_approx(fmaf(v[i + 1], c, o.y)) : 0.f;
    s2 += j <= w.z ? ex2_approx(fmaf(v[i + 2], c, o.z)) : 0.f;
    s3 += j <= w.w ? ex2_approx(fmaf(v[i + 3], c, o.w)) : 0.f;
  }
  return (s0 + s1) + (s2 + s3);
}

template <int PASS, int NCH>
__global__ void __launch_bounds__(kThreads, 1) score_kernel(const __grid_constant__ ScoreLaunch p) {
  using Cfg = ScoreCfg<PASS, NCH>;
  constexpr int S = Cfg::kStages;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = sm;
  uint8_t* sK = sm + Cfg::kQBytes;
  float* sNegOff = reinterpret_cast<float*>(sm + Cfg::kOffOff);
  int* sPw = reinterpret_cast<int*>(sm + Cfg::kPwOff);
  float2* sComb = reinterpret_cast<float2*>(sm + Cfg::kCombOff);
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + Cfg::kBarOff);
  uint64_t* k_full = bars;
  uint64_t* k_empty = bars + S;
  uint64_t* q_full = bars + 2 * S;
  uint64_t* q_empty = q_full + 1;
  uint64_t* acc_full = q_empty + 1;    // [2]
  uint64_t* acc_empty = acc_full + 2;  // [2]
  uint64_t* epi_bar = acc_empty + 2;  // [2], one per epilogue group
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sm + Cfg::kMiscOff);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(sm + Cfg::kMiscOff + 4);

  const ScoreGeom& g = p.g;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int U = p.n_units * g.n_tiles;
  const int t_lo = blockIdx.x * p.tpc;
  const int t_hi = min(U, t_lo + p.tpc);
  const int n_my = t_hi - t_lo;
  // Pass 2 walks the CTA's tile range backwards: the tiles pass 1 streamed last are still in L2.
  auto tile_at = [&](int k) { return PASS == 1 ? t_lo + k : t_hi - 1 - k; };

  if (threadIdx.x == 0) {
    for (int i = 0; i < S; ++i) {
      mbar_init(&k_full[i], 1);
      mbar_init(&k_empty[i], 1);
    }
    mbar_init(q_full, 1);
    mbar_init(q_empty, 1);
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], kGroupWarps);
    }
    mbar_init(&epi_bar[0], kGroupWarps);
    mbar_init(&epi_bar[1], kGroupWarps);
    *abort_flag = 0;
    mbar_fence_init();
  }
  if (warp == 0 && lane == 0) {
    for (int l = 0; l < p.n_layers; ++l) {
      tma_prefetch_desc(&p.tmK[l]);
      tma_prefetch_desc(&p.tmQ[l]);
    }
  }
  if (warp == 1) tmem_alloc(tmem_slot, kTmemCols);
  // Zero the Q staging area once: rows the TMA never writes (MMA padding) must hold finite values.
  for (int i = threadIdx.x; i < Cfg::kQBytes / 16; i += kThreads) reinterpret_cast<uint4*>(sQ)[i] = make_uint4(0, 0, 0, 0);
  fence_proxy_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  // Only shared memory, barriers and TMEM are set up before this point.  Every thread waits for the
  // earlier kernels on the stream before its first global access (a per-role wait placed later was
  // observed to let early-launched CTAs read pass-1 partials of the previous call).
  pdl_wait();
  pdl_launch_dependents();
  if (PASS == 1 && p.zero_acc) {
    for (int i = blockIdx.x * kThreads + threadIdx.x; i < g.T; i += gridDim.x * kThreads) p.t_acc[i] = 0ull;
  }

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer (one thread)
    if (lane == 0) {
      int stage = 0, cur = -1;
      uint32_t phase = 0, qe_phase = 0, q_issued = 0;
      uint32_t used = 0, last_par = 0;  // per-stage bit: loaded at least once / parity of its last load
      bool ok = true;
      for (int k = 0; k < n_my; ++k) {
        const int gt = tile_at(k);
        const int u = gt / g.n_tiles, tile = gt - u * g.n_tiles;
        const int pair = p.pair0 + u / g.n_rg, rg = u % g.n_rg;
        const int layer = pair / g.Hkv, h = pair - layer * g.Hkv;
        if (u != cur) {
          if (cur >= 0) {
            if (!mbar_wait(q_empty, qe_phase, abort_flag)) { ok = false; break; }
            qe_phase ^= 1;
          }
          const RowGroup r = row_group(g, rg);
          const int box_rows = min(g.W_pad, kMaxRows);
          mbar_arrive_expect_tx(q_full, (uint32_t)(r.n_blk * NCH * box_rows * 128));
          for (int b = 0; b < r.n_blk; ++b)
            for (int c = 0; c < NCH; ++c)
              tma_load_3d(sQ + c * kQChunkBytes + b * r.blk_rows * 128, &p.tmQ[layer], c * 64, r.w0,
                          h * g.G + r.g_first + b, q_full);
          ++q_issued;
          cur = u;
        }
        if (!mbar_wait(&k_empty[stage], phase ^ 1, abort_flag)) { ok = false; break; }
        mbar_arrive_expect_tx(&k_full[stage], (uint32_t)(NCH * kKChunkBytes));
        for (int c = 0; c < NCH; ++c)
          tma_load_3d(sK + stage * Cfg::kStageBytes + c * kKChunkBytes, &p.tmK[layer], c * 64, tile * kKeyTile, h,
                      &k_full[stage]);
        used |= 1u << stage;
        last_par = (last_par & ~(1u << stage)) | (phase << stage);
        if (++stage == S) { stage = 0; phase ^= 1; }
      }
      if (!ok) {
        *abort_flag = 1;
        record_status(p.status, STEPKV_ETIMEOUT);
      }
      // Drain: every copy this thread issued has landed before the CTA may exit.
      for (int i = 0; i < S; ++i)
        if (used >> i & 1u) mbar_wait_drain(&k_full[i], last_par >> i & 1u);
      if (q_issued) mbar_wait_drain(q_full, (q_issued - 1) & 1u);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer (one thread)
    if (lane == 0) {
      int stage = 0, buf = 0, cur = -1;
      uint32_t phase = 0, buf_phase = 0, q_phase = 0;
      bool issued = false, ok = true;
      int last_buf = 0;
      uint32_t last_buf_parity = 0;
      for (int k = 0; k < n_my; ++k) {
        const int u = tile_at(k) / g.n_tiles;
        const RowGroup r = row_group(g, u % g.n_rg);
        if (u != cur) {
          if (cur >= 0) umma_commit(q_empty);  // Q may be overwritten once the previous unit's MMAs finish
          if (!mbar_wait(q_full, q_phase, abort_flag)) { ok = false; break; }
          q_phase ^= 1;
          cur = u;
        }
        if (!mbar_wait(&acc_empty[buf], buf_phase ^ 1, abort_flag)) { ok = false; break; }
        if (!mbar_wait(&k_full[stage], phase, abort_flag)) { ok = false; break; }
        tc_fence_after();
        const uint32_t kst = smem_u32(sK + stage * Cfg::kStageBytes);
        const uint32_t qst = smem_u32(sQ);
        const uint32_t dcol = tmem_base + (uint32_t)(buf * 256);
        if (PASS == 1) {
          const int n_mt = r.rows > 128 ? 2 : 1;
          constexpr uint32_t idesc = umma_idesc_bf16(128, kKeyTile);
          for (int mt = 0; mt < n_mt; ++mt)
#pragma unroll
            for (int kk = 0; kk < NCH * 4; ++kk) {
              const uint32_t qoff = (uint32_t)((kk >> 2) * kQChunkBytes + mt * 128 * 128 + (kk & 3) * 32);
              const uint32_t koff = (uint32_t)((kk >> 2) * kKChunkBytes + (kk & 3) * 32);
              umma_bf16(dcol + (uint32_t)(mt * 128), umma_desc_sw128(qst + qoff), umma_desc_sw128(kst + koff), idesc,
                        kk > 0 ? 1u : 0u);
            }
        } else {
          const int n_mma = (r.rows + 31) & ~31;  // every TMEM column the epilogue loads is written
          const uint32_t idesc = umma_idesc_bf16(128, n_mma);
#pragma unroll
          for (int kk = 0; kk < NCH * 4; ++kk) {
            const uint32_t qoff = (uint32_t)((kk >> 2) * kQChunkBytes + (kk & 3) * 32);
            const uint32_t koff = (uint32_t)((kk >> 2) * kKChunkBytes + (kk & 3) * 32);
            umma_bf16(dcol, umma_desc_sw128(kst + koff), umma_desc_sw128(qst + qoff), idesc, kk > 0 ? 1u : 0u);
          }
        }
        umma_commit(&k_empty[stage]);
        umma_commit(&acc_full[buf]);
        issued = true;
        last_buf = buf;
        last_buf_parity = buf_phase;
        if (++stage == S) { stage = 0; phase ^= 1; }
        if (++buf == 2) { buf = 0; buf_phase ^= 1; }
      }
      if (!ok) {
        *abort_flag = 1;
        record_status(p.status, STEPKV_ETIMEOUT);
      }
      // Drain: the last MMA group has completed before TMEM is released.
      if (issued) mbar_wait_drain(&acc_full[last_buf], last_buf_parity);
    }
  } else {
    // ------------------------------------------------------------ epilogue (16 warps, 4 per lane quarter)
    // Two groups of 8 warps take alternate tiles (group g drains accumulator buffer g), so one group's
    // TMEM round trips and barrier waits overlap the other group's exponentials.  Within a group, two
    // warps share each TMEM lane quarter.
    const int ew = warp - 2;
    const int q = warp & 3;     // TMEM lane quarter this warp may access
    const int sub = ew >> 2;    // 0..3
    const int grp = sub >> 1;   // epilogue group = accumulator buffer
    const int s2 = sub & 1;     // which of the group's two warps on this quarter
    const float c = g.c;
    int cur = -1;
    uint32_t acc_phase = 0, eb_phase = 0;
    RowGroup r{};
    float m = -INFINITY, Z = 0.f;  // pass 1: running statistics of this thread's row over its columns
    int my_row = 0, my_pw = 0, my_e = 0;
    bool row_ok = false, two = false, ok = true;
    float* negoff = sNegOff + grp * kMaxRows;  // pass 2: this group's per-row offsets and causal limits
    int* pw_tab = sPw + grp * kMaxRows;
    float* combf = reinterpret_cast<float*>(sComb) + grp * (2 * 128);  // pass 2 rows output: [2 parity][128]
    int n_done = 0;                                                     // tiles this group has drained
    const uint32_t lane_base = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(grp * 256);

    // pass 1: this warp's (m, Z) over its share of the row's keys becomes entry my_e of the CTA's partial
    auto flush_partial = [&](int u) {
      p.part[((size_t)(u + (int)blockIdx.x) * kPartEntries + my_e) * kMaxRows + my_row] = make_float2(m, Z);
    };
    auto release_buffer = [&]() {
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acc_empty[grp]);
    };

    for (int k = 0; k < n_my && ok; ++k) {
      const int gt = tile_at(k);
      const int u = gt / g.n_tiles, tile = gt - u * g.n_tiles;
      if (PASS == 1 && u != cur) {
        // Every group flushes every unit the CTA touches (an untouched share flushes m = -inf, Z = 0),
        // so each of the unit's partial entries is written.
        if (cur >= 0) flush_partial(cur);
        r = row_group(g, u % g.n_rg);
        two = r.rows > 128;
        my_row = (two ? s2 * 128 : 0) + q * 32 + lane;
        my_e = two ? grp : grp * 2 + s2;
        const int w = r.w0 + my_row % r.blk_rows;
        row_ok = my_row < r.rows && w < g.W;
        my_pw = g.T - g.W + w;
        m = -INFINITY;
        Z = 0.f;
        cur = u;
      }
      if ((k & 1) != grp) continue;
      if (PASS == 2 && u != cur) {
        // Combine the pass-1 partials of unit u into this group's per-row offsets, in contributing-CTA
        // order (the group no longer reads the previous unit's offsets once all its warps arrive).
        if (!(ok = epi_sync(&epi_bar[grp], eb_phase, abort_flag))) break;
        r = row_group(g, u % g.n_rg);
        const int c0 = (u * g.n_tiles) / p.tpc;
        const int c1 = (u * g.n_tiles + g.n_tiles - 1) / p.tpc;
        const int n_e = r.rows > 128 ? 2 : kPartEntries;  // entries written per row in pass 1
        const int row = (ew & 7) * 32 + lane;             // 256 threads of the group, one row each
        const int w = r.w0 + row % r.blk_rows;
        const bool valid = row < r.rows && w < g.W;
        float off = INFINITY;
        if (valid) {
          float M = -INFINITY;
          for (int ci = c0; ci <= c1; ++ci)
            for (int e = 0; e < n_e; ++e)
              M = fmaxf(M, __ldcg(&p.part[((size_t)(u + ci) * kPartEntries + e) * kMaxRows + row]).x);
          float Zs = 0.f;
          for (int ci = c0; ci <= c1; ++ci)
            for (int e = 0; e < n_e; ++e) {
              const float2 pz = __ldcg(&p.part[((size_t)(u + ci) * kPartEntries + e) * kMaxRows + row]);
              if (pz.x != -INFINITY) Zs += pz.y * ex2_approx((pz.x - M) * c);
            }
          off = M * c + __log2f(Zs);
        }
        negoff[row] = -off;
        pw_tab[row] = valid ? g.T - g.W + w : -1;
        if (!(ok = epi_sync(&epi_bar[grp], eb_phase, abort_flag))) break;
        cur = u;
      }
      if (!(ok = mbar_wait(&acc_full[grp], acc_phase, abort_flag))) break;
      acc_phase ^= 1;
      tc_fence_after();
      const int key0 = tile * kKeyTile;
      const bool need_mask = key0 + kKeyTile - 1 > g.T - g.W;  // tile reaches into the causal window
      if (PASS == 1) {
        // Queries on the TMEM lanes.  Above 128 rows warp s2 takes M-tile s2 (128 columns = all 128 keys
        // of the tile); otherwise the two warps split the 128 columns (keys) in halves.
        const uint32_t col0 = two ? (uint32_t)(s2 * 128) : (uint32_t)(s2 * 64);
        const int kofs = two ? 0 : s2 * 64;
        const int n_pairs_ch = two ? 2 : 1;  // pairs of 32-column chunks
#pragma unroll 1
        for (int h2 = 0; h2 < n_pairs_ch; ++h2) {
          float va[32], vb[32];
          tmem_ld32x2(lane_base + col0 + (uint32_t)(h2 * 64), lane_base + col0 + (uint32_t)(h2 * 64 + 32), va, vb);
          if (h2 == n_pairs_ch - 1) release_buffer();
          if (row_ok) {
            const int j0 = key0 + kofs + h2 * 64;
            if (need_mask) {
#pragma unroll
              for (int i = 0; i < 32; ++i) {
                va[i] = (j0 + i <= my_pw) ? va[i] : -INFINITY;
                vb[i] = (j0 + 32 + i <= my_pw) ? vb[i] : -INFINITY;
              }
            }
            row_stats_update<2>(va, vb, c, m, Z);
          }
        }
      } else {
        // Keys on the TMEM lanes: this warp sums its key's mass over query columns s2*32 + 64 i, one
        // 32-column chunk at a time (holding two chunks in registers spills).  The buffer is released
        // once the warp's last chunk is in registers.
        const int n_cols = (r.rows + 31) & ~31;
        const int j = key0 + q * 32 + lane;
        float acc = 0.f;
        bool released = false;
#pragma unroll 1
        for (int cc = s2 * 32; cc < n_cols; cc += 64) {
          float v[32];
          tmem_ld32(lane_base + (uint32_t)cc, v);
          if (cc + 64 >= n_cols) {
            release_buffer();
            released = true;
          }
          acc += key_mass(v, negoff + cc, pw_tab + cc, j, need_mask, c);
        }
        if (!released) release_buffer();
        if (p.t_acc) {
          // fused pass: each warp adds its share of the rows straight into the per-token fixed-point
          // sum (integer addition: the total does not depend on the order of arrival)
          if (j < g.T) atomicAdd(&p.t_acc[j], to_fixed(acc * g.inv_G, p.acc_shift));
        } else {
          // saliency rows: the group's two warps on this quarter combine in a fixed order (the slot
          // alternates between the group's tiles, so a write never meets a pending read)
          float* comb = combf + (n_done & 1) * 128;
          if (s2 == 1) comb[q * 32 + lane] = acc;
          if (!(ok = epi_sync(&epi_bar[grp], eb_phase, abort_flag))) break;
          if (s2 == 0 && j < g.T) {
            const float val = (acc + comb[q * 32 + lane]) * g.inv_G;
            const int pair = p.pair0 + u / g.n_rg, rg = u % g.n_rg;
            p.out[(size_t)(pair * g.n_rg + rg) * p.out_stride + j] = val;
          }
        }
      }
      ++n_done;
    }
    if (PASS == 1 && ok && cur >= 0) flush_partial(cur);
    if (!ok) {
      *abort_flag = 1;
      record_status(p.status, STEPKV_ETIMEOUT);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
}

// -------------------------------------------------------------------------------------------------
// Sum of row-group partial rows into the [n_pairs][T] saliency output (only needed when n_rg > 1).
__global__ void sum_row_groups_kernel(const float* __restrict__ rows, int n_pairs, int n_rg, int T,
                                      float* __restrict__ sal) {
  pdl_wait();
  pdl_launch_dependents();
  const int64_t n = (int64_t)n_pairs * T;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t pair = i / T, j = i - pair * T;
    float s = 0.f;
    for (int rg = 0; rg < n_rg; ++rg) s += rows[(pair * n_rg + rg) * T + j];
    sal[i] = s;
  }
}

// -------------------------------------------------------------------------------------------------
// Host side
static ScoreGeom make_geom(int Hkv, int Hq, int d, int T, int W) {
  ScoreGeom g;
  memset(&g, 0, sizeof(g));
  g.Hkv = Hkv;
  g.Hq = Hq;
  g.G = Hq / Hkv;
  g.d = d;
  g.T = T;
  g.W = W;
  g.W_pad = (W + 7) & ~7;
  if (g.W_pad <= kMaxRows) {
    g.split = 0;
    g.hpr = kMaxRows / g.W_pad;
    g.rph = 1;
    g.n_rg = (g.G + g.hpr - 1) / g.hpr;
  } else {
    g.split = 1;
    g.hpr = 1;
    g.rph = (g.W_pad + kMaxRows - 1) / kMaxRows;
    g.n_rg = g.G * g.rph;
  }
  g.n_tiles = (T + kKeyTile - 1) / kKeyTile;
  g.c = (float)(1.4426950408889634 / sqrt((double)d));
  g.inv_G = 1.0f / (float)g.G;
  return g;
}

int score_row_groups(int Hkv, int Hq, int W) { return make_geom(Hkv, Hq, 64, W, W).n_rg; }

// Fixed-point shift for the per-token sum over (layer, KV head) pairs: each pair contributes at most W
// (a softmax row sums to one; W rows per query head, mean over the group), so the sum of n_pairs
// contributions stays below 2^60 with scale 2^shift.
int score_acc_shift(int n_pairs, int W) {
  const double bound = (double)n_pairs * (double)W;
  int e = 0;
  while (ldexp(1.0, e) < bound) ++e;
  return 60 - e;
}

size_t score_partial_bytes(int n_layers, int Hkv, int Hq, int W) {
  const int n_rg = score_row_groups(Hkv, Hq, W);
  return (size_t)(n_layers * Hkv * n_rg + kMaxGrid) * kPartEntries * kMaxRows * sizeof(float2);
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn get_encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(f);
  }
  return fn;
}

// 3-D bf16 tensor map over [heads][rows][d] with a 64 x box_rows x 1 box and 128-byte swizzle.
static bool encode_3d(CUtensorMap* map, const void* base, int d, int rows, int heads, int64_t head_stride,
                      int box_rows) {
  EncodeTiledFn enc = get_encode_fn();
  if (!enc) return false;
  cuuint64_t dims[3] = {(cuuint64_t)d, (cuuint64_t)rows, (cuuint64_t)heads};
  cuuint64_t strides[2] = {(cuuint64_t)d * 2, (cuuint64_t)head_stride * 2};
  cuuint32_t box[3] = {64, (cuuint32_t)box_rows, 1};
  cuuint32_t es[3] = {1, 1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, es,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int PASS, int NCH>
static cudaError_t launch_pass(const ScoreLaunch& L, int grid, cudaStream_t stream) {
  using Cfg = ScoreCfg<PASS, NCH>;
  void (*kern)(ScoreLaunch) = score_kernel<PASS, NCH>;
  cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(kern), Cfg::kDynSmem);
  if (e != cudaSuccess) return e;
  return launch_kernel(kern, dim3(grid), dim3(kThreads), Cfg::kDynSmem, stream, L);
}

stepkv_status_t score_run(int n_layers, const void* const* K, int64_t k_head_stride, const void* const* Q,
                          int64_t q_head_stride, int Hkv, int Hq, int d, int T, int W, float* rows_out,
                          int64_t out_stride, unsigned long long* t_acc, int acc_shift, float2* part, int32_t* status,
                          cudaStream_t stream) {
  const ScoreGeom g = make_geom(Hkv, Hq, d, T, W);
  ScoreLaunch L;
  memset(&L, 0, sizeof(L));
  L.g = g;
  L.n_layers = n_layers;
  L.part = part;
  L.out = rows_out;
  L.out_stride = out_stride;
  L.t_acc = t_acc;
  L.acc_shift = acc_shift;
  L.status = status;
  const int box_rows = std::min(g.W_pad, kMaxRows);
  for (int l = 0; l < n_layers; ++l) {
    if (!encode_3d(&L.tmK[l], K[l], d, T, Hkv, k_head_stride, kKeyTile)) return STEPKV_ECUDA;
    if (!encode_3d(&L.tmQ[l], Q[l], d, W, Hq, q_head_stride, box_rows)) return STEPKV_ECUDA;
  }
  int n_sm = 0;
  cudaError_t e = device_sm_count(&n_sm);
  if (e != cudaSuccess) { set_last_cuda_error(e); return STEPKV_ECUDA; }
  const int grid_cap = std::max(1, std::min(n_sm, kMaxGrid));
  // all (layer, KV head) pairs in one launch per pass
  const int n_pairs = n_layers * Hkv;
  const int ppg = n_pairs;
  for (int p0 = 0; p0 < n_pairs; p0 += ppg) {
    const int np = std::min(ppg, n_pairs - p0);
    L.pair0 = p0;
    L.zero_acc = (t_acc != nullptr && p0 == 0) ? 1 : 0;
    L.n_units = np * g.n_rg;
    const int U = L.n_units * g.n_tiles;
    const int grid0 = std::min(grid_cap, U);
    L.tpc = (U + grid0 - 1) / grid0;
    const int grid = (U + L.tpc - 1) / L.tpc;
    e = d == 128 ? launch_pass<1, 2>(L, grid, stream) : launch_pass<1, 1>(L, grid, stream);
    if (e == cudaSuccess) e = d == 128 ? launch_pass<2, 2>(L, grid, stream) : launch_pass<2, 1>(L, grid, stream);
    if (e != cudaSuccess) { set_last_cuda_error(e); return STEPKV_ECUDA; }
  }
  return STEPKV_OK;
}

stepkv_status_t score_sum_row_groups(const float* rows, int n_pairs, int n_rg, int T, float* sal,
                                     cudaStream_t stream) {
  const int64_t n = (int64_t)n_pairs * T;
  const int blocks = (int)std::min<int64_t>((n + 255) / 256, 4096);
  cudaError_t e = launch_kernel(sum_row_groups_kernel, dim3(blocks), dim3(256), 0, stream, rows, n_pairs, n_rg, T, sal);
  if (e != cudaSuccess) { set_last_cuda_error(e); return STEPKV_ECUDA; }
  return STEPKV_OK;
}

}  // namespace stepkv
