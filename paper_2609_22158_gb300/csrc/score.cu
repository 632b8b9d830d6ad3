// Stage 1 -- token saliency from the observation-window queries (Sec. 4.2 "Token Saliency";
// Table H: last 3 layers).  For layer l, KV head h, key j:
//   A[l,h,j] = (1/G) sum_{g in group(h)} sum_w softmax_{j' <= T-W+w}(q_{g,w} . k_{j'} / sqrt(d))[j]
//
// GB300 design.  The softmax normalises over keys while A sums over query rows, so the two
// reductions run in two tensor-core passes over K, each in the orientation that makes its
// reduction a per-thread loop over TMEM columns:
//   pass 1  S   = Q . K^T  (M = 128 query rows, N = 256 keys): per-row reference point m (a running
//                 maximum, moved only when a chunk would overflow) and Z = sum 2^((s - m) c),
//                 c = log2(e)/sqrt(d); one partial (m, Z) per CTA segment;
//   pass 2  S^T = K . Q^T  (M = 128 keys, N = up to 256 query rows): per-key
//                 sum_r 2^(s c - off_r), off_r = m_r c + log2 Z_r combined from the pass-1 partials.
// Both passes run in one cooperative launch.  Each CTA (one per SM) owns a contiguous range of
// (unit, key tile) items, unit = (layer, KV head, row group); it streams them forward for pass 1 and
// backward for pass 2, so pass 2 starts on the tiles pass 1 left in L2 and on the Q already staged.
// K tiles are TMA-staged (128-byte swizzle) through an mbarrier ring; one thread issues tcgen05.mma
// into a double-buffered TMEM accumulator (2 x 256 columns); 16 epilogue warps in two groups (one per
// accumulator buffer, alternate items) read TMEM with tcgen05.ld and spend one MUFU ex2 per logit.
// A unit has a few pass-1 partials (one set per contributing CTA); the pass-2 epilogue combines them
// in a fixed order (deterministic) once the CTAs that cover the unit have raised their pass-1 flags.
#include <math.h>

#include <algorithm>
#include <vector>
#include <atomic>
#include <chrono>

#include "common.cuh"
#include "fastdiv.h"
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
  // the divisors of the per-tile bookkeeping, as multiply-and-shift dividers
  FastDiv rg_div;    // n_rg
  FastDiv hkv_div;   // Hkv
  FastDiv rph_div;   // rph
};

// One trajectory of a batched launch: its items are [item_off, item_off + units_per * n_tiles).
struct ScoreTraj {
  int T;
  int n_tiles;                 // ceil(T / 128)
  FastDiv nt_div;              // n_tiles
  int item_off;
  unsigned long long* t_acc;   // pass 2: per-token fixed-point sum (when the launch accumulates)
};

struct ScoreLaunch {
  CUtensorMap tmK[kMaxScoreMaps];  // [traj * n_layers + layer]
  CUtensorMap tmQ[kMaxScoreMaps];
  ScoreTraj traj[kMaxScoreBatch];
  ScoreGeom g;                     // shared head geometry (T, n_tiles: see traj)
  int n_traj;
  int n_layers;
  int pair0;          // first (layer*Hkv + head) pair of this launch (rows output)
  int units_per;      // units per trajectory = n_layers x Hkv x n_rg
  int n_items;        // items of all trajectories
  int cta_first[kMaxGrid + 1];  // CTA b owns items [cta_first[b], cta_first[b + 1])
  FastDiv units_div;  // units_per
  float2* part;       // pass-1 partials: slot (unit + cta) x 256 rows
  float* out;         // pass-2 output rows: row (pair*n_rg + rg), stride out_stride (when not accumulating)
  int64_t out_stride;
  int accumulate;     // 1: pass 2 adds into each trajectory's t_acc (zeroed first) instead of writing rows
  int acc_shift;      // k: fixed-point scale 2^k of t_acc
  unsigned long long* flags;  // [grid] pass-1-done flags: CTA b stores the launch token once its partials are written
  unsigned long long* zflags; // [grid] CTA b stores the launch token once its share of the accumulators is zeroed
  unsigned long long* epoch;  // per-workspace launch counter, advanced by CTA 0 at the end of every launch
  unsigned long long token;   // host value, unique per call; mixed with the epoch into the launch token
  int selftest;               // 1: the pass-2 wait looks for a value no CTA publishes (failure-path self-test)
  int pass2_only;             // 1: the row statistics come from the caller (lse), pass 1 is skipped
  const float* lse[kMaxScoreMaps];  // [traj * n_layers + layer]: [Hq][W] natural-log row log-sum-exp
  unsigned long long wait_limit_ns;  // the pass-2 wait gives up (STEPKV_ETIMEOUT) after this long
  int32_t* status;
};

static_assert(sizeof(ScoreLaunch) <= 32000, "kernel parameter space");

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
    int w_blk;
    r.g_first = fdivmod(rg, g.rph_div, w_blk);
    r.n_blk = 1;
    r.w0 = w_blk * kMaxRows;
    r.blk_rows = min(kMaxRows, g.W_pad - r.w0);
  }
  r.rows = r.n_blk * r.blk_rows;
  return r;
}

// Where global item t of a launch sits: trajectory b, local unit ul (global unit b * units_per + ul),
// key tile of the unit.
struct ItemLoc {
  int b, ul, u, tile;
};
__device__ __forceinline__ ItemLoc locate(const ScoreLaunch& p, int t) {
  int b = 0;
  while (b + 1 < p.n_traj && p.traj[b + 1].item_off <= t) ++b;
  const int local = t - p.traj[b].item_off;
  ItemLoc r;
  r.b = b;
  r.ul = fdivmod(local, p.traj[b].nt_div, r.tile);
  r.u = b * p.units_per + r.ul;
  return r;
}
// First item of global unit u.
__device__ __forceinline__ int unit_first_item(const ScoreLaunch& p, int u) {
  int ul;
  const int b = fdivmod(u, p.units_div, ul);
  return p.traj[b].item_off + ul * p.traj[b].n_tiles;
}

// The CTA whose item range holds item t (binary search over the ranges' first items).
__device__ __forceinline__ int cta_of_item(const ScoreLaunch& p, int t) {
  int lo = 0, hi = (int)gridDim.x - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (p.cta_first[mid] <= t) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

// Shared memory of the kernel.
template <int NCH>
struct ScoreCfg {
  // Pass 1 streams pairs of key tiles: a slot is two stages whose chunks sit side by side, so one
  // N = 256 MMA reads 256 consecutive keys.  Pass 2 streams single tiles through kStages2 stages.
  static constexpr int kSlots1 = NCH == 2 ? 2 : 5;
  static constexpr int kStages2 = NCH == 2 ? 4 : 10;
  static constexpr int kStages = 2 * kSlots1 > kStages2 ? 2 * kSlots1 : kStages2;
  static constexpr int kQBytes = NCH * kQChunkBytes;
  static constexpr int kStageBytes = NCH * kKChunkBytes;
  static constexpr int kTabOff = kQBytes + kStages * kStageBytes;     // float negoff[2][256] | int pw[2][256]
  static constexpr int kCombOff = kTabOff + 2 * 2 * kMaxRows * 4;    // | float comb[2 grp][2 parity][128]
  static constexpr int kBarOff = kCombOff + 2 * 2 * 128 * 4;
  // k_full/k_empty per stage, q_full/q_empty, acc_full/acc_empty[2], epi[2], p1_flushed
  static constexpr int kNumBars = 2 * kStages + 2 + 4 + 2 + 1;
  static constexpr int kMiscOff = kBarOff + kNumBars * 8;                 // tmem base, abort flag
  static constexpr int kBytes = kMiscOff + 16;
  static constexpr int kDynSmem = kBytes + 1024;                          // + alignment slack
  static_assert(kDynSmem <= 232448, "shared memory budget");
  static_assert(kStages % 2 == 0, "stages come in pairs");
  // Byte offset (from the first stage) of chunk c of stage s: stages 2i and 2i+1 hold their chunk c
  // back to back, 256 consecutive keys.
  __host__ __device__ static constexpr int chunk_off(int s, int c) {
    return (s >> 1) * 2 * kStageBytes + c * 2 * kKChunkBytes + (s & 1) * kKChunkBytes;
  }
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

// Sum over NCHUNK x 32 logits of one query row of 2^((s - ref) c).
template <int NCHUNK>
__device__ __forceinline__ float chunk_sum(const float (&va)[32], const float (&vb)[32], float c, float ref) {
  const float nmc = -ref * c;
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
  return ((s0 + s1) + (s2 + s3)) + ((s4 + s5) + (s6 + s7));
}

// Pass 1: fold NCHUNK x 32 logits of one query row into its running (m, Z), Z = sum 2^((s - m) c).
// m is a reference point, not necessarily the maximum: any m that keeps every term below fp32
// overflow gives the same m c + log2 Z.  A chunk is summed against the current m and kept if the sum
// stays below 2^60; only the row's first chunk and a chunk with a logit far above m (sum >= 2^60,
// inf or nan) take the running maximum as the new m, so the per-chunk maximum is almost never needed.
template <int NCHUNK>
__device__ __forceinline__ void row_stats_update(const float (&va)[32], const float (&vb)[32], float c, float& m,
                                                 float& Z) {
  if (m != -INFINITY) {
    const float s = chunk_sum<NCHUNK>(va, vb, c, m);
    if (s < 0x1p60f) {
      Z += s;
      return;
    }
  }
  float mn = fmaxf(tree_max<32>(va), m);
  if (NCHUNK == 2) mn = fmaxf(mn, tree_max<32>(vb));
  if (mn == -INFINITY) return;  // every logit so far masked
  Z = Z * ex2_approx((m - mn) * c) + chunk_sum<NCHUNK>(va, vb, c, mn);
  m = mn;
}

// Pass 2: one 32-column chunk of a warp's 32 keys, read with two 16x256b loads (ra: the quarter's lanes
// 0-15, rb: lanes 16-31).  Register 4k + e of a load holds lane lane/4 + 8 (e >= 2) and column
// 8k + 2 (lane % 4) + (e & 1), so a thread sees 4 keys, lane/4 + 8 kk (kk < 4), and 8 columns of the
// chunk, whose offsets o2[k] (pairs of columns) it loaded from the unit's table.  acc2[kk] collects
// 2^(s c - off_r) over those columns for key kk in pairs; columns whose causal limit pw_r is below the
// key contribute nothing (only tiles that reach into the window need the test, jq = key of kk = 0).
__device__ __forceinline__ void chunk_mass(const uint32_t (&ra)[16], const uint32_t (&rb)[16], const uint64_t (&o2)[4],
                                           const int* pw, int jq, bool need_mask, float c, uint64_t (&acc2)[4]) {
  if (!need_mask) {
    const uint64_t c2 = f2_pack(c, c);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        const uint32_t* r = kk < 2 ? ra : rb;
        const int e = 4 * k + (kk & 1) * 2;
        float lo, hi;
        f2_unpack(f2_fma(f2_pack(__uint_as_float(r[e]), __uint_as_float(r[e + 1])), c2, o2[k]), lo, hi);
        acc2[kk] = f2_add(acc2[kk], f2_pack(ex2_approx(lo), ex2_approx(hi)));
      }
    }
    return;
  }
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const int2 w = *reinterpret_cast<const int2*>(&pw[8 * k]);
    float ox, oy;
    f2_unpack(o2[k], ox, oy);
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      const uint32_t* r = kk < 2 ? ra : rb;
      const int e = 4 * k + (kk & 1) * 2;
      const int jk = jq + 8 * kk;
      const float t0 = jk <= w.x ? ex2_approx(fmaf(__uint_as_float(r[e]), c, ox)) : 0.f;
      const float t1 = jk <= w.y ? ex2_approx(fmaf(__uint_as_float(r[e + 1]), c, oy)) : 0.f;
      acc2[kk] = f2_add(acc2[kk], f2_pack(t0, t1));
    }
  }
}

__device__ __forceinline__ unsigned long long ld_relaxed_u64(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void fence_acquire_gpu() { asm volatile("fence.acq_rel.gpu;" ::: "memory"); }
__device__ __forceinline__ void st_release_u64(unsigned long long* p, unsigned long long v) {
  asm volatile("st.release.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}

// The launch token every CTA publishes in its flags.  It mixes the host's per-call value with the
// workspace's epoch, which CTA 0 advances at the end of each launch, so a launch replayed from a CUDA
// graph (same host value) still differs from the launch before it, and flags left in the workspace by
// earlier launches never match.  All CTAs read the epoch after the stream's earlier work is complete
// and before CTA 0 can advance it: CTA 0 advances it only after every CTA has published its zero flag.
__device__ __forceinline__ unsigned long long launch_token(const ScoreLaunch& p) {
  const unsigned long long e = ld_relaxed_u64(p.epoch);
  const unsigned long long t = p.token ^ ((e + 1ull) * 0x9E3779B97F4A7C15ull);
  return t == 0ull ? 1ull : t;
}

// Both passes in one launch.  A CTA owns a contiguous range of (unit, key tile) items; it streams them
// forward for pass 1 (in pairs of tiles: one N = 256 MMA per query half) and backward for pass 2, so
// the TMA ring, the MMA issuer and the Q staging run on without a break at the change of pass (the
// first pass-2 tile is the last pass-1 tile, same Q).  Only the pass-2 epilogue depends on other CTAs:
// each unit starts once the CTAs covering it have published their pass-1 partials (a flag per CTA set
// to this launch's token; the launch is cooperative, so all CTAs are resident and the wait ends, else it
// gives up after the wait limit).
//
// Accumulator work is counted in "halves": a pass-1 pair item gives one half per 128-row query tile,
// a pass-2 item one half.  Half h goes to TMEM buffer h & 1 and is drained by epilogue group h & 1.
template <int NCH>
__global__ void __launch_bounds__(kThreads, 1) score_kernel(const __grid_constant__ ScoreLaunch p) {
  using Cfg = ScoreCfg<NCH>;
  constexpr int S2 = Cfg::kStages2, P1 = Cfg::kSlots1;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = sm;
  uint8_t* sK = sm + Cfg::kQBytes;
  float* sNegOff = reinterpret_cast<float*>(sm + Cfg::kTabOff);
  int* sPw = reinterpret_cast<int*>(sm + Cfg::kTabOff + 2 * kMaxRows * 4);
  float* sComb = reinterpret_cast<float*>(sm + Cfg::kCombOff);
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + Cfg::kBarOff);
  uint64_t* k_full = bars;
  uint64_t* k_empty = bars + Cfg::kStages;
  uint64_t* q_full = bars + 2 * Cfg::kStages;
  uint64_t* q_empty = q_full + 1;
  uint64_t* acc_full = q_empty + 1;    // [2]
  uint64_t* acc_empty = acc_full + 2;  // [2]
  uint64_t* epi_bar = acc_empty + 2;   // [2], one per epilogue group
  uint64_t* p1_flushed = epi_bar + 2;  // every epilogue warp has written its pass-1 partials
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sm + Cfg::kMiscOff);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(sm + Cfg::kMiscOff + 4);

  const ScoreGeom& g = p.g;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int U = p.n_items;
  const int t_lo = p.cta_first[blockIdx.x];
  const int t_hi = min(U, p.cta_first[blockIdx.x + 1]);
  const int n1 = max(0, t_hi - t_lo);  // tiles of the CTA (each is streamed once per pass)
  // Pass-1 items: two consecutive tiles of one unit where possible, else one.
  auto item_tiles = [&](const ItemLoc& l, int t) {
    return (t + 1 < t_hi && l.tile + 1 < p.traj[l.b].n_tiles) ? 2 : 1;
  };

  if (threadIdx.x == 0) {
    for (int i = 0; i < Cfg::kStages; ++i) {
      mbar_init(&k_full[i], 1);
      mbar_init(&k_empty[i], 1);
    }
    mbar_init(q_full, 1);
    mbar_init(q_empty, 1);
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], kGroupWarps);
      mbar_init(&epi_bar[b], kGroupWarps);
    }
    mbar_init(p1_flushed, kEpiWarps);
    *abort_flag = 0;
    mbar_fence_init();
  }
  if (warp == 0 && lane == 0) {
    for (int l = 0; l < p.n_traj * p.n_layers; ++l) {
      tma_prefetch_desc(&p.tmK[l]);
      tma_prefetch_desc(&p.tmQ[l]);
    }
  }
  if (warp == 1) tmem_alloc(tmem_slot, kTmemCols);
  // Zero the Q staging area once: rows the TMA never writes (MMA padding) must hold finite values.
  for (int i = threadIdx.x; i < Cfg::kQBytes / 16; i += kThreads) reinterpret_cast<uint4*>(sQ)[i] = make_uint4(0, 0, 0, 0);
  fence_proxy_async_smem();

  // Every thread waits for the earlier kernels on the stream before its first global access.
  pdl_wait();
  pdl_launch_dependents();
  const unsigned long long tok = launch_token(p);
  const unsigned long long wait_tok = p.selftest ? ~tok : tok;
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer (one thread)
    if (lane == 0) {
      int cur = -1;
      uint32_t qe_phase = 0, q_issued = 0;
      uint32_t par = 0, used = 0;  // per stage: parity of its next use / loaded at least once
      bool ok = true;
      auto load_tile = [&](int gt, int st) -> bool {
        const ItemLoc il = locate(p, gt);
        const int u = il.u, tile = il.tile;
        int rg, h;
        const int pair = p.pair0 + fdivmod(il.ul, g.rg_div, rg);
        const int layer = fdivmod(pair, g.hkv_div, h);
        const int map = il.b * p.n_layers + layer;
        if (u != cur) {
          if (cur >= 0) {
            if (!mbar_wait(q_empty, qe_phase, abort_flag)) return false;
            qe_phase ^= 1;
          }
          const RowGroup r = row_group(g, rg);
          const int box_rows = min(g.W_pad, kMaxRows);
          mbar_arrive_expect_tx(q_full, (uint32_t)(r.n_blk * NCH * box_rows * 128));
          for (int b = 0; b < r.n_blk; ++b)
            for (int c = 0; c < NCH; ++c)
              tma_load_3d(sQ + c * kQChunkBytes + b * r.blk_rows * 128, &p.tmQ[map], c * 64, r.w0,
                          h * g.G + r.g_first + b, q_full);
          ++q_issued;
          cur = u;
        }
        const uint32_t ph = (par >> st) & 1u;
        if (!mbar_wait(&k_empty[st], ph ^ 1u, abort_flag)) return false;
        mbar_arrive_expect_tx(&k_full[st], (uint32_t)(NCH * kKChunkBytes));
        for (int c = 0; c < NCH; ++c)
          tma_load_3d(sK + Cfg::chunk_off(st, c), &p.tmK[map], c * 64, tile * kKeyTile, h, &k_full[st]);
        used |= 1u << st;
        par ^= 1u << st;
        return true;
      };
      int slot = 0;
      for (int t = p.pass2_only ? t_hi : t_lo; t < t_hi && ok;) {
        const int nt = item_tiles(locate(p, t), t);
        for (int i = 0; i < nt && ok; ++i) ok = load_tile(t + i, 2 * slot + i);
        t += nt;
        if (++slot == P1) slot = 0;
      }
      for (int k = 0; k < n1 && ok; ++k) ok = load_tile(t_hi - 1 - k, k % S2);
      if (!ok) {
        *abort_flag = 1;
        record_status(p.status, STEPKV_ETIMEOUT);
      }
      // Drain: every copy this thread issued has landed before the CTA may exit.
      for (int i = 0; i < Cfg::kStages; ++i)
        if (used >> i & 1u) mbar_wait_drain(&k_full[i], ((par >> i) & 1u) ^ 1u);
      if (q_issued) mbar_wait_drain(q_full, (q_issued - 1) & 1u);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer (one thread)
    if (lane == 0) {
      int cur = -1;
      uint32_t par = 0, buf_par = 0, q_phase = 0;  // per stage / per accumulator buffer: use parity
      uint32_t hh = 0;                              // halves issued so far
      bool ok = true;
      const uint32_t qst = smem_u32(sQ);
      auto new_unit = [&](int u) -> bool {
        if (u == cur) return true;
        if (cur >= 0) umma_commit(q_empty);  // Q may be overwritten once the previous unit's MMAs finish
        if (!mbar_wait(q_full, q_phase, abort_flag)) return false;
        q_phase ^= 1;
        cur = u;
        return true;
      };
      auto take_buffer = [&](int& b) -> bool {
        b = (int)(hh & 1u);
        if (!mbar_wait(&acc_empty[b], ((buf_par >> b) & 1u) ^ 1u, abort_flag)) return false;
        tc_fence_after();
        return true;
      };
      auto give_buffer = [&](int b) {
        umma_commit(&acc_full[b]);
        buf_par ^= 1u << b;
        ++hh;
      };
      // pass 1: S = Q K^T, one half per 128-row query tile, N = the item's keys (256 or 128)
      int slot = 0;
      // This thread's work between two MMA groups is on the tensor pipe's critical path: it shares its
      // scheduler with four epilogue warps that issue back to back.  So the unit, its rows and the
      // instruction descriptors are worked out only where the unit changes, and every operand
      // descriptor is one of two bases plus a constant offset (the 14-bit start-address field holds
      // address / 16 of a shared-memory window below 256 KB, so adding offset / 16 never carries out).
      const uint64_t dK0 = umma_desc_sw128(smem_u32(sK)), dQ0 = umma_desc_sw128(qst);
      int t_unit_end = -1;  // pass 1: first item after the current unit
      int n_mt = 1;
      for (int t = p.pass2_only ? t_hi : t_lo; t < t_hi && ok;) {
        if (t >= t_unit_end) {
          const ItemLoc il = locate(p, t);
          const RowGroup r = row_group(g, fmodulo(il.u, g.rg_div));
          if (!(ok = new_unit(il.u))) break;
          n_mt = r.rows > 128 ? 2 : 1;
          t_unit_end = t - il.tile + p.traj[il.b].n_tiles;
        }
        const int nt = (t + 1 < t_hi && t + 1 < t_unit_end) ? 2 : 1;
        for (int i = 0; i < nt && ok; ++i) {
          const int st = 2 * slot + i;
          ok = mbar_wait(&k_full[st], (par >> st) & 1u, abort_flag);
        }
        if (!ok) break;
        tc_fence_after();
        const uint32_t idesc = nt == 2 ? umma_idesc_bf16(128, 2 * kKeyTile) : umma_idesc_bf16(128, kKeyTile);
        const uint64_t dK = dK0 + (uint64_t)(Cfg::chunk_off(2 * slot, 0) >> 4);
        for (int mt = 0; mt < n_mt && ok; ++mt) {
          int b;
          if (!(ok = take_buffer(b))) break;
          const uint32_t dcol = tmem_base + (uint32_t)(b * 256);
          const uint64_t dQ = dQ0 + (uint64_t)((mt * 128 * 128) >> 4);
#pragma unroll
          for (int kk = 0; kk < NCH * 4; ++kk) {
            const uint32_t qoff = (uint32_t)((kk >> 2) * kQChunkBytes + (kk & 3) * 32);
            const uint32_t koff = (uint32_t)((kk >> 2) * 2 * kKChunkBytes + (kk & 3) * 32);  // within the slot
            umma_bf16(dcol, dQ + (qoff >> 4), dK + (koff >> 4), idesc, kk > 0 ? 1u : 0u);
          }
          give_buffer(b);
        }
        if (!ok) break;
        for (int i = 0; i < nt; ++i) {
          const int st = 2 * slot + i;
          umma_commit(&k_empty[st]);
          par ^= 1u << st;
        }
        t += nt;
        if (++slot == P1) slot = 0;
      }
      // pass 2: S^T = K Q^T, the tile's keys on M, the query rows on N
      int k_unit_end = 0;  // pass 2: first item (in pass-2 order) after the current unit
      uint32_t idesc2 = 0;
      for (int k = 0; k < n1 && ok; ++k) {
        if (k == k_unit_end) {
          const int u = locate(p, t_hi - 1 - k).u;
          const RowGroup r = row_group(g, fmodulo(u, g.rg_div));
          if (!(ok = new_unit(u))) break;
          idesc2 = umma_idesc_bf16(128, (r.rows + 31) & ~31);  // every TMEM column the epilogue loads is written
          k_unit_end = t_hi - unit_first_item(p, u);
        }
        int b;
        if (!(ok = take_buffer(b))) break;
        const int st = k % S2;
        if (!(ok = mbar_wait(&k_full[st], (par >> st) & 1u, abort_flag))) break;
        tc_fence_after();
        const uint32_t dcol = tmem_base + (uint32_t)(b * 256);
        const uint64_t dK = dK0 + (uint64_t)(Cfg::chunk_off(st, 0) >> 4);
#pragma unroll
        for (int kk = 0; kk < NCH * 4; ++kk) {
          const uint32_t qoff = (uint32_t)((kk >> 2) * kQChunkBytes + (kk & 3) * 32);
          const uint32_t koff = (uint32_t)((kk >> 2) * 2 * kKChunkBytes + (kk & 3) * 32);  // within the stage
          umma_bf16(dcol, dK + (koff >> 4), dQ0 + (qoff >> 4), idesc2, kk > 0 ? 1u : 0u);
        }
        umma_commit(&k_empty[st]);
        par ^= 1u << st;
        give_buffer(b);
      }
      if (!ok) {
        *abort_flag = 1;
        record_status(p.status, STEPKV_ETIMEOUT);
      }
      // Drain: the last MMA group has completed before TMEM is released.
      if (hh > 0) {
        const int lb = (int)((hh - 1) & 1u);
        mbar_wait_drain(&acc_full[lb], ((buf_par >> lb) & 1u) ^ 1u);
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue (16 warps, 4 per lane quarter)
    // Two groups of 8 warps drain alternate halves (group g drains accumulator buffer g), so one group's
    // TMEM round trips and barrier waits overlap the other group's exponentials.  Within a group, two
    // warps share each TMEM lane quarter.
    const int ew = warp - 2;
    const int q = warp & 3;     // TMEM lane quarter this warp may access
    const int sub = ew >> 2;    // 0..3
    const int grp = sub >> 1;   // epilogue group = accumulator buffer
    const int s2 = sub & 1;     // which of the group's two warps on this quarter
    const bool leader = (ew & 7) == 0;
    const float c = g.c;
    uint32_t acc_phase = 0, eb_phase = 0, hh = 0;
    bool ok = true;
    const uint32_t lane_base = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(grp * 256);
    auto release_buffer = [&]() {
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acc_empty[grp]);
    };

    // The per-token accumulators (8 bytes per token) take an atomic per key and KV head in pass 2; an
    // evict-last L2 policy on their zeroing stores and atomics keeps them resident while the key tiles
    // stream through L2 (fused pass 279.6 -> 277.7 us at T = 32768).
    const uint64_t acc_pol = l2_policy_evict_last();
    // The first epilogue warp zeroes this CTA's share of the accumulators (when the launch accumulates)
    // while the first tiles stream in, then publishes its zero flag (fence + release store of the launch
    // token): a CTA adds into the accumulators only after it has seen every CTA's zero flag, and CTA 0
    // advances the epoch only after that too.
    if (ew == 0) {
      if (p.accumulate) {
        for (int b = 0; b < p.n_traj; ++b) {
          unsigned long long* acc = p.traj[b].t_acc;
          for (int i = blockIdx.x * 32 + lane; i < p.traj[b].T; i += gridDim.x * 32) st_u64_hint(acc + i, 0ull, acc_pol);
        }
      }
      __syncwarp();
      if (lane == 0) {
        __threadfence();
        st_release_u64(&p.zflags[blockIdx.x], tok);
      }
    }

    // ---- pass 1: per-row running (m, Z) over the keys this warp sees (skipped when the caller gives the
    // rows' log-sum-exp)
    if (!p.pass2_only) {
      int cur = -1, Tb = 0;
      float m = -INFINITY, Z = 0.f;
      int my_row = 0, my_pw = 0, my_e = 0;
      bool row_ok = false, two = false;
      // this warp's (m, Z) over its share of the row's keys becomes entry my_e of the CTA's partial
      auto flush_partial = [&](int u) {
        p.part[((size_t)(u + (int)blockIdx.x) * kPartEntries + my_e) * kMaxRows + my_row] = make_float2(m, Z);
      };
      for (int t = t_lo; t < t_hi && ok;) {
        const ItemLoc il = locate(p, t);
        const int nt = item_tiles(il, t);
        const int u = il.u, tile = il.tile;
        t += nt;
        if (u != cur) {
          Tb = p.traj[il.b].T;
          // Every warp flushes every unit the CTA touches (an untouched share flushes m = -inf, Z = 0),
          // so each of the unit's partial entries is written.
          if (cur >= 0) flush_partial(cur);
          const RowGroup r = row_group(g, fmodulo(u, g.rg_div));
          two = r.rows > 128;
          // Above 128 rows every item has two halves, query tile mt in buffer (h0 + mt) & 1 (h0 = halves
          // before the item, of fixed parity within the unit), so group g drains tile (g + h0) & 1 of
          // every item; otherwise the groups alternate items over the single query tile.
          const int mt_g = two ? (int)((grp + hh) & 1u) : 0;
          my_row = mt_g * 128 + q * 32 + lane;
          my_e = two ? s2 : grp * 2 + s2;
          const int w = r.w0 + my_row % r.blk_rows;
          row_ok = my_row < r.rows && w < g.W;
          my_pw = Tb - g.W + w;
          m = -INFINITY;
          Z = 0.f;
          cur = u;
        }
        const int n_halves = two ? 2 : 1;
        const bool mine = two || (hh & 1u) == (uint32_t)grp;
        hh += n_halves;
        if (!mine) continue;
        if (!(ok = mbar_wait(&acc_full[grp], acc_phase, abort_flag))) break;
        acc_phase ^= 1;
        tc_fence_after();
        // Keys on the TMEM columns: warp s2 takes half of the item's nt*128 keys, in pairs of 32-column
        // chunks (one TMEM round trip per pair); the buffer is released once the last pair is loaded.
        const int half_keys = nt * 64;
        const int key0 = tile * kKeyTile + s2 * half_keys;
        const bool need_mask = key0 + half_keys - 1 > Tb - g.W;  // reaches into the causal window
        const int n_pairs_ch = half_keys / 64;
#pragma unroll 1
        for (int h2 = 0; h2 < n_pairs_ch; ++h2) {
          float va[32], vb[32];
          const uint32_t col = (uint32_t)(s2 * half_keys + h2 * 64);
          tmem_ld32x2(lane_base + col, lane_base + col + 32u, va, vb);
          if (h2 == n_pairs_ch - 1) release_buffer();
          if (row_ok) {
            const int j0 = key0 + h2 * 64;
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
      }
      // End of pass 1: every warp writes its last partial; then one thread publishes the CTA's flag.
      // The partial stores are ordered before the flag by the mbarrier (release/acquire within the CTA)
      // followed by the publisher's GPU-scope fence and release store.
      if (ok) {
        if (cur >= 0) flush_partial(cur);
        __syncwarp();
        if (lane == 0) mbar_arrive(p1_flushed);
        if (ew == 0 && lane == 0) {
          if (mbar_wait(p1_flushed, 0, abort_flag)) {
            __threadfence();
            st_release_u64(&p.flags[blockIdx.x], tok);
          } else {
            ok = false;
          }
        }
        ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
      }
    }

    // ---- pass 2: per-key mass over the query rows, with the offsets of every row of the unit
    if (ok) {
      int cur = -1, n_done = 0;  // n_done: pass-2 items this group has drained
      RowGroup r{};
      bool zeros_seen = !p.accumulate;
      float* negoff = sNegOff + grp * kMaxRows;  // this group's per-row offsets and causal limits
      int* pw_tab = sPw + grp * kMaxRows;
      float* combf = sComb + grp * (2 * 128);     // rows output: [2 parity][128]
      // pass-2 item k is half hh + k: this group drains every other item, starting with the first of its parity
      const int k_first = (int)(((uint32_t)grp - hh) & 1u);
      for (int k = k_first; k < n1 && ok; k += 2) {
        const int gt = t_hi - 1 - k;
        const ItemLoc il = locate(p, gt);
        const int u = il.u, tile = il.tile;
        const int Tb = p.traj[il.b].T;
        if (u != cur) {
          // The CTAs whose pass-1 ranges cover unit u: their partials are combined below.
          const int f0 = unit_first_item(p, u);
          const int c0 = cta_of_item(p, f0);
          const int c1 = cta_of_item(p, f0 + p.traj[il.b].n_tiles - 1);
          // Wait until those CTAs have published their pass-1 partials (and, before the first addition,
          // every CTA its zeroed accumulators): the unit starts as soon as its own producers are done.
          if (leader) {
            // Relaxed polls (the lanes' loads overlap), then one acquire fence once all flags match.
            bool all = false;
            const uint64_t t0 = globaltimer_ns();
            for (uint32_t it = 0; !all; ++it) {
              bool mine = true;
              if (!p.pass2_only)  // no pass-1 partials to wait for when the caller gives the row statistics
                for (int b = c0 + lane; b <= c1; b += 32) mine &= ld_relaxed_u64(&p.flags[b]) == wait_tok;
              if (!zeros_seen) {
#pragma unroll 4
                for (int b = lane; b < (int)gridDim.x; b += 32) mine &= ld_relaxed_u64(&p.zflags[b]) == wait_tok;
              }
              all = __all_sync(0xffffffffu, mine);
              if (!all && (it & 15u) == 15u && (*abort_flag || globaltimer_ns() - t0 > p.wait_limit_ns)) break;
            }
            fence_acquire_gpu();
            if (!all) {
              *abort_flag = 1;
              if (lane == 0) record_status(p.status, STEPKV_ETIMEOUT);
            }
          }
          zeros_seen = true;
          // Combine the pass-1 partials of unit u into this group's per-row offsets, in contributing-CTA
          // order (the group no longer reads the previous unit's offsets once all its warps arrive).
          if (!(ok = epi_sync(&epi_bar[grp], eb_phase, abort_flag))) break;
          r = row_group(g, fmodulo(u, g.rg_div));
          const int n_e = r.rows > 128 ? 2 : kPartEntries;  // entries written per row in pass 1
          const int n_e_log2 = r.rows > 128 ? 1 : 2;
          const int row = (ew & 7) * 32 + lane;             // 256 threads of the group, one row each
          const int w = r.w0 + row % r.blk_rows;
          const bool valid = row < r.rows && w < g.W;
          float off = INFINITY;
          if (valid && p.pass2_only) {
            // the caller's natural-log row log-sum-exp, in the kernel's log2 units
            int rg_x, h_x;
            const int pair_x = p.pair0 + fdivmod(il.ul, g.rg_div, rg_x);
            const int layer_x = fdivmod(pair_x, g.hkv_div, h_x);
            const int q_head = h_x * g.G + r.g_first + row / r.blk_rows;
            off = __ldg(p.lse[il.b * p.n_layers + layer_x] + (size_t)q_head * g.W + w) * 1.4426950408889634f;
          } else if (valid) {
            // Log-sum-exp over the unit's entries in a fixed order.  Up to 16 entries (every unit spans
            // at most 8 CTAs for tile ranges of 32 or more) are loaded at once, so one L2 round trip
            // serves them all; longer lists continue in batches of 16.
            const int n_ent = (c1 - c0 + 1) * n_e;
            float M = -INFINITY, Zs = 0.f;
            for (int i0 = 0; i0 < n_ent; i0 += 16) {
              float2 pz[16];
#pragma unroll
              for (int t8 = 0; t8 < 16; ++t8) {
                const int i = i0 + t8;
                const int ci = c0 + (i >> n_e_log2), e = i & (n_e - 1);
                pz[t8] = i < n_ent ? __ldcg(&p.part[((size_t)(u + ci) * kPartEntries + e) * kMaxRows + row])
                                   : make_float2(-INFINITY, 0.f);
              }
              float Mb = M;
#pragma unroll
              for (int t8 = 0; t8 < 16; ++t8) Mb = fmaxf(Mb, pz[t8].x);
              if (Mb == -INFINITY) continue;
              float Zb = M == -INFINITY ? 0.f : Zs * ex2_approx((M - Mb) * c);
#pragma unroll
              for (int t8 = 0; t8 < 16; ++t8)
                Zb += pz[t8].x == -INFINITY ? 0.f : pz[t8].y * ex2_approx((pz[t8].x - Mb) * c);
              M = Mb;
              Zs = Zb;
            }
            off = M * c + __log2f(Zs);
          }
          negoff[row] = -off;
          pw_tab[row] = valid ? Tb - g.W + w : -1;
          if (!(ok = epi_sync(&epi_bar[grp], eb_phase, abort_flag))) break;
          cur = u;
        }
        if (!(ok = mbar_wait(&acc_full[grp], acc_phase, abort_flag))) break;
        acc_phase ^= 1;
        tc_fence_after();
        const int key0 = tile * kKeyTile;
        const bool need_mask = key0 + kKeyTile - 1 > Tb - g.W;  // tile reaches into the causal window
        // Keys on the TMEM lanes: this warp covers its quarter's 32 keys over query columns s2*32 + 64 i
        // (32-column chunks, one TMEM round trip each; holding two chunks in registers spills).  Per
        // chunk a thread needs 8 row offsets, so the shared-memory reads per logit drop fourfold against
        // the one-key-per-thread 32x32b layout.  The buffer is released once the warp's last chunk is in
        // registers.
        const int n_cols = (r.rows + 31) & ~31;
        const int lq = lane & 3;
        const int jq = key0 + q * 32 + (lane >> 2);
        uint64_t acc2[4] = {0ull, 0ull, 0ull, 0ull};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int cc = s2 * 32 + 64 * i;
          if (cc < n_cols) {
            uint64_t o2[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) o2[k] = *reinterpret_cast<const uint64_t*>(&negoff[cc + 8 * k + 2 * lq]);
            uint32_t ra[16], rb[16];
            tmem_ld16x256x4_pair(lane_base + (uint32_t)cc, lane_base + (16u << 16) + (uint32_t)cc, ra, rb);
            if (cc + 64 >= n_cols) release_buffer();
            chunk_mass(ra, rb, o2, pw_tab + cc + 2 * lq, jq, need_mask, c, acc2);
          }
        }
        if (s2 * 32 >= n_cols) release_buffer();  // no chunk for this warp
        // each key's sum is spread over the 4 threads of a quad (lane % 4): reduce in a fixed order, then
        // thread `lane` reports key lane/4 + 8 (lane % 4) of the quarter
        float sk[4];
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
          float lo, hi;
          f2_unpack(acc2[kk], lo, hi);
          sk[kk] = lo + hi;
          sk[kk] += __shfl_xor_sync(0xffffffffu, sk[kk], 1);
          sk[kk] += __shfl_xor_sync(0xffffffffu, sk[kk], 2);
        }
        const float acc = lq == 0 ? sk[0] : lq == 1 ? sk[1] : lq == 2 ? sk[2] : sk[3];
        const int lk = (lane >> 2) + 8 * lq;
        const int j = key0 + q * 32 + lk;
        if (p.accumulate) {
          // fused pass: each warp adds its share of the rows straight into the per-token fixed-point
          // sum (integer addition: the total does not depend on the order of arrival)
          if (j < Tb) red_add_u64_hint(&p.traj[il.b].t_acc[j], to_fixed(acc * g.inv_G, p.acc_shift), acc_pol);
        } else {
          // saliency rows: the group's two warps on this quarter combine in a fixed order (the slot
          // alternates between the group's items, so a write never meets a pending read)
          float* comb = combf + (n_done & 1) * 128;
          if (s2 == 1) comb[q * 32 + lk] = acc;
          if (!(ok = epi_sync(&epi_bar[grp], eb_phase, abort_flag))) break;
          if (s2 == 0 && j < Tb) {
            const float val = (acc + comb[q * 32 + lk]) * g.inv_G;
            int rg;
            const int pair = p.pair0 + fdivmod(il.ul, g.rg_div, rg);
            p.out[(size_t)(pair * g.n_rg + rg) * p.out_stride + j] = val;
          }
        }
        ++n_done;
      }
    }
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
  if (blockIdx.x == 0 && warp == 0) {
    // every CTA has read the epoch once its zero flag carries this launch's token (bounded wait; the
    // epoch advances in any case, so the next launch's token differs from this one)
    const uint64_t t0 = globaltimer_ns();
    for (uint32_t it = 0;; ++it) {
      bool mine = true;
      for (int b = lane; b < (int)gridDim.x; b += 32) mine &= ld_relaxed_u64(&p.zflags[b]) == tok;
      if (__all_sync(0xffffffffu, mine)) break;
      if ((it & 15u) == 15u && globaltimer_ns() - t0 > p.wait_limit_ns) break;
    }
    if (lane == 0) atomicAdd(p.epoch, 1ull);
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
// Contiguous item ranges for the persistent grid, balanced by cost rather than by tile count.  A key tile
// costs 1; a range that switches to another unit costs kUnitSwitchCost more, since the switch stages
// another Q block (the MMAs wait for it), flushes a pass-1 partial, and in pass 2 combines another
// unit's partials after another cross-CTA wait.  With equal tile counts the CTAs whose ranges cross a unit
// boundary finished pass 1 last, and every CTA sharing their units waited for them at the change of pass.
constexpr int kUnitSwitchCost = 3;

// Greedy split under a per-CTA cost cap: returns the number of ranges (max_ranges + 1 if they do not fit)
// and, with `first`, their first items (first[ranges] = the item count).
static int greedy_split(const std::vector<int>& unit_tiles, int cap, int max_ranges, int* first) {
  int ranges = 0, item = 0, cost = 0;
  bool open = false;
  for (const int n : unit_tiles) {
    int left = n;
    bool in_unit = false;  // the open range already holds tiles of this unit
    while (left > 0) {
      if (open && !in_unit && cost + kUnitSwitchCost + 1 > cap) open = false;  // switch would overflow
      if (!open || cost >= cap) {
        if (ranges == max_ranges) return max_ranges + 1;
        if (first) first[ranges] = item;
        ++ranges;
        open = true;
        cost = 0;
        in_unit = false;
      }
      if (!in_unit && cost > 0) cost += kUnitSwitchCost;
      in_unit = true;
      const int take = std::min(left, std::max(1, cap - cost));
      cost += take;
      left -= take;
      item += take;
    }
  }
  if (first) first[ranges] = item;
  return ranges;
}

// The smallest cap whose greedy split fits max_ranges CTAs; writes the ranges and returns their count.
static int split_items(const std::vector<int>& unit_tiles, int items, int max_ranges, int* first) {
  int lo = std::max(1, (items + max_ranges - 1) / max_ranges);
  int hi = items + kUnitSwitchCost * (int)unit_tiles.size();
  while (lo < hi) {
    const int mid = lo + (hi - lo) / 2;
    if (greedy_split(unit_tiles, mid, max_ranges, nullptr) <= max_ranges) hi = mid;
    else lo = mid + 1;
  }
  return greedy_split(unit_tiles, lo, max_ranges, first);
}

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
  g.rg_div = make_fastdiv(g.n_rg);
  g.hkv_div = make_fastdiv(g.Hkv);
  g.rph_div = make_fastdiv(g.rph);
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

// Pass-1 partial slots (one per (unit, CTA) pair a launch can form: units + grid), then one
// pass-1-done flag and one accumulators-zeroed flag per CTA.
static size_t score_partial_slots_bytes(int n_traj, int n_layers, int Hkv, int Hq, int W) {
  const int n_rg = score_row_groups(Hkv, Hq, W);
  return (size_t)(n_traj * n_layers * Hkv * n_rg + kMaxGrid) * kPartEntries * kMaxRows * sizeof(float2);
}
size_t score_partial_bytes(int n_layers, int Hkv, int Hq, int W, int n_traj) {
  // partial slots, pass-1 flags, zero flags, launch epoch (16 B)
  return score_partial_slots_bytes(n_traj, n_layers, Hkv, Hq, W) + 2 * (size_t)kMaxGrid * sizeof(unsigned long long) + 16;
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

// A value no earlier launch in this process used (and, with the per-process salt, vanishingly unlikely to
// be left in a workspace by another process); never zero.
static unsigned long long next_launch_token() {
  static std::atomic<unsigned long long> counter{0};
  static const unsigned long long salt = [] {
    unsigned long long x = (unsigned long long)std::chrono::steady_clock::now().time_since_epoch().count();
    x ^= (unsigned long long)reinterpret_cast<uintptr_t>(&counter) << 17;
    // splitmix64 finaliser
    x += 0x9E3779B97F4A7C15ull;
    x = (x ^ (x >> 30)) * 0xBF58476D1CE4E5B9ull;
    x = (x ^ (x >> 27)) * 0x94D049BB133111EBull;
    return x ^ (x >> 31);
  }();
  unsigned long long t = 0;
  while (t == 0) t = salt + (counter.fetch_add(1) + 1) * 0x9E3779B97F4A7C15ull;
  return t;
}

template <int NCH>
static cudaError_t launch_score(const ScoreLaunch& L, int grid, cudaStream_t stream) {
  using Cfg = ScoreCfg<NCH>;
  void (*kern)(ScoreLaunch) = score_kernel<NCH>;
  cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(kern), Cfg::kDynSmem);
  if (e != cudaSuccess) return e;
  // Cooperative: the pass-2 epilogue of each CTA waits for other CTAs' flags, so all CTAs must be
  // resident at once (the launch fails instead of starting if they cannot be).
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof(cfg));
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = Cfg::kDynSmem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, L);
}

stepkv_status_t score_run_batch(int n_layers, const ScoreTrajSpec* trajs, int n_traj, int Hkv, int Hq, int d,
                                int W, float* rows_out,
                                int64_t out_stride, int acc_shift, float2* part, int32_t* status, cudaStream_t stream,
                                unsigned long long selftest_wait_ns) {
  if (n_traj < 1 || n_traj > kMaxScoreBatch || n_traj * n_layers > kMaxScoreMaps) return STEPKV_EUNSUPPORTED;
  const ScoreGeom g = make_geom(Hkv, Hq, d, trajs[0].T, W);
  ScoreLaunch L;
  memset(&L, 0, sizeof(L));
  L.g = g;
  L.n_traj = n_traj;
  L.n_layers = n_layers;
  L.units_per = n_layers * Hkv * g.n_rg;
  L.units_div = make_fastdiv(L.units_per);
  L.part = part;
  L.flags = reinterpret_cast<unsigned long long*>(reinterpret_cast<uint8_t*>(part) +
                                                  score_partial_slots_bytes(n_traj, n_layers, Hkv, Hq, W));
  L.zflags = L.flags + kMaxGrid;
  L.epoch = L.zflags + kMaxGrid;
  L.out = rows_out;
  L.out_stride = out_stride;
  L.accumulate = trajs[0].t_acc != nullptr ? 1 : 0;
  L.pass2_only = trajs[0].lse != nullptr ? 1 : 0;
  L.acc_shift = acc_shift;
  L.status = status;
  const int box_rows = std::min(g.W_pad, kMaxRows);
  int items = 0;
  for (int b = 0; b < n_traj; ++b) {
    const ScoreTrajSpec& t = trajs[b];
    if ((t.t_acc != nullptr) != (L.accumulate != 0)) return STEPKV_EINVAL;
    if ((t.lse != nullptr) != (L.pass2_only != 0)) return STEPKV_EINVAL;
    for (int l = 0; l < n_layers; ++l) {
      if (t.lse && !t.lse[l]) return STEPKV_EINVAL;
      L.lse[b * n_layers + l] = t.lse ? t.lse[l] : nullptr;
      if (!encode_3d(&L.tmK[b * n_layers + l], t.K[l], d, t.T, Hkv, t.k_head_stride, kKeyTile)) return STEPKV_ECUDA;
      if (!encode_3d(&L.tmQ[b * n_layers + l], t.Q[l], d, W, Hq, t.q_head_stride, box_rows)) return STEPKV_ECUDA;
    }
    L.traj[b].T = t.T;
    L.traj[b].n_tiles = (t.T + kKeyTile - 1) / kKeyTile;
    L.traj[b].nt_div = make_fastdiv(L.traj[b].n_tiles);
    L.traj[b].item_off = items;
    L.traj[b].t_acc = t.t_acc;
    items += L.units_per * L.traj[b].n_tiles;
  }
  int n_sm = 0;
  cudaError_t e = device_sm_count(&n_sm);
  if (e != cudaSuccess) { set_last_cuda_error(e); return STEPKV_ECUDA; }
  const int grid_cap = std::max(1, std::min(n_sm, kMaxGrid));
  // all (trajectory, layer, KV head) pairs in one launch: every CTA gets a contiguous range of items
  L.pair0 = 0;
  L.n_items = items;
  std::vector<int> unit_tiles;
  unit_tiles.reserve((size_t)n_traj * L.units_per);
  for (int b = 0; b < n_traj; ++b) unit_tiles.insert(unit_tiles.end(), L.units_per, L.traj[b].n_tiles);
  const int grid = split_items(unit_tiles, items, grid_cap, L.cta_first);
  L.token = next_launch_token();
  // Self-test of the failure path: the pass-2 wait looks for a value no CTA ever publishes, so every
  // CTA's wait runs out after selftest_wait_ns and the kernel takes its abort path.
  L.selftest = selftest_wait_ns ? 1 : 0;
  L.wait_limit_ns = selftest_wait_ns ? selftest_wait_ns : kWaitLimitNs;
  e = d == 128 ? launch_score<2>(L, grid, stream) : launch_score<1>(L, grid, stream);
  if (e != cudaSuccess) { set_last_cuda_error(e); return STEPKV_ECUDA; }
  return STEPKV_OK;
}

stepkv_status_t score_run(int n_layers, const void* const* K, int64_t k_head_stride, const void* const* Q,
                          int64_t q_head_stride, int Hkv, int Hq, int d, int T, int W, float* rows_out,
                          int64_t out_stride, unsigned long long* t_acc, int acc_shift, float2* part, int32_t* status,
                          cudaStream_t stream, unsigned long long selftest_wait_ns, const float* const* lse) {
  const ScoreTrajSpec one{K, Q, T, t_acc, k_head_stride, q_head_stride, lse};
  return score_run_batch(n_layers, &one, 1, Hkv, Hq, d, W, rows_out, out_stride, acc_shift, part, status, stream,
                         selftest_wait_ns);
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
