// Step 3: block-causal GQA verify attention on GB300 (split-KV, Stream-K,
// warp-specialised persistent CTAs, 5th-generation tensor cores, all layers
// of a round in one launch).
//
// Work decomposition. For sequence b the verified block has M_b = (L_b+1)*g
// query rows per kv head (g = Hq/Hkv; row r is block position t = r / g of
// query head kvh*g + r % g) and N_b = kv_len_b + L_b + 1 visible keys. Rows
// are cut into groups of R = g * floor(128/g) (whole block positions, at most
// 128: one tcgen05 M=128 tile) and keys into 64-key tiles. All (row group,
// key tile) pairs of the batch form one tile sequence (sequence-major, then kv
// head, row group, key tile); CTA c of the persistent grid (one CTA per SM)
// takes the contiguous range [c*T/G, (c+1)*T/G) of it, so every CTA streams
// the same number of tiles whatever the ragged lengths; with more (sequence,
// kv head) pairs than CTAs the ranges are cut by cost instead (each row
// group weighs its tiles plus an item's fixed cost; tile_of_weighted). The
// plan is derived on the device from L[] and kv_len[] by every CTA, and it
// is the same for every layer (all layers share L and kv_len).
//
// Roles in a CTA (192 threads):
//  * producer warp: walks the CTA's range layer after layer in items (runs of
//    tiles of one row group); loads the group's Q rows (one 3-D TMA box per
//    64-column half: R/g positions x g heads) into a Q slot (two slots at
//    d = 64; one at d = 128, whose shared memory goes to a fifth stage) and
//    the K/V tiles (3-D TMA, 128-byte swizzle) into a ring of STAGES stages;
//  * MMA warp: one thread issues S = Q K^T (tcgen05.mma, A and B K-major from
//    shared memory, fp32 accumulator in tensor memory, double-buffered) and
//    O += P V (A = P from tensor memory, B = V MN-major from shared memory),
//    and signals completions with tcgen05.commit;
//  * softmax warpgroup (4 warps, thread i <-> tensor-memory lane i = row i of
//    the group): reads S, masks keys beyond kv_len_b + t, keeps the online
//    softmax in the log2 domain, writes P (bf16) back to tensor memory, and at
//    the end of an item normalises O and stores it (or a split partial).
// The running max is only raised when a tile's max exceeds it by more than 8
// (a factor 2^8), so O is rescaled in tensor memory rarely; p <= 2^8 keeps
// bf16 P and fp32 O exact in range, and O / l is unchanged by the choice of
// reference max.
//
// Layers. Layer l+1 may read Q, the block's own keys (positions >= kv_len_b)
// and layer l's partials only after every CTA has finished layer l: a
// grid-wide barrier (one counter per layer; the launch is cooperative, so all
// CTAs are resident and the bounded waits end). The cache prefix
// (keys < kv_len_b) is state from earlier rounds, so the producer streams the
// next layer's prefix tiles while the softmax warps still finish the current
// layer.
//
// Split groups. A row group covered by one CTA is written directly. A group
// spread over CTAs c0..c1 leaves one fp32 partial (O, m, l) per CTA, in slot
// 2c+1 for c0 (its last item) and 2c for the others (their first item), in a
// buffer chosen by the layer (l mod 3). After the barrier that ends layer
// l, each of those CTAs merges its share of the group's rows from all parts
// in CTA order (deterministic, spread over every contributing SM); the merge
// of layer l runs beside the CTA's items of layer l+1. The last layer waits
// for no grid barrier: a group's parts are counted in as they are written,
// and a small group is merged whole by the CTA whose part completes it.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <cstdio>
#include <cstdlib>
#include <memory>

#include "common.cuh"
#include "tc.cuh"

namespace libraspec {

constexpr int kSoftmaxWarps = 4;
constexpr int kProducerWarp = 4;
constexpr int kMmaWarp = 5;
constexpr int kMergeWarp = 6;
constexpr int kAttnThreads = 7 * 32;
constexpr int kPBufs = 4;  // P buffers in tensor memory
constexpr int kMaxWaitIters = 1 << 24;
constexpr int kSoftmaxBar = 1;  // named barrier of the softmax warpgroup
constexpr float kRescaleLog2 = 8.f;
constexpr int kTmemCols = 512;

__device__ __forceinline__ void softmax_sync() {
  asm volatile("bar.sync %0, %1;" ::"n"(kSoftmaxBar), "n"(kSoftmaxWarps * 32) : "memory");
}

// bits [0, n) set (n clamped to [0, 64])
__device__ __forceinline__ uint64_t low_bits(int n) {
  return n <= 0 ? 0ull : (n >= 64 ? ~0ull : ((1ull << n) - 1ull));
}

// Bits [o, o + 64) of the bit set row[0 .. words) (bits outside read as 0;
// o may be negative).
__device__ __forceinline__ uint64_t bit_window(const uint64_t* __restrict__ row, int words, int o) {
  const int q = o >> 6, r = o & 63;  // floor division
  const uint64_t lo = (q >= 0 && q < words) ? __ldg(row + q) : 0ull;
  const uint64_t hi = (q + 1 >= 0 && q + 1 < words) ? __ldg(row + q + 1) : 0ull;
  return r == 0 ? lo : (lo >> r) | (hi << (64 - r));
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// ---------------------------------------------------------------------------
// Device-side plan.
// ---------------------------------------------------------------------------
struct SeqPlan {
  int M, n_mg, N, n_tiles;  // rows, row groups, visible keys, key tiles
  bool ok;
};

__device__ __forceinline__ SeqPlan seq_plan(int b, int B, const int32_t* kv_len, const int32_t* Ls, int K, int g,
                                            int R, int S_cap) {
  SeqPlan p{0, 0, 0, 0, false};
  if (b >= B) return p;
  const int Lb = Ls[b], kv = kv_len[b];
  if (Lb < 0 || Lb > K || kv < 0 || (long)kv + Lb + 1 > S_cap) return p;
  p.ok = true;
  p.M = (Lb + 1) * g;
  p.n_mg = (p.M + R - 1) / R;
  p.N = kv + Lb + 1;
  p.n_tiles = (p.N + kAttnTileKeys - 1) / kAttnTileKeys;
  return p;
}

// Warp-wide: total tiles T of the batch and its row groups (*groups);
// flags invalid sequences.
__device__ long long total_tiles(int B, const int32_t* kv_len, const int32_t* Ls, int K, int g, int R, int Hkv,
                                 int S_cap, int* status, bool report, long long* groups) {
  const int lane = threadIdx.x & 31;
  long long tot = 0, ng = 0;
  bool bad = false;
  for (int b = lane; b < B; b += 32) {
    const SeqPlan p = seq_plan(b, B, kv_len, Ls, K, g, R, S_cap);
    if (!p.ok) bad = true;
    else {
      tot += (long long)Hkv * p.n_mg * p.n_tiles;
      ng += (long long)Hkv * p.n_mg;
    }
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    tot += __shfl_xor_sync(0xffffffffu, tot, off);
    ng += __shfl_xor_sync(0xffffffffu, ng, off);
  }
  *groups = ng;
  if (report && __any_sync(0xffffffffu, bad) && lane == 0) {
    int bits = 0;
    for (int b = 0; b < B; ++b) {
      const int Lb = Ls[b], kv = kv_len[b];
      if (Lb < 0 || Lb > K) bits |= LIBRASPEC_ST_BAD_LENGTH;
      else if (kv < 0 || (long)kv + Lb + 1 > S_cap) bits |= LIBRASPEC_ST_KV_OVERFLOW;
    }
    raise_status(status, bits);
  }
  return tot;
}

// Where tile position `pos` of the batch's tile sequence lies (warp-wide).
struct TileLoc {
  int b;                  // sequence (-1: past the end)
  long long seq_start;    // first tile of sequence b
  int group0;             // global index of b's first row group
  SeqPlan p;
};

__device__ TileLoc locate_tile(long long pos, int B, const int32_t* kv_len, const int32_t* Ls, int K, int g, int R,
                               int Hkv, int S_cap) {
  const int lane = threadIdx.x & 31;
  TileLoc loc{-1, 0, 0, {}};
  long long carry_t = 0;
  int carry_g = 0;
  for (int base = 0; base < B; base += 32) {
    const int b = base + lane;
    const SeqPlan p = seq_plan(b, B, kv_len, Ls, K, g, R, S_cap);
    const long long nt = p.ok ? (long long)Hkv * p.n_mg * p.n_tiles : 0;
    const int ng = p.ok ? Hkv * p.n_mg : 0;
    long long inc_t = nt;
    int inc_g = ng;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const long long a = __shfl_up_sync(0xffffffffu, inc_t, off);
      const int c = __shfl_up_sync(0xffffffffu, inc_g, off);
      if (lane >= off) { inc_t += a; inc_g += c; }
    }
    const long long st = carry_t + inc_t - nt;
    const bool mine = nt > 0 && pos >= st && pos < st + nt;
    const unsigned ball = __ballot_sync(0xffffffffu, mine);
    if (ball) {
      const int src = __ffs(ball) - 1;
      loc.b = base + src;
      loc.seq_start = __shfl_sync(0xffffffffu, st, src);
      loc.group0 = __shfl_sync(0xffffffffu, carry_g + inc_g - ng, src);
      loc.p = seq_plan(loc.b, B, kv_len, Ls, K, g, R, S_cap);
      return loc;
    }
    carry_t += __shfl_sync(0xffffffffu, inc_t, 31);
    carry_g += __shfl_sync(0xffffffffu, inc_g, 31);
  }
  return loc;
}

// a / b for a >= 0, b > 0: 32-bit when both fit (a 64-bit division is a
// long software sequence, and the plan runs on one warp before any copy)
__device__ __forceinline__ long long div_nn(long long a, long long b) {
  if ((((unsigned long long)a | (unsigned long long)b) >> 32) == 0) return (long long)((uint32_t)a / (uint32_t)b);
  return a / b;
}

__device__ __forceinline__ long long range_lo(int c, long long T, int G) { return div_nn((long long)c * T, G); }

// CTA whose range holds tile t: the largest c with c*T/G <= t.
__device__ __forceinline__ int cta_of(long long t, long long T, int G) {
  return (int)div_nn((t + 1) * (long long)G - 1, T);
}

// Cost-weighted Stream-K. A row group costs its key tiles plus C (an item's
// fixed cost: the Q load the first S waits for, the epilogue, a partial's
// merge, in tile-equivalents), placed before its tiles; the batch weighs
// W = T + C * groups, and CTA c takes the tiles of the weighted range
// [c W / G, (c+1) W / G). A boundary inside a group's C falls on the
// group's first tile. C = 0 is the plain split by tiles.
__device__ long long tile_of_weighted(long long x, long long W, long long T, int C, int B, const int32_t* kv_len,
                                      const int32_t* Ls, int K, int g, int R, int Hkv, int S_cap) {
  if (x >= W) return T;
  const int lane = threadIdx.x & 31;
  long long carry_w = 0, carry_t = 0;
  for (int base = 0; base < B; base += 32) {
    const int b = base + lane;
    const SeqPlan p = seq_plan(b, B, kv_len, Ls, K, g, R, S_cap);
    const long long nt = p.ok ? (long long)Hkv * p.n_mg * p.n_tiles : 0;
    const long long nw = p.ok ? nt + (long long)C * Hkv * p.n_mg : 0;
    long long inc_w = nw, inc_t = nt;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const long long a = __shfl_up_sync(0xffffffffu, inc_w, off);
      const long long t = __shfl_up_sync(0xffffffffu, inc_t, off);
      if (lane >= off) { inc_w += a; inc_t += t; }
    }
    const long long sw = carry_w + inc_w - nw;
    const bool mine = nw > 0 && x >= sw && x < sw + nw;
    const unsigned ball = __ballot_sync(0xffffffffu, mine);
    if (ball) {
      const int src = __ffs(ball) - 1;
      const long long wstart = __shfl_sync(0xffffffffu, sw, src);
      const long long tstart = __shfl_sync(0xffffffffu, carry_t + inc_t - nt, src);
      const SeqPlan q = seq_plan(base + src, B, kv_len, Ls, K, g, R, S_cap);
      const long long per = q.n_tiles + C;
      const long long o = x - wstart;
      const long long gib = div_nn(o, per);
      const long long r = o - gib * per;
      return tstart + gib * q.n_tiles + (r > C ? r - C : 0);
    }
    carry_w += __shfl_sync(0xffffffffu, inc_w, 31);
    carry_t += __shfl_sync(0xffffffffu, inc_t, 31);
  }
  return T;
}

// Weighted position of tile t of global row group `group` (the groups up to
// and including it each put C before their tiles).
__device__ __forceinline__ long long weighted_pos(long long t, long long group, int C) {
  return t + (long long)C * (group + 1);
}

// Bounded poll of a grid-barrier counter (acquire).
__device__ __forceinline__ bool wait_counter(const uint32_t* ctr, uint32_t target) {
  for (int i = 0; i < kMaxWaitIters; ++i) {
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(ctr) : "memory");
    if (v >= target) return true;
    __nanosleep(32);
  }
  return false;
}

// One item handed from the producer to the MMA and softmax warps.
struct ItemInfo {
  int b, kvh, mg, rows, kv;
  int key0, key1;     // keys [key0, key1)
  int partial;        // 1: write a partial, else write O
  int slot;           // partial slot
  int grp;            // global row group index
  int pad[6];
};

// A split row group this CTA helps merge (the same for every layer).
struct MergeTask {
  int b, kvh, mg, rows, c0, np;
  int grp;  // global row group index
  int epi;  // in the last layer, merged whole by the CTA completing it (small groups)
};
// A split group whose merge reads at most this many (row, 4-column) items
// over all its parts (rows x d/4 x parts) is merged, in a launch's last
// layer, by the CTA whose part completes it, in that part's epilogue (a few
// memory round trips, and no wait); a larger one (a long group spread over
// many CTAs) is merged share by share by all its CTAs.
constexpr int kEpiMaxItems = 8192;
static_assert(2 * sizeof(MergeTask) <= 64, "two merge tasks fit their shared-memory slot");

constexpr int kMaxLayers = kAttnMaxLayers;

struct LayerPtrs {
  const __nv_bfloat16* Q;
  __nv_bfloat16* O;
  float* lse;
};

// Everything a launch needs per layer, passed by value as one kernel
// parameter (< 32 KB).
struct LayerSet {
  CUtensorMap K[kMaxLayers];
  CUtensorMap V[kMaxLayers];
  CUtensorMap Q[kMaxLayers];
  LayerPtrs p[kMaxLayers];
  int n;
};
static_assert(sizeof(LayerSet) <= 32000, "kernel parameters are limited to 32764 bytes");

template <int D, int STAGES>
struct AttnSmem {
  // One Q slot at d = 128 (the next item's Q then waits for this one's last
  // S) buys a fifth K/V stage: more of the next layer's prefix streams in
  // before the layer barrier (8b: 9.76 -> 9.40 us per layer).
  static constexpr int kQSlots = (D == 128 && STAGES >= 5) ? 1 : 2;
  static constexpr int kBoxes = D / 64;
  static constexpr int kTileBytes = kBoxes * 8192;       // one 64-key x D bf16 tile (per box 64 x 128 B)
  static constexpr int kQBox = kAttnRows * 128;          // 128 rows x 64 columns
  static constexpr int kQSlot = kBoxes * kQBox;
  static constexpr int kQ = 0;                           // 2 slots
  static constexpr int kK = kQ + kQSlots * kQSlot;
  static constexpr int kV = kK + STAGES * kTileBytes;
  // mbarriers: full[S], empty[S], qfull[2], qempty[2], sfull[2], sfree[2],
  // pfull[4], pvdone[4], ofree[2], drain
  static constexpr int kBar = kV + STAGES * kTileBytes;
  static constexpr int kNumBars = 2 * STAGES + 2 * 4 + 2 * kPBufs + 2 + 1;
  static constexpr int kInfo = kBar + ((8 * kNumBars + 63) / 64) * 64;
  static constexpr int kTasks = kInfo + 2 * 64;
  static constexpr int kTmem = kTasks + 64;
  // [0] abort, [1] merge tasks, [2] items per layer, [3] merge chunks per
  // layer, [4] chunks claimed, [5] chunks done, [6] the last layer's shared
  // merges may start, [7] this item's epilogue merges its group
  static constexpr int kMisc = kTmem + 16;
  // kv_len and L of up to kPlanCap sequences, read once from global memory
  // for the CTA's tile plan (a larger batch plans from global memory)
  static constexpr int kPlanCap = 1024;
  static constexpr int kRange = kMisc + 32;  // the CTA's tile range [lo, hi)
  static constexpr int kPlan = kRange + 16;
  static constexpr int kBytes = kPlan + 2 * 4 * kPlanCap;
  static constexpr int kAlloc = kBytes + 1024;           // room to align the base to 1024
  // tensor-memory columns
  static constexpr int kColS = 0;                        // S[2]: 64 fp32 columns each
  static constexpr int kColP = 128;                      // P[4]: 64 bf16 = 32 columns each
  static constexpr int kColO = 256;                      // O[2]: D fp32 columns each
  static_assert(kColP + 32 * kPBufs <= kColO && kColO + 2 * D <= kTmemCols, "tensor memory");
  static_assert(kAlloc <= 227 * 1024, "shared memory per CTA");
  // paged caches: the page of each of the CTA's tiles, after everything else
  static constexpr int kPageCap = 4096;
  static constexpr int kAllocPaged = kAlloc + kPageCap * 4;
  static_assert(kAllocPaged <= 227 * 1024, "shared memory per CTA (paged)");
};

// Merging a layer's split groups. This CTA merges its share of rows
// [rows*k/np, rows*(k+1)/np) of each group it contributed to (k = its index
// among the group's np CTAs): O = sum_p w_p O_p / sum_p w_p l_p with
// w_p = 2^(m_p - M), M = max m_p, parts in CTA order. The share is cut into
// chunks of (row, 4-column) items that any warp may claim once the layer's
// grid barrier has passed: the merge warp right away (beside the next
// layer's items), the softmax warps once their own items are done. A lane
// loads (m_p, l_p) and its 4 columns of O_p for a batch of parts at once and
// folds the batch in with a running maximum, so a chunk costs one memory
// round trip per batch and no weights are staged in shared memory.

// This CTA's share [u0, u0 + nr) of task t's rows.
__device__ __forceinline__ int merge_share(const MergeTask& t, int& u0) {
  const int k_me = (int)blockIdx.x - t.c0;
  u0 = (int)((long long)t.rows * k_me / t.np);
  return (int)((long long)t.rows * (k_me + 1) / t.np) - u0;
}

// Between layers the softmax warps help with a merge of at least this many
// chunks; a smaller one is left to the merge warp, which keeps cold code off
// the softmax warps' path from one layer to the next (instruction fetch
// misses cost about a memory round trip). The last layer's merge, the tail
// of the launch, is always shared.
constexpr int kMergeHelpChunks = 8;

// Items per lane in a chunk of a group of np parts: J items x 16/J parts are
// in flight per batch, and a share of `items` items costs ceil(items / 32J)
// chunks x ceil(np / (16/J)) batches, one memory round trip each. J = 4 wins
// for many rows over few parts (tree and long blocks), J = 1 for one row
// over many parts (short blocks at B = 1); ties go to J = 1 (more chunks to
// share among helping warps).
__device__ __forceinline__ int merge_j(int np, int items) {
  const int trips1 = ((items + 31) / 32) * ((np + 15) / 16);
  const int trips4 = ((items + 127) / 128) * ((np + 3) / 4);
  return trips4 < trips1 ? 4 : 1;
}

template <int J, int D>
__device__ __forceinline__ void merge_chunk(const MergeTask& t, int u0, int nr, int lc, const float* __restrict__ part_o,
                                            const float* __restrict__ part_ml, int K, int Hq, int g, int R,
                                            __nv_bfloat16* __restrict__ O, float* __restrict__ lse);

// The whole of group t by the softmax warpgroup (warp w of 4 takes every
// fourth chunk), share by share with each share's chunk shape, so the result
// has the bits the group's CTAs would each give for their share. Out of line:
// it runs once per small split group of a launch's last layer, and keeps its
// code out of the item loop's instruction stream.
template <int D>
__device__ __noinline__ void merge_group_whole(const MergeTask t, int warp, const float* __restrict__ part_o,
                                               const float* __restrict__ part_ml, int K, int Hq, int g, int R,
                                               __nv_bfloat16* __restrict__ O, float* __restrict__ lse) {
  int gi = 0;
  for (int k = 0; k < t.np; ++k) {
    const int u0 = (int)((long long)t.rows * k / t.np);
    const int nr = (int)((long long)t.rows * (k + 1) / t.np) - u0;
    const int items = nr * (D / 4);
    const int J = merge_j(t.np, items);
    const int nc = (items + 32 * J - 1) / (32 * J);
    for (int lc = 0; lc < nc; ++lc, ++gi) {
      if (gi % kSoftmaxWarps != warp) continue;
      if (J == 1) merge_chunk<1, D>(t, u0, nr, lc, part_o, part_ml, K, Hq, g, R, O, lse);
      else merge_chunk<4, D>(t, u0, nr, lc, part_o, part_ml, K, Hq, g, R, O, lse);
    }
  }
}

// A part of a launch's last layer is written (softmax warpgroup, after its
// epilogue). The last layer's split groups need no grid barrier: each part is
// counted in as written (the named barrier orders the warpgroup's writes
// before the release). A small group is merged at once, whole, by the CTA
// whose part completes it (the acquire makes the other parts visible), share
// by share as its CTAs would merge it, so the result is the same bits; a
// larger one by the merge warps of all its CTAs once its count is complete.
// Out of line, like merge_group_whole: it runs once per split part of the
// last layer.
template <int D>
__device__ __noinline__ void last_layer_part_done(const MergeTask* tasks, int n_tasks, int grp,
                                                  uint32_t* __restrict__ grp_cnt, volatile int* misc,
                                                  const float* __restrict__ part_o, const float* __restrict__ part_ml,
                                                  int K, int Hq, int g, int R, __nv_bfloat16* __restrict__ O,
                                                  float* __restrict__ lse) {
  const int tid = threadIdx.x, warp = tid >> 5;
  int ti = 0;
  while (ti + 1 < n_tasks && tasks[ti].grp != grp) ++ti;
  const MergeTask t = tasks[ti];
  softmax_sync();
  if (tid == 0) {
    bool last = false;
    if (t.epi) {
      uint32_t old;
      asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], %2;" : "=r"(old) : "l"(grp_cnt + 2 * grp), "r"(1u) : "memory");
      last = old == (uint32_t)t.np - 1;
      if (last) grp_cnt[2 * grp] = 0u;  // every part is in: ready for the next launch
    } else {
      asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(grp_cnt + 2 * grp), "r"(1u) : "memory");
    }
    misc[7] = last ? 1 : 0;
  }
  softmax_sync();
  if (misc[7]) merge_group_whole<D>(t, warp, part_o, part_ml, K, Hq, g, R, O, lse);
}

template <int D>
__device__ __forceinline__ int merge_chunk_count(const MergeTask* tasks, int n_tasks) {
  int n = 0;
  for (int ti = 0; ti < n_tasks; ++ti) {
    int u0;
    const int items = merge_share(tasks[ti], u0) * (D / 4);
    const int ci = 32 * merge_j(tasks[ti].np, items);
    n += (items + ci - 1) / ci;
  }
  return n;
}

// Chunk lc of task t: items (lc*J + j)*32 + lane, j < J.
template <int J, int D>
__device__ __forceinline__ void merge_chunk(const MergeTask& t, int u0, int nr, int lc, const float* __restrict__ part_o,
                                            const float* __restrict__ part_ml, int K, int Hq, int g, int R,
                                            __nv_bfloat16* __restrict__ O, float* __restrict__ lse) {
  constexpr int PB = 16 / J, C4 = D / 4;
  const int lane = threadIdx.x & 31;
  const int np = t.np, c0 = t.c0, items = nr * C4;
  float M[J], Ls[J];
  float4 acc[J];
#pragma unroll
  for (int j = 0; j < J; ++j) {
    M[j] = -INFINITY;
    Ls[j] = 0.f;
    acc[j] = make_float4(0.f, 0.f, 0.f, 0.f);
  }
  for (int p0 = 0; p0 < np; p0 += PB) {
    float2 ml[J][PB];
    float4 v[J][PB];
#pragma unroll
    for (int j = 0; j < J; ++j) {
      const int i = (lc * J + j) * 32 + lane;
      const int r = i / C4, c = i - r * C4;
#pragma unroll
      for (int k = 0; k < PB; ++k) {
        const int p = p0 + k;
        if (i < items && p < np) {
          const size_t at = (size_t)(p == 0 ? 2 * c0 + 1 : 2 * (c0 + p)) * kAttnRows + u0 + r;
          ml[j][k] = __ldcg(reinterpret_cast<const float2*>(part_ml + at * 2));
          v[j][k] = __ldcg(reinterpret_cast<const float4*>(part_o + at * D) + c);
        } else {
          ml[j][k] = make_float2(-INFINITY, 0.f);
          v[j][k] = make_float4(0.f, 0.f, 0.f, 0.f);
        }
      }
    }
#pragma unroll
    for (int j = 0; j < J; ++j) {
      float bm = -INFINITY;
#pragma unroll
      for (int k = 0; k < PB; ++k) bm = fmaxf(bm, ml[j][k].x);
      const float Mn = fmaxf(M[j], bm);
      if (Mn == -INFINITY) continue;  // no visible key in these parts yet
      const float f = ex2_approx(M[j] - Mn);  // 0 while M is still -inf
      acc[j].x *= f;
      acc[j].y *= f;
      acc[j].z *= f;
      acc[j].w *= f;
      Ls[j] *= f;
      M[j] = Mn;
#pragma unroll
      for (int k = 0; k < PB; ++k) {
        const float w = ex2_approx(ml[j][k].x - Mn);  // 0 for a part with no visible key
        acc[j].x += w * v[j][k].x;
        acc[j].y += w * v[j][k].y;
        acc[j].z += w * v[j][k].z;
        acc[j].w += w * v[j][k].w;
        Ls[j] += w * ml[j][k].y;
      }
    }
  }
#pragma unroll
  for (int j = 0; j < J; ++j) {
    const int i = (lc * J + j) * 32 + lane;
    if (i >= items) continue;
    const int r = i / C4, c = i - r * C4;
    const float inv = 1.f / Ls[j];
    const int rr = t.mg * R + u0 + r;
    const int tt = rr / g, hq = t.kvh * g + rr % g;
    uint2 o;
    o.x = pack_bf16(acc[j].x * inv, acc[j].y * inv);
    o.y = pack_bf16(acc[j].z * inv, acc[j].w * inv);
    *reinterpret_cast<uint2*>(O + (((size_t)t.b * (K + 1) + tt) * Hq + hq) * D + c * 4) = o;
    if (lse && c == 0) lse[((size_t)t.b * (K + 1) + tt) * Hq + hq] = (M[j] + __log2f(Ls[j])) * kLn2;
  }
}

// Claims and merges chunks of layers up to `last_layer` until none is left,
// oldest first. Chunks are numbered [l * C, (l + 1) * C) for layer l on the
// CTA's monotonic counters; ctr_done counts the chunks merged (stores done).
template <int D>
__device__ void merge_chunks(int last_layer, const LayerSet& set, const MergeTask* tasks, int n_tasks, int C,
                             int* ctr_claim, int* ctr_done, int K, int Hq, int Hkv, int R,
                             const float* __restrict__ part_buf_o, const float* __restrict__ part_buf_ml,
                             size_t part_o_stride, size_t part_ml_stride, int epi_layer) {
  const int lane = threadIdx.x & 31;
  const int g = Hq / Hkv;
  const int hi = (last_layer + 1) * C;
  for (;;) {
    int u = 0;
    if (lane == 0) {
      u = *reinterpret_cast<volatile int*>(ctr_claim);
      while (u < hi) {
        const int prev = atomicCAS(ctr_claim, u, u + 1);
        if (prev == u) break;
        u = prev;
      }
    }
    u = __shfl_sync(0xffffffffu, u, 0);
    if (u >= hi) return;
    // the chunk's layer, task and index within the task
    const int layer = u / C;
    const float* part_o = part_buf_o + (layer % kAttnPartBufs) * part_o_stride;
    const float* part_ml = part_buf_ml + (layer % kAttnPartBufs) * part_ml_stride;
    __nv_bfloat16* O = set.p[layer].O;
    float* lse = set.p[layer].lse;
    int lc = u - layer * C, ti = 0, u0 = 0, nr = 0;
    for (; ti < n_tasks; ++ti) {
      nr = merge_share(tasks[ti], u0);
      const int ci = 32 * merge_j(tasks[ti].np, nr * (D / 4));
      const int nc = (nr * (D / 4) + ci - 1) / ci;
      if (lc < nc) break;
      lc -= nc;
    }
    if (ti < n_tasks && !(layer == epi_layer && tasks[ti].epi)) {  // (an epilogue merge: counted, no work)
      const MergeTask& t = tasks[ti];
      if (merge_j(t.np, nr * (D / 4)) == 1) merge_chunk<1, D>(t, u0, nr, lc, part_o, part_ml, K, Hq, g, R, O, lse);
      else merge_chunk<4, D>(t, u0, nr, lc, part_o, part_ml, K, Hq, g, R, O, lse);
    }
    __syncwarp();
    if (lane == 0) atomicAdd(ctr_done, 1);
  }
}

// PAGED: the caches are page pools [n_pages, Hkv, page_size, d] and key s of
// sequence b lives at page block_table[b * max_pages + s / page_size], row
// s % page_size (page_size a multiple of 64, so a key tile lies in one page);
// S_cap is then max_pages * page_size.
// tree_vis (optional, [B, K+1, tree_words]): the block is a draft tree and
// row t sees the block keys of the set bits (bit j <-> block position j + 1)
// besides the root and the prefix; nullptr: the chain draft (block-causal).
template <int D, int STAGES, bool PAGED, bool WEIGHTED>
__global__ void __launch_bounds__(kAttnThreads, 1) verify_attn_kernel(
    const __grid_constant__ LayerSet set, const int32_t* __restrict__ kv_len, const int32_t* __restrict__ Ls,
    const uint64_t* __restrict__ tree_vis, int tree_words,
    const int32_t* __restrict__ block_table, int max_pages, int page_size, int n_pages, int page_cache,
    int B, int K, int Hq, int Hkv, int S_cap, float scale_log2, int min_tiles, int item_tiles,
    float* __restrict__ part_buf_o,
    float* __restrict__ part_buf_ml, size_t part_o_stride, size_t part_ml_stride, uint32_t* __restrict__ bar_cnt,
    uint32_t* __restrict__ grp_cnt, int* __restrict__ status) {
  using SM = AttnSmem<D, STAGES>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sQ = smem_u32(smem + SM::kQ);
  const uint32_t sK = smem_u32(smem + SM::kK);
  const uint32_t sV = smem_u32(smem + SM::kV);
  const uint32_t bFull = smem_u32(smem + SM::kBar);
  const uint32_t bEmpty = bFull + 8 * STAGES;
  const uint32_t bQFull = bEmpty + 8 * STAGES;
  const uint32_t bQEmpty = bQFull + 16;
  const uint32_t bSFull = bQEmpty + 16;
  const uint32_t bSFree = bSFull + 16;
  const uint32_t bPFull = bSFree + 16;
  const uint32_t bPVDone = bPFull + 8 * kPBufs;
  const uint32_t bOFree = bPVDone + 8 * kPBufs;
  const uint32_t bDrain = bOFree + 16;
  ItemInfo* info = reinterpret_cast<ItemInfo*>(smem + SM::kInfo);
  MergeTask* tasks = reinterpret_cast<MergeTask*>(smem + SM::kTasks);
  volatile uint32_t* tmem_slot = reinterpret_cast<volatile uint32_t*>(smem + SM::kTmem);
  volatile int* misc = reinterpret_cast<int*>(smem + SM::kMisc);
  uint32_t* exit_cnt = bar_cnt + kMaxLayers;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = Hq / Hkv;
  const int R = g * (kAttnRows / g);  // rows per group: whole block positions
  const int n_layers = set.n;
  const uint32_t n_ctas = gridDim.x;
  // the tensor maps' first use then finds them on chip
  if (warp == kProducerWarp)
    for (int l = lane; l < n_layers; l += 32) {
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&set.Q[l])) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&set.K[l])) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&set.V[l])) : "memory");
    }
  // the plan reads kv_len and L from shared memory when the batch fits
  const bool plan_cached = B <= SM::kPlanCap;
  int32_t* plan_kv = reinterpret_cast<int32_t*>(smem + SM::kPlan);
  int32_t* plan_L = plan_kv + SM::kPlanCap;
  const int32_t* kvs = plan_cached ? plan_kv : kv_len;
  const int32_t* Lss = plan_cached ? plan_L : Ls;

  if (tid == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(bFull + 8 * s, 1);
      mbar_init(bEmpty + 8 * s, 1);  // the MMA warp's commit after the tile's PV
    }
    for (int q = 0; q < 2; ++q) {
      mbar_init(bQFull + 8 * q, 1);                   // the producer's arrive; Q bytes as transactions
      mbar_init(bQEmpty + 8 * q, 1 + kSoftmaxWarps);  // MMA commit (Q read) + softmax warps (info read)
      mbar_init(bSFull + 8 * q, 1);
      mbar_init(bSFree + 8 * q, kSoftmaxWarps);
      mbar_init(bOFree + 8 * q, kSoftmaxWarps);
    }
    for (int p = 0; p < kPBufs; ++p) {
      mbar_init(bPFull + 8 * p, kSoftmaxWarps);
      mbar_init(bPVDone + 8 * p, 1);
    }
    mbar_init(bDrain, 1);
    misc[0] = 0;
    misc[4] = 0;
    misc[5] = 0;
    misc[6] = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == kMmaWarp) {
    // one CTA per SM: the whole tensor memory
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(const_cast<uint32_t*>(tmem_slot))),
                 "n"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  // The plan (identical for every layer): this CTA's tile range, its item
  // count and the split groups it helps merge.
  if (warp == 0) {
    if (plan_cached) {
      // one round trip: four sequences per lane in flight
      for (int b0 = 0; b0 < B; b0 += 128) {
        int kv4[4], L4[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int b = b0 + u * 32 + lane;
          kv4[u] = b < B ? kv_len[b] : 0;
          L4[u] = b < B ? Ls[b] : 0;
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int b = b0 + u * 32 + lane;
          if (b < B) {
            plan_kv[b] = kv4[u];
            plan_L[b] = L4[u];
          }
        }
      }
      __syncwarp();
    }
    long long NG = 0;
    const long long T = total_tiles(B, kvs, Lss, K, g, R, Hkv, S_cap, status, blockIdx.x == 0, &NG);
    int G = (int)n_ctas;
    if (T > 0) {
      const long long g_cap = div_nn(T + min_tiles - 1, min_tiles);
      if ((long long)G > g_cap) G = (int)g_cap;
    }
    const int c = blockIdx.x;
    // weighted length (the unweighted instantiation splits by tiles alone)
    const long long W = WEIGHTED ? T + (long long)item_tiles * NG : T;
    long long lo = 0, hi = 0;
    if (T > 0 && c < G) {
      if constexpr (WEIGHTED) {
        lo = tile_of_weighted(range_lo(c, W, G), W, T, item_tiles, B, kvs, Lss, K, g, R, Hkv, S_cap);
        hi = tile_of_weighted(range_lo(c + 1, W, G), W, T, item_tiles, B, kvs, Lss, K, g, R, Hkv, S_cap);
      } else {
        lo = range_lo(c, T, G);
        hi = range_lo(c + 1, T, G);
      }
    }
    int n_items = 0, n_tasks = 0;
    long long* range = reinterpret_cast<long long*>(smem + SM::kRange);
    if (lane == 0) {
      range[0] = lo;
      range[1] = hi;
    }
    if (lo < hi) {
      int group_lo = 0;
      for (int e = 0; e < 2; ++e) {
        const long long pos = e == 0 ? lo : hi - 1;
        const TileLoc loc = locate_tile(pos, B, kvs, Lss, K, g, R, Hkv, S_cap);
        const int nt = loc.p.n_tiles;
        const int gib = (int)div_nn(pos - loc.seq_start, nt);
        const long long gstart = loc.seq_start + (long long)gib * nt, gend = gstart + nt;
        const int group = loc.group0 + gib;
        if (e == 0) group_lo = group;
        else n_items = group - group_lo + 1;
        if ((gstart < lo || gend > hi) && !(e == 1 && group == group_lo)) {
          if (lane == 0) {
            MergeTask t;
            t.b = loc.b;
            t.kvh = gib / loc.p.n_mg;
            t.mg = gib % loc.p.n_mg;
            t.rows = min(R, loc.p.M - t.mg * R);
            const int C = WEIGHTED ? item_tiles : 0;
            t.c0 = cta_of(weighted_pos(gstart, group, C), W, G);
            t.np = cta_of(weighted_pos(gend - 1, group, C), W, G) - t.c0 + 1;
            t.grp = group;
            t.epi = (long long)t.rows * (D / 4) * t.np <= kEpiMaxItems ? 1 : 0;
            tasks[n_tasks] = t;
          }
          ++n_tasks;
        }
      }
    }
    if (lane == 0) {
      misc[1] = n_tasks;
      misc[2] = n_items;
      misc[3] = merge_chunk_count<D>(tasks, n_tasks);  // merge chunks per layer
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const int n_tasks = misc[1], n_items = misc[2], merge_n = misc[3];
  int* merge_claimed = const_cast<int*>(misc) + 4;
  int* merge_done = const_cast<int*>(misc) + 5;
  // bounded wait until every CTA has finished `layer` (lane 0 polls)
  auto layer_done = [&](int layer) {
    bool ok = false;
    if ((threadIdx.x & 31) == 0) ok = wait_counter(bar_cnt + layer, n_ctas) && !misc[0];
    return __shfl_sync(0xffffffffu, ok, 0) != 0;
  };
  // bounded wait (warp-wide) until the merge warp has seen every split group
  // of the last layer complete
  auto last_groups_ready = [&]() {
    bool ok = false;
    if ((threadIdx.x & 31) == 0) {
      for (int i = 0; i < kMaxWaitIters; ++i) {
        if (misc[6]) { ok = true; break; }
        if (misc[0]) break;
        __nanosleep(64);
      }
    }
    return __shfl_sync(0xffffffffu, ok, 0) != 0;
  };
  // bounded wait (one lane) until the CTA has merged n chunks
  auto merged_upto = [&](int n) {
    for (int i = 0; i < kMaxWaitIters; ++i) {
      if (*reinterpret_cast<volatile int*>(merge_done) >= n) return true;
      if (misc[0]) return false;
      __nanosleep(64);
    }
    return false;
  };
  const uint32_t tmem = *tmem_slot;

  if (warp == kProducerWarp) {
    // ======================= producer =======================
    const int c = blockIdx.x;
    const long long lo = reinterpret_cast<const long long*>(smem + SM::kRange)[0];
    const long long hi = reinterpret_cast<const long long*>(smem + SM::kRange)[1];
    uint32_t item_ctr = 0, tile_ctr = 0;
    // lane 0 reads the abort flag for the whole warp (the loop body has warp-wide steps)
    auto aborted = [&]() { return __shfl_sync(0xffffffffu, misc[0], 0) != 0; };
    // paged: the page of every tile of the range, read once for all layers
    // (they share the block table); a range beyond the cache reads the
    // table tile by tile
    int32_t* tile_page = reinterpret_cast<int32_t*>(smem + SM::kBytes);
    const bool pages_cached = PAGED && hi - lo <= page_cache;
    auto page_of = [&](int b, int key) {
      int id = __ldg(block_table + (size_t)b * max_pages + key / page_size);
      if (id < 0 || id >= n_pages) {
        raise_status(status, LIBRASPEC_ST_BAD_PAGE);
        id = 0;  // read a valid page; the sequence's output is then meaningless
      }
      return id;
    };
    if (pages_cached) {
      for (long long pos = lo; pos < hi;) {
        const TileLoc loc = locate_tile(pos, B, kvs, Lss, K, g, R, Hkv, S_cap);
        const int nt = loc.p.n_tiles;
        const long long gstart = loc.seq_start + div_nn(pos - loc.seq_start, nt) * nt;
        const long long iend = gstart + nt < hi ? gstart + nt : hi;
        const int key0 = (int)(pos - gstart) * kAttnTileKeys;
        for (int i = lane; i < (int)(iend - pos); i += 32)
          tile_page[pos - lo + i] = page_of(loc.b, key0 + i * kAttnTileKeys);
        pos = iend;
      }
      __syncwarp();
    }
    for (int layer = 0; layer < n_layers && !aborted(); ++layer) {
      // layer's dependent data (Q, the block's keys) is readable once every
      // CTA has finished the previous layer
      bool ready = layer == 0;
      for (long long pos = lo; pos < hi && !aborted();) {
        ItemInfo it{};
        const TileLoc loc = locate_tile(pos, B, kvs, Lss, K, g, R, Hkv, S_cap);
        const int nt = loc.p.n_tiles;
        const int gib = (int)div_nn(pos - loc.seq_start, nt);
        const long long gstart = loc.seq_start + (long long)gib * nt;
        const long long gend = gstart + nt;
        const long long iend = gend < hi ? gend : hi;
        it.b = loc.b;
        it.kvh = gib / loc.p.n_mg;
        it.mg = gib % loc.p.n_mg;
        it.rows = min(R, loc.p.M - it.mg * R);
        it.kv = kvs[loc.b];
        it.key0 = (int)(pos - gstart) * kAttnTileKeys;
        it.key1 = min(loc.p.N, (int)(iend - gstart) * kAttnTileKeys);
        it.partial = ((pos == gstart) && (gend <= hi)) ? 0 : 1;
        it.slot = (pos == gstart) ? 2 * c + 1 : 2 * c;
        it.grp = loc.group0 + gib;
        const int n_tiles = (int)(iend - pos);
        const int zc = loc.b * Hkv + it.kvh;
        const long long item_pos = pos;  // the item's first tile in the tile sequence
        pos = iend;
        const uint32_t q = item_ctr % SM::kQSlots;
        if (lane == 0) {
          bool ok = true;
          int issued = 0;
          auto issue_tile = [&](int i) {
            const uint32_t s = tile_ctr % STAGES;
            const uint32_t bar = bFull + 8 * s;
            mbar_expect_tx(bar, 2 * SM::kTileBytes);
            int y = it.key0 + i * kAttnTileKeys, z = zc;
            if (PAGED) {
              const int page = pages_cached ? tile_page[item_pos - lo + i] : page_of(it.b, y);
              z = page * Hkv + it.kvh;
              y %= page_size;
            }
#pragma unroll
            for (int bx = 0; bx < SM::kBoxes; ++bx) {
              tma_load_3d(sK + s * SM::kTileBytes + bx * 8192, &set.K[layer], bar, bx * 64, y, z);
              tma_load_3d(sV + s * SM::kTileBytes + bx * 8192, &set.V[layer], bar, bx * 64, y, z);
            }
            ++tile_ctr;
          };
          // Tiles go out as their stages free, before the item's Q slot is
          // free (the previous item's last S), so the ring does not drain
          // between items; before the layer barrier only tiles that lie
          // wholly in the cache prefix (the block's keys are the previous
          // layer's output).
          // (a free Q slot at once: Q goes first, the item's first S needs it)
          if (!ready) {
            // Q is read once the layer barrier passes; bring it into L2 now
#pragma unroll
            for (int hb = 0; hb < SM::kBoxes; ++hb)
              tma_prefetch_3d(&set.Q[layer], hb * 64, it.kvh * g, it.b * (K + 1) + it.mg * (R / g));
          }
          int n_pre = ready ? n_tiles : min(n_tiles, max(0, (it.kv - it.key0) / kAttnTileKeys));
          // a layer's first item: its prefix tiles go out once the previous
          // layer's last S has read its Q slot (earlier copies only slow the
          // previous layer, whose barrier this layer waits for)
          bool q_free = !ready && mbar_wait(bQEmpty + 8 * q, ((item_ctr / SM::kQSlots) & 1) ^ 1);
          for (int spin = 0;; ++spin) {
            if (!q_free) q_free = mbar_test_wait(bQEmpty + 8 * q, ((item_ctr / SM::kQSlots) & 1) ^ 1);
            if (ready && q_free) break;
            while (issued < n_pre &&
                   mbar_test_wait(bEmpty + 8 * (tile_ctr % STAGES), ((tile_ctr / STAGES) & 1) ^ 1)) {
              issue_tile(issued);
              ++issued;
            }
            if (!ready) {
              uint32_t v;
              asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(bar_cnt + (layer - 1)) : "memory");
              if (v >= n_ctas) {
                ready = true;
                n_pre = n_tiles;
                continue;
              }
            }
            if (spin >= kMaxWaitIters) {
              ok = false;
              break;
            }
            __nanosleep(32);
          }
          if (ok) {
            // Q: R/g positions x g heads of kv head kvh, one box per 64-column half
            info[q] = it;
            mbar_expect_tx(bQFull + 8 * q, (uint32_t)R * D * 2);
            const uint32_t qdst = sQ + q * SM::kQSlot;
#pragma unroll
            for (int hb = 0; hb < SM::kBoxes; ++hb)
              tma_load_3d(qdst + hb * SM::kQBox, &set.Q[layer], bQFull + 8 * q, hb * 64, it.kvh * g,
                          it.b * (K + 1) + it.mg * (R / g));
            for (int i = issued; i < n_tiles && ok; ++i) {
              ok = mbar_wait(bEmpty + 8 * (tile_ctr % STAGES), ((tile_ctr / STAGES) & 1) ^ 1);
              if (ok) issue_tile(i);
            }
          }
          if (!ok) {
            raise_status(status, LIBRASPEC_ST_TIMEOUT);
            misc[0] = 1;
          }
        }
        ready = true;
        ++item_ctr;
        __syncwarp();
      }
    }
    // before leaving, wait (bounded) for this CTA's copies still in flight
    if (lane == 0) {
      for (uint32_t k = 0; k < STAGES && k < tile_ctr; ++k) {
        const uint32_t t = tile_ctr - 1 - k;
        mbar_wait(bFull + 8 * (t % STAGES), (t / STAGES) & 1);
      }
      for (uint32_t k = 0; k < (uint32_t)SM::kQSlots && k < item_ctr; ++k) {
        const uint32_t i = item_ctr - 1 - k;
        mbar_wait(bQFull + 8 * (i % SM::kQSlots), (i / SM::kQSlots) & 1);
      }
    }
    __syncwarp();
  } else if (warp == kMmaWarp) {
    // ======================= MMA issue =======================
    if (lane == 0) {
      constexpr uint32_t kIdescS = mma_idesc(128, kAttnTileKeys, 0);
      constexpr uint32_t kIdescPV = mma_idesc(128, D, 1);
      uint32_t item_ctr = 0, tile_ctr = 0;
      bool ok = true;
      // O[ob] += P(gt) V(gt); the first PV of an item overwrites O
      auto issue_pv = [&](uint32_t gt, uint32_t item, bool first) {
        const uint32_t pb = gt % kPBufs, s = gt % STAGES, ob = item & 1;
        ok = ok && mbar_spin(bPFull + 8 * pb, (gt / kPBufs) & 1);
        if (first) ok = ok && mbar_spin(bOFree + 8 * ob, ((item >> 1) & 1) ^ 1);
        if (!ok) return;
        tc_fence_after();
        const uint32_t vtile = sV + s * SM::kTileBytes;
#pragma unroll
        for (int kc = 0; kc < kAttnTileKeys / 16; ++kc)
          mma_ts(tmem + SM::kColO + ob * D, tmem + SM::kColP + pb * 32 + kc * 8,
                 smem_desc(vtile + kc * 2048, 8192, 1024), kIdescPV, (!first || kc > 0) ? 1u : 0u);
        mma_commit(bPVDone + 8 * pb);
        mma_commit(bEmpty + 8 * s);
      };
      for (int layer = 0; layer < n_layers && ok; ++layer) {
        for (int item = 0; item < n_items && ok; ++item) {
          const uint32_t q = item_ctr % SM::kQSlots;
          ok = mbar_spin(bQFull + 8 * q, (item_ctr / SM::kQSlots) & 1);
          if (!ok) break;
          const ItemInfo it = info[q];
          const int n_tiles = (it.key1 - it.key0 + kAttnTileKeys - 1) / kAttnTileKeys;
          const uint32_t qslot = sQ + q * SM::kQSlot;
          for (int t = 0; t < n_tiles && ok; ++t) {
            const uint32_t gt = tile_ctr;
            const uint32_t s = gt % STAGES, sb = gt & 1;
            ok = mbar_spin(bFull + 8 * s, (gt / STAGES) & 1) && mbar_spin(bSFree + 8 * sb, ((gt >> 1) & 1) ^ 1);
            if (!ok) break;
            tc_fence_after();
            const uint32_t ktile = sK + s * SM::kTileBytes;
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk)
              mma_ss(tmem + SM::kColS + sb * kAttnTileKeys,
                     smem_desc(qslot + (kk >> 2) * SM::kQBox + (kk & 3) * 32, 16, 1024),
                     smem_desc(ktile + (kk >> 2) * 8192 + (kk & 3) * 32, 16, 1024), kIdescS, kk > 0 ? 1u : 0u);
            mma_commit(bSFull + 8 * sb);
            if (t == n_tiles - 1) mma_commit(bQEmpty + 8 * q);
            // the previous tile's PV overlaps this tile's softmax
            if (t > 0) issue_pv(gt - 1, item_ctr, t == 1);
            ++tile_ctr;
          }
          if (ok && n_tiles > 0) issue_pv(tile_ctr - 1, item_ctr, n_tiles == 1);
          ++item_ctr;
        }
      }
      if (!ok) {
        raise_status(status, LIBRASPEC_ST_TIMEOUT);
        misc[0] = 1;
      }
      // every MMA issued has completed before the tensor memory is released
      mma_commit(bDrain);
      mbar_wait(bDrain, 0);
    }
    __syncwarp();
  } else if (warp < kSoftmaxWarps) {
    // ======================= softmax warpgroup =======================
    const int row = warp * 32 + lane;  // tensor-memory lane
    const uint32_t lane_off = (uint32_t)(warp * 32) << 16;
    uint32_t item_ctr = 0, tile_ctr = 0;
    bool ok = true;
    // layer n_layers has no items: it only helps with the last layer's merge
    for (int layer = 0; layer <= n_layers && ok; ++layer) {
      const bool has_items = layer < n_layers;
      float* part_o = part_buf_o + (layer % kAttnPartBufs) * part_o_stride;
      float* part_ml = part_buf_ml + (layer % kAttnPartBufs) * part_ml_stride;
      if (layer > 0 && has_items) {
        // layer's inputs are ready once every CTA is done with the previous layer
        if (tid == 0 && !wait_counter(bar_cnt + (layer - 1), n_ctas)) {
          raise_status(status, LIBRASPEC_ST_TIMEOUT);
          misc[0] = 1;
        }
        softmax_sync();
        if (misc[0]) {
          ok = false;
          break;
        }
      }
      __nv_bfloat16* O = has_items ? set.p[layer].O : nullptr;
      float* lse = has_items ? set.p[layer].lse : nullptr;
      for (int item = 0; item < n_items && ok && has_items; ++item) {
        const uint32_t q = item_ctr % SM::kQSlots, ob = item_ctr & 1;
        ok = warp_wait(bQFull + 8 * q, (item_ctr / SM::kQSlots) & 1);
        if (!ok) break;
        const ItemInfo it = info[q];
        __syncwarp();
        if (lane == 0) mbar_arrive(bQEmpty + 8 * q);  // info read; the Q slot is freed by the MMA commit
        const int n_tiles = (it.key1 - it.key0 + kAttnTileKeys - 1) / kAttnTileKeys;
        const bool valid = row < it.rows;
        // a warp without valid rows only keeps the barrier counts in step
        const bool warp_live = warp * 32 < it.rows;
        const int t_row = (it.mg * R + row) / g;
        // Keys seen by this row: the cache prefix and the root (keys <= kv),
        // then chain: the block positions up to t_row (keys <= kv + t_row);
        // tree: the ancestors of node t_row and itself, bit j of its
        // visibility row <-> key kv + 1 + j.
        const uint64_t* vrow =
            (tree_vis && valid) ? tree_vis + ((size_t)it.b * (K + 1) + t_row) * tree_words : nullptr;
        const int mask_from = tree_vis ? it.kv : it.kv + t_row;  // tiles past this key need the mask
        float m_run = -INFINITY, l_run = 0.f;
        for (int t = 0; t < n_tiles && ok; ++t) {
          const uint32_t gt = tile_ctr;
          const uint32_t sb = gt & 1, pb = gt % kPBufs;
          const int kt0 = it.key0 + t * kAttnTileKeys;
          ok = warp_wait(bSFull + 8 * sb, (gt >> 1) & 1);
          if (!ok) break;
          if (!warp_live) {
            __syncwarp();
            if (lane == 0) {
              mbar_arrive(bSFree + 8 * sb);
              mbar_arrive(bPFull + 8 * pb);
            }
            ++tile_ctr;
            continue;
          }
          tc_fence_after();
          uint32_t sr[2][32];
          tmem_ld32(tmem + lane_off + SM::kColS + sb * kAttnTileKeys, sr[0]);
          tmem_ld32(tmem + lane_off + SM::kColS + sb * kAttnTileKeys + 32, sr[1]);
          tmem_wait_ld();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(bSFree + 8 * sb);
          // raw scores; keys this row does not see (and rows past the
          // group) count as -inf; the scale (> 0) is applied below
          const bool need_mask = !valid || kt0 + kAttnTileKeys - 1 > mask_from;
          uint64_t tmask = ~0ull;  // bit c: key kt0 + c is seen
          if (need_mask) {
            if (!valid) tmask = 0ull;
            else if (!vrow) tmask = low_bits(it.kv + t_row + 1 - kt0);
            else tmask = low_bits(it.kv + 1 - kt0) | bit_window(vrow, tree_words, kt0 - it.kv - 1);
          }
          // two copies of the loop: per-column mask tests that every tile ran
          // took a fifth of the softmax's time on tiles with no masked key
          float xs[kAttnTileKeys];
          float mx[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
          if (need_mask) {
#pragma unroll
            for (int c = 0; c < kAttnTileKeys; ++c) {
              float v = __uint_as_float(sr[c >> 5][c & 31]);
              if (!((tmask >> c) & 1ull)) v = -INFINITY;
              xs[c] = v;
              mx[c & 3] = fmaxf(mx[c & 3], v);
            }
          } else {
#pragma unroll
            for (int c = 0; c < kAttnTileKeys; ++c) {
              xs[c] = __uint_as_float(sr[c >> 5][c & 31]);
              mx[c & 3] = fmaxf(mx[c & 3], xs[c]);
            }
          }
          const float tmax = fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])) * scale_log2;
          // raise the reference max only when it grows by more than 2^8
          float f = 1.f;
          const bool raise = tmax > m_run + kRescaleLog2;
          if (raise) {
            f = (m_run == -INFINITY) ? 0.f : ex2_approx(m_run - tmax);
            m_run = tmax;
          }
          const float neg_m = (m_run == -INFINITY) ? 0.f : -m_run;
          float ls[4] = {0.f, 0.f, 0.f, 0.f};
          uint32_t pk[32];
#pragma unroll
          for (int c = 0; c < kAttnTileKeys; c += 2) {
            const float p0 = ex2_approx(fmaf(xs[c], scale_log2, neg_m));
            const float p1 = ex2_approx(fmaf(xs[c + 1], scale_log2, neg_m));
            ls[(c >> 1) & 3] += p0 + p1;
            pk[c >> 1] = pack_bf16(p0, p1);
          }
          l_run = l_run * f + ((ls[0] + ls[1]) + (ls[2] + ls[3]));
          // O holds the earlier tiles of this item: rescale its rows once the
          // previous tile's PV has landed (rare: the max rose by > 2^8)
          if (t > 0 && __any_sync(0xffffffffu, raise)) {
            ok = warp_wait(bPVDone + 8 * ((gt - 1) % kPBufs), ((gt - 1) / kPBufs) & 1);
            if (!ok) break;
            tc_fence_after();
#pragma unroll 1
            for (int c0 = 0; c0 < D; c0 += 32) {
              uint32_t o[32];
              tmem_ld32(tmem + lane_off + SM::kColO + ob * D + c0, o);
              tmem_wait_ld();
#pragma unroll
              for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * f);
              tmem_st32(tmem + lane_off + SM::kColO + ob * D + c0, o);
            }
            tmem_wait_st();
          }
          // P buffer pb is free once PV(gt - kPBufs) has read it
          if (gt >= kPBufs) {
            ok = warp_wait(bPVDone + 8 * pb, ((gt / kPBufs) & 1) ^ 1);
            if (!ok) break;
            tc_fence_after();
          }
          tmem_st32(tmem + lane_off + SM::kColP + pb * 32, pk);
          tmem_wait_st();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(bPFull + 8 * pb);
          ++tile_ctr;
        }
        if (!ok) break;
        // epilogue: O of this item is complete once the last PV has landed
        {
          const uint32_t last = tile_ctr - 1;
          ok = warp_wait(bPVDone + 8 * (last % kPBufs), (last / kPBufs) & 1);
          if (!ok) break;
          tc_fence_after();
          if (warp_live) {
            const int rr = it.mg * R + row;
            const int hq = it.kvh * g + rr % g;
            const float inv = 1.f / l_run;
            const size_t slot = (size_t)it.slot;
#pragma unroll 1
            for (int c0 = 0; c0 < D; c0 += 32) {
              uint32_t o[32];
              tmem_ld32(tmem + lane_off + SM::kColO + ob * D + c0, o);
              tmem_wait_ld();
              if (valid) {
                if (!it.partial) {
                  uint4* dst =
                      reinterpret_cast<uint4*>(O + (((size_t)it.b * (K + 1) + t_row) * Hq + hq) * D + c0);
#pragma unroll
                  for (int i = 0; i < 4; ++i)
                    dst[i] = make_uint4(
                        pack_bf16(__uint_as_float(o[8 * i]) * inv, __uint_as_float(o[8 * i + 1]) * inv),
                        pack_bf16(__uint_as_float(o[8 * i + 2]) * inv, __uint_as_float(o[8 * i + 3]) * inv),
                        pack_bf16(__uint_as_float(o[8 * i + 4]) * inv, __uint_as_float(o[8 * i + 5]) * inv),
                        pack_bf16(__uint_as_float(o[8 * i + 6]) * inv, __uint_as_float(o[8 * i + 7]) * inv));
                } else {
                  uint4* dst = reinterpret_cast<uint4*>(part_o + (slot * kAttnRows + row) * D + c0);
#pragma unroll
                  for (int i = 0; i < 8; ++i) dst[i] = make_uint4(o[4 * i], o[4 * i + 1], o[4 * i + 2], o[4 * i + 3]);
                }
              }
            }
            if (valid) {
              if (it.partial) {
                *reinterpret_cast<float2*>(part_ml + (slot * kAttnRows + row) * 2) = make_float2(m_run, l_run);
              } else if (lse) {
                lse[((size_t)it.b * (K + 1) + t_row) * Hq + hq] = (m_run + __log2f(l_run)) * kLn2;
              }
            }
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(bOFree + 8 * ob);
          if (it.partial && layer == n_layers - 1)
            last_layer_part_done<D>(tasks, n_tasks, it.grp, grp_cnt, misc, part_o, part_ml, K, Hq, g, R, O, lse);
        }
        ++item_ctr;
      }
      if (!ok) break;
      // This CTA is done with the layer's items. Once its grid barrier
      // passes, CTAs write layer + 1's partials into the buffer of layer - 2,
      // whose merge must be done first. Help with the merge warp's backlog
      // (layers up to layer - 1) if it is large; after the last layer, help
      // with its merge (the tail of the launch) once its barrier has passed.
      if (layer > 0 && merge_n > 0 &&
          (has_items ? layer * merge_n - *reinterpret_cast<volatile int*>(merge_claimed) >= kMergeHelpChunks
                     : last_groups_ready()))
        merge_chunks<D>(layer - 1, set, tasks, n_tasks, merge_n, merge_claimed, merge_done, K, Hq, Hkv, R, part_buf_o,
                        part_buf_ml, part_o_stride, part_ml_stride, n_layers - 1);
      if (!has_items) break;
      if (layer >= kAttnPartBufs - 1 && merge_n > 0 && tid == 0 &&
          !merged_upto((layer - (kAttnPartBufs - 2)) * merge_n)) {
        raise_status(status, LIBRASPEC_ST_TIMEOUT);
        misc[0] = 1;
      }
      softmax_sync();
      if (misc[0]) {
        ok = false;
        break;
      }
      if (tid == 0)
        asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(bar_cnt + layer), "r"(1u) : "memory");
    }
    if (!ok) {
      if (lane == 0) raise_status(status, LIBRASPEC_ST_TIMEOUT);
      misc[0] = 1;
    }
  } else if (warp == kMergeWarp) {
    // ======================= merge warp =======================
    // Layer l's split groups, once every CTA has finished layer l (its grid
    // barrier), while the softmax warps already run the next layers.
    bool ok = true;
    for (int layer = 0; layer < n_layers && ok; ++layer) {
      if (layer < n_layers - 1) {
        ok = layer_done(layer);
      } else {
        // the last layer: each split group once its np parts are counted in
        // (no grid barrier); the last CTA past a group's wait resets its
        // counters for the next launch
        if (lane == 0) {
          for (int ti = 0; ti < n_tasks && ok; ++ti)
            if (!tasks[ti].epi) ok = wait_counter(grp_cnt + 2 * tasks[ti].grp, tasks[ti].np);
          if (ok) {
            misc[6] = 1;  // the softmax warps may help now
            for (int ti = 0; ti < n_tasks; ++ti) {
              if (tasks[ti].epi) continue;
              uint32_t* gc = grp_cnt + 2 * tasks[ti].grp;
              if (atomicAdd(gc + 1, 1u) == (uint32_t)tasks[ti].np - 1) {
                gc[0] = 0u;
                gc[1] = 0u;
              }
            }
          }
        }
        ok = __shfl_sync(0xffffffffu, ok, 0) != 0 && !misc[0];
      }
      if (!ok) break;
      if (merge_n > 0)
        merge_chunks<D>(layer, set, tasks, n_tasks, merge_n, merge_claimed, merge_done, K, Hq, Hkv, R, part_buf_o,
                        part_buf_ml, part_o_stride, part_ml_stride, n_layers - 1);
    }
    // every chunk of every layer is merged (by whichever warp) before the exit count
    if (ok && merge_n > 0 && n_layers > 0) {
      if (lane == 0) ok = merged_upto(n_layers * merge_n);
      ok = __shfl_sync(0xffffffffu, ok, 0) != 0;
    }
    if (!ok && lane == 0 && !misc[0]) {
      raise_status(status, LIBRASPEC_ST_TIMEOUT);
      misc[0] = 1;
    }
    __syncwarp();
  }
  // every role is done with the tensor memory
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (tid == 0 && !misc[0] && n_layers > 0) {
    // the last CTA out resets the barrier counters for the next launch (each
    // CTA has arrived at every layer's barrier by now)
    __threadfence();
    const uint32_t done = atomicAdd(exit_cnt, 1u);
    if (done == n_ctas - 1) {
      for (int l = 0; l < n_layers; ++l) bar_cnt[l] = 0u;
      *exit_cnt = 0u;
      __threadfence();
    }
  }
  if (warp == kMmaWarp)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "n"(kTmemCols) : "memory");
}

// ---------------------------------------------------------------------------
// Host side.
// ---------------------------------------------------------------------------
int num_sms_current();

// Q [B*(K+1), Hq, D] as 3-D; box = 64 columns x g heads x R/g positions (one
// row group of one kv head), 128-byte swizzle.
static bool make_q_map(CUtensorMap* map, const void* base, int D, int Hq, int BT, int g, int R) {
  auto enc = get_encode();
  if (!enc) return false;
  cuuint64_t dims[3] = {(cuuint64_t)D, (cuuint64_t)Hq, (cuuint64_t)BT};
  cuuint64_t strides[2] = {(cuuint64_t)D * 2, (cuuint64_t)Hq * D * 2};
  cuuint32_t box[3] = {64, (cuuint32_t)g, (cuuint32_t)(R / g)};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

static bool make_kv_map(CUtensorMap* map, const void* base, int D, int S_cap, int BH) {
  auto enc = get_encode();
  if (!enc) return false;
  cuuint64_t dims[3] = {(cuuint64_t)D, (cuuint64_t)S_cap, (cuuint64_t)BH};
  cuuint64_t strides[2] = {(cuuint64_t)D * 2, (cuuint64_t)S_cap * D * 2};
  cuuint32_t box[3] = {64, (cuuint32_t)kAttnTileKeys, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// Smallest tile range per CTA; the LIBRASPEC_ATTN_MIN_TILES environment
// variable overrides the default, read once per process.
static int attn_min_tiles() {
  static int t = [] {
    int v = 2;
    if (const char* e = getenv("LIBRASPEC_ATTN_MIN_TILES")) {
      int a = 0;
      if (sscanf(e, "%d", &a) == 1 && a >= 1 && a <= 4096) v = a;
    }
    return v;
  }();
  return t;
}

// Tile-equivalents an item costs in the Stream-K split (see
// tile_of_weighted); the LIBRASPEC_ATTN_ITEM_TILES environment variable
// overrides the default, read once per process.
static int attn_item_tiles() {
  static int t = [] {
    int v = 2;
    if (const char* e = getenv("LIBRASPEC_ATTN_ITEM_TILES")) {
      int a = 0;
      if (sscanf(e, "%d", &a) == 1 && a >= 0 && a <= 64) v = a;
    }
    return v;
  }();
  return t;
}

// Ancestor sets of a draft tree, one CTA per sequence, by pointer jumping:
// after round r, m[t] holds the nodes on the path from t up to (not
// including) up[t], the ancestor at distance 2^r (the root absorbs: m[0] =
// 0, up[0] = 0); rounds stop once every up[] is the root (depth <= 2^r).
// vis[b, t] = m[t] as `words` 64-bit words, bit j <-> block position j + 1;
// rows t > L_b get 0. A parent outside [0, t) raises LIBRASPEC_ST_BAD_TREE
// and is read as the root. Each round reads all (node, word) pairs into
// registers before any is written.
constexpr int kTreeThreads = 256;
constexpr int kTreeWords = (LIBRASPEC_MAX_TREE_NODES + 63) / 64;
constexpr int kTreePer = ((LIBRASPEC_MAX_TREE_NODES + 1) * kTreeWords + kTreeThreads - 1) / kTreeThreads;

__global__ void __launch_bounds__(kTreeThreads) tree_vis_kernel(const int32_t* __restrict__ parent,
                                                                 const int32_t* __restrict__ Ls, int K, int words,
                                                                 uint64_t* __restrict__ vis,
                                                                 int* __restrict__ status) {
  __shared__ int up[LIBRASPEC_MAX_TREE_NODES + 1];
  __shared__ uint64_t m[(LIBRASPEC_MAX_TREE_NODES + 1) * kTreeWords];
  const int b = blockIdx.x, tid = threadIdx.x;
  int Lb = Ls[b];
  if (Lb < 0 || Lb > K) Lb = 0;  // the attention kernel reports the bad length
  const int pairs = (K + 1) * words;
  for (int t = tid; t <= K; t += kTreeThreads) {
    int p = 0;
    if (t >= 1 && t <= Lb) {
      p = parent[(size_t)b * (K + 1) + t];
      if (p < 0 || p >= t) {
        raise_status(status, LIBRASPEC_ST_BAD_TREE);
        p = 0;
      }
    }
    up[t] = p;
  }
  for (int i = tid; i < pairs; i += kTreeThreads) {
    const int t = i / words, w = i % words;
    m[i] = (t >= 1 && t <= Lb && (t - 1) / 64 == w) ? 1ull << ((t - 1) % 64) : 0ull;
  }
  __syncthreads();
  for (int r = 0; r < 16; ++r) {  // depth <= 512 needs at most 10 rounds
    uint64_t nm[kTreePer];
    int nu[kTreePer];
    bool more = false;
#pragma unroll
    for (int k = 0; k < kTreePer; ++k) {
      const int i = tid + k * kTreeThreads;
      if (i < pairs) {
        const int t = i / words, w = i % words;
        const int u = up[t];
        nm[k] = m[i] | m[u * words + w];
        nu[k] = up[u];
        more |= nu[k] != 0;
      }
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < kTreePer; ++k) {
      const int i = tid + k * kTreeThreads;
      if (i < pairs) {
        m[i] = nm[k];
        if (i % words == 0) up[i / words] = nu[k];
      }
    }
    if (!__syncthreads_or(more)) break;
  }
  for (int i = tid; i < pairs; i += kTreeThreads) vis[(size_t)b * pairs + i] = m[i];
}

inline int tree_words(int K) { return K <= 64 ? 1 : (K + 63) / 64; }

// parent != nullptr: fill the tree visibility masks of the workspace first.
static cudaError_t tree_vis(const int32_t* parent, const int32_t* L, int B, int K, char* ws, const WsLayout& lay,
                            cudaStream_t stream, const uint64_t** out) {
  *out = nullptr;
  if (!parent) return cudaSuccess;
  auto* vis = reinterpret_cast<uint64_t*>(ws + lay.tree_vis);
  tree_vis_kernel<<<B, kTreeThreads, 0, stream>>>(parent, L, K, tree_words(K), vis,
                                                  reinterpret_cast<int*>(ws + lay.status));
  *out = vis;
  return cudaGetLastError();
}

// Paged caches (block_table != nullptr): Kc / Vc are page pools of n_pages
// pages of page_size keys and S_cap = max_pages * page_size.
// Tiles per CTA whose page ids are cached in shared memory (at most cap);
// the LIBRASPEC_ATTN_PAGE_CACHE environment variable lowers it (0: read the
// block table tile by tile). Read once per process.
static int attn_page_cache(int cap) {
  static int v = [] {
    int a = -1;
    if (const char* e = getenv("LIBRASPEC_ATTN_PAGE_CACHE")) {
      if (sscanf(e, "%d", &a) != 1 || a < 0) a = -1;
    }
    return a;
  }();
  return v < 0 || v > cap ? cap : v;
}

// The tensor maps of a launch cost the host about a microsecond each (3 per
// layer); a caller that runs round after round on the same buffers (the
// staged round) gets them from this per-thread cache of the last launch of
// each chunk of layers, keyed by every pointer and shape they encode.
struct LayerSetCache {
  bool valid = false;
  int rows = 0, planes = 0, Hq = 0, BT = 0, g = 0, R = 0;
  const void* Kp[kMaxLayers];
  const void* Vp[kMaxLayers];
  LayerSet set;
};
constexpr int kCachedChunks = 4;

template <int D, int STAGES, bool PAGED>
static cudaError_t launch_layers_t(const uint16_t* const* Q, const uint16_t* const* Kc, const uint16_t* const* Vc,
                                   int n_layers, const int32_t* kv_len, const int32_t* L, const uint64_t* tree_vis,
                                   const int32_t* block_table,
                                   int max_pages, int page_size, int n_pages, int B, int K, int Hq, int Hkv, int S_cap,
                                   float scale, uint16_t* const* O, float* const* lse, char* ws, const WsLayout& lay,
                                   cudaStream_t stream) {
  using SM = AttnSmem<D, STAGES>;
  constexpr int kSmem = PAGED ? SM::kAllocPaged : SM::kAlloc;
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(verify_attn_kernel<D, STAGES, PAGED, false>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(verify_attn_kernel<D, STAGES, PAGED, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               kSmem);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  int grid = num_sms_current();  // one CTA per SM (it holds all 512 tensor-memory columns)
  if (grid > kAttnMaxCtas) grid = kAttnMaxCtas;
  // The cost-weighted split pays where CTAs hold many items: more (sequence,
  // kv head) pairs than CTAs. Otherwise the instantiation without it runs
  // (its code alone measured 2.5% faster on the latency-bound B = 1 layers).
  const int item_tiles = attn_item_tiles();
  const bool weighted = item_tiles > 0 && (long long)B * Hkv > grid;
  auto kern = weighted ? verify_attn_kernel<D, STAGES, PAGED, true> : verify_attn_kernel<D, STAGES, PAGED, false>;
  const int g = Hq / Hkv;
  const int R = g * (kAttnRows / g);
  // layers beyond kMaxLayers go in further launches of the same kernel
  for (int l0 = 0; l0 < n_layers; l0 += kMaxLayers) {
    const int n = n_layers - l0 < kMaxLayers ? n_layers - l0 : kMaxLayers;
    // dense: [B*Hkv, S_cap, D]; paged: [n_pages*Hkv, page_size, D]
    const int rows = PAGED ? page_size : S_cap;
    const int planes = PAGED ? n_pages * Hkv : B * Hkv;
    const int BT = B * (K + 1);
    static thread_local std::unique_ptr<LayerSetCache[]> caches;
    const int ci = l0 / kMaxLayers;
    LayerSetCache* c = nullptr;
    if (ci < kCachedChunks) {
      if (!caches) caches.reset(new (std::nothrow) LayerSetCache[kCachedChunks]);
      if (caches) c = &caches[ci];
    }
    bool hit = c && c->valid && c->set.n == n && c->rows == rows && c->planes == planes && c->Hq == Hq &&
               c->BT == BT && c->g == g && c->R == R;
    for (int i = 0; i < n && hit; ++i) {
      const int l = l0 + i;
      hit = c->Kp[i] == Kc[l] && c->Vp[i] == Vc[l] && c->set.p[i].Q == reinterpret_cast<const __nv_bfloat16*>(Q[l]) &&
            c->set.p[i].O == reinterpret_cast<__nv_bfloat16*>(O[l]) && c->set.p[i].lse == (lse ? lse[l] : nullptr);
    }
    LayerSet local;
    LayerSet& set = c ? c->set : local;  // ~26 KB: built on the host, copied into the launch parameters
    if (!hit) {
      if (c) c->valid = false;
      set.n = n;
      for (int i = 0; i < n; ++i) {
        const int l = l0 + i;
        if (!make_kv_map(&set.K[i], Kc[l], D, rows, planes) || !make_kv_map(&set.V[i], Vc[l], D, rows, planes) ||
            !make_q_map(&set.Q[i], Q[l], D, Hq, BT, g, R))
          return cudaErrorInvalidValue;
        set.p[i].Q = reinterpret_cast<const __nv_bfloat16*>(Q[l]);
        set.p[i].O = reinterpret_cast<__nv_bfloat16*>(O[l]);
        set.p[i].lse = lse ? lse[l] : nullptr;
        if (c) {
          c->Kp[i] = Kc[l];
          c->Vp[i] = Vc[l];
        }
      }
      if (c) {
        c->rows = rows;
        c->planes = planes;
        c->Hq = Hq;
        c->BT = BT;
        c->g = g;
        c->R = R;
        c->valid = true;
      }
    }
    // one partial buffer's share, kept 256-byte aligned
    const size_t o_part = ((lay.attn_ml - lay.attn_o) / kAttnPartBufs) & ~size_t(255);
    const size_t ml_part = ((lay.attn_cnt - lay.attn_ml) / kAttnPartBufs) & ~size_t(255);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kAttnThreads);
    cfg.dynamicSmemBytes = kSmem;
    cfg.stream = stream;
    // cooperative: every CTA is resident at once, which the layer barriers rely on
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cudaError_t e = cudaLaunchKernelEx(
        &cfg, kern, set, kv_len, L, tree_vis, tree_words(K), block_table, max_pages, page_size, n_pages, attn_page_cache(SM::kPageCap), B, K,
        Hq, Hkv, S_cap, scale * kLog2e, attn_min_tiles(), item_tiles,
        reinterpret_cast<float*>(ws + lay.attn_o), reinterpret_cast<float*>(ws + lay.attn_ml), o_part / sizeof(float),
        ml_part / sizeof(float), reinterpret_cast<uint32_t*>(ws + lay.attn_cnt),
        reinterpret_cast<uint32_t*>(ws + lay.attn_grp), reinterpret_cast<int*>(ws + lay.status));
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

// parent (optional, [B, K+1]): the block is a draft tree (nullptr: the chain).
cudaError_t launch_verify_attn_layers(const uint16_t* const* Q, const uint16_t* const* Kc,
                                      const uint16_t* const* Vc, int n_layers, const int32_t* parent,
                                      const int32_t* kv_len, const int32_t* L, int B, int K, int Hq, int Hkv, int D,
                                      int S_cap, float scale, uint16_t* const* O, float* const* lse, char* ws,
                                      const WsLayout& lay, cudaStream_t stream) {
  if (B == 0 || n_layers == 0) return cudaSuccess;
  const uint64_t* vis = nullptr;
  cudaError_t e = tree_vis(parent, L, B, K, ws, lay, stream, &vis);
  if (e != cudaSuccess) return e;
  if (D == 128)
    return launch_layers_t<128, 5, false>(Q, Kc, Vc, n_layers, kv_len, L, vis, nullptr, 0, 0, 0, B, K, Hq, Hkv, S_cap,
                                          scale, O, lse, ws, lay, stream);
  return launch_layers_t<64, 8, false>(Q, Kc, Vc, n_layers, kv_len, L, vis, nullptr, 0, 0, 0, B, K, Hq, Hkv, S_cap,
                                       scale, O, lse, ws, lay, stream);
}

cudaError_t launch_verify_attn_paged_layers(const uint16_t* const* Q, const uint16_t* const* Kp,
                                            const uint16_t* const* Vp, int n_layers, const int32_t* parent,
                                            const int32_t* block_table, int max_pages, int page_size, int n_pages,
                                            const int32_t* kv_len, const int32_t* L, int B, int K, int Hq, int Hkv,
                                            int D, float scale, uint16_t* const* O, float* const* lse, char* ws,
                                            const WsLayout& lay, cudaStream_t stream) {
  if (B == 0 || n_layers == 0) return cudaSuccess;
  const int S_cap = max_pages * page_size;
  const uint64_t* vis = nullptr;
  cudaError_t e = tree_vis(parent, L, B, K, ws, lay, stream, &vis);
  if (e != cudaSuccess) return e;
  if (D == 128)
    return launch_layers_t<128, 5, true>(Q, Kp, Vp, n_layers, kv_len, L, vis, block_table, max_pages, page_size,
                                         n_pages, B, K, Hq, Hkv, S_cap, scale, O, lse, ws, lay, stream);
  return launch_layers_t<64, 8, true>(Q, Kp, Vp, n_layers, kv_len, L, vis, block_table, max_pages, page_size, n_pages,
                                      B, K, Hq, Hkv, S_cap, scale, O, lse, ws, lay, stream);
}

cudaError_t launch_verify_attn(const uint16_t* Q, const uint16_t* Kc, const uint16_t* Vc, const int32_t* kv_len,
                               const int32_t* L, int B, int K, int Hq, int Hkv, int D, int S_cap, float scale,
                               uint16_t* O, float* lse, char* ws, const WsLayout& lay, cudaStream_t stream) {
  float* lse_arr[1] = {lse};
  return launch_verify_attn_layers(&Q, &Kc, &Vc, 1, nullptr, kv_len, L, B, K, Hq, Hkv, D, S_cap, scale, &O,
                                   lse ? lse_arr : nullptr, ws, lay, stream);
}

}  // namespace libraspec
