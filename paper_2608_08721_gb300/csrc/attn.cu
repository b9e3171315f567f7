// Step 3: block-causal GQA verify attention on GB300 (split-KV, Stream-K,
// warp-specialised persistent CTAs, all layers of a round in one launch).
//
// Work decomposition. For sequence b the verified block has M_b = (L_b+1)*g
// query rows per kv head (g = Hq/Hkv; row r is block position t = r / g of
// query head kvh*g + r % g) and N_b = kv_len_b + L_b + 1 visible keys. Rows
// are cut into groups of 64 (one m16 tile per consumer warp) and keys into
// 64-key tiles. All (row group, key tile) pairs of the batch form one tile
// sequence (sequence-major, then kv head, row group, key tile); CTA c of the
// persistent grid takes the contiguous range [c*T/G, (c+1)*T/G) of it, so
// every CTA streams the same number of tiles whatever the ragged lengths.
// The plan is derived on the device from L[] and kv_len[] by every CTA, and
// it is the same for every layer (all layers share L and kv_len).
//
// Inside a CTA one producer warp walks the CTA's range layer after layer: for
// each run of tiles of one row group (an "item") it loads the group's Q rows
// into a double-buffered shared slot (cp.async) and issues the K/V tiles by
// TMA (3-D tensor map per layer, 128-byte swizzle) into a ring of STAGES
// stages. Four consumer warps compute S = Q K^T and O += P V with
// mma.sync m16n8k16 (bf16 in, fp32 accumulate), mask keys beyond
// kv_len_b + t and keep an online softmax in the log2 domain; with few rows
// the warps also split each tile's keys. Full/empty mbarriers hand stages
// between the two roles.
//
// Layers. Layer l+1 may read Q, the block's own keys (positions >= kv_len_b)
// and the merged output of layer l only after every CTA has finished layer l:
// a grid-wide barrier (one counter per layer; the launch is cooperative, so
// all CTAs are resident and the bounded waits end). The cache prefix
// (keys < kv_len_b) is state from earlier rounds, so the producer streams the
// next layer's prefix tiles while the consumers still finish the current
// layer: HBM stays busy across layer boundaries.
//
// Split groups. A row group covered by one CTA is written directly. A group
// spread over CTAs c0..c1 leaves one fp32 partial (O, m, l) per CTA, in slot
// 2c+1 for c0 (its last item) and 2c for the others (their first item), in a
// buffer chosen by the layer parity. After the barrier that ends layer l,
// each of those CTAs merges its share of the group's rows from all parts in
// CTA order (deterministic, spread over every contributing SM).
#include <cuda.h>
#include <cudaTypedefs.h>

#include <cstdio>
#include <cstdlib>

#include "common.cuh"

namespace libraspec {

constexpr int kConsumerWarps = 4;
constexpr int kAttnThreads = (kConsumerWarps + 1) * 32;
constexpr int kProducerWarp = kConsumerWarps;
constexpr int kMaxWaitIters = 1 << 24;
constexpr int kConsumerBar = 1;  // named barrier of the consumer warps

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ bool mbar_test_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait: false after kMaxWaitIters polls (each poll may suspend).
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
  for (int i = 0; i < kMaxWaitIters; ++i)
    if (mbar_try_wait(bar, parity)) return true;
  return false;
}

__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* map, uint32_t bar, int x, int y,
                                            int z) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(bar)
      : "memory");
}

// Bulk async copy global -> shared of `bytes` (multiple of 16; both addresses
// 16-byte aligned), completing as transaction bytes on `bar`.
__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
               "l"(src), "r"(bytes), "r"(bar)
               : "memory");
}

__device__ __forceinline__ void consumer_sync() {
  asm volatile("bar.sync %0, %1;" ::"n"(kConsumerBar), "n"(kConsumerWarps * 32) : "memory");
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                          uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

__device__ __forceinline__ void mma_bf16(float* d, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// Byte offset of (row, col) in a [64 rows][D] bf16 tile held as D/64 boxes of
// 64 rows x 128 bytes with the 128-byte swizzle (16-byte chunk index XOR
// row % 8). col is a multiple of 8.
__device__ __forceinline__ uint32_t sw128(int row, int col) {
  const int box = col >> 6, chunk = (col & 63) >> 3;
  return (uint32_t)(box * 8192 + row * 128 + ((chunk ^ (row & 7)) << 4));
}

// ---------------------------------------------------------------------------
// Device-side plan.
// ---------------------------------------------------------------------------
struct SeqPlan {
  int M, n_mg, N, n_tiles;  // rows, row groups, visible keys, key tiles
  bool ok;
};

__device__ __forceinline__ SeqPlan seq_plan(int b, int B, const int32_t* kv_len, const int32_t* Ls, int K, int g,
                                            int S_cap) {
  SeqPlan p{0, 0, 0, 0, false};
  if (b >= B) return p;
  const int Lb = Ls[b], kv = kv_len[b];
  if (Lb < 0 || Lb > K || kv < 0 || (long)kv + Lb + 1 > S_cap) return p;
  p.ok = true;
  p.M = (Lb + 1) * g;
  p.n_mg = (p.M + kAttnRows - 1) / kAttnRows;
  p.N = kv + Lb + 1;
  p.n_tiles = (p.N + kAttnTileKeys - 1) / kAttnTileKeys;
  return p;
}

// Warp-wide: total tiles T of the batch; flags invalid sequences.
__device__ long long total_tiles(int B, const int32_t* kv_len, const int32_t* Ls, int K, int g, int Hkv,
                                 int S_cap, int* status, bool report) {
  const int lane = threadIdx.x & 31;
  long long tot = 0;
  bool bad = false;
  for (int b = lane; b < B; b += 32) {
    const SeqPlan p = seq_plan(b, B, kv_len, Ls, K, g, S_cap);
    if (!p.ok) bad = true;
    else tot += (long long)Hkv * p.n_mg * p.n_tiles;
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) tot += __shfl_xor_sync(0xffffffffu, tot, off);
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

__device__ TileLoc locate_tile(long long pos, int B, const int32_t* kv_len, const int32_t* Ls, int K, int g, int Hkv,
                               int S_cap) {
  const int lane = threadIdx.x & 31;
  TileLoc loc{-1, 0, 0, {}};
  long long carry_t = 0;
  int carry_g = 0;
  for (int base = 0; base < B; base += 32) {
    const int b = base + lane;
    const SeqPlan p = seq_plan(b, B, kv_len, Ls, K, g, S_cap);
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
      loc.p = seq_plan(loc.b, B, kv_len, Ls, K, g, S_cap);
      return loc;
    }
    carry_t += __shfl_sync(0xffffffffu, inc_t, 31);
    carry_g += __shfl_sync(0xffffffffu, inc_g, 31);
  }
  return loc;
}

__device__ __forceinline__ long long range_lo(int c, long long T, int G) { return (long long)c * T / G; }

// CTA whose range holds tile t: the largest c with c*T/G <= t.
__device__ __forceinline__ int cta_of(long long t, long long T, int G) {
  return (int)(((t + 1) * (long long)G - 1) / T);
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

// One item handed from the producer to the consumers.
struct ItemInfo {
  int layer;
  int b, kvh, mg, rows, kv;
  int key0, key1;     // keys [key0, key1)
  int partial;        // 1: write a partial, else write O
  int slot;           // partial slot
  int pad[3];
};

// A split row group this CTA helps merge (the same for every layer).
struct MergeTask {
  int b, kvh, mg, rows, c0, np;
};

constexpr int kMaxLayers = kAttnMaxLayers;
constexpr int kMaxParts = kAttnMaxCtas;  // parts of one split group <= grid size

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
  CUtensorMap Q[kMaxLayers];  // used when g divides 64 (q_tma)
  LayerPtrs p[kMaxLayers];
  int n;
  int q_tma;
};
static_assert(sizeof(LayerSet) <= 32000, "kernel parameters are limited to 32764 bytes");

template <int D, int STAGES>
struct AttnSmem {
  static constexpr int kBoxes = D / 64;
  static constexpr int kTileBytes = kBoxes * 8192;  // one 64 x D bf16 tile
  // 2 Q slots; each also serves as the key-split combine scratch of its item
  // (two 16-row fp32 partials with their (m, l)), so it is rounded up to 1 KB
  static constexpr int kQSlot = ((kTileBytes > 2 * (16 * D + 32) * 4 ? kTileBytes : 2 * (16 * D + 32) * 4) +
                                 1023) / 1024 * 1024;
  static constexpr int kQ = 0;
  static constexpr int kK = kQ + 2 * kQSlot;
  static constexpr int kV = kK + STAGES * kTileBytes;
  static constexpr int kBar = kV + STAGES * kTileBytes;  // full[S], empty[S], qfull[2], qempty[2]
  static constexpr int kInfo = kBar + 8 * (2 * STAGES + 4);
  static constexpr int kTasks = kInfo + 2 * 64;
  // merge scratch: (m or weight, l) for rows x parts of one share, whose
  // product is at most kAttnRows + kMaxParts, then 1/L and lse of its rows
  static constexpr int kMergeCap = kAttnRows + kMaxParts;
  static constexpr int kMergeW = kTasks + 64;
  static constexpr int kMisc = kMergeW + (2 * kMergeCap + 2 * kAttnRows) * 4;
  static constexpr int kBytes = kMisc + 16;
  static constexpr int kAlloc = kBytes + 1024;           // room to align the base to 1024
};

// Merge, for layer l's split groups this CTA contributed to, its share of
// rows [rows*k/np, rows*(k+1)/np) (k = this CTA's index among the group's np
// CTAs): O = sum_p w_p O_p / sum_p w_p l_p, w_p = 2^(m_p - M), M = max m_p,
// parts in CTA order. Consumer warps only. Three batched phases (all (m, l)
// of the share; weights and sums per row; the weighted O rows), so that each
// phase issues all of its loads at once.
template <int D, int STAGES>
__device__ void merge_layer(uint8_t* smem, const MergeTask* tasks, int n_tasks, int K, int Hq, int Hkv,
                            const float* __restrict__ part_o, const float* __restrict__ part_ml,
                            __nv_bfloat16* __restrict__ O, float* __restrict__ lse) {
  using SM = AttnSmem<D, STAGES>;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  constexpr int kT = kConsumerWarps * 32;
  constexpr int C4 = D / 4;  // float4 columns of a row
  const int g = Hq / Hkv;
  float* m_sh = reinterpret_cast<float*>(smem + SM::kMergeW);  // [nr * np] m, then weights
  float* l_sh = m_sh + SM::kMergeCap;                           // [nr * np] l
  float* row_sh = l_sh + SM::kMergeCap;                         // [nr] 1/L, [nr] lse (log2)
  for (int ti = 0; ti < n_tasks; ++ti) {
    const MergeTask it = tasks[ti];
    const int c0 = it.c0, np = it.np;
    const int k_me = (int)blockIdx.x - c0;
    const int u0 = (int)((long long)it.rows * k_me / np), u1 = (int)((long long)it.rows * (k_me + 1) / np);
    const int nr = u1 - u0;
    if (nr <= 0) continue;
    auto slot_of = [&](int p) { return (size_t)(p == 0 ? 2 * c0 + 1 : 2 * (c0 + p)); };
    // 1) (m, l) of every part of every row of the share
    for (int idx = tid; idx < nr * np; idx += kT) {
      const int r = idx / np, p = idx - r * np;
      const float2 ml = __ldcg(reinterpret_cast<const float2*>(part_ml + (slot_of(p) * kAttnRows + u0 + r) * 2));
      m_sh[idx] = ml.x;
      l_sh[idx] = ml.y;
    }
    consumer_sync();
    // 2) per row (one warp): M, the weights, 1/L and lse
    for (int r = warp; r < nr; r += kConsumerWarps) {
      float M = -INFINITY;
      for (int p = lane; p < np; p += 32) M = fmaxf(M, m_sh[r * np + p]);
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
      float Ls = 0.f;
      for (int p = lane; p < np; p += 32) {
        const float mp = m_sh[r * np + p];
        const float w = (mp == -INFINITY) ? 0.f : ex2_approx(mp - M);
        m_sh[r * np + p] = w;
        Ls += w * l_sh[r * np + p];
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) Ls += __shfl_xor_sync(0xffffffffu, Ls, off);
      if (lane == 0) {
        row_sh[r] = 1.f / Ls;
        row_sh[kAttnRows + r] = M + __log2f(Ls);
      }
    }
    consumer_sync();
    // 3) the weighted sum of the part rows, one float4 column per thread
    for (int idx = tid; idx < nr * C4; idx += kT) {
      const int r = idx / C4, c = idx - r * C4;
      const float* wr = m_sh + r * np;
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 8
      for (int p = 0; p < np; ++p) {
        const float4 v =
            __ldcg(reinterpret_cast<const float4*>(part_o + (slot_of(p) * kAttnRows + u0 + r) * D) + c);
        const float w = wr[p];
        acc.x += w * v.x;
        acc.y += w * v.y;
        acc.z += w * v.z;
        acc.w += w * v.w;
      }
      const float inv = row_sh[r];
      const int rr = it.mg * kAttnRows + u0 + r;
      const int t = rr / g, hq = it.kvh * g + rr % g;
      __nv_bfloat16* dst = O + (((size_t)it.b * (K + 1) + t) * Hq + hq) * D + c * 4;
      *reinterpret_cast<__nv_bfloat162*>(dst) = __floats2bfloat162_rn(acc.x * inv, acc.y * inv);
      *reinterpret_cast<__nv_bfloat162*>(dst + 2) = __floats2bfloat162_rn(acc.z * inv, acc.w * inv);
      if (lse && c == 0) lse[((size_t)it.b * (K + 1) + t) * Hq + hq] = row_sh[kAttnRows + r] * kLn2;
    }
    consumer_sync();  // the scratch is reused by the next task
  }
}

template <int D, int STAGES>
__global__ void __launch_bounds__(kAttnThreads, 2) verify_attn_kernel(
    const __grid_constant__ LayerSet set, const int32_t* __restrict__ kv_len, const int32_t* __restrict__ Ls,
    int B, int K, int Hq, int Hkv, int S_cap, float scale_log2, int min_tiles, float* __restrict__ part_buf_o,
    float* __restrict__ part_buf_ml, size_t part_o_stride, size_t part_ml_stride, uint32_t* __restrict__ bar_cnt,
    int* __restrict__ status) {
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
  ItemInfo* info = reinterpret_cast<ItemInfo*>(smem + SM::kInfo);
  MergeTask* tasks = reinterpret_cast<MergeTask*>(smem + SM::kTasks);
  volatile int* misc = reinterpret_cast<int*>(smem + SM::kMisc);  // [0] abort, [1] n_tasks, [2] n_items
  uint32_t* exit_cnt = bar_cnt + kMaxLayers;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = Hq / Hkv;
  const int n_layers = set.n;
  const uint32_t n_ctas = gridDim.x;

  if (tid == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(bFull + 8 * s, 1);
      mbar_init(bEmpty + 8 * s, kConsumerWarps);
    }
    for (int q = 0; q < 2; ++q) {
      mbar_init(bQFull + 8 * q, 1);  // the producer's arrive; the Q bytes complete as transactions
      mbar_init(bQEmpty + 8 * q, kConsumerWarps);
    }
    misc[0] = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  // The plan (identical for every layer): this CTA's tile range, its item
  // count and the split groups it helps merge.
  if (warp == 0) {
    const long long T = total_tiles(B, kv_len, Ls, K, g, Hkv, S_cap, status, blockIdx.x == 0);
    int G = (int)n_ctas;
    if (T > 0) {
      const long long g_cap = (T + min_tiles - 1) / min_tiles;
      if ((long long)G > g_cap) G = (int)g_cap;
    }
    const int c = blockIdx.x;
    int n_items = 0, n_tasks = 0;
    if (T > 0 && c < G) {
      const long long lo = range_lo(c, T, G), hi = range_lo(c + 1, T, G);
      int group_lo = 0;
      for (int e = 0; e < 2; ++e) {
        const long long pos = e == 0 ? lo : hi - 1;
        const TileLoc loc = locate_tile(pos, B, kv_len, Ls, K, g, Hkv, S_cap);
        const int nt = loc.p.n_tiles;
        const int gib = (int)((pos - loc.seq_start) / nt);
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
            t.rows = min(kAttnRows, loc.p.M - t.mg * kAttnRows);
            t.c0 = cta_of(gstart, T, G);
            t.np = cta_of(gend - 1, T, G) - t.c0 + 1;
            tasks[n_tasks] = t;
          }
          ++n_tasks;
        }
      }
    }
    if (lane == 0) {
      misc[1] = n_tasks;
      misc[2] = n_items;
    }
  }
  __syncthreads();
  const int n_tasks = misc[1], n_items = misc[2];

  if (warp == kProducerWarp) {
    // ======================= producer =======================
    const long long T = total_tiles(B, kv_len, Ls, K, g, Hkv, S_cap, status, false);
    int G = (int)n_ctas;
    if (T > 0) {
      const long long g_cap = (T + min_tiles - 1) / min_tiles;
      if ((long long)G > g_cap) G = (int)g_cap;
    }
    const int c = blockIdx.x;
    const long long lo = (T > 0 && c < G) ? range_lo(c, T, G) : 0;
    const long long hi = (T > 0 && c < G) ? range_lo(c + 1, T, G) : 0;
    uint32_t item_ctr = 0, tile_ctr = 0;
    for (int layer = 0; layer < n_layers; ++layer) {
      // layer's dependent data (Q, the block's keys) is readable once every
      // CTA has finished the previous layer
      bool ready = layer == 0;
      for (long long pos = lo; pos < hi;) {
        ItemInfo it{};
        const TileLoc loc = locate_tile(pos, B, kv_len, Ls, K, g, Hkv, S_cap);
        const int nt = loc.p.n_tiles;
        const int gib = (int)((pos - loc.seq_start) / nt);
        const long long gstart = loc.seq_start + (long long)gib * nt;
        const long long gend = gstart + nt;
        const long long iend = gend < hi ? gend : hi;
        it.layer = layer;
        it.b = loc.b;
        it.kvh = gib / loc.p.n_mg;
        it.mg = gib % loc.p.n_mg;
        it.rows = min(kAttnRows, loc.p.M - it.mg * kAttnRows);
        it.kv = kv_len[loc.b];
        it.key0 = (int)(pos - gstart) * kAttnTileKeys;
        it.key1 = min(loc.p.N, (int)(iend - gstart) * kAttnTileKeys);
        it.partial = ((pos == gstart) && (gend <= hi)) ? 0 : 1;
        it.slot = (pos == gstart) ? 2 * c + 1 : 2 * c;
        const int n_tiles = (int)(iend - pos);
        const int zc = loc.b * Hkv + it.kvh;
        pos = iend;
        const uint32_t q = item_ctr & 1;
        if (!mbar_wait(bQEmpty + 8 * q, ((item_ctr >> 1) & 1) ^ 1)) {
          if (lane == 0) raise_status(status, LIBRASPEC_ST_TIMEOUT);
          misc[0] = 1;
          return;
        }
        int issued = 0;
        auto issue_tile = [&](int i) {
          const uint32_t s = tile_ctr % STAGES;
          const uint32_t bar = bFull + 8 * s;
          mbar_expect_tx(bar, 2 * SM::kTileBytes);
          const int y = it.key0 + i * kAttnTileKeys;
#pragma unroll
          for (int bx = 0; bx < SM::kBoxes; ++bx) {
            tma_load_3d(sK + s * SM::kTileBytes + bx * 8192, &set.K[layer], bar, bx * 64, y, zc);
            tma_load_3d(sV + s * SM::kTileBytes + bx * 8192, &set.V[layer], bar, bx * 64, y, zc);
          }
          ++tile_ctr;
        };
        if (lane == 0) {
          // tiles whose stage is free go out first; before the barrier only
          // tiles that lie wholly in the cache prefix, issued as the consumers
          // free stages while the barrier is polled
          const int n_pre = ready ? n_tiles : min(n_tiles, max(0, (it.kv - it.key0) / kAttnTileKeys));
          for (int spin = 0;; ++spin) {
            while (issued < n_pre &&
                   mbar_test_wait(bEmpty + 8 * (tile_ctr % STAGES), ((tile_ctr / STAGES) & 1) ^ 1)) {
              issue_tile(issued);
              ++issued;
            }
            if (ready) break;
            uint32_t v;
            asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(bar_cnt + (layer - 1)) : "memory");
            if (v >= n_ctas) break;
            if (spin >= kMaxWaitIters) {
              raise_status(status, LIBRASPEC_ST_TIMEOUT);
              misc[0] = 1;
              break;
            }
            __nanosleep(32);
          }
        }
        __syncwarp();
        if (misc[0]) return;
        ready = true;
        // Q rows of the item's row group into the slot, unswizzled: row r of
        // 64-column half hb at hb * 8192 + r * 128. When g divides 64 a group is
        // 64/g whole positions of its kv head's g query heads: one TMA box per
        // half (rows past `rows` are read but never used). Otherwise one bulk
        // copy per row and half. Both complete as transaction bytes on the
        // slot's mbarrier; the producer issues no non-bulk cp.async copies
        // (on GB300, non-bulk copies in flight in the warp issuing TMA loads
        // were seen to lose their mbarrier arrival).
        const uint32_t qdst = sQ + q * SM::kQSlot;
        if (set.q_tma) {
          if (lane == 0) {
            info[q] = it;
            mbar_expect_tx(bQFull + 8 * q, (uint32_t)kAttnRows * D * 2);
#pragma unroll
            for (int hb = 0; hb < SM::kBoxes; ++hb)
              tma_load_3d(qdst + hb * 8192, &set.Q[layer], bQFull + 8 * q, hb * 64, it.kvh * g,
                          it.b * (K + 1) + it.mg * (kAttnRows / g));
          }
        } else {
          if (lane == 0) {
            info[q] = it;
            mbar_expect_tx(bQFull + 8 * q, (uint32_t)it.rows * D * 2);
          }
          __syncwarp();
          const __nv_bfloat16* Qb = set.p[layer].Q;
          for (int idx = lane; idx < it.rows * SM::kBoxes; idx += 32) {
            const int r = idx / SM::kBoxes, hb = idx - r * SM::kBoxes;
            const int rr = it.mg * kAttnRows + r;
            const int t = rr / g, h = it.kvh * g + (rr - t * g);
            const __nv_bfloat16* src = Qb + (((size_t)it.b * (K + 1) + t) * Hq + h) * D + hb * 64;
            bulk_load(qdst + hb * 8192 + r * 128, src, 128u, bQFull + 8 * q);
          }
        }
        ++item_ctr;
        if (lane == 0) {
          for (int i = issued; i < n_tiles; ++i) {
            const uint32_t par = ((tile_ctr / STAGES) & 1) ^ 1;
            if (!mbar_wait(bEmpty + 8 * (tile_ctr % STAGES), par)) {
              raise_status(status, LIBRASPEC_ST_TIMEOUT);
              misc[0] = 1;
              break;
            }
            issue_tile(i);
          }
        }
        tile_ctr = __shfl_sync(0xffffffffu, tile_ctr, 0);
        __syncwarp();
        if (misc[0]) return;
      }
    }
    return;
  }

  // ======================= consumers =======================
  // Warp roles per item: the item's rows form n_rt tiles of 16 rows. With
  // n_rt <= 2 the four warps are split across each KV tile's keys as well
  // (ks warps per row tile, each taking kq of the tile's four 16-key chunks),
  // so that small verified blocks still keep every warp busy; their (m, l, O)
  // are combined through shared memory when the item ends.
  uint32_t item_ctr = 0, tile_ctr = 0;
  for (int layer = 0; layer < n_layers; ++layer) {
    float* part_o = part_buf_o + (layer & 1) * part_o_stride;
    float* part_ml = part_buf_ml + (layer & 1) * part_ml_stride;
    if (layer > 0) {
      // layer's inputs are ready once every CTA is done with the previous layer
      if (tid == 0 && !wait_counter(bar_cnt + (layer - 1), n_ctas)) {
        raise_status(status, LIBRASPEC_ST_TIMEOUT);
        misc[0] = 1;
      }
      consumer_sync();
      if (misc[0]) return;
    }
    __nv_bfloat16* O = set.p[layer].O;
    float* lse = set.p[layer].lse;
    for (int item = 0; item < n_items; ++item) {
    const uint32_t q = item_ctr & 1;
    if (!mbar_wait(bQFull + 8 * q, (item_ctr >> 1) & 1)) {
      if (lane == 0) raise_status(status, LIBRASPEC_ST_TIMEOUT);
      return;
    }
    const ItemInfo it = info[q];
    const int rows = it.rows, kv = it.kv, b = it.b, kvh = it.kvh;
    const int r_base = it.mg * kAttnRows;
    const int n_rt = (rows + 15) >> 4;
    const int ks = n_rt == 1 ? 4 : (n_rt == 2 ? 2 : 1);
    const int rt = warp / ks;            // row tile of this warp
    const int kq = 4 / ks;               // 16-key chunks per tile for this warp
    const int c_lo = (warp % ks) * kq;   // its first chunk
    const bool warp_live = rt < n_rt;
    const uint32_t qslot = sQ + q * SM::kQSlot;
    uint32_t qf[D / 16][4];
    if (warp_live) {
#pragma unroll
      for (int kk = 0; kk < D / 16; ++kk) {
        const int mi = lane >> 3, rr = lane & 7;
        const int row = rt * 16 + (mi & 1) * 8 + rr;
        const int col = kk * 16 + (mi >> 1) * 8;
        ldsm_x4(qslot + (col >> 6) * 8192 + row * 128 + (col & 63) * 2, qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3]);
      }
    }
    ++item_ctr;

    float o[D / 8][4];
#pragma unroll
    for (int n = 0; n < D / 8; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.f;
    float m_run[2] = {-INFINITY, -INFINITY}, l_run[2] = {0.f, 0.f};
    const int row_a = r_base + rt * 16 + (lane >> 2);
    const int lim_a = kv + row_a / g;  // last visible key of row_a
    const int lim_b = kv + (row_a + 8) / g;
    const int n_tiles = (it.key1 - it.key0 + kAttnTileKeys - 1) / kAttnTileKeys;

    for (int i = 0; i < n_tiles; ++i) {
      const uint32_t s = tile_ctr % STAGES;
      if (!mbar_wait(bFull + 8 * s, (tile_ctr / STAGES) & 1)) {
        if (lane == 0) raise_status(status, LIBRASPEC_ST_TIMEOUT);
        return;
      }
      const int kt0 = it.key0 + i * kAttnTileKeys;
      const uint32_t tK = sK + s * SM::kTileBytes, tV = sV + s * SM::kTileBytes;
      if (kt0 + kAttnTileKeys > it.key1) {
        // zero V rows past the visible keys so that 0 * garbage cannot poison O
        const int first = it.key1 - kt0;
        for (int idx = warp * 32 + lane; idx < (kAttnTileKeys - first) * (D / 8); idx += kConsumerWarps * 32) {
          const int r = first + idx / (D / 8), ch = idx % (D / 8);
          *reinterpret_cast<uint4*>(smem + SM::kV + s * SM::kTileBytes + sw128(r, ch * 8)) =
              make_uint4(0, 0, 0, 0);
        }
        // these generic writes precede the next TMA write of the stage
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        consumer_sync();
      }
      if (warp_live) {
        float sc[8][4];
#pragma unroll
        for (int n = 0; n < 8; ++n) sc[n][0] = sc[n][1] = sc[n][2] = sc[n][3] = 0.f;
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
#pragma unroll
          for (int np = 0; np < 4; ++np) {
            if (np < c_lo || np >= c_lo + kq) continue;
            const int mi = lane >> 3, rr = lane & 7;
            const int key = np * 16 + (mi >> 1) * 8 + rr;
            const int col = kk * 16 + (mi & 1) * 8;
            uint32_t b0, b1, b2, b3;
            ldsm_x4(tK + sw128(key, col), b0, b1, b2, b3);
            mma_bf16(sc[2 * np], qf[kk], b0, b1);
            mma_bf16(sc[2 * np + 1], qf[kk], b2, b3);
          }
        }
        const bool need_mask = kt0 + kAttnTileKeys - 1 > kv;
        float tmax[2] = {-INFINITY, -INFINITY};
#pragma unroll
        for (int n = 0; n < 8; ++n) {
          const bool mine = (n >> 1) >= c_lo && (n >> 1) < c_lo + kq;
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            float x = sc[n][e] * scale_log2;
            if (!mine) x = -INFINITY;
            if (need_mask) {
              const int key = kt0 + n * 8 + 2 * (lane & 3) + (e & 1);
              if (key > ((e < 2) ? lim_a : lim_b)) x = -INFINITY;
            }
            sc[n][e] = x;
            tmax[e >> 1] = fmaxf(tmax[e >> 1], x);
          }
        }
        float corr[2], m_use[2];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          tmax[h] = fmaxf(tmax[h], __shfl_xor_sync(0xffffffffu, tmax[h], 1));
          tmax[h] = fmaxf(tmax[h], __shfl_xor_sync(0xffffffffu, tmax[h], 2));
          const float m_new = fmaxf(m_run[h], tmax[h]);
          m_use[h] = (m_new == -INFINITY) ? 0.f : m_new;
          corr[h] = ex2_approx(m_run[h] - m_use[h]);
          m_run[h] = m_new;
          l_run[h] *= corr[h];
        }
#pragma unroll
        for (int n = 0; n < D / 8; ++n) {
          o[n][0] *= corr[0]; o[n][1] *= corr[0];
          o[n][2] *= corr[1]; o[n][3] *= corr[1];
        }
#pragma unroll
        for (int n = 0; n < 8; ++n) {
          sc[n][0] = ex2_approx(sc[n][0] - m_use[0]);
          sc[n][1] = ex2_approx(sc[n][1] - m_use[0]);
          sc[n][2] = ex2_approx(sc[n][2] - m_use[1]);
          sc[n][3] = ex2_approx(sc[n][3] - m_use[1]);
          l_run[0] += sc[n][0] + sc[n][1];
          l_run[1] += sc[n][2] + sc[n][3];
        }
#pragma unroll
        for (int kc = 0; kc < 4; ++kc) {
          if (kc < c_lo || kc >= c_lo + kq) continue;
          uint32_t a[4];
          a[0] = pack_bf16(sc[2 * kc][0], sc[2 * kc][1]);
          a[1] = pack_bf16(sc[2 * kc][2], sc[2 * kc][3]);
          a[2] = pack_bf16(sc[2 * kc + 1][0], sc[2 * kc + 1][1]);
          a[3] = pack_bf16(sc[2 * kc + 1][2], sc[2 * kc + 1][3]);
#pragma unroll
          for (int dp = 0; dp < D / 16; ++dp) {
            const int mi = lane >> 3, rr = lane & 7;
            const int key = kc * 16 + (mi & 1) * 8 + rr;
            const int col = dp * 16 + (mi >> 1) * 8;
            uint32_t b0, b1, b2, b3;
            ldsm_x4_t(tV + sw128(key, col), b0, b1, b2, b3);
            mma_bf16(o[2 * dp], a, b0, b1);
            mma_bf16(o[2 * dp + 1], a, b2, b3);
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(bEmpty + 8 * s);
      ++tile_ctr;
    }

    // ---- epilogue ----
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      l_run[h] += __shfl_xor_sync(0xffffffffu, l_run[h], 1);
      l_run[h] += __shfl_xor_sync(0xffffffffu, l_run[h], 2);
    }
    // combine the key-split warps of each row tile through the (now free) Q slot
    if (ks > 1) {
      float* scr = reinterpret_cast<float*>(smem + SM::kQ + q * SM::kQSlot);
      constexpr int kPart = 16 * D + 32;  // floats: O rows, then (m, l) of 16 rows
      auto put = [&](int slot_i) {
        float* dst = scr + slot_i * kPart;
#pragma unroll
        for (int n = 0; n < D / 8; ++n) {
          const int col = n * 8 + 2 * (lane & 3);
          *reinterpret_cast<float2*>(dst + (lane >> 2) * D + col) = make_float2(o[n][0], o[n][1]);
          *reinterpret_cast<float2*>(dst + ((lane >> 2) + 8) * D + col) = make_float2(o[n][2], o[n][3]);
        }
        if ((lane & 3) == 0) {
          dst[16 * D + 2 * (lane >> 2)] = m_run[0];
          dst[16 * D + 2 * (lane >> 2) + 1] = l_run[0];
          dst[16 * D + 2 * ((lane >> 2) + 8)] = m_run[1];
          dst[16 * D + 2 * ((lane >> 2) + 8) + 1] = l_run[1];
        }
      };
      auto take = [&](int slot_i) {
        const float* src = scr + slot_i * kPart;
        float wa[2], wb[2];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int r = (lane >> 2) + 8 * h;
          const float mo = src[16 * D + 2 * r], lo = src[16 * D + 2 * r + 1];
          const float M = fmaxf(m_run[h], mo);
          wa[h] = (M == -INFINITY) ? 0.f : ex2_approx(m_run[h] - M);
          wb[h] = (M == -INFINITY) ? 0.f : ex2_approx(mo - M);
          l_run[h] = l_run[h] * wa[h] + lo * wb[h];
          m_run[h] = M;
        }
#pragma unroll
        for (int n = 0; n < D / 8; ++n) {
          const int col = n * 8 + 2 * (lane & 3);
          const float2 u = *reinterpret_cast<const float2*>(src + (lane >> 2) * D + col);
          const float2 v = *reinterpret_cast<const float2*>(src + ((lane >> 2) + 8) * D + col);
          o[n][0] = o[n][0] * wa[0] + u.x * wb[0];
          o[n][1] = o[n][1] * wa[0] + u.y * wb[0];
          o[n][2] = o[n][2] * wa[1] + v.x * wb[1];
          o[n][3] = o[n][3] * wa[1] + v.y * wb[1];
        }
      };
      const int kw = warp % ks;
      consumer_sync();  // every warp has its Q fragments before the slot is overwritten
      if (ks == 4) {
        if (kw >= 2) put(kw - 2);
        consumer_sync();
        if (kw < 2) take(kw);
        consumer_sync();
        if (kw == 1) put(0);
        consumer_sync();
        if (kw == 0) take(0);
      } else {  // ks == 2: warps 1 and 3 hand over to warps 0 and 2
        if (kw == 1) put(rt);
        consumer_sync();
        if (kw == 0) take(rt);
      }
    }
    consumer_sync();
    if (lane == 0) mbar_arrive(bQEmpty + 8 * q);  // the slot may take the next Q now
    const bool owner = warp_live && (warp % ks) == 0;
    const int lr0 = rt * 16 + (lane >> 2);
    if (!it.partial) {
      if (owner) {
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int lr = lr0 + 8 * h;
          if (lr >= rows) continue;
          const int rr = r_base + lr;
          const int t = rr / g, hq = kvh * g + rr % g;
          const float inv = 1.f / l_run[h];
          __nv_bfloat16* dst = O + (((size_t)b * (K + 1) + t) * Hq + hq) * D;
#pragma unroll
          for (int n = 0; n < D / 8; ++n) {
            const int col = n * 8 + 2 * (lane & 3);
            *reinterpret_cast<__nv_bfloat162*>(dst + col) =
                __floats2bfloat162_rn(o[n][2 * h] * inv, o[n][2 * h + 1] * inv);
          }
          if (lse && (lane & 3) == 0)
            lse[((size_t)b * (K + 1) + t) * Hq + hq] = (m_run[h] + __log2f(l_run[h])) * kLn2;
        }
      }
      continue;
    }
    // partial of a row group spread over several CTAs
    const size_t slot = (size_t)it.slot;
    if (owner) {
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int lr = lr0 + 8 * h;
        if (lr >= rows) continue;
        float* dst = part_o + (slot * kAttnRows + lr) * D;
#pragma unroll
        for (int n = 0; n < D / 8; ++n) {
          const int col = n * 8 + 2 * (lane & 3);
          *reinterpret_cast<float2*>(dst + col) = make_float2(o[n][2 * h], o[n][2 * h + 1]);
        }
        if ((lane & 3) == 0) {
          part_ml[(slot * kAttnRows + lr) * 2] = m_run[h];
          part_ml[(slot * kAttnRows + lr) * 2 + 1] = l_run[h];
        }
      }
    }
    }
    // the previous layer's split groups: its partials (the other parity
    // buffer) stay untouched until every CTA has passed this layer's barrier,
    // and the producer already streams the next layer's first tiles meanwhile
    if (layer > 0) {
      consumer_sync();
      merge_layer<D, STAGES>(smem, tasks, n_tasks, K, Hq, Hkv, part_buf_o + ((layer - 1) & 1) * part_o_stride,
                             part_buf_ml + ((layer - 1) & 1) * part_ml_stride, set.p[layer - 1].O,
                             set.p[layer - 1].lse);
    }
    // this CTA is done with the layer
    consumer_sync();
    if (tid == 0) asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(bar_cnt + layer), "r"(1u) : "memory");
  }
  // merge the last layer, then the last CTA out resets the counters
  if (n_layers > 0) {
    if (tid == 0 && !wait_counter(bar_cnt + (n_layers - 1), n_ctas)) {
      raise_status(status, LIBRASPEC_ST_TIMEOUT);
      misc[0] = 1;
    }
    consumer_sync();
    if (misc[0]) return;
    merge_layer<D, STAGES>(smem, tasks, n_tasks, K, Hq, Hkv, part_buf_o + ((n_layers - 1) & 1) * part_o_stride,
                           part_buf_ml + ((n_layers - 1) & 1) * part_ml_stride, set.p[n_layers - 1].O,
                           set.p[n_layers - 1].lse);
  }
  consumer_sync();
  if (tid == 0) {
    const uint32_t done = atomicAdd(exit_cnt, 1u);
    if (done == n_ctas - 1) {
      for (int l = 0; l < n_layers; ++l) bar_cnt[l] = 0u;
      *exit_cnt = 0u;
      __threadfence();
    }
  }
}

// ---------------------------------------------------------------------------
// Host side.
// ---------------------------------------------------------------------------
int num_sms_current();

static PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

// Q [B*(K+1), Hq, D] as 3-D; box = 64 columns x g heads x 64/g positions
// (one 64-row group of one kv head), no swizzle.
static bool make_q_map(CUtensorMap* map, const void* base, int D, int Hq, int BT, int g) {
  auto enc = get_encode();
  if (!enc) return false;
  cuuint64_t dims[3] = {(cuuint64_t)D, (cuuint64_t)Hq, (cuuint64_t)BT};
  cuuint64_t strides[2] = {(cuuint64_t)D * 2, (cuuint64_t)Hq * D * 2};
  cuuint32_t box[3] = {64, (cuuint32_t)g, (cuuint32_t)(kAttnRows / g)};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
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

// Launch tuning: pipeline depth variant and the smallest tile range per CTA.
// Defaults were chosen by measurement on GB300; the LIBRASPEC_ATTN_TUNING
// environment variable ("deep:min_tiles", deep = 0 for the two-CTAs-per-SM
// pipeline, 1 for the deeper one-CTA-per-SM one) overrides them, read once
// per process.
struct AttnTuning {
  int deep = 0;
  int min_tiles = 2;
};

static const AttnTuning& attn_tuning() {
  static AttnTuning t = [] {
    AttnTuning v;
    if (const char* e = getenv("LIBRASPEC_ATTN_TUNING")) {
      int a = 0, b = 0;
      if (sscanf(e, "%d:%d", &a, &b) == 2 && b >= 1 && b <= 4096) {
        v.deep = a != 0;
        v.min_tiles = b;
      }
    }
    return v;
  }();
  return t;
}

template <int D, int STAGES>
static cudaError_t launch_layers_t(const uint16_t* const* Q, const uint16_t* const* Kc, const uint16_t* const* Vc,
                                   int n_layers, const int32_t* kv_len, const int32_t* L, int B, int K, int Hq,
                                   int Hkv, int S_cap, float scale, int min_tiles, uint16_t* const* O,
                                   float* const* lse, char* ws, const WsLayout& lay, cudaStream_t stream) {
  using SM = AttnSmem<D, STAGES>;
  auto kern = verify_attn_kernel<D, STAGES>;
  static int occ = 0;
  if (occ == 0) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, SM::kAlloc);
    if (e != cudaSuccess) return e;
    int o = 1;
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&o, kern, kAttnThreads, SM::kAlloc);
    occ = o < 1 ? 1 : o;
  }
  int grid = num_sms_current() * occ;
  if (grid > kAttnMaxCtas) grid = kAttnMaxCtas;
  // layers beyond kMaxLayers go in further launches of the same kernel
  for (int l0 = 0; l0 < n_layers; l0 += kMaxLayers) {
    LayerSet set;  // ~27 KB: built on the host, copied into the launch parameters
    const int n = n_layers - l0 < kMaxLayers ? n_layers - l0 : kMaxLayers;
    set.n = n;
    const int g = Hq / Hkv;
    set.q_tma = (kAttnRows % g == 0) ? 1 : 0;
    for (int i = 0; i < n; ++i) {
      const int l = l0 + i;
      if (!make_kv_map(&set.K[i], Kc[l], D, S_cap, B * Hkv) || !make_kv_map(&set.V[i], Vc[l], D, S_cap, B * Hkv))
        return cudaErrorInvalidValue;
      if (set.q_tma && !make_q_map(&set.Q[i], Q[l], D, Hq, B * (K + 1), g)) return cudaErrorInvalidValue;
      set.p[i].Q = reinterpret_cast<const __nv_bfloat16*>(Q[l]);
      set.p[i].O = reinterpret_cast<__nv_bfloat16*>(O[l]);
      set.p[i].lse = lse ? lse[l] : nullptr;
    }
    const size_t o_half = (lay.attn_ml - lay.attn_o) / 2, ml_half = (lay.attn_cnt - lay.attn_ml) / 2;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kAttnThreads);
    cfg.dynamicSmemBytes = SM::kAlloc;
    cfg.stream = stream;
    // cooperative: every CTA is resident at once, which the layer barriers rely on
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cudaError_t e = cudaLaunchKernelEx(
        &cfg, kern, set, kv_len, L, B, K, Hq, Hkv, S_cap, scale * kLog2e, min_tiles,
        reinterpret_cast<float*>(ws + lay.attn_o), reinterpret_cast<float*>(ws + lay.attn_ml), o_half / sizeof(float),
        ml_half / sizeof(float), reinterpret_cast<uint32_t*>(ws + lay.attn_cnt), reinterpret_cast<int*>(ws + lay.status));
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

cudaError_t launch_verify_attn_layers(const uint16_t* const* Q, const uint16_t* const* Kc,
                                      const uint16_t* const* Vc, int n_layers, const int32_t* kv_len,
                                      const int32_t* L, int B, int K, int Hq, int Hkv, int D, int S_cap, float scale,
                                      uint16_t* const* O, float* const* lse, char* ws, const WsLayout& lay,
                                      cudaStream_t stream) {
  if (B == 0 || n_layers == 0) return cudaSuccess;
  const AttnTuning& t = attn_tuning();
  if (D == 128) {
    if (t.deep)
      return launch_layers_t<128, 4>(Q, Kc, Vc, n_layers, kv_len, L, B, K, Hq, Hkv, S_cap, scale, t.min_tiles, O,
                                     lse, ws, lay, stream);
    return launch_layers_t<128, 2>(Q, Kc, Vc, n_layers, kv_len, L, B, K, Hq, Hkv, S_cap, scale, t.min_tiles, O, lse,
                                   ws, lay, stream);
  }
  if (t.deep)
    return launch_layers_t<64, 8>(Q, Kc, Vc, n_layers, kv_len, L, B, K, Hq, Hkv, S_cap, scale, t.min_tiles, O, lse,
                                  ws, lay, stream);
  return launch_layers_t<64, 4>(Q, Kc, Vc, n_layers, kv_len, L, B, K, Hq, Hkv, S_cap, scale, t.min_tiles, O, lse,
                                ws, lay, stream);
}

cudaError_t launch_verify_attn(const uint16_t* Q, const uint16_t* Kc, const uint16_t* Vc, const int32_t* kv_len,
                               const int32_t* L, int B, int K, int Hq, int Hkv, int D, int S_cap, float scale,
                               uint16_t* O, float* lse, char* ws, const WsLayout& lay, cudaStream_t stream) {
  float* lse_arr[1] = {lse};
  return launch_verify_attn_layers(&Q, &Kc, &Vc, 1, kv_len, L, B, K, Hq, Hkv, D, S_cap, scale, &O,
                                   lse ? lse_arr : nullptr, ws, lay, stream);
}

}  // namespace libraspec
