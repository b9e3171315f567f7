// Step 3: block-causal GQA verify attention (split-KV, persistent grid).
//
// Work decomposition. For sequence b the verified block has M_b = (L_b+1)*g
// query rows per kv head (g = Hq/Hkv; row r is block position t = r / g of
// query head kvh*g + r % g) and N_b = kv_len_b + L_b + 1 visible keys. Rows
// are cut into groups of 64 (one m16 tile per warp, 4 warps) and keys into
// 64-key tiles. A work item is (b, kv head, row group, run of consecutive
// key tiles); every CTA derives the item list itself from L[] and kv_len[]
// (both device-resident), so the grid never depends on values the host does
// not know. Items are dealt round-robin over a persistent grid.
//
// Per item: K/V tiles arrive by TMA (128-byte swizzle, mbarrier pipeline of
// STAGES tiles); each warp computes S = Q K^T for its 16 rows with
// mma.sync m16n8k16 (bf16 in, fp32 accumulate), masks keys beyond
// kv_len_b + t, keeps an online softmax in the log2 domain and accumulates
// O += P V. An item that covers all of a row group's keys writes O directly;
// otherwise it writes an fp32 partial (O, m, l) and the last item of the
// group to finish (atomic ticket) merges the partials in a fixed order.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <cstdio>
#include <cstdlib>

#include "common.cuh"

namespace libraspec {

constexpr int kAttnThreads = 128;
constexpr int kMaxWaitIters = 1 << 24;

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
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

struct ItemInfo {
  int b, kvh, mg, split, nsplit, kv, Lb, rows, key0, key1, group, item_base, n_mg;
};

// Per-sequence quantities of the item list.
struct SeqPlan {
  int M, n_mg, N, n_tiles, n_split, items, groups;
  bool ok;
};

__device__ __forceinline__ SeqPlan seq_plan(int b, int B, const int32_t* kv_len, const int32_t* Ls, int K, int g,
                                            int Hkv, int S_cap, int tpi) {
  SeqPlan p{0, 0, 0, 0, 0, 0, 0, false};
  if (b >= B) return p;
  const int Lb = Ls[b], kv = kv_len[b];
  if (Lb < 0 || Lb > K || kv < 0 || (long)kv + Lb + 1 > S_cap) return p;
  p.ok = true;
  p.M = (Lb + 1) * g;
  p.n_mg = (p.M + kAttnRows - 1) / kAttnRows;
  p.N = kv + Lb + 1;
  p.n_tiles = (p.N + kAttnTileKeys - 1) / kAttnTileKeys;
  if (tpi > 0) {
    p.n_split = (p.n_tiles + tpi - 1) / tpi;
    p.items = Hkv * p.n_mg * p.n_split;
  }
  p.groups = Hkv * p.n_mg;
  return p;
}

// Warp 0: total key tiles over all row groups (sets tpi for everyone) and
// flags invalid sequences.
__device__ int total_tiles(int B, const int32_t* kv_len, const int32_t* Ls, int K, int g, int Hkv, int S_cap,
                           int* status, bool report) {
  const int lane = threadIdx.x & 31;
  long tot = 0;
  bool bad = false;
  for (int b = lane; b < B; b += 32) {
    const SeqPlan p = seq_plan(b, B, kv_len, Ls, K, g, Hkv, S_cap, 0);
    if (!p.ok) bad = true;
    else tot += (long)Hkv * p.n_mg * p.n_tiles;
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) tot += __shfl_xor_sync(0xffffffffu, tot, off);
  if (report && __any_sync(0xffffffffu, bad) && lane == 0) {
    // report which condition: re-check on lane 0 (cheap, B small)
    int bits = 0;
    for (int b = 0; b < B; ++b) {
      const int Lb = Ls[b], kv = kv_len[b];
      if (Lb < 0 || Lb > K) bits |= LIBRASPEC_ST_BAD_LENGTH;
      else if (kv < 0 || (long)kv + Lb + 1 > S_cap) bits |= LIBRASPEC_ST_KV_OVERFLOW;
    }
    raise_status(status, bits);
  }
  return (int)(tot > 0x7fffffff ? 0x7fffffff : tot);
}

// Warp 0: locate item i. Returns false when i is past the last item.
__device__ bool locate_item(int item, int B, const int32_t* kv_len, const int32_t* Ls, int K, int g, int Hkv,
                            int S_cap, int tpi, ItemInfo& info) {
  const int lane = threadIdx.x & 31;
  int item_carry = 0, group_carry = 0;
  for (int base = 0; base < B; base += 32) {
    const int b = base + lane;
    const SeqPlan p = seq_plan(b, B, kv_len, Ls, K, g, Hkv, S_cap, tpi);
    const int it = p.ok ? p.items : 0, gr = p.ok ? p.groups : 0;
    int inc_it = it, inc_gr = gr;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int a = __shfl_up_sync(0xffffffffu, inc_it, off);
      const int c = __shfl_up_sync(0xffffffffu, inc_gr, off);
      if (lane >= off) { inc_it += a; inc_gr += c; }
    }
    const int start_it = item_carry + inc_it - it, start_gr = group_carry + inc_gr - gr;
    const bool mine = it > 0 && item >= start_it && item < start_it + it;
    const unsigned ball = __ballot_sync(0xffffffffu, mine);
    if (ball) {
      const int src = __ffs(ball) - 1;
      if (lane == src) {
        const int local = item - start_it;
        info.b = b;
        info.mg = local % p.n_mg;
        const int rem = local / p.n_mg;
        info.split = rem % p.n_split;
        info.kvh = rem / p.n_split;
        info.nsplit = p.n_split;
        info.kv = kv_len[b];
        info.Lb = Ls[b];
        const int r0 = info.mg * kAttnRows;
        info.rows = min(kAttnRows, p.M - r0);
        const int t0 = info.split * tpi, t1 = min(p.n_tiles, t0 + tpi);
        info.key0 = t0 * kAttnTileKeys;
        info.key1 = min(p.N, t1 * kAttnTileKeys);
        info.group = start_gr + info.kvh * p.n_mg + info.mg;
        info.item_base = start_it + info.kvh * p.n_split * p.n_mg + info.mg;  // + split * n_mg
        info.n_mg = p.n_mg;
      }
      return true;
    }
    item_carry += __shfl_sync(0xffffffffu, inc_it, 31);
    group_carry += __shfl_sync(0xffffffffu, inc_gr, 31);
  }
  return false;
}

template <int D, int STAGES>
struct AttnSmem {
  static constexpr int kBoxes = D / 64;
  static constexpr int kTileBytes = kBoxes * 8192;  // one 64 x D bf16 tile
  static constexpr int kQ = 0;
  static constexpr int kK = kQ + kTileBytes;
  static constexpr int kV = kK + STAGES * kTileBytes;
  static constexpr int kBar = kV + STAGES * kTileBytes;
  static constexpr int kInfo = kBar + 8 * STAGES;
  static constexpr int kMerge = kInfo + 128;            // m, l of the merged rows (64 x 2 floats)
  static constexpr int kBytes = kMerge + 64 * 2 * 4;
  static constexpr int kAlloc = kBytes + 1024;          // room to align the base to 1024
};

template <int D, int STAGES>
__global__ void __launch_bounds__(kAttnThreads, 1) verify_attn_kernel(
    const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
    const __nv_bfloat16* __restrict__ Q, const int32_t* __restrict__ kv_len, const int32_t* __restrict__ Ls,
    int B, int K, int Hq, int Hkv, int S_cap, float scale_log2, int min_tiles, __nv_bfloat16* __restrict__ O,
    float* __restrict__ lse, float* __restrict__ part_o, float* __restrict__ part_ml, int* __restrict__ status) {
  using SM = AttnSmem<D, STAGES>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sQ = smem_u32(smem + SM::kQ);
  const uint32_t sK = smem_u32(smem + SM::kK);
  const uint32_t sV = smem_u32(smem + SM::kV);
  const uint32_t sBar = smem_u32(smem + SM::kBar);
  ItemInfo& info = *reinterpret_cast<ItemInfo*>(smem + SM::kInfo);
  float* merge_ml = reinterpret_cast<float*>(smem + SM::kMerge);
  __shared__ int sh_tpi, sh_found, sh_abort;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = Hq / Hkv;

  if (tid == 0) {
    for (int s = 0; s < STAGES; ++s) mbar_init(sBar + 8 * s, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    sh_abort = 0;
  }
  if (warp == 0) {
    const int tot = total_tiles(B, kv_len, Ls, K, g, Hkv, S_cap, status, blockIdx.x == 0);
    if (lane == 0) {
      int tpi = (tot + (int)gridDim.x - 1) / (int)gridDim.x;
      sh_tpi = tpi < min_tiles ? min_tiles : tpi;
    }
  }
  __syncthreads();
  const int tpi = sh_tpi;
  uint32_t tile_ctr = 0;  // tiles consumed by this CTA so far (stage / phase)
  // let the merge kernel (launched as a programmatic dependent) get resident
  // as soon as SMs free up; it waits for this grid's completion itself
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  for (int item = blockIdx.x;; item += gridDim.x) {
    __syncthreads();  // everyone is done with the previous item's shared state
    if (warp == 0) {
      const bool found = locate_item(item, B, kv_len, Ls, K, g, Hkv, S_cap, tpi, info);
      if (lane == 0) sh_found = found;
    }
    __syncthreads();
    if (!sh_found || sh_abort) break;
    const int b = info.b, kvh = info.kvh, rows = info.rows, kv = info.kv;
    const int r_base = info.mg * kAttnRows;
    const int key0 = info.key0, key1 = info.key1;
    const int nsplit = info.nsplit, split = info.split, n_mg = info.n_mg;
    const int group = info.group, item_base = info.item_base;
    const int n_tiles = (key1 - key0 + kAttnTileKeys - 1) / kAttnTileKeys;
    const int zcoord = b * Hkv + kvh;

    // ---- producer prologue: first STAGES tiles ----
    if (tid == 0) {
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      for (int i = 0; i < n_tiles && i < STAGES; ++i) {
        const uint32_t s = (tile_ctr + i) % STAGES;
        const uint32_t bar = sBar + 8 * s;
        mbar_expect_tx(bar, 2 * SM::kTileBytes);
        const int y = key0 + i * kAttnTileKeys;
#pragma unroll
        for (int bx = 0; bx < SM::kBoxes; ++bx) {
          tma_load_3d(sK + s * SM::kTileBytes + bx * 8192, &tmK, bar, bx * 64, y, zcoord);
          tma_load_3d(sV + s * SM::kTileBytes + bx * 8192, &tmV, bar, bx * 64, y, zcoord);
        }
      }
    }

    // ---- Q rows of this group into shared memory (zero beyond `rows`) ----
    {
      constexpr int kChunks = D / 8;  // 16-byte chunks per row
      for (int idx = tid; idx < kAttnRows * kChunks; idx += kAttnThreads) {
        const int r = idx / kChunks, ch = idx % kChunks;
        uint4 val = make_uint4(0, 0, 0, 0);
        if (r < rows) {
          const int rr = r_base + r;
          const int t = rr / g, h = kvh * g + rr % g;
          const __nv_bfloat16* src = Q + (((size_t)b * (K + 1) + t) * Hq + h) * D + ch * 8;
          val = *reinterpret_cast<const uint4*>(src);
        }
        *reinterpret_cast<uint4*>(smem + SM::kQ + sw128(r, ch * 8)) = val;
      }
    }
    __syncthreads();

    const bool warp_live = warp * 16 < rows;
    uint32_t qf[D / 16][4];
    if (warp_live) {
#pragma unroll
      for (int kk = 0; kk < D / 16; ++kk) {
        const int mi = lane >> 3, rr = lane & 7;
        const int row = warp * 16 + (mi & 1) * 8 + rr;
        const int col = kk * 16 + (mi >> 1) * 8;
        ldsm_x4(sQ + sw128(row, col), qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3]);
      }
    }
    float o[D / 8][4];
#pragma unroll
    for (int n = 0; n < D / 8; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.f;
    float m_run[2] = {-INFINITY, -INFINITY}, l_run[2] = {0.f, 0.f};
    // block row (t) of this thread's two rows, for the causal limit
    const int row_a = r_base + warp * 16 + (lane >> 2);
    const int lim_a = kv + row_a / g;            // last visible key of row_a
    const int lim_b = kv + (row_a + 8) / g;

    for (int i = 0; i < n_tiles; ++i) {
      const uint32_t s = tile_ctr % STAGES;
      const uint32_t par = (tile_ctr / STAGES) & 1;
      if (!mbar_wait(sBar + 8 * s, par)) {
        if (lane == 0) raise_status(status, LIBRASPEC_ST_TIMEOUT);
        sh_abort = 1;
        return;
      }
      const int kt0 = key0 + i * kAttnTileKeys;
      const uint32_t tK = sK + s * SM::kTileBytes, tV = sV + s * SM::kTileBytes;
      // zero V rows past the visible keys so that 0 * garbage cannot poison O
      if (kt0 + kAttnTileKeys > key1) {
        __syncwarp();
        const int first = key1 - kt0;
        for (int idx = lane; idx < (kAttnTileKeys - first) * (D / 8); idx += 32) {
          const int r = first + idx / (D / 8), ch = idx % (D / 8);
          if (warp == 0) *reinterpret_cast<uint4*>(smem + SM::kV + s * SM::kTileBytes + sw128(r, ch * 8)) =
              make_uint4(0, 0, 0, 0);
        }
        __syncthreads();
      }
      if (warp_live) {
        float sc[8][4];
#pragma unroll
        for (int n = 0; n < 8; ++n) sc[n][0] = sc[n][1] = sc[n][2] = sc[n][3] = 0.f;
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
#pragma unroll
          for (int np = 0; np < 4; ++np) {
            const int mi = lane >> 3, rr = lane & 7;
            const int key = np * 16 + (mi >> 1) * 8 + rr;
            const int col = kk * 16 + (mi & 1) * 8;
            uint32_t b0, b1, b2, b3;
            ldsm_x4(tK + sw128(key, col), b0, b1, b2, b3);
            mma_bf16(sc[2 * np], qf[kk], b0, b1);
            mma_bf16(sc[2 * np + 1], qf[kk], b2, b3);
          }
        }
        // scale into the log2 domain and mask
        const bool need_mask = kt0 + kAttnTileKeys - 1 > kv;
        float tmax[2] = {-INFINITY, -INFINITY};
#pragma unroll
        for (int n = 0; n < 8; ++n) {
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            float x = sc[n][e] * scale_log2;
            if (need_mask) {
              const int key = kt0 + n * 8 + 2 * (lane & 3) + (e & 1);
              const int lim = (e < 2) ? lim_a : lim_b;
              if (key > lim) x = -INFINITY;
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
        // O += P V
#pragma unroll
        for (int kc = 0; kc < 4; ++kc) {
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
      ++tile_ctr;
      __syncthreads();  // every warp is done with stage s
      if (tid == 0 && i + STAGES < n_tiles) {
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        const uint32_t bar = sBar + 8 * s;
        mbar_expect_tx(bar, 2 * SM::kTileBytes);
        const int y = key0 + (i + STAGES) * kAttnTileKeys;
#pragma unroll
        for (int bx = 0; bx < SM::kBoxes; ++bx) {
          tma_load_3d(tK + bx * 8192, &tmK, bar, bx * 64, y, zcoord);
          tma_load_3d(tV + bx * 8192, &tmV, bar, bx * 64, y, zcoord);
        }
      }
    }

    // ---- epilogue ----
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      l_run[h] += __shfl_xor_sync(0xffffffffu, l_run[h], 1);
      l_run[h] += __shfl_xor_sync(0xffffffffu, l_run[h], 2);
    }
    const int lr0 = warp * 16 + (lane >> 2);  // local rows lr0, lr0 + 8
    if (nsplit == 1) {
      if (warp_live) {
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
    // several items share this row group: write the fp32 partial (O, m, l);
    // attn_merge_kernel combines them once the whole grid is done
    const size_t slot = (size_t)item_base + (size_t)split * n_mg;
    if (warp_live) {
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
    (void)group;
  }
}

// ---------------------------------------------------------------------------
// Merge of the split-KV partials. Launched right after verify_attn_kernel as
// a programmatic dependent: it becomes resident early and waits
// (griddepcontrol.wait) until every attention CTA has finished and its
// writes are visible. One warp per (sequence, kv head, row) whose row group
// was split: O = sum_s 2^(m_s - M) O_s / sum_s 2^(m_s - M) l_s, M = max_s m_s,
// splits combined in a fixed order (deterministic). Spread over the whole
// GPU, so no single SM reads all of a group's partials.
// ---------------------------------------------------------------------------
constexpr int kMergeThreads = 256;

template <int D>
__global__ void __launch_bounds__(kMergeThreads) attn_merge_kernel(
    const int32_t* __restrict__ kv_len, const int32_t* __restrict__ Ls, int B, int K, int Hq, int Hkv, int S_cap,
    int attn_grid, int min_tiles, __nv_bfloat16* __restrict__ O, float* __restrict__ lse,
    const float* __restrict__ part_o, const float* __restrict__ part_ml) {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  __shared__ int sh_tpi;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int g = Hq / Hkv;
  if (warp == 0) {
    const int tot = total_tiles(B, kv_len, Ls, K, g, Hkv, S_cap, nullptr, false);
    if (lane == 0) {
      const int tpi = (tot + attn_grid - 1) / attn_grid;
      sh_tpi = tpi < min_tiles ? min_tiles : tpi;
    }
  }
  __syncthreads();
  const int tpi = sh_tpi;
  const int warps_total = gridDim.x * (kMergeThreads / 32);
  for (int unit = blockIdx.x * (kMergeThreads / 32) + warp;; unit += warps_total) {
    // locate the unit: units of sequence b (split row groups only) are
    // Hkv * M_b rows, kv head major
    int carry_u = 0, carry_it = 0;
    int b = -1, local = 0, start_it = 0;
    SeqPlan p{};
    for (int base = 0; base < B; base += 32) {
      const int bb = base + lane;
      const SeqPlan q = seq_plan(bb, B, kv_len, Ls, K, g, Hkv, S_cap, tpi);
      const int it = q.ok ? q.items : 0;
      const int un = (q.ok && q.n_split > 1) ? Hkv * q.M : 0;
      int inc_u = un, inc_it = it;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const int a = __shfl_up_sync(0xffffffffu, inc_u, off);
        const int c = __shfl_up_sync(0xffffffffu, inc_it, off);
        if (lane >= off) { inc_u += a; inc_it += c; }
      }
      const int su = carry_u + inc_u - un;
      const bool mine = un > 0 && unit >= su && unit < su + un;
      const unsigned ball = __ballot_sync(0xffffffffu, mine);
      if (ball) {
        const int src = __ffs(ball) - 1;
        b = base + src;
        local = unit - __shfl_sync(0xffffffffu, su, src);
        start_it = __shfl_sync(0xffffffffu, carry_it + inc_it - it, src);
        p = seq_plan(b, B, kv_len, Ls, K, g, Hkv, S_cap, tpi);
        break;
      }
      carry_u += __shfl_sync(0xffffffffu, inc_u, 31);
      carry_it += __shfl_sync(0xffffffffu, inc_it, 31);
    }
    if (b < 0) break;
    const int kvh = local / p.M, r = local % p.M;
    const int mg = r / kAttnRows, lr = r % kAttnRows;
    const int nsp = p.n_split;
    auto slot_of = [&](int sp) { return (size_t)start_it + ((size_t)kvh * nsp + sp) * p.n_mg + mg; };
    // row max and denominator over the splits
    float M = -INFINITY;
    for (int sp = lane; sp < nsp; sp += 32) M = fmaxf(M, __ldcg(&part_ml[(slot_of(sp) * kAttnRows + lr) * 2]));
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
    float Lsum = 0.f;
    for (int sp = lane; sp < nsp; sp += 32) {
      const size_t e = (slot_of(sp) * kAttnRows + lr) * 2;
      const float ms = __ldcg(&part_ml[e]);
      if (ms != -INFINITY) Lsum += __ldcg(&part_ml[e + 1]) * ex2_approx(ms - M);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) Lsum += __shfl_xor_sync(0xffffffffu, Lsum, off);
    // weighted sum of the partial rows; lane covers D/32 consecutive columns
    constexpr int CPL = D / 32;
    float acc[CPL];
#pragma unroll
    for (int i = 0; i < CPL; ++i) acc[i] = 0.f;
    for (int base = 0; base < nsp; base += 32) {
      float wl = 0.f;
      if (base + lane < nsp) {
        const float ms = __ldcg(&part_ml[(slot_of(base + lane) * kAttnRows + lr) * 2]);
        wl = (ms == -INFINITY) ? 0.f : ex2_approx(ms - M);
      }
      const int n = min(32, nsp - base);
#pragma unroll 8
      for (int j = 0; j < n; ++j) {
        const float w = __shfl_sync(0xffffffffu, wl, j);
        const float* src = part_o + (slot_of(base + j) * kAttnRows + lr) * D + lane * CPL;
        if (CPL == 4) {
          const float4 v = __ldcg(reinterpret_cast<const float4*>(src));
          acc[0] += w * v.x; acc[1] += w * v.y; acc[2 % CPL] += w * v.z; acc[3 % CPL] += w * v.w;
        } else {
          const float2 v = __ldcg(reinterpret_cast<const float2*>(src));
          acc[0] += w * v.x; acc[1 % CPL] += w * v.y;
        }
      }
    }
    const float inv = 1.f / Lsum;
    const int t = r / g, hq = kvh * g + r % g;
    __nv_bfloat16* dst = O + (((size_t)b * (K + 1) + t) * Hq + hq) * D + lane * CPL;
#pragma unroll
    for (int i = 0; i < CPL; i += 2)
      *reinterpret_cast<__nv_bfloat162*>(dst + i) = __floats2bfloat162_rn(acc[i] * inv, acc[i + 1] * inv);
    if (lse && lane == 0) lse[((size_t)b * (K + 1) + t) * Hq + hq] = (M + __log2f(Lsum)) * kLn2;
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

template <int D, int STAGES>
static cudaError_t launch_attn_t(const CUtensorMap& mK, const CUtensorMap& mV, const uint16_t* Q,
                                 const int32_t* kv_len, const int32_t* L, int B, int K, int Hq, int Hkv, int S_cap,
                                 float scale, int min_tiles, uint16_t* O, float* lse, char* ws, const WsLayout& lay,
                                 cudaStream_t stream) {
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
  auto* part_o = reinterpret_cast<float*>(ws + lay.attn_o);
  auto* part_ml = reinterpret_cast<float*>(ws + lay.attn_ml);
  auto* st = reinterpret_cast<int*>(ws + lay.status);
  auto* Ob = reinterpret_cast<__nv_bfloat16*>(O);
  kern<<<grid, kAttnThreads, SM::kAlloc, stream>>>(mK, mV, reinterpret_cast<const __nv_bfloat16*>(Q), kv_len, L, B,
                                                   K, Hq, Hkv, S_cap, scale * kLog2e, min_tiles, Ob, lse, part_o,
                                                   part_ml, st);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  // merge kernel as a programmatic dependent launch
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * num_sms_current());
  cfg.blockDim = dim3(kMergeThreads);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, attn_merge_kernel<D>, kv_len, L, B, K, Hq, Hkv, S_cap, grid, min_tiles, Ob, lse,
                            (const float*)part_o, (const float*)part_ml);
}

// Launch tuning: pipeline depth variant and the smallest run of key tiles
// per work item. Defaults were chosen by measurement on GB300; the
// LIBRASPEC_ATTN_TUNING environment variable ("deep:min_tiles", deep = 0 for
// the shallow two-CTAs-per-SM pipeline, 1 for the deep one-CTA-per-SM one)
// overrides them, read once per process.
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

cudaError_t launch_verify_attn(const uint16_t* Q, const uint16_t* Kc, const uint16_t* Vc, const int32_t* kv_len,
                               const int32_t* L, int B, int K, int Hq, int Hkv, int D, int S_cap, float scale,
                               uint16_t* O, float* lse, char* ws, const WsLayout& lay, cudaStream_t stream) {
  if (B == 0) return cudaSuccess;
  CUtensorMap mK, mV;
  if (!make_kv_map(&mK, Kc, D, S_cap, B * Hkv) || !make_kv_map(&mV, Vc, D, S_cap, B * Hkv))
    return cudaErrorInvalidValue;
  const AttnTuning& t = attn_tuning();
  if (D == 128) {
    if (t.deep)
      return launch_attn_t<128, 6>(mK, mV, Q, kv_len, L, B, K, Hq, Hkv, S_cap, scale, t.min_tiles, O, lse, ws, lay,
                                   stream);
    return launch_attn_t<128, 2>(mK, mV, Q, kv_len, L, B, K, Hq, Hkv, S_cap, scale, t.min_tiles, O, lse, ws, lay,
                                 stream);
  }
  if (t.deep)
    return launch_attn_t<64, 10>(mK, mV, Q, kv_len, L, B, K, Hq, Hkv, S_cap, scale, t.min_tiles, O, lse, ws, lay,
                                 stream);
  return launch_attn_t<64, 4>(mK, mV, Q, kv_len, L, B, K, Hq, Hkv, S_cap, scale, t.min_tiles, O, lse, ws, lay,
                              stream);
}

}  // namespace libraspec
