// The LM head with the confidence / acceptance row statistics in its
// epilogue: logits x = H W^T (H [M, Dm] hidden states, W [V, Dm] the head,
// bf16) are accumulated by the 5th-generation tensor cores in tensor memory
// and reduced there to per-row (max, sum of exp, argmax, logit of one token)
// partials per 128-column vocabulary tile, so the logits never reach HBM;
// a second kernel merges each row's partials in binary64 (Assumption 1's
// confidence q = softmax(x / T)[token], and the max / argmax / Z of the
// acceptance rows, Sec. 3.1).
//
// Work: items = (row tile of 128, vocabulary tile of 128), vocabulary-major
// so that CTAs running at the same time share the head's tile through L2;
// CTA c of a grid of one CTA per SM takes items c, c + G, ... Roles (192
// threads): warp 4 streams H and W k-slabs (64 columns, 128-byte swizzle)
// by TMA into a ring of stages; warp 5 issues tcgen05.mma (M = 128, N =
// 128, K = 16, fp32 accumulate) into one of two tensor-memory accumulators;
// warps 0-3 (thread i <-> row i) read an accumulator, fold its 128 columns
// into the row's partial and free it. Rows past M and columns past V come
// from the TMA's zero fill and are left out of the statistics.
//
// Decode batches have few rows (M <= 128: one row tile), and the head's
// bytes set the time. There a stage holds only a_rows = M rounded up to 8
// rows of H (the MMA still reads 128 rows: the rest is whatever follows in
// shared memory, and only feeds accumulator rows that are never used), so
// the ring has room for more stages and keeps more of W in flight per SM.
#include <cstdio>

#include "tc.cuh"

namespace libraspec {

constexpr int kLmBM = 128, kLmBN = 128, kLmBK = 64, kLmMaxStages = 16;
constexpr int kLmEpiWarps = 4, kLmProducer = 4, kLmMma = 5, kLmThreads = 6 * 32;
constexpr uint32_t kLmATile = kLmBM * kLmBK * 2;  // 16 KB: a full H tile
constexpr uint32_t kLmBTile = kLmBN * kLmBK * 2;  // 16 KB
constexpr int kLmBarBytes = (2 * kLmMaxStages + 5) * 8 + 16;  // barriers and the tensor-memory slot
constexpr int kLmSmemMax = 227 * 1024;
constexpr int kLmTmemCols = 2 * kLmBN;
constexpr int kLmSub = 2;  // k-slabs per stage (fewer when Dm / 64 is not a multiple)
constexpr uint32_t kLmIdesc = mma_idesc(kLmBM, kLmBN, 0);

// Shared memory of a ring of `stages` stages of stage_bytes: barriers first,
// then the ring at the next 1024-byte boundary, then the 16 KB the MMA may
// read past the last stage's short H tile; plus room to align the base.
__host__ __device__ constexpr int lm_ring_offset() { return (kLmBarBytes + 1023) / 1024 * 1024; }
__host__ __device__ constexpr int lm_smem_bytes(int stages, int stage_bytes) {
  return 1024 + lm_ring_offset() + stages * stage_bytes + (int)kLmATile;
}

struct LmPartial {
  float m, z;  // max of the tile's logits, sum of 2^((x - m) c)
  int arg;     // first column of the max
  float xtok;  // the row's token logit if its column is in the tile, else NaN
};

__global__ void __launch_bounds__(kLmThreads, 1) lm_head_stats_kernel(
    const __grid_constant__ CUtensorMap mapH, const __grid_constant__ CUtensorMap mapW,
    const float* __restrict__ temperature, int rows_per_seq, const int32_t* __restrict__ tokens, int M, int V,
    int Dm, int m_tiles, int n_tiles, int a_rows, int stages, int sub, LmPartial* __restrict__ part,
    int* __restrict__ status) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  // a stage holds `sub` consecutive k-slabs (H slab, then W slab, each 1024-byte aligned), so every
  // row of W is read `sub` * 128 contiguous bytes at a time
  const uint32_t a_bytes = (uint32_t)a_rows * kLmBK * 2, slab_bytes = a_bytes + kLmBTile;
  const uint32_t stage_bytes = sub * slab_bytes;
  const uint32_t sbase = smem_u32(smem) + lm_ring_offset();
  const uint32_t bFull = smem_u32(smem), bEmpty = bFull + 8 * kLmMaxStages;
  const uint32_t bAccFull = bEmpty + 8 * kLmMaxStages, bAccEmpty = bAccFull + 16, bDrain = bAccEmpty + 16;
  volatile uint32_t* tmem_slot = reinterpret_cast<volatile uint32_t*>(smem + (2 * kLmMaxStages + 5) * 8);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int items = m_tiles * n_tiles, nk = Dm / kLmBK / sub;  // stages per item

  if (threadIdx.x == 0) {
    for (int s = 0; s < stages; ++s) {
      mbar_init(bFull + 8 * s, 1);   // the producer's expect_tx; bytes as transactions
      mbar_init(bEmpty + 8 * s, 1);  // the MMA warp's commit
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(bAccFull + 8 * a, 1);
      mbar_init(bAccEmpty + 8 * a, kLmEpiWarps);
    }
    mbar_init(bDrain, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == kLmMma) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(const_cast<uint32_t*>(tmem_slot))),
                 "n"(kLmTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  bool ok = true;

  if (warp == kLmProducer) {
    if (lane == 0) {
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&mapH)) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&mapW)) : "memory");
      uint32_t it = 0;
      for (int item = blockIdx.x; item < items && ok; item += gridDim.x) {
        const int n = item / m_tiles, m = item - n * m_tiles;
        for (int k = 0; k < nk; ++k, ++it) {
          const uint32_t s = it % stages, ph = (it / stages) & 1;
          if (!(ok = mbar_wait(bEmpty + 8 * s, ph ^ 1))) break;
          const uint32_t a = sbase + s * stage_bytes;
          mbar_expect_tx(bFull + 8 * s, stage_bytes);
          for (int j = 0; j < sub; ++j) {
            const int kc = (k * sub + j) * kLmBK;
            tma_load_2d(a + j * slab_bytes, &mapH, bFull + 8 * s, kc, m * kLmBM);
            tma_load_2d(a + j * slab_bytes + a_bytes, &mapW, bFull + 8 * s, kc, n * kLmBN);
          }
        }
      }
      if (!ok) raise_status(status, LIBRASPEC_ST_TIMEOUT);
    }
    __syncwarp();
  } else if (warp == kLmMma) {
    if (lane == 0) {
      uint32_t it = 0, t = 0;
      for (int item = blockIdx.x; item < items && ok; item += gridDim.x, ++t) {
        const uint32_t ab = t & 1, aph = (t >> 1) & 1;
        if (!(ok = mbar_wait(bAccEmpty + 8 * ab, aph ^ 1))) break;
        tc_fence_after();
        const uint32_t d = tmem + ab * kLmBN;
        for (int k = 0; k < nk; ++k, ++it) {
          const uint32_t s = it % stages, ph = (it / stages) & 1;
          if (!(ok = mbar_wait(bFull + 8 * s, ph))) break;
          tc_fence_after();
          for (int j = 0; j < sub; ++j) {
            const uint32_t a = sbase + s * stage_bytes + j * slab_bytes;
#pragma unroll
            for (int kk = 0; kk < kLmBK / 16; ++kk)
              mma_ss(d, smem_desc(a + kk * 32, 16, 1024), smem_desc(a + a_bytes + kk * 32, 16, 1024), kLmIdesc,
                     (k | j | kk) != 0 ? 1u : 0u);
          }
          mma_commit(bEmpty + 8 * s);  // the stage is free once these MMAs have read it
        }
        if (ok) mma_commit(bAccFull + 8 * ab);
      }
      if (!ok) raise_status(status, LIBRASPEC_ST_TIMEOUT);
      // every MMA issued has completed before the tensor memory is released
      mma_commit(bDrain);
      if (!mbar_wait(bDrain, 0)) raise_status(status, LIBRASPEC_ST_TIMEOUT);
    }
    __syncwarp();
  } else {
    // ===== epilogue: thread i <-> accumulator lane i = row i of the tile =====
    const int row = warp * 32 + lane;
    const uint32_t lane_off = (uint32_t)(warp * 32) << 16;
    uint32_t t = 0;
    for (int item = blockIdx.x; item < items && ok; item += gridDim.x, ++t) {
      const int n = item / m_tiles, m = item - n * m_tiles;
      const uint32_t ab = t & 1, aph = (t >> 1) & 1;
      if (!(ok = warp_wait(bAccFull + 8 * ab, aph))) break;
      tc_fence_after();
      const int grow = m * kLmBM + row;
      const bool valid = grow < M;
      float T = (valid && temperature) ? temperature[grow / rows_per_seq] : 1.f;
      if (!(T > 0.f)) T = 1.f;
      const float c = log2e_over(T);
      const int tok = (valid && tokens) ? tokens[grow] : -1;
      const int v0 = n * kLmBN;
      float mrun = -INFINITY, z = 0.f, xt = __int_as_float(0x7fc00000);
      int arg = 0x7fffffff;
#pragma unroll 1
      for (int ch = 0; ch < kLmBN / 32; ++ch) {
        uint32_t r[32];
        tmem_ld32(tmem + lane_off + ab * kLmBN + ch * 32, r);
        tmem_wait_ld();
        const int vc = v0 + ch * 32, nvalid = min(32, V - vc);
        float cm = -INFINITY;
        int ca = 0x7fffffff;
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const float x = __uint_as_float(r[i]);
          if (i < nvalid && x > cm) {
            cm = x;
            ca = vc + i;
          }
        }
        if (cm > mrun) {
          z = (mrun == -INFINITY) ? 0.f : z * ex2_approx((mrun - cm) * c);
          mrun = cm;
          arg = ca;
        }
        float zs[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int i = 0; i < 32; ++i)
          if (i < nvalid) zs[i & 3] += ex2_approx((__uint_as_float(r[i]) - mrun) * c);
        z += (zs[0] + zs[1]) + (zs[2] + zs[3]);
        if ((unsigned)(tok - vc) < 32u) {
#pragma unroll
          for (int i = 0; i < 32; ++i)
            if (i == tok - vc) xt = __uint_as_float(r[i]);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(bAccEmpty + 8 * ab);
      if (valid) {
        LmPartial p;
        p.m = mrun;
        p.z = z;
        p.arg = arg;
        p.xtok = xt;
        part[(size_t)grow * n_tiles + n] = p;
      }
    }
    if (!ok && lane == 0) raise_status(status, LIBRASPEC_ST_TIMEOUT);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == kLmMma)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "n"(kLmTmemCols) : "memory");
}

// One warp per row: the row's n_tiles partials in binary64. Z = sum_n z_n
// 2^((m_n - m) c); the argmax is the first column of the largest max (the
// partials are in column order); the token probability is
// 2^((x_tok - m) c) / Z.
// A token outside [-1, V) sets LIBRASPEC_ST_BAD_TOKEN (probability NaN).
__global__ void __launch_bounds__(128) lm_head_merge_kernel(const LmPartial* __restrict__ part, int M, int V,
                                                            int n_tiles, const float* __restrict__ temperature,
                                                            int rows_per_seq, const int32_t* __restrict__ tokens,
                                                            float* __restrict__ row_stat,
                                                            int32_t* __restrict__ row_argmax,
                                                            float* __restrict__ token_prob, int* __restrict__ status) {
  const int lane = threadIdx.x & 31;
  const int r = blockIdx.x * 4 + (threadIdx.x >> 5);
  if (r >= M) return;
  const LmPartial* p = part + (size_t)r * n_tiles;
  float T = temperature ? temperature[r / rows_per_seq] : 1.f;
  if (!(T > 0.f)) T = 1.f;
  const double c = (double)log2e_over(T);
  float mx = -INFINITY;
  int arg = 0x7fffffff;
  for (int n = lane; n < n_tiles; n += 32) argmax_combine(mx, arg, __ldg(&p[n].m), __ldg(&p[n].arg));
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, mx, off);
    const int a2 = __shfl_xor_sync(0xffffffffu, arg, off);
    argmax_combine(mx, arg, m2, a2);
  }
  double Z = 0.0;
  for (int n = lane; n < n_tiles; n += 32) {
    const float mn = __ldg(&p[n].m);
    if (mn > -INFINITY) Z += (double)__ldg(&p[n].z) * exp2(((double)mn - (double)mx) * c);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) Z += __shfl_xor_sync(0xffffffffu, Z, off);
  if (lane == 0) {
    if (row_stat) {
      row_stat[2 * (size_t)r] = mx;
      row_stat[2 * (size_t)r + 1] = (float)Z;
    }
    if (row_argmax) row_argmax[r] = arg;
    if (token_prob) {
      const int tok = tokens ? tokens[r] : -1;
      if (tok >= V || tok < -1) {
        raise_status(status, LIBRASPEC_ST_BAD_TOKEN);
        token_prob[r] = __int_as_float(0x7fc00000);
      } else {
        token_prob[r] = tok >= 0 ? (float)(exp2(((double)__ldg(&p[tok / kLmBN].xtok) - (double)mx) * c) / Z) : 0.f;
      }
    }
  }
}

int num_sms_current();

size_t lm_head_workspace_bytes(int M, int V) {
  const size_t n_tiles = ((size_t)V + kLmBN - 1) / kLmBN;
  return 256 + align256((size_t)M * n_tiles * sizeof(LmPartial));
}

static bool make_2d_map(CUtensorMap* map, const void* base, int cols, int rows, int box_rows) {
  // box_rows <= 256 (TMA), a multiple of 8 (whole 1024-byte swizzle atoms)
  auto enc = get_encode();
  if (!enc) return false;
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
  cuuint32_t box[2] = {(cuuint32_t)kLmBK, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// Workspace: the status word, then the partials [M, n_tiles].
cudaError_t launch_lm_head_stats(const uint16_t* H, const uint16_t* W, const float* temperature, int rows_per_seq,
                                 const int32_t* tokens, int M, int V, int Dm, float* row_stat, int32_t* row_argmax,
                                 float* token_prob, char* ws, cudaStream_t stream) {
  if (M == 0) return cudaSuccess;
  const int m_tiles = (M + kLmBM - 1) / kLmBM, n_tiles = (V + kLmBN - 1) / kLmBN;
  // one row tile: load only its rows (rounded up to 8), and spend the room on stages
  const int a_rows = m_tiles == 1 ? (M + 7) / 8 * 8 : kLmBM;
  const int slab_bytes = a_rows * kLmBK * 2 + (int)kLmBTile;
  const int nk = Dm / kLmBK;
  // k-slabs per stage: kLmSub, fewer while they do not divide Dm / 64 or leave under 3 stages
  int sub = kLmSub, stages = 0;
  for (;; sub >>= 1) {
    stages = (kLmSmemMax - lm_smem_bytes(0, sub * slab_bytes)) / (sub * slab_bytes);
    if (sub == 1 || (nk % sub == 0 && stages >= 3)) break;
  }
  const int stage_bytes = sub * slab_bytes;
  if (stages > kLmMaxStages) stages = kLmMaxStages;
  const int smem = lm_smem_bytes(stages, stage_bytes);
  CUtensorMap mapH, mapW;
  if (!make_2d_map(&mapH, H, Dm, M, a_rows) || !make_2d_map(&mapW, W, Dm, V, kLmBN)) return cudaErrorInvalidValue;
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(lm_head_stats_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         kLmSmemMax);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  const long long items = (long long)m_tiles * n_tiles;
  const int grid = (int)(items < num_sms_current() ? items : num_sms_current());
  auto* part = reinterpret_cast<LmPartial*>(ws + 256);
  auto* status = reinterpret_cast<int*>(ws);
  lm_head_stats_kernel<<<grid, kLmThreads, smem, stream>>>(mapH, mapW, temperature, rows_per_seq, tokens, M, V, Dm,
                                                          m_tiles, n_tiles, a_rows, stages, sub, part, status);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  lm_head_merge_kernel<<<(M + 3) / 4, 128, 0, stream>>>(part, M, V, n_tiles, temperature, rows_per_seq, tokens,
                                                        row_stat, row_argmax, token_prob, status);
  return cudaGetLastError();
}

}  // namespace libraspec
