// Step 1 (drafter confidence) and step 2 (LibraSpec length selection).
#include "rowpass.cuh"

namespace libraspec {

// ---------------------------------------------------------------------------
// Confidence: grid (nsplit, B*K), 256 threads. CTA `split` of row r streams
// columns [split*chunk, (split+1)*chunk) once, keeping the running max and
// sum of exp((x - m)/T). With several splits the last CTA to finish (atomic
// ticket) merges the row's partials (binary64 sums) and finalises
// q = exp((x_tok - m)/T) / Z (Assumption 1: q_k, the drafter's probability
// of its drafted token).
// ---------------------------------------------------------------------------
// ---------------------------------------------------------------------------
// Selection (Thm. 4): one warp per sequence, binary64. Lane k of a 32-wide
// chunk evaluates the step L = k -> k+1:
//   P_{k+1} = prod_{i<=k} q_i          (multiplicative inclusive scan)
//   E_k     = 1 + sum_{j<=k} P_j       (additive exclusive scan of P)
//   extend  iff P_{k+1} * T(k) > (T(k+1) - T(k)) * E_k
// L is the first lane (in chunk order) whose test fails, or K. Executed by
// one full warp; conf is read through L2 (it may have been written by other
// CTAs of the same launch).
// ---------------------------------------------------------------------------
__device__ void select_seq(const float* __restrict__ conf, const float* __restrict__ cost, int K, int seq,
                           int32_t* __restrict__ L, int* __restrict__ status) {
  const int lane = threadIdx.x & 31;
  bool bad = false;
  for (int l = lane; l <= K; l += 32) {
    const float t = cost[l];
    if (!(t > 0.f) || !isfinite(t)) bad = true;
  }
  if (__any_sync(0xffffffffu, bad)) {
    if (lane == 0) {
      L[seq] = 0;
      raise_status(status, LIBRASPEC_ST_BAD_COST);
    }
    return;
  }
  double carryP = 1.0, carryE = 1.0;
  int result = K;
  for (int base = 0; base < K; base += 32) {
    const int k = base + lane;
    const bool live = k < K;
    const double q = live ? (double)__ldcg(&conf[(size_t)seq * K + k]) : 1.0;
    double P = q;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const double o = __shfl_up_sync(0xffffffffu, P, off);
      if (lane >= off) P = __dmul_rn(P, o);
    }
    P = __dmul_rn(P, carryP);                 // P_{k+1}
    double S = P;                             // inclusive sum of P over the chunk
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const double o = __shfl_up_sync(0xffffffffu, S, off);
      if (lane >= off) S = __dadd_rn(S, o);
    }
    double Sx = __shfl_up_sync(0xffffffffu, S, 1);
    if (lane == 0) Sx = 0.0;
    const double E = __dadd_rn(carryE, Sx);   // E_k
    bool fail = false;
    if (live) {
      const double Tk = (double)cost[k], Tk1 = (double)cost[k + 1];
      const double lhs = __dmul_rn(P, Tk);
      const double rhs = __dmul_rn(E, __dsub_rn(Tk1, Tk));
      fail = !(lhs > rhs);
    }
    const unsigned ball = __ballot_sync(0xffffffffu, fail);
    if (ball) {
      result = base + __ffs(ball) - 1;
      break;
    }
    carryP = __shfl_sync(0xffffffffu, P, 31);
    carryE = __dadd_rn(carryE, __shfl_sync(0xffffffffu, S, 31));
  }
  if (lane == 0) L[seq] = result;
}

__global__ void __launch_bounds__(128) select_kernel(const float* __restrict__ conf,
                                                     const float* __restrict__ cost, int B, int K,
                                                     int32_t* __restrict__ L, int* __restrict__ status) {
  const int seq = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  if (seq >= B) return;
  select_seq(conf, cost, K, seq, L, status);
}

template <bool VEC, typename E>
__global__ void __launch_bounds__(kRowThreads) conf_kernel(
    const E* __restrict__ x, const int32_t* __restrict__ tokens, const float* __restrict__ temperature,
    int K, int V, int nsplit, int chunk, float* __restrict__ conf, float* __restrict__ dstat,
    RowPartial* __restrict__ part, uint32_t* __restrict__ cnt, const float* __restrict__ cost,
    int32_t* __restrict__ L, uint32_t* __restrict__ seq_cnt, int* __restrict__ status) {
  __shared__ float sm[64];
  __shared__ int last;
  const int row = blockIdx.y, split = blockIdx.x;
  const int b = row / K;
  const float tb = temperature[b];
  const float T = tb > 0.f ? tb : 1.f;
  const float c = log2e_over(T);
  const E* xr = x + (size_t)row * V;
  const int c0 = split * chunk, c1 = min(V, c0 + chunk);

  SumAcc sa;
  ArgAcc aa;
  sa.init();
  row_slice_pass<true, false, VEC, E>(xr, c0, c1, c, sa, aa);
  float m = sa.m, s = sa.value();
  cta_reduce_sum(m, s, c, sm);

  double Z;
  float M;
  if (nsplit == 1) {
    if (threadIdx.x >= 32) return;
    M = m;
    Z = (double)s;
  } else {
    if (threadIdx.x == 0) {
      RowPartial p;
      p.m = m;
      p.arg = 0;
      p.s = (double)s;
      part[(size_t)row * kConfMaxSplits + split] = p;
      __threadfence();
      const uint32_t ticket = atomicAdd(&cnt[row], 1u);
      last = (ticket == (uint32_t)(nsplit - 1));
    }
    __syncthreads();
    if (!last) return;
    if (threadIdx.x >= 32) return;
    __threadfence();
    int dummy;
    warp_merge_partials(part + (size_t)row * kConfMaxSplits, nsplit, c, false, M, dummy, Z);
    if (threadIdx.x == 0) cnt[row] = 0u;  // ready for the next call
  }
  // warp 0 of the CTA that completed the row
  bool seq_done = false;
  if (threadIdx.x == 0) {
    const int tok = tokens[row];
    float q = 0.f;
    if (tok < 0 || tok >= V) {
      raise_status(status, LIBRASPEC_ST_BAD_TOKEN);
    } else {
      // x_tok - M is exact for the near-maximal tokens that matter (Sterbenz)
      q = (float)((double)exp2f((Logit<E>::at(xr, tok) - M) * c) / Z);
    }
    conf[row] = q;
    if (dstat) {
      dstat[2 * (size_t)row] = M;
      dstat[2 * (size_t)row + 1] = (float)Z;
    }
    if (cost) {
      __threadfence();
      seq_done = atomicAdd(&seq_cnt[b], 1u) == (uint32_t)(K - 1);
    }
  }
  // With a cost table, the CTA that completes a sequence's last row selects
  // its length (Thm. 4) right away instead of in a separate launch.
  if (cost == nullptr || !__shfl_sync(0xffffffffu, seq_done, 0)) return;
  __threadfence();
  if (threadIdx.x == 0) seq_cnt[b] = 0u;  // ready for the next call
  select_seq(conf, cost, K, b, L, status);
}

// ---------------------------------------------------------------------------
// Alpha-mode length search (Algorithm 1), one warp per sequence, binary64.
// eps_i = floor(alpha * S_i + i) with S_i = sum_{j=i}^{d} prod_{k=i}^{j} q_k,
// eps* = min_i eps_i. S_i = q_i (1 + S_{i+1}), S_{d+1} = 0: lane i-1 holds
// the affine map x -> q_i + q_i x and a suffix scan of map compositions
// gives every S_i at once (positions 33..64 in a second chunk whose S_33
// feeds the first). From d = n: eps* <= d rolls back once and stops, else
// d = min(eps*, K) and ceil(-budget/n) blocks are drafted when the budget
// of drafted-but-unused tokens turns negative.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void suffix_compose(double& a, double& b) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const double ao = __shfl_down_sync(0xffffffffu, a, off);
    const double bo = __shfl_down_sync(0xffffffffu, b, off);
    if (lane + off < 32) {
      b = __dadd_rn(__dmul_rn(a, bo), b);  // (this map) o (the maps after it)
      a = __dmul_rn(a, ao);
    }
  }
}

__global__ void __launch_bounds__(128) select_alpha_kernel(const float* __restrict__ conf, int B, int K, int n,
                                                           double alpha, int32_t* __restrict__ L,
                                                           int32_t* __restrict__ n_blocks) {
  const int seq = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (seq >= B) return;
  const float* q = conf + (size_t)seq * K;
  const double q0 = lane < K ? (double)q[lane] : 0.0;            // q_{lane+1}
  const double q1 = lane + 32 < K ? (double)q[lane + 32] : 0.0;  // q_{lane+33}
  int d = n, blocks = 1;
  int budget = 0;
  while (d < K) {
    int best = K + 1;
    double carry = 0.0;  // S_33
    if (d > 32) {
      const bool live = lane + 33 <= d;
      double a = live ? q1 : 1.0, b = live ? q1 : 0.0;
      suffix_compose(a, b);
      carry = __shfl_sync(0xffffffffu, b, 0);
      if (live) {
        const double x = __dadd_rn(__dmul_rn(alpha, b), (double)(lane + 33));
        const double f = floor(x);
        best = min(best, f >= (double)(K + 1) ? K + 1 : (f >= 1.0 ? (int)f : 1));
      }
    }
    const bool live = lane + 1 <= d;
    double a = live ? q0 : 1.0, b = live ? q0 : 0.0;
    suffix_compose(a, b);
    if (live) {
      const double S = __dadd_rn(__dmul_rn(a, carry), b);
      const double x = __dadd_rn(__dmul_rn(alpha, S), (double)(lane + 1));
      const double f = floor(x);
      best = min(best, f >= (double)(K + 1) ? K + 1 : (f >= 1.0 ? (int)f : 1));
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) best = min(best, __shfl_xor_sync(0xffffffffu, best, off));
    if (best <= d) {
      d = best;  // the single rollback
      break;
    }
    if (best > K) best = K;
    budget -= best - d;
    d = best;
    if (budget < 0) {
      const int more = (-budget + n - 1) / n;
      blocks += more;
      budget += more * n;
    }
  }
  if (lane == 0) {
    L[seq] = d;
    if (n_blocks) n_blocks[seq] = blocks;
  }
}

// ---------------------------------------------------------------------------
// Host launchers (arguments already validated by the ABI layer).
// ---------------------------------------------------------------------------
int num_sms_current();

// cost != nullptr: also select every sequence's length (Thm. 4) into L, in
// the same launch (K >= 1).
template <typename T>
cudaError_t launch_confidence(const T* x, const int32_t* tokens, const float* temperature, int B, int K, int V,
                              float* conf, float* dstat, char* ws, const WsLayout& lay, cudaStream_t stream,
                              const float* cost, int32_t* L) {
  const long rows = (long)B * K;
  if (rows == 0) return cudaSuccess;
  const int nsplit0 = conf_row_splits(rows, V, num_sms_current(), kConfMaxSplits, 4096);
  const int chunk = row_chunk(V, nsplit0);
  const int nsplit = (V + chunk - 1) / chunk;
  const bool vec = rows_vectorizable(x, V);
  dim3 grid(nsplit, (unsigned)rows);
  auto* part = reinterpret_cast<RowPartial*>(ws + lay.conf_part);
  auto* cnt = reinterpret_cast<uint32_t*>(ws + lay.conf_cnt);
  auto* st = reinterpret_cast<int*>(ws + lay.status);
  auto* seq_cnt = reinterpret_cast<uint32_t*>(ws + lay.seq_cnt);
  if (vec)
    conf_kernel<true, T><<<grid, kRowThreads, 0, stream>>>(x, tokens, temperature, K, V, nsplit, chunk, conf,
                                                           dstat, part, cnt, cost, L, seq_cnt, st);
  else
    conf_kernel<false, T><<<grid, kRowThreads, 0, stream>>>(x, tokens, temperature, K, V, nsplit, chunk, conf,
                                                            dstat, part, cnt, cost, L, seq_cnt, st);
  return cudaGetLastError();
}
template cudaError_t launch_confidence<float>(const float*, const int32_t*, const float*, int, int, int, float*,
                                              float*, char*, const WsLayout&, cudaStream_t, const float*, int32_t*);
template cudaError_t launch_confidence<uint16_t>(const uint16_t*, const int32_t*, const float*, int, int, int,
                                                 float*, float*, char*, const WsLayout&, cudaStream_t, const float*,
                                                 int32_t*);

cudaError_t launch_select_alpha(const float* conf, int B, int K, int n, double alpha, int32_t* L,
                                int32_t* n_blocks, cudaStream_t stream) {
  if (B == 0) return cudaSuccess;
  const int threads = 128;
  const int blocks = (B * 32 + threads - 1) / threads;
  select_alpha_kernel<<<blocks, threads, 0, stream>>>(conf, B, K, n, alpha, L, n_blocks);
  return cudaGetLastError();
}

cudaError_t launch_select(const float* conf, const float* cost, int B, int K, int32_t* L, char* ws,
                          const WsLayout& lay, cudaStream_t stream) {
  if (B == 0) return cudaSuccess;
  const int threads = 128;
  const int blocks = (B * 32 + threads - 1) / threads;
  select_kernel<<<blocks, threads, 0, stream>>>(conf, cost, B, K, L, reinterpret_cast<int*>(ws + lay.status));
  return cudaGetLastError();
}

}  // namespace libraspec
