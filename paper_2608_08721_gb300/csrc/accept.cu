// Step 4: acceptance (greedy argmax match / rejection sampling).
#include "rowpass.cuh"

namespace libraspec {

// ---------------------------------------------------------------------------
// Row statistics of the verified target rows. Grid (nsplit, K+1, B); rows
// j > L_b exit at once. Greedy sequences need only max / argmax; sampling
// sequences need (m, Z) at their temperature. Partials of a row are merged by
// the last CTA to finish (atomic ticket) into row_stat[b, j].
// ---------------------------------------------------------------------------
template <bool VEC, typename E>
__global__ void __launch_bounds__(kRowThreads) accept_rows_kernel(
    const E* __restrict__ target, const int32_t* __restrict__ Ls, const float* __restrict__ temperature,
    int K, int V, int nsplit, int chunk, RowPartial* __restrict__ part, uint32_t* __restrict__ cnt,
    RowStat* __restrict__ stat, int* __restrict__ status) {
  __shared__ float smf[64];
  __shared__ int smi[32];
  __shared__ int last;
  const int split = blockIdx.x, j = blockIdx.y, b = blockIdx.z;
  const int Lb = Ls[b];
  if (Lb < 0 || Lb > K) {
    if (split == 0 && j == 0 && threadIdx.x == 0) raise_status(status, LIBRASPEC_ST_BAD_LENGTH);
    return;
  }
  if (j > Lb) return;
  const int row = b * (K + 1) + j;
  const float tb = temperature ? temperature[b] : 0.f;  // none: every sequence greedy
  const bool sampling = tb > 0.f;
  const float T = sampling ? tb : 1.f;
  const float c = (float)(1.4426950408889634 / (double)T);
  const E* xr = target + (size_t)row * V;
  const int c0 = split * chunk, c1 = min(V, c0 + chunk);

  SumAcc sa;
  ArgAcc aa;
  sa.init();
  aa.init();
  float m;
  int arg = 0;
  float s = 0.f;
  if (sampling) {
    row_slice_pass<true, false, VEC, E>(xr, c0, c1, c, sa, aa);
    m = sa.m;
    s = sa.value();
    cta_reduce_sum(m, s, c, smf);
  } else {
    row_slice_pass<false, true, VEC, E>(xr, c0, c1, c, sa, aa);
    m = aa.m;
    arg = aa.arg;
    cta_reduce_arg(m, arg, smf, smi);
  }
  if (nsplit == 1) {
    if (threadIdx.x == 0) {
      RowStat st;
      st.m = m;
      st.arg = arg;
      st.Z = (double)s;
      stat[row] = st;
    }
    return;
  }
  if (threadIdx.x == 0) {
    RowPartial p;
    p.m = m;
    p.arg = arg;
    p.s = (double)s;
    part[(size_t)row * kRowMaxSplits + split] = p;
    __threadfence();
    const uint32_t ticket = atomicAdd(&cnt[row], 1u);
    last = (ticket == (uint32_t)(nsplit - 1));
  }
  __syncthreads();
  if (!last || threadIdx.x >= 32) return;
  __threadfence();
  float M;
  int A;
  double Z;
  warp_merge_partials(part + (size_t)row * kRowMaxSplits, nsplit, sampling ? c : 0.f, !sampling, M, A, Z);
  if (threadIdx.x == 0) {
    RowStat st;
    st.m = M;
    st.arg = sampling ? 0 : A;
    st.Z = Z;
    stat[row] = st;
    cnt[row] = 0u;
  }
}

// ---------------------------------------------------------------------------
// Decision and draw. Grid (nsplit, B). Every CTA of sequence b first takes
// the sequence's accept / reject decisions itself (they are cheap and
// deterministic), then, for sampling sequences, streams its slice of the
// vocabulary for the exponential race (argmin_v E_v / w_v, E_v = -ln u_v):
// w = max(0, p_r - q_r) after a rejection at r, or w = p_{L_b} (unnormalised)
// when all L_b drafts were accepted. The last CTA merges the slices.
// ---------------------------------------------------------------------------
struct Decision {
  int n;       // accepted drafts (r)
  int bonus;   // greedy: emitted token; sampling: -1 (drawn below)
  bool ok;
};

template <typename E>
__device__ Decision decide(int b, int K, int V, const E* __restrict__ target,
                           const int32_t* __restrict__ tokens, const float* __restrict__ conf,
                           const int32_t* __restrict__ Ls, const float* __restrict__ temperature,
                           const RowStat* __restrict__ stat, uint64_t seed, uint64_t round_offset,
                           uint32_t seq_offset, int* __restrict__ status) {
  // executed by one full warp
  const int lane = threadIdx.x & 31;
  Decision d{0, -1, true};
  const int Lb = Ls[b];
  if (Lb < 0 || Lb > K) {
    d.ok = false;
    return d;
  }
  const float tb = temperature[b];
  const RowStat* st = stat + (size_t)b * (K + 1);
  int n = Lb;
  for (int base = 0; base < Lb; base += 32) {
    const int jj = base + lane;
    bool reject = false;
    if (jj < Lb) {
      const int x = tokens[(size_t)b * K + jj];
      if (x < 0 || x >= V) {
        raise_status(status, LIBRASPEC_ST_BAD_TOKEN);
        reject = true;
      } else if (tb == 0.f) {
        reject = __ldcg(&st[jj].arg) != x;
      } else if (conf == nullptr) {
        reject = true;
      } else {
        const float c = (float)(1.4426950408889634 / (double)tb);
        const float y = Logit<E>::at(target, ((size_t)b * (K + 1) + jj) * V + x);
        const double p = (double)exp2f((y - __ldcg(&st[jj].m)) * c) / __ldcg(&st[jj].Z);
        const double q = (double)conf[(size_t)b * K + jj];
        const double ratio = (q <= p) ? 1.0 : p / q;
        const uint4 w = philox_block(seed, 0u, (uint32_t)jj, seq_offset + (uint32_t)b, 0u, round_offset);
        const double u = (double)word_to_uniform(w.x);
        reject = !(u < ratio);
      }
    }
    const unsigned ball = __ballot_sync(0xffffffffu, reject);
    if (ball) {
      n = base + __ffs(ball) - 1;
      break;
    }
  }
  d.n = n;
  if (tb == 0.f) d.bonus = __ldcg(&st[n].arg);
  return d;
}

template <bool VEC, typename E>
__global__ void __launch_bounds__(kRowThreads) accept_decide_kernel(
    const E* __restrict__ target, const E* __restrict__ draft, const int32_t* __restrict__ tokens,
    const float* __restrict__ conf, const float* __restrict__ dstat, const int32_t* __restrict__ Ls,
    const float* __restrict__ temperature, int K, int V, int nsplit, int chunk, uint64_t seed,
    uint64_t round_offset, uint32_t seq_offset, const uint64_t* __restrict__ rng, const RowStat* __restrict__ stat,
    RacePartial* __restrict__ part, uint32_t* __restrict__ cnt, int32_t* __restrict__ n_accepted,
    int32_t* __restrict__ bonus_token, int* __restrict__ status) {
  __shared__ int sh_n, sh_bonus, sh_ok, last;
  __shared__ float smk[32];
  __shared__ int smi[32];
  const int split = blockIdx.x, b = blockIdx.y;
  if (rng) {  // the generator's arguments from device memory (a replayed graph of a staged round)
    seed = rng[0];
    round_offset = rng[1];
    seq_offset = (uint32_t)rng[2];
  }
  if (threadIdx.x < 32) {
    const Decision d = decide<E>(b, K, V, target, tokens, conf, Ls, temperature, stat, seed, round_offset,
                                 seq_offset, status);
    if (threadIdx.x == 0) {
      sh_n = d.n;
      sh_bonus = d.bonus;
      sh_ok = d.ok;
    }
  }
  __syncthreads();
  const int n = sh_n;
  if (!sh_ok) {
    if (split == 0 && threadIdx.x == 0) {
      n_accepted[b] = 0;
      bonus_token[b] = 0;
      raise_status(status, LIBRASPEC_ST_BAD_LENGTH);
    }
    return;
  }
  const float tb = temperature[b];
  if (tb == 0.f) {
    if (split == 0 && threadIdx.x == 0) {
      n_accepted[b] = n;
      bonus_token[b] = sh_bonus;
    }
    return;
  }
  if (conf == nullptr || dstat == nullptr) {  // sampling needs q and the drafter row statistics
    if (split == 0 && threadIdx.x == 0) {
      n_accepted[b] = 0;
      bonus_token[b] = 0;
      raise_status(status, LIBRASPEC_ST_MISSING_INPUT);
    }
    return;
  }
  // ---- sampling: exponential race over the vocabulary at position n ----
  const int Lb = Ls[b];
  const bool residual = n < Lb;
  const float c = (float)(1.4426950408889634 / (double)tb);
  const RowStat st = stat[(size_t)b * (K + 1) + n];
  const E* yr = target + ((size_t)b * (K + 1) + n) * V;
  const E* dr = residual ? draft + ((size_t)b * K + n) * V : nullptr;
  const float mp = st.m;
  const float invZp = (float)(1.0 / st.Z);
  float mq = 0.f, invZq = 0.f;
  if (residual) {
    mq = dstat[2 * ((size_t)b * K + n)];
    invZq = 1.0f / dstat[2 * ((size_t)b * K + n) + 1];
  }
  const uint32_t seq = seq_offset + (uint32_t)b;
  const int c0 = split * chunk, c1 = min(V, c0 + chunk);
  float best = INFINITY;
  int besti = 0x7fffffff;
  // groups of 4 consecutive tokens share one Philox block
  for (int g = (c0 >> 2) + threadIdx.x; 4 * g < c1; g += kRowThreads) {
    const uint4 w4 = philox_block(seed, (uint32_t)g, (uint32_t)n, seq, 1u, round_offset);
    const uint32_t ws[4] = {w4.x, w4.y, w4.z, w4.w};
    float yv[4], dv[4];
    if (VEC) {
      Logit<E>::stream4(yr + 4 * g, yv);
      if (residual) Logit<E>::stream4(dr + 4 * g, dv);
    } else {
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        const int v = 4 * g + t;
        yv[t] = v < V ? Logit<E>::at(yr, v) : -INFINITY;
        dv[t] = (residual && v < V) ? Logit<E>::at(dr, v) : 0.f;
      }
    }
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      const int v = 4 * g + t;
      if (v >= c1) break;
      // exponents are <= 0 (below the row maxima), so the fast base-2
      // exponential is exact to a few ulp
      const float e = (yv[t] - mp) * c;
      float wv = ex2_approx(e);
      if (residual) wv = wv * invZp - ex2_approx((dv[t] - mq) * c) * invZq;
      if (wv > 0.f) {
        // E / w < best  <=>  u > exp(-best * w): a candidate whose uniform is
        // below that (with a margin far above the rounding of the test)
        // cannot win, and skips the logarithm
        const float u = word_to_uniform(ws[t]);
        if (best == INFINITY || u > ex2_approx(-best * wv * kLog2e) * (1.f - 9.5367431640625e-7f)) {
          const float E = -logf(u);
          const float key = residual ? __fdividef(E, wv) : E * ex2_approx(-e);
          argmin_combine(best, besti, key, v);
        }
      }
    }
  }
  // CTA reduction of (key, index)
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const float k2 = __shfl_xor_sync(0xffffffffu, best, off);
    const int i2 = __shfl_xor_sync(0xffffffffu, besti, off);
    argmin_combine(best, besti, k2, i2);
  }
  if (lane == 0) { smk[warp] = best; smi[warp] = besti; }
  __syncthreads();
  if (threadIdx.x == 0) {
    best = smk[0];
    besti = smi[0];
    for (int w = 1; w < kRowThreads / 32; ++w) argmin_combine(best, besti, smk[w], smi[w]);
    RacePartial p;
    p.key = best;
    p.idx = besti;
    part[(size_t)b * kRaceMaxSplits + split] = p;
    __threadfence();
    const uint32_t ticket = atomicAdd(&cnt[b], 1u);
    last = (ticket == (uint32_t)(nsplit - 1));
  }
  __syncthreads();
  if (!last) return;
  __threadfence();
  if (threadIdx.x < 32) {
    float kb = INFINITY;
    int ib = 0x7fffffff;
    for (int i = lane; i < nsplit; i += 32)
      argmin_combine(kb, ib, __ldcg(&part[(size_t)b * kRaceMaxSplits + i].key),
                     __ldcg(&part[(size_t)b * kRaceMaxSplits + i].idx));
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const float k2 = __shfl_xor_sync(0xffffffffu, kb, off);
      const int i2 = __shfl_xor_sync(0xffffffffu, ib, off);
      argmin_combine(kb, ib, k2, i2);
    }
    if (lane == 0) {
      cnt[b] = 0u;
      sh_bonus = ib;
      sh_ok = (kb < INFINITY);
    }
  }
  __syncthreads();
  if (sh_ok) {
    if (threadIdx.x == 0) {
      n_accepted[b] = n;
      bonus_token[b] = sh_bonus;
    }
    return;
  }
  // Residual identically zero (p_r == q_r to rounding): draw from p_r
  // instead, in this CTA alone (rare).
  best = INFINITY;
  besti = 0x7fffffff;
  for (int v = threadIdx.x; v < V; v += kRowThreads) {
    const uint4 w4 = philox_block(seed, (uint32_t)(v >> 2), (uint32_t)n, seq, 1u, round_offset);
    const uint32_t wsel = (v & 3) == 0 ? w4.x : (v & 3) == 1 ? w4.y : (v & 3) == 2 ? w4.z : w4.w;
    const float wv = exp2f((Logit<E>::at(yr, v) - mp) * c);
    if (wv > 0.f) argmin_combine(best, besti, -logf(word_to_uniform(wsel)) / wv, v);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const float k2 = __shfl_xor_sync(0xffffffffu, best, off);
    const int i2 = __shfl_xor_sync(0xffffffffu, besti, off);
    argmin_combine(best, besti, k2, i2);
  }
  if (lane == 0) { smk[warp] = best; smi[warp] = besti; }
  __syncthreads();
  if (threadIdx.x == 0) {
    best = smk[0];
    besti = smi[0];
    for (int w = 1; w < kRowThreads / 32; ++w) argmin_combine(best, besti, smk[w], smi[w]);
    n_accepted[b] = n;
    bonus_token[b] = besti == 0x7fffffff ? 0 : besti;
  }
}

// ---------------------------------------------------------------------------
// Per-node draws of a draft tree. Grid (nsplit, N+1, B); nodes t > L_b exit
// at once. A greedy sequence (temperature 0) takes the argmax of the node's
// target row; a sampling one draws from softmax(row / T) by the exponential
// race x = argmin_v key_v, key_v = log2(E_v) - y_v log2(e) / T, E_v = -ln u_v,
// u_v from Philox at (v >> 2, node t, sequence, purpose 2), word v & 3. The
// race is carried as an argmax of -key so the partials merge like argmaxes
// (lowest index on ties). A candidate can only win if key_v < best, i.e.
// u_v > exp(-2^(best + y_v c)); that test (two fast exponentials, with a
// margin above their error) skips the logarithms of almost every token.
// The draw of node t lands in stat[b, t].arg for the walk.
// ---------------------------------------------------------------------------
template <bool VEC, typename E>
__global__ void __launch_bounds__(kRowThreads) tree_rows_kernel(
    const E* __restrict__ target, const int32_t* __restrict__ Ls, const float* __restrict__ temperature, int K,
    int V, int nsplit, int chunk, uint64_t seed, uint64_t round_offset, uint32_t seq_offset,
    RowPartial* __restrict__ part, uint32_t* __restrict__ cnt, RowStat* __restrict__ stat, int* __restrict__ status) {
  __shared__ float smf[64];
  __shared__ int smi[32];
  __shared__ int last;
  const int split = blockIdx.x, j = blockIdx.y, b = blockIdx.z;
  const int Lb = Ls[b];
  if (Lb < 0 || Lb > K) {
    if (split == 0 && j == 0 && threadIdx.x == 0) raise_status(status, LIBRASPEC_ST_BAD_LENGTH);
    return;
  }
  if (j > Lb) return;
  const int row = b * (K + 1) + j;
  const float tb = temperature[b];
  const E* xr = target + (size_t)row * V;
  const int c0 = split * chunk, c1 = min(V, c0 + chunk);
  float m;
  int arg;
  if (!(tb > 0.f)) {
    SumAcc sa;
    ArgAcc aa;
    sa.init();
    aa.init();
    row_slice_pass<false, true, VEC, E>(xr, c0, c1, 1.f, sa, aa);
    m = aa.m;
    arg = aa.arg;
  } else {
    const float c = (float)(1.4426950408889634 / (double)tb);
    const uint32_t seq = seq_offset + (uint32_t)b;
    float best = INFINITY;
    int besti = 0x7fffffff;
    for (int g = (c0 >> 2) + threadIdx.x; 4 * g < c1; g += kRowThreads) {
      const uint4 w4 = philox_block(seed, (uint32_t)g, (uint32_t)j, seq, 2u, round_offset);
      const uint32_t ws[4] = {w4.x, w4.y, w4.z, w4.w};
      float yv[4];
      if (VEC) {
        Logit<E>::stream4(xr + 4 * g, yv);
      } else {
#pragma unroll
        for (int t = 0; t < 4; ++t) yv[t] = 4 * g + t < V ? Logit<E>::at(xr, 4 * g + t) : -INFINITY;
      }
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        const int v = 4 * g + t;
        if (v >= c1) break;
        const float yc = yv[t] * c;
        if (!(yc > -INFINITY)) continue;
        const float u = word_to_uniform(ws[t]);
        // key < best  <=>  u > exp(-2^(best + yc)) =: h. The fast exponentials
        // give h to a relative 2e-4 while h is a normal float (exponent above
        // -150; below, h flushes to 0 and every candidate passes): a margin of
        // 2^-12 keeps every possible winner, whose key is then compared exactly.
        if (best == INFINITY || u > ex2_approx(-ex2_approx(best + yc) * kLog2e) * 0.999755859375f) {
          const float key = log2f(-logf(u)) - yc;
          argmin_combine(best, besti, key, v);
        }
      }
    }
    m = -best;
    arg = besti;
  }
  cta_reduce_arg(m, arg, smf, smi);
  if (nsplit == 1) {
    if (threadIdx.x == 0) {
      RowStat st;
      st.m = m;
      st.arg = arg;
      st.Z = 0.0;
      stat[row] = st;
    }
    return;
  }
  if (threadIdx.x == 0) {
    RowPartial p;
    p.m = m;
    p.arg = arg;
    p.s = 0.0;
    part[(size_t)row * kRowMaxSplits + split] = p;
    __threadfence();
    const uint32_t ticket = atomicAdd(&cnt[row], 1u);
    last = (ticket == (uint32_t)(nsplit - 1));
  }
  __syncthreads();
  if (!last || threadIdx.x >= 32) return;
  __threadfence();
  float M;
  int A;
  double Z;
  warp_merge_partials(part + (size_t)row * kRowMaxSplits, nsplit, 0.f, true, M, A, Z);
  if (threadIdx.x == 0) {
    RowStat st;
    st.m = M;
    st.arg = A;
    st.Z = 0.0;
    stat[row] = st;
    cnt[row] = 0u;
  }
}

// ---------------------------------------------------------------------------
// Greedy walk of a draft tree, one warp per sequence. Node t in [1, L_b] has
// parent parent[b, t] < t and token tokens[b, t-1]. The warp first finds, for
// every node p, its matching child next[p]: the lowest-numbered child whose
// token is the argmax of p's target row (argmaxes from accept_rows_kernel),
// by shared-memory atomicMin over the nodes; then it follows next[] from the
// root. n = nodes walked, last = the final node, bonus = its argmax. A parent
// outside [0, t) or a token outside [0, V) never matches and raises its
// status bit.
// ---------------------------------------------------------------------------
constexpr int kWalkWarps = 4;
constexpr int kWalkNodes = LIBRASPEC_MAX_TREE_NODES + 1;

__global__ void __launch_bounds__(kWalkWarps * 32) tree_walk_kernel(
    const int32_t* __restrict__ tokens, const int32_t* __restrict__ parent, const int32_t* __restrict__ Ls, int B,
    int K, int V, const RowStat* __restrict__ stat, int32_t* __restrict__ n_accepted,
    int32_t* __restrict__ last_node, int32_t* __restrict__ bonus, int* __restrict__ status) {
  __shared__ int arg_s[kWalkWarps][kWalkNodes];
  __shared__ int next_s[kWalkWarps][kWalkNodes];
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int b = blockIdx.x * kWalkWarps + w;
  if (b >= B) return;
  const int Lb = Ls[b];
  if (Lb < 0 || Lb > K) {  // accept_rows_kernel raised the status
    if (lane == 0) {
      n_accepted[b] = 0;
      if (last_node) last_node[b] = 0;
      bonus[b] = 0;
    }
    return;
  }
  int* arg = arg_s[w];
  int* next = next_s[w];
  constexpr int kNone = 0x7fffffff;
  for (int t = lane; t <= Lb; t += 32) {
    const int a = __ldcg(&stat[(size_t)b * (K + 1) + t].arg);
    arg[t] = a == 0x7fffffff ? 0 : a;  // a row without a finite logit
    next[t] = kNone;
  }
  __syncwarp();
  for (int t = lane + 1; t <= Lb; t += 32) {
    const int p = parent[(size_t)b * (K + 1) + t];
    const int x = tokens[(size_t)b * K + t - 1];
    if (p < 0 || p >= t) raise_status(status, LIBRASPEC_ST_BAD_TREE);
    else if (x < 0 || x >= V) raise_status(status, LIBRASPEC_ST_BAD_TOKEN);
    else if (x == arg[p]) atomicMin(&next[p], t);
  }
  __syncwarp();
  if (lane == 0) {
    int cur = 0, n = 0;
    while (n < Lb && next[cur] != kNone) {  // next[] only points to higher nodes
      cur = next[cur];
      ++n;
    }
    n_accepted[b] = n;
    if (last_node) last_node[b] = cur;
    bonus[b] = arg[cur];
  }
}

// ---------------------------------------------------------------------------
// Host launchers.
// ---------------------------------------------------------------------------
int num_sms_current();

// temperature == nullptr: every sequence greedy (argmax rows); else per
// sequence, greedy at 0 and drawing at T > 0 (tree_rows_kernel).
template <typename T>
cudaError_t launch_accept_tree(const T* target, const int32_t* tokens, const int32_t* parent, const int32_t* L,
                               const float* temperature, int B, int K, int V, uint64_t seed, uint64_t round_offset,
                               uint32_t seq_offset, int32_t* n_accepted, int32_t* last_node, int32_t* bonus,
                               char* ws, const WsLayout& lay, cudaStream_t stream) {
  if (B == 0) return cudaSuccess;
  const int sms = num_sms_current();
  auto* st = reinterpret_cast<int*>(ws + lay.status);
  auto* rstat = reinterpret_cast<RowStat*>(ws + lay.row_stat);
  const long rows = (long)B * (K + 1);
  const int nsplit0 = row_splits(rows, V, sms, kRowMaxSplits, 4096);
  const int chunk = row_chunk(V, nsplit0);
  const int nsplit = (V + chunk - 1) / chunk;
  dim3 grid(nsplit, K + 1, B);
  auto* part = reinterpret_cast<RowPartial*>(ws + lay.row_part);
  auto* cnt = reinterpret_cast<uint32_t*>(ws + lay.row_cnt);
  const bool vec = rows_vectorizable(target, V);
  if (temperature == nullptr) {
    if (vec)
      accept_rows_kernel<true, T><<<grid, kRowThreads, 0, stream>>>(target, L, nullptr, K, V, nsplit, chunk, part,
                                                                     cnt, rstat, st);
    else
      accept_rows_kernel<false, T><<<grid, kRowThreads, 0, stream>>>(target, L, nullptr, K, V, nsplit, chunk, part,
                                                                      cnt, rstat, st);
  } else if (vec) {
    tree_rows_kernel<true, T><<<grid, kRowThreads, 0, stream>>>(target, L, temperature, K, V, nsplit, chunk, seed,
                                                                 round_offset, seq_offset, part, cnt, rstat, st);
  } else {
    tree_rows_kernel<false, T><<<grid, kRowThreads, 0, stream>>>(target, L, temperature, K, V, nsplit, chunk, seed,
                                                                  round_offset, seq_offset, part, cnt, rstat, st);
  }
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  tree_walk_kernel<<<(B + kWalkWarps - 1) / kWalkWarps, kWalkWarps * 32, 0, stream>>>(
      tokens, parent, L, B, K, V, rstat, n_accepted, last_node, bonus, st);
  return cudaGetLastError();
}
template cudaError_t launch_accept_tree<float>(const float*, const int32_t*, const int32_t*, const int32_t*,
                                               const float*, int, int, int, uint64_t, uint64_t, uint32_t, int32_t*,
                                               int32_t*, int32_t*, char*, const WsLayout&, cudaStream_t);
template cudaError_t launch_accept_tree<uint16_t>(const uint16_t*, const int32_t*, const int32_t*, const int32_t*,
                                                  const float*, int, int, int, uint64_t, uint64_t, uint32_t, int32_t*,
                                                  int32_t*, int32_t*, char*, const WsLayout&, cudaStream_t);

// rng (optional, device): {seed, round_offset, seq_offset} read by the
// kernels in place of the three arguments.
template <typename T>
cudaError_t launch_accept(const T* target, const T* draft, const int32_t* tokens, const float* conf,
                          const float* dstat, const int32_t* L, const float* temperature, int B, int K, int V,
                          uint64_t seed, uint64_t round_offset, uint32_t seq_offset, int32_t* n_accepted,
                          int32_t* bonus, char* ws, const WsLayout& lay, cudaStream_t stream,
                          const uint64_t* rng) {
  if (B == 0) return cudaSuccess;
  const int sms = num_sms_current();
  // the race reads groups of 4 logits: both rows must allow those loads too
  const bool vec = rows_vectorizable(target, V) && (draft == nullptr || rows_vectorizable(draft, V));
  auto* st = reinterpret_cast<int*>(ws + lay.status);
  auto* rstat = reinterpret_cast<RowStat*>(ws + lay.row_stat);
  {
    const long rows = (long)B * (K + 1);
    const int nsplit0 = row_splits(rows, V, sms, kRowMaxSplits, 4096);
    const int chunk = row_chunk(V, nsplit0);
    const int nsplit = (V + chunk - 1) / chunk;
    dim3 grid(nsplit, K + 1, B);
    auto* part = reinterpret_cast<RowPartial*>(ws + lay.row_part);
    auto* cnt = reinterpret_cast<uint32_t*>(ws + lay.row_cnt);
    if (vec)
      accept_rows_kernel<true, T><<<grid, kRowThreads, 0, stream>>>(target, L, temperature, K, V, nsplit, chunk,
                                                                     part, cnt, rstat, st);
    else
      accept_rows_kernel<false, T><<<grid, kRowThreads, 0, stream>>>(target, L, temperature, K, V, nsplit, chunk,
                                                                      part, cnt, rstat, st);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  {
    // race slices: enough CTAs per sequence to stream one or two V-rows fast
    long target_ctas = 4L * sms;
    int nsplit = (int)((target_ctas + B - 1) / B);
    const int cap = (V + 4095) / 4096;
    if (nsplit > cap) nsplit = cap;
    if (nsplit > kRaceMaxSplits) nsplit = kRaceMaxSplits;
    if (nsplit < 1) nsplit = 1;
    int chunk = row_chunk(V, nsplit);
    nsplit = (V + chunk - 1) / chunk;
    dim3 grid(nsplit, B);
    auto* part = reinterpret_cast<RacePartial*>(ws + lay.race_part);
    auto* cnt = reinterpret_cast<uint32_t*>(ws + lay.race_cnt);
    if (vec)
      accept_decide_kernel<true, T><<<grid, kRowThreads, 0, stream>>>(
          target, draft, tokens, conf, dstat, L, temperature, K, V, nsplit, chunk, seed, round_offset, seq_offset,
          rng, rstat, part, cnt, n_accepted, bonus, st);
    else
      accept_decide_kernel<false, T><<<grid, kRowThreads, 0, stream>>>(
          target, draft, tokens, conf, dstat, L, temperature, K, V, nsplit, chunk, seed, round_offset, seq_offset,
          rng, rstat, part, cnt, n_accepted, bonus, st);
    return cudaGetLastError();
  }
}
template cudaError_t launch_accept<float>(const float*, const float*, const int32_t*, const float*, const float*,
                                          const int32_t*, const float*, int, int, int, uint64_t, uint64_t, uint32_t,
                                          int32_t*, int32_t*, char*, const WsLayout&, cudaStream_t,
                                          const uint64_t*);
template cudaError_t launch_accept<uint16_t>(const uint16_t*, const uint16_t*, const int32_t*, const float*,
                                             const float*, const int32_t*, const float*, int, int, int, uint64_t,
                                             uint64_t, uint32_t, int32_t*, int32_t*, char*, const WsLayout&,
                                             cudaStream_t, const uint64_t*);

}  // namespace libraspec
