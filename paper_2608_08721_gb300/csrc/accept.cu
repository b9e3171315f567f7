// Step 4: acceptance (greedy argmax match / rejection sampling).
#include "rowpass.cuh"

namespace libraspec {

// ---------------------------------------------------------------------------
// Row statistics of the node rows of a draft tree (the greedy walk reads
// their argmaxes). Grid (nsplit, K+1, B); rows j > L_b exit at once. Greedy
// sequences need only max / argmax; sampling sequences need (m, Z) at their
// temperature. Partials of a row are merged by the last CTA to finish
// (atomic ticket) into row_stat[b, j].
// ---------------------------------------------------------------------------
template <bool VEC, typename E>
__global__ void __launch_bounds__(kRowThreads) tree_argmax_kernel(
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
  const float c = log2e_over(T);
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
// Acceptance of a chain draft (Sec. 3.1: the target verifies every drafted
// position; the rule is the rejection sampler of Leviathan et al. at T > 0
// and the argmax match at T = 0), in three launches:
//
// accept_plan_kernel (one CTA). From L[] and the temperatures, the rows the
//   decisions read: j <= L_b of a greedy sequence (the argmax of row L_b is
//   its bonus token), j < L_b of a sampling one; cut into S slices, S chosen
//   so that the units fill the rows grid (one unit per CTA); one 8-byte
//   descriptor per unit (sequence, row, slice, L_b, and log2(e)/T of a
//   sampling sequence). A sampling sequence with L_b = 0 is decided here
//   (its bonus draw). In a whole round this launch runs before the attention
//   layers.
// accept_rows_kernel. CTA u reads descriptor u: a greedy row's slice yields
//   (max, argmax); a sampling row's slice (max, sum of exp((y - max) / T))
//   and, from the slice that holds the drafted token x_j, y_{j, x_j}. The CTA
//   completing a sequence's last slice merges its rows and takes the
//   decisions (binary64 p/q against the Philox uniform, or the argmax
//   match): a greedy sequence writes its result; a sampling one records its
//   draw, the bonus draw from row L_b when all drafts were accepted, else the
//   residual draw max(0, p_n - q_n) after the rejection at n.
// accept_race_kernel (a programmatic dependent launch). Grid (slices, B):
//   every recorded draw is an exponential race over the vocabulary, split
//   into slices; the CTA completing a sequence's last slice merges it and
//   writes the result. The bonus race's winner argmin_v E_v / exp((y_v -
//   m) / T) does not depend on the row's max m or normaliser, so its
//   candidates are carried as (E_v, y_v) and compared pairwise and the row
//   needs no statistics pass.
// ---------------------------------------------------------------------------
constexpr int kAccMaxRows = LIBRASPEC_MAX_K + 1;
constexpr int kPlanThreads = 1024;

struct AccPlanHeader {
  int R;      // rows
  int S;      // slices per row
  int chunk;  // logits per slice
  int U;      // units (R * S)
};

// descriptor: b | j << 12 | s << 19 | L_b << 25 (b < 4096, j, L_b <= 64,
// s < 64), and log2(e)/T as float bits (0: a greedy sequence)
__device__ __forceinline__ uint32_t pack_unit(int b, int j, int s, int Lb) {
  return (uint32_t)b | ((uint32_t)j << 12) | ((uint32_t)s << 19) | ((uint32_t)Lb << 25);
}

template <typename E>
struct AcceptArgs {
  const E* target;          // [B, K+1, V]
  const E* draft;           // [B, K, V]
  const int32_t* tokens;    // [B, K]
  const float* conf;        // [B, K] q_j(x_j)
  const float* dstat;       // [B, K, 2] drafter (max, Z)
  const float* temperature; // [B]
  int B, K, V;
  int chunkB, SB;           // race slices: length and count per row
  uint64_t seed, round_offset;
  uint32_t seq_offset;
  const uint64_t* rng;      // optional {seed, round_offset, seq_offset} in device memory
  const AccPlanHeader* hdr;
  const uint2* desc;        // [max(kAccMaxGrid, B*(K+1))]
  RowPartial* part;         // [B*(K+1), kRowMaxSplits]
  float* yx;                // [B*(K+1)]
  uint32_t* seq_cnt;        // [B]
  ResEntry* res;            // [B]
  uint32_t* ready;          // [B] res[b] published (reset by the draw's last CTA)
  RaceCand* rpart;          // [B, kRaceMaxSplits]
  uint32_t* rcnt;           // [B]
  int32_t* n_accepted;
  int32_t* bonus;
  int* status;
};

// (E, y, idx) candidates of a race whose key is E * 2^(-y c): candidate 2
// replaces 1 iff E2 < E1 * 2^((y2 - y1) c), or on equality at a lower index.
__device__ __forceinline__ void race_combine(float& E, float& y, int& i, float E2, float y2, int i2, float c) {
  if (!(E2 < INFINITY)) return;
  if (!(E < INFINITY)) {
    E = E2; y = y2; i = i2;
    return;
  }
  const float X = E * ex2_approx((y2 - y) * c);
  if (E2 < X || (E2 == X && i2 < i)) {
    E = E2; y = y2; i = i2;
  }
}

// The best candidate that any lane of the warp holds, (bEw, byw); bEw = inf
// when no lane has one. Lanes rank their candidates by the log2 key
// log2(bE) - by c with the fast logarithm: a slightly wrong pick only makes
// the screen below a little looser, never unsafe, since the picked
// candidate is a token some lane has drawn. All 32 lanes take part.
__device__ __forceinline__ void warp_best_candidate(float bE, float by, float c, float& bEw, float& byw) {
  const bool has = bE < INFINITY;
  const float lk = has ? __log2f(bE) - by * c : INFINITY;
  float mn = lk;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, off));
  const unsigned ball = __ballot_sync(0xffffffffu, has && lk == mn);
  const int src = ball ? __ffs(ball) - 1 : 0;
  const float e = __shfl_sync(0xffffffffu, bE, src);
  byw = __shfl_sync(0xffffffffu, by, src);
  bEw = ball ? e : INFINITY;
}

// Token v (logit y, Philox word w) in the bonus race. v beats a candidate
// (E, y') iff E_v = -ln u_v < X = E 2^((y - y') c), i.e. u_v > exp(-X). The
// screen tests that against the warp's best candidate (bEw, byw), a token
// already drawn, with a margin of 2^-12 above the fast exponentials' error,
// so every token that can still win the race passes it; a token that
// passes takes the exact logarithm and is compared with the lane's own
// candidate (bE, by, bi). Screening against the warp's candidate rather
// than the lane's own skips the logarithm for most of the slice: a warp
// runs the exact step whenever any of its lanes needs it.
__device__ __forceinline__ void bonus_race_token(float y, uint32_t w, int v, float c, float bEw, float byw, float& bE,
                                                 float& by, int& bi) {
  const float u = word_to_uniform(w);
  if (bEw < INFINITY) {
    const float Xw = bEw * ex2_approx((y - byw) * c);
    if (!(u > ex2_approx(-Xw * kLog2e) * 0.999755859375f)) return;
  }
  const float Ev = -logf(u);
  if (!(bE < INFINITY) || Ev < bE * ex2_approx((y - by) * c)) {
    bE = Ev; by = y; bi = v;
  }
}

// The bonus race over logits [c0, c1) of row j (sampling at c = log2(e)/T):
// uniforms from Philox at (v >> 2, j, seq, purpose 1), word v & 3. Four
// groups of four logits are loaded before any is used. The trip counts are
// the warp's (lanes past the slice's end idle), so that every lane joins
// the refreshes of the warp's candidate: after the first token, then
// before every later group.
template <bool VEC, typename E>
__device__ __forceinline__ void bonus_race_slice(const E* __restrict__ yr, int c0, int c1, int V, float c,
                                                 uint64_t seed, uint32_t j, uint32_t seq, uint64_t round_offset,
                                                 float& bE, float& by, int& bi) {
  const int g1 = (c1 + 3) >> 2;
  const int lane = threadIdx.x & 31;
  float bEw = INFINITY, byw = 0.f;
  bool first = true;
  for (int gw = (c0 >> 2) + (int)(threadIdx.x & ~31u); gw < g1; gw += 4 * kRowThreads) {
    const int g = gw + lane;
    float yv[4][4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int gg = g + k * kRowThreads;
      if (gg < g1) {
        if (VEC) {
          Logit<E>::stream4(yr + 4 * gg, yv[k]);
        } else {
#pragma unroll
          for (int t = 0; t < 4; ++t) yv[k][t] = 4 * gg + t < V ? Logit<E>::at(yr, 4 * gg + t) : -INFINITY;
        }
      } else {
#pragma unroll
        for (int t = 0; t < 4; ++t) yv[k][t] = -INFINITY;
      }
    }
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      if (gw + k * kRowThreads >= g1) break;  // the same for the whole warp
      if (!first) warp_best_candidate(bE, by, c, bEw, byw);
      const int gg = g + k * kRowThreads;
      uint4 w4 = make_uint4(0u, 0u, 0u, 0u);
      if (gg < g1) w4 = philox_block(seed, (uint32_t)gg, j, seq, 1u, round_offset);
      const uint32_t ws[4] = {w4.x, w4.y, w4.z, w4.w};
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        const int v = 4 * gg + t;
        if (v < c1 && yv[k][t] > -INFINITY) bonus_race_token(yv[k][t], ws[t], v, c, bEw, byw, bE, by, bi);
        if (t == 0 && first) warp_best_candidate(bE, by, c, bEw, byw);
      }
      first = false;
    }
  }
}

// CTA reduction of race candidates; result in thread 0.
__device__ __forceinline__ void cta_reduce_race(float& E, float& y, int& i, float c, float* smE /*[32]*/,
                                                float* smy /*[32]*/, int* smi /*[32]*/) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const float E2 = __shfl_xor_sync(0xffffffffu, E, off);
    const float y2 = __shfl_xor_sync(0xffffffffu, y, off);
    const int i2 = __shfl_xor_sync(0xffffffffu, i, off);
    race_combine(E, y, i, E2, y2, i2, c);
  }
  if (lane == 0) { smE[warp] = E; smy[warp] = y; smi[warp] = i; }
  __syncthreads();
  if (threadIdx.x == 0) {
    E = smE[0]; y = smy[0]; i = smi[0];
    for (int w = 1; w < (int)(blockDim.x >> 5); ++w) race_combine(E, y, i, smE[w], smy[w], smi[w], c);
  }
}

// Largest b with start[b] <= r (rows of empty sequences are skipped).
__device__ __forceinline__ int seq_of_row(const int* start, int B, int r) {
  int lo = 0, hi = B - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (start[mid] <= r) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

// The smallest key any lane of the warp holds (all 32 lanes take part).
__device__ __forceinline__ float warp_min_key(float k) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) k = fminf(k, __shfl_xor_sync(0xffffffffu, k, off));
  return k;
}

// Residual race of queued entry e over slice s: w_v = max(0, p_v - q_v),
// key E_v / w_v, uniforms at (v >> 2, n, seq, purpose 1). The screen tests
// each token against the smaller of the lane's best key and the warp's best
// at its last refresh (a key some lane has drawn); the trip counts are the
// warp's, so every lane joins the refreshes.
template <bool VEC, typename E>
__device__ __forceinline__ void residual_race_slice(const E* __restrict__ yr, const E* __restrict__ dr, int c0,
                                                    int c1, int V, float c, float mp, float invZp, float mq,
                                                    float invZq, uint64_t seed, uint32_t n, uint32_t seq,
                                                    uint64_t round_offset, float& best, int& besti) {
  const int g1 = (c1 + 3) >> 2;
  const int lane = threadIdx.x & 31;
  float bw = INFINITY;
  bool first = true;
  for (int gw = (c0 >> 2) + (int)(threadIdx.x & ~31u); gw < g1; gw += 2 * kRowThreads) {
    const int g = gw + lane;
    float yv[2][4], dv[2][4];
#pragma unroll
    for (int k = 0; k < 2; ++k) {
      const int gg = g + k * kRowThreads;
      if (gg < g1) {
        if (VEC) {
          Logit<E>::stream4(yr + 4 * gg, yv[k]);
          Logit<E>::stream4(dr + 4 * gg, dv[k]);
        } else {
#pragma unroll
          for (int t = 0; t < 4; ++t) {
            const int v = 4 * gg + t;
            yv[k][t] = v < V ? Logit<E>::at(yr, v) : -INFINITY;
            dv[k][t] = v < V ? Logit<E>::at(dr, v) : 0.f;
          }
        }
      } else {
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          yv[k][t] = -INFINITY;
          dv[k][t] = 0.f;
        }
      }
    }
#pragma unroll
    for (int k = 0; k < 2; ++k) {
      if (gw + k * kRowThreads >= g1) break;  // the same for the whole warp
      if (!first) bw = warp_min_key(best);
      const int gg = g + k * kRowThreads;
      uint4 w4 = make_uint4(0u, 0u, 0u, 0u);
      if (gg < g1) w4 = philox_block(seed, (uint32_t)gg, n, seq, 1u, round_offset);
      const uint32_t ws[4] = {w4.x, w4.y, w4.z, w4.w};
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        const int v = 4 * gg + t;
        if (v < c1 && gg < g1) {
          // exponents are <= 0 (below the row maxima), so the fast base-2
          // exponential is exact to a few ulp
          const float wv = ex2_approx((yv[k][t] - mp) * c) * invZp - ex2_approx((dv[k][t] - mq) * c) * invZq;
          if (wv > 0.f) {
            // E / w < thr  <=>  u > exp(-thr * w): a candidate whose uniform is
            // below that (with a margin far above the rounding of the test)
            // cannot win, and skips the logarithm
            const float u = word_to_uniform(ws[t]);
            const float thr = fminf(best, bw);
            if (thr == INFINITY || u > ex2_approx(-thr * wv * kLog2e) * (1.f - 9.5367431640625e-7f)) {
              const float Ev = -logf(u);
              argmin_combine(best, besti, __fdividef(Ev, wv), v);
            }
          }
        }
        if (t == 0 && first) bw = warp_min_key(best);
      }
      first = false;
    }
  }
}

// CTA argmin of (key, index); result in thread 0.
__device__ __forceinline__ void cta_reduce_min(float& best, int& besti, float* smk, int* smi) {
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
    for (int w = 1; w < (int)(blockDim.x >> 5); ++w) argmin_combine(best, besti, smk[w], smi[w]);
  }
}

__device__ __forceinline__ uint32_t ld_acquire_u32(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Publish sequence b's draw (release: the entry is visible before the flag).
__device__ __forceinline__ void publish_draw(ResEntry* res, uint32_t* ready, int b, const ResEntry& en) {
  res[b] = en;
  __threadfence();
  asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(ready + b), "r"(1u) : "memory");
}

// Bounded wait for a published flag: false after limit_ns (LIBRASPEC_ST_TIMEOUT).
__device__ bool wait_published(const uint32_t* flag, int* status, uint64_t limit_ns = 2000000000ull) {
  uint64_t t0 = 0;
  for (uint32_t it = 0;; ++it) {
    if (ld_acquire_u32(flag) != 0u) return true;
    if (it == 0) {
      asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t0));
    } else if ((it & 7u) == 0u) {
      uint64_t t;
      asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
      if (t - t0 > limit_ns) {
        raise_status(status, LIBRASPEC_ST_TIMEOUT);
        return false;
      }
    }
    __nanosleep(it < 8 ? 128u : 1024u);
  }
}

// The plan of the rows grid (G CTAs). A sequence whose L_b lies outside
// [0, K], or that samples without q, gets no rows and its result at once.
__global__ void __launch_bounds__(kPlanThreads) accept_plan_kernel(const int32_t* __restrict__ Ls,
                                                                   const float* __restrict__ temperature,
                                                                   int have_q, int B, int K, int V, int G,
                                                                   AccPlanHeader* __restrict__ hdr,
                                                                   uint2* __restrict__ desc,
                                                                   int32_t* __restrict__ n_accepted,
                                                                   int32_t* __restrict__ bonus,
                                                                   ResEntry* __restrict__ res,
                                                                   uint32_t* __restrict__ ready,
                                                                   int* __restrict__ status) {
  __shared__ int s_start[LIBRASPEC_MAX_B + 1];
  __shared__ float s_c[LIBRASPEC_MAX_B];
  __shared__ int s_L[LIBRASPEC_MAX_B];
  __shared__ int smi[32];
  __shared__ int s_tot;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int per = (B + kPlanThreads - 1) / kPlanThreads;
  int loc = 0;
  for (int i = 0; i < per; ++i) {
    const int b = tid * per + i;
    if (b >= B) break;
    const int Lb = Ls[b];
    const float tb = temperature[b];
    const bool sampling = tb > 0.f;
    const bool bad_len = Lb < 0 || Lb > K;
    int r = 0;
    ResEntry en;
    en.n = -1;
    en.mode = 0;
    en.mp = 0.f;
    en.invZp = 0.f;
    if (bad_len || (sampling && !have_q)) {
      n_accepted[b] = 0;
      bonus[b] = 0;
      if (sampling) publish_draw(res, ready, b, en);  // its draw CTAs wait for a draw (none)
      raise_status(status, bad_len ? LIBRASPEC_ST_BAD_LENGTH : LIBRASPEC_ST_MISSING_INPUT);
    } else if (!sampling) {
      r = Lb + 1;
    } else if (Lb > 0) {
      r = Lb;
    } else {  // no draft to verify: the bonus draw from row 0
      en.n = 0;
      en.mode = 1;
      publish_draw(res, ready, b, en);
    }
    s_start[b] = r;  // rows for now, turned into the prefix below
    s_c[b] = sampling ? log2e_over(tb) : 0.f;
    s_L[b] = Lb;
    loc += r;
  }
  int incl = loc;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int o = __shfl_up_sync(0xffffffffu, incl, off);
    if (lane >= off) incl += o;
  }
  if (lane == 31) smi[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    const int t = smi[lane];
    int ti = t;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int o = __shfl_up_sync(0xffffffffu, ti, off);
      if (lane >= off) ti += o;
    }
    smi[lane] = ti - t;  // exclusive prefix of the warp totals
    if (lane == 31) s_tot = ti;
  }
  __syncthreads();
  {
    int run = smi[warp] + incl - loc;
    for (int i = 0; i < per; ++i) {
      const int b = tid * per + i;
      if (b >= B) break;
      const int r = s_start[b];
      s_start[b] = run;
      run += r;
    }
  }
  const int R = s_tot;
  // slices per row: as many as the grid holds (one unit per CTA), each of at
  // least 2048 logits
  const int smax = max(1, min(kRowMaxSplits, (V + 2047) / 2048));
  int S = R > 0 ? G / R : 1;
  S = max(1, min(S, smax));
  const int chunk = (((V + S - 1) / S) + kRowAlign - 1) & ~(kRowAlign - 1);
  S = (V + chunk - 1) / chunk;
  const int U = R * S;
  if (tid == 0) {
    s_start[B] = R;
    AccPlanHeader h;
    h.R = R;
    h.S = S;
    h.chunk = chunk;
    h.U = U;
    *hdr = h;
  }
  __syncthreads();
  for (int u = tid; u < U; u += kPlanThreads) {
    const int r = u / S, s = u - r * S;
    const int b = seq_of_row(s_start, B, r);
    desc[u] = make_uint2(pack_unit(b, r - s_start[b], s, s_L[b]), __float_as_uint(s_c[b]));
  }
}

template <bool VEC, typename E>
__global__ void __launch_bounds__(kRowThreads, 6) accept_rows_kernel(const AcceptArgs<E> a) {
  __shared__ float s_m[kAccMaxRows];
  __shared__ double s_Z[kAccMaxRows];
  __shared__ int s_arg[kAccMaxRows];
  __shared__ float smf[64];
  __shared__ int smi[32];
  __shared__ int sh[1];
  __shared__ float s_yx;
  // the race launch may start its CTAs (they wait for this grid's end)
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int G = gridDim.x;
  const int K = a.K, V = a.V;
  const AccPlanHeader h = *a.hdr;
  uint2 d = a.desc[blockIdx.x];  // read beside the header (stale beyond the plan's units)
  if ((int)blockIdx.x >= h.U) return;
  const int S = h.S, chunk = h.chunk;

  for (int u = blockIdx.x; u < h.U; u += G) {
    if (u != (int)blockIdx.x) d = a.desc[u];
    const int b = (int)(d.x & 0xfffu), j = (int)((d.x >> 12) & 0x7fu), s = (int)((d.x >> 19) & 0x3fu);
    const int Lb = (int)(d.x >> 25);
    const float c = __uint_as_float(d.y);
    const bool sampling = c > 0.f;
    const int rows_b = sampling ? Lb : Lb + 1;
    const size_t row = (size_t)b * (K + 1) + j;
    const E* yr = a.target + row * V;
    const int c0 = s * chunk, c1 = min(V, c0 + chunk);
    RowPartial* pp = a.part + row * kRowMaxSplits + s;
    if (!sampling) {
      SumAcc sa;
      ArgAcc aa;
      sa.init();
      aa.init();
      row_slice_pass<false, true, VEC, E>(yr, c0, c1, 1.f, sa, aa);
      float m = aa.m;
      int arg = aa.arg;
      cta_reduce_arg(m, arg, smf, smi);
      if (tid == 0) {
        RowPartial p;
        p.m = m;
        p.arg = arg;
        p.s = 0.0;
        *pp = p;
      }
    } else {
      // the drafted token's logit: kept by the thread that streams it
      const int x = a.tokens[(size_t)b * K + j];
      SumAcc sa;
      ArgAcc aa;
      sa.init();
      row_slice_pass<true, false, VEC, E, true>(yr, c0, c1, c, sa, aa, x, &s_yx);
      float m = sa.m, sum = sa.value();
      cta_reduce_sum(m, sum, c, smf);  // its barrier also publishes s_yx
      if (tid == 0) {
        RowPartial p;
        p.m = m;
        p.arg = 0;
        p.s = (double)sum;
        *pp = p;
        if (x >= c0 && x < c1) a.yx[row] = s_yx;
      }
    }
    if (tid == 0) {
      __threadfence();
      sh[0] = atomicAdd(&a.seq_cnt[b], 1u) == (uint32_t)(rows_b * S - 1);
    }
    __syncthreads();
    if (!sh[0]) continue;

    // ---- decision for sequence b (this CTA completed its last slice) ----
    __threadfence();
    const size_t row0 = (size_t)b * (K + 1);
    // the first 32 decisions' inputs, loaded beside the merges
    int xj = 0;
    float yj = 0.f, qj = 0.f;
    if (warp == 0 && lane < Lb) {
      xj = a.tokens[(size_t)b * K + lane];
      if (sampling) {
        yj = __ldcg(&a.yx[row0 + lane]);
        qj = a.conf[(size_t)b * K + lane];
      }
    }
    for (int jj = warp; jj < rows_b; jj += kRowThreads / 32) {
      const RowPartial* p = a.part + (row0 + jj) * kRowMaxSplits;
      float M;
      int A;
      double Z;
      if (!sampling) {
        warp_merge_partials(p, S, 0.f, true, M, A, Z);
        if (lane == 0) s_arg[jj] = A;
      } else {
        warp_merge_partials(p, S, c, false, M, A, Z);
        if (lane == 0) { s_m[jj] = M; s_Z[jj] = Z; }
      }
    }
    __syncthreads();
    if (warp == 0) {
      uint64_t seed = a.seed, round_offset = a.round_offset;
      uint32_t seq_offset = a.seq_offset;
      if (a.rng) {  // the generator's arguments from device memory (a replayed graph of a staged round)
        seed = a.rng[0];
        round_offset = a.rng[1];
        seq_offset = (uint32_t)a.rng[2];
      }
      int n = Lb;
      for (int base = 0; base < Lb; base += 32) {
        const int jj = base + lane;
        bool reject = false;
        if (jj < Lb) {
          const int x = base == 0 ? xj : a.tokens[(size_t)b * K + jj];
          if (x < 0 || x >= V) {
            raise_status(a.status, LIBRASPEC_ST_BAD_TOKEN);
            reject = true;
          } else if (!sampling) {
            reject = s_arg[jj] != x;
          } else {
            const float y = base == 0 ? yj : __ldcg(&a.yx[row0 + jj]);
            const double p = (double)exp2f((y - s_m[jj]) * c) / s_Z[jj];
            const double q = (double)(base == 0 ? qj : a.conf[(size_t)b * K + jj]);
            const double ratio = (q <= p) ? 1.0 : p / q;
            const uint4 w = philox_block(seed, 0u, (uint32_t)jj, seq_offset + (uint32_t)b, 0u, round_offset);
            reject = !((double)word_to_uniform(w.x) < ratio);
          }
        }
        const unsigned ball = __ballot_sync(0xffffffffu, reject);
        if (ball) {
          n = base + __ffs(ball) - 1;
          break;
        }
      }
      if (lane == 0) {
        a.seq_cnt[b] = 0u;  // ready for the next call
        ResEntry en;
        en.n = n;
        en.mode = 0;
        en.mp = 0.f;
        en.invZp = 0.f;
        if (!sampling) {
          const int w = s_arg[n];
          a.n_accepted[b] = n;
          a.bonus[b] = w == 0x7fffffff ? 0 : w;  // a row without a finite logit
        } else {
          if (n == Lb) {
            en.mode = 1;  // all drafts accepted: the bonus draw from row L_b
          } else {
            en.mode = 2;  // rejected at n: the residual draw
            en.mp = s_m[n];
            en.invZp = (float)(1.0 / s_Z[n]);
          }
          publish_draw(a.res, a.ready, b, en);
        }
      }
    }
    __syncthreads();
  }
}

// The draws: CTA (s, b) runs slice s of sequence b's race, if b recorded
// one; the CTA completing the last slice merges the race and writes
// (n, the drawn token). A programmatic dependent launch of the rows grid:
// it starts once every rows CTA has started, and each CTA waits (bounded)
// only for its own sequence's decision, so a sequence's race overlaps the
// rows still streaming for the others.
template <bool VEC, typename E>
__global__ void __launch_bounds__(kRowThreads, 4) accept_race_kernel(const AcceptArgs<E> a) {
  __shared__ float smk[32];
  __shared__ float smy[32];
  __shared__ int smi[32];
  __shared__ int sh[2];
  __shared__ ResEntry s_en;
  __shared__ float s_c;
  const int s = blockIdx.x, b = blockIdx.y;
  // a greedy sequence has no draw (and publishes none): its CTAs leave at
  // once, so they hold no slot while the sampling races wait and run
  if (!(a.temperature[b] > 0.f)) return;
  if (threadIdx.x == 0) {
    sh[0] = wait_published(a.ready + b, a.status);
    s_en = a.res[b];
    s_c = log2e_over(a.temperature[b]);  // once per CTA: a binary32 division and reciprocal
  }
  __syncthreads();
  if (!sh[0]) return;
  const ResEntry en = s_en;
  if (en.mode == 0) {  // nothing to draw: the last CTA of b resets the flag
    if (threadIdx.x == 0 && atomicAdd(&a.rcnt[b], 1u) == (uint32_t)(a.SB - 1)) {
      a.rcnt[b] = 0u;
      a.ready[b] = 0u;
    }
    return;
  }
  const int n = en.n;
  uint64_t seed = a.seed, round_offset = a.round_offset;
  uint32_t seq_offset = a.seq_offset;
  if (a.rng) {
    seed = a.rng[0];
    round_offset = a.rng[1];
    seq_offset = (uint32_t)a.rng[2];
  }
  const int K = a.K, V = a.V;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const float c = s_c;
  const E* yr = a.target + ((size_t)b * (K + 1) + n) * V;
  const uint32_t seq = seq_offset + (uint32_t)b;
  const int c0 = s * a.chunkB, c1 = min(V, c0 + a.chunkB);
  const bool residual = en.mode == 2;
  float bE = INFINITY, by = 0.f;
  int bi = 0x7fffffff;
  if (residual) {
    const E* dr = a.draft + ((size_t)b * K + n) * V;
    const float mq = a.dstat[2 * ((size_t)b * K + n)];
    const float invZq = 1.0f / a.dstat[2 * ((size_t)b * K + n) + 1];
    residual_race_slice<VEC, E>(yr, dr, c0, c1, V, c, en.mp, en.invZp, mq, invZq, seed, (uint32_t)n, seq,
                                round_offset, bE, bi);
    cta_reduce_min(bE, bi, smk, smi);
  } else {
    bonus_race_slice<VEC, E>(yr, c0, c1, V, c, seed, (uint32_t)n, seq, round_offset, bE, by, bi);
    cta_reduce_race(bE, by, bi, c, smk, smy, smi);
  }
  if (tid == 0) {
    RaceCand p;
    p.E = bE;
    p.y = by;
    p.idx = bi;
    p.pad = 0;
    a.rpart[(size_t)b * kRaceMaxSplits + s] = p;
    __threadfence();
    sh[0] = atomicAdd(&a.rcnt[b], 1u) == (uint32_t)(a.SB - 1);
  }
  __syncthreads();
  if (!sh[0]) return;
  __threadfence();
  if (warp == 0) {
    float kb = INFINITY, ky = 0.f;
    int ib = 0x7fffffff;
    const RaceCand* rp = a.rpart + (size_t)b * kRaceMaxSplits;
    for (int i = lane; i < a.SB; i += 32) {
      if (residual) argmin_combine(kb, ib, __ldcg(&rp[i].E), __ldcg(&rp[i].idx));
      else race_combine(kb, ky, ib, __ldcg(&rp[i].E), __ldcg(&rp[i].y), __ldcg(&rp[i].idx), c);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const float k2 = __shfl_xor_sync(0xffffffffu, kb, off);
      const float y2 = __shfl_xor_sync(0xffffffffu, ky, off);
      const int i2 = __shfl_xor_sync(0xffffffffu, ib, off);
      if (residual) argmin_combine(kb, ib, k2, i2);
      else race_combine(kb, ky, ib, k2, y2, i2, c);
    }
    if (lane == 0) {
      a.rcnt[b] = 0u;  // ready for the next call
      a.ready[b] = 0u;
      sh[1] = kb < INFINITY ? ib : (residual ? -1 : 0);  // a bonus row without a finite logit: token 0
    }
  }
  __syncthreads();
  int win = sh[1];
  if (win < 0) {
    // residual identically zero (p_n == q_n to rounding): draw from p_n
    // instead, in this CTA alone (rare)
    float bk = INFINITY;
    int bkI = 0x7fffffff;
    for (int v = tid; v < V; v += kRowThreads) {
      const uint4 w4 = philox_block(seed, (uint32_t)(v >> 2), (uint32_t)n, seq, 1u, round_offset);
      const uint32_t wsel = (v & 3) == 0 ? w4.x : (v & 3) == 1 ? w4.y : (v & 3) == 2 ? w4.z : w4.w;
      const float wv = exp2f((Logit<E>::at(yr, v) - en.mp) * c);
      if (wv > 0.f) argmin_combine(bk, bkI, -logf(word_to_uniform(wsel)) / wv, v);
    }
    cta_reduce_min(bk, bkI, smk, smi);
    win = bkI == 0x7fffffff ? 0 : bkI;
  }
  if (tid == 0) {
    a.n_accepted[b] = n;
    a.bonus[b] = win;
  }
}

// Failure-detection self-test: the draws' bounded wait on a device flag with
// a caller-given limit; observed = 1 if the flag was seen, 0 if the wait
// gave up (and raised LIBRASPEC_ST_TIMEOUT).
__global__ void selftest_wait_kernel(const uint32_t* __restrict__ flag, uint64_t limit_ns,
                                     int32_t* __restrict__ observed, int* __restrict__ status) {
  if (threadIdx.x == 0) *observed = wait_published(flag, status, limit_ns) ? 1 : 0;
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
    const float c = log2e_over(tb);
    const uint32_t seq = seq_offset + (uint32_t)b;
    float best = INFINITY;
    int besti = 0x7fffffff;
    // the screen's threshold: the smaller of the lane's best key and the
    // warp's best at its last refresh (a key some lane has drawn), refreshed
    // after the first token and then before groups 1, 2, 3 and every fourth;
    // the trip counts are the warp's, so every lane joins the refreshes
    float bw = INFINITY;
    const int lane = threadIdx.x & 31;
    int it = 0;
    for (int gw = (c0 >> 2) + (int)(threadIdx.x & ~31u); 4 * gw < c1; gw += kRowThreads, ++it) {
      if (it > 0 && (it < 4 || (it & 3) == 0)) bw = warp_min_key(best);
      const int g = gw + lane;
      const bool live = 4 * g < c1;
      uint4 w4 = make_uint4(0u, 0u, 0u, 0u);
      float yv[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
      if (live) {
        w4 = philox_block(seed, (uint32_t)g, (uint32_t)j, seq, 2u, round_offset);
        if (VEC) {
          Logit<E>::stream4(xr + 4 * g, yv);
        } else {
#pragma unroll
          for (int t = 0; t < 4; ++t) yv[t] = 4 * g + t < V ? Logit<E>::at(xr, 4 * g + t) : -INFINITY;
        }
      }
      const uint32_t ws[4] = {w4.x, w4.y, w4.z, w4.w};
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        const int v = 4 * g + t;
        const float yc = yv[t] * c;
        if (v < c1 && yc > -INFINITY) {
          const float u = word_to_uniform(ws[t]);
          // key < thr  <=>  u > exp(-2^(thr + yc)) =: h. The fast exponentials
          // give h to a relative 2e-4 while h is a normal float (exponent above
          // -150; below, h flushes to 0 and every candidate passes): a margin of
          // 2^-12 keeps every possible winner, whose key is then compared exactly.
          const float thr = fminf(best, bw);
          if (thr == INFINITY || u > ex2_approx(-ex2_approx(thr + yc) * kLog2e) * 0.999755859375f) {
            const float key = log2f(-logf(u)) - yc;
            argmin_combine(best, besti, key, v);
          }
        }
        if (t == 0 && it == 0) bw = warp_min_key(best);
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
// token is the argmax of p's target row (argmaxes from tree_argmax_kernel),
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
  if (Lb < 0 || Lb > K) {  // tree_argmax_kernel raised the status
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
      tree_argmax_kernel<true, T><<<grid, kRowThreads, 0, stream>>>(target, L, nullptr, K, V, nsplit, chunk, part,
                                                                     cnt, rstat, st);
    else
      tree_argmax_kernel<false, T><<<grid, kRowThreads, 0, stream>>>(target, L, nullptr, K, V, nsplit, chunk, part,
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

// CTAs of the acceptance rows kernel resident at once on the current device;
// its grid is two waves of them (at most kAccMaxGrid; measured on the ragged
// batch: 51.5 us back to back against 54.3 with four waves, 53.0 with three).
template <bool VEC, typename T>
int accept_grid() {
  static int cached[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  int g = cached[dev];
  if (g == 0) {
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, accept_rows_kernel<VEC, T>, kRowThreads, 0) !=
            cudaSuccess ||
        per_sm < 1)
      per_sm = 1;
    g = std::min(2 * per_sm * num_sms_current(), kAccMaxGrid);
    cached[dev] = g;
  }
  return g;
}

template <typename T>
bool accept_vec(const T* target, const T* draft, int V) {
  // the races read groups of 4 logits: both rows must allow those loads too
  return rows_vectorizable(target, V) && (draft == nullptr || rows_vectorizable(draft, V));
}

// The acceptance plan for the rows grid of launch_accept<T> with the same
// pointers' alignment (one CTA; needs only L and the temperatures).
template <typename T>
cudaError_t launch_accept_plan(const T* target, const T* draft, const float* conf, const float* dstat,
                               const int32_t* L, const float* temperature, int B, int K, int V, int32_t* n_accepted,
                               int32_t* bonus, char* ws, const WsLayout& lay, cudaStream_t stream) {
  if (B == 0) return cudaSuccess;
  const int G = accept_vec(target, draft, V) ? accept_grid<true, T>() : accept_grid<false, T>();
  if (G <= 0) return cudaErrorInvalidConfiguration;
  accept_plan_kernel<<<1, kPlanThreads, 0, stream>>>(
      L, temperature, conf != nullptr && dstat != nullptr, B, K, V, G,
      reinterpret_cast<AccPlanHeader*>(ws + lay.acc_plan), reinterpret_cast<uint2*>(ws + lay.acc_plan + 16),
      n_accepted, bonus, reinterpret_cast<ResEntry*>(ws + lay.acc_res),
      reinterpret_cast<uint32_t*>(ws + lay.acc_ready), reinterpret_cast<int*>(ws + lay.status));
  return cudaGetLastError();
}

// rng (optional, device): {seed, round_offset, seq_offset} read by the
// kernels in place of the three arguments. plan_ready: launch_accept_plan
// already ran for these inputs on this stream.
template <typename T>
cudaError_t launch_accept(const T* target, const T* draft, const int32_t* tokens, const float* conf,
                          const float* dstat, const int32_t* L, const float* temperature, int B, int K, int V,
                          uint64_t seed, uint64_t round_offset, uint32_t seq_offset, int32_t* n_accepted,
                          int32_t* bonus, char* ws, const WsLayout& lay, cudaStream_t stream,
                          const uint64_t* rng, bool plan_ready) {
  if (B == 0) return cudaSuccess;
  if (!plan_ready) {
    const cudaError_t e = launch_accept_plan<T>(target, draft, conf, dstat, L, temperature, B, K, V, n_accepted,
                                                bonus, ws, lay, stream);
    if (e != cudaSuccess) return e;
  }
  const bool vec = accept_vec(target, draft, V);
  AcceptArgs<T> a;
  a.target = target;
  a.draft = draft;
  a.tokens = tokens;
  a.conf = conf;
  a.dstat = dstat;
  a.temperature = temperature;
  a.B = B;
  a.K = K;
  a.V = V;
  // race slices of about 4096 logits of each row
  int SB = (V + 4095) / 4096;
  if (SB > kRaceMaxSplits) SB = kRaceMaxSplits;
  const int chunkB = row_chunk(V, SB);
  a.SB = (V + chunkB - 1) / chunkB;
  a.chunkB = chunkB;
  a.seed = seed;
  a.round_offset = round_offset;
  a.seq_offset = seq_offset;
  a.rng = rng;
  a.hdr = reinterpret_cast<const AccPlanHeader*>(ws + lay.acc_plan);
  a.desc = reinterpret_cast<const uint2*>(ws + lay.acc_plan + 16);
  a.part = reinterpret_cast<RowPartial*>(ws + lay.row_part);
  a.yx = reinterpret_cast<float*>(ws + lay.acc_yx);
  a.seq_cnt = reinterpret_cast<uint32_t*>(ws + lay.acc_seq);
  a.res = reinterpret_cast<ResEntry*>(ws + lay.acc_res);
  a.ready = reinterpret_cast<uint32_t*>(ws + lay.acc_ready);
  a.rpart = reinterpret_cast<RaceCand*>(ws + lay.race_part);
  a.rcnt = reinterpret_cast<uint32_t*>(ws + lay.race_cnt);
  a.n_accepted = n_accepted;
  a.bonus = bonus;
  a.status = reinterpret_cast<int*>(ws + lay.status);
  const int G = vec ? accept_grid<true, T>() : accept_grid<false, T>();
  if (G <= 0) return cudaErrorInvalidConfiguration;
  if (vec)
    accept_rows_kernel<true, T><<<G, kRowThreads, 0, stream>>>(a);
  else
    accept_rows_kernel<false, T><<<G, kRowThreads, 0, stream>>>(a);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  // the draws: launched once every rows CTA has started (each waits for its sequence)
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.SB, B);
  cfg.blockDim = dim3(kRowThreads);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (vec) return cudaLaunchKernelEx(&cfg, accept_race_kernel<true, T>, a);
  return cudaLaunchKernelEx(&cfg, accept_race_kernel<false, T>, a);
}
template cudaError_t launch_accept<float>(const float*, const float*, const int32_t*, const float*, const float*,
                                          const int32_t*, const float*, int, int, int, uint64_t, uint64_t, uint32_t,
                                          int32_t*, int32_t*, char*, const WsLayout&, cudaStream_t,
                                          const uint64_t*, bool);
template cudaError_t launch_accept_plan<float>(const float*, const float*, const float*, const float*,
                                               const int32_t*, const float*, int, int, int, int32_t*, int32_t*,
                                               char*, const WsLayout&, cudaStream_t);
template cudaError_t launch_accept_plan<uint16_t>(const uint16_t*, const uint16_t*, const float*, const float*,
                                                  const int32_t*, const float*, int, int, int, int32_t*, int32_t*,
                                                  char*, const WsLayout&, cudaStream_t);
cudaError_t launch_selftest_wait(const uint32_t* flag, uint64_t limit_ns, int32_t* observed, int* status,
                                 cudaStream_t stream) {
  selftest_wait_kernel<<<1, 32, 0, stream>>>(flag, limit_ns, observed, status);
  return cudaGetLastError();
}

template cudaError_t launch_accept<uint16_t>(const uint16_t*, const uint16_t*, const int32_t*, const float*,
                                             const float*, const int32_t*, const float*, int, int, int, uint64_t,
                                             uint64_t, uint32_t, int32_t*, int32_t*, char*, const WsLayout&,
                                             cudaStream_t, const uint64_t*, bool);

}  // namespace libraspec
