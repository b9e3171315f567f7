/*
 * LibraSpec verify-round ORACLE — plain, slow, CPU-only, fp64.
 *
 * This file is TEST INFRASTRUCTURE. Only the tests, the smoke check and the
 * benchmark's CPU-baseline leg load it. It shares no code, header, table or
 * helper with the CUDA library; the two meet only through the seeded input
 * arrays both are given.
 *
 * What it computes, step by step, and where each step comes from:
 *
 *   oracle_confidence      drafter confidence q_k of the drafted token
 *                          (Sec. 3.4, Assumption 1: q stands in for the
 *                          acceptance probability p; Algorithm 1 uses q_k).
 *   oracle_select_lengths  marginal-gain length selection: extend L -> L+1
 *                          while prod_{k<=L+1} q_k * T(L) > c_L * E[tau_L]
 *                          (Thm. 4, derived from Thm. 1's ratio comparison;
 *                          prefix acceptance Pr = prod q, E[tau] = sum of
 *                          cumulative products, proof of Thm. 2).
 *   oracle_select_iterate  iterated single beneficial adjustments (Def. 1,
 *                          Thm. 1 both cases, Thm. 5) from any start length.
 *   oracle_select_alpha    the alpha-mode length search of Algorithm 1:
 *                          position-wise bounds eps_i (Thm. 2 / Thm. 3 with
 *                          the trade-off weight alpha), eps* = min_i eps_i,
 *                          block-wise drafting budget, one rollback.
 *   oracle_gather_pages    the dense KV cache a paged cache (page pool and
 *                          block table) describes.
 *   oracle_verify_attn_tree, oracle_accept_tree_greedy, oracle_accept_tree
 *                          verification of a draft tree (the tree drafters
 *                          of Sec. 2, e.g. DDTree): ancestor-masked
 *                          attention, the greedy longest accepted path and
 *                          its sampling counterpart.
 *   oracle_lm_head_stats   confidence / acceptance row statistics from an LM
 *                          head's hidden states and weights (logits
 *                          never stored).
 *   oracle_verify_attn     block-causal GQA attention of the d+1 verified
 *                          positions against the target KV cache (Sec. 3.1:
 *                          the target scores all drafted positions in one
 *                          forward pass).
 *   oracle_accept          verification: greedy argmax match, or the
 *                          standard rejection rule of speculative sampling
 *                          (Sec. 3.1, which cites Leviathan et al.; lossless
 *                          with respect to the target distribution) with a
 *                          residual / bonus draw by an exponential race.
 *   oracle_philox4x32_10   counter-based generator of Salmon, Moraes, Dror
 *                          and Shaw, "Parallel random numbers: as easy as
 *                          1, 2, 3" (SC'11), written from that definition.
 *
 * Readings of points the paper leaves open are stated where they are used.
 * Floating point: every reduction is a plain left-to-right loop in double;
 * the file is compiled with -ffp-contract=off so no multiply-add is fused.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define ORACLE_OK 0
#define ORACLE_EINVAL (-1)

/* Relative distance below which a comparison that decides an integer is
 * reported as "near the threshold" (flagged): 1e-6, as the contract states. */
static const double FLAG_REL = 1e-6;

/* ------------------------------------------------------------------ */
/* threads                                                             */
/* ------------------------------------------------------------------ */
static int g_threads = 1;

void oracle_set_threads(int n) {
  g_threads = n < 1 ? 1 : n;
#ifdef _OPENMP
  omp_set_num_threads(g_threads);
#endif
}

int oracle_get_threads(void) {
#ifdef _OPENMP
  return g_threads;
#else
  return 1;
#endif
}

int oracle_has_openmp(void) {
#ifdef _OPENMP
  return 1;
#else
  return 0;
#endif
}

/* ------------------------------------------------------------------ */
/* Philox4x32-10 (Salmon et al., SC'11).                               */
/* One round maps (X0,X1,X2,X3) with key (k0,k1) to                    */
/*   (hi(M1*X2) ^ X1 ^ k0,  lo(M1*X2),  hi(M0*X0) ^ X3 ^ k1,  lo(M0*X0)) */
/* and the key is bumped by the Weyl constants (W0,W1) between rounds. */
/* ------------------------------------------------------------------ */
static const uint32_t PHILOX_M0 = 0xD2511F53u;
static const uint32_t PHILOX_M1 = 0xCD9E8D57u;
static const uint32_t PHILOX_W0 = 0x9E3779B9u;
static const uint32_t PHILOX_W1 = 0xBB67AE85u;

void oracle_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]) {
  uint32_t x0 = ctr[0], x1 = ctr[1], x2 = ctr[2], x3 = ctr[3];
  uint32_t k0 = key[0], k1 = key[1];
  for (int round = 0; round < 10; ++round) {
    if (round > 0) {
      k0 += PHILOX_W0;
      k1 += PHILOX_W1;
    }
    uint64_t p0 = (uint64_t)PHILOX_M0 * (uint64_t)x0;
    uint64_t p1 = (uint64_t)PHILOX_M1 * (uint64_t)x2;
    uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
    uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
    uint32_t y0 = hi1 ^ x1 ^ k0;
    uint32_t y1 = lo1;
    uint32_t y2 = hi0 ^ x3 ^ k1;
    uint32_t y3 = lo0;
    x0 = y0; x1 = y1; x2 = y2; x3 = y3;
  }
  out[0] = x0; out[1] = x1; out[2] = x2; out[3] = x3;
}

/* The stream layout used for every uniform of the verify round:
 *   key     = (seed low 32 bits, seed high 32 bits)
 *   counter = (idx, position j, global sequence index, purpose + 4*round)
 * purpose 0: accept test of draft position j (idx 0, word 0)
 * purpose 1: residual / bonus race over the vocabulary (idx = v >> 2,
 *            word v & 3) at the position where the draw happens
 * A 32-bit word w becomes u = ((w >> 9) + 1/2) * 2^-23, which lies strictly
 * inside (0,1) and is exact in binary32 and binary64. */
double oracle_uniform(uint64_t seed, uint32_t idx, uint32_t j, uint32_t seq,
                      uint32_t purpose, uint64_t round_offset, int word) {
  uint32_t ctr[4] = {idx, j, seq, purpose + 4u * (uint32_t)round_offset};
  uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
  uint32_t out[4];
  oracle_philox4x32_10(ctr, key, out);
  uint32_t w = out[word & 3];
  return ((double)(w >> 9) + 0.5) * (1.0 / 8388608.0);
}

static double bf16_to_double(uint16_t h) {
  uint32_t bits = ((uint32_t)h) << 16;
  float f;
  memcpy(&f, &bits, sizeof f);
  return (double)f;
}

/* Softmax statistics of one logit row at temperature T:
 * m = max_v x_v and Z = sum_v exp((x_v - m)/T), so that
 * softmax_T(x)_v = exp((x_v - m)/T) / Z. The maximum is subtracted before
 * dividing by T (a reading: the paper does not fix the form; this keeps the
 * largest terms exact). */
static void row_softmax_stats(const float* x, int V, double T, double* m_out, double* Z_out) {
  double m = (double)x[0];
  for (int v = 1; v < V; ++v)
    if ((double)x[v] > m) m = (double)x[v];
  double Z = 0.0;
  for (int v = 0; v < V; ++v) Z += exp(((double)x[v] - m) / T);
  *m_out = m;
  *Z_out = Z;
}

static int row_argmax(const float* x, int V) {
  int best = 0;
  for (int v = 1; v < V; ++v)
    if (x[v] > x[best]) best = v; /* strict: the lowest index wins ties */
  return best;
}

static int all_finite(const float* x, size_t n) {
  for (size_t i = 0; i < n; ++i)
    if (!isfinite(x[i])) return 0;
  return 1;
}

/* ------------------------------------------------------------------ */
/* Confidence (Assumption 1; Algorithm 1's q_k).                       */
/* Reading: the confidence of draft position k is the drafter's softmax */
/* probability of the token it drafted there. Greedy sequences          */
/* (temperature 0) use the drafter's native distribution (T = 1);       */
/* sampling sequences use the sampling temperature, the same q that the */
/* rejection test divides by.                                           */
/* conf[b,k] = q, dstat[b,k] = (m, Z) of the drafter row.               */
/* ------------------------------------------------------------------ */
int oracle_confidence(const float* draft_logits, const int32_t* draft_tokens,
                      const float* temperature, int B, int K, int V,
                      double* conf, double* dstat) {
  if (B < 0 || K < 0 || V < 1 || !draft_logits || !draft_tokens || !temperature || !conf)
    return ORACLE_EINVAL;
  for (int i = 0; i < B * K; ++i)
    if (draft_tokens[i] < 0 || draft_tokens[i] >= V) return ORACLE_EINVAL;
  for (int b = 0; b < B; ++b)
    if (!(temperature[b] >= 0.0f) || !isfinite(temperature[b])) return ORACLE_EINVAL;
  if (!all_finite(draft_logits, (size_t)B * K * V)) return ORACLE_EINVAL;
#pragma omp parallel for schedule(dynamic, 1)
  for (int r = 0; r < B * K; ++r) {
    int b = r / K;
    double T = temperature[b] > 0.0f ? (double)temperature[b] : 1.0;
    const float* x = draft_logits + (size_t)r * V;
    double m, Z;
    row_softmax_stats(x, V, T, &m, &Z);
    conf[r] = exp(((double)x[draft_tokens[r]] - m) / T) / Z;
    if (dstat) {
      dstat[2 * r] = m;
      dstat[2 * r + 1] = Z;
    }
  }
  return ORACLE_OK;
}

/* ------------------------------------------------------------------ */
/* Selector (Thm. 4 criterion scanned from L = 0; Thm. 5).             */
/*                                                                     */
/* P_L = prod_{k=1}^{L} q_k (prefix acceptance, proof of Thm. 2);      */
/* E_L = e0 + sum_{j=1}^{L} P_j is the expected number of tokens one    */
/* verification of L drafts yields. Reading: e0 = 1 counts the token   */
/* verification always emits (correction or bonus), so T(0) describes  */
/* plain autoregressive decoding with speedup 1; e0 = 0 is the          */
/* alternative reading, kept for tests.                                 */
/* Extending L -> L+1 adds P_{L+1} tokens for c_L = T(L+1) - T(L) time; */
/* by Thm. 1 (the mediant / ratio comparison) it raises E/T iff        */
/* P_{L+1} * T(L) > c_L * E_L (Thm. 4's cross-multiplied form; exact   */
/* for any sign of c_L as long as T(L), T(L+1) > 0). The scan stops at  */
/* the first L where the test fails, or at K. The comparison is strict */
/* (Def. 1), so a tie does not extend.                                 */
/* A sequence is flagged when any comparison the scan made lies within */
/* a relative 1e-6 of its threshold.                                    */
/* ------------------------------------------------------------------ */
int oracle_select_lengths(const double* conf, const double* cost_table, int B, int K,
                          double e0, int32_t* L_out, int32_t* flag_out) {
  if (B < 0 || K < 0 || !conf || !cost_table || !L_out) return ORACLE_EINVAL;
  for (int l = 0; l <= K; ++l)
    if (!(cost_table[l] > 0.0) || !isfinite(cost_table[l])) return ORACLE_EINVAL;
  for (int b = 0; b < B; ++b) {
    const double* q = conf + (size_t)b * K;
    double P = 1.0, E = e0;
    int L = 0, flag = 0;
    while (L < K) {
      P = P * q[L];
      double c = cost_table[L + 1] - cost_table[L];
      double lhs = P * cost_table[L];
      double rhs = E * c;
      double scale = fmax(fabs(lhs), fabs(rhs));
      if (fabs(lhs - rhs) <= FLAG_REL * scale) flag = 1;
      if (!(lhs > rhs)) break;
      E = E + P;
      L = L + 1;
    }
    L_out[b] = L;
    if (flag_out) flag_out[b] = flag;
  }
  return ORACLE_OK;
}

/* Expected speedup up to the constant L_target (Eq. 2 with negligible
 * drafting): eta_L = E_L / T(L). Used by the iteration below. */
static double expected_tokens(const double* q, int L, double e0) {
  double P = 1.0, E = e0;
  for (int j = 0; j < L; ++j) {
    P = P * q[j];
    E = E + P;
  }
  return E;
}

/* Iterated single beneficial adjustments (Def. 1), each one step long,
 * judged by Thm. 1's criterion with the segment quantities written out:
 *   extend d -> d+1   iff E[tau_{d:d+1}] / T_{d:d+1} > E[tau_d] / T_d
 *                     (E[tau_{d:d+1}] = P_{d+1}, T_{d:d+1} = T(d+1) - T(d));
 *   truncate d -> d-1 iff E[tau_{d-1:d}] / T_{d-1:d} < E[tau_d] / T_d
 *                     (E[tau_{d-1:d}] = P_d,     T_{d-1:d} = T(d) - T(d-1));
 *   otherwise stop.
 * Thm. 1's ratio comparison needs positive segment costs, so the cost
 * table must be strictly increasing here. Writes the visited lengths into
 * path[0..] (path[0] = start) and returns how many it wrote (<= cap).
 * Thm. 5 states the walk ends at argmax_d E[eta_d]. */
int oracle_select_iterate(const double* q, const double* cost_table, int K, double e0,
                          int start, int32_t* path, int cap) {
  if (start < 0 || start > K || cap < 1 || !q || !cost_table || !path) return ORACLE_EINVAL;
  for (int l = 0; l <= K; ++l)
    if (!(cost_table[l] > 0.0)) return ORACLE_EINVAL;
  for (int l = 0; l < K; ++l)
    if (!(cost_table[l + 1] > cost_table[l])) return ORACLE_EINVAL;
  int d = start, n = 0;
  path[n++] = d;
  while (n < cap) {
    double Ed = expected_tokens(q, d, e0);
    double avg = Ed / cost_table[d];
    int next = d;
    if (d < K) {
      double seg_gain = expected_tokens(q, d + 1, e0) - Ed;
      double seg_cost = cost_table[d + 1] - cost_table[d];
      if (seg_gain / seg_cost > avg) next = d + 1;
    }
    if (next == d && d > 0) {
      double seg_gain = Ed - expected_tokens(q, d - 1, e0);
      double seg_cost = cost_table[d] - cost_table[d - 1];
      if (seg_gain / seg_cost < avg) next = d - 1;
    }
    if (next == d) break;
    d = next;
    path[n++] = d;
  }
  return n;
}

/* ------------------------------------------------------------------ */
/* Alpha-mode length search (Algorithm 1, Sec. 3.3; Thm. 2 and Thm. 3 */
/* give the position-wise bounds it evaluates, alpha = 2.0 / 2.2 in    */
/* Sec. 4).                                                            */
/*                                                                     */
/* With q_k the drafter confidence of position k (1-based, q_k =       */
/* conf[b, k-1]) and the current length d:                              */
/*   eps_i = floor(alpha * sum_{j=i}^{d} prod_{k=i}^{j} q_k + i),       */
/*           i = 1 .. d,   eps* = min_i eps_i.                          */
/* Starting from one drafted block, d = n, budget B = 0, while          */
/* d < d_max: if eps* <= d, d = eps* and stop (the single rollback);    */
/* otherwise B -= eps* - d, d = eps*, and when B < 0 ceil(-B/n) more    */
/* blocks are drafted and B += ceil(-B/n) * n. d tokens are verified.  */
/* Readings of points the algorithm leaves open:                        */
/*  * the floor form of Algorithm 1 is used as printed (the theorems'   */
/*    strict "<" bound would give ceil(x) - 1; the two differ only when */
/*    alpha*S_i + i is an integer, which is flagged);                  */
/*  * the sum runs to the current d, as in Algorithm 1;                 */
/*  * eps* above d_max is clamped to d_max (the loop then ends);        */
/*  * the first block holds n <= d_max positions (1 <= n <= d_max);     */
/*  * q_k of every position up to d_max is given: the search only ever  */
/*    reads q_1 .. q_d of the current d, so this matches drafting the   */
/*    blocks on demand; blocks_out counts the blocks drafted.          */
/* The sums are written out as the definition reads (a fresh product   */
/* for every j). A sequence is flagged when some alpha*S_i + i lies     */
/* within a relative 1e-6 of an integer (there floor is ambiguous      */
/* between binary64 evaluations in different orders).                  */
/* ------------------------------------------------------------------ */
int oracle_select_alpha(const double* conf, int B, int K, int n, double alpha, int32_t* L_out,
                        int32_t* blocks_out, int32_t* flag_out) {
  if (B < 0 || K < 1 || n < 1 || n > K || !conf || !L_out || !(alpha > 0.0) || !isfinite(alpha))
    return ORACLE_EINVAL;
  for (int b = 0; b < B; ++b) {
    const double* q = conf + (size_t)b * K; /* q_k = q[k - 1] */
    int d = n, blocks = 1, flag = 0;
    long budget = 0;
    while (d < K) {
      long eps_star = 0;
      for (int i = 1; i <= d; ++i) {
        double S = 0.0;
        for (int j = i; j <= d; ++j) {
          double P = 1.0;
          for (int k = i; k <= j; ++k) P = P * q[k - 1];
          S = S + P;
        }
        const double x = alpha * S + (double)i;
        const double fl = floor(x);
        if (fabs(x - nearbyint(x)) <= FLAG_REL * fmax(1.0, fabs(x))) flag = 1;
        const long eps_i = (long)fl;
        if (i == 1 || eps_i < eps_star) eps_star = eps_i;
      }
      if (eps_star <= d) {
        d = (int)eps_star; /* the single rollback */
        break;
      }
      if (eps_star > K) eps_star = K;
      budget -= eps_star - d;
      d = (int)eps_star;
      if (budget < 0) {
        const long more = (-budget + n - 1) / n;
        blocks += (int)more;
        budget += more * n;
      }
    }
    L_out[b] = d;
    if (blocks_out) blocks_out[b] = blocks;
    if (flag_out) flag_out[b] = flag;
  }
  return ORACLE_OK;
}

/* ------------------------------------------------------------------ */
/* Paged KV cache: the dense cache a block table describes.            */
/* Reading (the paper does not address memory layout): key s of        */
/* sequence b is row s % page_size of page block_table[b * max_pages + */
/* s / page_size] of a pool [n_pages, Hkv, page_size, dh]; the verify  */
/* attention over a paged cache is the dense one on                    */
/*   dense[b, h, s, :] = pool[block_table[b][s / P], h, s % P, :],      */
/* s < S_out <= max_pages * P. An entry outside [0, n_pages) that some  */
/* s < S_out needs is an error.                                        */
/* ------------------------------------------------------------------ */
int oracle_gather_pages(const uint16_t* pool, const int32_t* block_table, int B, int max_pages, int page_size,
                        int n_pages, int Hkv, int dh, int S_out, uint16_t* dense) {
  if (B < 0 || max_pages < 1 || page_size < 1 || n_pages < 1 || Hkv < 1 || dh < 1 || S_out < 0 ||
      (long)S_out > (long)max_pages * page_size || !pool || !block_table || !dense)
    return ORACLE_EINVAL;
  for (int b = 0; b < B; ++b)
    for (int s = 0; s < S_out; ++s) {
      const int page = block_table[(size_t)b * max_pages + s / page_size];
      if (page < 0 || page >= n_pages) return ORACLE_EINVAL;
      for (int h = 0; h < Hkv; ++h) {
        const uint16_t* src = pool + (((size_t)page * Hkv + h) * page_size + s % page_size) * dh;
        uint16_t* dst = dense + (((size_t)b * Hkv + h) * S_out + s) * dh;
        for (int c = 0; c < dh; ++c) dst[c] = src[c];
      }
    }
  return ORACLE_OK;
}

/* ------------------------------------------------------------------ */
/* Verify attention (Sec. 3.1: one target forward pass scores the d+1 */
/* verified positions).                                                */
/* Readings (the paper does not write the layer out): scale 1/sqrt(d)  */
/* is passed in; Q and K are already position-encoded; grouped-query   */
/* heads map query head h to kv head floor(h / g), g = Hq / Hkv; the    */
/* block's own L_b + 1 keys are in the cache at kv_len_b .. kv_len_b +  */
/* L_b; block row t sees keys 0 .. kv_len_b + t (a causal chain draft); */
/* rows t > L_b are not computed (left as the caller filled them).     */
/* Layouts: Q, O [B, K+1, Hq, dh]; Kc, Vc [B, Hkv, S_cap, dh] (bf16    */
/* bit patterns); lse [B, K+1, Hq] natural log.                        */
/* If rows != NULL only the n_rows listed triples (b, h, t) are done.  */
/* ------------------------------------------------------------------ */
/* One query row over the visible keys keys[0..n_keys) (ascending), as
 * verify attention computes it: scores, max, exponentials, weighted sum. */
static void attn_row(const double* qv, const uint16_t* Kh, const uint16_t* Vh, int dh, double scale,
                     const int* keys, int n_keys, double* s, double* acc, double* out, double* lse_out) {
  double m = -INFINITY;
  for (int jj = 0; jj < n_keys; ++jj) {
    const int j = keys[jj];
    double dot = 0.0;
    for (int i = 0; i < dh; ++i) dot += qv[i] * bf16_to_double(Kh[(size_t)j * dh + i]);
    s[jj] = dot * scale;
    if (s[jj] > m) m = s[jj];
  }
  double l = 0.0;
  for (int i = 0; i < dh; ++i) acc[i] = 0.0;
  for (int jj = 0; jj < n_keys; ++jj) {
    const int j = keys[jj];
    double w = exp(s[jj] - m);
    l += w;
    for (int i = 0; i < dh; ++i) acc[i] += w * bf16_to_double(Vh[(size_t)j * dh + i]);
  }
  for (int i = 0; i < dh; ++i) out[i] = acc[i] / l;
  if (lse_out) *lse_out = m + log(l);
}

/* parent == NULL: the chain draft (row t sees keys 0 .. kv_len_b + t).
 * Otherwise a draft tree: node t in [0, L_b] has parent[b * (K+1) + t] in
 * [0, t) (node 0, the last accepted token, is the root), its keys sit at
 * kv_len_b + t, and node t sees the cache prefix and the keys of its
 * ancestors and itself. A chain tree (parent t-1) is the chain draft. */
static int verify_attn_impl(const uint16_t* Q, const uint16_t* Kc, const uint16_t* Vc,
                            const int32_t* kv_len, const int32_t* L, const int32_t* parent, int B, int K,
                            int Hq, int Hkv, int dh, int S_cap, double scale, double* O, double* lse,
                            const int32_t* rows, int n_rows) {
  if (B < 0 || K < 0 || Hq < 1 || Hkv < 1 || Hq % Hkv != 0 || dh < 1 || S_cap < 1) return ORACLE_EINVAL;
  for (int b = 0; b < B; ++b)
    if (L[b] < 0 || L[b] > K || kv_len[b] < 0 || (long)kv_len[b] + L[b] + 1 > S_cap) return ORACLE_EINVAL;
  if (parent)
    for (int b = 0; b < B; ++b)
      for (int t = 1; t <= L[b]; ++t) {
        const int p = parent[(size_t)b * (K + 1) + t];
        if (p < 0 || p >= t) return ORACLE_EINVAL;
      }
  const int g = Hq / Hkv;
  long total = rows ? n_rows : (long)B * Hq * (K + 1);
#pragma omp parallel
  {
    double* s = (double*)malloc(sizeof(double) * (size_t)S_cap);
    double* qv = (double*)malloc(sizeof(double) * (size_t)dh);
    double* acc = (double*)malloc(sizeof(double) * (size_t)dh);
    int* keys = (int*)malloc(sizeof(int) * (size_t)S_cap);
    char* anc = (char*)malloc((size_t)K + 1);
#pragma omp for schedule(dynamic, 1)
    for (long it = 0; it < total; ++it) {
      int b, h, t;
      if (rows) {
        b = rows[3 * it]; h = rows[3 * it + 1]; t = rows[3 * it + 2];
      } else {
        b = (int)(it / ((long)Hq * (K + 1)));
        int rem = (int)(it % ((long)Hq * (K + 1)));
        t = rem / Hq; h = rem % Hq;
      }
      if (b < 0 || b >= B || h < 0 || h >= Hq || t < 0 || t > L[b]) continue;
      int kvh = h / g;
      size_t qoff = (((size_t)b * (K + 1) + t) * Hq + h) * dh;
      for (int i = 0; i < dh; ++i) qv[i] = bf16_to_double(Q[qoff + i]);
      const uint16_t* Kh = Kc + ((size_t)b * Hkv + kvh) * (size_t)S_cap * dh;
      const uint16_t* Vh = Vc + ((size_t)b * Hkv + kvh) * (size_t)S_cap * dh;
      int n_keys = 0;
      for (int j = 0; j < kv_len[b]; ++j) keys[n_keys++] = j;
      if (!parent) {
        for (int a = 0; a <= t; ++a) keys[n_keys++] = kv_len[b] + a;
      } else {
        for (int a = 0; a <= t; ++a) anc[a] = 0;
        for (int a = t; a > 0; a = parent[(size_t)b * (K + 1) + a]) anc[a] = 1;
        anc[0] = 1;
        for (int a = 0; a <= t; ++a)
          if (anc[a]) keys[n_keys++] = kv_len[b] + a;
      }
      attn_row(qv, Kh, Vh, dh, scale, keys, n_keys, s, acc, O + qoff,
               lse ? lse + ((size_t)b * (K + 1) + t) * Hq + h : NULL);
    }
    free(s); free(qv); free(acc); free(keys); free(anc);
  }
  return ORACLE_OK;
}

int oracle_verify_attn(const uint16_t* Q, const uint16_t* Kc, const uint16_t* Vc,
                       const int32_t* kv_len, const int32_t* L, int B, int K, int Hq, int Hkv,
                       int dh, int S_cap, double scale, double* O, double* lse,
                       const int32_t* rows, int n_rows) {
  return verify_attn_impl(Q, Kc, Vc, kv_len, L, NULL, B, K, Hq, Hkv, dh, S_cap, scale, O, lse, rows, n_rows);
}

/* Verify attention of a draft tree (tree verification as in the tree
 * drafters the paper builds on, Sec. 2): parent [B, K+1], see above. */
int oracle_verify_attn_tree(const uint16_t* Q, const uint16_t* Kc, const uint16_t* Vc,
                            const int32_t* kv_len, const int32_t* L, const int32_t* parent, int B, int K,
                            int Hq, int Hkv, int dh, int S_cap, double scale, double* O, double* lse,
                            const int32_t* rows, int n_rows) {
  if (!parent) return ORACLE_EINVAL;
  return verify_attn_impl(Q, Kc, Vc, kv_len, L, parent, B, K, Hq, Hkv, dh, S_cap, scale, O, lse, rows, n_rows);
}

/* Greedy acceptance of a draft tree: from the root (node 0), follow the
 * lowest-numbered child whose token is the target's argmax at the current
 * node (lowest index on ties) while there is one; n = nodes accepted
 * below the root, last = the final node, bonus = the argmax there. Node
 * t >= 1 carries draft token tokens[b * K + t - 1] (the chain layout). A
 * chain tree gives the chain's greedy acceptance. */
int oracle_accept_tree_greedy(const float* target, const int32_t* tokens, const int32_t* parent,
                              const int32_t* L, int B, int K, int V, int32_t* n_accepted, int32_t* last_node,
                              int32_t* bonus) {
  if (B < 0 || K < 0 || V < 1 || !target || !tokens || !parent || !L || !n_accepted || !bonus) return ORACLE_EINVAL;
  for (int b = 0; b < B; ++b) {
    if (L[b] < 0 || L[b] > K) return ORACLE_EINVAL;
    for (int t = 1; t <= L[b]; ++t) {
      const int p = parent[(size_t)b * (K + 1) + t];
      if (p < 0 || p >= t) return ORACLE_EINVAL;
      if (tokens[(size_t)b * K + t - 1] < 0 || tokens[(size_t)b * K + t - 1] >= V) return ORACLE_EINVAL;
    }
    int cur = 0, n = 0, arg = 0;
    for (;;) {
      arg = row_argmax(target + ((size_t)b * (K + 1) + cur) * V, V);
      int next = -1;
      for (int c = cur + 1; c <= L[b]; ++c)
        if (parent[(size_t)b * (K + 1) + c] == cur && tokens[(size_t)b * K + c - 1] == arg) {
          next = c;
          break;
        }
      if (next < 0) break;
      cur = next;
      ++n;
    }
    n_accepted[b] = n;
    if (last_node) last_node[b] = cur;
    bonus[b] = arg;
  }
  return ORACLE_OK;
}

/* Acceptance of a draft tree at temperature[b] (the greedy walk above when
 * it is 0). At the current node the walk draws the target's token x from
 * softmax(row / T) and moves to the lowest-numbered child carrying x while
 * there is one; the round emits the walked nodes' tokens and then the last
 * draw (bonus). Every emitted token is a draw from the target given the
 * prefix it extends, so the output follows the target's distribution; a
 * child is accepted with the target's probability of its token. Draw at
 * node t: the race x = argmin_v key_v, key_v = log2(E_v) - y_v log2(e) / T,
 * E_v = -ln u_v, u_v the Philox uniform of (v >> 2, position t, sequence
 * seq_offset + b, purpose 2), word v & 3 (the exponential race in log2
 * units; lowest index on equal keys). flag[b] = 1 when at a visited node
 * the two smallest keys lie within 4e-5 + 1e-6 |y_v log2(e) / T| of each
 * other (the fp32 keys of a GPU could order them differently). */
static const uint32_t TREE_PURPOSE = 2u;

static int tree_draw(const float* row, int V, double T, uint64_t seed, uint32_t t, uint32_t seq,
                     uint64_t round_offset, int* flag) {
  const double c = 1.4426950408889634 / T;
  double best = INFINITY, second = INFINITY, yc_best = 0.0, yc_second = 0.0;
  int arg = 0;
  for (int v = 0; v < V; ++v) {
    const double yc = (double)row[v] * c;
    if (!(yc > -INFINITY)) continue;
    const double u = oracle_uniform(seed, (uint32_t)(v >> 2), t, seq, TREE_PURPOSE, round_offset, v & 3);
    const double key = log2(-log(u)) - yc;
    if (key < best) {
      second = best; yc_second = yc_best;
      best = key; yc_best = yc; arg = v;
    } else if (key < second) {
      second = key; yc_second = yc;
    }
  }
  if (second < INFINITY && second - best <= 4e-5 + 1e-6 * fmax(fabs(yc_best), fabs(yc_second))) *flag = 1;
  return arg;
}

int oracle_accept_tree(const float* target, const int32_t* tokens, const int32_t* parent, const int32_t* L,
                       const float* temperature, int B, int K, int V, uint64_t seed, uint64_t round_offset,
                       uint32_t seq_offset, int32_t* n_accepted, int32_t* last_node, int32_t* bonus,
                       int32_t* flag_out) {
  if (B < 0 || K < 0 || V < 1 || !target || !tokens || !parent || !L || !temperature || !n_accepted || !bonus)
    return ORACLE_EINVAL;
  for (int b = 0; b < B; ++b) {
    if (L[b] < 0 || L[b] > K) return ORACLE_EINVAL;
    if (!(temperature[b] >= 0.0f) || !isfinite(temperature[b])) return ORACLE_EINVAL;
    for (int t = 1; t <= L[b]; ++t) {
      const int p = parent[(size_t)b * (K + 1) + t];
      if (p < 0 || p >= t) return ORACLE_EINVAL;
      if (tokens[(size_t)b * K + t - 1] < 0 || tokens[(size_t)b * K + t - 1] >= V) return ORACLE_EINVAL;
    }
  }
#pragma omp parallel for schedule(dynamic, 1)
  for (int b = 0; b < B; ++b) {
    const double T = (double)temperature[b];
    const uint32_t seq = seq_offset + (uint32_t)b;
    int cur = 0, n = 0, x = 0, flag = 0;
    for (;;) {
      const float* row = target + ((size_t)b * (K + 1) + cur) * V;
      x = T == 0.0 ? row_argmax(row, V) : tree_draw(row, V, T, seed, (uint32_t)cur, seq, round_offset, &flag);
      int next = -1;
      for (int c = cur + 1; c <= L[b]; ++c)
        if (parent[(size_t)b * (K + 1) + c] == cur && tokens[(size_t)b * K + c - 1] == x) {
          next = c;
          break;
        }
      if (next < 0) break;
      cur = next;
      ++n;
    }
    n_accepted[b] = n;
    if (last_node) last_node[b] = cur;
    bonus[b] = x;
    if (flag_out) flag_out[b] = flag;
  }
  return ORACLE_OK;
}

/* ------------------------------------------------------------------ */
/* Exponential race: among the weights w_v >= 0 of a distribution,     */
/* argmin_v E_v / w_v with E_v = -ln u_v i.i.d. Exp(1) draws picks v   */
/* with probability w_v / sum w (the "exponential clocks" form of the  */
/* Gumbel-max identity). Ties go to the lower index.                   */
/* The race is flagged when some other candidate's key lies within the */
/* combined relative uncertainty of the winner's: each key carries a    */
/* relative uncertainty rel_v (1e-6, widened where w_v was obtained by */
/* cancellation).                                                      */
/* ------------------------------------------------------------------ */
typedef struct {
  int winner;
  int flag;
} race_result;

static race_result exp_race(const double* w, const double* rel, int V, uint64_t seed,
                            uint32_t j, uint32_t seq, uint64_t round_offset, double* keybuf) {
  race_result res = {-1, 0};
  double best = INFINITY;
  for (int v = 0; v < V; ++v) {
    keybuf[v] = INFINITY;
    if (!(w[v] > 0.0)) continue;
    double u = oracle_uniform(seed, (uint32_t)(v >> 2), j, seq, 1u, round_offset, v & 3);
    double E = -log(u);
    keybuf[v] = E / w[v];
    if (keybuf[v] < best) {
      best = keybuf[v];
      res.winner = v;
    }
  }
  if (res.winner < 0) return res;
  double hi = best * (1.0 + rel[res.winner]);
  for (int v = 0; v < V; ++v) {
    if (v == res.winner || !(keybuf[v] < INFINITY)) continue;
    if (keybuf[v] * (1.0 - rel[v]) <= hi) {
      res.flag = 1;
      break;
    }
  }
  return res;
}

/* ------------------------------------------------------------------ */
/* Row statistics straight from an LM head (the confidence of Assumption */
/* 1 and the acceptance row statistics of Sec. 3.1, with the logits     */
/* x[r, v] = sum_k H[r, k] W[v, k] never stored): H [M, Dm] and W [V, Dm]  */
/* bf16 bit patterns; T_r = temperature[r / rows_per_seq] (1 when 0 or   */
/* when temperature is NULL). Per row: max m, lowest-index argmax, Z =   */
/* sum_v exp((x_v - m) / T_r), and for token[r] >= 0 the probability     */
/* exp((x_tok - m) / T_r) / Z. Logits are sums of exact bf16 products in */
/* binary64. flag[r] = 1 when the two largest logits lie within          */
/* 2^-16 (a_1 + a_2), a_v = sum_k |H[r,k] W[v,k]|: a binary32            */
/* accumulation may order them differently.                              */
/* ------------------------------------------------------------------ */
int oracle_lm_head_stats(const uint16_t* H, const uint16_t* W, const float* temperature, int rows_per_seq,
                         const int32_t* token, int M, int V, int Dm, double* row_max, double* row_Z,
                         int32_t* row_arg, double* token_prob, int32_t* flag) {
  if (M < 0 || V < 1 || Dm < 1 || !H || !W || rows_per_seq < 1) return ORACLE_EINVAL;
  for (int r = 0; r < M; ++r)
    if (token && token[r] >= V) return ORACLE_EINVAL;
#pragma omp parallel
  {
    double* x = (double*)malloc(sizeof(double) * (size_t)V);
    double* a = (double*)malloc(sizeof(double) * (size_t)V);
    double* h = (double*)malloc(sizeof(double) * (size_t)Dm);
#pragma omp for schedule(dynamic, 1)
    for (int r = 0; r < M; ++r) {
      for (int k = 0; k < Dm; ++k) h[k] = bf16_to_double(H[(size_t)r * Dm + k]);
      for (int v = 0; v < V; ++v) {
        double s = 0.0, sa = 0.0;
        const uint16_t* w = W + (size_t)v * Dm;
        for (int k = 0; k < Dm; ++k) {
          const double p = h[k] * bf16_to_double(w[k]);
          s += p;
          sa += fabs(p);
        }
        x[v] = s;
        a[v] = sa;
      }
      double T = temperature ? (double)temperature[r / rows_per_seq] : 1.0;
      if (!(T > 0.0)) T = 1.0;
      int arg = 0, second = -1;
      for (int v = 1; v < V; ++v) {
        if (x[v] > x[arg]) { second = arg; arg = v; }
        else if (second < 0 || x[v] > x[second]) second = v;
      }
      const double m = x[arg];
      double Z = 0.0;
      for (int v = 0; v < V; ++v) Z += exp((x[v] - m) / T);
      if (row_max) row_max[r] = m;
      if (row_Z) row_Z[r] = Z;
      if (row_arg) row_arg[r] = arg;
      if (token_prob) token_prob[r] = (token && token[r] >= 0) ? exp((x[token[r]] - m) / T) / Z : 0.0;
      if (flag) flag[r] = (second >= 0 && x[arg] - x[second] <= ldexp(a[arg] + a[second], -16)) ? 1 : 0;
    }
    free(x); free(a); free(h);
  }
  return ORACLE_OK;
}

/* ------------------------------------------------------------------ */
/* Acceptance (Sec. 3.1; the rule of Leviathan et al. the paper cites). */
/*                                                                     */
/* Row j of target_logits [B, K+1, V] is the target's distribution for  */
/* draft position j (row L_b is the bonus row). draft_logits [B, K, V], */
/* draft_tokens [B, K].                                                 */
/*                                                                     */
/* temperature[b] == 0 (greedy): accept x_j while argmax p_j = x_j     */
/*   (lowest index on ties); n = first mismatch or L_b; the emitted    */
/*   token is argmax p_n.                                              */
/* temperature[b] > 0 (sampling): p, q = softmax at that temperature.  */
/*   For j < L_b draw u_j (purpose 0) and accept iff u_j < min(1,      */
/*   p_j(x_j)/q_j(x_j)) (q <= p accepts outright). At the first          */
/*   rejection r draw the token from norm(max(0, p_r - q_r)); if all    */
/*   L_b are accepted draw it from p_{L_b}. Both draws are exponential  */
/*   races over purpose-1 uniforms at position r (resp. L_b). If the    */
/*   residual is identically zero (p_r == q_r) the draw falls back to   */
/*   p_r and the sequence is flagged.                                   */
/* Outputs n_accepted[b] = number of accepted drafts, bonus_token[b] =  */
/* the token emitted after them; flag[b] = 1 when an accept test or the */
/* race lies within the flag tolerance. rejected_at[b] (optional) =    */
/* r or L_b.                                                            */
/* seq_offset is added to b to form the global sequence index used in   */
/* the generator counters (a batch split over several workers draws the */
/* same numbers as the unsplit batch).                                 */
/* ------------------------------------------------------------------ */
int oracle_accept(const float* target_logits, const float* draft_logits, const int32_t* draft_tokens,
                  const int32_t* L, const float* temperature, int B, int K, int V,
                  uint64_t seed, uint64_t round_offset, uint32_t seq_offset,
                  int32_t* n_accepted, int32_t* bonus_token, int32_t* flag_out) {
  if (B < 0 || K < 0 || V < 1 || !target_logits || !draft_logits || !draft_tokens || !L ||
      !temperature || !n_accepted || !bonus_token)
    return ORACLE_EINVAL;
  for (int b = 0; b < B; ++b) {
    if (L[b] < 0 || L[b] > K) return ORACLE_EINVAL;
    if (!(temperature[b] >= 0.0f) || !isfinite(temperature[b])) return ORACLE_EINVAL;
    for (int j = 0; j < L[b]; ++j)
      if (draft_tokens[(size_t)b * K + j] < 0 || draft_tokens[(size_t)b * K + j] >= V) return ORACLE_EINVAL;
  }
  int status = ORACLE_OK;
#pragma omp parallel
  {
    double* w = (double*)malloc(sizeof(double) * (size_t)V);
    double* rel = (double*)malloc(sizeof(double) * (size_t)V);
    double* keys = (double*)malloc(sizeof(double) * (size_t)V);
#pragma omp for schedule(dynamic, 1)
    for (int b = 0; b < B; ++b) {
      const float* tb = target_logits + (size_t)b * (K + 1) * V;
      const float* db = draft_logits + (size_t)b * K * V;
      const int32_t* xb = draft_tokens + (size_t)b * K;
      uint32_t seq = seq_offset + (uint32_t)b;
      int Lb = L[b], flag = 0;
      if (temperature[b] == 0.0f) {
        int n = Lb, emit = -1;
        for (int j = 0; j < Lb; ++j) {
          int a = row_argmax(tb + (size_t)j * V, V);
          if (a != xb[j]) { n = j; emit = a; break; }
        }
        if (emit < 0) emit = row_argmax(tb + (size_t)Lb * V, V);
        n_accepted[b] = n;
        bonus_token[b] = emit;
      } else {
        double T = (double)temperature[b];
        int r = Lb;
        for (int j = 0; j < Lb; ++j) {
          double mp, Zp, mq, Zq;
          row_softmax_stats(tb + (size_t)j * V, V, T, &mp, &Zp);
          row_softmax_stats(db + (size_t)j * V, V, T, &mq, &Zq);
          int x = xb[j];
          double p = exp(((double)tb[(size_t)j * V + x] - mp) / T) / Zp;
          double q = exp(((double)db[(size_t)j * V + x] - mq) / T) / Zq;
          double ratio = (q <= p) ? 1.0 : p / q;
          double u = oracle_uniform(seed, 0u, (uint32_t)j, seq, 0u, round_offset, 0);
          if (fabs(u - ratio) < FLAG_REL) flag = 1;
          if (!(u < ratio)) { r = j; break; }
        }
        int emit;
        if (r < Lb) {
          /* residual max(0, p_r - q_r); the normaliser does not change the race */
          double mp, Zp, mq, Zq;
          const float* pr = tb + (size_t)r * V;
          const float* qr = db + (size_t)r * V;
          row_softmax_stats(pr, V, T, &mp, &Zp);
          row_softmax_stats(qr, V, T, &mq, &Zq);
          for (int v = 0; v < V; ++v) {
            double p = exp(((double)pr[v] - mp) / T) / Zp;
            double q = exp(((double)qr[v] - mq) / T) / Zq;
            double d = p - q;
            w[v] = d > 0.0 ? d : 0.0;
            rel[v] = d > 0.0 ? FLAG_REL * (1.0 + (p + q) / d) : FLAG_REL;
          }
          race_result rr = exp_race(w, rel, V, seed, (uint32_t)r, seq, round_offset, keys);
          if (rr.winner < 0) {
            for (int v = 0; v < V; ++v) { w[v] = exp(((double)pr[v] - mp) / T); rel[v] = FLAG_REL; }
            rr = exp_race(w, rel, V, seed, (uint32_t)r, seq, round_offset, keys);
            rr.flag = 1;
          }
          emit = rr.winner;
          flag |= rr.flag;
        } else {
          double mp, Zp;
          const float* pr = tb + (size_t)Lb * V;
          row_softmax_stats(pr, V, T, &mp, &Zp);
          for (int v = 0; v < V; ++v) { w[v] = exp(((double)pr[v] - mp) / T); rel[v] = FLAG_REL; }
          race_result rr = exp_race(w, rel, V, seed, (uint32_t)Lb, seq, round_offset, keys);
          emit = rr.winner;
          flag |= rr.flag;
        }
        n_accepted[b] = r;
        bonus_token[b] = emit;
      }
      if (flag_out) flag_out[b] = flag;
    }
    free(w); free(rel); free(keys);
  }
  return status;
}
