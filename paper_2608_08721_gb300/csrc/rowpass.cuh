// One CTA's streaming pass over a slice of a logit row: max / argmax and the
// sum of exponentials, in a single read of HBM with 128-bit loads.
#pragma once

#include "common.cuh"

namespace libraspec {

constexpr int kRowThreads = 256;

// Per-thread running sum of 2^((x - m) * c), c = log2(e) / T, with the max
// tracked online (the sum is rescaled when the max grows) and Kahan
// compensation of the running sum.
struct SumAcc {
  float m, s, comp;
  __device__ __forceinline__ void init() { m = -INFINITY; s = 0.f; comp = 0.f; }
  __device__ __forceinline__ void add4(float4 v, float c) {
    const float gm = fmaxf(fmaxf(v.x, v.y), fmaxf(v.z, v.w));
    if (gm > m) {
      const float f = ex2_approx((m - gm) * c);
      s *= f;
      comp *= f;
      m = gm;
    }
    const float t = (ex2_approx((v.x - m) * c) + ex2_approx((v.y - m) * c)) +
                    (ex2_approx((v.z - m) * c) + ex2_approx((v.w - m) * c));
    const float y = t - comp;
    const float ts = s + y;
    comp = (ts - s) - y;
    s = ts;
  }
  __device__ __forceinline__ void add1(float x, float c) {
    if (x > m) {
      const float f = ex2_approx((m - x) * c);
      s *= f;
      comp *= f;
      m = x;
    }
    const float y = ex2_approx((x - m) * c) - comp;
    const float ts = s + y;
    comp = (ts - s) - y;
    s = ts;
  }
  __device__ __forceinline__ float value() const { return s - comp; }
};

// Per-thread running max with the lowest index among equal maxima
// (elements are visited in increasing index order within a thread).
struct ArgAcc {
  float m;
  int arg;
  __device__ __forceinline__ void init() { m = -INFINITY; arg = 0x7fffffff; }
  __device__ __forceinline__ void add4(float4 v, int i0) {
    if (v.x > m) { m = v.x; arg = i0; }
    if (v.y > m) { m = v.y; arg = i0 + 1; }
    if (v.z > m) { m = v.z; arg = i0 + 2; }
    if (v.w > m) { m = v.w; arg = i0 + 3; }
  }
  __device__ __forceinline__ void add1(float x, int i) {
    if (x > m) { m = x; arg = i; }
  }
};

// Logit `watch` of a group of four starting at index i0, if it lies there.
__device__ __forceinline__ void watch4(float4 f, int i0, int watch, float& watched) {
  const unsigned d = (unsigned)(watch - i0);
  if (d < 4u) watched = d == 0 ? f.x : d == 1 ? f.y : d == 2 ? f.z : f.w;
}

// Stream x[c0, c1) of logits of type T (c0 a multiple of kRowAlign). VEC: x
// is 16-byte aligned and the row length a multiple of the elements one
// 128-bit load holds, so 128-bit loads cover the slice. WATCH: the thread
// that streams logit `watch` also keeps it in `watched` (a drafted token's
// logit, read with the stream instead of by a dependent load).
template <bool SUM, bool ARG, bool VEC, typename T, bool WATCH = false>
__device__ __forceinline__ void row_slice_pass(const T* __restrict__ x, int c0, int c1, float c, SumAcc& sa,
                                               ArgAcc& aa, int watch = -1, float* watched = nullptr) {
  using LT = Logit<T>;
  constexpr int W = LT::kVec;  // elements per 128-bit load
  const int tid = threadIdx.x;
  float wv = 0.f;
  if (VEC) {
    const int g0 = c0 / W, g1 = c1 / W;  // groups of W
    int g = g0 + tid;
    constexpr int U = 16 / W;  // 16 elements in flight per thread
    for (; g + (U - 1) * kRowThreads < g1; g += U * kRowThreads) {
      float v[U][W];
#pragma unroll
      for (int u = 0; u < U; ++u) LT::stream_vec(x + W * (g + u * kRowThreads), v[u]);
#pragma unroll
      for (int u = 0; u < U; ++u)
#pragma unroll
        for (int h = 0; h < W; h += 4) {
          const float4 f = make_float4(v[u][h], v[u][h + 1], v[u][h + 2], v[u][h + 3]);
          if (SUM) sa.add4(f, c);
          if (ARG) aa.add4(f, W * (g + u * kRowThreads) + h);
          if (WATCH) watch4(f, W * (g + u * kRowThreads) + h, watch, wv);
        }
    }
    for (; g < g1; g += kRowThreads) {
      float v[W];
      LT::stream_vec(x + W * g, v);
#pragma unroll
      for (int h = 0; h < W; h += 4) {
        const float4 f = make_float4(v[h], v[h + 1], v[h + 2], v[h + 3]);
        if (SUM) sa.add4(f, c);
        if (ARG) aa.add4(f, W * g + h);
        if (WATCH) watch4(f, W * g + h, watch, wv);
      }
    }
  } else {
    for (int i = c0 + tid; i < c1; i += kRowThreads) {
      const float v = LT::stream1(x + i);
      if (SUM) sa.add1(v, c);
      if (ARG) aa.add1(v, i);
      if (WATCH && i == watch) wv = v;
    }
  }
  if (WATCH && watch >= c0 && watch < c1 && (VEC ? ((watch / W) - c0 / W) % kRowThreads == tid
                                                 : (watch - c0) % kRowThreads == tid))
    *watched = wv;
}

// Combine the (m, s) pairs of all threads of the CTA; result valid in thread 0.
__device__ __forceinline__ void cta_reduce_sum(float& m, float& s, float c, float* sm /*[2*32]*/) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, off);
    const float s2 = __shfl_xor_sync(0xffffffffu, s, off);
    const float M = fmaxf(m, m2);
    if (M != -INFINITY) {
      s = s * ex2_approx((m - M) * c) + s2 * ex2_approx((m2 - M) * c);
      m = M;
    }
  }
  if (lane == 0) { sm[2 * warp] = m; sm[2 * warp + 1] = s; }
  __syncthreads();
  if (threadIdx.x == 0) {
    m = sm[0];
    s = sm[1];
    for (int w = 1; w < (int)(blockDim.x >> 5); ++w) {
      const float m2 = sm[2 * w], s2 = sm[2 * w + 1];
      const float M = fmaxf(m, m2);
      if (M != -INFINITY) {
        s = s * ex2_approx((m - M) * c) + s2 * ex2_approx((m2 - M) * c);
        m = M;
      }
    }
  }
}

// Combine (max, argmax) of all threads; result valid in thread 0.
__device__ __forceinline__ void cta_reduce_arg(float& m, int& arg, float* smf /*[32]*/, int* smi /*[32]*/) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, off);
    const int a2 = __shfl_xor_sync(0xffffffffu, arg, off);
    argmax_combine(m, arg, m2, a2);
  }
  if (lane == 0) { smf[warp] = m; smi[warp] = arg; }
  __syncthreads();
  if (threadIdx.x == 0) {
    m = smf[0];
    arg = smi[0];
    for (int w = 1; w < (int)(blockDim.x >> 5); ++w) argmax_combine(m, arg, smf[w], smi[w]);
  }
}

// Merge nsplit partials of one row (one warp; result in lane 0). Each share
// s_i was summed relative to its own max m_i; it is rescaled to the row max M
// by 2^((m_i - M) c), c = log2(e)/T, and the shares are added in binary64
// (additions only: GB300 runs binary64 at a small fraction of the fp32 rate).
// A lane reads each of its partials whole (one 16-byte load) and keeps up to
// kMergeHeld of them, so up to 32 * kMergeHeld partials cost one memory round
// trip; the sums are taken in the same order either way.
constexpr int kMergeHeld = 2;
__device__ __forceinline__ void warp_merge_partials(const RowPartial* __restrict__ p, int nsplit, float c,
                                                    bool want_arg, float& m_out, int& arg_out,
                                                    double& s_out) {
  const int lane = threadIdx.x & 31;
  float mh[kMergeHeld];
  double sh[kMergeHeld];
  float m = -INFINITY;
  int arg = 0x7fffffff;
#pragma unroll
  for (int k = 0; k < kMergeHeld; ++k) {
    const int i = lane + 32 * k;
    mh[k] = -INFINITY;
    sh[k] = 0.0;
    if (i < nsplit) {
      const double2 raw = __ldcg(reinterpret_cast<const double2*>(p + i));
      const long long mw = __double_as_longlong(raw.x);
      mh[k] = __int_as_float((int)(mw & 0xffffffffll));
      const int ai = (int)(mw >> 32);
      sh[k] = raw.y;
      if (want_arg) argmax_combine(m, arg, mh[k], ai);
      else m = fmaxf(m, mh[k]);
    }
  }
  for (int i = lane + 32 * kMergeHeld; i < nsplit; i += 32) {
    const float mi = __ldcg(&p[i].m);
    const int ai = __ldcg(&p[i].arg);
    if (want_arg) argmax_combine(m, arg, mi, ai);
    else m = fmaxf(m, mi);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, off);
    const int a2 = __shfl_xor_sync(0xffffffffu, arg, off);
    if (want_arg) argmax_combine(m, arg, m2, a2);
    else m = fmaxf(m, m2);
  }
  double s = 0.0;
  if (m != -INFINITY) {
#pragma unroll
    for (int k = 0; k < kMergeHeld; ++k)
      if (mh[k] != -INFINITY) s += sh[k] * (double)ex2_approx((mh[k] - m) * c);
    for (int i = lane + 32 * kMergeHeld; i < nsplit; i += 32) {
      const float mi = __ldcg(&p[i].m);
      const double si = __ldcg(&p[i].s);
      if (mi != -INFINITY) s += si * (double)ex2_approx((mi - m) * c);
    }
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
  m_out = m;
  arg_out = arg;
  s_out = s;
}

// Choose how many CTAs share a row: enough CTAs in total to fill the GPU
// several times over, each with at least min_elems elements.
inline int row_splits(long rows, int V, int num_sms, int max_splits, int min_elems) {
  if (rows <= 0) return 1;
  const long target = 2L * 8 * num_sms;
  long ns = (target + rows - 1) / rows;
  const long cap = (V + min_elems - 1) / min_elems;  // at least min_elems per CTA
  if (ns > cap) ns = cap;
  if (ns > max_splits) ns = max_splits;
  if (ns < 1) ns = 1;
  return (int)ns;
}

// Splits per drafter row for the confidence pass: the fewest that give about
// 0.6 of one wave of resident CTAs (8 per SM), each of at least min_elems
// elements. Long CTAs amortise each CTA's reduction and ticket, and a count
// below a whole wave leaves no straggling wave (measured: sampling's 256
// rows 37.2 us at 10 splits, 33.1 at 3; ragged's 2048 rows 156.7 us at 2,
// 152.2 at 1).
inline int conf_row_splits(long rows, int V, int num_sms, int max_splits, int min_elems) {
  if (rows <= 0) return 1;
  const long target = (6L * 8 * num_sms + 9) / 10;
  long ns = (target + rows - 1) / rows;
  const long cap = (V + min_elems - 1) / min_elems;
  if (ns > cap) ns = cap;
  if (ns > max_splits) ns = max_splits;
  if (ns < 1) ns = 1;
  return (int)ns;
}

// Split length: a multiple of 8 elements (whole 128-bit loads of fp32 or bf16).
constexpr int kRowAlign = 8;
inline int row_chunk(int V, int nsplit) {
  int ch = (V + nsplit - 1) / nsplit;
  return (ch + kRowAlign - 1) & ~(kRowAlign - 1);
}

// 128-bit loads cover a row of V logits of type T at base x.
template <typename T>
inline bool rows_vectorizable(const T* x, int V) {
  return (V % Logit<T>::kVec == 0) && ((reinterpret_cast<uintptr_t>(x) & 15) == 0);
}

}  // namespace libraspec
