// Shared device helpers of the libraspec kernels (sm_103a).
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include <algorithm>

#include "libraspec.h"

namespace libraspec {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

// ---------------------------------------------------------------------------
// Workspace layout. Every region is 256-byte aligned; counters are reset to
// zero by the kernel that uses them, so one zero-fill serves every call.
// ---------------------------------------------------------------------------
constexpr int kConfMaxSplits = 64;    // CTAs per drafter row
constexpr int kRowMaxSplits = 64;     // CTAs per target row (acceptance)
constexpr int kRaceMaxSplits = 128;   // CTAs per sequence for a vocabulary draw
constexpr int kAttnMaxCtas = 192;     // persistent attention grid cap (one CTA per SM)
// Buffers of split-group partials: layer l writes buffer l % 3, so layer l's
// merge may run until layer l + 2 starts, a layer after the one it overlaps.
constexpr int kAttnPartBufs = 3;
constexpr int kAttnRows = 128;        // query rows per attention row group (at most)
constexpr int kAttnTileKeys = 64;     // keys per KV tile
constexpr int kAttnMaxLayers = LIBRASPEC_ATTN_LAYERS_PER_LAUNCH;  // layers per attention launch
constexpr int kAccMaxGrid = 6144;     // acceptance rows grid cap (4 waves of 8 CTAs on <= 192 SMs)

struct RowPartial {      // one CTA's share of a logit row
  float m;               // max
  int arg;               // argmax (lowest index among maxima)
  double s;              // sum of exp((x - m) / T)
};
static_assert(sizeof(RowPartial) == 16, "a partial is read as one 16-byte load");

struct RowStat {         // merged statistics of a target row
  float m;
  int arg;
  double Z;
};

struct RacePartial {
  float key;
  int idx;
};

// A race candidate carried without the row's normaliser: the key of token v
// is E_v * 2^(-y_v c) (E_v = -ln u_v, c = log2(e) / T), compared between two
// candidates as E_a < E_b * 2^((y_a - y_b) c).
struct RaceCand {
  float E;
  float y;
  int idx;
  int pad;
};

// The draw that ends a sampling sequence's acceptance: mode 1, the bonus
// draw from target row n = L_b (all drafts accepted); mode 2, the residual
// draw max(0, p_n - q_n) after a rejection at n (with row n's max and
// normaliser); mode 0, none (a sampling sequence without units: a length
// out of range, or no drafter statistics). A greedy sequence publishes none.
struct ResEntry {
  int n;
  int mode;
  float mp;     // max of target row n (mode 2)
  float invZp;  // 1 / sum of exp((y - mp) / T) of target row n (mode 2)
};

struct WsLayout {
  size_t status, conf_part, conf_cnt, seq_cnt, row_part, row_cnt, row_stat, race_part, race_cnt;
  size_t acc_seq, acc_yx, acc_res, acc_ready, acc_plan;
  size_t attn_o, attn_ml, attn_cnt, attn_grp, tree_vis, total;
  int max_items, max_groups;
};

inline size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

inline WsLayout ws_layout(int B, int K, int V, int Hq, int Hkv, int d, int S_cap) {
  (void)V; (void)S_cap;
  WsLayout w{};
  size_t off = 0;
  auto take = [&](size_t bytes) { size_t o = off; off = align256(off + bytes); return o; };
  const size_t rows_d = size_t(B) * K, rows_t = size_t(B) * (K + 1);
  const int g = Hkv > 0 ? Hq / Hkv : 1;
  const int m_max = (K + 1) * g;
  const int rows = g >= 1 && g <= kAttnRows ? g * (kAttnRows / g) : 1;
  const int n_mg = (m_max + rows - 1) / rows;
  w.max_groups = B * Hkv * n_mg;
  w.max_items = kAttnMaxCtas + w.max_groups;
  w.status = take(256);
  w.conf_part = take(rows_d * kConfMaxSplits * sizeof(RowPartial));
  w.conf_cnt = take(rows_d * sizeof(uint32_t));
  w.seq_cnt = take(size_t(B) * sizeof(uint32_t));  // rows of a sequence done (fused selection)
  w.row_part = take(rows_t * kRowMaxSplits * sizeof(RowPartial));
  w.row_cnt = take(rows_t * sizeof(uint32_t));
  w.row_stat = take(rows_t * sizeof(RowStat));
  w.race_part = take(size_t(B) * kRaceMaxSplits * sizeof(RaceCand));
  w.race_cnt = take(size_t(B) * sizeof(uint32_t));
  // acceptance: slices done per sequence, the target logit at each drafted
  // token, and each sequence's residual draw (or none)
  w.acc_seq = take(size_t(B) * sizeof(uint32_t));
  w.acc_yx = take(rows_t * sizeof(float));
  w.acc_res = take(size_t(B) * sizeof(ResEntry));
  w.acc_ready = take(size_t(B) * sizeof(uint32_t));  // res[b] published
  // the acceptance plan: a header, then one 8-byte descriptor per unit
  w.acc_plan = take(16 + 8 * std::max(size_t(kAccMaxGrid), rows_t));
  // two partial slots per attention CTA (its first and its last item), in
  // kAttnPartBufs buffers that rotate with the layer (layer % kAttnPartBufs)
  w.attn_o = take(kAttnPartBufs * size_t(2 * kAttnMaxCtas) * kAttnRows * d * sizeof(float));
  w.attn_ml = take(kAttnPartBufs * size_t(2 * kAttnMaxCtas) * kAttnRows * 2 * sizeof(float));
  // grid-barrier counters, one per layer of a launch, then the exit counter
  w.attn_cnt = take((kAttnMaxLayers + 1) * sizeof(uint32_t));
  // per row group: parts of the last layer counted in, CTAs past its wait
  w.attn_grp = take(2 * size_t(w.max_groups) * sizeof(uint32_t));
  // ancestor masks of a draft tree, ceil(K / 64) words per block position
  w.tree_vis = take(rows_t * size_t(K <= 64 ? 1 : (K + 63) / 64) * sizeof(uint64_t));
  w.total = off;
  return w;
}

// ---------------------------------------------------------------------------
// Status word (device side): bits are OR-ed in, never cleared by kernels.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void raise_status(int* status, int bits) {
  if (status) atomicOr(status, bits);
}

// ---------------------------------------------------------------------------
// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11), from its definition:
// a round maps (x0,x1,x2,x3) with key (k0,k1) to
// (hi(M1 x2) ^ x1 ^ k0, lo(M1 x2), hi(M0 x0) ^ x3 ^ k1, lo(M0 x0)); the key
// advances by (W0, W1) between rounds.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint2 k) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const uint32_t lo0 = 0xD2511F53u * c.x, hi0 = __umulhi(0xD2511F53u, c.x);
    const uint32_t lo1 = 0xCD9E8D57u * c.z, hi1 = __umulhi(0xCD9E8D57u, c.z);
    c = make_uint4(hi1 ^ c.y ^ k.x, lo1, hi0 ^ c.w ^ k.y, lo0);
    k.x += 0x9E3779B9u;
    k.y += 0xBB67AE85u;
  }
  return c;
}

// Counter of a draw: (idx, position j, global sequence, purpose + 4 * round).
__device__ __forceinline__ uint4 philox_block(uint64_t seed, uint32_t idx, uint32_t j, uint32_t seq,
                                              uint32_t purpose, uint64_t round_offset) {
  return philox4x32_10(make_uint4(idx, j, seq, purpose + 4u * (uint32_t)round_offset),
                       make_uint2((uint32_t)seed, (uint32_t)(seed >> 32)));
}

// u = ((w >> 9) + 1/2) * 2^-23: strictly inside (0,1), exact in binary32.
// Formed without an integer-to-float conversion: the word's top 23 bits as
// the mantissa of a = 1 + (w >> 9) 2^-23 in [1, 2), then a - (1 - 2^-24),
// which is exact (Sterbenz: the operands are within a factor of two), so u
// has the same bits as the conversion-and-scale form.
__device__ __forceinline__ float word_to_uniform(uint32_t w) {
  return __fsub_rn(__uint_as_float(0x3F800000u | (w >> 9)), 0.999999940395355224609375f);
}

// ---------------------------------------------------------------------------
// Fast base-2 exponential (the MUFU instruction); used where the result only
// needs relative accuracy of a few ulp.
// ---------------------------------------------------------------------------
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// c = log2(e) / T in binary32 arithmetic alone (GB300 runs binary64 at a
// small fraction of the binary32 rate, so one binary64 division per thread
// costs more than the thread's share of a logit row). log2(e) = hi + lo; the
// rounded quotient q = hi / T is corrected once by the exact remainder
// hi - q T (an FMA) plus lo: the result is log2(e) / T rounded to binary32,
// up to a residual far below half an ulp.
__device__ __forceinline__ float log2e_over(float T) {
  const float hi = 1.44269502162933349609375f;  // binary32 log2(e)
  const float lo = 1.925963033500011e-08f;      // log2(e) - hi
  const float q = __fdiv_rn(hi, T);
  const float r = __fadd_rn(__fmaf_rn(-q, T, hi), lo);
  return __fmaf_rn(r, __frcp_rn(T), q);
}

// Streaming 128-bit load that does not allocate in L1.
__device__ __forceinline__ float4 ld_stream4(const float* p) {
  float4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.f32 {%0,%1,%2,%3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "l"(p));
  return v;
}

__device__ __forceinline__ float ld_stream(const float* p) {
  float v;
  asm volatile("ld.global.nc.L1::no_allocate.f32 %0, [%1];" : "=f"(v) : "l"(p));
  return v;
}

// Logit element types: fp32, or bf16 passed as its 16-bit pattern. A bf16
// value widens to fp32 exactly (its bits are the top half of the fp32 word).
__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

template <typename T>
struct Logit;

template <>
struct Logit<float> {
  static constexpr int kVec = 4;  // elements per 16-byte load
  __device__ static __forceinline__ float at(const float* p, size_t i) { return p[i]; }
  __device__ static __forceinline__ float stream1(const float* p) { return ld_stream(p); }
  // kVec elements from a 16-byte-aligned address
  __device__ static __forceinline__ void stream_vec(const float* p, float (&v)[4]) {
    const float4 a = ld_stream4(p);
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
  }
  // 4 elements from an address aligned to 4 elements
  __device__ static __forceinline__ void stream4(const float* p, float (&v)[4]) { stream_vec(p, v); }
};

template <>
struct Logit<uint16_t> {
  static constexpr int kVec = 8;
  __device__ static __forceinline__ float at(const uint16_t* p, size_t i) {
    return __uint_as_float((uint32_t)p[i] << 16);
  }
  __device__ static __forceinline__ float stream1(const uint16_t* p) {
    unsigned short h;
    asm volatile("ld.global.nc.L1::no_allocate.u16 %0, [%1];" : "=h"(h) : "l"(p));
    return __uint_as_float((uint32_t)h << 16);
  }
  __device__ static __forceinline__ void stream_vec(const uint16_t* p, float (&v)[8]) {
    uint32_t w0, w1, w2, w3;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(w0), "=r"(w1), "=r"(w2), "=r"(w3)
                 : "l"(p));
    v[0] = bf16_lo(w0); v[1] = bf16_hi(w0); v[2] = bf16_lo(w1); v[3] = bf16_hi(w1);
    v[4] = bf16_lo(w2); v[5] = bf16_hi(w2); v[6] = bf16_lo(w3); v[7] = bf16_hi(w3);
  }
  __device__ static __forceinline__ void stream4(const uint16_t* p, float (&v)[4]) {
    uint32_t w0, w1;
    asm volatile("ld.global.nc.L1::no_allocate.v2.u32 {%0,%1}, [%2];" : "=r"(w0), "=r"(w1) : "l"(p));
    v[0] = bf16_lo(w0); v[1] = bf16_hi(w0); v[2] = bf16_lo(w1); v[3] = bf16_hi(w1);
  }
};

// Combine two (m, s) pairs (binary64 sums); c = log2(e) / T.
__device__ __forceinline__ void combine_ms(float& m, double& s, float m2, double s2, float c) {
  if (m2 == -INFINITY) return;
  if (m == -INFINITY) { m = m2; s = s2; return; }
  if (m2 > m) {
    s = s * (double)exp2f((m - m2) * c) + s2;
    m = m2;
  } else {
    s = s + s2 * (double)exp2f((m2 - m) * c);
  }
}

// (value, index) max with the lowest index winning ties.
__device__ __forceinline__ void argmax_combine(float& v, int& i, float v2, int i2) {
  if (v2 > v || (v2 == v && i2 < i)) { v = v2; i = i2; }
}

// (key, index) min with the lowest index winning ties.
__device__ __forceinline__ void argmin_combine(float& k, int& i, float k2, int i2) {
  if (k2 < k || (k2 == k && i2 < i)) { k = k2; i = i2; }
}

}  // namespace libraspec
