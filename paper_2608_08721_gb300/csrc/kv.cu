// Appending the verified block's keys and values to the KV caches: before
// the verify attention reads them, the rows of block positions 0..T-1 of
// sequence b go to cache rows kv_len_b .. kv_len_b + T - 1 of every layer
// (the target model computes them for the block, Sec. 3.1). One thread moves
// 16 bytes; all layers of a call go in one launch per 64 layers.
#include "common.cuh"

namespace libraspec {

constexpr int kAppendLayers = 64;
constexpr int kAppendThreads = 256;

struct AppendPtrs {
  uint16_t* K[kAppendLayers];
  uint16_t* V[kAppendLayers];
};

// kv_new [n_layers, 2, B, Hkv, T, d] (K then V). Dense caches [B, Hkv, S_cap,
// d]; paged (block_table != nullptr): pools [n_pages, Hkv, page_size, d] and
// cache row s of sequence b at page block_table[b * max_pages + s / page_size].
__global__ void __launch_bounds__(kAppendThreads) kv_append_kernel(
    const __grid_constant__ AppendPtrs ptrs, const uint4* __restrict__ kv_new, int n_layers,
    const int32_t* __restrict__ kv_len, const int32_t* __restrict__ block_table, int max_pages, int page_size,
    int n_pages, int B, int T, int Hkv, int d, int S_cap, int* __restrict__ status) {
  const int c16 = d / 8;  // 16-byte chunks per row
  const long long per_kv = (long long)B * Hkv * T * c16;
  const long long total = (long long)n_layers * 2 * per_kv;
  for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total;
       i += (long long)gridDim.x * blockDim.x) {
    long long q = i;
    const int c = (int)(q % c16);
    q /= c16;
    const int r = (int)(q % T);
    q /= T;
    const int h = (int)(q % Hkv);
    q /= Hkv;
    const int b = (int)(q % B);
    q /= B;
    const int which = (int)(q % 2);
    const int l = (int)(q / 2);
    const int kv = kv_len[b];
    const long long s = (long long)kv + r;
    if (kv < 0 || s >= S_cap) {
      if (c == 0) raise_status(status, LIBRASPEC_ST_KV_OVERFLOW);
      continue;
    }
    size_t row;
    if (block_table) {
      int page = block_table[(size_t)b * max_pages + s / page_size];
      if (page < 0 || page >= n_pages) {
        if (c == 0) raise_status(status, LIBRASPEC_ST_BAD_PAGE);
        continue;
      }
      row = ((size_t)page * Hkv + h) * page_size + (size_t)(s % page_size);
    } else {
      row = ((size_t)b * Hkv + h) * S_cap + (size_t)s;
    }
    uint16_t* dst = which ? ptrs.V[l] : ptrs.K[l];
    reinterpret_cast<uint4*>(dst + row * d)[c] = kv_new[i];
  }
}

cudaError_t launch_kv_append(const uint16_t* kv_new, uint16_t* const* Kc, uint16_t* const* Vc, int n_layers,
                             const int32_t* kv_len, const int32_t* block_table, int max_pages, int page_size,
                             int n_pages, int B, int T, int Hkv, int d, int S_cap, int* status,
                             cudaStream_t stream) {
  if (B == 0 || T == 0 || n_layers == 0) return cudaSuccess;
  const size_t layer_elems = (size_t)2 * B * Hkv * T * d;
  for (int l0 = 0; l0 < n_layers; l0 += kAppendLayers) {
    const int n = n_layers - l0 < kAppendLayers ? n_layers - l0 : kAppendLayers;
    AppendPtrs p{};
    for (int i = 0; i < n; ++i) {
      p.K[i] = Kc[l0 + i];
      p.V[i] = Vc[l0 + i];
    }
    const long long total = (long long)n * 2 * B * Hkv * T * (d / 8);
    long long blocks = (total + kAppendThreads - 1) / kAppendThreads;
    if (blocks > 16 * 152) blocks = 16 * 152;
    kv_append_kernel<<<(int)blocks, kAppendThreads, 0, stream>>>(
        p, reinterpret_cast<const uint4*>(kv_new + (size_t)l0 * layer_elems), n, kv_len, block_table, max_pages,
        page_size, n_pages, B, T, Hkv, d, S_cap, status);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace libraspec
