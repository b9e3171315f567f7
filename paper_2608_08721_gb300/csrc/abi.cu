// The C ABI (include/libraspec.h): argument checks, workspace, status and
// the whole-round entry point. Kernels live in conf_select.cu, attn.cu and
// accept.cu.
#include <cstdio>
#include <cstring>
#include <vector>

#include "common.cuh"

namespace libraspec {

template <typename T>
cudaError_t launch_confidence(const T*, const int32_t*, const float*, int, int, int, float*, float*, char*,
                              const WsLayout&, cudaStream_t, const float*, int32_t*);
cudaError_t launch_select(const float*, const float*, int, int, int32_t*, char*, const WsLayout&, cudaStream_t);
cudaError_t launch_select_alpha(const float*, int, int, int, double, int32_t*, int32_t*, cudaStream_t);
cudaError_t launch_verify_attn(const uint16_t*, const uint16_t*, const uint16_t*, const int32_t*, const int32_t*,
                               int, int, int, int, int, int, float, uint16_t*, float*, char*, const WsLayout&,
                               cudaStream_t);
cudaError_t launch_verify_attn_paged_layers(const uint16_t* const*, const uint16_t* const*, const uint16_t* const*,
                                            int, const int32_t*, const int32_t*, int, int, int, const int32_t*,
                                            const int32_t*, int, int, int, int, int, float, uint16_t* const*,
                                            float* const*, char*, const WsLayout&, cudaStream_t);
cudaError_t launch_verify_attn_layers(const uint16_t* const*, const uint16_t* const*, const uint16_t* const*, int,
                                      const int32_t*, const int32_t*, const int32_t*, int, int, int, int, int, int,
                                      float, uint16_t* const*, float* const*, char*, const WsLayout&, cudaStream_t);
size_t lm_head_workspace_bytes(int M, int V);
cudaError_t launch_lm_head_stats(const uint16_t*, const uint16_t*, const float*, int, const int32_t*, int, int, int,
                                 float*, int32_t*, float*, char*, cudaStream_t);
cudaError_t launch_kv_append(const uint16_t*, uint16_t* const*, uint16_t* const*, int, const int32_t*,
                             const int32_t*, int, int, int, int, int, int, int, int, int*, cudaStream_t);
template <typename T>
cudaError_t launch_accept_tree(const T*, const int32_t*, const int32_t*, const int32_t*, const float*, int, int, int,
                               uint64_t, uint64_t, uint32_t, int32_t*, int32_t*, int32_t*, char*, const WsLayout&,
                               cudaStream_t);
template <typename T>
cudaError_t launch_accept(const T*, const T*, const int32_t*, const float*, const float*, const int32_t*,
                          const float*, int, int, int, uint64_t, uint64_t, uint32_t, int32_t*, int32_t*, char*,
                          const WsLayout&, cudaStream_t, const uint64_t*, bool);
cudaError_t launch_selftest_wait(const uint32_t*, uint64_t, int32_t*, int*, cudaStream_t);
template <typename T>
cudaError_t launch_accept_plan(const T*, const T*, const float*, const float*, const int32_t*, const float*, int,
                               int, int, int32_t*, int32_t*, char*, const WsLayout&, cudaStream_t);

int num_sms_current() {
  static int cached_dev = -1, cached_sms = 0;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 148;
  if (dev != cached_dev) {
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0) sms = 148;
    cached_sms = sms;
    cached_dev = dev;
  }
  return cached_sms;
}

}  // namespace libraspec

using namespace libraspec;

namespace {

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

bool shapes_ok(int B, int K, int V) {
  return B >= 0 && B <= LIBRASPEC_MAX_B && K >= 0 && K <= LIBRASPEC_MAX_K && V >= 1;
}

// tree: K is the node budget N (<= LIBRASPEC_MAX_TREE_NODES) and the block
// may hold any number of query rows per kv head.
bool attn_shapes_ok(int B, int K, int Hq, int Hkv, int D, int S_cap, bool tree = false) {
  if (B < 0 || B > LIBRASPEC_MAX_B || K < 0 || K > (tree ? LIBRASPEC_MAX_TREE_NODES : LIBRASPEC_MAX_K)) return false;
  if (Hq < 1 || Hkv < 1 || Hq % Hkv != 0 || S_cap < 1) return false;
  if (!tree && (long)(K + 1) * (Hq / Hkv) > 512) return false;
  if (Hq / Hkv > kAttnRows) return false;  // a row group holds at least one block position
  if ((long)B * Hkv > (1L << 30)) return false;
  (void)D;
  return true;
}

int from_cuda(cudaError_t e) { return e == cudaSuccess ? LIBRASPEC_OK : LIBRASPEC_ECUDA; }

}  // namespace

extern "C" {

const char* libraspec_version(void) { return "libraspec 0.1 (sm_103a)"; }

const char* libraspec_status_string(int status) {
  switch (status) {
    case LIBRASPEC_OK: return "ok";
    case LIBRASPEC_EINVAL: return "invalid argument";
    case LIBRASPEC_EUNSUPPORTED: return "unsupported shape";
    case LIBRASPEC_ECUDA: return "CUDA error";
    case LIBRASPEC_EDEVICE: return "device-reported violation";
    default: return "unknown status";
  }
}

size_t libraspec_workspace_size(int B, int K, int V, int Hq, int Hkv, int head_dim, int S_cap) {
  if (B < 0 || B > LIBRASPEC_MAX_B || K < 0 || K > LIBRASPEC_MAX_TREE_NODES || V < 1 || Hq < 1 || Hkv < 1 || Hq % Hkv != 0 || (head_dim != 64 && head_dim != 128) ||
      S_cap < 1)
    return 0;
  return ws_layout(B, K, V, Hq, Hkv, head_dim, S_cap).total;
}

int libraspec_workspace_init(void* workspace, size_t bytes, void* stream) {
  if (!workspace || !aligned(workspace, 256)) return LIBRASPEC_EINVAL;
  return from_cuda(cudaMemsetAsync(workspace, 0, bytes, static_cast<cudaStream_t>(stream)));
}

int libraspec_selftest_wait(const uint32_t* flag, uint64_t limit_ns, int32_t* observed, void* workspace,
                            size_t ws_bytes, void* stream) {
  if (!flag || !observed || !workspace || !aligned(workspace, 256) || ws_bytes < 256 || !aligned(flag, 4) ||
      !aligned(observed, 4) || limit_ns < 1 || limit_ns > 2000000000ull)
    return LIBRASPEC_EINVAL;
  return from_cuda(launch_selftest_wait(flag, limit_ns, observed, static_cast<int*>(workspace),
                                        static_cast<cudaStream_t>(stream)));
}

int libraspec_get_status(void* workspace, void* stream, int32_t* host_status) {
  if (!workspace || !host_status) return LIBRASPEC_EINVAL;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int32_t v = 0;
  cudaError_t e = cudaMemcpyAsync(&v, workspace, sizeof(v), cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e == cudaSuccess && v != 0) e = cudaMemsetAsync(workspace, 0, sizeof(v), s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return LIBRASPEC_ECUDA;
  *host_status = v;
  return v == 0 ? LIBRASPEC_OK : LIBRASPEC_EDEVICE;
}

// The workspace must hold the regions of the layout computed from the call's
// own shapes; the layout puts every region after the ones of smaller calls,
// so we check the bytes the call touches.
static bool ws_ok(const void* ws, size_t ws_bytes, const WsLayout& lay) {
  return ws && aligned(ws, 256) && ws_bytes >= lay.total;
}

extern "C++" {
template <typename T>
static int confidence_t(const T* draft_logits, const int32_t* draft_tokens, const float* temperature, int B, int K,
                        int V, float* conf, float* dstat, void* workspace, size_t ws_bytes, void* stream,
                        const float* cost = nullptr, int32_t* L = nullptr) {
  if (!shapes_ok(B, K, V)) return LIBRASPEC_EINVAL;
  if (B * K == 0) return LIBRASPEC_OK;
  if (!draft_logits || !draft_tokens || !temperature || !conf) return LIBRASPEC_EINVAL;
  if (!aligned(draft_logits, sizeof(T)) || !aligned(conf, 4) || (dstat && !aligned(dstat, 4)))
    return LIBRASPEC_EINVAL;
  const WsLayout lay = ws_layout(B, K, V, 1, 1, 64, 1);
  if (!ws_ok(workspace, ws_bytes, lay)) return LIBRASPEC_EINVAL;
  return from_cuda(launch_confidence<T>(draft_logits, draft_tokens, temperature, B, K, V, conf, dstat,
                                        static_cast<char*>(workspace), lay, static_cast<cudaStream_t>(stream), cost,
                                        L));
}
}  // extern "C++"

int libraspec_confidence(const float* draft_logits, const int32_t* draft_tokens, const float* temperature, int B,
                         int K, int V, float* conf, float* dstat, void* workspace, size_t ws_bytes, void* stream) {
  return confidence_t(draft_logits, draft_tokens, temperature, B, K, V, conf, dstat, workspace, ws_bytes, stream);
}

int libraspec_confidence_bf16(const uint16_t* draft_logits, const int32_t* draft_tokens, const float* temperature,
                              int B, int K, int V, float* conf, float* dstat, void* workspace, size_t ws_bytes,
                              void* stream) {
  return confidence_t(draft_logits, draft_tokens, temperature, B, K, V, conf, dstat, workspace, ws_bytes, stream);
}

int libraspec_confidence_select(const float* draft_logits, const int32_t* draft_tokens, const float* temperature,
                                const float* cost_table, int B, int K, int V, float* conf, float* dstat, int32_t* L,
                                void* workspace, size_t ws_bytes, void* stream) {
  if (!cost_table || !L) return LIBRASPEC_EINVAL;
  if (K == 0) return libraspec_select_lengths(conf, cost_table, B, K, L, workspace, ws_bytes, stream);
  return confidence_t(draft_logits, draft_tokens, temperature, B, K, V, conf, dstat, workspace, ws_bytes, stream,
                      cost_table, L);
}

int libraspec_confidence_select_bf16(const uint16_t* draft_logits, const int32_t* draft_tokens,
                                     const float* temperature, const float* cost_table, int B, int K, int V,
                                     float* conf, float* dstat, int32_t* L, void* workspace, size_t ws_bytes,
                                     void* stream) {
  if (!cost_table || !L) return LIBRASPEC_EINVAL;
  if (K == 0) return libraspec_select_lengths(conf, cost_table, B, K, L, workspace, ws_bytes, stream);
  return confidence_t(draft_logits, draft_tokens, temperature, B, K, V, conf, dstat, workspace, ws_bytes, stream,
                      cost_table, L);
}

int libraspec_select_lengths(const float* conf, const float* cost_table, int B, int K, int32_t* L, void* workspace,
                             size_t ws_bytes, void* stream) {
  if (!shapes_ok(B, K, 1)) return LIBRASPEC_EINVAL;
  if (B == 0) return LIBRASPEC_OK;
  if ((!conf && K > 0) || !cost_table || !L) return LIBRASPEC_EINVAL;
  const WsLayout lay = ws_layout(B, K, 1, 1, 1, 64, 1);
  if (!workspace || !aligned(workspace, 256) || ws_bytes < 256) return LIBRASPEC_EINVAL;
  return from_cuda(
      launch_select(conf, cost_table, B, K, L, static_cast<char*>(workspace), lay, static_cast<cudaStream_t>(stream)));
}

int libraspec_select_alpha(const float* conf, int B, int K, int block_size, float alpha, int32_t* L,
                           int32_t* n_blocks, void* stream) {
  if (B < 0 || K < 1 || K > LIBRASPEC_MAX_K || block_size < 1 || block_size > K) return LIBRASPEC_EINVAL;
  if (!(alpha > 0.f) || !isfinite(alpha)) return LIBRASPEC_EINVAL;
  if (B == 0) return LIBRASPEC_OK;
  if (!conf || !L) return LIBRASPEC_EINVAL;
  return from_cuda(launch_select_alpha(conf, B, K, block_size, (double)alpha, L, n_blocks,
                                       static_cast<cudaStream_t>(stream)));
}

int libraspec_verify_attn(const uint16_t* Q, const uint16_t* Kc, const uint16_t* Vc, const int32_t* kv_len,
                          const int32_t* L, int B, int K, int Hq, int Hkv, int head_dim, int S_cap, float softmax_scale,
                          uint16_t* O, float* lse, void* workspace, size_t ws_bytes, void* stream) {
  if (head_dim != 64 && head_dim != 128) return LIBRASPEC_EUNSUPPORTED;
  if (!attn_shapes_ok(B, K, Hq, Hkv, head_dim, S_cap)) return LIBRASPEC_EINVAL;
  if (B == 0) return LIBRASPEC_OK;
  if (!Q || !Kc || !Vc || !kv_len || !L || !O) return LIBRASPEC_EINVAL;
  if (!aligned(Q, 16) || !aligned(Kc, 16) || !aligned(Vc, 16) || !aligned(O, 16)) return LIBRASPEC_EINVAL;
  if (lse && !aligned(lse, 4)) return LIBRASPEC_EINVAL;
  if (!(softmax_scale > 0.f)) return LIBRASPEC_EINVAL;
  const WsLayout lay = ws_layout(B, K, 1, Hq, Hkv, head_dim, S_cap);
  if (!ws_ok(workspace, ws_bytes, lay)) return LIBRASPEC_EINVAL;
  return from_cuda(launch_verify_attn(Q, Kc, Vc, kv_len, L, B, K, Hq, Hkv, head_dim, S_cap, softmax_scale, O, lse,
                                      static_cast<char*>(workspace), lay, static_cast<cudaStream_t>(stream)));
}

namespace {

int attn_layers(const uint16_t* const* Q, const uint16_t* const* Kc, const uint16_t* const* Vc, int n_layers,
                const int32_t* parent, bool tree, const int32_t* kv_len, const int32_t* L, int B, int K, int Hq,
                int Hkv, int head_dim, int S_cap, float softmax_scale, uint16_t* const* O, float* const* lse,
                void* workspace, size_t ws_bytes, void* stream) {
  if (head_dim != 64 && head_dim != 128) return LIBRASPEC_EUNSUPPORTED;
  if (!attn_shapes_ok(B, K, Hq, Hkv, head_dim, S_cap, tree) || n_layers < 0) return LIBRASPEC_EINVAL;
  if (B == 0 || n_layers == 0) return LIBRASPEC_OK;
  if (!Q || !Kc || !Vc || !O || !kv_len || !L || (tree && !parent)) return LIBRASPEC_EINVAL;
  for (int l = 0; l < n_layers; ++l) {
    if (!Q[l] || !Kc[l] || !Vc[l] || !O[l]) return LIBRASPEC_EINVAL;
    if (!aligned(Q[l], 16) || !aligned(Kc[l], 16) || !aligned(Vc[l], 16) || !aligned(O[l], 16))
      return LIBRASPEC_EINVAL;
    if (lse && lse[l] && !aligned(lse[l], 4)) return LIBRASPEC_EINVAL;
  }
  if (!(softmax_scale > 0.f)) return LIBRASPEC_EINVAL;
  const WsLayout lay = ws_layout(B, K, 1, Hq, Hkv, head_dim, S_cap);
  if (!ws_ok(workspace, ws_bytes, lay)) return LIBRASPEC_EINVAL;
  return from_cuda(launch_verify_attn_layers(Q, Kc, Vc, n_layers, parent, kv_len, L, B, K, Hq, Hkv, head_dim,
                                             S_cap, softmax_scale, O, lse, static_cast<char*>(workspace), lay,
                                             static_cast<cudaStream_t>(stream)));
}

int attn_paged_layers(const uint16_t* const* Q, const uint16_t* const* Kp, const uint16_t* const* Vp, int n_layers,
                      const int32_t* parent, bool tree, const int32_t* block_table, int max_pages, int page_size,
                      int n_pages, const int32_t* kv_len, const int32_t* L, int B, int K, int Hq, int Hkv,
                      int head_dim, float softmax_scale, uint16_t* const* O, float* const* lse, void* workspace,
                      size_t ws_bytes, void* stream) {
  if (head_dim != 64 && head_dim != 128) return LIBRASPEC_EUNSUPPORTED;
  if (page_size < 64 || page_size % 64 != 0 || page_size > 65536) return LIBRASPEC_EUNSUPPORTED;
  if (max_pages < 1 || n_pages < 1 || (long)max_pages * page_size > 0x7fffffffL ||
      (long)n_pages * (Hkv > 0 ? Hkv : 1) > 0x7fffffffL || n_layers < 0)
    return LIBRASPEC_EINVAL;
  const int S_cap = max_pages * page_size;
  if (!attn_shapes_ok(B, K, Hq, Hkv, head_dim, S_cap, tree)) return LIBRASPEC_EINVAL;
  if (B == 0 || n_layers == 0) return LIBRASPEC_OK;
  if (!Q || !Kp || !Vp || !O || !kv_len || !L || !block_table || !aligned(block_table, 4)) return LIBRASPEC_EINVAL;
  if (tree && !parent) return LIBRASPEC_EINVAL;
  for (int l = 0; l < n_layers; ++l) {
    if (!Q[l] || !Kp[l] || !Vp[l] || !O[l]) return LIBRASPEC_EINVAL;
    if (!aligned(Q[l], 16) || !aligned(Kp[l], 16) || !aligned(Vp[l], 16) || !aligned(O[l], 16))
      return LIBRASPEC_EINVAL;
    if (lse && lse[l] && !aligned(lse[l], 4)) return LIBRASPEC_EINVAL;
  }
  if (!(softmax_scale > 0.f)) return LIBRASPEC_EINVAL;
  const WsLayout lay = ws_layout(B, K, 1, Hq, Hkv, head_dim, S_cap);
  if (!ws_ok(workspace, ws_bytes, lay)) return LIBRASPEC_EINVAL;
  return from_cuda(launch_verify_attn_paged_layers(Q, Kp, Vp, n_layers, parent, block_table, max_pages, page_size,
                                                   n_pages, kv_len, L, B, K, Hq, Hkv, head_dim, softmax_scale, O, lse,
                                                   static_cast<char*>(workspace), lay,
                                                   static_cast<cudaStream_t>(stream)));
}

}  // namespace

int libraspec_verify_attn_layers(const uint16_t* const* Q, const uint16_t* const* Kc, const uint16_t* const* Vc,
                                 int n_layers, const int32_t* kv_len, const int32_t* L, int B, int K, int Hq, int Hkv,
                                 int head_dim, int S_cap, float softmax_scale, uint16_t* const* O, float* const* lse,
                                 void* workspace, size_t ws_bytes, void* stream) {
  return attn_layers(Q, Kc, Vc, n_layers, nullptr, false, kv_len, L, B, K, Hq, Hkv, head_dim, S_cap, softmax_scale,
                     O, lse, workspace, ws_bytes, stream);
}

int libraspec_verify_attn_tree_layers(const uint16_t* const* Q, const uint16_t* const* Kc,
                                      const uint16_t* const* Vc, int n_layers, const int32_t* parent,
                                      const int32_t* kv_len, const int32_t* L, int B, int K, int Hq, int Hkv,
                                      int head_dim, int S_cap, float softmax_scale, uint16_t* const* O,
                                      float* const* lse, void* workspace, size_t ws_bytes, void* stream) {
  return attn_layers(Q, Kc, Vc, n_layers, parent, true, kv_len, L, B, K, Hq, Hkv, head_dim, S_cap, softmax_scale, O,
                     lse, workspace, ws_bytes, stream);
}

int libraspec_verify_attn_paged_layers(const uint16_t* const* Q, const uint16_t* const* Kp,
                                       const uint16_t* const* Vp, int n_layers, const int32_t* block_table,
                                       int max_pages, int page_size, int n_pages, const int32_t* kv_len,
                                       const int32_t* L, int B, int K, int Hq, int Hkv, int head_dim,
                                       float softmax_scale, uint16_t* const* O, float* const* lse, void* workspace,
                                       size_t ws_bytes, void* stream) {
  return attn_paged_layers(Q, Kp, Vp, n_layers, nullptr, false, block_table, max_pages, page_size, n_pages, kv_len, L,
                           B, K, Hq, Hkv, head_dim, softmax_scale, O, lse, workspace, ws_bytes, stream);
}

int libraspec_verify_attn_tree_paged_layers(const uint16_t* const* Q, const uint16_t* const* Kp,
                                            const uint16_t* const* Vp, int n_layers, const int32_t* parent,
                                            const int32_t* block_table, int max_pages, int page_size, int n_pages,
                                            const int32_t* kv_len, const int32_t* L, int B, int K, int Hq, int Hkv,
                                            int head_dim, float softmax_scale, uint16_t* const* O,
                                            float* const* lse, void* workspace, size_t ws_bytes, void* stream) {
  return attn_paged_layers(Q, Kp, Vp, n_layers, parent, true, block_table, max_pages, page_size, n_pages, kv_len, L,
                           B, K, Hq, Hkv, head_dim, softmax_scale, O, lse, workspace, ws_bytes, stream);
}

extern "C++" {
template <typename T>
static int accept_t(const T* target_logits, const T* draft_logits, const int32_t* draft_tokens, const float* conf,
                    const float* dstat, const int32_t* L, const float* temperature, int B, int K, int V, uint64_t seed,
                    uint64_t round_offset, uint32_t seq_offset, int32_t* n_accepted, int32_t* bonus_token,
                    void* workspace, size_t ws_bytes, void* stream, const uint64_t* rng = nullptr,
                    bool plan_ready = false) {
  if (!shapes_ok(B, K, V)) return LIBRASPEC_EINVAL;
  if (B == 0) return LIBRASPEC_OK;
  if (!target_logits || (!draft_logits && K > 0) || (!draft_tokens && K > 0) || !L || !temperature ||
      !n_accepted || !bonus_token)
    return LIBRASPEC_EINVAL;
  if (!aligned(target_logits, sizeof(T)) || (draft_logits && !aligned(draft_logits, sizeof(T))))
    return LIBRASPEC_EINVAL;
  const WsLayout lay = ws_layout(B, K, V, 1, 1, 64, 1);
  if (!ws_ok(workspace, ws_bytes, lay)) return LIBRASPEC_EINVAL;
  return from_cuda(launch_accept<T>(target_logits, draft_logits, draft_tokens, conf, dstat, L, temperature, B, K, V,
                                    seed, round_offset, seq_offset, n_accepted, bonus_token,
                                    static_cast<char*>(workspace), lay, static_cast<cudaStream_t>(stream), rng,
                                    plan_ready));
}
}  // extern "C++"

int libraspec_accept(const float* target_logits, const float* draft_logits, const int32_t* draft_tokens,
                     const float* conf, const float* dstat, const int32_t* L, const float* temperature, int B, int K,
                     int V, uint64_t seed, uint64_t round_offset, uint32_t seq_offset, int32_t* n_accepted,
                     int32_t* bonus_token, void* workspace, size_t ws_bytes, void* stream) {
  return accept_t(target_logits, draft_logits, draft_tokens, conf, dstat, L, temperature, B, K, V, seed,
                  round_offset, seq_offset, n_accepted, bonus_token, workspace, ws_bytes, stream);
}

int libraspec_accept_bf16(const uint16_t* target_logits, const uint16_t* draft_logits, const int32_t* draft_tokens,
                          const float* conf, const float* dstat, const int32_t* L, const float* temperature, int B,
                          int K, int V, uint64_t seed, uint64_t round_offset, uint32_t seq_offset,
                          int32_t* n_accepted, int32_t* bonus_token, void* workspace, size_t ws_bytes,
                          void* stream) {
  return accept_t(target_logits, draft_logits, draft_tokens, conf, dstat, L, temperature, B, K, V, seed,
                  round_offset, seq_offset, n_accepted, bonus_token, workspace, ws_bytes, stream);
}

namespace {

int kv_append_checked(const uint16_t* kv_new, uint16_t* const* Kc, uint16_t* const* Vc, int n_layers,
                      const int32_t* kv_len, const int32_t* block_table, int max_pages, int page_size, int n_pages,
                      int B, int T, int Hkv, int head_dim, int S_cap, void* workspace, size_t ws_bytes,
                      void* stream) {
  if (head_dim != 64 && head_dim != 128) return LIBRASPEC_EUNSUPPORTED;
  if (B < 0 || B > LIBRASPEC_MAX_B || T < 0 || T > LIBRASPEC_MAX_TREE_NODES + 1 || Hkv < 1 || n_layers < 0 ||
      S_cap < 1)
    return LIBRASPEC_EINVAL;
  if (B == 0 || T == 0 || n_layers == 0) return LIBRASPEC_OK;
  if (!kv_new || !aligned(kv_new, 16) || !Kc || !Vc || !kv_len) return LIBRASPEC_EINVAL;
  for (int l = 0; l < n_layers; ++l)
    if (!Kc[l] || !Vc[l] || !aligned(Kc[l], 16) || !aligned(Vc[l], 16)) return LIBRASPEC_EINVAL;
  if (!workspace || !aligned(workspace, 256) || ws_bytes < 256) return LIBRASPEC_EINVAL;
  return from_cuda(launch_kv_append(kv_new, Kc, Vc, n_layers, kv_len, block_table, max_pages, page_size, n_pages, B,
                                    T, Hkv, head_dim, S_cap, static_cast<int*>(workspace),
                                    static_cast<cudaStream_t>(stream)));
}

}  // namespace

size_t libraspec_lm_head_workspace_size(int M, int V) {
  if (M < 0 || M > (1 << 20) || V < 1) return 0;
  return lm_head_workspace_bytes(M, V);
}

int libraspec_lm_head_stats(const uint16_t* H, const uint16_t* W, const float* temperature, int rows_per_seq,
                            const int32_t* tokens, int M, int V, int Dm, float* row_stat, int32_t* row_argmax,
                            float* token_prob, void* workspace, size_t ws_bytes, void* stream) {
  if (M < 0 || M > (1 << 20) || V < 1 || rows_per_seq < 1) return LIBRASPEC_EINVAL;
  if (Dm < 64 || Dm % 64 != 0 || Dm > 65536) return LIBRASPEC_EUNSUPPORTED;
  if (M == 0) return LIBRASPEC_OK;
  if (!H || !W || !aligned(H, 16) || !aligned(W, 16)) return LIBRASPEC_EINVAL;
  if (token_prob && !tokens) return LIBRASPEC_EINVAL;
  if (!workspace || !aligned(workspace, 256) || ws_bytes < lm_head_workspace_bytes(M, V)) return LIBRASPEC_EINVAL;
  return from_cuda(launch_lm_head_stats(H, W, temperature, rows_per_seq, tokens, M, V, Dm, row_stat, row_argmax,
                                        token_prob, static_cast<char*>(workspace),
                                        static_cast<cudaStream_t>(stream)));
}

int libraspec_kv_append(const uint16_t* kv_new, uint16_t* const* Kc, uint16_t* const* Vc, int n_layers,
                        const int32_t* kv_len, int B, int T, int Hkv, int head_dim, int S_cap, void* workspace,
                        size_t ws_bytes, void* stream) {
  return kv_append_checked(kv_new, Kc, Vc, n_layers, kv_len, nullptr, 0, 0, 0, B, T, Hkv, head_dim, S_cap, workspace,
                           ws_bytes, stream);
}

int libraspec_kv_append_paged(const uint16_t* kv_new, uint16_t* const* Kp, uint16_t* const* Vp, int n_layers,
                              const int32_t* block_table, int max_pages, int page_size, int n_pages,
                              const int32_t* kv_len, int B, int T, int Hkv, int head_dim, void* workspace,
                              size_t ws_bytes, void* stream) {
  if (page_size < 1 || max_pages < 1 || n_pages < 1 || (long)max_pages * page_size > 0x7fffffffL) return LIBRASPEC_EINVAL;
  if (B > 0 && (!block_table || !aligned(block_table, 4))) return LIBRASPEC_EINVAL;
  return kv_append_checked(kv_new, Kp, Vp, n_layers, kv_len, block_table, max_pages, page_size, n_pages, B, T, Hkv,
                           head_dim, max_pages * page_size, workspace, ws_bytes, stream);
}

extern "C++" {
template <typename T>
static int accept_tree_t(const T* target_logits, const int32_t* draft_tokens, const int32_t* parent,
                         const int32_t* L, const float* temperature, int B, int K, int V, uint64_t seed,
                         uint64_t round_offset, uint32_t seq_offset, int32_t* n_accepted, int32_t* last_node,
                         int32_t* bonus_token, void* workspace, size_t ws_bytes, void* stream) {
  if (B < 0 || B > LIBRASPEC_MAX_B || K < 0 || K > LIBRASPEC_MAX_TREE_NODES || V < 1) return LIBRASPEC_EINVAL;
  if (B == 0) return LIBRASPEC_OK;
  if (!target_logits || (!draft_tokens && K > 0) || (!parent && K > 0) || !L || !n_accepted || !bonus_token)
    return LIBRASPEC_EINVAL;
  if (!aligned(target_logits, sizeof(T))) return LIBRASPEC_EINVAL;
  const WsLayout lay = ws_layout(B, K, V, 1, 1, 64, 1);
  if (!ws_ok(workspace, ws_bytes, lay)) return LIBRASPEC_EINVAL;
  return from_cuda(launch_accept_tree<T>(target_logits, draft_tokens, parent, L, temperature, B, K, V, seed,
                                         round_offset, seq_offset, n_accepted, last_node, bonus_token,
                                         static_cast<char*>(workspace), lay, static_cast<cudaStream_t>(stream)));
}
}  // extern "C++"

int libraspec_accept_tree_greedy(const float* target_logits, const int32_t* draft_tokens, const int32_t* parent,
                                 const int32_t* L, int B, int K, int V, int32_t* n_accepted, int32_t* last_node,
                                 int32_t* bonus_token, void* workspace, size_t ws_bytes, void* stream) {
  return accept_tree_t(target_logits, draft_tokens, parent, L, nullptr, B, K, V, 0, 0, 0, n_accepted, last_node,
                       bonus_token, workspace, ws_bytes, stream);
}

int libraspec_accept_tree_greedy_bf16(const uint16_t* target_logits, const int32_t* draft_tokens,
                                      const int32_t* parent, const int32_t* L, int B, int K, int V,
                                      int32_t* n_accepted, int32_t* last_node, int32_t* bonus_token, void* workspace,
                                      size_t ws_bytes, void* stream) {
  return accept_tree_t(target_logits, draft_tokens, parent, L, nullptr, B, K, V, 0, 0, 0, n_accepted, last_node,
                       bonus_token, workspace, ws_bytes, stream);
}

int libraspec_accept_tree(const float* target_logits, const int32_t* draft_tokens, const int32_t* parent,
                          const int32_t* L, const float* temperature, int B, int N, int V, uint64_t seed,
                          uint64_t round_offset, uint32_t seq_offset, int32_t* n_accepted, int32_t* last_node,
                          int32_t* bonus_token, void* workspace, size_t ws_bytes, void* stream) {
  if (!temperature && B > 0) return LIBRASPEC_EINVAL;
  return accept_tree_t(target_logits, draft_tokens, parent, L, temperature, B, N, V, seed, round_offset, seq_offset,
                       n_accepted, last_node, bonus_token, workspace, ws_bytes, stream);
}

int libraspec_accept_tree_bf16(const uint16_t* target_logits, const int32_t* draft_tokens, const int32_t* parent,
                               const int32_t* L, const float* temperature, int B, int N, int V, uint64_t seed,
                               uint64_t round_offset, uint32_t seq_offset, int32_t* n_accepted, int32_t* last_node,
                               int32_t* bonus_token, void* workspace, size_t ws_bytes, void* stream) {
  if (!temperature && B > 0) return LIBRASPEC_EINVAL;
  return accept_tree_t(target_logits, draft_tokens, parent, L, temperature, B, N, V, seed, round_offset, seq_offset,
                       n_accepted, last_node, bonus_token, workspace, ws_bytes, stream);
}

namespace {

// Inputs of a staged round: three host parts copied in on copy_stream (the
// drafter part, then the layers' queries and new keys/values, then the
// target rows), each step of the round waiting only for its part; the block's
// keys and values appended from kv_new; results read back into host memory.
struct Staged {
  const void* const* host_parts;
  void* const* dev_parts;
  const size_t* part_bytes;
  cudaStream_t copy_stream;
  const uint16_t* kv_new;
  int32_t* n_host;
  int32_t* bonus_host;
  const uint64_t* rng_dev;  // {seed, round_offset, seq_offset} inside part 2 on the device
  cudaEvent_t ev[4];
};

// Creates the events, orders copy_stream after the work already on `s` and
// enqueues the three copies, recording one event after each.
int staged_begin(Staged* st, cudaStream_t s) {
  for (int i = 0; i < 4; ++i) st->ev[i] = nullptr;
  for (int i = 0; i < 4; ++i)
    if (cudaEventCreateWithFlags(&st->ev[i], cudaEventDisableTiming) != cudaSuccess) return LIBRASPEC_ECUDA;
  cudaError_t e = cudaEventRecord(st->ev[3], s);
  if (e == cudaSuccess) e = cudaStreamWaitEvent(st->copy_stream, st->ev[3], 0);
  for (int i = 0; i < 3 && e == cudaSuccess; ++i) {
    if (st->part_bytes[i] > 0)
      e = cudaMemcpyAsync(st->dev_parts[i], st->host_parts[i], st->part_bytes[i], cudaMemcpyHostToDevice,
                          st->copy_stream);
    if (e == cudaSuccess) e = cudaEventRecord(st->ev[i], st->copy_stream);
  }
  return from_cuda(e);
}

void staged_end(Staged* st) {
  for (int i = 0; i < 4; ++i)
    if (st->ev[i]) cudaEventDestroy(st->ev[i]);  // released once the recorded work completes
}

int staged_wait(const Staged* st, int part, cudaStream_t s) {
  return st ? from_cuda(cudaStreamWaitEvent(s, st->ev[part], 0)) : LIBRASPEC_OK;
}

}  // namespace

extern "C++" {
template <typename T>
static int verify_round_t(const T* draft_logits, const int32_t* draft_tokens, const float* temperature,
                           const float* cost_table, const T* target_logits, const uint16_t* const* Q,
                           const uint16_t* const* Kc, const uint16_t* const* Vc, uint16_t* const* O,
                           float* const* lse, int n_layers, const int32_t* kv_len, int B, int K, int V, int Hq,
                           int Hkv, int head_dim, int S_cap, float softmax_scale, uint64_t seed,
                           uint64_t round_offset, uint32_t seq_offset, float* conf, float* dstat, int32_t* L,
                           int32_t* n_accepted, int32_t* bonus_token, void* workspace, size_t ws_bytes,
                           void* stream, Staged* st = nullptr) {
  if (!shapes_ok(B, K, V) || n_layers < 0) return LIBRASPEC_EINVAL;
  if (head_dim != 64 && head_dim != 128) return LIBRASPEC_EUNSUPPORTED;
  if (!attn_shapes_ok(B, K, Hq, Hkv, head_dim, S_cap)) return LIBRASPEC_EINVAL;
  if (B == 0) return LIBRASPEC_OK;
  if (n_layers > 0 && (!Q || !Kc || !Vc || !O)) return LIBRASPEC_EINVAL;
  if (!conf || !dstat || !L || !kv_len) return LIBRASPEC_EINVAL;
  const WsLayout lay = ws_layout(B, K, V, Hq, Hkv, head_dim, S_cap);
  if (!ws_ok(workspace, ws_bytes, lay)) return LIBRASPEC_EINVAL;
  for (int l = 0; l < n_layers; ++l) {
    if (!Q[l] || !Kc[l] || !Vc[l] || !O[l]) return LIBRASPEC_EINVAL;
    if (!aligned(Q[l], 16) || !aligned(Kc[l], 16) || !aligned(Vc[l], 16) || !aligned(O[l], 16))
      return LIBRASPEC_EINVAL;
  }
  if (!(softmax_scale > 0.f)) return LIBRASPEC_EINVAL;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  char* ws = static_cast<char*>(workspace);
  int rc = LIBRASPEC_OK;
  if (st && (rc = staged_begin(st, s)) != LIBRASPEC_OK) return rc;
  if ((rc = staged_wait(st, 0, s)) != LIBRASPEC_OK) return rc;
  if (!cost_table) return LIBRASPEC_EINVAL;
  if (K > 0) {  // confidence, and the selection in the same launch
    rc = confidence_t(draft_logits, draft_tokens, temperature, B, K, V, conf, dstat, workspace, ws_bytes, stream,
                      cost_table, L);
  } else {
    rc = from_cuda(launch_select(conf, cost_table, B, K, L, ws, lay, s));
  }
  if (rc != LIBRASPEC_OK) return rc;
  // the acceptance plan needs only L and the temperatures: it runs here, off
  // the acceptance's critical path
  const bool plan = target_logits != nullptr && (draft_logits != nullptr || K == 0) && aligned(target_logits, sizeof(T));
  if (plan && (rc = from_cuda(launch_accept_plan<T>(target_logits, draft_logits, conf, dstat, L, temperature, B, K,
                                                    V, n_accepted, bonus_token, ws, lay, s))) != LIBRASPEC_OK)
    return rc;
  if ((rc = staged_wait(st, 1, s)) != LIBRASPEC_OK) return rc;
  if (st && (rc = from_cuda(launch_kv_append(st->kv_new, const_cast<uint16_t* const*>(Kc),
                                             const_cast<uint16_t* const*>(Vc), n_layers, kv_len, nullptr, 0, 0, 0, B,
                                             K + 1, Hkv, head_dim, S_cap, reinterpret_cast<int*>(ws + lay.status),
                                             s))) != LIBRASPEC_OK)
    return rc;
  rc = from_cuda(launch_verify_attn_layers(Q, Kc, Vc, n_layers, nullptr, kv_len, L, B, K, Hq, Hkv, head_dim, S_cap,
                                           softmax_scale, O, lse, ws, lay, s));
  if (rc != LIBRASPEC_OK) return rc;
  if ((rc = staged_wait(st, 2, s)) != LIBRASPEC_OK) return rc;
  rc = accept_t(target_logits, draft_logits, draft_tokens, conf, dstat, L, temperature, B, K, V, seed, round_offset,
                seq_offset, n_accepted, bonus_token, workspace, ws_bytes, stream, st ? st->rng_dev : nullptr, plan);
  if (rc != LIBRASPEC_OK || !st) return rc;
  cudaError_t e = cudaMemcpyAsync(st->n_host, n_accepted, sizeof(int32_t) * B, cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaMemcpyAsync(st->bonus_host, bonus_token, sizeof(int32_t) * B, cudaMemcpyDeviceToHost, s);
  return from_cuda(e);
}

// A staged round replays as one CUDA graph: the first call with a set of
// buffers and shapes runs eagerly, the second captures the round (copies,
// events, kernels, read-back) on the caller's stream and keeps the
// instantiated graph; later calls with the same set launch it. The generator
// arguments travel in part 2 (rng_host -> rng_dev), so a graph serves every
// seed and round. One cached graph per thread.
inline uintptr_t float_bits(float f) {
  uint32_t u;
  memcpy(&u, &f, sizeof(u));
  return u;
}

struct StagedGraph {
  std::vector<uintptr_t> key;
  int seen = 0;
  cudaGraphExec_t exec = nullptr;
};

template <typename T>
static int verify_round_staged_t(const void* const* host_parts, void* const* dev_parts, const size_t* part_bytes,
                                 void* copy_stream, const uint16_t* kv_new, uint64_t* rng_host,
                                 const uint64_t* rng_dev, int32_t* n_accepted_host, int32_t* bonus_host,
                                 const T* draft_logits, const int32_t* draft_tokens, const float* temperature,
                                 const float* cost_table, const T* target_logits, const uint16_t* const* Q,
                                 uint16_t* const* Kc, uint16_t* const* Vc, uint16_t* const* O, int n_layers,
                                 const int32_t* kv_len, int B, int K, int V, int Hq, int Hkv, int head_dim,
                                 int S_cap, float softmax_scale, uint64_t seed, uint64_t round_offset,
                                 uint32_t seq_offset, float* conf, float* dstat, int32_t* L, int32_t* n_accepted,
                                 int32_t* bonus_token, void* workspace, size_t ws_bytes, void* stream) {
  if (!host_parts || !dev_parts || !part_bytes || !n_accepted_host || !bonus_host || !n_accepted || !bonus_token ||
      !rng_host || !rng_dev || !aligned(rng_dev, 8))
    return LIBRASPEC_EINVAL;
  for (int i = 0; i < 3; ++i)
    if (part_bytes[i] > 0 && (!host_parts[i] || !dev_parts[i])) return LIBRASPEC_EINVAL;
  if (n_layers > 0 && (!kv_new || !aligned(kv_new, 16) || !Q || !Kc || !Vc || !O)) return LIBRASPEC_EINVAL;
  if (n_layers < 0 || n_layers > 4096) return LIBRASPEC_EINVAL;
  const uintptr_t fixed[] = {
      (uintptr_t)host_parts[0], (uintptr_t)host_parts[1], (uintptr_t)host_parts[2], (uintptr_t)dev_parts[0],
      (uintptr_t)dev_parts[1], (uintptr_t)dev_parts[2], part_bytes[0], part_bytes[1], part_bytes[2],
      (uintptr_t)copy_stream, (uintptr_t)kv_new, (uintptr_t)rng_dev, (uintptr_t)n_accepted_host,
      (uintptr_t)bonus_host, (uintptr_t)draft_logits, (uintptr_t)draft_tokens, (uintptr_t)temperature,
      (uintptr_t)cost_table, (uintptr_t)target_logits, (uintptr_t)n_layers, (uintptr_t)kv_len, (uintptr_t)B,
      (uintptr_t)K, (uintptr_t)V, (uintptr_t)Hq, (uintptr_t)Hkv, (uintptr_t)head_dim, (uintptr_t)S_cap,
      float_bits(softmax_scale), (uintptr_t)conf, (uintptr_t)dstat, (uintptr_t)L,
      (uintptr_t)n_accepted, (uintptr_t)bonus_token, (uintptr_t)workspace, ws_bytes, (uintptr_t)stream,
      (uintptr_t)sizeof(T)};
  std::vector<uintptr_t> key(fixed, fixed + sizeof(fixed) / sizeof(fixed[0]));
  for (int l = 0; l < n_layers; ++l) {
    key.push_back((uintptr_t)Q[l]);
    key.push_back((uintptr_t)Kc[l]);
    key.push_back((uintptr_t)Vc[l]);
    key.push_back((uintptr_t)O[l]);
  }
  // the generator arguments of this round, copied in with part 2
  rng_host[0] = seed;
  rng_host[1] = round_offset;
  rng_host[2] = seq_offset;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  static thread_local StagedGraph cache;
  if (cache.exec && cache.key == key) return from_cuda(cudaGraphLaunch(cache.exec, s));
  const bool capture = cache.key == key && cache.seen >= 1;
  if (cache.key != key) {
    if (cache.exec) cudaGraphExecDestroy(cache.exec);
    cache.exec = nullptr;
    cache.key = key;
    cache.seen = 0;
  }
  ++cache.seen;
  Staged st{host_parts, dev_parts, part_bytes, static_cast<cudaStream_t>(copy_stream), kv_new, n_accepted_host,
            bonus_host, rng_dev, {}};
  bool capturing = false;
  if (capture) {
    // not possible on the legacy default stream, for one: then this set of
    // buffers always runs eagerly
    capturing = cudaStreamBeginCapture(s, cudaStreamCaptureModeThreadLocal) == cudaSuccess;
    if (!capturing) {
      cudaGetLastError();
      cache.seen = -(1 << 30);
    }
  }
  if (capturing) {
    int rc = verify_round_t(draft_logits, draft_tokens, temperature, cost_table, target_logits, Q,
                            const_cast<const uint16_t* const*>(Kc), const_cast<const uint16_t* const*>(Vc), O,
                            nullptr, n_layers, kv_len, B, K, V, Hq, Hkv, head_dim, S_cap, softmax_scale, seed,
                            round_offset, seq_offset, conf, dstat, L, n_accepted, bonus_token, workspace, ws_bytes,
                            stream, &st);
    cudaGraph_t graph = nullptr;
    const cudaError_t e = cudaStreamEndCapture(s, &graph);
    staged_end(&st);
    cudaGraphExec_t exec = nullptr;
    if (rc == LIBRASPEC_OK && e == cudaSuccess && graph &&
        cudaGraphInstantiate(&exec, graph, 0) == cudaSuccess) {
      cudaGraphDestroy(graph);
      cache.exec = exec;
      return from_cuda(cudaGraphLaunch(exec, s));
    }
    if (graph) cudaGraphDestroy(graph);
    cudaGetLastError();  // the failed capture's error; run the round eagerly below, and from now on
    cache.seen = -(1 << 30);
    st = Staged{host_parts, dev_parts, part_bytes, static_cast<cudaStream_t>(copy_stream), kv_new, n_accepted_host,
                bonus_host, rng_dev, {}};
  }
  const int rc = verify_round_t(draft_logits, draft_tokens, temperature, cost_table, target_logits, Q,
                                const_cast<const uint16_t* const*>(Kc), const_cast<const uint16_t* const*>(Vc), O,
                                nullptr, n_layers, kv_len, B, K, V, Hq, Hkv, head_dim, S_cap, softmax_scale, seed,
                                round_offset, seq_offset, conf, dstat, L, n_accepted, bonus_token, workspace,
                                ws_bytes, stream, &st);
  staged_end(&st);
  return rc;
}
}  // extern "C++"

int libraspec_verify_round_staged(const void* const* host_parts, void* const* dev_parts, const size_t* part_bytes,
                                  void* copy_stream, const uint16_t* kv_new, uint64_t* rng_host,
                                  const uint64_t* rng_dev, int32_t* n_accepted_host, int32_t* bonus_host, const float* draft_logits, const int32_t* draft_tokens,
                                  const float* temperature, const float* cost_table, const float* target_logits,
                                  const uint16_t* const* Q, uint16_t* const* Kc, uint16_t* const* Vc,
                                  uint16_t* const* O, int n_layers, const int32_t* kv_len, int B, int K, int V,
                                  int Hq, int Hkv, int head_dim, int S_cap, float softmax_scale, uint64_t seed,
                                  uint64_t round_offset, uint32_t seq_offset, float* conf, float* dstat, int32_t* L,
                                  int32_t* n_accepted, int32_t* bonus_token, void* workspace, size_t ws_bytes,
                                  void* stream) {
  return verify_round_staged_t(host_parts, dev_parts, part_bytes, copy_stream, kv_new, rng_host, rng_dev,
                               n_accepted_host, bonus_host,
                               draft_logits, draft_tokens, temperature, cost_table, target_logits, Q, Kc, Vc, O,
                               n_layers, kv_len, B, K, V, Hq, Hkv, head_dim, S_cap, softmax_scale, seed, round_offset,
                               seq_offset, conf, dstat, L, n_accepted, bonus_token, workspace, ws_bytes, stream);
}

int libraspec_verify_round_staged_bf16(const void* const* host_parts, void* const* dev_parts,
                                       const size_t* part_bytes, void* copy_stream, const uint16_t* kv_new,
                                       uint64_t* rng_host, const uint64_t* rng_dev, int32_t* n_accepted_host,
                                       int32_t* bonus_host, const uint16_t* draft_logits,
                                       const int32_t* draft_tokens, const float* temperature,
                                       const float* cost_table, const uint16_t* target_logits,
                                       const uint16_t* const* Q, uint16_t* const* Kc, uint16_t* const* Vc,
                                       uint16_t* const* O, int n_layers, const int32_t* kv_len, int B, int K, int V,
                                       int Hq, int Hkv, int head_dim, int S_cap, float softmax_scale, uint64_t seed,
                                       uint64_t round_offset, uint32_t seq_offset, float* conf, float* dstat,
                                       int32_t* L, int32_t* n_accepted, int32_t* bonus_token, void* workspace,
                                       size_t ws_bytes, void* stream) {
  return verify_round_staged_t(host_parts, dev_parts, part_bytes, copy_stream, kv_new, rng_host, rng_dev,
                               n_accepted_host, bonus_host,
                               draft_logits, draft_tokens, temperature, cost_table, target_logits, Q, Kc, Vc, O,
                               n_layers, kv_len, B, K, V, Hq, Hkv, head_dim, S_cap, softmax_scale, seed, round_offset,
                               seq_offset, conf, dstat, L, n_accepted, bonus_token, workspace, ws_bytes, stream);
}

int libraspec_verify_round(const float* draft_logits, const int32_t* draft_tokens, const float* temperature,
                           const float* cost_table, const float* target_logits, const uint16_t* const* Q,
                           const uint16_t* const* Kc, const uint16_t* const* Vc, uint16_t* const* O,
                           float* const* lse, int n_layers, const int32_t* kv_len, int B, int K, int V, int Hq,
                           int Hkv, int head_dim, int S_cap, float softmax_scale, uint64_t seed,
                           uint64_t round_offset, uint32_t seq_offset, float* conf, float* dstat, int32_t* L,
                           int32_t* n_accepted, int32_t* bonus_token, void* workspace, size_t ws_bytes,
                           void* stream) {
  return verify_round_t(draft_logits, draft_tokens, temperature, cost_table, target_logits, Q, Kc, Vc, O, lse,
                        n_layers, kv_len, B, K, V, Hq, Hkv, head_dim, S_cap, softmax_scale, seed, round_offset,
                        seq_offset, conf, dstat, L, n_accepted, bonus_token, workspace, ws_bytes, stream);
}

int libraspec_verify_round_bf16(const uint16_t* draft_logits, const int32_t* draft_tokens, const float* temperature,
                                const float* cost_table, const uint16_t* target_logits, const uint16_t* const* Q,
                                const uint16_t* const* Kc, const uint16_t* const* Vc, uint16_t* const* O,
                                float* const* lse, int n_layers, const int32_t* kv_len, int B, int K, int V, int Hq,
                                int Hkv, int head_dim, int S_cap, float softmax_scale, uint64_t seed,
                                uint64_t round_offset, uint32_t seq_offset, float* conf, float* dstat, int32_t* L,
                                int32_t* n_accepted, int32_t* bonus_token, void* workspace, size_t ws_bytes,
                                void* stream) {
  return verify_round_t(draft_logits, draft_tokens, temperature, cost_table, target_logits, Q, Kc, Vc, O, lse,
                        n_layers, kv_len, B, K, V, Hq, Hkv, head_dim, S_cap, softmax_scale, seed, round_offset,
                        seq_offset, conf, dstat, L, n_accepted, bonus_token, workspace, ws_bytes, stream);
}

}  // extern "C"
