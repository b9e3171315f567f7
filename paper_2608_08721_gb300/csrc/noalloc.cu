// libraspec_confidence_noalloc: the drafter-confidence step for callers that
// cannot allocate device memory. Its scratch (the split-row partials, the
// per-row merge tickets and the status word) lives in one file-scope
// __device__ array of fixed size instead of a caller workspace; the kernels
// are the ones libraspec_confidence launches.
#include <atomic>
#include <mutex>

#include "common.cuh"

namespace libraspec {

template <typename T>
cudaError_t launch_confidence(const T*, const int32_t*, const float*, int, int, int, float*, float*, char*,
                              const WsLayout&, cudaStream_t, const float*, int32_t*);

namespace {

constexpr size_t kNoAllocRows = LIBRASPEC_NOALLOC_MAX_ROWS;
// [status 256 B][tickets: one u32 per row][partials: kConfMaxSplits per row]
constexpr size_t kCntOff = 256;
constexpr size_t kPartOff = kCntOff + ((kNoAllocRows * sizeof(uint32_t) + 255) & ~size_t(255));
constexpr size_t kScratchBytes = kPartOff + kNoAllocRows * kConfMaxSplits * sizeof(RowPartial);

__device__ __align__(256) char g_noalloc_scratch[kScratchBytes];

constexpr int kMaxDevices = 64;
// per device: the CUDA context the address was looked up in, and the address
struct ScratchAddr {
  std::atomic<void*> ctx{nullptr};
  std::atomic<char*> addr{nullptr};
};
ScratchAddr g_scratch_addr[kMaxDevices];
std::mutex g_setup_mu;

// The driver's cuCtxGetCurrent, resolved once.
typedef int (*CtxGetCurrentFn)(void**);
CtxGetCurrentFn ctx_get_current() {
  static std::atomic<CtxGetCurrentFn> fn{nullptr};
  CtxGetCurrentFn f = fn.load(std::memory_order_acquire);
  if (!f) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess) {
      f = reinterpret_cast<CtxGetCurrentFn>(p);
      fn.store(f, std::memory_order_release);
    }
  }
  return f;
}

// Address of the scratch array on the current device, looked up once per
// device and context (cudaGetSymbolAddress, with that device current). A new
// context on the device (after cudaDeviceReset, say) reloads the module, so
// the address is looked up again.
cudaError_t scratch_on_current_device(char** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  CtxGetCurrentFn get = ctx_get_current();
  if (!get) return cudaErrorDeviceUninitialized;
  void* ctx = nullptr;
  if (get(&ctx) != 0) return cudaErrorDeviceUninitialized;  // null: no context current yet
  ScratchAddr& slot = g_scratch_addr[dev];
  char* p = slot.addr.load(std::memory_order_acquire);
  if (!p || !ctx || slot.ctx.load(std::memory_order_acquire) != ctx) {
    std::lock_guard<std::mutex> lock(g_setup_mu);
    p = slot.addr.load(std::memory_order_relaxed);
    if (!p || !ctx || slot.ctx.load(std::memory_order_relaxed) != ctx) {
      // the lookup makes the device's primary context current if none was
      void* a = nullptr;
      e = cudaGetSymbolAddress(&a, g_noalloc_scratch);
      if (e != cudaSuccess) return e;
      if (get(&ctx) != 0 || !ctx) return cudaErrorDeviceUninitialized;
      p = static_cast<char*>(a);
      slot.addr.store(nullptr, std::memory_order_release);
      slot.ctx.store(ctx, std::memory_order_release);
      slot.addr.store(p, std::memory_order_release);
    }
  }
  *out = p;
  return cudaSuccess;
}

}  // namespace
}  // namespace libraspec

using namespace libraspec;

extern "C" int libraspec_confidence_noalloc(const float* draft_logits, const int32_t* draft_tokens,
                                            const float* temperature, int B, int K, int V, float* conf,
                                            float* dstat, int32_t* status, void* stream) {
  if (B < 0 || B > LIBRASPEC_MAX_B || K < 0 || K > LIBRASPEC_MAX_K || V < 1) return LIBRASPEC_EINVAL;
  const size_t rows = (size_t)B * K;
  if (rows > kNoAllocRows) return LIBRASPEC_EUNSUPPORTED;
  if (rows == 0) return LIBRASPEC_OK;
  if (!draft_logits || !draft_tokens || !temperature || !conf) return LIBRASPEC_EINVAL;
  if ((reinterpret_cast<uintptr_t>(draft_logits) & 3) || (reinterpret_cast<uintptr_t>(conf) & 3) ||
      (reinterpret_cast<uintptr_t>(dstat) & 3) || (reinterpret_cast<uintptr_t>(status) & 3))
    return LIBRASPEC_EINVAL;
  char* scratch = nullptr;
  if (scratch_on_current_device(&scratch) != cudaSuccess) return LIBRASPEC_ECUDA;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // the status word and this call's tickets start at zero
  cudaError_t e = cudaMemsetAsync(scratch, 0, kCntOff + rows * sizeof(uint32_t), s);
  if (e != cudaSuccess) return LIBRASPEC_ECUDA;
  WsLayout lay{};
  lay.status = 0;
  lay.conf_cnt = kCntOff;
  lay.conf_part = kPartOff;
  e = launch_confidence(draft_logits, draft_tokens, temperature, B, K, V, conf, dstat, scratch, lay, s,
                        static_cast<const float*>(nullptr), nullptr);
  if (e != cudaSuccess) return LIBRASPEC_ECUDA;
  if (status) {
    e = cudaMemcpyAsync(status, scratch, sizeof(int32_t), cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess) return LIBRASPEC_ECUDA;
  }
  return LIBRASPEC_OK;
}
