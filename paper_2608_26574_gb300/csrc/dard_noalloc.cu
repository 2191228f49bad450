// dard_noalloc.cu - dard_score_and_transition_noalloc: the scoring call with its scratch in a
// fixed array inside the library, for callers that cannot hand device memory to it.
//
// The scoring scratch is three counters per sequence (zero between calls) and two bytes
// per block row (the promotion / demotion outcome of each C row, and each row's new
// state). Here it is a file-scope __device__ array sized for DARD_SCORE_NOALLOC_MAX_ROWS
// rows and DARD_MAX_SEQS sequences. Its address on a device is looked up once
// (cudaGetSymbolAddress, with that device current) on the first call made on that device,
// cached per device together with the context it belongs to (looked up again when the
// current context changes), and then passed as the workspace of dard_score_and_transition, whose
// kernels and validation run unchanged. Every call first clears the counters with an
// asynchronous memset on its stream, so a call never depends on what an earlier one left
// behind. No call allocates or frees device memory.
#include <mutex>

#include "dard_internal.h"


namespace {

// score_workspace_bytes(DARD_SCORE_NOALLOC_MAX_ROWS, DARD_MAX_SEQS): counters, then the
// outcome and new-state bytes, each part 256-byte aligned
constexpr size_t kScratchBytes = ((3 * 4 * DARD_MAX_SEQS + 255) / 256) * 256 +
                                 2 * (((DARD_SCORE_NOALLOC_MAX_ROWS + 255) / 256) * 256);
__device__ __align__(256) uint8_t g_score_scratch[kScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
void* g_scratch_ptr[kMaxDevices] = {};
void* g_scratch_ctx[kMaxDevices] = {};  // the context the cached address belongs to

// The current CUDA context (driver entry point, so that the library needs no -lcuda).
cudaError_t current_context(void** ctx) {
  using GetCurrent = int (*)(void**);
  static GetCurrent fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<GetCurrent>(f);
  });
  if (fn == nullptr) return cudaErrorNotSupported;
  return fn(ctx) == 0 ? cudaSuccess : cudaErrorUnknown;
}

// Device address of g_score_scratch on the current device: looked up on the first call in
// a context, and again whenever the current context has changed (a device reset or a new
// primary context loads the module again, at another address).
cudaError_t scratch_on_current_device(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  void* ctx = nullptr;
  e = current_context(&ctx);  // NULL before the runtime has initialised the device
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (g_scratch_ptr[dev] == nullptr || ctx == nullptr || g_scratch_ctx[dev] != ctx) {
    void* ptr = nullptr;
    e = cudaGetSymbolAddress(&ptr, g_score_scratch);  // initialises the context if needed
    if (e != cudaSuccess) return e;
    if (ptr == nullptr) return cudaErrorInvalidSymbol;
    e = current_context(&ctx);
    if (e != cudaSuccess) return e;
    g_scratch_ptr[dev] = ptr;
    g_scratch_ctx[dev] = ctx;
  }
  *out = g_scratch_ptr[dev];
  return cudaSuccess;
}

}  // namespace

extern "C" dard_status dard_score_and_transition_noalloc(const dard_score_args* a, void* stream) {
  using namespace dard;
  if (!a) return report(DARD_ERR_NULL, "args is NULL");
  // Sizes that dard_score_and_transition itself rejects are passed on to it for its message.
  long long rows = 0;
  bool sizes_ok = a->block_len != nullptr && a->num_seqs >= 1 && a->num_seqs <= DARD_MAX_SEQS;
  for (int s = 0; sizes_ok && s < a->num_seqs; ++s) {
    const int B = a->block_len[s];
    sizes_ok = B >= 0 && B <= DARD_MAX_BLOCK;
    rows += B;
  }
  dard_score_args b = *a;
  b.workspace = nullptr;
  b.workspace_bytes = 0;
  if (sizes_ok && rows > 0) {
    if (rows > DARD_SCORE_NOALLOC_MAX_ROWS)
      return report(DARD_ERR_WORKSPACE,
                    "%lld block rows exceed the %d rows the built-in scratch of "
                    "dard_score_and_transition_noalloc holds; use dard_score_and_transition "
                    "with a workspace",
                    rows, DARD_SCORE_NOALLOC_MAX_ROWS);
    void* scratch = nullptr;
    const cudaError_t e = scratch_on_current_device(&scratch);
    if (e != cudaSuccess)
      return report(DARD_ERR_CUDA, "looking up the built-in scratch failed: %s",
                    cudaGetErrorString(e));
    b.workspace = scratch;
    b.workspace_bytes = sizeof(g_score_scratch);
  }
  ScoreParams p;
  const dard_status st = prepare_score(&b, p);
  if (st != DARD_OK) return st;
  if (b.workspace != nullptr) {
    // the counters start at zero on every call (cudaMemsetAsync allocates nothing)
    const cudaError_t m = cudaMemsetAsync(b.workspace, 0, score_counter_bytes(b.num_seqs),
                                          static_cast<cudaStream_t>(stream));
    if (m != cudaSuccess)
      return report(DARD_ERR_CUDA, "clearing the built-in scratch failed: %s",
                    cudaGetErrorString(m));
  }
  char err[256];
  const dard_status ls = launch_score(b, p, static_cast<cudaStream_t>(stream), err, sizeof(err));
  if (ls != DARD_OK) return report(ls, "%s", err);
  return DARD_OK;
}
