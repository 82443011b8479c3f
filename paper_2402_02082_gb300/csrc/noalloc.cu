// glide_cross_attn_noalloc: GliDe cross-attention for callers that cannot
// allocate device memory when they call us.
//
// Typical such callers: an engine plugin whose enqueue path is forbidden to
// allocate because the host engine owns and budgets all device memory, or a
// serving loop that has handed nearly all of HBM to its KV cache and bans
// allocator calls on its per-token path (an allocation there can block,
// fragment the pool, or fail at the worst moment).  They still own their
// inputs and outputs, but have no workspace to lend.
//
// This entry point keeps the scratch that glide_cross_attn takes as a
// workspace (status word, per-(b,h) arrival counters, split partials) in one
// fixed-size array in the library's own device memory instead.  Its size,
// kScratchBytes, is reserved on every GPU that loads the library until the
// process exits.  Nothing here calls cudaMalloc, cudaFree or any allocating
// library routine.
#include <cuda_runtime.h>

#include "../../include/glide.h"
#include "common.cuh"
#include "kernels.h"

namespace {

constexpr size_t kScratchBytes = 32u << 20;  // 32 MiB per GPU

// The scratch itself.  In host code this name is only a host-side stand-in
// for the symbol, never a device address: host code obtains the real address
// with cudaGetSymbolAddress (below) and passes that to the kernel.
static __device__ __align__(256) unsigned char g_scratch[kScratchBytes];

// Device address of g_scratch in the current device's context.  Looked up on
// every call (a lookup allocates nothing and enqueues nothing), so a context
// that was torn down and created again, after cudaDeviceReset for instance,
// gets the array's new address, never a stale one.  The first lookup on a
// device loads the library's device code there.
cudaError_t scratch_address(void** out) {
  void* p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_scratch);
  if (e != cudaSuccess) return e;
  if (p == nullptr) return cudaErrorInvalidSymbol;
  *out = p;
  return cudaSuccess;
}

}  // namespace

extern "C" glide_status glide_cross_attn_noalloc(const glide_attn_desc* desc, const void* q_draft,
                                                 const void* K_cache, const void* V_cache,
                                                 const int32_t* kv_len, int32_t max_kv_len, float* out,
                                                 glide_stream_t stream) {
  // The same workspace glide_cross_attn would need; reject shapes whose
  // scratch would not fit in the fixed array.
  const size_t need = glide_attn_workspace_bytes(desc, 1);
  if (need == 0) return GLIDE_ERR_INVALID;
  if (need > kScratchBytes) return GLIDE_ERR_UNSUPPORTED;
  void* scratch = nullptr;
  if (scratch_address(&scratch) != cudaSuccess) return GLIDE_ERR_CUDA;
  // The array keeps whatever the previous call left.  The counters after the
  // status word must start at zero; the status word itself (bytes 0..3) is
  // left alone, so a wait that ran out in an earlier call stays reported
  // until glide_noalloc_read_device_status reads and clears it.
  // (cudaMemsetAsync does not allocate.)
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const size_t first = glide::WsLayout::kClaimOff;
  const size_t zeroed = glide::WsLayout::partials_off(desc->B, desc->H) - first;
  if (cudaMemsetAsync(static_cast<unsigned char*>(scratch) + first, 0, zeroed, st) != cudaSuccess)
    return GLIDE_ERR_CUDA;
  return glide_cross_attn(desc, q_draft, K_cache, V_cache, kv_len, max_kv_len, out, scratch, kScratchBytes,
                          stream);
}

extern "C" glide_status glide_noalloc_read_device_status(glide_stream_t stream) {
  void* scratch = nullptr;
  if (scratch_address(&scratch) != cudaSuccess) return GLIDE_ERR_CUDA;
  return glide_read_device_status(scratch, stream);
}

extern "C" glide_status glide_noalloc_scratch(void** device_ptr) {
  if (!device_ptr) return GLIDE_ERR_INVALID;
  return scratch_address(device_ptr) == cudaSuccess ? GLIDE_OK : GLIDE_ERR_CUDA;
}
