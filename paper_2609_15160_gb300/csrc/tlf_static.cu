// tlf_attn_decode_static: the recursion-wise decode attention for callers
// that cannot allocate device memory (declared in include/tlf.h).
//
// Same kernels and results as tlf_attn_decode; the scratch (work plan and
// split-K partials) is a fixed array in the library's device image instead
// of a caller buffer. Host code cannot use the array's name as a device
// address, so the first call on each device looks the address up with
// cudaGetSymbolAddress while that device is current and remembers it, keyed
// by the device and by the id of its current CUDA context: a context that is
// torn down and re-created (cudaDeviceReset, for one) loads the module again,
// possibly elsewhere, and gets a new id, so the next call looks again instead
// of handing the kernels a stale address.
#include <atomic>
#include <cstdio>
#include <mutex>

#include "tlf.h"
#include "tlf_internal.cuh"

// 4 MiB on every GPU that loads the library, held until the process exits.
static constexpr size_t kStaticScratchBytes = size_t(4) << 20;
static __device__ __align__(256) uint8_t g_static_scratch[kStaticScratchBytes];

namespace {
std::mutex g_scratch_mu;
constexpr int kMaxDevices = 64;
struct ScratchEntry {
  unsigned long long ctx_id = 0;  // CUDA context the address belongs to
  void* addr = nullptr;
};
ScratchEntry g_scratch[kMaxDevices];

// Device address of g_static_scratch in the current device's current context (looked up
// once per device and context).
int static_scratch_address(void** out) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return tlf::set_thread_error(TLF_ERR_CUDA, cudaGetErrorString(e));
  if (dev < 0 || dev >= kMaxDevices) return tlf::set_thread_error(TLF_ERR_CUDA, "device ordinal out of range");
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  ScratchEntry& ent = g_scratch[dev];
  unsigned long long id = 0;
  const bool have_id = tlf::current_context_id(&id);
  if (!have_id || !ent.addr || ent.ctx_id != id) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_static_scratch);  // makes the runtime's context current if none was
    if (e != cudaSuccess || !p)
      return tlf::set_thread_error(TLF_ERR_CUDA, e != cudaSuccess ? cudaGetErrorString(e)
                                                                  : "cudaGetSymbolAddress returned NULL");
    if (!tlf::current_context_id(&id))
      return tlf::set_thread_error(TLF_ERR_CUDA, "no current CUDA context after the symbol lookup");
    ent.ctx_id = id;
    ent.addr = p;
  }
  *out = ent.addr;
  return TLF_OK;
}
}  // namespace

extern "C" int tlf_attn_decode_static(const tlf_attn_args* a, void* stream) {
  using namespace tlf;
  if (const char* why = attn_op_validate(a)) return set_thread_error(TLF_ERR_INVALID_ARG, why);
  const int sms = current_num_sms();
  if (sms <= 0) return set_thread_error(TLF_ERR_CUDA, "no current CUDA device");
  const AttnOpLayout L = attn_op_layout(a, sms);
  if (L.total > kStaticScratchBytes) {
    char msg[256];
    snprintf(msg, sizeof msg,
             "tlf_attn_decode_static: these arguments need %zu bytes of scratch but the built-in buffer holds "
             "%zu; use tlf_attn_decode with caller scratch",
             L.total, kStaticScratchBytes);
    return set_thread_error(TLF_ERR_INVALID_ARG, msg);
  }
  void* base = nullptr;
  if (int rc = static_scratch_address(&base)) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  uint8_t* scratch = static_cast<uint8_t*>(base);
  // Only the internal error word must start at zero (it is OR-ed into); every
  // other scratch byte is written before it is read within a call.
  if (!a->err) {
    const cudaError_t e = cudaMemsetAsync(scratch + L.errw, 0, 4, st);
    if (e != cudaSuccess) return set_thread_error(TLF_ERR_CUDA, cudaGetErrorString(e));
  }
  const cudaError_t e = attn_op_run(a, scratch, L, st);
  if (e != cudaSuccess) return set_thread_error(TLF_ERR_CUDA, cudaGetErrorString(e));
  return TLF_OK;
}
