// Kernel-level entry point: the recursion-wise split-K decode attention on a
// caller-described paged cache (declared in include/tlf.h).
//
// It runs the same kernels as a decode step, with one loop (M = 1) and row b
// standing for sequence slot b: a prep kernel turns the key counts into cache
// lengths, the plan kernel cuts every (row, kv head) key range into chunks,
// k_attn_decode streams the pages and k_attn_combine merges the chunk
// partials. The scratch holds the plan and the partials.
#include <cudaTypedefs.h>

#include <atomic>
#include <mutex>
#include <vector>

#include "tlf.h"
#include "tlf_internal.cuh"

namespace tlf {

// Id of the calling thread's current CUDA context (unique for the life of the process);
// false when no context is current yet or the driver entry points are unavailable.
bool current_context_id(unsigned long long* id) {
  static std::atomic<PFN_cuCtxGetCurrent_v4000> get_current{nullptr};
  static std::atomic<PFN_cuCtxGetId_v12000> get_id{nullptr};
  if (!get_current.load() || !get_id.load()) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 4000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess || !p)
      return false;
    get_current.store(reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(p));
    p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess || !p)
      return false;
    get_id.store(reinterpret_cast<PFN_cuCtxGetId_v12000>(p));
  }
  CUcontext c = nullptr;
  if (get_current.load()(&c) != CUDA_SUCCESS || !c) return false;
  return get_id.load()(c, id) == CUDA_SUCCESS;
}

// Kernel attributes belong to a CUDA context: a device reset, or the same kernel on another
// device, needs them set again. Each (kernel, context) pair is set once; without a context id
// the attributes are set on every call.
cudaError_t ensure_kernel_attrs(const void* func, int max_dyn_smem, bool nonportable_cluster) {
  struct Entry {
    const void* func;
    unsigned long long ctx;
    int smem;
    bool nonportable;
  };
  static std::mutex mu;
  static std::vector<Entry> done;
  unsigned long long ctx = 0;
  const bool have = current_context_id(&ctx);
  std::lock_guard<std::mutex> lock(mu);
  Entry* hit = nullptr;
  if (have)
    for (Entry& e : done)
      if (e.func == func && e.ctx == ctx) hit = &e;
  if (hit && hit->smem >= max_dyn_smem && (hit->nonportable || !nonportable_cluster)) return cudaSuccess;
  cudaError_t r = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, max_dyn_smem);
  if (r == cudaSuccess && nonportable_cluster)
    r = cudaFuncSetAttribute(func, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (r == cudaSuccess && have) {
    if (hit) {
      hit->smem = max_dyn_smem;
      hit->nonportable = hit->nonportable || nonportable_cluster;
    } else {
      done.push_back({func, ctx, max_dyn_smem, nonportable_cluster});
    }
  }
  return r;
}

__global__ void k_attn_prep(int n, const int* __restrict__ lens, int max_keys, int* m, int* slots, int* len,
                            uint32_t* err) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= n) return;
  int L = lens[b];
  if (L < 1 || L > max_keys) {
    atomicOr(err, DEVERR_INDEX);
    L = 1;
  }
  m[b] = 1;
  slots[b] = b;
  len[b] = L - 1;  // the kernels attend to len + 1 entries
}

static size_t up(size_t x, size_t a) { return (x + a - 1) / a * a; }

AttnOpLayout attn_op_layout(const tlf_attn_args* a, int num_sms) {
  AttnOpLayout L{};
  const int n = a->n, G = a->n_heads / a->n_kv_heads;
  L.grid = 2 * num_sms;
  const size_t part_floats = ((size_t)n * a->n_kv_heads + L.grid) * G * (a->head_dim + 2);
  size_t o = 0;
  auto take = [&](size_t bytes) { size_t at = o; o = up(o + bytes, 16); return at; };
  L.m = take(4 * (size_t)n);
  L.slots = take(4 * (size_t)n);
  L.len = take(4 * (size_t)n);
  L.idx = take(4 * (size_t)n);
  L.count = take(4);
  L.item_base = take(4 * ((size_t)n + 1));
  L.nch = take(4 * (size_t)n);
  L.chunk = take(4);
  L.errw = take(4);
  L.cnt = take(4 * (size_t)n * a->n_kv_heads);
  o = up(o, 256);
  L.part = take(4 * part_floats);
  L.total = up(o, 256);
  return L;
}

const char* attn_op_validate(const tlf_attn_args* a) {
  if (!a) return "args is NULL";
  if (a->n < 1 || a->n > 256) return "n must be in 1..256";
  if (a->dtype != TLF_DTYPE_F32 && a->dtype != TLF_DTYPE_BF16) return "unknown dtype";
  if (a->n_heads < 1 || a->n_kv_heads < 1 || a->n_heads % a->n_kv_heads) return "n_kv_heads must divide n_heads";
  const int g = a->n_heads / a->n_kv_heads;
  if (!(g == 1 || g == 2 || (g == 4 && a->dtype == TLF_DTYPE_BF16 && a->head_dim >= 64)))
    return "query heads per kv head must be 1 or 2 (or 4 for bf16 with head_dim >= 64)";
  if (a->dtype == TLF_DTYPE_BF16 ? !(a->head_dim == 32 || a->head_dim == 64 || a->head_dim == 128)
                                 : !(a->head_dim == 16 || a->head_dim == 32 || a->head_dim == 64 || a->head_dim == 128))
    return "unsupported head_dim for this dtype";
  if (a->n_layers < 1 || a->layer < 0 || a->layer >= a->n_layers) return "layer out of range";
  if (a->page_size != 64) return "page_size must be 64";
  if (a->max_pages < 1 || a->n_pages < 1 || a->n_pages > 0x7fffffff) return "bad page counts";
  if (a->max_pages > 0x7fffffff / a->page_size) return "max_pages * page_size exceeds the int32 key range";
  if (!a->q || !a->pool || !a->page_table || !a->lens || !a->out) return "a device pointer is NULL";
  return nullptr;
}

int current_num_sms() {
  // one entry per device ordinal, filled on first use; concurrent first uses store the same value
  static std::atomic<int> cache[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (dev < 0 || dev >= 64) return 0;
  int n = cache[dev].load(std::memory_order_relaxed);
  if (!n) {
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    cache[dev].store(n, std::memory_order_relaxed);
  }
  return n;
}

cudaError_t attn_op_run(const tlf_attn_args* a, uint8_t* scratch, const AttnOpLayout& L, cudaStream_t st) {
  ModelDims md{};
  md.Hq = a->n_heads;
  md.Hkv = a->n_kv_heads;
  md.hd = a->head_dim;
  md.J = a->n_layers;
  md.M = 1;
  md.q_dim = md.Hq * md.hd;
  md.kv_dim = md.Hkv * md.hd;
  md.qkv_dim = md.q_dim + 2 * md.kv_dim;
  md.max_seqs = a->n;
  md.max_batch = a->n;
  md.max_pages = a->max_pages;
  md.page_size = a->page_size;
  md.n_pages = a->n_pages;
  md.page_elems = (long long)md.J * 2 * md.Hkv * md.page_size * md.hd;
  md.dtype = a->dtype;

  StepDev s{};
  s.m = reinterpret_cast<int*>(scratch + L.m);
  s.slots = reinterpret_cast<int*>(scratch + L.slots);
  s.len = reinterpret_cast<int*>(scratch + L.len);
  s.idx = reinterpret_cast<int*>(scratch + L.idx);
  s.n = reinterpret_cast<int*>(scratch + L.count);
  s.item_base = reinterpret_cast<int*>(scratch + L.item_base);
  s.nch = reinterpret_cast<int*>(scratch + L.nch);
  s.chunk = reinterpret_cast<int*>(scratch + L.chunk);
  s.page_table = const_cast<int*>(a->page_table);
  s.pool = const_cast<void*>(a->pool);
  s.err = a->err ? a->err : reinterpret_cast<uint32_t*>(scratch + L.errw);
  s.cnt = reinterpret_cast<int*>(scratch + L.cnt);
  float* part = reinterpret_cast<float*>(scratch + L.part);

  k_attn_prep<<<(a->n + 127) / 128, 128, 0, st>>>(a->n, a->lens, a->max_pages * a->page_size, s.m,
                                                  const_cast<int*>(s.slots), s.len, s.err);
  launch_plan(md, s, a->n, st);
  launch_attn_decode(md, s, 0, a->layer, a->q, part, a->out, s.cnt, L.grid, st);
  return cudaGetLastError();
}

}  // namespace tlf

using namespace tlf;

extern "C" size_t tlf_attn_decode_scratch_bytes(const tlf_attn_args* a) {
  if (attn_op_validate(a)) return 0;
  const int sms = current_num_sms();
  if (sms <= 0) return 0;
  return attn_op_layout(a, sms).total;
}

extern "C" int tlf_attn_decode(const tlf_attn_args* a, void* scratch, size_t scratch_bytes, void* stream) {
  if (const char* why = attn_op_validate(a)) return set_thread_error(TLF_ERR_INVALID_ARG, why);
  const int sms = current_num_sms();
  if (sms <= 0) return set_thread_error(TLF_ERR_CUDA, "no current CUDA device");
  const AttnOpLayout L = attn_op_layout(a, sms);
  if (!scratch || scratch_bytes < L.total) return set_thread_error(TLF_ERR_INVALID_ARG, "scratch too small");
  const cudaError_t e = attn_op_run(a, static_cast<uint8_t*>(scratch), L, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return set_thread_error(TLF_ERR_CUDA, cudaGetErrorString(e));
  return TLF_OK;
}
