// Internal declarations shared by the kernels and the host runtime of libtlf.
//
// Device helpers here are thin inline-PTX wrappers (mbarrier, 1-D bulk copy,
// 2-D tensor copy, tcgen05) written from the public PTX ISA. Every wait on an
// mbarrier is bounded by wall-clock time (%globaltimer); when it runs out the
// kernel records TLF_DEVERR_WAIT in the context's error word and returns, so
// no kernel of this library can spin forever.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "tlf.h"

namespace tlf {

// ----------------------------------------------------------------------------
// Error word bits written by kernels (read by the host after each step).
// ----------------------------------------------------------------------------
enum : uint32_t {
  DEVERR_WAIT = 1u,       // an mbarrier wait ran past its time limit
  DEVERR_INDEX = 2u,      // a page id / slot / row index was out of range
  DEVERR_TMEM = 4u,       // TMEM allocation returned an unusable address
};

constexpr uint64_t kWaitLimitNs = 4000000000ull;  // 4 s

// ----------------------------------------------------------------------------
// Programmatic dependent launch. Every kernel of the step is launched with
// programmatic stream serialisation: it may start while its predecessor in the
// stream is still running, does work that reads nothing the predecessors write
// (barrier set-up, TMEM allocation, weight tiles), then waits for them with
// pdl_wait() and lets its own successor start with pdl_trigger(). Without the
// launch attribute both instructions are no-ops.
// ----------------------------------------------------------------------------
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// Launch with the programmatic-serialisation attribute when `pdl` is set.
extern bool g_use_pdl;
template <typename... KArgs, typename... Args>
inline cudaError_t launch_k(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                            Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = g_use_pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// ----------------------------------------------------------------------------
// Element helpers
// ----------------------------------------------------------------------------
typedef __nv_bfloat16 bf16;

__device__ __forceinline__ float to_f32(float x) { return x; }
__device__ __forceinline__ float to_f32(bf16 x) { return __bfloat162float(x); }
template <typename T> __device__ __forceinline__ T from_f32(float x);
template <> __device__ __forceinline__ float from_f32<float>(float x) { return x; }
template <> __device__ __forceinline__ bf16 from_f32<bf16>(float x) { return __float2bfloat16_rn(x); }

// 16 bytes of T widened to float: 4 floats or 8 bf16.
template <typename T> struct Vec16;
template <> struct Vec16<float> {
  static constexpr int N = 4;
  __device__ __forceinline__ static void load(const float* p, float* out) {
    float4 v = *reinterpret_cast<const float4*>(p);
    out[0] = v.x; out[1] = v.y; out[2] = v.z; out[3] = v.w;
  }
};
template <> struct Vec16<bf16> {
  static constexpr int N = 8;
  __device__ __forceinline__ static void load(const bf16* p, float* out) {
    uint4 v = *reinterpret_cast<const uint4*>(p);
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      out[2 * i] = __uint_as_float(w[i] << 16);
      out[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
    }
  }
};

// ----------------------------------------------------------------------------
// Shared-memory address, timers, mbarrier
// ----------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

// Make barrier initialisation visible to the async proxy (TMA, tcgen05.commit).
__device__ __forceinline__ void fence_barrier_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// Wait for the phase with the given parity to complete; false after the time limit
// (the error word then carries DEVERR_WAIT).
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, uint32_t* err) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (globaltimer_ns() - t0 > kWaitLimitNs) {
      atomicOr(err, DEVERR_WAIT);
      return false;
    }
  }
}

// 1-D bulk copy global -> shared (TMA engine), completing tx bytes on `bar`.
// dst, src and bytes must be multiples of 16.
__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
      "l"(src), "r"(bytes), "r"(bar)
      : "memory");
}

// L2 access policies for the cache_hint forms of the bulk copies: streamed data
// that is read once per launch (KV pages, decode weight tiles) is marked for
// early eviction so it does not displace the step's small, reused buffers.
__device__ __forceinline__ uint64_t l2_policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint64_t l2_policy_evict_normal() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_normal.b64 %0, 1.0;" : "=l"(p));
  return p;
}

// bulk_g2s with an L2 access policy.
__device__ __forceinline__ void bulk_g2s_hint(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar,
                                              uint64_t policy) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::"r"(
          dst),
      "l"(src), "r"(bytes), "r"(bar), "l"(policy)
      : "memory");
}

// 2-D tiled tensor copy global -> shared with a tensor map (coordinates in elements,
// innermost first). The innermost coordinate times the element size is a multiple of 16.
// This form carries an L2 access policy; tma_load_2d below has none.
__device__ __forceinline__ void tma_load_2d_hint(uint32_t dst, const CUtensorMap* map, int32_t c0, int32_t c1,
                                                 uint32_t bar, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1, {%2, "
      "%3}], [%4], %5;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(bar), "l"(policy)
      : "memory");
}

// 3-D tiled tensor copy global -> shared (coordinates innermost first).
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* map, int32_t c0, int32_t c1, int32_t c2,
                                            uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(
          dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(bar)
      : "memory");
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int32_t c0, int32_t c1,
                                            uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
          dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(bar)
      : "memory");
}

__device__ __forceinline__ void prefetch_tensormap(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

// ----------------------------------------------------------------------------
// tcgen05 (5th-generation tensor core, accumulators in tensor memory)
// ----------------------------------------------------------------------------
__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// D(tmem) (+)= A(smem desc) * B(smem desc), kind::f16 (bf16 inputs, f32 accumulate).
__device__ __forceinline__ void tc_mma_f16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                           uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive on an mbarrier once every tcgen05.mma issued so far by this thread has completed.
__device__ __forceinline__ void tc_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
               : "memory");
}

// 32 lanes x 32-bit, 16 consecutive columns per thread.
__device__ __forceinline__ void tmem_ld_16(uint32_t taddr, float* v) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// The same load without the wait: several loads may be in flight before one tmem_ld_wait(),
// after which their registers may be read.
__device__ __forceinline__ void tmem_ld_16_issue(uint32_t taddr, uint32_t* r) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

// 32 lanes x 32-bit, 16 consecutive columns per thread, register -> TMEM; waits for completion.
__device__ __forceinline__ void tmem_st_16(uint32_t taddr, const float* v) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(taddr),
      "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])), "r"(__float_as_uint(v[3])),
      "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])), "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])),
      "r"(__float_as_uint(v[8])), "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
      "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
      "r"(__float_as_uint(v[15]))
      : "memory");
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// Makes this thread's ordinary shared-memory stores visible to the tensor cores
// (the async proxy) once a barrier orders them before the MMA issue.
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Byte offset of 16-byte chunk q of row `row` in a K-major tile with 128-byte
// swizzling (rows of 128 B = 64 bf16, 8-row atoms; the tile base is 1024-byte
// aligned), the layout TMA writes with CU_TENSOR_MAP_SWIZZLE_128B.
__host__ __device__ constexpr uint32_t sw128_off(int row, int q) {
  return (uint32_t)row * 128u + (uint32_t)((q ^ (row & 7)) << 4);
}

// Shared-memory matrix descriptor for an MN-major operand tile (N contiguous) written by TMA
// with 128-byte swizzling: rows of 128 B = 64 elements along N, one row per K index, 8-row
// swizzle atoms 1024 B apart along K (stride byte offset) and 64-element atom columns
// col_stride bytes apart along N (leading byte offset). A K step of 16 advances the start
// address by 2048 B. (Checked on the device against a direct product.)
__device__ __forceinline__ uint64_t smem_desc_sw128_mn(uint32_t saddr, uint32_t col_stride) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr >> 4) & 0x3FFFu);
  d |= (uint64_t)((col_stride >> 4) & 0x3FFFu) << 16;  // leading byte offset: next 64 N-elements
  d |= (uint64_t)(1024u >> 4) << 32;                   // stride byte offset: next 8 K-rows
  d |= (uint64_t)1u << 46;
  d |= (uint64_t)2u << 61;
  return d;
}

// Shared-memory matrix descriptor for a K-major operand tile written by TMA with
// 128-byte swizzling: rows of 128 B, 8-row swizzle atoms 1024 B apart.
__device__ __forceinline__ uint64_t smem_desc_sw128(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr >> 4) & 0x3FFFu);        // start address
  d |= (uint64_t)1u << 16;                        // leading byte offset (unused for swizzled K-major)
  d |= (uint64_t)(1024u >> 4) << 32;              // stride byte offset: 8 rows * 128 B
  d |= (uint64_t)1u << 46;                        // descriptor version (sm_100 family)
  d |= (uint64_t)2u << 61;                        // layout: 128-byte swizzle
  return d;
}

// Instruction descriptor: kind::f16, A = B = bf16, D = f32, both K-major, M x N.
__host__ __device__ constexpr uint32_t idesc_bf16_f32(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}
// The same with B MN-major (bit 16).
__host__ __device__ constexpr uint32_t idesc_bf16_f32_bmn(int M, int N) { return idesc_bf16_f32(M, N) | (1u << 16); }

// 32 lanes x 32-bit, 32 consecutive columns per thread (one wait).
__device__ __forceinline__ void tmem_ld_32(uint32_t taddr, float* v) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,"
      "%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
        "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// ----------------------------------------------------------------------------
// Thread-block clusters: rank, distributed shared memory, cluster barrier.
// Every CTA of a cluster is resident at the same time, so the barrier always
// completes once each CTA of the cluster reaches it (no CTA returns early).
// ----------------------------------------------------------------------------
__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// Address of the same shared-memory location in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t dsmem_map(uint32_t saddr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(saddr), "r"(rank));
  return r;
}
// Not volatile: the address comes from dsmem_map (volatile, issued after the
// cluster barrier), so these loads cannot move above the barrier but can be
// batched freely.
__device__ __forceinline__ float dsmem_ld_f32(uint32_t addr) {
  float v;
  asm("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(addr));
  return v;
}
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// ----------------------------------------------------------------------------
// Warp / block reductions and scans
// ----------------------------------------------------------------------------
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// ----------------------------------------------------------------------------
// Kernel argument blocks
// ----------------------------------------------------------------------------
enum GemmEpilogue : int {
  EPI_PARTIAL = 0,    // out[s][row][col] = acc (split-K partial sums, float32)
  EPI_RESID = 1,      // atomicAdd(resid[idx[row]][col], acc) (residual add + scatter, Eq. 7)
  EPI_STORE = 2,      // out[row][col] = acc (float32; single split)
  // Cluster epilogues: the split-K CTAs of a tile form one cluster and sum their
  // partial tiles through distributed shared memory, then:
  EPI_CL_RESID = 3,   // resid[idx[row]][col] += sum (one writer per element; Eq. 7)
  EPI_CL_QKV = 4,     // RoPE on q and k at the original position, q -> Q, k and v appended to
                      // the loop-r page of the token's sequence (Eq. 9, 11)
  EPI_CL_SWIGLU = 5,  // U[row][64*tile + f] = silu(gate_f) * up_f; each 128-row weight tile holds
                      // 64 gate rows then the 64 matching up rows
};

struct StepDev {
  // per-step inputs / outputs (device)
  const int* tokens;   // [B]
  const int* forced;   // [B]
  const int* slots;    // [B] sequence slot of each row
  int* m;              // [B] loop counts
  float* margin;       // [B]
  float* H;            // [B][d] residual stream, float32
  // compaction / plan, written by the plan kernel
  int* idx;            // [M][maxB] rows of A_r in increasing order
  int* n;              // [M] |A_r|
  int* item_base;      // [M][maxB+1]
  int* nch;            // [M][maxB] keys each kv head of the token attends to (0: no work)
  int* act;            // [M][maxB] 1 if compact row k runs loop r (always, except rows masked
                       // by TLF_ABLATION_NO_GATHER)
  int* chunk;          // [M] keys per page
  int* cnt;            // [maxB * Hkv] attention merge tickets (zeroed by the plan kernel)
  int4* rowinfo;       // [M][maxB] per compact row k of A_r: {page, slot in page, position, 0} of the
                       // token's new loop-r cache entry (page -1 if the page table is corrupt);
                       // NULL for callers that only attend (the plan then writes no append targets)
  int* col;            // [M][maxB] compact row of residual-stream row b in A_r, -1 if not listed
                       // (inverse of idx; NULL: not written)
  // cache state
  int* len;            // [max_seqs][M] entries per (sequence, loop)
  int* page_table;     // [max_seqs][M][max_pages]
  int* pos_table;      // [n_pages][page_size]
  void* pool;          // KV pages
  uint32_t* err;
};

struct ModelDims {
  int V, d, Hq, Hkv, hd, J, ff, M;
  int qkv_dim, q_dim, kv_dim;
  int max_seqs, max_batch, max_pages, page_size;
  long long n_pages;
  long long page_elems;  // elements per page
  float eps, rope_base, threshold;
  int exit_rule;
  int dtype;             // 0 f32, 1 bf16
  int max_pos;           // positions 0..max_pos-1 have a row in the rotary table
  int ablation;          // tlf_ablation
  int router_hidden;     // > 0: two-layer MLP router with this hidden width
};

// Time/step conditioning (Sec. 3.1, App. A) inside the step. The modulation of
// layer j for a token of depth m at loop r (0-based) is built once per context
// into the table [J][M(M+1)/2][4][d]: depth-major (m, r) pairs, then the four
// vectors alpha_msa, alpha_mlp, gamma_msa, gamma_mlp.
struct CondArgs {
  const float* mod = nullptr;  // the table; NULL = no conditioning
  const int* m = nullptr;      // loop count of each row, indexed like the residual stream's rows
  int M = 0, d = 0, r = 0, j = 0;
  int part = 0;                // which of the four vectors
};
// Row of the table for residual-stream row b. Rows that do not run loop r (masked
// rows of the no-gather ablation, discarded) read the vectors of depth r + 1.
__device__ __forceinline__ const float* cond_row(const CondArgs& c, int b) {
  int m = c.m[b];
  m = m < c.r + 1 ? c.r + 1 : (m > c.M ? c.M : m);
  const int combo = m * (m - 1) / 2 + c.r;
  return c.mod + (((size_t)c.j * (c.M * (c.M + 1) / 2) + combo) * 4 + c.part) * c.d;
}

struct GemmArgs {
  int N;             // output features (rows of W)
  int K;             // reduction length
  int splits;        // split-K factor (gridDim.y; the cluster size for EPI_CL_*)
  int stages;        // depth of the tcgen05 kernel's operand ring (set by the launcher)
  const int* act;    // RESID epilogues: rows with act[row] == 0 keep their residual (NULL: none)
  CondArgs alpha;    // RESID epilogues: the update is gated by alpha (conditioning; mod NULL: none)
  const int* n_dev;  // token rows n (device scalar), or NULL to use n_host
  int n_host;
  int epi;           // GemmEpilogue
  float* out;        // EPI_PARTIAL: [splits][max_rows][N]; EPI_STORE: [rows][ldo]
  int ldo;
  int max_rows;
  float* resid;      // EPI_RESID / EPI_CL_RESID: [*][ldr]
  int ldr;
  const int* idx;    // residual row map (NULL = identity)
  uint32_t* err;
  // EPI_CL_QKV / EPI_CL_SWIGLU
  ModelDims md;
  StepDev s;
  int r, j;
  const float2* rope;      // [max_pos][hd/2] (cos, sin) of position x rotary frequency
  float* Q;                // [max_rows][Hq][hd]
  void* U;                 // [max_rows][ff] bf16
  // token tiling (prefill): gridDim.z = tok_tiles tiles of NT rows
  int tok_tiles;
  // prefill QKV epilogue: per compact row, sequence slot, loop-r cache slot and position
  const int* row_slot;
  const int* row_cslot;
  const int* row_pos;
  // RMSNorm split across two GEMMs (EPI_CL_* decode path). The producer (a RESID
  // epilogue) writes the next pre-norm's operand unscaled, xn[dst][f] =
  // h[f] * gain[f] * (1 + gamma[f]), and per 128-feature tile t the partial sum
  // ss[dst][t] = sum of h[f]^2 over the tile; the consumer (QKV or SwiGLU epilogue)
  // scales column c of its product by rsqrt(sum_t ss[c][t] / K + eps), which is
  // the row's RMSNorm factor moved past the (linear) projection. Rows of ss hold
  // ldss = ceil(d / 128) rounded up to 4 entries, the padding kept at zero.
  bf16* xn;                // producer: next operand [max_rows][N] (NULL: no fused norm)
  float* ss_out;           // producer: [max_rows][ldss]
  const float* gain;       // producer: the next norm's gain [N]
  CondArgs gamma;          // producer: the next norm's conditioning (mod NULL: none)
  const int* next_col;     // producer: column of residual row b in the next operand (NULL: same column)
  const float* ss_in;      // consumer: [max_rows][ldss] (NULL: operand already normalised)
  int ldss;
  float norm_eps;
  // Two-term bf16 operand (tcgen05 decode path). An activation v is
  // stored as hi = bf16(v) and lo = bf16(v - hi) in two planes of one buffer, lo at row
  // offset max_rows, and the GEMM multiplies both (MMA N = 2 x tile, halves summed in the
  // epilogue), so the operand keeps about 16 significant bits instead of 8.
  int blo;                 // consumer: row offset of the token operand's lo plane (0: one plane)
  bf16* xn_lo;             // producer (split norm): lo plane of xn (NULL: none)
  void* U_lo;              // EPI_CL_SWIGLU: lo plane of U (NULL: none)
  // One-split cluster epilogues (prefill) may stage their fp32 tile in windows of this many token
  // columns, so the CTA needs less shared memory and two share an SM (0: the whole tile at once).
  int red_window;
};
// Entries per row of the split-norm partial sums for model width d.
inline int split_norm_ldss(int d) { return (((d + 127) / 128) + 3) / 4 * 4; }

// ----------------------------------------------------------------------------
// Launchers (host functions, one .cu file each)
// ----------------------------------------------------------------------------
struct PageUpdate {
  int index;  // into page_table
  int page;
};

void launch_router(const ModelDims& md, const StepDev& s, int B, const void* emb, const void* router_w,
                   const float* router_b, const PageUpdate* upd, const int* n_upd, cudaStream_t st,
                   const void* router_w1 = nullptr, const float* router_b1 = nullptr);
void launch_plan(const ModelDims& md, const StepDev& s, int B, cudaStream_t st);

void launch_norm_rows(int dtype, const float* H, int ldh, const int* idx, const int* n_dev, int n_host,
                      int rows_max, const float* gain, int d, float eps, void* X, int ldx, cudaStream_t st,
                      const CondArgs& gamma = CondArgs{}, float* ss_out = nullptr, void* X_lo = nullptr);
// Builds the conditioning table (see CondArgs) from the float32 weights on the device, in float64.
int build_cond_table(const ModelDims& md, const float* t_w1, const float* t_b1, const float* t_w2, const float* t_b2,
                     const float* dt_w1, const float* dt_b1, const float* dt_w2, const float* dt_b2,
                     const float* mod_w, const float* mod_b, float* table, cudaStream_t st);

void launch_gemm_simt(int dtype, const void* W, const void* X, int ldx, const GemmArgs& a, cudaStream_t st);
void launch_gemm_tc(const CUtensorMap* mapW, const CUtensorMap* mapX, int nt_max, const GemmArgs& a,
                    cudaStream_t st);
// operand-ring depth of a tcgen05 GEMM whose CTAs each reduce ceil(ceil(K/64)/splits) k-tiles
// with token tile nt (and a two-term operand when lo), and the dynamic shared memory one CTA
// then needs
int gemm_tc_stages(int K, int splits, int nt, bool lo);
int gemm_tc_smem_bytes(int nt, int stages, bool lo = false);

void launch_rope_table(const ModelDims& md, const double* inv_freq, float2* table, cudaStream_t st);
void launch_rope_append(const ModelDims& md, const StepDev& s, int r, int j, const float* part, int splits,
                        float* Q, const float2* rope, cudaStream_t st);
// o_lo (bf16 models): also write O's lo plane (bf16 of the rounding remainder) at row offset
// max_batch, the two-term operand of the output projection
void launch_attn_decode(const ModelDims& md, const StepDev& s, int r, int j, const float* Q, float* part, void* O,
                        int* cnt, int grid, cudaStream_t st, bool o_lo = false);
// Id of the calling thread's current CUDA context (unique for the life of the process); false when
// no context is current yet or the driver entry points are unavailable.
bool current_context_id(unsigned long long* id);
// A kernel's dynamic shared-memory limit (and, if asked, non-portable cluster sizes), set once per
// (kernel, CUDA context).
cudaError_t ensure_kernel_attrs(const void* func, int max_dyn_smem, bool nonportable_cluster = false);
int attn_decode_grid(const ModelDims& md, int num_sms);
size_t attn_partial_floats(const ModelDims& md, int grid);

void launch_swiglu(int dtype, const float* part, int splits, int max_rows, const int* n_dev, int ff, void* U,
                   cudaStream_t st);
void launch_final(const ModelDims& md, const StepDev& s, int B, const float* gain, void* Xf, cudaStream_t st);

void launch_scatter_cache(const ModelDims& md, int slot, int r, int n, const void* k, const void* v,
                          const int* positions, const int* page_table, void* pool, int* pos_table,
                          cudaStream_t st);
void launch_fill_cache(const ModelDims& md, int slot, int r, int n, const int* positions, const int* page_table,
                       void* pool, int* pos_table, cudaStream_t st);

// Batched prefill of one chunk of prompt tokens (ordered by sequence, then position).
struct PrefillDev {
  int T;               // tokens in the chunk
  int S;               // sequences in the chunk (<= Smax <= 1024)
  int C;               // chunk capacity (row stride of the per-loop arrays)
  int Smax;            // sequence capacity (row stride of the per-sequence arrays)
  const int* seqidx;   // [T] sequence of each token (0..S-1)
  const int* pos;      // [T] original position of each token
  const int* seq_slot; // [S] sequence slot
  const int* m;        // [T] loop counts
  int* idx;            // [M][C] chunk rows of A_r
  int* n;              // [M] |A_r|
  int* row_slot;       // [M][C] sequence slot of each compact row
  int* row_cslot;      // [M][C] loop-r cache slot of each compact row
  int* row_pos;        // [M][C] position of each compact row
  int* first;          // [M][Smax] first compact row of each sequence
  int* cnt;            // [M][Smax] compact rows of each sequence
  int* s0;             // [M][Smax] loop-r cache length of each sequence before the chunk
  int* tile_base;      // [M][Smax + 1] attention query blocks, prefix over sequences
  int qblock;          // queries per attention block (the attention kernel's tile)
  int* len;            // [max_seqs][M] cache lengths
};
void launch_pf_plan(const ModelDims& md, const PrefillDev& p, cudaStream_t st);
// pool_map: 3-D tensor map over the KV pool, {head_dim, J * 2 * Hkv * 64 rows of a page, pages}, box
// {64, 64, 1}, 128-byte swizzle (NULL: the kernel without tensor-map loads)
void launch_pf_attn(const ModelDims& md, const PrefillDev& p, const StepDev& s, int r, int j, const float* Q,
                    void* O, int tiles_bound, cudaStream_t st, const CUtensorMap* pool_map = nullptr);
void launch_pf_len(const ModelDims& md, const PrefillDev& p, cudaStream_t st);
// Queries per block of the prefill attention kernel that launch_pf_attn picks for this model.
int pf_attn_qblock(const ModelDims& md);

// Kernel-level attention operation (tlf_attn_decode): scratch layout and launch.
struct AttnOpLayout {
  size_t m, slots, len, idx, count, item_base, nch, chunk, errw, cnt, part, total;
  int grid;
};
AttnOpLayout attn_op_layout(const tlf_attn_args* a, int num_sms);
const char* attn_op_validate(const tlf_attn_args* a);
cudaError_t attn_op_run(const tlf_attn_args* a, uint8_t* scratch, const AttnOpLayout& L, cudaStream_t st);
int current_num_sms();

// Record a message for tlf_last_error(NULL) on this thread; returns code.
int set_thread_error(int code, const char* msg);

}  // namespace tlf
