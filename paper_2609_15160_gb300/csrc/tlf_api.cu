// Host runtime and C ABI of libtlf (declared in include/tlf.h).
//
// The runtime owns the device copies of the weights, the paged KV pool of the
// recursion-wise caches and the per-step workspaces. Host-side bookkeeping:
// a sequence table (id -> slot), a free list of KV pages, and a host mirror of
// every (sequence, loop) cache length and page table. Before a step launches
// anything, the host checks the batch and reserves, for every sequence, one
// free slot in each of the M loop caches (a page is taken only when a loop
// cache is at a page boundary); so a failing call changes nothing, and a step
// never needs the host between kernels. The loop counts come back at the end
// of the step and advance the host mirror.
//
// One decode step (T-LoopFormer Sec. 3.2-3.3):
//   router (Eq. 2-5) -> compaction + attention plan (Eq. 6) ->
//   for loop r, layer j: gather+RMSNorm -> QKV GEMM -> RoPE + append (Eq. 9, 11)
//     -> recursion-wise split-K attention + combine (Eq. 10) -> O GEMM + residual
//     scatter (Eq. 7) -> gather+RMSNorm -> gate/up GEMM -> SwiGLU -> down GEMM +
//     residual scatter
//   -> final RMSNorm + cache-length update -> tied LM head.
// Kernels of a loop with no active token exit on the device-side count.
#include <cudaTypedefs.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <string>
#include <unordered_map>
#include <unordered_set>
#include <vector>

#include "tlf.h"
#include "tlf_internal.cuh"

using namespace tlf;

namespace {
thread_local std::string g_create_error = "no error";

struct DeviceMat {
  void* ptr = nullptr;
  int N = 0, K = 0;
  CUtensorMap map;
};
}  // namespace

struct tlf_ctx {
  tlf_config cfg{};
  ModelDims md{};
  std::string err = "no error";
  bool host_only = false;
  int num_sms = 0;
  size_t eb = 4;
  bool use_tc = false;
  int nt_max = 0;

  // weights
  void* d_emb = nullptr;
  void* d_router_w = nullptr;
  void* d_router_w1 = nullptr;   // MLP router hidden layer [H_r][d]
  float* d_router_b1 = nullptr;
  float* d_router_b = nullptr;
  float* d_attn_norm = nullptr;
  float* d_mlp_norm = nullptr;
  float* d_final_norm = nullptr;
  double* d_inv_freq = nullptr;
  float2* d_rope = nullptr;     // [max_pos][hd/2] (cos, sin)
  float* d_cond = nullptr;      // [J][M(M+1)/2][4][d] time/step modulation (conditioning only)
  int4* d_rowinfo = nullptr;    // [M][max_batch]
  int* d_act = nullptr;         // [M][max_batch]
  int* d_col = nullptr;         // [M][max_batch] compact row of each residual row per loop
  float* d_ss = nullptr;        // [max_batch][split_norm_ldss(d)] split RMSNorm partial sums of squares
  bool split_norm = false;      // pre-norms split across the neighbouring GEMMs (tcgen05 path)
  bool operand_lo = false;      // X, O, U carry a lo plane (two-term GEMM operands, tcgen05 path)
  bool pf_ws = true;            // prefill attention: the warp-specialised tensor-map kernel
  std::vector<DeviceMat> wqkv, wo, wgu, wd;
  DeviceMat emb_mat;

  // KV pool and tables
  void* d_pool = nullptr;
  CUtensorMap map_pool;         // prefill attention's tensor map over the pool (has_pool_map)
  bool has_pool_map = false;
  int* d_pos_table = nullptr;
  int64_t n_pages = 0;
  std::vector<int> free_pages;
  int* d_page_table = nullptr;
  std::vector<int> h_page_table;
  int* d_len = nullptr;
  std::vector<int> h_len;
  std::unordered_map<uint64_t, int> seq_slot;
  std::vector<int> free_slots;

  // step workspaces
  int* d_upload = nullptr;
  int* h_upload = nullptr;
  size_t upload_ints = 0;
  int* d_m = nullptr;
  float* d_margin = nullptr;
  float* d_H = nullptr;
  void* d_X = nullptr;
  void* d_O = nullptr;
  void* d_U = nullptr;
  void* d_Xf = nullptr;
  CUtensorMap map_X, map_O, map_U, map_Xf;
  float* d_part = nullptr;
  float* d_Q = nullptr;
  int* d_idx = nullptr;
  int* d_n = nullptr;
  int* d_item_base = nullptr;
  int* d_nch = nullptr;
  int* d_chunk = nullptr;
  float* d_attn_part = nullptr;
  int* d_attn_cnt = nullptr;
  int attn_grid = 0;
  float* d_logits = nullptr;
  uint32_t* d_err = nullptr;
  int* h_m = nullptr;
  float* h_margin = nullptr;
  uint32_t* h_err = nullptr;
  int s_qkv = 1, s_o = 1, s_gu = 1, s_d = 1, split_cap = 8;

  // batched prefill (bf16 models): chunk workspaces, allocated on first use
  int pf_C = 0, pf_Smax = 0;
  size_t pf_in_ints = 0;
  int* d_pf_in = nullptr;
  int* h_pf_in = nullptr;
  int* d_pf_m = nullptr;
  float* d_pf_margin = nullptr;
  float* d_pf_H = nullptr;
  void* d_pf_X = nullptr;
  float* d_pf_Q = nullptr;
  void* d_pf_O = nullptr;
  void* d_pf_U = nullptr;
  CUtensorMap pf_map_X, pf_map_O, pf_map_U;
  int *d_pf_idx = nullptr, *d_pf_n = nullptr, *d_pf_row_slot = nullptr, *d_pf_row_cslot = nullptr,
      *d_pf_row_pos = nullptr, *d_pf_first = nullptr, *d_pf_cnt = nullptr, *d_pf_s0 = nullptr,
      *d_pf_tile_base = nullptr;
  int* h_pf_m = nullptr;
  int* h_pf_nr = nullptr;  // [M] rows of every loop of the current prefill chunk
  float pf_last_ms = 0.f;

  // profiling
  bool profiling = false;
  float last_attn_ms = 0.f;
  double last_attn_bytes = 0.0;
  int last_launches = 0;
  std::vector<cudaEvent_t> events;
  std::vector<int> ev_class;  // kernel class closed by each profiling event
  float class_ms[13] = {};
  int last_batch = 0;

  // CUDA graphs of the step
  struct StepGraph {
    int B;
    bool logits;
    cudaGraphExec_t exec;
    int launches;
  };
  std::vector<StepGraph> graphs;
  cudaStream_t cap_stream = nullptr;
  bool use_graphs = true;
  bool warmed = false;
};

// ----------------------------------------------------------------------------
// small helpers
// ----------------------------------------------------------------------------
static int fail(tlf_ctx* ctx, int code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  if (ctx) ctx->err = buf;
  else g_create_error = buf;
  return code;
}

#define CK(ctx, call)                                                                          \
  do {                                                                                         \
    cudaError_t e_ = (call);                                                                   \
    if (e_ != cudaSuccess) return fail((ctx), TLF_ERR_CUDA, "%s: %s", #call, cudaGetErrorString(e_)); \
  } while (0)

static int64_t page_bytes_of(const tlf_config& c) {
  const int64_t eb = c.dtype == TLF_DTYPE_BF16 ? 2 : 4;
  return (int64_t)c.n_layers * 2 * c.n_kv_heads * c.page_size * c.head_dim * eb;
}

static int max_pages_of(const tlf_config& c) { return (c.max_seq_len + c.page_size - 1) / c.page_size; }

static bool is_device_ptr(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged;
}

extern "C" int tlf_validate_config(const tlf_config* c, char* msg, size_t msg_len) {
  auto bad = [&](const char* why) {
    if (msg && msg_len) snprintf(msg, msg_len, "%s", why);
    return TLF_ERR_INVALID_ARG;
  };
  if (!c) return bad("config is NULL");
  if (c->dtype != TLF_DTYPE_F32 && c->dtype != TLF_DTYPE_BF16) return bad("dtype must be TLF_DTYPE_F32 or TLF_DTYPE_BF16");
  if (c->vocab < 1) return bad("vocab must be >= 1");
  if (c->d_model < 64 || c->d_model % 64 || c->d_model > 8192) return bad("d_model must be a multiple of 64 in 64..8192");
  if (c->n_heads < 1 || c->n_kv_heads < 1 || c->n_heads % c->n_kv_heads) return bad("n_kv_heads must divide n_heads");
  const int g = c->n_heads / c->n_kv_heads;
  if (!(g == 1 || g == 2 || (g == 4 && c->dtype == TLF_DTYPE_BF16 && c->head_dim >= 64)))
    return bad("query heads per kv head must be 1 or 2 (or 4 for bf16 with head_dim >= 64)");
  if (c->dtype == TLF_DTYPE_BF16) {
    if (c->head_dim != 32 && c->head_dim != 64 && c->head_dim != 128) return bad("bf16 head_dim must be 32, 64 or 128");
  } else if (c->head_dim != 16 && c->head_dim != 32 && c->head_dim != 64 && c->head_dim != 128) {
    return bad("float32 head_dim must be 16, 32, 64 or 128");
  }
  if (c->n_layers < 1) return bad("n_layers must be >= 1");
  if (c->ffn_hidden < 16 || c->ffn_hidden % 16) return bad("ffn_hidden must be a positive multiple of 16");
  if (c->max_loops < 1 || c->max_loops > 16) return bad("max_loops must be in 1..16");
  if (!(c->rope_base > 1.0f)) return bad("rope_base must be > 1");
  if (!(c->norm_eps > 0.0f)) return bad("norm_eps must be > 0");
  if (c->exit_rule != TLF_EXIT_ARGMAX && c->exit_rule != TLF_EXIT_SURVIVAL) return bad("unknown exit_rule");
  if (c->exit_rule == TLF_EXIT_SURVIVAL && !(c->threshold > 0.0f && c->threshold < 1.0f))
    return bad("threshold must be in (0, 1)");
  if (c->max_seqs < 1) return bad("max_seqs must be >= 1");
  if (c->max_batch < 1 || c->max_batch > 256) return bad("max_batch must be in 1..256");
  if (c->max_batch > c->max_seqs) return bad("max_batch must not exceed max_seqs");
  if (c->max_seq_len < 1) return bad("max_seq_len must be >= 1");
  if (c->page_size != 64) return bad("page_size must be 64");
  if (c->gemm_impl != TLF_GEMM_AUTO && c->gemm_impl != TLF_GEMM_SIMT) return bad("unknown gemm_impl");
  if (c->kv_pool_pages < 0) return bad("kv_pool_pages must be >= 0");
  if (c->prefill_chunk < 0 || (c->prefill_chunk > 0 && c->prefill_chunk < 64))
    return bad("prefill_chunk must be 0 (default) or >= 64");
  if (c->ablation != TLF_ABLATION_NONE && c->ablation != TLF_ABLATION_NO_GATHER &&
      c->ablation != TLF_ABLATION_DENSE_CACHE)
    return bad("unknown ablation");
  if (c->ablation == TLF_ABLATION_DENSE_CACHE && c->dtype != TLF_DTYPE_BF16)
    return bad("the dense-cache ablation needs a bf16 model");
  if (c->conditioning != 0 && c->conditioning != 1) return bad("conditioning must be 0 or 1");
  if (c->router_hidden < 0 || c->router_hidden > 8192 || c->router_hidden % 8)
    return bad("router_hidden must be 0 or a multiple of 8 up to 8192");
  if (c->reserved != 0) return bad("reserved must be 0");
  if (msg && msg_len) snprintf(msg, msg_len, "ok");
  return TLF_OK;
}

// Programmatic dependent launch for the step kernels (TLF_NO_PDL=1 turns it off).
bool tlf::g_use_pdl = [] {
  const char* e = getenv("TLF_NO_PDL");
  return !(e && e[0] == '1');
}();

int tlf::set_thread_error(int code, const char* msg) {
  g_create_error = msg;
  return code;
}

extern "C" int64_t tlf_page_bytes(const tlf_config* c) {
  if (tlf_validate_config(c, nullptr, 0) != TLF_OK) return 0;
  return page_bytes_of(*c);
}

extern "C" const char* tlf_last_error(const tlf_ctx* ctx) {
  return ctx ? ctx->err.c_str() : g_create_error.c_str();
}

// ----------------------------------------------------------------------------
// creation
// ----------------------------------------------------------------------------
static PFN_cuTensorMapEncodeTiled_v12000 get_encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    cudaDriverEntryPointQueryResult q;
    void* p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

// 2-D bf16 tensor map over a row-major [rows][cols] matrix with row stride ld
// elements; box = 64 columns x box_rows rows, 128-byte swizzle, zero fill.
static bool make_map(CUtensorMap* m, const void* base, int rows, int cols, int ld, int box_rows) {
  auto fn = get_encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)ld * 2};
  cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
  cuuint32_t es[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// 3-D bf16 tensor map over the KV pool for the prefill attention's page loads: {head_dim,
// J * 2 * Hkv * page_size rows of a page, pages}, box {64, 64, 1}, 128-byte swizzle (a page keeps
// its own coordinate, so coordinates stay within int32 for any pool size).
static bool make_pool_map(CUtensorMap* m, const void* base, const ModelDims& md) {
  auto fn = get_encode_fn();
  if (!fn) return false;
  cuuint64_t dims[3] = {(cuuint64_t)md.hd, (cuuint64_t)md.J * 2 * md.Hkv * md.page_size, (cuuint64_t)md.n_pages};
  cuuint64_t strides[2] = {(cuuint64_t)md.hd * 2, (cuuint64_t)md.page_elems * 2};
  cuuint32_t box[3] = {64, 64, 1};
  cuuint32_t es[3] = {1, 1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, es,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

template <typename T>
static int dev_alloc(tlf_ctx* ctx, T** p, size_t bytes, const char* what) {
  void* q = nullptr;
  cudaError_t e = cudaMalloc(&q, bytes < 16 ? 16 : bytes);
  if (e != cudaSuccess) return fail(ctx, TLF_ERR_CUDA, "cudaMalloc(%s, %zu bytes): %s", what, bytes, cudaGetErrorString(e));
  *p = static_cast<T*>(q);
  return TLF_OK;
}

static int upload(tlf_ctx* ctx, void** dst, const void* src, size_t bytes, const char* what) {
  int rc = dev_alloc(ctx, dst, bytes, what);
  if (rc) return rc;
  CK(ctx, cudaMemcpy(*dst, src, bytes, cudaMemcpyHostToDevice));
  return TLF_OK;
}

static int make_mat(tlf_ctx* ctx, DeviceMat* m, const std::vector<const uint8_t*>& parts,
                    const std::vector<int>& part_rows, int K, const char* what) {
  int N = 0;
  for (int r : part_rows) N += r;
  const size_t row_bytes = (size_t)K * ctx->eb;
  std::vector<uint8_t> host((size_t)N * row_bytes);
  size_t off = 0;
  for (size_t i = 0; i < parts.size(); ++i) {
    memcpy(host.data() + off, parts[i], (size_t)part_rows[i] * row_bytes);
    off += (size_t)part_rows[i] * row_bytes;
  }
  int rc = upload(ctx, &m->ptr, host.data(), host.size(), what);
  if (rc) return rc;
  m->N = N;
  m->K = K;
  if (ctx->use_tc && !make_map(&m->map, m->ptr, N, K, K, 128))
    return fail(ctx, TLF_ERR_CUDA, "cuTensorMapEncodeTiled failed for %s", what);
  return TLF_OK;
}

static int choose_splits(int tiles, int nkb, int target_ctas, int cap) {
  int s = (target_ctas + tiles - 1) / tiles;
  s = std::max(1, std::min(s, std::min(nkb, cap)));
  return s;
}

static int create_impl(tlf_ctx* ctx, const tlf_weights* w) {
  const tlf_config& c = ctx->cfg;
  ModelDims& md = ctx->md;
  md.V = c.vocab; md.d = c.d_model; md.Hq = c.n_heads; md.Hkv = c.n_kv_heads; md.hd = c.head_dim;
  md.J = c.n_layers; md.ff = c.ffn_hidden; md.M = c.max_loops;
  md.q_dim = md.Hq * md.hd; md.kv_dim = md.Hkv * md.hd; md.qkv_dim = md.q_dim + 2 * md.kv_dim;
  md.max_seqs = c.max_seqs; md.max_batch = c.max_batch; md.max_pages = max_pages_of(c); md.page_size = c.page_size;
  md.eps = c.norm_eps; md.rope_base = c.rope_base; md.threshold = c.threshold; md.exit_rule = c.exit_rule;
  md.dtype = c.dtype;
  md.max_pos = c.max_seq_len;
  md.ablation = c.ablation;
  md.router_hidden = c.router_hidden;
  ctx->eb = c.dtype == TLF_DTYPE_BF16 ? 2 : 4;
  md.page_elems = (long long)md.J * 2 * md.Hkv * md.page_size * md.hd;
  ctx->n_pages = c.kv_pool_pages > 0 ? c.kv_pool_pages : (int64_t)c.max_seqs * c.max_loops * md.max_pages;
  if (ctx->n_pages > 0x7fffffff) return fail(ctx, TLF_ERR_INVALID_ARG, "too many KV pages");
  md.n_pages = ctx->n_pages;

  ctx->free_pages.resize(ctx->n_pages);
  for (int64_t i = 0; i < ctx->n_pages; ++i) ctx->free_pages[i] = (int)(ctx->n_pages - 1 - i);
  ctx->free_slots.resize(c.max_seqs);
  for (int i = 0; i < c.max_seqs; ++i) ctx->free_slots[i] = c.max_seqs - 1 - i;
  ctx->h_page_table.assign((size_t)c.max_seqs * c.max_loops * md.max_pages, -1);
  ctx->h_len.assign((size_t)c.max_seqs * c.max_loops, 0);
  if (ctx->host_only) return TLF_OK;

  if (!w || !w->embedding || !w->router_w || !w->router_b || !w->wq || !w->wk || !w->wv || !w->wo || !w->w_gate ||
      !w->w_up || !w->w_down || !w->attn_norm || !w->mlp_norm || !w->final_norm)
    return fail(ctx, TLF_ERR_BAD_WEIGHTS, "a weight pointer is NULL");

  int dev = 0;
  CK(ctx, cudaGetDevice(&dev));
  CK(ctx, cudaDeviceGetAttribute(&ctx->num_sms, cudaDevAttrMultiProcessorCount, dev));
  int major = 0, minor = 0;
  CK(ctx, cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev));
  CK(ctx, cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev));
  if (major != 10) return fail(ctx, TLF_ERR_CUDA, "libtlf is built for sm_103a; device is sm_%d%d", major, minor);
  ctx->use_tc = (c.dtype == TLF_DTYPE_BF16 && c.gemm_impl == TLF_GEMM_AUTO);
  if (ctx->use_tc && !get_encode_fn()) return fail(ctx, TLF_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable");
  {
    int nt = ((c.max_batch + 15) / 16) * 16, b = 16;
    while (b < nt) b <<= 1;
    ctx->nt_max = b;
  }

  const size_t eb = ctx->eb;
  const int d = md.d, J = md.J, ff = md.ff, V = md.V, M = md.M, B = md.max_batch;
  int rc;
  const int Hr = c.router_hidden;
  if ((rc = upload(ctx, &ctx->d_router_w, w->router_w, (size_t)M * (Hr > 0 ? Hr : d) * eb, "router_w"))) return rc;
  if (Hr > 0) {
    if (!w->router_w1 || !w->router_b1) return fail(ctx, TLF_ERR_BAD_WEIGHTS, "MLP router weights are NULL");
    if ((rc = upload(ctx, &ctx->d_router_w1, w->router_w1, (size_t)Hr * d * eb, "router_w1"))) return rc;
    if ((rc = upload(ctx, (void**)&ctx->d_router_b1, w->router_b1, (size_t)Hr * 4, "router_b1"))) return rc;
  }
  if ((rc = upload(ctx, (void**)&ctx->d_router_b, w->router_b, (size_t)M * 4, "router_b"))) return rc;
  if ((rc = upload(ctx, (void**)&ctx->d_attn_norm, w->attn_norm, (size_t)J * d * 4, "attn_norm"))) return rc;
  if ((rc = upload(ctx, (void**)&ctx->d_mlp_norm, w->mlp_norm, (size_t)J * d * 4, "mlp_norm"))) return rc;
  if ((rc = upload(ctx, (void**)&ctx->d_final_norm, w->final_norm, (size_t)d * 4, "final_norm"))) return rc;
  if ((rc = make_mat(ctx, &ctx->emb_mat, {(const uint8_t*)w->embedding}, {V}, d, "embedding"))) return rc;
  ctx->d_emb = ctx->emb_mat.ptr;
  ctx->wqkv.resize(J);
  ctx->wo.resize(J);
  ctx->wgu.resize(J);
  ctx->wd.resize(J);
  for (int j = 0; j < J; ++j) {
    const uint8_t* q = (const uint8_t*)w->wq + (size_t)j * md.q_dim * d * eb;
    const uint8_t* k = (const uint8_t*)w->wk + (size_t)j * md.kv_dim * d * eb;
    const uint8_t* v = (const uint8_t*)w->wv + (size_t)j * md.kv_dim * d * eb;
    if ((rc = make_mat(ctx, &ctx->wqkv[j], {q, k, v}, {md.q_dim, md.kv_dim, md.kv_dim}, d, "wqkv"))) return rc;
    const uint8_t* o = (const uint8_t*)w->wo + (size_t)j * d * md.q_dim * eb;
    if ((rc = make_mat(ctx, &ctx->wo[j], {o}, {d}, md.q_dim, "wo"))) return rc;
    const uint8_t* gt = (const uint8_t*)w->w_gate + (size_t)j * ff * d * eb;
    const uint8_t* up = (const uint8_t*)w->w_up + (size_t)j * ff * d * eb;
    if (ctx->use_tc) {
      // 128-row tiles of 64 gate rows then the 64 matching up rows (zero rows past ff), so the
      // GEMM epilogue sees both halves of SwiGLU in one tile
      const int tiles = (ff + 63) / 64;
      const size_t rb = (size_t)d * eb;
      std::vector<uint8_t> zero(rb * 64, 0);
      std::vector<const uint8_t*> parts;
      std::vector<int> rows;
      for (int t = 0; t < tiles; ++t) {
        const int cnt = std::min(64, ff - 64 * t);
        parts.push_back(gt + (size_t)64 * t * rb); rows.push_back(cnt);
        if (cnt < 64) { parts.push_back(zero.data()); rows.push_back(64 - cnt); }
        parts.push_back(up + (size_t)64 * t * rb); rows.push_back(cnt);
        if (cnt < 64) { parts.push_back(zero.data()); rows.push_back(64 - cnt); }
      }
      if ((rc = make_mat(ctx, &ctx->wgu[j], parts, rows, d, "w_gate_up"))) return rc;
    } else if ((rc = make_mat(ctx, &ctx->wgu[j], {gt, up}, {ff, ff}, d, "w_gate_up"))) {
      return rc;
    }
    const uint8_t* dn = (const uint8_t*)w->w_down + (size_t)j * d * ff * eb;
    if ((rc = make_mat(ctx, &ctx->wd[j], {dn}, {d}, ff, "w_down"))) return rc;
  }
  {
    std::vector<double> inv(md.hd / 2);
    for (int i = 0; i < md.hd / 2; ++i) inv[i] = std::pow((double)c.rope_base, -2.0 * i / md.hd);
    if ((rc = upload(ctx, (void**)&ctx->d_inv_freq, inv.data(), inv.size() * sizeof(double), "inv_freq"))) return rc;
    if ((rc = dev_alloc(ctx, &ctx->d_rope, (size_t)md.max_pos * (md.hd / 2) * sizeof(float2), "rotary table")))
      return rc;
    launch_rope_table(md, ctx->d_inv_freq, ctx->d_rope, 0);
    CK(ctx, cudaGetLastError());
    CK(ctx, cudaStreamSynchronize(0));
  }
  if (c.conditioning) {
    // time/step conditioning: the weights are needed only to build the per-(depth, loop) table
    const size_t F = 256, dd = (size_t)d * d, J4 = (size_t)J * 4 * d;
    const float* src[10] = {w->cond_t_w1, w->cond_t_b1, w->cond_t_w2, w->cond_t_b2, w->cond_dt_w1,
                            w->cond_dt_b1, w->cond_dt_w2, w->cond_dt_b2, w->mod_w, w->mod_b};
    const size_t cnt[10] = {d * F, (size_t)d, dd, (size_t)d, d * F, (size_t)d, dd, (size_t)d, J4 * d, J4};
    float* dev[10] = {};
    rc = 0;
    for (int i = 0; i < 10 && rc == 0; ++i) {
      if (!src[i]) rc = fail(ctx, TLF_ERR_BAD_WEIGHTS, "a conditioning weight pointer is NULL");
      else rc = upload(ctx, (void**)&dev[i], src[i], cnt[i] * 4, "conditioning weights");
    }
    const size_t P = (size_t)M * (M + 1) / 2;
    if (rc == 0) rc = dev_alloc(ctx, &ctx->d_cond, (size_t)J * P * 4 * d * 4, "conditioning table");
    if (rc == 0) {
      const int e = build_cond_table(md, dev[0], dev[1], dev[2], dev[3], dev[4], dev[5], dev[6], dev[7], dev[8],
                                     dev[9], ctx->d_cond, 0);
      if (e) rc = fail(ctx, TLF_ERR_CUDA, "conditioning table: %s", cudaGetErrorString((cudaError_t)e));
    }
    for (float* p : dev)
      if (p) cudaFree(p);
    if (rc) return rc;
  }

  // KV pool and tables
  if ((rc = dev_alloc(ctx, &ctx->d_pool, (size_t)ctx->n_pages * page_bytes_of(c), "kv pool"))) return rc;
  // every slot holds a finite value from the start (a page's slots past its cache length are read
  // as masked keys by the prefill attention, whose zero weights must not meet a NaN)
  CK(ctx, cudaMemset(ctx->d_pool, 0, (size_t)ctx->n_pages * page_bytes_of(c)));
  if (ctx->use_tc && md.page_size == 64 && (md.hd == 64 || md.hd == 128)) {
    if (!make_pool_map(&ctx->map_pool, ctx->d_pool, md))
      return fail(ctx, TLF_ERR_CUDA, "cuTensorMapEncodeTiled failed for the KV pool");
    ctx->has_pool_map = true;
  }
  if ((rc = dev_alloc(ctx, &ctx->d_pos_table, (size_t)ctx->n_pages * md.page_size * 4, "pos table"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_page_table, ctx->h_page_table.size() * 4, "page table"))) return rc;
  CK(ctx, cudaMemset(ctx->d_page_table, 0xFF, ctx->h_page_table.size() * 4));
  if ((rc = dev_alloc(ctx, &ctx->d_len, ctx->h_len.size() * 4, "lengths"))) return rc;
  CK(ctx, cudaMemset(ctx->d_len, 0, ctx->h_len.size() * 4));

  // step workspaces
  ctx->upload_ints = (size_t)3 * B + 2 * (size_t)B * M + 16;
  if ((rc = dev_alloc(ctx, &ctx->d_upload, ctx->upload_ints * 4, "upload"))) return rc;
  CK(ctx, cudaMallocHost((void**)&ctx->h_upload, ctx->upload_ints * 4));
  if ((rc = dev_alloc(ctx, &ctx->d_m, (size_t)B * 4, "m"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_margin, (size_t)B * 4, "margin"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_H, (size_t)B * d * 4, "H"))) return rc;
  {
    // two-term operands (hi + lo planes) for every decode GEMM of the tcgen05 path;
    // TLF_NO_OPERAND_LO=1 keeps one bf16 plane (comparison runs)
    const char* e = getenv("TLF_NO_OPERAND_LO");
    ctx->operand_lo = ctx->use_tc && !(e && e[0] == '1');
  }
  const int planes = ctx->operand_lo ? 2 : 1;
  if ((rc = dev_alloc(ctx, &ctx->d_X, (size_t)planes * B * d * eb, "X"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_O, (size_t)planes * B * md.q_dim * eb, "O"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_U, (size_t)planes * B * ff * eb, "U"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_Xf, (size_t)B * d * eb, "Xf"))) return rc;
  CK(ctx, cudaMemset(ctx->d_X, 0, (size_t)planes * B * d * eb));
  CK(ctx, cudaMemset(ctx->d_O, 0, (size_t)planes * B * md.q_dim * eb));
  CK(ctx, cudaMemset(ctx->d_U, 0, (size_t)planes * B * ff * eb));
  CK(ctx, cudaMemset(ctx->d_Xf, 0, (size_t)B * d * eb));
  if (ctx->use_tc) {
    if (!make_map(&ctx->map_X, ctx->d_X, planes * B, d, d, ctx->nt_max) ||
        !make_map(&ctx->map_O, ctx->d_O, planes * B, md.q_dim, md.q_dim, ctx->nt_max) ||
        !make_map(&ctx->map_U, ctx->d_U, planes * B, ff, ff, ctx->nt_max) ||
        !make_map(&ctx->map_Xf, ctx->d_Xf, B, d, d, ctx->nt_max))
      return fail(ctx, TLF_ERR_CUDA, "cuTensorMapEncodeTiled failed for an activation buffer");
  }
  // split-K factors. tcgen05 path: the largest cluster size (<= 8, the portable
  // limit) whose grid still fits in one wave, counting how many CTAs of the
  // resulting ring depth share an SM (10 % margin for cluster placement).
  if (ctx->use_tc) {
    auto pick = [&](int tiles, int K) {
      const int nkb = (K + 63) / 64;
      for (int S = std::min(8, nkb); S > 1; --S) {
        const int bytes =
            gemm_tc_smem_bytes(ctx->nt_max, gemm_tc_stages(K, S, ctx->nt_max, ctx->operand_lo), ctx->operand_lo);
        const int per_sm = std::min(16, 232448 / (bytes + 1024));
        if (10LL * tiles * S <= 9LL * per_sm * ctx->num_sms) return S;
      }
      return 1;
    };
    ctx->s_qkv = pick((md.qkv_dim + 127) / 128, d);
    ctx->s_o = pick((d + 127) / 128, md.q_dim);
    ctx->s_gu = pick(ctx->wgu[0].N / 128, d);
    ctx->s_d = pick((d + 127) / 128, ff);
  } else {
    const int target = 2 * ctx->num_sms;
    ctx->s_qkv = choose_splits((md.qkv_dim + 63) / 64, (d + 31) / 32, target, ctx->split_cap);
    ctx->s_o = choose_splits((d + 63) / 64, (md.q_dim + 31) / 32, target, 32);
    ctx->s_gu = choose_splits((2 * ff + 63) / 64, (d + 31) / 32, target, ctx->split_cap);
    ctx->s_d = choose_splits((d + 63) / 64, (ff + 31) / 32, target, 32);
  }
  const size_t part_n = std::max((size_t)md.qkv_dim, (size_t)2 * ff);
  if ((rc = dev_alloc(ctx, &ctx->d_part, (size_t)ctx->split_cap * B * part_n * 4, "split-K partials"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_Q, (size_t)B * md.q_dim * 4, "Q"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_idx, (size_t)M * B * 4, "idx"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_n, (size_t)M * 4, "n"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_item_base, (size_t)M * (B + 1) * 4, "item_base"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_nch, (size_t)M * B * 4, "nch"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_chunk, (size_t)M * 4, "chunk"))) return rc;
  ctx->attn_grid = attn_decode_grid(md, ctx->num_sms);
  if ((rc = dev_alloc(ctx, &ctx->d_attn_part, attn_partial_floats(md, ctx->attn_grid) * 4, "attention partials")))
    return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_attn_cnt, (size_t)B * md.Hkv * 4, "attention tickets"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_rowinfo, (size_t)M * B * sizeof(int4), "row info"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_act, (size_t)M * B * 4, "row masks"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_col, (size_t)M * B * 4, "row columns"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_ss, (size_t)split_norm_ldss(d) * B * 4, "norm partial sums"))) return rc;
  CK(ctx, cudaMemset(ctx->d_ss, 0, (size_t)split_norm_ldss(d) * B * 4));
  {
    // TLF_PF_ATTN_V1=1: prefill attention with the thread-staged page ring (comparison runs)
    const char* e = getenv("TLF_PF_ATTN_V1");
    ctx->pf_ws = !(e && e[0] == '1');
  }
  {
    // TLF_NO_SPLIT_NORM=1 keeps every pre-norm a kernel of its own (comparison runs)
    const char* e = getenv("TLF_NO_SPLIT_NORM");
    ctx->split_norm = ctx->use_tc && !(e && e[0] == '1');
  }
  CK(ctx, cudaMemset(ctx->d_attn_cnt, 0, (size_t)B * md.Hkv * 4));
  if ((rc = dev_alloc(ctx, &ctx->d_logits, (size_t)B * V * 4, "logits"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_err, 16, "error word"))) return rc;
  CK(ctx, cudaMemset(ctx->d_err, 0, 16));
  CK(ctx, cudaMallocHost((void**)&ctx->h_m, (size_t)B * 4));
  CK(ctx, cudaMallocHost((void**)&ctx->h_margin, (size_t)B * 4));
  CK(ctx, cudaMallocHost((void**)&ctx->h_err, 16));
  CK(ctx, cudaStreamCreateWithFlags(&ctx->cap_stream, cudaStreamNonBlocking));
  {
    const char* e = getenv("TLF_NO_GRAPH");
    ctx->use_graphs = !(e && e[0] == '1');
  }
  ctx->events.resize(4 + 9 * (size_t)M * J + 2);
  for (auto& e : ctx->events) CK(ctx, cudaEventCreate(&e));
  CK(ctx, cudaDeviceSynchronize());
  return TLF_OK;
}

extern "C" void tlf_destroy(tlf_ctx* ctx) {
  if (!ctx) return;
  if (!ctx->host_only) {
    cudaDeviceSynchronize();
    auto f = [](void* p) { if (p) cudaFree(p); };
    f(ctx->d_emb); f(ctx->d_router_w); f(ctx->d_router_w1); f(ctx->d_router_b1); f(ctx->d_router_b); f(ctx->d_attn_norm); f(ctx->d_mlp_norm);
    f(ctx->d_final_norm); f(ctx->d_inv_freq); f(ctx->d_rope); f(ctx->d_rowinfo); f(ctx->d_act); f(ctx->d_col); f(ctx->d_ss); f(ctx->d_cond);
    for (auto* v : {&ctx->wqkv, &ctx->wo, &ctx->wgu, &ctx->wd})
      for (auto& m : *v) f(m.ptr);
    f(ctx->d_pool); f(ctx->d_pos_table); f(ctx->d_page_table); f(ctx->d_len); f(ctx->d_upload);
    f(ctx->d_m); f(ctx->d_margin); f(ctx->d_H); f(ctx->d_X); f(ctx->d_O); f(ctx->d_U); f(ctx->d_Xf);
    f(ctx->d_part); f(ctx->d_Q); f(ctx->d_idx); f(ctx->d_n); f(ctx->d_item_base); f(ctx->d_nch); f(ctx->d_chunk);
    f(ctx->d_attn_part); f(ctx->d_attn_cnt); f(ctx->d_logits); f(ctx->d_err);
    if (ctx->h_upload) cudaFreeHost(ctx->h_upload);
    if (ctx->h_m) cudaFreeHost(ctx->h_m);
    if (ctx->h_margin) cudaFreeHost(ctx->h_margin);
    if (ctx->h_err) cudaFreeHost(ctx->h_err);
    for (auto e : ctx->events) if (e) cudaEventDestroy(e);
    for (auto& g : ctx->graphs) cudaGraphExecDestroy(g.exec);
    f(ctx->d_pf_in); f(ctx->d_pf_m); f(ctx->d_pf_margin); f(ctx->d_pf_H); f(ctx->d_pf_X); f(ctx->d_pf_Q);
    f(ctx->d_pf_O); f(ctx->d_pf_U); f(ctx->d_pf_idx); f(ctx->d_pf_n); f(ctx->d_pf_row_slot); f(ctx->d_pf_row_cslot);
    f(ctx->d_pf_row_pos); f(ctx->d_pf_first); f(ctx->d_pf_cnt); f(ctx->d_pf_s0); f(ctx->d_pf_tile_base);
    if (ctx->h_pf_in) cudaFreeHost(ctx->h_pf_in);
    if (ctx->h_pf_m) cudaFreeHost(ctx->h_pf_m);
    if (ctx->h_pf_nr) cudaFreeHost(ctx->h_pf_nr);
    if (ctx->cap_stream) cudaStreamDestroy(ctx->cap_stream);
  }
  delete ctx;
}

extern "C" int tlf_create(const tlf_config* cfg, const tlf_weights* w, tlf_ctx** out) {
  if (!out) return fail(nullptr, TLF_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  char msg[256];
  if (tlf_validate_config(cfg, msg, sizeof msg) != TLF_OK) return fail(nullptr, TLF_ERR_INVALID_ARG, "%s", msg);
  tlf_ctx* ctx = new tlf_ctx();
  ctx->cfg = *cfg;
  ctx->host_only = cfg->host_only != 0;
  int rc = create_impl(ctx, w);
  if (rc != TLF_OK) {
    g_create_error = ctx->err;
    tlf_destroy(ctx);
    return rc;
  }
  *out = ctx;
  return TLF_OK;
}

// ----------------------------------------------------------------------------
// sequences and pages
// ----------------------------------------------------------------------------
static inline int& pt_at(tlf_ctx* ctx, int slot, int r, int p) {
  return ctx->h_page_table[((size_t)slot * ctx->md.M + r) * ctx->md.max_pages + p];
}

static void free_slot(tlf_ctx* ctx, int slot) {
  const int M = ctx->md.M, P = ctx->md.max_pages;
  for (int r = 0; r < M; ++r) {
    for (int p = 0; p < P; ++p) {
      int& e = pt_at(ctx, slot, r, p);
      if (e >= 0) {
        ctx->free_pages.push_back(e);
        e = -1;
      }
    }
    ctx->h_len[(size_t)slot * M + r] = 0;
  }
  ctx->free_slots.push_back(slot);
}

extern "C" int tlf_release(tlf_ctx* ctx, uint64_t seq_id) {
  if (!ctx) return TLF_ERR_INVALID_ARG;
  auto it = ctx->seq_slot.find(seq_id);
  if (it == ctx->seq_slot.end()) return fail(ctx, TLF_ERR_UNKNOWN_SEQ, "sequence %llu is not live", (unsigned long long)seq_id);
  free_slot(ctx, it->second);
  ctx->seq_slot.erase(it);
  return TLF_OK;
}

// Check that one cache slot can be reserved in each of the M loops of every row.
static int check_reserve(tlf_ctx* ctx, int B, const int* slots) {
  const int M = ctx->md.M, ps = ctx->md.page_size;
  size_t need = 0;
  for (int b = 0; b < B; ++b) {
    const int s = slots[b];
    if (ctx->h_len[(size_t)s * M] + 1 > ctx->cfg.max_seq_len)
      return fail(ctx, TLF_ERR_SEQ_TOO_LONG, "a sequence would exceed max_seq_len=%d", ctx->cfg.max_seq_len);
    for (int r = 0; r < M; ++r) {
      const int L = ctx->h_len[(size_t)s * M + r];
      if (L % ps == 0 && pt_at(ctx, s, r, L / ps) < 0) ++need;
    }
  }
  if (need > ctx->free_pages.size())
    return fail(ctx, TLF_ERR_OUT_OF_PAGES, "step needs %zu new KV pages, %zu free", need, ctx->free_pages.size());
  return TLF_OK;
}

// Reserve the slots checked by check_reserve; fills the page-table updates of the step.
static int reserve_step(tlf_ctx* ctx, int B, const int* slots, std::vector<PageUpdate>* upd) {
  const int M = ctx->md.M, ps = ctx->md.page_size;
  const int rc = check_reserve(ctx, B, slots);
  if (rc) return rc;
  upd->clear();
  for (int b = 0; b < B; ++b) {
    const int s = slots[b];
    for (int r = 0; r < M; ++r) {
      const int L = ctx->h_len[(size_t)s * M + r];
      int& e = pt_at(ctx, s, r, L / ps);
      if (L % ps == 0 && e < 0) {
        e = ctx->free_pages.back();
        ctx->free_pages.pop_back();
        upd->push_back({(int)(((size_t)s * M + r) * ctx->md.max_pages + L / ps), e});
      }
    }
  }
  return TLF_OK;
}

static int new_slot(tlf_ctx* ctx, uint64_t id, cudaStream_t st) {
  const int slot = ctx->free_slots.back();
  ctx->free_slots.pop_back();
  ctx->seq_slot[id] = slot;
  for (int r = 0; r < ctx->md.M; ++r) ctx->h_len[(size_t)slot * ctx->md.M + r] = 0;
  if (!ctx->host_only) cudaMemsetAsync(ctx->d_len + (size_t)slot * ctx->md.M, 0, ctx->md.M * 4, st);
  return slot;
}

// ----------------------------------------------------------------------------
// one step on the device
// ----------------------------------------------------------------------------
static void gemm(tlf_ctx* ctx, const DeviceMat& W, const CUtensorMap* xmap, const void* X, int ldx, GemmArgs a,
                 cudaStream_t st) {
  a.N = W.N;
  a.K = W.K;
  a.err = ctx->d_err;
  if (ctx->use_tc) launch_gemm_tc(&W.map, xmap, ctx->nt_max, a, st);
  else launch_gemm_simt(ctx->md.dtype, W.ptr, X, ldx, a, st);
  ++ctx->last_launches;
}

// All device work of one step on `st`: upload of the step inputs from the pinned
// buffer, every kernel, and the download of loop counts, margins and the error
// word. Capturable in a CUDA graph (nothing here depends on host values that
// change between steps with the same batch size).
// Lookup of one of the four conditioning vectors (0 alpha_msa, 1 alpha_mlp, 2 gamma_msa,
// 3 gamma_mlp) of layer j at loop r for rows whose loop counts are m; empty without conditioning.
static CondArgs cond_args(const tlf_ctx* ctx, const int* m, int r, int j, int part) {
  CondArgs c;
  if (!ctx->d_cond) return c;
  c.mod = ctx->d_cond;
  c.m = m;
  c.M = ctx->md.M;
  c.d = ctx->md.d;
  c.r = r;
  c.j = j;
  c.part = part;
  return c;
}

static int enqueue_step(tlf_ctx* ctx, int B, bool need_logits, bool prof, cudaStream_t st) {
  const ModelDims& md = ctx->md;
  const int M = md.M, J = md.J, maxB = md.max_batch;
  CK(ctx, cudaMemcpyAsync(ctx->d_upload, ctx->h_upload, ctx->upload_ints * 4, cudaMemcpyHostToDevice, st));

  StepDev s{};
  s.tokens = ctx->d_upload + 1;
  s.forced = ctx->d_upload + 1 + B;
  s.slots = ctx->d_upload + 1 + 2 * B;
  s.m = ctx->d_m;
  s.margin = ctx->d_margin;
  s.H = ctx->d_H;
  s.idx = ctx->d_idx;
  s.n = ctx->d_n;
  s.item_base = ctx->d_item_base;
  s.nch = ctx->d_nch;
  s.chunk = ctx->d_chunk;
  s.len = ctx->d_len;
  s.page_table = ctx->d_page_table;
  s.pos_table = ctx->d_pos_table;
  s.pool = ctx->d_pool;
  s.err = ctx->d_err;
  s.cnt = ctx->d_attn_cnt;
  s.rowinfo = ctx->d_rowinfo;
  s.act = ctx->d_act;
  s.col = ctx->d_col;
  const PageUpdate* d_upd = reinterpret_cast<const PageUpdate*>(ctx->d_upload + 1 + 3 * B);

  ctx->last_launches = 0;
  int ev = 0;
  ctx->ev_class.clear();
  // profiling: an event after every launch, tagged with the kernel class it closes
  auto mark = [&](int cls) {
    if (!prof) return;
    cudaEventRecord(ctx->events[ev++], st);
    if (cls >= 0) ctx->ev_class.push_back(cls);
  };
  mark(-1);
  launch_router(md, s, B, ctx->d_emb, ctx->d_router_w, ctx->d_router_b, d_upd, ctx->d_upload, st, ctx->d_router_w1,
                ctx->d_router_b1);
  mark(0);
  launch_plan(md, s, B, st);
  mark(1);
  ctx->last_launches += 2;
  // two-term GEMM operands: lo planes of X, U (and O, written by the attention kernel) sit
  // max_batch rows below the hi planes
  const int lo_rows = ctx->operand_lo ? maxB : 0;
  void* x_lo = ctx->operand_lo ? static_cast<void*>(reinterpret_cast<bf16*>(ctx->d_X) + (size_t)maxB * md.d) : nullptr;
  void* u_lo = ctx->operand_lo ? static_cast<void*>(reinterpret_cast<bf16*>(ctx->d_U) + (size_t)maxB * md.ff) : nullptr;
  for (int r = 0; r < M; ++r) {
    const int* n_dev = ctx->d_n + r;
    const int* idx_r = ctx->d_idx + (size_t)r * maxB;
    // rows that do not run loop r but are computed anyway (no-gather ablation) keep their residual
    const int* act_r = md.ablation == TLF_ABLATION_NO_GATHER ? ctx->d_act + (size_t)r * maxB : nullptr;
    for (int j = 0; j < J; ++j) {
      // Split pre-norms: after the first, each norm's operand and partial sums are written by the
      // residual epilogue before it and its factor applied by the GEMM after it.
      const bool split = ctx->split_norm;
      if (!split || (r == 0 && j == 0)) {
        launch_norm_rows(md.dtype, ctx->d_H, md.d, idx_r, n_dev, 0, maxB, ctx->d_attn_norm + (size_t)j * md.d, md.d,
                         md.eps, ctx->d_X, md.d, st, cond_args(ctx, s.m, r, j, 2), split ? ctx->d_ss : nullptr,
                         x_lo);
        ++ctx->last_launches;
        mark(2);
      }
      GemmArgs a{};
      a.n_dev = n_dev;
      a.max_rows = maxB;
      a.splits = ctx->s_qkv;
      a.blo = lo_rows;
      if (split) {
        a.ss_in = ctx->d_ss;
        a.ldss = split_norm_ldss(md.d);
        a.norm_eps = md.eps;
      }
      if (ctx->use_tc) {
        // split-K reduction, RoPE and the K/V append run in the GEMM's cluster epilogue
        a.epi = EPI_CL_QKV;
        a.md = md;
        a.s = s;
        a.r = r;
        a.j = j;
        a.rope = ctx->d_rope;
        a.Q = ctx->d_Q;
        gemm(ctx, ctx->wqkv[j], &ctx->map_X, ctx->d_X, md.d, a, st);
        mark(3);
      } else {
        a.epi = EPI_PARTIAL;
        a.out = ctx->d_part;
        gemm(ctx, ctx->wqkv[j], &ctx->map_X, ctx->d_X, md.d, a, st);
        mark(3);
        launch_rope_append(md, s, r, j, ctx->d_part, ctx->s_qkv, ctx->d_Q, ctx->d_rope, st);
        ++ctx->last_launches;
        mark(4);
      }
      launch_attn_decode(md, s, r, j, ctx->d_Q, ctx->d_attn_part, ctx->d_O, ctx->d_attn_cnt, ctx->attn_grid, st,
                         ctx->operand_lo);
      mark(5);
      a = GemmArgs{};
      a.n_dev = n_dev;
      a.max_rows = maxB;
      a.epi = ctx->use_tc ? EPI_CL_RESID : EPI_RESID;
      a.resid = ctx->d_H;
      a.ldr = md.d;
      a.idx = idx_r;
      a.act = act_r;
      a.alpha = cond_args(ctx, s.m, r, j, 0);
      a.splits = ctx->s_o;
      a.blo = lo_rows;
      if (split) {  // the MLP pre-norm of this layer, same rows
        a.xn = reinterpret_cast<bf16*>(ctx->d_X);
        a.xn_lo = reinterpret_cast<bf16*>(x_lo);
        a.ss_out = ctx->d_ss;
        a.ldss = split_norm_ldss(md.d);
        a.gain = ctx->d_mlp_norm + (size_t)j * md.d;
        a.gamma = cond_args(ctx, s.m, r, j, 3);
      }
      gemm(ctx, ctx->wo[j], &ctx->map_O, ctx->d_O, md.q_dim, a, st);
      mark(6);
      if (!split) {
        launch_norm_rows(md.dtype, ctx->d_H, md.d, idx_r, n_dev, 0, maxB, ctx->d_mlp_norm + (size_t)j * md.d, md.d,
                         md.eps, ctx->d_X, md.d, st, cond_args(ctx, s.m, r, j, 3), nullptr, x_lo);
        ++ctx->last_launches;
        mark(7);
      }
      a = GemmArgs{};
      a.n_dev = n_dev;
      a.max_rows = maxB;
      a.splits = ctx->s_gu;
      a.blo = lo_rows;
      if (split) {
        a.ss_in = ctx->d_ss;
        a.ldss = split_norm_ldss(md.d);
        a.norm_eps = md.eps;
      }
      if (ctx->use_tc) {
        a.epi = EPI_CL_SWIGLU;  // SwiGLU in the cluster epilogue
        a.md = md;
        a.U = ctx->d_U;
        a.U_lo = u_lo;
        gemm(ctx, ctx->wgu[j], &ctx->map_X, ctx->d_X, md.d, a, st);
        mark(8);
      } else {
        a.epi = EPI_PARTIAL;
        a.out = ctx->d_part;
        gemm(ctx, ctx->wgu[j], &ctx->map_X, ctx->d_X, md.d, a, st);
        mark(8);
        launch_swiglu(md.dtype, ctx->d_part, ctx->s_gu, maxB, n_dev, md.ff, ctx->d_U, st);
        ++ctx->last_launches;
        mark(9);
      }
      a = GemmArgs{};
      a.n_dev = n_dev;
      a.max_rows = maxB;
      a.epi = ctx->use_tc ? EPI_CL_RESID : EPI_RESID;
      a.resid = ctx->d_H;
      a.ldr = md.d;
      a.idx = idx_r;
      a.act = act_r;
      a.alpha = cond_args(ctx, s.m, r, j, 1);
      a.splits = ctx->s_d;
      a.blo = lo_rows;
      if (split && (j + 1 < J || r + 1 < M)) {
        // the attention pre-norm of the next layer, or of layer 0 of loop r + 1 for the rows
        // that continue (they move to their compact row of A_{r+1})
        const int rn = j + 1 < J ? r : r + 1, jn = j + 1 < J ? j + 1 : 0;
        a.xn = reinterpret_cast<bf16*>(ctx->d_X);
        a.xn_lo = reinterpret_cast<bf16*>(x_lo);
        a.ss_out = ctx->d_ss;
        a.ldss = split_norm_ldss(md.d);
        a.gain = ctx->d_attn_norm + (size_t)jn * md.d;
        a.gamma = cond_args(ctx, s.m, rn, jn, 2);
        a.next_col = rn != r ? ctx->d_col + (size_t)rn * maxB : nullptr;
      }
      gemm(ctx, ctx->wd[j], &ctx->map_U, ctx->d_U, md.ff, a, st);
      mark(10);
      ++ctx->last_launches;  // the attention (GEMMs counted in gemm(), norms where launched)
    }
  }
  launch_final(md, s, B, ctx->d_final_norm, ctx->d_Xf, st);
  mark(11);
  ++ctx->last_launches;
  if (need_logits) {
    GemmArgs a{};
    a.n_host = B;
    a.max_rows = maxB;
    a.epi = EPI_STORE;
    a.out = ctx->d_logits;
    a.ldo = md.V;
    a.splits = 1;
    gemm(ctx, ctx->emb_mat, &ctx->map_Xf, ctx->d_Xf, md.d, a, st);
    mark(12);
  }
  CK(ctx, cudaGetLastError());
  CK(ctx, cudaMemcpyAsync(ctx->h_m, ctx->d_m, (size_t)B * 4, cudaMemcpyDeviceToHost, st));
  CK(ctx, cudaMemcpyAsync(ctx->h_margin, ctx->d_margin, (size_t)B * 4, cudaMemcpyDeviceToHost, st));
  CK(ctx, cudaMemcpyAsync(ctx->h_err, ctx->d_err, 4, cudaMemcpyDeviceToHost, st));
  return TLF_OK;
}

// The step as one CUDA graph per (batch size, logits on/off), built on first
// use after the kernels have run once directly (their attributes are set).
static cudaGraphExec_t step_graph(tlf_ctx* ctx, int B, bool need_logits) {
  for (auto& g : ctx->graphs)
    if (g.B == B && g.logits == need_logits) {
      ctx->last_launches = g.launches;
      return g.exec;
    }
  if (!ctx->use_graphs || !ctx->warmed || ctx->graphs.size() >= 32) return nullptr;
  cudaGraph_t graph = nullptr;
  cudaGraphExec_t exec = nullptr;
  if (cudaStreamBeginCapture(ctx->cap_stream, cudaStreamCaptureModeThreadLocal) != cudaSuccess) {
    cudaGetLastError();
    ctx->use_graphs = false;
    return nullptr;
  }
  const int rc = enqueue_step(ctx, B, need_logits, false, ctx->cap_stream);
  const cudaError_t e1 = cudaStreamEndCapture(ctx->cap_stream, &graph);
  if (rc != TLF_OK || e1 != cudaSuccess || cudaGraphInstantiate(&exec, graph, 0) != cudaSuccess) {
    cudaGetLastError();
    if (graph) cudaGraphDestroy(graph);
    ctx->use_graphs = false;  // run the kernels directly from now on
    return nullptr;
  }
  cudaGraphDestroy(graph);
  ctx->graphs.push_back({B, need_logits, exec, ctx->last_launches});
  return exec;
}

static int run_step(tlf_ctx* ctx, int B, const int* slots, const int* tokens, const int* forced,
                    const std::vector<PageUpdate>& upd, bool need_logits, cudaStream_t st) {
  const ModelDims& md = ctx->md;
  const int M = md.M, J = md.J;
  const bool prof = ctx->profiling;
  int* h = ctx->h_upload;
  const size_t nu = upd.size();
  h[0] = (int)nu;
  for (int b = 0; b < B; ++b) {
    h[1 + b] = tokens[b];
    h[1 + B + b] = forced ? forced[b] : -1;
    h[1 + 2 * B + b] = slots[b];
  }
  memcpy(h + 1 + 3 * B, upd.data(), nu * sizeof(PageUpdate));
  cudaGraphExec_t exec = prof ? nullptr : step_graph(ctx, B, need_logits);
  if (exec) {
    CK(ctx, cudaGraphLaunch(exec, st));
  } else {
    const int rc = enqueue_step(ctx, B, need_logits, prof, st);
    if (rc) return rc;
    ctx->warmed = true;
  }
  CK(ctx, cudaStreamSynchronize(st));
  if (*ctx->h_err) {
    const uint32_t e = *ctx->h_err;
    cudaMemsetAsync(ctx->d_err, 0, 4, st);
    return fail(ctx, TLF_ERR_DEVICE, "device error word 0x%x (1 = bounded wait expired, 2 = bad index)", e);
  }
  if (prof) {
    for (float& c : ctx->class_ms) c = 0.f;
    for (size_t i = 0; i < ctx->ev_class.size(); ++i) {
      float ms = 0.f;
      cudaEventElapsedTime(&ms, ctx->events[i], ctx->events[i + 1]);
      ctx->class_ms[ctx->ev_class[i]] += ms;
    }
    ctx->last_attn_ms = ctx->class_ms[5];
    // KV bytes visited: for every row b and loop r < m_b, (len + 1) entries x J layers x K,V;
    // without the gather, every loop that runs also reads the caches of the exited rows
    double bytes = 0.0;
    int loops_run = 0;
    for (int b = 0; b < B; ++b) loops_run = std::max(loops_run, ctx->h_m[b]);
    for (int b = 0; b < B; ++b)
      for (int r = 0; r < (md.ablation == TLF_ABLATION_NO_GATHER ? loops_run : ctx->h_m[b]); ++r) {
        const double keys = ctx->h_len[(size_t)slots[b] * M + r] + (r < ctx->h_m[b] ? 1 : 0);
        bytes += keys * J * 2.0 * md.Hkv * md.hd * ctx->eb;
        // a full-length cache (dense-cache ablation) also reads each page's 64 positions per kv head
        if (md.ablation == TLF_ABLATION_DENSE_CACHE)
          bytes += std::ceil(keys / md.page_size) * J * md.Hkv * md.page_size * 4.0;
      }
    ctx->last_attn_bytes = bytes;
  }
  ctx->last_batch = B;
  return TLF_OK;
}

static void advance_lengths(tlf_ctx* ctx, int B, const int* slots) {
  const int M = ctx->md.M;
  const bool dense = ctx->md.ablation == TLF_ABLATION_DENSE_CACHE;  // every cache holds a slot per token
  for (int b = 0; b < B; ++b)
    for (int r = 0; r < (dense ? M : ctx->h_m[b]); ++r) ctx->h_len[(size_t)slots[b] * M + r] += 1;
}

// ----------------------------------------------------------------------------
// public calls
// ----------------------------------------------------------------------------
extern "C" int tlf_decode_step(tlf_ctx* ctx, int32_t batch, const uint64_t* seq_ids, const int32_t* tokens,
                               const int32_t* forced, float* logits, int32_t* loops, float* router_margin,
                               void* stream) {
  if (!ctx) return TLF_ERR_INVALID_ARG;
  if (batch < 1 || batch > ctx->cfg.max_batch)
    return fail(ctx, TLF_ERR_CAPACITY, "batch %d not in 1..max_batch=%d", batch, ctx->cfg.max_batch);
  if (!seq_ids || !tokens || !loops) return fail(ctx, TLF_ERR_INVALID_ARG, "seq_ids, tokens and loops are required");
  std::vector<int> slots(batch);
  std::unordered_set<uint64_t> seen;
  for (int b = 0; b < batch; ++b) {
    if (tokens[b] < 0 || tokens[b] >= ctx->md.V) return fail(ctx, TLF_ERR_INVALID_ARG, "token %d out of range", tokens[b]);
    if (forced && forced[b] > ctx->md.M) return fail(ctx, TLF_ERR_INVALID_ARG, "forced loop count %d > max_loops", forced[b]);
    auto it = ctx->seq_slot.find(seq_ids[b]);
    if (it == ctx->seq_slot.end())
      return fail(ctx, TLF_ERR_UNKNOWN_SEQ, "sequence %llu is not live", (unsigned long long)seq_ids[b]);
    if (!seen.insert(seq_ids[b]).second)
      return fail(ctx, TLF_ERR_INVALID_ARG, "sequence %llu appears twice in the batch", (unsigned long long)seq_ids[b]);
    slots[b] = it->second;
  }
  int rc = check_reserve(ctx, batch, slots.data());
  if (rc) return rc;
  if (ctx->host_only) return fail(ctx, TLF_ERR_NO_DEVICE, "host-only context cannot run a decode step");
  std::vector<PageUpdate> upd;
  rc = reserve_step(ctx, batch, slots.data(), &upd);
  if (rc) return rc;
  cudaStream_t st = (cudaStream_t)stream;
  const bool want = logits != nullptr;
  rc = run_step(ctx, batch, slots.data(), tokens, forced, upd, want, st);
  if (rc) return rc;
  advance_lengths(ctx, batch, slots.data());
  for (int b = 0; b < batch; ++b) loops[b] = ctx->h_m[b];
  if (router_margin) memcpy(router_margin, ctx->h_margin, (size_t)batch * 4);
  if (want) {
    const size_t bytes = (size_t)batch * ctx->md.V * 4;
    if (is_device_ptr(logits)) CK(ctx, cudaMemcpyAsync(logits, ctx->d_logits, bytes, cudaMemcpyDeviceToDevice, st));
    else CK(ctx, cudaMemcpyAsync(logits, ctx->d_logits, bytes, cudaMemcpyDeviceToHost, st));
    CK(ctx, cudaStreamSynchronize(st));
  }
  return TLF_OK;
}

// ----------------------------------------------------------------------------
// batched prefill (tensor-core models)
// ----------------------------------------------------------------------------
static int ensure_prefill_buffers(tlf_ctx* ctx) {
  if (ctx->pf_C) return TLF_OK;
  const ModelDims& md = ctx->md;
  int C = ctx->cfg.prefill_chunk > 0 ? ctx->cfg.prefill_chunk : 8192;
  C = (C + 255) / 256 * 256;
  const int Smax = std::min(1024, std::min(C, ctx->cfg.max_seqs));
  const int M = md.M, d = md.d;
  const size_t max_upd = (size_t)M * (C / 64 + 2 * (size_t)Smax);
  ctx->pf_in_ints = 1 + 4 * (size_t)C + 2 * (size_t)Smax + 2 * max_upd;
  int rc;
  if ((rc = dev_alloc(ctx, &ctx->d_pf_in, ctx->pf_in_ints * 4, "prefill inputs"))) return rc;
  CK(ctx, cudaMallocHost((void**)&ctx->h_pf_in, ctx->pf_in_ints * 4));
  CK(ctx, cudaMallocHost((void**)&ctx->h_pf_m, (size_t)C * 4));
  CK(ctx, cudaMallocHost((void**)&ctx->h_pf_nr, (size_t)M * 4));
  if ((rc = dev_alloc(ctx, &ctx->d_pf_m, (size_t)C * 4, "prefill m"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_pf_margin, (size_t)C * 4, "prefill margin"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_pf_H, (size_t)C * d * 4, "prefill H"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_pf_X, (size_t)C * d * 2, "prefill X"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_pf_Q, (size_t)C * md.q_dim * 4, "prefill Q"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_pf_O, (size_t)C * md.q_dim * 2, "prefill O"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_pf_U, (size_t)C * md.ff * 2, "prefill U"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_pf_idx, (size_t)M * C * 4, "prefill idx"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_pf_row_slot, (size_t)M * C * 4, "prefill rows"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_pf_row_cslot, (size_t)M * C * 4, "prefill rows"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_pf_row_pos, (size_t)M * C * 4, "prefill rows"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_pf_n, (size_t)M * 4, "prefill n"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_pf_first, (size_t)M * Smax * 4, "prefill seqs"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_pf_cnt, (size_t)M * Smax * 4, "prefill seqs"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_pf_s0, (size_t)M * Smax * 4, "prefill seqs"))) return rc;
  if ((rc = dev_alloc(ctx, &ctx->d_pf_tile_base, (size_t)M * (Smax + 1) * 4, "prefill tiles"))) return rc;
  CK(ctx, cudaMemset(ctx->d_pf_X, 0, (size_t)C * d * 2));
  CK(ctx, cudaMemset(ctx->d_pf_O, 0, (size_t)C * md.q_dim * 2));
  CK(ctx, cudaMemset(ctx->d_pf_U, 0, (size_t)C * md.ff * 2));
  if (!make_map(&ctx->pf_map_X, ctx->d_pf_X, C, d, d, 256) ||
      !make_map(&ctx->pf_map_O, ctx->d_pf_O, C, md.q_dim, md.q_dim, 256) ||
      !make_map(&ctx->pf_map_U, ctx->d_pf_U, C, md.ff, md.ff, 256))
    return fail(ctx, TLF_ERR_CUDA, "cuTensorMapEncodeTiled failed for a prefill buffer");
  ctx->pf_C = C;
  ctx->pf_Smax = Smax;
  return TLF_OK;
}

// rows: the chunk's token count (an upper bound on the rows of every loop)
static void gemm_pf(tlf_ctx* ctx, const DeviceMat& W, const CUtensorMap* xmap, GemmArgs a, int rows,
                    cudaStream_t st) {
  a.N = W.N;
  a.K = W.K;
  a.err = ctx->d_err;
  a.splits = 1;
  const int ntiles = (W.N + 127) / 128, ttiles = (rows + 255) / 256;
  // A chunk of few token tiles (a short prompt) would stream the weights through few CTAs, one per
  // (128-row tile, token tile): K is split over a cluster instead (up to 8 CTAs, at least two k-tiles
  // each), as in the decode step, while the tiles x splits still fit one CTA per SM.
  if (a.epi >= EPI_CL_RESID) {
    const int nkb = (W.K + 63) / 64;
    while (a.splits < 8 && (long long)ntiles * ttiles * a.splits * 2 <= ctx->num_sms && nkb >= 4 * a.splits)
      a.splits *= 2;
  }
  // Stage 128 of the 256 token columns at a time (2-stage ring): two CTAs share an SM, so one
  // CTA's epilogue overlaps the other's main loop. Only worth it when the grid has more tiles
  // than SMs; a smaller grid keeps one CTA per SM and the deeper ring.
  const long long tiles = (long long)ntiles * ttiles;
  a.red_window = (a.splits == 1 && tiles > ctx->num_sms) ? 128 : 0;
  a.max_rows = ctx->pf_C;
  // token tiles of the chunk's rows (every loop's rows are among them), not of its capacity: a short
  // prompt would otherwise launch a grid of CTAs that only wait for the kernel before and exit
  a.tok_tiles = ttiles;
  launch_gemm_tc(&W.map, xmap, 256, a, st);
}

// Prompts of the (already created) sequences slot_of[0..n), chunk by chunk: every chunk is routed,
// runs all loops on its gathered tokens (Eq. 6-7) with causal attention over each sequence's
// loop caches (Eq. 10), and appends its k, v at the following cache slots (Eq. 11, App. B).
static int prefill_batched(tlf_ctx* ctx, int n_seqs, const int* slot_of, const int32_t* offsets,
                           const int32_t* tokens, const int32_t* forced, float* last_logits, bool logits_dev,
                           int32_t* loops, cudaStream_t st) {
  int rc = ensure_prefill_buffers(ctx);
  if (rc) return rc;
  const ModelDims& md = ctx->md;
  const int M = md.M, J = md.J, C = ctx->pf_C, Smax = ctx->pf_Smax, ps = md.page_size, maxB = md.max_batch;
  struct Seg {
    int s, start, count;
  };
  int s_next = 0, pos_next = 0;
  while (s_next < n_seqs) {
    std::vector<Seg> segs;
    int T = 0;
    while (s_next < n_seqs && T < C && (int)segs.size() < Smax) {
      const int len = offsets[s_next + 1] - offsets[s_next];
      const int take = std::min(len - pos_next, C - T);
      segs.push_back({s_next, pos_next, take});
      T += take;
      pos_next += take;
      if (pos_next == len) {
        ++s_next;
        pos_next = 0;
      }
    }
    const int S = (int)segs.size();
    // pages: worst case (every chunk token runs every loop); trimmed once the loop counts are known
    size_t need = 0;
    for (const Seg& g : segs)
      for (int r = 0; r < M; ++r) {
        const int L = ctx->h_len[(size_t)slot_of[g.s] * M + r];
        for (int p = L / ps; p <= (L + g.count - 1) / ps; ++p)
          if (pt_at(ctx, slot_of[g.s], r, p) < 0) ++need;
      }
    if (need > ctx->free_pages.size())
      return fail(ctx, TLF_ERR_OUT_OF_PAGES, "prefill chunk needs %zu KV pages, %zu free", need,
                  ctx->free_pages.size());
    int* h = ctx->h_pf_in;
    int* h_upd = h + 1 + 4 * C + 2 * Smax;
    int nu = 0;
    for (const Seg& g : segs)
      for (int r = 0; r < M; ++r) {
        const int slot = slot_of[g.s];
        const int L = ctx->h_len[(size_t)slot * M + r];
        for (int p = L / ps; p <= (L + g.count - 1) / ps; ++p) {
          int& e = pt_at(ctx, slot, r, p);
          if (e < 0) {
            e = ctx->free_pages.back();
            ctx->free_pages.pop_back();
            h_upd[2 * nu] = (int)(((size_t)slot * M + r) * md.max_pages + p);
            h_upd[2 * nu + 1] = e;
            ++nu;
          }
        }
      }
    h[0] = nu;
    std::vector<int> ending;  // prompts whose last token is in this chunk
    int nend = 0;
    for (int si = 0, t = 0; si < S; ++si) {
      const Seg& g = segs[si];
      for (int i = 0; i < g.count; ++i, ++t) {
        const int gi = offsets[g.s] + g.start + i;
        h[1 + t] = tokens[gi];
        h[1 + C + t] = forced ? forced[gi] : -1;
        h[1 + 2 * C + t] = si;
        h[1 + 3 * C + t] = g.start + i;
      }
      h[1 + 4 * C + si] = slot_of[g.s];
      if (g.start + g.count == offsets[g.s + 1] - offsets[g.s]) {
        h[1 + 4 * C + Smax + nend++] = t - 1;
        ending.push_back(g.s);
      }
    }
    CK(ctx, cudaMemcpyAsync(ctx->d_pf_in, h, (size_t)(1 + 4 * C + 2 * Smax + 2 * nu) * 4, cudaMemcpyHostToDevice, st));

    StepDev sr{};
    sr.tokens = ctx->d_pf_in + 1;
    sr.forced = ctx->d_pf_in + 1 + C;
    sr.m = ctx->d_pf_m;
    sr.margin = ctx->d_pf_margin;
    sr.H = ctx->d_pf_H;
    sr.page_table = ctx->d_page_table;
    sr.err = ctx->d_err;
    launch_router(md, sr, T, ctx->d_emb, ctx->d_router_w, ctx->d_router_b,
                  reinterpret_cast<const PageUpdate*>(ctx->d_pf_in + 1 + 4 * C + 2 * Smax), ctx->d_pf_in, st,
                  ctx->d_router_w1, ctx->d_router_b1);
    PrefillDev P{};
    P.T = T;
    P.S = S;
    P.C = C;
    P.Smax = Smax;
    P.seqidx = ctx->d_pf_in + 1 + 2 * C;
    P.pos = ctx->d_pf_in + 1 + 3 * C;
    P.seq_slot = ctx->d_pf_in + 1 + 4 * C;
    P.m = ctx->d_pf_m;
    P.idx = ctx->d_pf_idx;
    P.n = ctx->d_pf_n;
    P.row_slot = ctx->d_pf_row_slot;
    P.row_cslot = ctx->d_pf_row_cslot;
    P.row_pos = ctx->d_pf_row_pos;
    P.first = ctx->d_pf_first;
    P.cnt = ctx->d_pf_cnt;
    P.s0 = ctx->d_pf_s0;
    P.tile_base = ctx->d_pf_tile_base;
    P.qblock = pf_attn_qblock(md);
    P.len = ctx->d_len;
    launch_pf_plan(md, P, st);
    // For a chunk of more than one 256-token tile, the rows of every loop come to the host: each
    // loop's grids follow them (deeper loops hold fewer of the chunk's tokens, so their grids shrink
    // and their GEMMs may split K), and a loop that no token reaches launches nothing. A chunk of one
    // tile has nothing to shrink and skips the wait.
    const bool per_loop_rows = T > 256;
    if (per_loop_rows) {
      CK(ctx, cudaMemcpyAsync(ctx->h_pf_nr, ctx->d_pf_n, (size_t)M * 4, cudaMemcpyDeviceToHost, st));
      CK(ctx, cudaStreamSynchronize(st));
    }
    StepDev sp{};
    sp.page_table = ctx->d_page_table;
    sp.pool = ctx->d_pool;
    sp.pos_table = ctx->d_pos_table;
    sp.len = ctx->d_len;
    sp.err = ctx->d_err;
    for (int r = 0; r < M; ++r) {
      const int* n_dev = ctx->d_pf_n + r;
      const int* idx_r = ctx->d_pf_idx + (size_t)r * C;
      // rows of loop r (the kernels read the count itself from n_dev)
      const int nr = per_loop_rows ? std::min(std::max(ctx->h_pf_nr[r], 0), T) : T;
      if (nr == 0) continue;
      for (int j = 0; j < J; ++j) {
        // one CTA per row of the loop
        launch_norm_rows(md.dtype, ctx->d_pf_H, md.d, idx_r, n_dev, 0, nr, ctx->d_attn_norm + (size_t)j * md.d, md.d,
                         md.eps, ctx->d_pf_X, md.d, st, cond_args(ctx, ctx->d_pf_m, r, j, 2));
        GemmArgs a{};
        a.n_dev = n_dev;
        a.epi = EPI_CL_QKV;
        a.md = md;
        a.s = sp;
        a.r = r;
        a.j = j;
        a.rope = ctx->d_rope;
        a.Q = ctx->d_pf_Q;
        a.row_slot = ctx->d_pf_row_slot + (size_t)r * C;
        a.row_cslot = ctx->d_pf_row_cslot + (size_t)r * C;
        a.row_pos = ctx->d_pf_row_pos + (size_t)r * C;
        gemm_pf(ctx, ctx->wqkv[j], &ctx->pf_map_X, a, nr, st);
        // attention blocks of loop r: sum over sequences of ceil(count / qblock) <= nr / qblock + S
        launch_pf_attn(md, P, sp, r, j, ctx->d_pf_Q, ctx->d_pf_O, nr / P.qblock + S + 1, st,
                       ctx->has_pool_map && ctx->pf_ws ? &ctx->map_pool : nullptr);
        a = GemmArgs{};
        a.n_dev = n_dev;
        a.epi = EPI_CL_RESID;
        a.resid = ctx->d_pf_H;
        a.ldr = md.d;
        a.idx = idx_r;
        a.alpha = cond_args(ctx, ctx->d_pf_m, r, j, 0);
        gemm_pf(ctx, ctx->wo[j], &ctx->pf_map_O, a, nr, st);
        launch_norm_rows(md.dtype, ctx->d_pf_H, md.d, idx_r, n_dev, 0, nr, ctx->d_mlp_norm + (size_t)j * md.d, md.d,
                         md.eps, ctx->d_pf_X, md.d, st, cond_args(ctx, ctx->d_pf_m, r, j, 3));
        a = GemmArgs{};
        a.n_dev = n_dev;
        a.epi = EPI_CL_SWIGLU;
        a.md = md;
        a.U = ctx->d_pf_U;
        gemm_pf(ctx, ctx->wgu[j], &ctx->pf_map_X, a, nr, st);
        a = GemmArgs{};
        a.n_dev = n_dev;
        a.epi = EPI_CL_RESID;
        a.resid = ctx->d_pf_H;
        a.ldr = md.d;
        a.idx = idx_r;
        a.alpha = cond_args(ctx, ctx->d_pf_m, r, j, 1);
        gemm_pf(ctx, ctx->wd[j], &ctx->pf_map_U, a, nr, st);
      }
    }
    if (last_logits && nend > 0) {
      for (int e0 = 0; e0 < nend; e0 += maxB) {
        const int cnt = std::min(maxB, nend - e0);
        launch_norm_rows(md.dtype, ctx->d_pf_H, md.d, ctx->d_pf_in + 1 + 4 * C + Smax + e0, nullptr, cnt, cnt,
                         ctx->d_final_norm, md.d, md.eps, ctx->d_Xf, md.d, st);
        GemmArgs a{};
        a.n_host = cnt;
        a.max_rows = maxB;
        a.epi = EPI_STORE;
        a.out = ctx->d_logits;
        a.ldo = md.V;
        a.splits = 1;
        gemm(ctx, ctx->emb_mat, &ctx->map_Xf, ctx->d_Xf, md.d, a, st);
        for (int e = 0; e < cnt; ++e)
          CK(ctx, cudaMemcpyAsync(last_logits + (size_t)ending[e0 + e] * md.V, ctx->d_logits + (size_t)e * md.V,
                                  (size_t)md.V * 4, logits_dev ? cudaMemcpyDeviceToDevice : cudaMemcpyDeviceToHost,
                                  st));
      }
    }
    launch_pf_len(md, P, st);
    CK(ctx, cudaGetLastError());
    CK(ctx, cudaMemcpyAsync(ctx->h_pf_m, ctx->d_pf_m, (size_t)T * 4, cudaMemcpyDeviceToHost, st));
    CK(ctx, cudaMemcpyAsync(ctx->h_err, ctx->d_err, 4, cudaMemcpyDeviceToHost, st));
    CK(ctx, cudaStreamSynchronize(st));
    if (*ctx->h_err) {
      const uint32_t e = *ctx->h_err;
      cudaMemsetAsync(ctx->d_err, 0, 4, st);
      return fail(ctx, TLF_ERR_DEVICE, "device error word 0x%x during prefill", e);
    }
    // loop counts out, host lengths, and the pages the worst-case reservation did not need
    for (int si = 0, t = 0; si < S; ++si) {
      const Seg& g = segs[si];
      const int slot = slot_of[g.s];
      for (int i = 0; i < g.count; ++i, ++t) {
        const int m = ctx->h_pf_m[t];
        if (loops) loops[offsets[g.s] + g.start + i] = m;
        for (int r = 0; r < m; ++r) ctx->h_len[(size_t)slot * M + r] += 1;
      }
      for (int r = 0; r < M; ++r) {
        const int keep = (ctx->h_len[(size_t)slot * M + r] + ps - 1) / ps;
        for (int p = keep; p < md.max_pages; ++p) {
          int& e = pt_at(ctx, slot, r, p);
          if (e < 0) break;
          ctx->free_pages.push_back(e);
          e = -1;
        }
      }
    }
  }
  return TLF_OK;
}

extern "C" int tlf_prefill(tlf_ctx* ctx, int32_t n_seqs, const uint64_t* seq_ids, const int32_t* offsets,
                           const int32_t* tokens, const int32_t* forced, float* last_logits, int32_t* loops,
                           void* stream) {
  if (!ctx) return TLF_ERR_INVALID_ARG;
  if (n_seqs < 1 || !seq_ids || !offsets || !tokens)
    return fail(ctx, TLF_ERR_INVALID_ARG, "n_seqs >= 1 and seq_ids, offsets, tokens are required");
  if ((size_t)n_seqs > ctx->free_slots.size())
    return fail(ctx, TLF_ERR_CAPACITY, "%d new sequences but only %zu free slots", n_seqs, ctx->free_slots.size());
  std::unordered_set<uint64_t> seen;
  if (offsets[0] != 0) return fail(ctx, TLF_ERR_INVALID_ARG, "offsets[0] must be 0");
  for (int s = 0; s < n_seqs; ++s) {
    const int len = offsets[s + 1] - offsets[s];
    if (len < 1) return fail(ctx, TLF_ERR_INVALID_ARG, "prompt %d is empty", s);
    if (len > ctx->cfg.max_seq_len) return fail(ctx, TLF_ERR_SEQ_TOO_LONG, "prompt %d longer than max_seq_len", s);
    if (ctx->seq_slot.count(seq_ids[s])) return fail(ctx, TLF_ERR_DUPLICATE_SEQ, "sequence %llu is live", (unsigned long long)seq_ids[s]);
    if (!seen.insert(seq_ids[s]).second) return fail(ctx, TLF_ERR_INVALID_ARG, "sequence id repeated in the call");
  }
  for (int i = 0; i < offsets[n_seqs]; ++i) {
    if (tokens[i] < 0 || tokens[i] >= ctx->md.V) return fail(ctx, TLF_ERR_INVALID_ARG, "token %d out of range", tokens[i]);
    if (forced && forced[i] > ctx->md.M) return fail(ctx, TLF_ERR_INVALID_ARG, "forced loop count > max_loops");
  }
  if (ctx->host_only) return fail(ctx, TLF_ERR_NO_DEVICE, "host-only context cannot run a prefill");
  cudaStream_t st = (cudaStream_t)stream;
  std::vector<int> slot_of(n_seqs);
  for (int s = 0; s < n_seqs; ++s) slot_of[s] = new_slot(ctx, seq_ids[s], st);
  auto rollback = [&](int rc) {
    for (int s = 0; s < n_seqs; ++s) {
      free_slot(ctx, slot_of[s]);
      ctx->seq_slot.erase(seq_ids[s]);
    }
    return rc;
  };
  const bool logits_dev = last_logits && is_device_ptr(last_logits);
  if (ctx->use_tc && ctx->md.ablation != TLF_ABLATION_DENSE_CACHE) {  // batched, chunked prefill (tcgen05)
    const int rc = prefill_batched(ctx, n_seqs, slot_of.data(), offsets, tokens, forced, last_logits, logits_dev,
                                   loops, st);
    return rc ? rollback(rc) : TLF_OK;
  }
  // float32 models and the dense-cache ablation: the prompt runs position by position through the
  // decode kernels
  const int maxB = ctx->cfg.max_batch;
  std::vector<PageUpdate> upd;
  for (int g0 = 0; g0 < n_seqs; g0 += maxB) {
    const int g1 = std::min(n_seqs, g0 + maxB);
    int maxlen = 0;
    for (int s = g0; s < g1; ++s) maxlen = std::max(maxlen, offsets[s + 1] - offsets[s]);
    std::vector<int> rows, slots, toks, frc;
    for (int t = 0; t < maxlen; ++t) {
      rows.clear(); slots.clear(); toks.clear(); frc.clear();
      bool need = false;
      for (int s = g0; s < g1; ++s) {
        const int len = offsets[s + 1] - offsets[s];
        if (t < len) {
          rows.push_back(s);
          slots.push_back(slot_of[s]);
          toks.push_back(tokens[offsets[s] + t]);
          frc.push_back(forced ? forced[offsets[s] + t] : -1);
          if (t == len - 1 && last_logits) need = true;
        }
      }
      const int B = (int)rows.size();
      int rc = reserve_step(ctx, B, slots.data(), &upd);
      if (rc) return rollback(rc);
      rc = run_step(ctx, B, slots.data(), toks.data(), frc.data(), upd, need, st);
      if (rc) return rollback(rc);
      advance_lengths(ctx, B, slots.data());
      for (int b = 0; b < B; ++b) {
        const int s = rows[b];
        if (loops) loops[offsets[s] + t] = ctx->h_m[b];
        if (need && t == offsets[s + 1] - offsets[s] - 1) {
          const size_t bytes = (size_t)ctx->md.V * 4;
          cudaError_t e = cudaMemcpyAsync(last_logits + (size_t)s * ctx->md.V, ctx->d_logits + (size_t)b * ctx->md.V,
                                          bytes, logits_dev ? cudaMemcpyDeviceToDevice : cudaMemcpyDeviceToHost, st);
          if (e != cudaSuccess) return rollback(fail(ctx, TLF_ERR_CUDA, "logits copy: %s", cudaGetErrorString(e)));
        }
      }
      if (need) CK(ctx, cudaStreamSynchronize(st));
    }
  }
  return TLF_OK;
}

extern "C" int tlf_load_cache(tlf_ctx* ctx, uint64_t seq_id, const int32_t* lens, const int32_t* positions,
                              const void* k, const void* v) {
  if (!ctx) return TLF_ERR_INVALID_ARG;
  if (!lens || !positions || (!k) != (!v)) return fail(ctx, TLF_ERR_INVALID_ARG, "NULL argument");
  const bool fill = (k == nullptr);  // entries filled on the device with a counter-based pattern
  const int M = ctx->md.M, ps = ctx->md.page_size;
  if (ctx->seq_slot.count(seq_id)) return fail(ctx, TLF_ERR_DUPLICATE_SEQ, "sequence %llu is live", (unsigned long long)seq_id);
  if (ctx->free_slots.empty()) return fail(ctx, TLF_ERR_CAPACITY, "no free sequence slot");
  if (lens[0] < 1 || lens[0] >= ctx->cfg.max_seq_len)
    return fail(ctx, TLF_ERR_SEQ_TOO_LONG, "loop-1 length must be in 1..max_seq_len-1");
  size_t need = 0, off = 0;
  std::vector<size_t> offs(M);
  for (int r = 0; r < M; ++r) {
    if (lens[r] < 0 || (r > 0 && lens[r] > lens[r - 1])) return fail(ctx, TLF_ERR_INVALID_ARG, "loop lengths must not grow with depth");
    offs[r] = off;
    const int32_t* p = positions + off;
    for (int i = 0; i < lens[r]; ++i) {
      if (r == 0 && p[i] != i) return fail(ctx, TLF_ERR_INVALID_ARG, "loop-1 positions must be 0..L-1");
      if (i > 0 && p[i] <= p[i - 1]) return fail(ctx, TLF_ERR_INVALID_ARG, "positions must increase");
    }
    if (r > 0) {  // subset of the previous loop's positions
      const int32_t* q = positions + offs[r - 1];
      int a = 0;
      for (int i = 0; i < lens[r]; ++i) {
        while (a < lens[r - 1] && q[a] < p[i]) ++a;
        if (a >= lens[r - 1] || q[a] != p[i]) return fail(ctx, TLF_ERR_INVALID_ARG, "loop caches must nest");
      }
    }
    need += (lens[r] + ps - 1) / ps;
    off += lens[r];
  }
  // without recursion-wise caches (dense-cache ablation) every loop cache holds a slot per position:
  // slot t of loop r holds position t if the token ran loop r, else a masked slot (position -1)
  std::vector<int32_t> dlens, dpos;
  std::vector<uint8_t> hk, hv;
  if (ctx->md.ablation == TLF_ABLATION_DENSE_CACHE) {
    const int L0 = lens[0];
    const size_t ebytes = (size_t)ctx->md.J * ctx->md.Hkv * ctx->md.hd * ctx->eb;
    dlens.assign(M, L0);
    dpos.assign((size_t)M * L0, -1);
    if (!fill) {
      hk.assign((size_t)M * L0 * ebytes, 0);
      hv.assign((size_t)M * L0 * ebytes, 0);
    }
    for (int r = 0; r < M; ++r)
      for (int i = 0; i < lens[r]; ++i) {
        const int t = positions[offs[r] + i];
        dpos[(size_t)r * L0 + t] = t;
        if (!fill) {
          memcpy(&hk[((size_t)r * L0 + t) * ebytes], (const uint8_t*)k + (offs[r] + i) * ebytes, ebytes);
          memcpy(&hv[((size_t)r * L0 + t) * ebytes], (const uint8_t*)v + (offs[r] + i) * ebytes, ebytes);
        }
      }
    for (int r = 0; r < M; ++r) offs[r] = (size_t)r * L0;
    lens = dlens.data();
    positions = dpos.data();
    if (!fill) {
      k = hk.data();
      v = hv.data();
    }
    need = (size_t)M * ((L0 + ps - 1) / ps);
  }
  if (need > ctx->free_pages.size()) return fail(ctx, TLF_ERR_OUT_OF_PAGES, "snapshot needs %zu pages", need);
  const int slot = new_slot(ctx, seq_id, 0);
  for (int r = 0; r < M; ++r) {
    for (int p = 0; p < (lens[r] + ps - 1) / ps; ++p) {
      pt_at(ctx, slot, r, p) = ctx->free_pages.back();
      ctx->free_pages.pop_back();
    }
    ctx->h_len[(size_t)slot * M + r] = lens[r];
  }
  if (ctx->host_only) return TLF_OK;  // bookkeeping only: a host-only context holds no cache data
  const size_t rowsz = (size_t)M * ctx->md.max_pages;
  auto undo = [&](int rc) {
    free_slot(ctx, slot);
    ctx->seq_slot.erase(seq_id);
    return rc;
  };
  cudaError_t e = cudaMemcpy(ctx->d_page_table + (size_t)slot * rowsz, &ctx->h_page_table[(size_t)slot * rowsz],
                             rowsz * 4, cudaMemcpyHostToDevice);
  if (e == cudaSuccess)
    e = cudaMemcpy(ctx->d_len + (size_t)slot * M, &ctx->h_len[(size_t)slot * M], M * 4, cudaMemcpyHostToDevice);
  const size_t per = (size_t)ctx->md.J * ctx->md.Hkv * ctx->md.hd;
  void *dk = nullptr, *dv = nullptr;
  int* dp = nullptr;
  if (e == cudaSuccess && lens[0] > 0) {
    if (!fill) {
      e = cudaMalloc(&dk, (size_t)lens[0] * per * ctx->eb);
      if (e == cudaSuccess) e = cudaMalloc(&dv, (size_t)lens[0] * per * ctx->eb);
    }
    if (e == cudaSuccess) e = cudaMalloc(&dp, (size_t)lens[0] * 4);
  }
  for (int r = 0; r < M && e == cudaSuccess; ++r) {
    if (lens[r] == 0) continue;
    if (!fill) {
      e = cudaMemcpy(dk, (const uint8_t*)k + offs[r] * per * ctx->eb, (size_t)lens[r] * per * ctx->eb,
                     cudaMemcpyHostToDevice);
      if (e == cudaSuccess)
        e = cudaMemcpy(dv, (const uint8_t*)v + offs[r] * per * ctx->eb, (size_t)lens[r] * per * ctx->eb,
                       cudaMemcpyHostToDevice);
    }
    if (e == cudaSuccess) e = cudaMemcpy(dp, positions + offs[r], (size_t)lens[r] * 4, cudaMemcpyHostToDevice);
    if (e == cudaSuccess) {
      if (fill)
        launch_fill_cache(ctx->md, slot, r, lens[r], dp, ctx->d_page_table, ctx->d_pool, ctx->d_pos_table, 0);
      else
        launch_scatter_cache(ctx->md, slot, r, lens[r], dk, dv, dp, ctx->d_page_table, ctx->d_pool,
                             ctx->d_pos_table, 0);
      e = cudaDeviceSynchronize();
    }
  }
  if (dk) cudaFree(dk);
  if (dv) cudaFree(dv);
  if (dp) cudaFree(dp);
  if (e != cudaSuccess) return undo(fail(ctx, TLF_ERR_CUDA, "load_cache: %s", cudaGetErrorString(e)));
  return TLF_OK;
}

// ----------------------------------------------------------------------------
// inspection
// ----------------------------------------------------------------------------
extern "C" int tlf_stats(const tlf_ctx* ctx, int32_t* live_seqs, int64_t* free_pages, int64_t* total_pages) {
  if (!ctx) return TLF_ERR_INVALID_ARG;
  if (live_seqs) *live_seqs = (int32_t)ctx->seq_slot.size();
  if (free_pages) *free_pages = (int64_t)ctx->free_pages.size();
  if (total_pages) *total_pages = ctx->n_pages;
  return TLF_OK;
}

extern "C" int tlf_cache_len(const tlf_ctx* ctx, uint64_t seq_id, int32_t loop, int32_t* len) {
  if (!ctx || !len) return TLF_ERR_INVALID_ARG;
  auto it = ctx->seq_slot.find(seq_id);
  if (it == ctx->seq_slot.end()) return TLF_ERR_UNKNOWN_SEQ;
  if (loop < 1 || loop > ctx->md.M) return TLF_ERR_INVALID_ARG;
  *len = ctx->h_len[(size_t)it->second * ctx->md.M + loop - 1];
  return TLF_OK;
}

static float widen(const uint8_t* p, size_t i, size_t eb) {
  if (eb == 4) {
    float f;
    memcpy(&f, p + 4 * i, 4);
    return f;
  }
  uint16_t h;
  memcpy(&h, p + 2 * i, 2);
  uint32_t u = (uint32_t)h << 16;
  float f;
  memcpy(&f, &u, 4);
  return f;
}

extern "C" int tlf_read_cache(tlf_ctx* ctx, uint64_t seq_id, int32_t loop, int32_t layer, int32_t* positions, float* k,
                              float* v) {
  if (!ctx) return TLF_ERR_INVALID_ARG;
  if (ctx->host_only) return fail(ctx, TLF_ERR_NO_DEVICE, "host-only context");
  auto it = ctx->seq_slot.find(seq_id);
  if (it == ctx->seq_slot.end()) return fail(ctx, TLF_ERR_UNKNOWN_SEQ, "sequence not live");
  const ModelDims& md = ctx->md;
  if (loop < 1 || loop > md.M || layer < 0 || layer >= md.J) return fail(ctx, TLF_ERR_INVALID_ARG, "loop/layer out of range");
  const int slot = it->second, r = loop - 1, ps = md.page_size;
  const int L = ctx->h_len[(size_t)slot * md.M + r];
  const size_t seg = (size_t)md.Hkv * ps * md.hd;  // elements of K (or V) of one layer in a page
  std::vector<uint8_t> kb(seg * ctx->eb), vb(seg * ctx->eb);
  std::vector<int> pb(ps);
  for (int p = 0; p * ps < L; ++p) {
    const int page = pt_at(ctx, slot, r, p);
    const uint8_t* base = (const uint8_t*)ctx->d_pool + (size_t)page * md.page_elems * ctx->eb;
    CK(ctx, cudaMemcpy(kb.data(), base + (size_t)(layer * 2 + 0) * seg * ctx->eb, seg * ctx->eb, cudaMemcpyDeviceToHost));
    CK(ctx, cudaMemcpy(vb.data(), base + (size_t)(layer * 2 + 1) * seg * ctx->eb, seg * ctx->eb, cudaMemcpyDeviceToHost));
    CK(ctx, cudaMemcpy(pb.data(), ctx->d_pos_table + (size_t)page * ps, ps * 4, cudaMemcpyDeviceToHost));
    for (int o = 0; o < ps && p * ps + o < L; ++o) {
      const int e = p * ps + o;
      if (positions) positions[e] = pb[o];
      for (int h = 0; h < md.Hkv; ++h)
        for (int i = 0; i < md.hd; ++i) {
          const size_t src = ((size_t)h * ps + o) * md.hd + i;
          const size_t dst = ((size_t)e * md.Hkv + h) * md.hd + i;
          if (k) k[dst] = widen(kb.data(), src, ctx->eb);
          if (v) v[dst] = widen(vb.data(), src, ctx->eb);
        }
    }
  }
  return TLF_OK;
}

extern "C" int tlf_last_active_sets(tlf_ctx* ctx, int32_t* counts, int32_t* idx) {
  if (!ctx || !counts || !idx) return TLF_ERR_INVALID_ARG;
  if (ctx->host_only) return fail(ctx, TLF_ERR_NO_DEVICE, "host-only context");
  const int M = ctx->md.M, maxB = ctx->md.max_batch, B = ctx->last_batch;
  std::vector<int> n(M), id((size_t)M * maxB);
  CK(ctx, cudaMemcpy(n.data(), ctx->d_n, M * 4, cudaMemcpyDeviceToHost));
  CK(ctx, cudaMemcpy(id.data(), ctx->d_idx, id.size() * 4, cudaMemcpyDeviceToHost));
  for (int r = 0; r < M; ++r) {
    counts[r] = n[r];
    for (int i = 0; i < B; ++i) idx[(size_t)r * B + i] = i < n[r] ? id[(size_t)r * maxB + i] : -1;
  }
  return TLF_OK;
}

extern "C" int tlf_set_profiling(tlf_ctx* ctx, int32_t on) {
  if (!ctx) return TLF_ERR_INVALID_ARG;
  ctx->profiling = on != 0;
  return TLF_OK;
}

extern "C" int tlf_last_step_profile(const tlf_ctx* ctx, float* attn_ms, double* attn_kv_bytes, int32_t* kernel_launches) {
  if (!ctx) return TLF_ERR_INVALID_ARG;
  if (attn_ms) *attn_ms = ctx->last_attn_ms;
  if (attn_kv_bytes) *attn_kv_bytes = ctx->last_attn_bytes;
  if (kernel_launches) *kernel_launches = ctx->last_launches;
  return TLF_OK;
}

extern "C" int tlf_last_step_kernel_times(const tlf_ctx* ctx, float* ms, int32_t n) {
  if (!ctx || !ms || n < 0) return TLF_ERR_INVALID_ARG;
  for (int i = 0; i < n && i < 13; ++i) ms[i] = ctx->class_ms[i];
  return TLF_OK;
}
