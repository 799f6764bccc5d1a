// Token-choice router and active-set compaction (T-LoopFormer Sec. 3.2, Eq. 2-6).
//
// k_router: four warps per token, each over a quarter of the row. h^(0) = E[x]
// is written to the float32 residual stream H, RMSNorm (no gain) is applied,
// the M router logits z = W_r x + b_r are reduced across the warps, and the
// loop count m and its decision margin are taken in float32 (ARGMAX or
// SURVIVAL rule, see tlf.h).
// The same kernel applies the page-table updates the host queued for the step.
//
// k_plan: one CTA per loop r. It builds A_r = {b : m_b >= r} in
// increasing b with a warp ballot plus a block prefix scan, the page, slot
// and position of each active token's new loop-r cache entry (read by the
// QKV epilogue that appends k, v), and the work plan of the decode attention
// over the loop-r caches: the pages of every (token, kv head) item, from the
// device-side cache lengths, laid out in one flat order (prefix sums), which
// the attention grid splits evenly.
#include "tlf_internal.cuh"

namespace tlf {

// Loop count from the M router logits z (entries >= M are ignored): the ARGMAX or
// SURVIVAL rule of Eq. 2-5 (see tlf.h), with the decision margin.
__device__ __forceinline__ void router_decide(const ModelDims& md, const float z[16], int& m, float& margin) {
  const int M = md.M;
  m = 1;
  if (md.exit_rule == 0) {
    // ARGMAX: first maximum wins (ties go to the smaller depth); indices stay compile-time
    // constants so z lives in registers
    int top = 0;
    float best = z[0];
#pragma unroll
    for (int l = 1; l < 16; ++l)
      if (l < M && z[l] > best) {
        best = z[l];
        top = l;
      }
    float second = -INFINITY;
#pragma unroll
    for (int l = 0; l < 16; ++l)
      if (l < M && l != top) second = fmaxf(second, z[l]);
    m = top + 1;
    margin = best - second;  // +inf when M == 1
  } else {
    // SURVIVAL (Eq. 2-5): softmax, suffix sums p^(i), m = max{i : p^(i) > threshold}
    float mx = z[0];
#pragma unroll
    for (int l = 1; l < 16; ++l)
      if (l < M) mx = fmaxf(mx, z[l]);
    float ex[16], sum = 0.f;
#pragma unroll
    for (int l = 0; l < 16; ++l) {
      ex[l] = (l < M) ? expf(z[l] - mx) : 0.f;
      sum += ex[l];
    }
    float p[17];
    p[16] = 0.f;
    float acc = 0.f;
#pragma unroll
    for (int l = 15; l >= 0; --l) {
      acc += ex[l] / sum;
      p[l] = acc;
    }
    m = 1;
#pragma unroll
    for (int l = 0; l < 16; ++l)
      if (l < M && p[l] > md.threshold) m = l + 1;
    float pm = 0.f, pnext = 0.f;  // p^(m) and p^(m+1) (0 past M)
#pragma unroll
    for (int l = 0; l < 16; ++l) {
      if (l == m - 1) pm = p[l];
      if (l == m && l < M) pnext = p[l];
    }
    margin = fminf(pm - md.threshold, md.threshold - pnext);
  }
}

// Warps per token of k_router: each reads a quarter of the row, so the dependent chain of
// 16-byte loads per lane is a quarter as long; a CTA of 8 warps serves two tokens.
constexpr int RT_WPT = 4;

template <typename T>
__global__ void __launch_bounds__(256) k_router(ModelDims md, StepDev s, int B, const T* __restrict__ emb,
                                                const T* __restrict__ rw, const float* __restrict__ rb,
                                                const PageUpdate* __restrict__ upd, const int* __restrict__ n_upd_dev) {
  pdl_wait();
  pdl_trigger();
  const int n_upd = *n_upd_dev;
  for (int u = blockIdx.x * blockDim.x + threadIdx.x; u < n_upd; u += gridDim.x * blockDim.x) {
    const PageUpdate p = upd[u];
    s.page_table[p.index] = p.page;
  }
  __shared__ float part_sum[8][17];  // per warp: sum of squares, then the M dot products
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int quarter = warp % RT_WPT;
  const int b = blockIdx.x * (8 / RT_WPT) + warp / RT_WPT;
  const int d = md.d, M = md.M;
  if (b < B) {
    int tok = s.tokens[b];
    if (tok < 0 || tok >= md.V) {
      if (lane == 0 && quarter == 0) atomicOr(s.err, DEVERR_INDEX);
      tok = 0;
    }
    // One pass over 16-byte chunks: each chunk of E[x] is loaded once, written to the residual
    // stream, squared into the norm, and dotted with all M router rows; the RMSNorm scale (a
    // per-row scalar) multiplies the dot products afterwards.
    constexpr int VEC = Vec16<T>::N;
    const T* e = emb + (size_t)tok * d;
    float* h = s.H + (size_t)b * d;
    float ss = 0.f, dot[16];
#pragma unroll
    for (int l = 0; l < 16; ++l) dot[l] = 0.f;
#pragma unroll 2
    for (int c = quarter * 32 + lane; c < d / VEC; c += 32 * RT_WPT) {
      float x[VEC];
      Vec16<T>::load(e + c * VEC, x);
#pragma unroll
      for (int u = 0; u < VEC; u += 4)
        *reinterpret_cast<float4*>(h + c * VEC + u) = make_float4(x[u], x[u + 1], x[u + 2], x[u + 3]);
#pragma unroll
      for (int u = 0; u < VEC; ++u) ss = fmaf(x[u], x[u], ss);
#pragma unroll
      for (int l = 0; l < 16; ++l) {
        if (l < M) {
          float w[VEC];
          Vec16<T>::load(rw + (size_t)l * d + c * VEC, w);
#pragma unroll
          for (int u = 0; u < VEC; ++u) dot[l] = fmaf(x[u], w[u], dot[l]);
        }
      }
    }
    ss = warp_sum(ss);
#pragma unroll
    for (int l = 0; l < 16; ++l)
      if (l < M) dot[l] = warp_sum(dot[l]);
    if (lane == 0) {
      part_sum[warp][0] = ss;
#pragma unroll
      for (int l = 0; l < 16; ++l)
        if (l < M) part_sum[warp][1 + l] = dot[l];
    }
  }
  __syncthreads();
  if (b >= B || quarter != 0) return;
  // the token's first warp adds the quarters (in a fixed order) and takes the decision
  const int w0 = warp;
  float ss = 0.f;
#pragma unroll
  for (int q = 0; q < RT_WPT; ++q) ss += part_sum[w0 + q][0];
  const float inv = rsqrtf(ss / (float)d + md.eps);
  float z[16];
#pragma unroll
  for (int l = 0; l < 16; ++l) {
    float t = 0.f;
    if (l < M) {
#pragma unroll
      for (int q = 0; q < RT_WPT; ++q) t += part_sum[w0 + q][1 + l];
    }
    z[l] = (l < M) ? t * inv + rb[l] : -INFINITY;
  }

  int m;
  float margin;
  router_decide(md, z, m, margin);
  const int f = s.forced[b];
  if (f >= 1) m = min(f, M);
  if (lane == 0) {
    s.m[b] = m;
    s.margin[b] = margin;
  }
}

// The two-layer MLP router of Sec. 3.2: z = W_r GELU(W_1 RMSNorm(h0) + b_1) + b_r (exact GELU).
// One CTA per token: the embedding row goes to the residual stream and, unnormalised, to shared
// memory; a warp per hidden unit reads its W_1 row in 16-byte chunks (the RMSNorm scale, a
// per-token scalar, multiplies the dot product), then a warp per logit reads W_r.
template <typename T>
__global__ void __launch_bounds__(256) k_router_mlp(ModelDims md, StepDev s, int B, const T* __restrict__ emb,
                                                    const T* __restrict__ w1, const float* __restrict__ b1,
                                                    const T* __restrict__ rw, const float* __restrict__ rb,
                                                    const PageUpdate* __restrict__ upd,
                                                    const int* __restrict__ n_upd_dev) {
  pdl_wait();
  pdl_trigger();
  const int n_upd = *n_upd_dev;
  for (int u = blockIdx.x * blockDim.x + threadIdx.x; u < n_upd; u += gridDim.x * blockDim.x) {
    const PageUpdate p = upd[u];
    s.page_table[p.index] = p.page;
  }
  const int b = blockIdx.x;
  if (b >= B) return;
  extern __shared__ float rsm[];
  const int d = md.d, Hr = md.router_hidden, M = md.M;
  float* xs = rsm;           // [d]  h0
  float* hs = rsm + d;       // [Hr] hidden activations
  __shared__ float zs[16], red[8];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int tok = s.tokens[b];
  if (tok < 0 || tok >= md.V) {
    if (threadIdx.x == 0) atomicOr(s.err, DEVERR_INDEX);
    tok = 0;
  }
  constexpr int VEC = Vec16<T>::N;
  const T* e = emb + (size_t)tok * d;
  float* h = s.H + (size_t)b * d;
  float ss = 0.f;
  for (int c = threadIdx.x; c < d / VEC; c += blockDim.x) {
    float x[VEC];
    Vec16<T>::load(e + c * VEC, x);
#pragma unroll
    for (int u = 0; u < VEC; ++u) {
      xs[c * VEC + u] = x[u];
      h[c * VEC + u] = x[u];
      ss = fmaf(x[u], x[u], ss);
    }
  }
  ss = warp_sum(ss);
  if (lane == 0) red[warp] = ss;
  __syncthreads();
  float tot = 0.f;
#pragma unroll
  for (int w = 0; w < 8; ++w) tot += red[w];
  const float inv = rsqrtf(tot / (float)d + md.eps);
  for (int u = warp; u < Hr; u += 8) {
    const T* wr = w1 + (size_t)u * d;
    float acc = 0.f;
    for (int c = lane; c < d / VEC; c += 32) {
      float wv[VEC];
      Vec16<T>::load(wr + c * VEC, wv);
#pragma unroll
      for (int q = 0; q < VEC; ++q) acc = fmaf(wv[q], xs[c * VEC + q], acc);
    }
    acc = warp_sum(acc) * inv + b1[u];
    if (lane == 0) hs[u] = 0.5f * acc * (1.f + erff(acc * 0.70710678118654752f));
  }
  __syncthreads();
  for (int l = warp; l < M; l += 8) {
    const T* wr = rw + (size_t)l * Hr;
    float acc = 0.f;
    for (int c = lane; c < Hr / VEC; c += 32) {
      float wv[VEC];
      Vec16<T>::load(wr + c * VEC, wv);
#pragma unroll
      for (int q = 0; q < VEC; ++q) acc = fmaf(wv[q], hs[c * VEC + q], acc);
    }
    acc = warp_sum(acc);
    if (lane == 0) zs[l] = acc + rb[l];
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float z[16];
#pragma unroll
    for (int l = 0; l < 16; ++l) z[l] = (l < M) ? zs[l] : -INFINITY;
    int m;
    float margin;
    router_decide(md, z, m, margin);
    const int f = s.forced[b];
    if (f >= 1) m = min(f, M);
    s.m[b] = m;
    s.margin[b] = margin;
  }
}

// Exclusive scan of one int per thread over the block (blockDim.x <= 1024).
__device__ int block_exclusive_scan(int v, int* total) {
  __shared__ int warp_tot[32];
  __shared__ int tot;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_tot[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int t = (lane < nw) ? warp_tot[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, t, o);
      if (lane >= o) t += y;
    }
    if (lane < nw) warp_tot[lane] = t;  // inclusive
    if (lane == 31) tot = t;
  }
  __syncthreads();
  const int excl = x - v + (warp > 0 ? warp_tot[warp - 1] : 0);
  *total = tot;
  __syncthreads();
  return excl;
}

// One CTA per loop r (the loops' lists and plans are independent), one thread per batch row.
__global__ void __launch_bounds__(256) k_plan(ModelDims md, StepDev s, int B) {
  pdl_wait();
  pdl_trigger();
  const int b = threadIdx.x;
  const int lane = b & 31;
  const int mb = (b < B) ? s.m[b] : 0;
  const int slot = (b < B) ? s.slots[b] : 0;
  const int maxB = md.max_batch, M = md.M, ps = md.page_size;
  // attention merge tickets start at zero every step
  if (blockIdx.x == 0)
    for (int i = b; i < maxB * md.Hkv; i += blockDim.x) s.cnt[i] = 0;
  // without the gather (an ablation), every row of the step is listed at every loop that runs
  const bool all_rows = md.ablation == TLF_ABLATION_NO_GATHER;
  const bool dense = md.ablation == TLF_ABLATION_DENSE_CACHE;
  {
    const int r = blockIdx.x;
    const bool active = mb > r;
    // compaction: ballot gives each active lane its rank in the warp, the block scan the warp offsets
    const unsigned ball = __ballot_sync(0xffffffffu, active);
    const int rank = __popc(ball & ((1u << lane) - 1u));
    int n_r;
    const int warp_off = block_exclusive_scan((lane == 0) ? __popc(ball) : 0, &n_r);
    const int n_list = all_rows ? (n_r > 0 ? B : 0) : n_r;
    const bool listed = all_rows ? (b < B && n_r > 0) : active;
    const int k = all_rows ? b : __shfl_sync(0xffffffffu, warp_off, 0) + rank;
    if (listed) {
      s.idx[r * maxB + k] = b;
      if (s.act) s.act[r * maxB + k] = active ? 1 : 0;
    }
    if (s.col && b < B) s.col[r * maxB + b] = listed ? k : -1;
    // attention plan over the loop-r caches: an active token attends to its cache including its own
    // new entry; a masked row (no gather) to the entries already there. Every (token, kv head) item
    // spans ceil(keys / page) pages; items are laid out token-major in one flat page order
    const int L = listed ? s.len[slot * M + r] + (active ? 1 : 0) : 0;
    const int np = (L + ps - 1) / ps;
    int pages;
    const int base = block_exclusive_scan(np * md.Hkv, &pages);
    if (listed) {
      s.item_base[r * (maxB + 1) + k] = base;
      s.nch[r * maxB + k] = L;
    }
    if (listed && s.rowinfo) {  // NULL for callers that only attend (no append this step)
      int page = -1, e = 0, pos = 0;
      if (active) {
        // where the token's k, v go (Eq. 11): slot L - 1 of the loop-r cache, at its original
        // position (its loop-1 length, since every token runs loop 1); the position table of the
        // page is filled here once for all layers
        e = L - 1;
        pos = s.len[slot * M];
        page = s.page_table[((size_t)slot * M + r) * md.max_pages + e / ps];
        if (page < 0 || page >= md.n_pages || pos >= md.max_pos) {
          atomicOr(s.err, DEVERR_INDEX);
          page = -1;
          pos = 0;
        } else {
          s.pos_table[(size_t)page * ps + e % ps] = pos;
        }
      }
      s.rowinfo[r * maxB + k] = make_int4(page, e % ps, pos, b);
    }
    if (dense && b < B && !active && s.rowinfo) {
      // no recursion-wise cache (an ablation): the exited token still takes its slot in the loop-r
      // cache, masked with position -1, so every loop's cache keeps one slot per position
      const int e = s.len[slot * M + r];
      const int page = s.page_table[((size_t)slot * M + r) * md.max_pages + e / ps];
      if (page < 0 || page >= md.n_pages) atomicOr(s.err, DEVERR_INDEX);
      else s.pos_table[(size_t)page * ps + e % ps] = -1;
    }
    if (b == 0) {
      s.n[r] = n_list;
      s.item_base[r * (maxB + 1) + n_list] = pages;
      s.chunk[r] = ps;
    }
  }
}

void launch_router(const ModelDims& md, const StepDev& s, int B, const void* emb, const void* router_w,
                   const float* router_b, const PageUpdate* upd, const int* n_upd, cudaStream_t st,
                   const void* router_w1, const float* router_b1) {
  if (md.router_hidden > 0) {
    const size_t smem = (size_t)(md.d + md.router_hidden) * 4;
    // (a failure shows at launch)
    (void)ensure_kernel_attrs(md.dtype == 1 ? (const void*)k_router_mlp<bf16> : (const void*)k_router_mlp<float>,
                              65536);
    if (md.dtype == 1)
      launch_k(k_router_mlp<bf16>, B, 256, smem, st, md, s, B, (const bf16*)emb, (const bf16*)router_w1, router_b1,
               (const bf16*)router_w, router_b, upd, n_upd);
    else
      launch_k(k_router_mlp<float>, B, 256, smem, st, md, s, B, (const float*)emb, (const float*)router_w1,
               router_b1, (const float*)router_w, router_b, upd, n_upd);
    return;
  }
  const int grid = (B + 8 / RT_WPT - 1) / (8 / RT_WPT);
  if (md.dtype == 1)
    launch_k(k_router<bf16>, grid, 256, 0, st, md, s, B, (const bf16*)emb, (const bf16*)router_w, router_b, upd,
             n_upd);
  else
    launch_k(k_router<float>, grid, 256, 0, st, md, s, B, (const float*)emb, (const float*)router_w, router_b, upd,
             n_upd);
}

void launch_plan(const ModelDims& md, const StepDev& s, int B, cudaStream_t st) {
  launch_k(k_plan, md.M, 256, 0, st, md, s, B);
}

}  // namespace tlf
