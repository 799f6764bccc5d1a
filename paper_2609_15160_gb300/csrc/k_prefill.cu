// Batched prefill of a chunk of prompt tokens (T-LoopFormer Sec. 3.3 and App. B).
//
// A chunk holds up to C prompt tokens of one or more sequences, ordered by
// sequence and position. All its tokens are routed at once; loop r gathers the
// chunk tokens with m >= r (Eq. 6), runs the shared block on them, and writes
// their k, v into the loop-r caches of their sequences at the slots after the
// entries of earlier chunks, in position order (the original positions rho^(r)
// of App. B). Attention at loop r is causal over the loop-r cache of each
// sequence: the token with cache slot s sees slots 0..s, i.e. exactly the
// tokens before it (this or earlier chunks) that also ran loop r (Eq. 10 with
// the block-causal mask among gathered tokens).
//
// k_pf_plan       per loop r: compact rows A_r, each row's sequence slot, cache
//                 slot and position, per-sequence counts, first rows and query
//                 blocks of the attention.
// k_pf_attn       causal attention of one block of QB queries of one sequence
//                 against that sequence's loop-r cache, for the G query heads of
//                 one kv head; K is staged transposed in shared memory so each
//                 lane scores whole keys, online softmax in float32 (base 2).
// k_pf_len        cache lengths += tokens of the chunk that ran each loop.
#include "tlf_internal.cuh"

namespace tlf {

constexpr int PF_QB = 32;       // queries per attention block
constexpr int PF_WARPS = 8;     // 4 queries per warp

// Exclusive scan over a block of up to 1024 threads (one value per thread).
__device__ int pf_block_scan(int v, int* total, int* warp_tot) {
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
    if (lane < nw) warp_tot[lane] = t;
    if (lane == 31) warp_tot[32] = t;
  }
  __syncthreads();
  const int excl = x - v + (warp > 0 ? warp_tot[warp - 1] : 0);
  *total = warp_tot[32];
  __syncthreads();
  return excl;
}

__global__ void __launch_bounds__(1024) k_pf_plan(ModelDims md, PrefillDev p) {
  __shared__ int warp_tot[33];
  __shared__ int cnt_s[1024];
  __shared__ int first_s[1024];
  __shared__ int s0_s[1024];
  pdl_wait();
  pdl_trigger();
  const int tid = threadIdx.x, T = p.T, S = p.S, C = p.C, M = md.M;
  for (int r = 0; r < M; ++r) {
    if (tid < S) cnt_s[tid] = 0;
    __syncthreads();
    for (int t = tid; t < T; t += blockDim.x)
      if (p.m[t] > r) atomicAdd(&cnt_s[p.seqidx[t]], 1);
    __syncthreads();
    const int v = tid < S ? cnt_s[tid] : 0;
    int n_r;
    const int first = pf_block_scan(v, &n_r, warp_tot);
    const int qb = (v + PF_QB - 1) / PF_QB;
    int tiles;
    const int tb = pf_block_scan(qb, &tiles, warp_tot);
    if (tid < S) {
      first_s[tid] = first;
      s0_s[tid] = p.len[p.seq_slot[tid] * M + r];
      p.first[r * p.Smax + tid] = first;
      p.cnt[r * p.Smax + tid] = v;
      p.s0[r * p.Smax + tid] = s0_s[tid];
      p.tile_base[r * (p.Smax + 1) + tid] = tb;
    }
    if (tid == 0) {
      p.n[r] = n_r;
      p.tile_base[r * (p.Smax + 1) + S] = tiles;
    }
    __syncthreads();
    int running = 0;
    for (int base = 0; base < T; base += blockDim.x) {
      const int t = base + tid;
      const bool act = t < T && p.m[t] > r;
      int btot;
      const int k = running + pf_block_scan(act ? 1 : 0, &btot, warp_tot);
      if (act) {
        const int sq = p.seqidx[t];
        p.idx[r * C + k] = t;
        p.row_slot[r * C + k] = p.seq_slot[sq];
        p.row_cslot[r * C + k] = s0_s[sq] + (k - first_s[sq]);
        p.row_pos[r * C + k] = p.pos[t];
      }
      running += btot;
    }
    __syncthreads();
  }
}

template <typename T, int HD, int G>
__global__ void __launch_bounds__(32 * PF_WARPS) k_pf_attn(ModelDims md, PrefillDev p, StepDev s, int r, int j,
                                                           const float* __restrict__ Q, T* __restrict__ O) {
  constexpr int QH = (PF_QB / PF_WARPS) * G;  // query-heads per warp
  constexpr int DPL = HD / 32;                 // output dims per lane
  extern __shared__ float sm[];
  float* Qs = sm;                              // [QB][G][HD]
  float* Kt = Qs + PF_QB * G * HD;             // [HD][65]
  float* Vs = Kt + HD * 65;                    // [64][HD]
  float* Ps = Vs + 64 * HD;                    // [warps][QH][64]

  pdl_wait();
  pdl_trigger();
  const int S = p.S;
  const int* tbase = p.tile_base + r * (p.Smax + 1);
  const int tile = blockIdx.x, kvh = blockIdx.y;
  if (tile >= tbase[S]) return;
  int lo = 0, hi = S;  // sequence: largest sq with tbase[sq] <= tile
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (tbase[mid] <= tile) lo = mid; else hi = mid;
  }
  const int sq = lo, qb = tile - tbase[sq];
  const int cnt = p.cnt[r * p.Smax + sq], first = p.first[r * p.Smax + sq], s0 = p.s0[r * p.Smax + sq];
  const int slot = p.seq_slot[sq];
  const int q0 = qb * PF_QB, nq = min(PF_QB, cnt - q0);
  const int last = s0 + q0 + nq - 1;  // cache slot of the block's last query
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const float scale = 1.4426950408889634f * rsqrtf((float)HD);

  for (int e = tid; e < PF_QB * G * HD; e += blockDim.x) {
    const int qi = e / (G * HD), rem = e % (G * HD), g = rem / HD, d = rem % HD;
    Qs[e] = (qi < nq) ? Q[((size_t)(first + q0 + qi) * md.Hq + kvh * G + g) * HD + d] * scale : 0.f;
  }

  float m_run[QH], l_run[QH], acc[QH][DPL];
#pragma unroll
  for (int qh = 0; qh < QH; ++qh) {
    m_run[qh] = -INFINITY;
    l_run[qh] = 0.f;
#pragma unroll
    for (int t = 0; t < DPL; ++t) acc[qh][t] = 0.f;
  }
  const int* ptab = s.page_table + ((size_t)slot * md.M + r) * md.max_pages;
  const int npages = last / 64 + 1;
  for (int pg = 0; pg < npages; ++pg) {
    __syncthreads();  // previous page fully consumed
    const int page = ptab[pg];
    if (page < 0 || page >= md.n_pages) {
      if (tid == 0) atomicOr(s.err, DEVERR_INDEX);
      return;
    }
    const T* kseg = reinterpret_cast<const T*>(s.pool) + (size_t)page * md.page_elems +
                    ((size_t)(j * 2 + 0) * md.Hkv + kvh) * 64 * HD;
    const T* vseg = kseg + (size_t)md.Hkv * 64 * HD;
    const int valid = min(64, last + 1 - pg * 64);
    for (int e = tid; e < 64 * HD; e += blockDim.x) {
      const int key = e / HD, d = e % HD;
      const float kv = key < valid ? to_f32(kseg[e]) : 0.f;
      const float vv = key < valid ? to_f32(vseg[e]) : 0.f;
      Kt[d * 65 + key] = kv;
      Vs[e] = vv;
    }
    __syncthreads();
    // scores of keys lane and lane + 32 for this warp's query-heads
    float sc[QH][2];
#pragma unroll
    for (int qh = 0; qh < QH; ++qh) sc[qh][0] = sc[qh][1] = 0.f;
    const float* qw = Qs + (warp * (PF_QB / PF_WARPS)) * G * HD;  // QH consecutive [G][HD] rows
    for (int d = 0; d < HD; d += 4) {
      float k0[4], k1[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        k0[u] = Kt[(d + u) * 65 + lane];
        k1[u] = Kt[(d + u) * 65 + lane + 32];
      }
#pragma unroll
      for (int qh = 0; qh < QH; ++qh) {
        const float4 q4 = *reinterpret_cast<const float4*>(qw + qh * HD + d);
        sc[qh][0] = fmaf(q4.x, k0[0], fmaf(q4.y, k0[1], fmaf(q4.z, k0[2], fmaf(q4.w, k0[3], sc[qh][0]))));
        sc[qh][1] = fmaf(q4.x, k1[0], fmaf(q4.y, k1[1], fmaf(q4.z, k1[2], fmaf(q4.w, k1[3], sc[qh][1]))));
      }
    }
    float* pw = Ps + warp * QH * 64;
#pragma unroll
    for (int qh = 0; qh < QH; ++qh) {
      const int qi = warp * (PF_QB / PF_WARPS) + qh / G;
      const int qslot = s0 + q0 + qi;
#pragma unroll
      for (int h2 = 0; h2 < 2; ++h2) {
        const int ks = pg * 64 + lane + 32 * h2;
        if (qi >= nq || ks > qslot) sc[qh][h2] = -INFINITY;  // causal within the cache
      }
      const float pm = warp_max(fmaxf(sc[qh][0], sc[qh][1]));
      if (pm > m_run[qh]) {
        const float cr = exp2f(m_run[qh] - pm);
        l_run[qh] *= cr;
#pragma unroll
        for (int t = 0; t < DPL; ++t) acc[qh][t] *= cr;
        m_run[qh] = pm;
      }
      const float p0 = (sc[qh][0] == -INFINITY) ? 0.f : exp2f(sc[qh][0] - m_run[qh]);
      const float p1 = (sc[qh][1] == -INFINITY) ? 0.f : exp2f(sc[qh][1] - m_run[qh]);
      l_run[qh] += p0 + p1;
      pw[qh * 64 + lane] = p0;
      pw[qh * 64 + lane + 32] = p1;
    }
    __syncwarp();
    for (int key = 0; key < valid; key += 4) {
      float4 pk[QH];
#pragma unroll
      for (int qh = 0; qh < QH; ++qh) pk[qh] = *reinterpret_cast<const float4*>(pw + qh * 64 + key);
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        float vv[DPL];
#pragma unroll
        for (int t = 0; t < DPL; ++t) vv[t] = Vs[(key + u) * HD + lane + 32 * t];
#pragma unroll
        for (int qh = 0; qh < QH; ++qh) {
          const float pr = u == 0 ? pk[qh].x : (u == 1 ? pk[qh].y : (u == 2 ? pk[qh].z : pk[qh].w));
#pragma unroll
          for (int t = 0; t < DPL; ++t) acc[qh][t] = fmaf(pr, vv[t], acc[qh][t]);
        }
      }
    }
  }
#pragma unroll
  for (int qh = 0; qh < QH; ++qh) {
    const int qi = warp * (PF_QB / PF_WARPS) + qh / G, g = qh % G;
    const float l = warp_sum(l_run[qh]);
    if (qi < nq) {
      T* orow = O + (size_t)(first + q0 + qi) * md.q_dim + (kvh * G + g) * HD;
#pragma unroll
      for (int t = 0; t < DPL; ++t) orow[lane + 32 * t] = from_f32<T>(acc[qh][t] / l);
    }
  }
}

__global__ void k_pf_len(ModelDims md, PrefillDev p) {
  pdl_wait();
  pdl_trigger();
  for (int e = threadIdx.x; e < p.S * md.M; e += blockDim.x) {
    const int sq = e / md.M, r = e % md.M;
    p.len[p.seq_slot[sq] * md.M + r] += p.cnt[r * p.Smax + sq];
  }
}

template <typename T, int HD, int G>
static void pf_attn_launch(const ModelDims& md, const PrefillDev& p, const StepDev& s, int r, int j, const float* Q,
                           void* O, int tiles_bound, cudaStream_t st) {
  static bool attr = false;
  constexpr int smem = (PF_QB * G * HD + HD * 65 + 64 * HD + PF_WARPS * (PF_QB / PF_WARPS) * G * 64) * 4;
  if (!attr) {
    cudaFuncSetAttribute(k_pf_attn<T, HD, G>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    attr = true;
  }
  launch_k(k_pf_attn<T, HD, G>, dim3(tiles_bound, md.Hkv), 32 * PF_WARPS, smem, st, md, p, s, r, j, Q, (T*)O);
}

void launch_pf_plan(const ModelDims& md, const PrefillDev& p, cudaStream_t st) {
  launch_k(k_pf_plan, 1, 1024, 0, st, md, p);
}

void launch_pf_attn(const ModelDims& md, const PrefillDev& p, const StepDev& s, int r, int j, const float* Q,
                    void* O, int tiles_bound, cudaStream_t st) {
  const int G = md.Hq / md.Hkv;
  if (md.hd == 128 && G == 1) pf_attn_launch<bf16, 128, 1>(md, p, s, r, j, Q, O, tiles_bound, st);
  else if (md.hd == 128 && G == 2) pf_attn_launch<bf16, 128, 2>(md, p, s, r, j, Q, O, tiles_bound, st);
  else if (md.hd == 128 && G == 4) pf_attn_launch<bf16, 128, 4>(md, p, s, r, j, Q, O, tiles_bound, st);
  else if (md.hd == 64 && G == 1) pf_attn_launch<bf16, 64, 1>(md, p, s, r, j, Q, O, tiles_bound, st);
  else if (md.hd == 64 && G == 2) pf_attn_launch<bf16, 64, 2>(md, p, s, r, j, Q, O, tiles_bound, st);
  else if (md.hd == 64 && G == 4) pf_attn_launch<bf16, 64, 4>(md, p, s, r, j, Q, O, tiles_bound, st);
  else if (md.hd == 32 && G == 1) pf_attn_launch<bf16, 32, 1>(md, p, s, r, j, Q, O, tiles_bound, st);
  else pf_attn_launch<bf16, 32, 2>(md, p, s, r, j, Q, O, tiles_bound, st);
}

void launch_pf_len(const ModelDims& md, const PrefillDev& p, cudaStream_t st) {
  launch_k(k_pf_len, 1, 256, 0, st, md, p);
}

}  // namespace tlf
