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
    const int qb = (v + p.qblock - 1) / p.qblock;
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

// ----------------------------------------------------------------------------
// Tensor-core causal attention of a chunk (bf16 models, head_dim 64 or 128)
// ----------------------------------------------------------------------------
// One CTA of 256 threads per (sequence, block of QT = 128/G queries, kv head): the 128 MMA rows
// are the G query heads of QT queries (row = query * G + head). For every page of 64 cache slots:
//   S = Q K^T   tcgen05.mma M=128, N=64, K=hd into TMEM; q enters as two bf16 terms (q = hi + lo),
//               so the scores keep q's float32 precision;
//   softmax     two threads share a row (warps w and w+4 reach the same TMEM lanes), each owning
//               32 of its 64 columns: they read S (tcgen05.ld), mask causally by cache slot (only
//               pages on the query's diagonal need the per-key test), exchange the row maximum
//               through shared memory and keep an online softmax in float32 (base 2); P goes to
//               shared memory in bf16;
//   O += P V    tcgen05.mma M=128, N=hd, K=64 accumulating in TMEM.
// The loop is software-pipelined: S has two TMEM buffers and the K / V^T operand tiles two
// shared-memory buffers, so the S product of page p+1 runs on the tensor cores while the threads
// do the softmax of page p, and the re-layout of page p+1 overlaps the P V product of page p.
// The running maximum is refreshed lazily: O (TMEM load, scale, store) and the row sum are
// rescaled only when a row's maximum grows by more than 8 (a factor of 256), so exponentials stay
// below 256 and rescaling is rare. The K and V segments of each page arrive by 1-D bulk copies in
// a two-deep staging ring; threads rewrite them into the swizzled K-major operand tiles (V
// transposed so that keys run along K), with zeros past the last valid slot.
constexpr int PFT_THREADS = 256;

template <int HD>
struct PfTcShape {
  static constexpr int A_BYTES = 128 * HD * 2;   // one of the hi / lo Q tiles [128][HD]
  static constexpr int BK_BYTES = 64 * HD * 2;   // K tile [64 keys][HD]
  static constexpr int BV_BYTES = HD * 64 * 2;   // V^T tile [HD][64 keys]
  static constexpr int P_BYTES = 128 * 64 * 2;   // P tile [128][64 keys]
  static constexpr int SEG = 64 * HD * 2;        // raw K (or V) segment of a page
  static constexpr int RAW_BYTES = 2 * SEG;
  static constexpr int OFF_AHI = 0;
  static constexpr int OFF_ALO = OFF_AHI + A_BYTES;
  static constexpr int OFF_BK = OFF_ALO + A_BYTES;   // two K tiles
  static constexpr int OFF_BV = OFF_BK + 2 * BK_BYTES;  // two V^T tiles
  static constexpr int OFF_P = OFF_BV + 2 * BV_BYTES;
  static constexpr int OFF_RAW = OFF_P + P_BYTES;
  static constexpr int OFF_BAR = OFF_RAW + 2 * RAW_BYTES;
  static constexpr int OFF_XCH = OFF_BAR + 64;         // [2][128] floats: row maxima, then row sums
  static constexpr int BYTES = OFF_XCH + 1024 + 1024;  // exchange, alignment slack
  static constexpr uint32_t TMEM_COLS = 256;          // S buffers in columns 0..127, O in 128..128+HD
  static constexpr int ACOL = 128 * 128;              // bytes of one 128-byte atom column of a Q tile
  static constexpr int BCOL = 64 * 128;               // ... of a K tile
};

// 2^x with the hardware approximation (relative error ~2^-22; the probabilities are then rounded
// to bf16)
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
  return (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(a)) |
         ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(b)) << 16);
}

template <int HD, int G>
__global__ void __launch_bounds__(PFT_THREADS) k_pf_attn_tc(ModelDims md, PrefillDev p, StepDev s, int r, int j,
                                                             const float* __restrict__ Q, bf16* __restrict__ O) {
  using Sh = PfTcShape<HD>;
  constexpr int QT = 128 / G;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  // staging 0, staging 1, S buffer 0 done, S buffer 1 done, P V done
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + Sh::OFF_BAR);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 5);

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
  const int q0 = qb * QT, nq = min(QT, cnt - q0);
  const int last = s0 + q0 + nq - 1;  // cache slot of the block's last query
  const int npages = last / 64 + 1;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int quad = warp & 3, half = warp >> 2;  // TMEM lane quadrant and column half of this warp
  const int row = quad * 32 + lane;             // the MMA row (query * G + head) this thread serves
  float* xch = reinterpret_cast<float*>(sm + Sh::OFF_XCH);
  const int* ptab = s.page_table + ((size_t)slot * md.M + r) * md.max_pages;
  const uint32_t stg0 = smem_u32(&bars[0]), stg1 = smem_u32(&bars[1]);
  const uint32_t bar_s0 = smem_u32(&bars[2]), bar_s1 = smem_u32(&bars[3]), bar_o = smem_u32(&bars[4]);

  if (tid == 0) {
    for (int i = 0; i < 5; ++i) mbar_init(smem_u32(&bars[i]), 1);
    fence_barrier_init();
  }
  if (warp == 0) {
    tmem_alloc(smem_u32(tmem_slot), Sh::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t t_row = tmem + ((uint32_t)(quad * 32) << 16);  // this warp's 32 TMEM lanes
  constexpr uint32_t OCOL = 128;                                 // first TMEM column of O

  auto stage_page = [&](int pg) {  // thread 0: K and V segments of page pg into staging buffer pg & 1
    const uint32_t bar = (pg & 1) ? stg1 : stg0;
    const int page = ptab[pg];
    if (page < 0 || page >= md.n_pages) {
      atomicOr(s.err, DEVERR_INDEX);
      mbar_arrive(bar);  // complete the phase without data
      return;
    }
    const bf16* kseg = reinterpret_cast<const bf16*>(s.pool) + (size_t)page * md.page_elems +
                       ((size_t)(j * 2 + 0) * md.Hkv + kvh) * 64 * HD;
    const bf16* vseg = kseg + (size_t)md.Hkv * 64 * HD;
    uint8_t* dst = sm + Sh::OFF_RAW + (pg & 1) * Sh::RAW_BYTES;
    mbar_arrive_expect_tx(bar, Sh::RAW_BYTES);
    bulk_g2s(smem_u32(dst), kseg, Sh::SEG, bar);
    bulk_g2s(smem_u32(dst + Sh::SEG), vseg, Sh::SEG, bar);
  };
  // K tile of page pg (from its staging buffer) into K buffer pg & 1; rows = keys
  auto relayout_k = [&](int pg) {
    mbar_wait((pg & 1) ? stg1 : stg0, (pg >> 1) & 1, s.err);
    const uint8_t* raw = sm + Sh::OFF_RAW + (pg & 1) * Sh::RAW_BYTES;
    uint8_t* bk = sm + Sh::OFF_BK + (pg & 1) * Sh::BK_BYTES;
    const int valid = min(64, last + 1 - pg * 64);
    for (int e = tid; e < 64 * (HD / 8); e += PFT_THREADS) {
      const int key = e / (HD / 8), c = e % (HD / 8);
      const uint4 v = key < valid ? *reinterpret_cast<const uint4*>(raw + key * HD * 2 + c * 16) : make_uint4(0, 0, 0, 0);
      *reinterpret_cast<uint4*>(bk + (c / 8) * Sh::BCOL + sw128_off(key, c % 8)) = v;
    }
  };
  // V^T tile of page pg into V buffer pg & 1: row = hd index n, chunk c = keys 8c..8c+7
  auto relayout_v = [&](int pg) {
    const uint8_t* raw = sm + Sh::OFF_RAW + (pg & 1) * Sh::RAW_BYTES;
    uint8_t* bv = sm + Sh::OFF_BV + (pg & 1) * Sh::BV_BYTES;
    const int valid = min(64, last + 1 - pg * 64);
    const uint32_t* rv = reinterpret_cast<const uint32_t*>(raw + Sh::SEG);  // [64 keys][HD / 2] pairs
    for (int e = tid; e < (HD / 2) * 8; e += PFT_THREADS) {
      const int n2 = e % (HD / 2), c = e / (HD / 2);  // hd indices 2 n2, 2 n2 + 1; keys 8c..8c+7
      uint32_t x[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) x[u] = 8 * c + u < valid ? rv[(8 * c + u) * (HD / 2) + n2] : 0u;
      uint32_t we[4], wo[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        we[u] = __byte_perm(x[2 * u], x[2 * u + 1], 0x5410);  // low halves: hd index 2 n2
        wo[u] = __byte_perm(x[2 * u], x[2 * u + 1], 0x7632);  // high halves: hd index 2 n2 + 1
      }
      *reinterpret_cast<uint4*>(bv + sw128_off(2 * n2, c)) = make_uint4(we[0], we[1], we[2], we[3]);
      *reinterpret_cast<uint4*>(bv + sw128_off(2 * n2 + 1, c)) = make_uint4(wo[0], wo[1], wo[2], wo[3]);
    }
  };
  constexpr uint32_t IDS = idesc_bf16_f32(128, 64), IDO = idesc_bf16_f32(128, HD);
  auto issue_s = [&](int pg) {  // thread 0: S of page pg into TMEM columns 64 * (pg & 1)
    tc_fence_after();
    const uint32_t bk = smem_u32(sm + Sh::OFF_BK + (pg & 1) * Sh::BK_BYTES);
#pragma unroll
    for (int kc = 0; kc < HD / 64; ++kc)
#pragma unroll
      for (int k = 0; k < 4; ++k) {  // K = 16 per MMA: +32 bytes (encoded +2) inside the atom column
        const uint64_t db = smem_desc_sw128(bk + kc * Sh::BCOL) + 2 * k;
        const uint32_t d = tmem + 64u * (uint32_t)(pg & 1);
        tc_mma_f16(d, smem_desc_sw128(smem_u32(sm + Sh::OFF_AHI + kc * Sh::ACOL)) + 2 * k, db, IDS, (kc | k) ? 1u : 0u);
        tc_mma_f16(d, smem_desc_sw128(smem_u32(sm + Sh::OFF_ALO + kc * Sh::ACOL)) + 2 * k, db, IDS, 1u);
      }
    tc_commit((pg & 1) ? bar_s1 : bar_s0);
  };

  if (tid == 0) {
    stage_page(0);
    if (npages > 1) stage_page(1);
  }

  // Q tile: row = query * G + head, as hi and lo bf16 parts (zeros past the block's queries)
  for (int e = tid; e < 128 * (HD / 8); e += PFT_THREADS) {
    const int qr = e / (HD / 8), c = e % (HD / 8);
    const int qq = qr / G, gg = qr % G;
    float x[8];
    if (qq < nq) {
      const float4* q4 = reinterpret_cast<const float4*>(Q + ((size_t)(first + q0 + qq) * md.Hq + kvh * G + gg) * HD);
      const float4 a = q4[2 * c], b = q4[2 * c + 1];
      x[0] = a.x; x[1] = a.y; x[2] = a.z; x[3] = a.w; x[4] = b.x; x[5] = b.y; x[6] = b.z; x[7] = b.w;
    } else {
#pragma unroll
      for (int u = 0; u < 8; ++u) x[u] = 0.f;
    }
    uint32_t h[4], l[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const float a0 = __bfloat162float(__float2bfloat16_rn(x[2 * u]));
      const float a1 = __bfloat162float(__float2bfloat16_rn(x[2 * u + 1]));
      h[u] = pack_bf16(a0, a1);
      l[u] = pack_bf16(x[2 * u] - a0, x[2 * u + 1] - a1);
    }
    const uint32_t off = (c / 8) * Sh::ACOL + sw128_off(qr, c % 8);
    *reinterpret_cast<uint4*>(sm + Sh::OFF_AHI + off) = make_uint4(h[0], h[1], h[2], h[3]);
    *reinterpret_cast<uint4*>(sm + Sh::OFF_ALO + off) = make_uint4(l[0], l[1], l[2], l[3]);
  }
  const int qi = row / G, g = row % G;
  const bool row_ok = qi < nq;
  // prologue: page 0's operand tiles and its S product
  relayout_k(0);
  relayout_v(0);
  fence_proxy_async_smem();
  __syncthreads();
  if (tid == 0) {
    if (npages > 2) stage_page(2);  // staging buffer 0 has been read
    issue_s(0);
  }
  __syncwarp();

  const int qslot = s0 + q0 + qi;  // cache slot of this row's query
  const float scale = 1.4426950408889634f * rsqrtf((float)HD);
  float m_run = -INFINITY, l_run = 0.f;

  for (int pg = 0; pg < npages; ++pg) {
    const bool more = pg + 1 < npages;
    // operand tiles of page pg+1: its K buffer was last read by S of page pg-1 (complete), its V^T
    // buffer by P V of page pg-1, which also frees P and lets O be rescaled
    if (more) relayout_k(pg + 1);
    if (pg > 0) mbar_wait(bar_o, (pg - 1) & 1, s.err);
    if (more) relayout_v(pg + 1);
    fence_proxy_async_smem();
    __syncthreads();
    if (tid == 0 && more) {
      if (pg + 3 < npages) stage_page(pg + 3);  // staging buffer (pg+1) & 1 has been read
      issue_s(pg + 1);
    }
    __syncwarp();
    mbar_wait((pg & 1) ? bar_s1 : bar_s0, (pg >> 1) & 1, s.err);
    tc_fence_after();

    // this thread's 32 columns of the row
    float sc[32];
    tmem_ld_16(t_row + 64u * (uint32_t)(pg & 1) + 32u * half, sc);
    tmem_ld_16(t_row + 64u * (uint32_t)(pg & 1) + 32u * half + 16u, sc + 16);
    const int valid = min(64, last + 1 - pg * 64);
    const int kb = pg * 64 + 32 * half;  // cache slot of this thread's first column
    float pm = -INFINITY;
    if (row_ok && kb + 31 <= qslot && 32 * half + 31 < valid) {  // every key visible
#pragma unroll
      for (int c = 0; c < 32; ++c) {
        sc[c] *= scale;
        pm = fmaxf(pm, sc[c]);
      }
    } else if (!row_ok || kb > qslot || 32 * half >= valid) {  // none visible
#pragma unroll
      for (int c = 0; c < 32; ++c) sc[c] = -INFINITY;
    } else {  // the diagonal: causal by cache slot
#pragma unroll
      for (int c = 0; c < 32; ++c) {
        const bool use = 32 * half + c < valid && kb + c <= qslot;
        sc[c] = use ? sc[c] * scale : -INFINITY;
        pm = fmaxf(pm, sc[c]);
      }
    }
    xch[half * 128 + row] = pm;
    __syncthreads();
    pm = fmaxf(pm, xch[(half ^ 1) * 128 + row]);
    // lazy maximum: rescale only when it grows by more than 8 (warp-uniform TMEM access); both
    // threads of a row take the same decision, each for its half of O and of the row sum
    const bool grow = pm > m_run + 8.f;
    const float cr = grow ? exp2f(m_run - pm) : 1.f;  // 0 when m_run was -inf
    if (__any_sync(0xffffffffu, grow) && pg > 0) {
#pragma unroll
      for (int c0 = 0; c0 < HD / 2; c0 += 16) {
        float o[16];
        tmem_ld_16(t_row + OCOL + (uint32_t)(half * (HD / 2) + c0), o);
#pragma unroll
        for (int i = 0; i < 16; ++i) o[i] *= cr;
        tmem_st_16(t_row + OCOL + (uint32_t)(half * (HD / 2) + c0), o);
      }
    }
    if (grow) {
      l_run *= cr;
      m_run = pm;
    }
    uint32_t pk[16];
    float psum = 0.f;
#pragma unroll
    for (int c = 0; c < 32; c += 2) {
      const float p0 = sc[c] == -INFINITY ? 0.f : ex2_approx(sc[c] - m_run);
      const float p1 = sc[c + 1] == -INFINITY ? 0.f : ex2_approx(sc[c + 1] - m_run);
      psum += p0 + p1;
      pk[c / 2] = pack_bf16(p0, p1);
    }
    l_run += psum;
#pragma unroll
    for (int q = 0; q < 4; ++q)
      *reinterpret_cast<uint4*>(sm + Sh::OFF_P + sw128_off(row, 4 * half + q)) =
          make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]);
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    if (tid == 0) {
      tc_fence_after();
      const uint32_t bv = smem_u32(sm + Sh::OFF_BV + (pg & 1) * Sh::BV_BYTES);
#pragma unroll
      for (int k = 0; k < 4; ++k)
        tc_mma_f16(tmem + OCOL, smem_desc_sw128(smem_u32(sm + Sh::OFF_P)) + 2 * k, smem_desc_sw128(bv) + 2 * k, IDO,
                   (pg > 0 || k > 0) ? 1u : 0u);
      tc_commit(bar_o);
    }
    __syncwarp();
  }
  mbar_wait(bar_o, (npages - 1) & 1, s.err);
  tc_fence_after();
  xch[half * 128 + row] = l_run;  // the two halves of each row sum
  __syncthreads();
  const float l_tot = l_run + xch[(half ^ 1) * 128 + row];
  const float inv_l = l_tot > 0.f ? 1.f / l_tot : 0.f;
  bf16* orow = O + (size_t)(first + q0 + qi) * md.q_dim + (kvh * G + g) * HD + half * (HD / 2);
#pragma unroll
  for (int c0 = 0; c0 < HD / 2; c0 += 16) {
    float o[16];
    tmem_ld_16(t_row + OCOL + (uint32_t)(half * (HD / 2) + c0), o);
    if (row_ok) {
      uint32_t w[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) w[i] = pack_bf16(o[2 * i] * inv_l, o[2 * i + 1] * inv_l);
      *reinterpret_cast<uint4*>(orow + c0) = make_uint4(w[0], w[1], w[2], w[3]);
      *reinterpret_cast<uint4*>(orow + c0 + 8) = make_uint4(w[4], w[5], w[6], w[7]);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, Sh::TMEM_COLS);
}

// ----------------------------------------------------------------------------
// Warp-specialised tensor-core causal attention of a chunk (bf16, head_dim 64 or 128)
// ----------------------------------------------------------------------------
// Same work split as k_pf_attn_tc (one CTA per sequence, block of QT = 128/G queries and kv head;
// the 128 MMA rows are query * G + head; cache pages of 64 slots), with the roles split across
// warps so that no block-wide barrier sits in the page loop:
//   warp 4      TMA producer: the block's q rows (bulk copies, staged in the empty rings), then the
//               K and V segments of every page, straight from the paged pool through a 3-D tensor
//               map (128-byte swizzle), into K and V rings (three deep for head_dim 128);
//   warp 5      MMA issuer: S(p) = Q K(p)^T into one of two TMEM buffers (q as bf16 hi + lo terms,
//               so the scores keep q's float32 precision), then O += P(p-1) V(p-1) with V taken as
//               an MN-major operand (no transpose);
//   warps 0-3   softmax, one thread per row: read the row of S(p) from TMEM, mask causally by cache
//               slot, keep the running maximum (refreshed lazily: O is rescaled in TMEM only when a
//               row's maximum grows by more than 8 in base 2) and sum in float32, and write P(p) in
//               bf16 to one of two shared-memory buffers; at the end they normalise O and store it.
// mbarriers connect the roles (ring full / empty, S full / free, P full / free); every wait is
// bounded. Slots past the block's last query in its last page hold finite values (the pool is
// zeroed when created and only ever holds finite entries), which the mask turns into P = 0.
constexpr int PFW_THREADS = 192;

template <int HD>
struct PfWsShape {
  static constexpr int ATOMS = HD / 64;                // 128-byte atom columns of a row
  static constexpr int Q_BYTES = 128 * HD * 2;         // one of the hi / lo Q tiles [128][HD]
  static constexpr int QCOL = 128 * 128;               // bytes of one atom column of a Q tile
  static constexpr int KV_BYTES = 64 * HD * 2;         // a K (or V) stage: [64 keys][HD]
  static constexpr int KVCOL = 64 * 128;               // bytes of one atom column of a stage
  // ring depth: with head_dim 128 a K copy is issued once the S product three pages back has freed
  // its stage, which covers the copy's latency (two stages left the MMA waiting for K); head_dim 64
  // keeps two stages so that two CTAs (101 KB each) share an SM and cover it between them
  static constexpr int NST = HD == 128 ? 3 : 2;
  static constexpr int P_BYTES = 128 * 64 * 2;         // a P buffer [128][64 keys]
  static constexpr int OFF_QHI = 0;
  static constexpr int OFF_QLO = OFF_QHI + Q_BYTES;
  static constexpr int OFF_K = OFF_QLO + Q_BYTES;
  static constexpr int OFF_V = OFF_K + NST * KV_BYTES;
  static constexpr int OFF_P = OFF_V + NST * KV_BYTES;
  static constexpr int OFF_BAR = OFF_P + 2 * P_BYTES;
  static constexpr int NBAR = 4 * NST + 9;
  static_assert(128 * HD * 4 <= 2 * NST * KV_BYTES, "the float32 Q tile is staged in the K/V rings");
  static constexpr int BYTES = OFF_BAR + NBAR * 8 + 16 + 1024;  // barriers, TMEM slot, alignment slack
  static constexpr uint32_t TMEM_COLS = 256;          // S buffers in columns 0..127, O in 128..128+HD
};

template <int HD, int G>
__global__ void __launch_bounds__(PFW_THREADS, HD == 64 ? 2 : 1) k_pf_attn_ws(ModelDims md, PrefillDev p, StepDev s, int r, int j,
                                                             const float* __restrict__ Q, bf16* __restrict__ O,
                                                             const __grid_constant__ CUtensorMap pool_map) {
  using Sh = PfWsShape<HD>;
  constexpr int QT = 128 / G, NST = Sh::NST;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + Sh::OFF_BAR);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + Sh::NBAR);
  auto bar = [&](int i) { return smem_u32(&bars[i]); };
  // K full / empty, V full / empty (NST each), then S full x2, S free x2, P full x2, P free x2
  auto k_full = [&](int st) { return bar(st); };
  auto k_empty = [&](int st) { return bar(NST + st); };
  auto v_full = [&](int st) { return bar(2 * NST + st); };
  auto v_empty = [&](int st) { return bar(3 * NST + st); };
  auto s_full = [&](int b) { return bar(4 * NST + b); };
  auto s_free = [&](int b) { return bar(4 * NST + 2 + b); };
  auto p_full = [&](int b) { return bar(4 * NST + 4 + b); };
  auto p_free = [&](int b) { return bar(4 * NST + 6 + b); };
  const uint32_t q_full = bar(4 * NST + 8);

  pdl_wait();
  pdl_trigger();
  const int S = p.S;
  const int* tbase = p.tile_base + r * (p.Smax + 1);
  // 1-D grid, kv head fastest and query blocks in reverse order: the blocks with the most pages
  // (the last queries of a sequence) are dispatched first, so the last wave holds short ones
  const int ntiles = tbase[S];
  const int kvh = blockIdx.x % md.Hkv, tile = ntiles - 1 - (int)(blockIdx.x / md.Hkv);
  if (tile < 0) return;
  int lo = 0, hi = S;  // sequence: largest sq with tbase[sq] <= tile
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (tbase[mid] <= tile) lo = mid; else hi = mid;
  }
  const int sq = lo, qb = tile - tbase[sq];
  const int cnt = p.cnt[r * p.Smax + sq], first = p.first[r * p.Smax + sq], s0 = p.s0[r * p.Smax + sq];
  const int slot = p.seq_slot[sq];
  const int q0 = qb * QT, nq = min(QT, cnt - q0);
  const int last = s0 + q0 + nq - 1;  // cache slot of the block's last query
  const int npages = last / 64 + 1;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int* ptab = s.page_table + ((size_t)slot * md.M + r) * md.max_pages;

  if (tid == 0) {
    for (int i = 0; i < NST; ++i) {
      mbar_init(k_full(i), 1);
      mbar_init(k_empty(i), 1);
      mbar_init(v_full(i), 1);
      mbar_init(v_empty(i), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(s_full(b), 1);
      mbar_init(s_free(b), 4);
      mbar_init(p_full(b), 4);
      mbar_init(p_free(b), 1);
    }
    mbar_init(q_full, 1);
    fence_barrier_init();
    prefetch_tensormap(&pool_map);
    // the block's float32 q rows, staged in the (still unused) K/V rings: the G heads of a query
    // are contiguous, so one bulk copy per query
    mbar_arrive_expect_tx(q_full, (uint32_t)(nq * G * HD * 4));
    for (int qq = 0; qq < nq; ++qq)
      bulk_g2s(smem_u32(sm + Sh::OFF_K + qq * G * HD * 4), Q + ((size_t)(first + q0 + qq) * md.Hq + kvh * G) * HD,
               (uint32_t)(G * HD * 4), q_full);
  }
  if (warp == 5) {
    tmem_alloc(smem_u32(tmem_slot), Sh::TMEM_COLS);
    tmem_relinquish();
  }
  __syncthreads();  // barriers initialised
  const bool q_ok = __all_sync(0xffffffffu, mbar_wait(q_full, 0, s.err));
  // Q tile: row = query * G + head, as hi and lo bf16 parts (zeros past the block's queries)
  const float* qstage = reinterpret_cast<const float*>(sm + Sh::OFF_K);
  for (int e = tid; e < 128 * (HD / 8); e += PFW_THREADS) {
    const int qr = e / (HD / 8), c = e % (HD / 8);
    const int qq = qr / G;
    float x[8];
    if (qq < nq && q_ok) {
      const float4* q4 = reinterpret_cast<const float4*>(qstage + (size_t)qr * HD);
      const float4 a = q4[2 * c], b = q4[2 * c + 1];
      x[0] = a.x; x[1] = a.y; x[2] = a.z; x[3] = a.w; x[4] = b.x; x[5] = b.y; x[6] = b.z; x[7] = b.w;
    } else {
#pragma unroll
      for (int u = 0; u < 8; ++u) x[u] = 0.f;
    }
    uint32_t h[4], l[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const float a0 = __bfloat162float(__float2bfloat16_rn(x[2 * u]));
      const float a1 = __bfloat162float(__float2bfloat16_rn(x[2 * u + 1]));
      h[u] = pack_bf16(a0, a1);
      l[u] = pack_bf16(x[2 * u] - a0, x[2 * u + 1] - a1);
    }
    const uint32_t off = (c / 8) * Sh::QCOL + sw128_off(qr, c % 8);
    *reinterpret_cast<uint4*>(sm + Sh::OFF_QHI + off) = make_uint4(h[0], h[1], h[2], h[3]);
    *reinterpret_cast<uint4*>(sm + Sh::OFF_QLO + off) = make_uint4(l[0], l[1], l[2], l[3]);
  }
  fence_proxy_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  constexpr uint32_t OCOL = 128;  // first TMEM column of O
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  if (tid == 0) *abort_flag = 0;
  __syncthreads();
  // a bounded wait; once any role has given up, the others skip their waits and wind down
  auto wait = [&](uint32_t b, uint32_t parity) {
    if (*abort_flag) return false;
    if (!mbar_wait(b, parity, s.err)) {
      *abort_flag = 1;
      return false;
    }
    return true;
  };

  if (warp == 4) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      const int rowK = ((j * 2 + 0) * md.Hkv + kvh) * 64, rowV = ((j * 2 + 1) * md.Hkv + kvh) * 64;
      for (int pg = 0; pg < npages; ++pg) {
        const int st = pg % NST;
        const uint32_t par = (uint32_t)((pg / NST) - 1) & 1u;
        int page = ptab[pg];
        const bool okp = page >= 0 && page < md.n_pages;
        if (!okp) atomicOr(s.err, DEVERR_INDEX);
        if (pg >= NST && !wait(k_empty(st), par)) break;
        if (okp) {
          mbar_arrive_expect_tx(k_full(st), Sh::KV_BYTES);
#pragma unroll
          for (int a = 0; a < Sh::ATOMS; ++a)
            tma_load_3d(smem_u32(sm + Sh::OFF_K + st * Sh::KV_BYTES + a * Sh::KVCOL), &pool_map, a * 64, rowK, page,
                        k_full(st));
        } else {
          mbar_arrive(k_full(st));  // complete the phase without data
        }
        if (pg >= NST && !wait(v_empty(st), par)) break;
        if (okp) {
          mbar_arrive_expect_tx(v_full(st), Sh::KV_BYTES);
#pragma unroll
          for (int a = 0; a < Sh::ATOMS; ++a)
            tma_load_3d(smem_u32(sm + Sh::OFF_V + st * Sh::KV_BYTES + a * Sh::KVCOL), &pool_map, a * 64, rowV, page,
                        v_full(st));
        } else {
          mbar_arrive(v_full(st));
        }
      }
    }
  } else if (warp == 5) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      constexpr uint32_t IDS = idesc_bf16_f32(128, 64), IDO = idesc_bf16_f32_bmn(128, HD);
      // every operand descriptor is a base plus a constant step (encoded in 16-byte units), built
      // once: this thread's instruction count per page is what paces the loop
      const uint64_t dqh = smem_desc_sw128(smem_u32(sm + Sh::OFF_QHI));
      const uint64_t dql = smem_desc_sw128(smem_u32(sm + Sh::OFF_QLO));
      const uint64_t dk0 = smem_desc_sw128(smem_u32(sm + Sh::OFF_K));
      const uint64_t dp0 = smem_desc_sw128(smem_u32(sm + Sh::OFF_P));
      const uint64_t dv0 = smem_desc_sw128_mn(smem_u32(sm + Sh::OFF_V), Sh::KVCOL);
      constexpr uint64_t QCOL_E = Sh::QCOL >> 4, KVCOL_E = Sh::KVCOL >> 4, KV_E = Sh::KV_BYTES >> 4,
                         P_E = Sh::P_BYTES >> 4, V16_E = 2048 >> 4;
      // Two streams, each issued as soon as its inputs are there: S(ns) once K(ns) has landed and the
      // softmax has read the S buffer two pages back, and P V(npv) once P(npv) and V(npv) are in.
      // S therefore runs ahead of the softmax instead of behind the P V product before it. One time
      // limit covers the whole loop.
      int ns = 0, npv = 0;
      const uint64_t t0 = globaltimer_ns();
      while (npv < npages) {
        bool did = false;
        if (ns < npages) {
          const int b = ns & 1, st = ns % NST;
          if (mbar_try_wait(k_full(st), (uint32_t)(ns / NST) & 1u) &&
              (ns < 2 || mbar_try_wait(s_free(b), (uint32_t)((ns - 2) >> 1) & 1u))) {
            tc_fence_after();
            const uint64_t kb = dk0 + st * KV_E;
            const uint32_t d = tmem + 64u * (uint32_t)b;
#pragma unroll
            for (int kc = 0; kc < Sh::ATOMS; ++kc)
#pragma unroll
              for (int k = 0; k < 4; ++k) {  // K = 16 per MMA: +32 bytes (encoded +2) inside the atom column
                const uint64_t db = kb + kc * KVCOL_E + 2 * k;
                tc_mma_f16(d, dqh + kc * QCOL_E + 2 * k, db, IDS, (kc | k) ? 1u : 0u);
                tc_mma_f16(d, dql + kc * QCOL_E + 2 * k, db, IDS, 1u);
              }
            tc_commit(s_full(b));
            tc_commit(k_empty(st));
            ++ns;
            did = true;
          }
        }
        if (npv < ns) {
          const int bq = npv & 1, st = npv % NST;
          if (mbar_try_wait(p_full(bq), (uint32_t)(npv >> 1) & 1u) &&
              mbar_try_wait(v_full(st), (uint32_t)(npv / NST) & 1u)) {  // O += P(npv) V(npv)
            tc_fence_after();
            const uint64_t pa = dp0 + bq * P_E, vb = dv0 + st * KV_E;
#pragma unroll
            for (int k = 0; k < 4; ++k)  // K = 16 keys per MMA: +32 B in P's rows, +2048 B (16 rows) in V
              tc_mma_f16(tmem + OCOL, pa + 2 * k, vb + V16_E * k, IDO, (npv > 0 || k > 0) ? 1u : 0u);
            tc_commit(p_free(bq));
            tc_commit(v_empty(st));
            ++npv;
            did = true;
          }
        }
        if (!did && (*abort_flag || globaltimer_ns() - t0 > kWaitLimitNs)) {
          atomicOr(s.err, DEVERR_WAIT);
          *abort_flag = 1;
          break;
        }
      }
    }
  } else {
    // ---------------- softmax: thread = MMA row = TMEM lane ----------------
    // The page's work per thread is short; what bounds it is the length of its dependent chains,
    // so the row maximum and sum run as four independent partials and no per-key select is taken
    // (ex2 of -inf is 0 once the reference maximum is finite).
    const int row = warp * 32 + lane;
    const uint32_t t_row = tmem + ((uint32_t)(warp * 32) << 16);
    const int qi = row / G, g = row % G;
    const bool row_ok = qi < nq;
    const int qslot = s0 + q0 + qi;  // cache slot of this row's query
    const float scale = 1.4426950408889634f * rsqrtf((float)HD);
    float m_run = -INFINITY, l_run = 0.f;
    bool ok = true;
    // waits taken by the whole warp: the TMEM accesses after them are warp-collective
    auto wait_w = [&](uint32_t bq, uint32_t parity) { return __all_sync(0xffffffffu, wait(bq, parity)); };
    for (int pg = 0; pg < npages && ok; ++pg) {
      const int b = pg & 1;
      if (!wait_w(s_full(b), (uint32_t)(pg >> 1) & 1u)) { ok = false; break; }
      tc_fence_after();
      float sc[64];
      tmem_ld_32(t_row + 64u * (uint32_t)b, sc);
      tmem_ld_32(t_row + 64u * (uint32_t)b + 32u, sc + 32);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(s_free(b));
      const int kb = pg * 64;  // cache slot of column 0
      float pm4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
      if (row_ok && kb + 63 <= qslot) {  // every key visible
#pragma unroll
        for (int c = 0; c < 64; ++c) {
          sc[c] *= scale;
          pm4[c & 3] = fmaxf(pm4[c & 3], sc[c]);
        }
      } else if (!row_ok || kb > qslot) {  // none visible
#pragma unroll
        for (int c = 0; c < 64; ++c) sc[c] = -INFINITY;
      } else {  // the diagonal: causal by cache slot
#pragma unroll
        for (int c = 0; c < 64; ++c) {
          sc[c] = kb + c <= qslot ? sc[c] * scale : -INFINITY;
          pm4[c & 3] = fmaxf(pm4[c & 3], sc[c]);
        }
      }
      const float pm = fmaxf(fmaxf(pm4[0], pm4[1]), fmaxf(pm4[2], pm4[3]));
      // lazy maximum: O is rescaled only when a row's maximum grows by more than 8, after the
      // P V product before has landed (warp-uniform TMEM access)
      const bool grow = pm > m_run + 8.f;
      const float cr = grow ? exp2f(m_run - pm) : 1.f;  // 0 when m_run was -inf
      if (pg > 0 && __any_sync(0xffffffffu, grow)) {
        if (!wait_w(p_free((pg - 1) & 1), (uint32_t)((pg - 1) >> 1) & 1u)) { ok = false; break; }
        tc_fence_after();
#pragma unroll
        for (int c0 = 0; c0 < HD; c0 += 16) {
          float o[16];
          tmem_ld_16(t_row + OCOL + (uint32_t)c0, o);
#pragma unroll
          for (int i = 0; i < 16; ++i) o[i] *= cr;
          tmem_st_16(t_row + OCOL + (uint32_t)c0, o);
        }
        tc_fence_before();
      }
      if (grow) {
        l_run *= cr;
        m_run = pm;
      }
      const float mref = m_run == -INFINITY ? 0.f : m_run;  // rows with no visible key so far
      uint32_t pk[32];
      float ps4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int c = 0; c < 64; c += 2) {
        const float p0 = ex2_approx(sc[c] - mref), p1 = ex2_approx(sc[c + 1] - mref);
        ps4[(c >> 1) & 3] += p0 + p1;
        pk[c / 2] = pack_bf16(p0, p1);
      }
      l_run += (ps4[0] + ps4[1]) + (ps4[2] + ps4[3]);
      // P buffer b was last read by P V of page pg - 2
      if (pg >= 2 && !wait_w(p_free(b), (uint32_t)((pg - 2) >> 1) & 1u)) { ok = false; break; }
      uint8_t* pb = sm + Sh::OFF_P + b * Sh::P_BYTES;
#pragma unroll
      for (int q = 0; q < 8; ++q)
        *reinterpret_cast<uint4*>(pb + sw128_off(row, q)) = make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]);
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(p_full(b));
    }
    // the last P V product, then O / l out
    if (ok && wait_w(p_free((npages - 1) & 1), (uint32_t)((npages - 1) >> 1) & 1u)) {
      tc_fence_after();
      const float inv_l = l_run > 0.f ? 1.f / l_run : 0.f;
      bf16* orow = O + (size_t)(first + q0 + qi) * md.q_dim + (kvh * G + g) * HD;
#pragma unroll
      for (int c0 = 0; c0 < HD; c0 += 16) {
        float o[16];
        tmem_ld_16(t_row + OCOL + (uint32_t)c0, o);
        if (row_ok) {
          uint32_t w[8];
#pragma unroll
          for (int i = 0; i < 8; ++i) w[i] = pack_bf16(o[2 * i] * inv_l, o[2 * i + 1] * inv_l);
          *reinterpret_cast<uint4*>(orow + c0) = make_uint4(w[0], w[1], w[2], w[3]);
          *reinterpret_cast<uint4*>(orow + c0 + 8) = make_uint4(w[4], w[5], w[6], w[7]);
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 5) tmem_dealloc(tmem, Sh::TMEM_COLS);
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
  constexpr int smem = (PF_QB * G * HD + HD * 65 + 64 * HD + PF_WARPS * (PF_QB / PF_WARPS) * G * 64) * 4;
  (void)ensure_kernel_attrs((const void*)k_pf_attn<T, HD, G>, smem);  // a failure shows at launch
  launch_k(k_pf_attn<T, HD, G>, dim3(tiles_bound, md.Hkv), 32 * PF_WARPS, smem, st, md, p, s, r, j, Q, (T*)O);
}

void launch_pf_plan(const ModelDims& md, const PrefillDev& p, cudaStream_t st) {
  launch_k(k_pf_plan, 1, 1024, 0, st, md, p);
}

template <int HD, int G>
static void pf_attn_tc_launch(const ModelDims& md, const PrefillDev& p, const StepDev& s, int r, int j,
                              const float* Q, void* O, int tiles_bound, cudaStream_t st) {
  constexpr int smem = PfTcShape<HD>::BYTES;
  (void)ensure_kernel_attrs((const void*)k_pf_attn_tc<HD, G>, smem);  // a failure shows at launch
  launch_k(k_pf_attn_tc<HD, G>, dim3(tiles_bound, md.Hkv), PFT_THREADS, smem, st, md, p, s, r, j, Q, (bf16*)O);
}

template <int HD, int G>
static void pf_attn_ws_launch(const ModelDims& md, const PrefillDev& p, const StepDev& s, int r, int j,
                              const float* Q, void* O, int tiles_bound, cudaStream_t st, const CUtensorMap* pool_map) {
  constexpr int smem = PfWsShape<HD>::BYTES;
  (void)ensure_kernel_attrs((const void*)k_pf_attn_ws<HD, G>, smem);  // a failure shows at launch
  launch_k(k_pf_attn_ws<HD, G>, dim3(tiles_bound * md.Hkv), PFW_THREADS, smem, st, md, p, s, r, j, Q, (bf16*)O,
           *pool_map);
}

// Tensor-core kernel for head_dim 64 and 128 (128-byte rows for the swizzled operand tiles); the
// CUDA-core kernel for head_dim 32.
static bool pf_attn_uses_tc(const ModelDims& md) { return md.hd == 64 || md.hd == 128; }

int pf_attn_qblock(const ModelDims& md) { return pf_attn_uses_tc(md) ? 128 / (md.Hq / md.Hkv) : PF_QB; }

void launch_pf_attn(const ModelDims& md, const PrefillDev& p, const StepDev& s, int r, int j, const float* Q,
                    void* O, int tiles_bound, cudaStream_t st, const CUtensorMap* pool_map) {
  const int G = md.Hq / md.Hkv;
  if (pool_map && (md.hd == 64 || md.hd == 128)) {
    if (md.hd == 128 && G == 1) pf_attn_ws_launch<128, 1>(md, p, s, r, j, Q, O, tiles_bound, st, pool_map);
    else if (md.hd == 128 && G == 2) pf_attn_ws_launch<128, 2>(md, p, s, r, j, Q, O, tiles_bound, st, pool_map);
    else if (md.hd == 128 && G == 4) pf_attn_ws_launch<128, 4>(md, p, s, r, j, Q, O, tiles_bound, st, pool_map);
    else if (md.hd == 64 && G == 1) pf_attn_ws_launch<64, 1>(md, p, s, r, j, Q, O, tiles_bound, st, pool_map);
    else if (md.hd == 64 && G == 2) pf_attn_ws_launch<64, 2>(md, p, s, r, j, Q, O, tiles_bound, st, pool_map);
    else pf_attn_ws_launch<64, 4>(md, p, s, r, j, Q, O, tiles_bound, st, pool_map);
    return;
  }
  if (md.hd == 128 && G == 1) pf_attn_tc_launch<128, 1>(md, p, s, r, j, Q, O, tiles_bound, st);
  else if (md.hd == 128 && G == 2) pf_attn_tc_launch<128, 2>(md, p, s, r, j, Q, O, tiles_bound, st);
  else if (md.hd == 128 && G == 4) pf_attn_tc_launch<128, 4>(md, p, s, r, j, Q, O, tiles_bound, st);
  else if (md.hd == 64 && G == 1) pf_attn_tc_launch<64, 1>(md, p, s, r, j, Q, O, tiles_bound, st);
  else if (md.hd == 64 && G == 2) pf_attn_tc_launch<64, 2>(md, p, s, r, j, Q, O, tiles_bound, st);
  else if (md.hd == 64 && G == 4) pf_attn_tc_launch<64, 4>(md, p, s, r, j, Q, O, tiles_bound, st);
  else if (md.hd == 32 && G == 1) pf_attn_launch<bf16, 32, 1>(md, p, s, r, j, Q, O, tiles_bound, st);
  else pf_attn_launch<bf16, 32, 2>(md, p, s, r, j, Q, O, tiles_bound, st);
}

void launch_pf_len(const ModelDims& md, const PrefillDev& p, cudaStream_t st) {
  launch_k(k_pf_len, 1, 256, 0, st, md, p);
}

}  // namespace tlf
