// Dense projections of the shared block on the compacted tokens (Eq. 6, 9):
// Y[row][o] = sum_k X[row][k] * W[o][k] for the n rows of the active set.
//
// k_gemm_tc (bf16): tcgen05 tensor-core GEMM. Operand roles are swapped so that
// the weight tile fills the 128-row MMA dimension and the n <= 256 tokens form
// the N dimension (decode has few tokens and many output features).
// - Warp 0 lane 0 streams 128x64 weight tiles and NTx64 token tiles into a
//   shared-memory ring of 1-4 stages with 2-D TMA (128-byte swizzle).
// - The first stages' weight tiles go out before the grid-dependency wait
//   (programmatic dependent launch). Decode weights carry an L2 evict-first
//   hint, because each tile is read once per launch.
// - Warp 1 lane 0 issues tcgen05.mma (M=128, K=16) accumulating in TMEM and
//   releases each stage with tcgen05.commit.
// - All four warps then read the accumulator with tcgen05.ld (warp w owns TMEM
//   lanes 32w..32w+31 = output features) and run the epilogue. Split-K over
//   gridDim.y keeps enough CTAs in flight to stream the weights at HBM speed.
// Two-term operands (decode): the token operand arrives as bf16 hi and lo
// planes, loaded as one B tile of 2 x NT rows; the MMA runs with N = 2 x NT
// (two MMAs of N = 256 for a 256-token tile, whose halves fill TMEM) and the
// epilogue adds the two accumulator halves.
//
// k_gemm_simt: CUDA-core tiled GEMM with the same epilogues, for float32
// models (tcgen05 has no exact float32 mode) and as a second GPU path.
//
// Cluster epilogues: the S split-K CTAs of one 128-feature tile are launched as
// a (1, S, 1) thread-block cluster. Each stages its partial tile in shared
// memory. After a cluster barrier every CTA sums a 1/S share of the tile over
// the cluster through distributed shared memory, in a fixed order, so results
// are deterministic. It then finishes the share in one of three ways:
// - residual add + scatter into the float32 stream H[idx[row]] (Eq. 7, one
//   writer per element); with a split pre-norm it also writes the next GEMM's
//   unscaled operand and per-tile sums of squares;
// - RoPE on q and k at the token's original position, with k and v appended to
//   its loop-r page (Eq. 9, 11);
// - silu(gate) * up (SwiGLU; gate and up rows interleave per 64-feature tile, so
//   one tile holds both halves).
// No partial sum leaves the chip and no separate kernel runs. Consumers of a
// split pre-norm scale each token column by its RMSNorm factor first. With one
// split (prefill) the CTA reads its own tile with plain shared loads and may
// stage it in 128-column windows, so two CTAs share an SM.
//
// Other epilogues (SIMT path, LM head): split-K partial sums to a buffer
// consumed by k_rope_append / k_swiglu, atomic residual add + scatter, or a
// plain float32 store (logits).
#include <type_traits>

#include "tlf_internal.cuh"

namespace tlf {

__device__ __forceinline__ void gemm_write(const GemmArgs& a, int split, int row, int col, float v) {
  if (a.epi == EPI_PARTIAL) {
    a.out[((size_t)split * a.max_rows + row) * a.N + col] = v;
  } else if (a.epi == EPI_RESID) {
    if (a.act && !a.act[row]) return;  // masked row (no-gather ablation): residual unchanged
    const int r = a.idx ? a.idx[row] : row;
    if (a.alpha.mod) v *= cond_row(a.alpha, r)[col];  // time/step conditioning gate
    atomicAdd(a.resid + (size_t)r * a.ldr + col, v);
  } else {
    a.out[(size_t)row * a.ldo + col] = v;
  }
}

// ----------------------------------------------------------------------------
// tcgen05 kernel
// ----------------------------------------------------------------------------
constexpr int TC_BM = 128;
constexpr int TC_BK = 64;  // 64 bf16 = one 128-byte swizzle row
constexpr int TC_STAGES = 4;  // deepest operand ring; a launch uses min(4, k-tiles per CTA) stages

// Dynamic shared memory of one CTA: the operand ring (reused after the main loop
// for the cluster epilogue's fp32 partial tile [NT columns][128 features]), the
// mbarriers and TMEM slot, and per token column one int4 of information, one
// float norm factor and four per-warp partial sums of squares. With a two-term
// operand (lo) a stage holds 2 x NT token rows.
constexpr int tc_b_bytes(int nt, bool lo) { return (lo ? 2 : 1) * nt * TC_BK * 2; }
constexpr int tc_ring_bytes(int nt, int stages, bool lo) { return stages * (TC_BM * TC_BK * 2 + tc_b_bytes(nt, lo)); }
constexpr int tc_red_bytes(int red_cols) { return TC_BM * red_cols * 4; }
// red_cols: token columns of the staged fp32 tile (nt, or the window of a one-split epilogue)
constexpr int tc_body_bytes(int nt, int stages, bool lo, int red_cols) {
  return tc_ring_bytes(nt, stages, lo) > tc_red_bytes(red_cols) ? tc_ring_bytes(nt, stages, lo)
                                                                : tc_red_bytes(red_cols);
}
// TMEM columns of one CTA: the accumulator of 2 x NT columns (hi and lo halves) with a
// two-term operand, NT otherwise, at least 32 (always a power of two).
constexpr int tc_tmem_cols(int nt, bool lo) {
  return lo ? (2 * nt < 32 ? 32 : 2 * nt) : (nt < 32 ? 32 : nt);
}
// tcgen05.alloc blocks until columns are free, so the CTAs that shared memory lets
// share an SM must fit in its 512 TMEM columns (otherwise clusters waiting for
// partners could wait on each other): launches request at least this much.
constexpr int SM_SMEM = 232448;  // shared memory per SM available to CTAs (227 KB + 1 KB per CTA)
constexpr int tc_min_smem(int nt, bool lo) { return SM_SMEM / (512 / tc_tmem_cols(nt, lo) + 1) - 1024 + 1; }
constexpr int tc_smem_bytes(int nt, int stages, bool lo, int red_cols = 0) {
  const int raw = 1024 /*align slack*/ + tc_body_bytes(nt, stages, lo, red_cols > 0 ? red_cols : nt) +
                  256 /*barriers, tmem slot*/ +
                  nt * (16 + 4 + 16);
  return raw > tc_min_smem(nt, lo) ? raw : tc_min_smem(nt, lo);
}
// Deepest operand ring of a token tile: a 256-token two-term stage holds 80 KB, so two fit.
constexpr int tc_max_stages(int nt, bool lo) { return (lo && nt >= 256) ? 2 : TC_STAGES; }
constexpr bool tmem_fits(int nt, bool lo) {
  return (SM_SMEM / (tc_smem_bytes(nt, 1, lo) + 1024)) * tc_tmem_cols(nt, lo) <= 512 &&
         tc_smem_bytes(nt, tc_max_stages(nt, lo), lo) <= SM_SMEM - 1024;
}
static_assert(tmem_fits(16, false) && tmem_fits(32, false) && tmem_fits(64, false) && tmem_fits(128, false) &&
                  tmem_fits(256, false) && tmem_fits(16, true) && tmem_fits(32, true) && tmem_fits(64, true) &&
                  tmem_fits(128, true) && tmem_fits(256, true),
              "co-resident CTAs would oversubscribe TMEM, or a ring does not fit in shared memory");

// Second half of a cluster epilogue. Every CTA of the cluster has staged its
// fp32 partial tile [NT columns][128 features] at `red`; this CTA sums the
// partners' tiles over its share of the token columns through distributed
// shared memory and finishes them according to the mode. `ci[c]` holds what
// the mode needs per token column c: for RESID the gate offset (.x), the next
// norm's conditioning offset (.y), the column of the next operand (.z, -1:
// none) and the residual row (.w, ~row for a row whose residual stays); for
// QKV the page, slot in page and position of the token's new cache entry.
// `scale[c]` is the column's RMSNorm factor when the operand arrives unscaled
// (split norm), and `ssp` [4][NT] holds per-warp sums of squares (RESID).
constexpr int CL_MAX = 8;  // largest cluster (split-K factor) of the cluster epilogues

// Sums over the cluster of the staged values at feature f, columns c..c+3
// (columns >= c1 give 0). All partner loads of the four columns are issued
// before any is used.
// With one split (prefill) the CTA's own staged tile is read with plain shared loads; it may
// hold the window of columns starting at roff.
__device__ __forceinline__ void cluster_sum4(const uint32_t* pb, const float* red, int roff, int S, int f, int c,
                                             int c1, float out[4]) {
  if (S == 1) {
#pragma unroll
    for (int q = 0; q < 4; ++q) out[q] = (c + q < c1) ? red[(c + q - roff) * 128 + f] : 0.f;
    return;
  }
  float v[CL_MAX][4];
#pragma unroll
  for (int p = 0; p < CL_MAX; ++p)
#pragma unroll
    for (int q = 0; q < 4; ++q)
      v[p][q] = (p < S && c + q < c1) ? dsmem_ld_f32(pb[p] + 4u * (uint32_t)((c + q) * 128 + f)) : 0.f;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    float s = 0.f;
#pragma unroll
    for (int p = 0; p < CL_MAX; ++p) s += v[p][q];
    out[q] = s;
  }
}

// Columns of a cluster rank's share whose residual values the split-norm
// epilogue takes from registers loaded before the main loop's end.
constexpr int HPRE = 8;

// The token columns [c0, c1) this CTA finishes in a cluster epilogue.
__device__ __forceinline__ void cluster_cols(int n, int S, int& c0, int& c1) {
  const int per = (n + S - 1) / S;
  c0 = (int)cluster_ctarank() * per;
  c1 = min(n, c0 + per);
}

template <int NT>
__device__ void cluster_epilogue(const GemmArgs& a, float* red, int4* ci, const float* scale, float* ssp,
                                 const float (&hpre)[HPRE], int m0, int n, int tok0, int cw0, int cw1) {
  const int S = a.splits;
  int c0, c1;
  cluster_cols(n, S, c0, c1);
  // columns of this pass: the CTA's share within the staged window [cw0, cw1) (the whole share
  // unless a one-split epilogue stages in windows; the split-norm path is never windowed)
  const int w0 = c0 > cw0 ? c0 : cw0, w1 = c1 < cw1 ? c1 : cw1;
  const int tid = threadIdx.x;
  uint32_t pb[CL_MAX];
  const uint32_t base = smem_u32(red);
#pragma unroll
  for (int p = 0; p < CL_MAX; ++p) pb[p] = (p < S) ? dsmem_map(base, (uint32_t)p) : 0u;

  if (a.epi == EPI_CL_RESID) {
    const int col = m0 + tid;
    if (!a.xn) {
      if (col < a.N)
        for (int c = w0; c < w1; c += 4) {
          float sm[4];
          cluster_sum4(pb, red, cw0, S, tid, c, w1, sm);
#pragma unroll
          for (int q = 0; q < 4; ++q)
            if (c + q < w1 && ci[c + q].w >= 0) {  // the only writer of this element
              const float g = a.alpha.mod ? a.alpha.mod[ci[c + q].x + col] : 1.f;
              atomicAdd(a.resid + (size_t)ci[c + q].w * a.ldr + col, g * sm[q]);
            }
        }
      return;
    }
    // Split norm: the new residual value also feeds the next pre-norm. Every thread runs
    // every column (features >= N count as 0) so the warp sums see full warps.
    const bool fin = col < a.N;
    const float gain = fin ? a.gain[col] : 0.f;
    const int warp = tid >> 5, lane = tid & 31;
    // column c (uniform over the CTA): h is its residual value before the update; returns the
    // square of the updated value (the next norm's share of this feature)
    auto update = [&](int c, float h, float sm) {
      const int4 e = ci[c];
      if (fin && e.w >= 0) {  // the only writer of this element
        const float g = a.alpha.mod ? a.alpha.mod[e.x + col] : 1.f;
        h += g * sm;
        a.resid[(size_t)e.w * a.ldr + col] = h;
      }
      if (e.z >= 0 && fin) {
        const float gm = a.gamma.mod ? 1.f + a.gamma.mod[e.y + col] : 1.f;
        const float y = h * gain * gm;
        const bf16 yh = __float2bfloat16_rn(y);
        a.xn[(size_t)e.z * a.N + col] = yh;
        if (a.xn_lo) a.xn_lo[(size_t)e.z * a.N + col] = __float2bfloat16_rn(y - __bfloat162float(yh));
      }
      return h * h;
    };
    // the warp sums of Q columns' squares, their shuffle chains interleaved
    auto sums = [&](int c, float* t, auto qn) {
      constexpr int Q = decltype(qn)::value;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1)
#pragma unroll
        for (int q = 0; q < Q; ++q) t[q] += __shfl_xor_sync(0xffffffffu, t[q], o);
      if (lane == 0)
#pragma unroll
        for (int q = 0; q < Q; ++q)
          if (c + q < c1 && ci[c + q].z >= 0) ssp[warp * NT + c + q] = t[q];
    };
    if (c1 - c0 <= HPRE) {
      float sm[HPRE];
#pragma unroll
      for (int q = 0; q < HPRE; q += 4) cluster_sum4(pb, red, 0, S, tid, c0 + q, c1, sm + q);
      float t[HPRE];
#pragma unroll
      for (int q = 0; q < HPRE; ++q) t[q] = (c0 + q < c1) ? update(c0 + q, hpre[q], sm[q]) : 0.f;
      sums(c0, t, std::integral_constant<int, HPRE>{});
    } else {
      for (int c = c0; c < c1; c += 4) {
        float hv[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int w = (c + q < c1) ? ci[c + q].w : -1;
          hv[q] = (fin && c + q < c1) ? a.resid[(size_t)(w >= 0 ? w : ~w) * a.ldr + col] : 0.f;
        }
        float sm[4];
        cluster_sum4(pb, red, 0, S, tid, c, c1, sm);
        float t[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) t[q] = (c + q < c1) ? update(c + q, hv[q], sm[q]) : 0.f;
        sums(c, t, std::integral_constant<int, 4>{});
      }
    }
    __syncthreads();
    for (int c = c0 + tid; c < c1; c += blockDim.x) {
      const int dst = ci[c].z;
      if (dst >= 0)
        a.ss_out[(size_t)dst * a.ldss + m0 / TC_BM] = ssp[c] + ssp[NT + c] + ssp[2 * NT + c] + ssp[3 * NT + c];
    }
    return;
  }
  // With a pair of rows per output (gate and up, or the two halves of a rotary pair), the
  // threads of the pair's upper row take the second half of the token columns.
  const int cm = w0 + (w1 - w0 + 1) / 2;
  if (a.epi == EPI_CL_SWIGLU) {
    const int f = tid & 63, hs = tid >> 6;
    const int gf = (m0 >> 1) + f;  // 64 gate rows then 64 up rows per 128-row tile
    const int ca = hs ? cm : w0, cb = hs ? w1 : cm;
    if (gf < a.md.ff)
      for (int c = ca; c < cb; c += 4) {
        float g[4], u[4];
        cluster_sum4(pb, red, cw0, S, f, c, cb, g);
        cluster_sum4(pb, red, cw0, S, f + 64, c, cb, u);
#pragma unroll
        for (int q = 0; q < 4; ++q)
          if (c + q < cb) {
            const float f = a.ss_in ? scale[c + q] : 1.f;
            const float gq = g[q] * f;
            const float y = gq / (1.f + expf(-gq)) * (u[q] * f);
            const bf16 yh = __float2bfloat16_rn(y);
            const size_t at = (size_t)(tok0 + c + q) * a.md.ff + gf;
            reinterpret_cast<bf16*>(a.U)[at] = yh;
            if (a.U_lo) reinterpret_cast<bf16*>(a.U_lo)[at] = __float2bfloat16_rn(y - __bfloat162float(yh));
          }
      }
    return;
  }
  // EPI_CL_QKV: column c is token k = tok0 + c of A_r
  const ModelDims& md = a.md;
  const StepDev& s = a.s;
  const int ps = md.page_size, hd = md.hd, half = hd / 2;
  if (a.row_cslot && cw0 == 0) {
    // prefill: sequence slot, cache slot and position of each row from the prefill plan (once, in
    // the first window)
    for (int c = c0 + tid; c < c1; c += blockDim.x) {
      const int row = tok0 + c;
      const int slot = a.row_slot[row], L = a.row_cslot[row];
      int pos = a.row_pos[row];
      int page = s.page_table[((size_t)slot * md.M + a.r) * md.max_pages + L / ps];
      if (page < 0 || page >= md.n_pages || pos < 0 || pos >= md.max_pos) {
        atomicOr(s.err, DEVERR_INDEX);
        page = -1;
        pos = 0;
      } else if (a.j == 0) {
        s.pos_table[(size_t)page * ps + L % ps] = pos;
      }
      ci[c] = make_int4(page, L % ps, pos, 0);
    }
    __syncthreads();
  }
  const int gfeat = m0 + tid;
  if (gfeat >= md.qkv_dim) return;
  bf16* pool = reinterpret_cast<bf16*>(s.pool);
  if (gfeat < md.q_dim + md.kv_dim) {
    const bool is_q = gfeat < md.q_dim;
    const int fr = is_q ? gfeat : gfeat - md.q_dim;
    const int h = fr / hd, hs = (fr % hd) >= half;
    const int i = (fr % hd) - hs * half;   // rotary pair (i, i + half) of head h
    const int tlo = tid - hs * half;       // tile row of the pair's lower element
    const int ca = hs ? cm : w0, cb = hs ? w1 : cm;
    for (int c = ca; c < cb; c += 4) {
      float2 csn[4];
#pragma unroll
      for (int q = 0; q < 4; ++q)
        csn[q] = (c + q < cb) ? a.rope[(size_t)ci[c + q].z * half + i] : make_float2(1.f, 0.f);
      float x0[4], x1[4];
      cluster_sum4(pb, red, cw0, S, tlo, c, cb, x0);
      cluster_sum4(pb, red, cw0, S, tlo + half, c, cb, x1);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int cc = c + q;
        if (cc >= cb) break;
        if (a.ss_in) {
          x0[q] *= scale[cc];
          x1[q] *= scale[cc];
        }
        const float r0 = x0[q] * csn[q].x - x1[q] * csn[q].y, r1 = x0[q] * csn[q].y + x1[q] * csn[q].x;
        if (is_q) {
          float* qo = a.Q + ((size_t)(tok0 + cc) * md.Hq + h) * hd;
          qo[i] = r0;
          qo[i + half] = r1;
        } else {
          const int4 e = ci[cc];
          if (e.x >= 0) {
            bf16* kp = pool + (size_t)e.x * md.page_elems + ((size_t)(a.j * 2 + 0) * md.Hkv + h) * ps * hd +
                       (size_t)e.y * hd;
            kp[i] = __float2bfloat16_rn(r0);
            kp[i + half] = __float2bfloat16_rn(r1);
          }
        }
      }
    }
  } else {
    const int fr = gfeat - md.q_dim - md.kv_dim;
    const int h = fr / hd, i = fr % hd;
    for (int c = w0; c < w1; c += 4) {
      float x[4];
      cluster_sum4(pb, red, cw0, S, tid, c, w1, x);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int cc = c + q;
        if (cc < w1 && ci[cc].x >= 0) {
          bf16* vp = pool + (size_t)ci[cc].x * md.page_elems + ((size_t)(a.j * 2 + 1) * md.Hkv + h) * ps * hd +
                     (size_t)ci[cc].y * hd;
          vp[i] = __float2bfloat16_rn(a.ss_in ? x[q] * scale[cc] : x[q]);
        }
      }
    }
  }
}

// 16 accumulator columns; with a two-term operand (lo_off > 0) plus the lo half lo_off columns on
// (both loads in flight before one wait).
__device__ __forceinline__ void tmem_ld_acc(uint32_t taddr, int lo_off, float* v) {
  uint32_t r[16], w[16];
  tmem_ld_16_issue(taddr, r);
  if (lo_off > 0) tmem_ld_16_issue(taddr + (uint32_t)lo_off, w);
  tmem_ld_wait();
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = lo_off > 0 ? __uint_as_float(r[i]) + __uint_as_float(w[i]) : __uint_as_float(r[i]);
}

// LO: the token operand is two-term (hi + lo planes); a compile-time choice, so the one-plane
// instantiations (prefill, the LM head) carry none of its code.
template <int NT, bool LO>
__global__ void __launch_bounds__(128) k_gemm_tc(const __grid_constant__ CUtensorMap mapW,
                                                 const __grid_constant__ CUtensorMap mapX, GemmArgs a) {
  constexpr int A_BYTES = TC_BM * TC_BK * 2;
  constexpr bool lo = LO;
  constexpr uint32_t TMEM_COLS = (uint32_t)tc_tmem_cols(NT, lo);
  const int B_BYTES = tc_b_bytes(NT, lo);
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int NS = a.stages;  // 1..TC_STAGES
  uint8_t* sA = smem;
  uint8_t* sB = smem + NS * A_BYTES;
  // one-split epilogues may stage the tile in windows of red_window columns (smaller smem)
  const int RW = (a.red_window > 0 && a.splits == 1 && a.red_window < NT) ? a.red_window : NT;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + tc_body_bytes(NT, NS, lo, RW));
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * TC_STAGES + 1);
  int4* colinfo = reinterpret_cast<int4*>(reinterpret_cast<uint8_t*>(bars) + 256);  // [NT]
  float* colscale = reinterpret_cast<float*>(colinfo + NT);                          // [NT]
  float* ssp = colscale + NT;                                                       // [4][NT]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // The token count comes from the plan kernel, which completed before this
  // grid was launched (every kernel triggers its successor only after its own
  // wait), so it is read before pdl_wait(), bypassing L1.
  const int n_all = a.n_dev ? __ldcg(a.n_dev) : a.n_host;
  const int tok0 = blockIdx.z * NT;  // token tile of this CTA (prefill has many)
  if (n_all <= tok0) {
    pdl_wait();
    pdl_trigger();
    return;
  }
  const int n = min(NT, n_all - tok0);      // token columns of this tile
  const int ncols = ((n + 15) / 16) * 16;  // MMA N: multiple of 16, <= NT
  const int m0 = blockIdx.x * TC_BM;
  const int split = blockIdx.y;
  const int nkb = (a.K + TC_BK - 1) / TC_BK;
  const int kb0 = (int)((long long)split * nkb / a.splits);
  const int kb1 = (int)((long long)(split + 1) * nkb / a.splits);
  const int nk = kb1 - kb0;

  auto full = [&](int i) { return smem_u32(&bars[i]); };
  auto empty = [&](int i) { return smem_u32(&bars[TC_STAGES + i]); };
  const uint32_t done = smem_u32(&bars[2 * TC_STAGES]);

  if (threadIdx.x == 0) {
    for (int i = 0; i < NS; ++i) {
      mbar_init(full(i), 1);
      mbar_init(empty(i), 1);
    }
    mbar_init(done, 1);
    fence_barrier_init();
    prefetch_tensormap(&mapW);
    prefetch_tensormap(&mapX);
  }
  if (warp == 0) {
    tmem_alloc(smem_u32(tmem_slot), TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0 && lane == 0) {
    // TMA producer. Weight tiles of the first stages go out before the wait on
    // the preceding kernels (weights are never written by them); token tiles after.
    // decode reads each weight tile once per launch (streamed, evicted first); prefill's token
    // tiles share them
    const uint64_t w_policy = gridDim.z == 1 ? l2_policy_evict_first() : l2_policy_evict_normal();
    const int pre = nk < NS ? nk : NS;
    for (int i = 0; i < pre; ++i) {
      mbar_arrive_expect_tx(full(i), A_BYTES + B_BYTES);
      tma_load_2d_hint(smem_u32(sA + i * A_BYTES), &mapW, (kb0 + i) * TC_BK, m0, full(i), w_policy);
    }
    pdl_wait();
    pdl_trigger();
    // token tiles; a two-term operand adds its lo plane (a.blo rows down) as rows NT..2NT-1
    auto load_x = [&](int st, int kx) {
      tma_load_2d(smem_u32(sB + st * B_BYTES), &mapX, kx, tok0, full(st));
      if (lo) tma_load_2d(smem_u32(sB + st * B_BYTES + NT * TC_BK * 2), &mapX, kx, tok0 + a.blo, full(st));
    };
    for (int i = 0; i < pre; ++i) load_x(i, (kb0 + i) * TC_BK);
    for (int i = pre; i < nk; ++i) {
      const int st = i % NS;
      const uint32_t ph = (uint32_t)(i / NS) & 1u;
      if (!mbar_wait(empty(st), ph ^ 1u, a.err)) break;
      mbar_arrive_expect_tx(full(st), A_BYTES + B_BYTES);
      const int kx = (kb0 + i) * TC_BK;
      tma_load_2d_hint(smem_u32(sA + st * A_BYTES), &mapW, kx, m0, full(st), w_policy);
      load_x(st, kx);
    }
  } else {
    pdl_wait();
    pdl_trigger();
    if (warp >= 2) {
      // idle during the main loop: fetch what the epilogue needs per token column
      // (outputs of the plan kernel and of the preceding GEMM, read after the wait)
      for (int c = threadIdx.x - 64; c < n; c += 64) {
        if (a.ss_in) {
          // split norm: the column's factor from the producer's per-tile sums of squares
          const float4* p4 = reinterpret_cast<const float4*>(a.ss_in + (size_t)(tok0 + c) * a.ldss);
          float t = 0.f;
#pragma unroll 4
          for (int k = 0; k < a.ldss / 4; ++k) {
            const float4 v = p4[k];
            t += (v.x + v.y) + (v.z + v.w);
          }
          colscale[c] = rsqrtf(t / (float)a.K + a.norm_eps);
        }
        if (a.epi == EPI_CL_QKV && !a.row_cslot) {
          colinfo[c] = a.s.rowinfo[a.r * a.md.max_batch + tok0 + c];
        } else if (a.epi == EPI_CL_RESID) {
          // residual row, ~row for a row masked by the no-gather ablation (residual unchanged);
          // with time/step conditioning, the offset of the row's gate vector in the table;
          // with a split norm, the row's column in the next operand and its conditioning offset
          const int row = a.idx ? a.idx[tok0 + c] : tok0 + c;
          const bool masked = a.act && !a.act[tok0 + c];
          const int aoff = (a.alpha.mod && !masked) ? (int)(cond_row(a.alpha, row) - a.alpha.mod) : 0;
          int goff = 0, dst = -1;
          if (a.xn) {
            dst = a.next_col ? a.next_col[row] : tok0 + c;
            if (a.gamma.mod && dst >= 0) goff = (int)(cond_row(a.gamma, row) - a.gamma.mod);
          }
          colinfo[c] = make_int4(aoff, goff, dst, masked ? ~row : row);
        }
      }
    }
  }
  if (nk > 0) {
    if (warp == 1 && lane == 0) {
      // MMA issuer
      // a two-term operand: MMA N covers the hi rows (NT) and the lo rows (NT); N is at most
      // 256, so a 256-token tile multiplies its lo rows (32 KB further into the stage) in a
      // second MMA into TMEM columns 256..511
      constexpr bool SPLIT_LO = 2 * NT > 256;
      const uint32_t idesc = idesc_bf16_f32(TC_BM, lo ? (SPLIT_LO ? NT : 2 * NT) : ncols);
      constexpr uint64_t LO_DESC_OFF = (uint64_t)(NT * TC_BK * 2) >> 4;  // encoded start-address step
      for (int i = 0; i < nk; ++i) {
        const int st = i % NS;
        const uint32_t ph = (uint32_t)(i / NS) & 1u;
        if (!mbar_wait(full(st), ph, a.err)) break;
        tc_fence_after();
        const uint64_t da = smem_desc_sw128(smem_u32(sA + st * A_BYTES));
        const uint64_t db = smem_desc_sw128(smem_u32(sB + st * B_BYTES));
#pragma unroll
        for (int k = 0; k < TC_BK / 16; ++k) {  // +32 bytes per K step of 16 bf16 (encoded >> 4)
          const uint32_t acc = (i > 0 || k > 0) ? 1u : 0u;
          tc_mma_f16(tmem, da + 2 * k, db + 2 * k, idesc, acc);
          if (SPLIT_LO && lo) tc_mma_f16(tmem + (uint32_t)NT, da + 2 * k, db + LO_DESC_OFF + 2 * k, idesc, acc);
        }
        tc_commit(empty(st));
      }
      tc_commit(done);
    }
  }
  __syncwarp();

  // Split norm: load this thread's residual values (feature m0 + tid of its first
  // HPRE columns) while the last MMAs drain; the epilogue updates them in place.
  // (Issued earlier, right after the wait, these loads measured slower.)
  float hpre[HPRE];
#pragma unroll
  for (int q = 0; q < HPRE; ++q) hpre[q] = 0.f;
  if (a.epi == EPI_CL_RESID && a.xn) {
    int c0, c1;
    cluster_cols(n, a.splits, c0, c1);
    const int col = m0 + threadIdx.x;
    if (c1 - c0 <= HPRE && col < a.N) {
#pragma unroll
      for (int q = 0; q < HPRE; ++q)
        if (c0 + q < c1) {
          const int row = a.idx ? a.idx[tok0 + c0 + q] : tok0 + c0 + q;
          hpre[q] = a.resid[(size_t)row * a.ldr + col];
        }
    }
  }

  // Epilogue: warp w holds output features m0 + 32w + lane; columns are token rows.
  bool ok = true;
  if (nk > 0) ok = mbar_wait(done, 0, a.err);
  ok = __all_sync(0xffffffffu, ok);  // tcgen05.ld is warp-collective
  tc_fence_after();
  if (a.epi >= EPI_CL_RESID) {
    // Stage the partial tile in shared memory (the operand ring is free now),
    // then reduce across the cluster. Every CTA reaches both cluster barriers.
    // tile layout [column][128 features]: a warp's partner reads are 128 contiguous bytes
    float* red = reinterpret_cast<float*>(smem);
    const int f = warp * 32 + lane;
    for (int w = 0; w < ncols; w += RW) {  // one pass unless a one-split tile is staged in windows
      const int wend = w + RW < ncols ? w + RW : ncols;
      if (w > 0) __syncthreads();  // every thread is done with the previous window
      for (int c0 = w; c0 < wend; c0 += 16) {
        float v[16];
        if (ok && nk > 0) {
          tmem_ld_acc(tmem + ((uint32_t)(warp * 32) << 16) + (uint32_t)c0, lo ? NT : 0, v);
        } else {
#pragma unroll
          for (int i = 0; i < 16; ++i) v[i] = 0.f;
        }
#pragma unroll
        for (int i = 0; i < 16; ++i) red[(c0 - w + i) * 128 + f] = v[i];
      }
      tc_fence_before();
      __syncthreads();
      if (wend == ncols && warp == 0) tmem_dealloc(tmem, TMEM_COLS);
      cluster_sync_all();  // every partner's tile is staged
      cluster_epilogue<NT>(a, red, colinfo, colscale, ssp, hpre, m0, n, tok0, w, w + RW);
      __syncwarp();
      cluster_sync_all();  // partners have finished reading this CTA's tile
    }
    return;
  }
  if (ok) {
    const int col = m0 + warp * 32 + lane;
    for (int c0 = 0; c0 < ncols; c0 += 16) {
      float v[16];
      if (nk > 0) {
        tmem_ld_acc(tmem + ((uint32_t)(warp * 32) << 16) + (uint32_t)c0, lo ? NT : 0, v);
      } else {
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] = 0.f;
      }
      if (col < a.N) {
#pragma unroll
        for (int i = 0; i < 16; ++i)
          if (c0 + i < n && (nk > 0 || a.epi == EPI_PARTIAL)) gemm_write(a, split, tok0 + c0 + i, col, v[i]);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, TMEM_COLS);
}

int gemm_tc_stages(int K, int splits, int nt, bool lo) {
  const int nkb = (K + TC_BK - 1) / TC_BK;
  const int per_cta = (nkb + splits - 1) / splits;
  const int cap = tc_max_stages(nt, lo);
  return per_cta < 1 ? 1 : (per_cta > cap ? cap : per_cta);
}

int gemm_tc_smem_bytes(int nt, int stages, bool lo) { return tc_smem_bytes(nt, stages, lo); }


template <int NT, bool LO>
static void launch_tc_nt(const CUtensorMap* mapW, const CUtensorMap* mapX, GemmArgs a, cudaStream_t st) {
  // (a failure shows at launch)
  (void)ensure_kernel_attrs((const void*)k_gemm_tc<NT, LO>, tc_smem_bytes(NT, tc_max_stages(NT, LO), LO));
  a.stages = gemm_tc_stages(a.K, a.splits, NT, LO);
  int red_cols = NT;
  if (a.red_window > 0 && a.splits == 1 && a.red_window < NT) {
    // windowed one-split epilogue: with a 2-stage ring two CTAs share an SM, so one CTA's
    // epilogue overlaps the other's main loop
    red_cols = a.red_window;
    if (a.stages > 2) a.stages = 2;
  } else {
    a.red_window = 0;
  }
  const int smem = tc_smem_bytes(NT, a.stages, LO, red_cols);
  dim3 grid((a.N + TC_BM - 1) / TC_BM, a.splits, a.tok_tiles > 0 ? a.tok_tiles : 1);
  if (a.epi < EPI_CL_RESID) {
    launch_k(k_gemm_tc<NT, LO>, grid, 128, smem, st, *mapW, *mapX, a);
    return;
  }
  // cluster epilogue: the splits of one tile form a (1, splits, 1) cluster
  if (a.splits > 8)
    (void)ensure_kernel_attrs((const void*)k_gemm_tc<NT, LO>, tc_smem_bytes(NT, tc_max_stages(NT, LO), LO), true);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(128);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 1;
  attr[0].val.clusterDim.y = a.splits;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = g_use_pdl ? 2 : 1;
  cudaLaunchKernelEx(&cfg, k_gemm_tc<NT, LO>, *mapW, *mapX, a);
}

template <bool LO>
static void launch_tc(const CUtensorMap* mapW, const CUtensorMap* mapX, int nt_max, const GemmArgs& a,
                      cudaStream_t st) {
  switch (nt_max) {
    case 16: launch_tc_nt<16, LO>(mapW, mapX, a, st); break;
    case 32: launch_tc_nt<32, LO>(mapW, mapX, a, st); break;
    case 64: launch_tc_nt<64, LO>(mapW, mapX, a, st); break;
    case 128: launch_tc_nt<128, LO>(mapW, mapX, a, st); break;
    default: launch_tc_nt<256, LO>(mapW, mapX, a, st); break;
  }
}

void launch_gemm_tc(const CUtensorMap* mapW, const CUtensorMap* mapX, int nt_max, const GemmArgs& a,
                    cudaStream_t st) {
  if (a.blo > 0) launch_tc<true>(mapW, mapX, nt_max, a, st);
  else launch_tc<false>(mapW, mapX, nt_max, a, st);
}

// ----------------------------------------------------------------------------
// SIMT kernel: 64 features x 32 rows per CTA, K in steps of 32
// ----------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(256) k_gemm_simt(const T* __restrict__ W, const T* __restrict__ X, int ldx,
                                                   GemmArgs a) {
  __shared__ float Ws[32][65];
  __shared__ float Xs[32][33];
  pdl_wait();
  pdl_trigger();
  const int n = a.n_dev ? *a.n_dev : a.n_host;
  if (n <= 0) return;
  const int f0 = blockIdx.x * 64;
  const int split = blockIdx.y;
  const int nkb = (a.K + 31) / 32;
  const int kb0 = (int)((long long)split * nkb / a.splits);
  const int kb1 = (int)((long long)(split + 1) * nkb / a.splits);
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  for (int row0 = 0; row0 < n; row0 += 32) {
    float acc[4][2] = {{0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}};
    for (int kb = kb0; kb < kb1; ++kb) {
      const int k0 = kb * 32;
      for (int e = tid; e < 64 * 32; e += 256) {
        const int fi = e >> 5, kk = e & 31, f = f0 + fi, k = k0 + kk;
        Ws[kk][fi] = (f < a.N && k < a.K) ? to_f32(W[(size_t)f * a.K + k]) : 0.f;
      }
      for (int e = tid; e < 32 * 32; e += 256) {
        const int ri = e >> 5, kk = e & 31, rr = row0 + ri, k = k0 + kk;
        Xs[kk][ri] = (rr < n && k < a.K) ? to_f32(X[(size_t)rr * ldx + k]) : 0.f;
      }
      __syncthreads();
#pragma unroll 8
      for (int kk = 0; kk < 32; ++kk) {
        float w[4], x[2];
#pragma unroll
        for (int i = 0; i < 4; ++i) w[i] = Ws[kk][ty * 4 + i];
        x[0] = Xs[kk][tx * 2];
        x[1] = Xs[kk][tx * 2 + 1];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          acc[i][0] = fmaf(w[i], x[0], acc[i][0]);
          acc[i][1] = fmaf(w[i], x[1], acc[i][1]);
        }
      }
      __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        const int f = f0 + ty * 4 + i, rr = row0 + tx * 2 + c;
        if (f < a.N && rr < n) gemm_write(a, split, rr, f, acc[i][c]);
      }
  }
}

void launch_gemm_simt(int dtype, const void* W, const void* X, int ldx, const GemmArgs& a, cudaStream_t st) {
  dim3 grid((a.N + 63) / 64, a.splits);
  if (dtype == 1)
    launch_k(k_gemm_simt<bf16>, grid, 256, 0, st, (const bf16*)W, (const bf16*)X, ldx, a);
  else
    launch_k(k_gemm_simt<float>, grid, 256, 0, st, (const float*)W, (const float*)X, ldx, a);
}

}  // namespace tlf
