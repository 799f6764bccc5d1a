// Dense projections of the shared block on the compacted tokens (Eq. 6, 9):
// Y[row][o] = sum_k X[row][k] * W[o][k] for the n rows of the active set.
//
// k_gemm_tc (bf16): tcgen05 tensor-core GEMM. Operand roles are swapped so
// that the weight tile fills the 128-row MMA dimension and the n <= 256 tokens
// form the N dimension (decode has few tokens and many output features).
// Warp 0 lane 0 streams 128x64 weight tiles and NTx64 token tiles into a
// 4-stage shared-memory ring with 2-D TMA (128-byte swizzle); warp 1 lane 0
// issues tcgen05.mma (M=128, N=round16(n), K=16) accumulating in TMEM and
// releases each stage with tcgen05.commit; then all four warps read the
// accumulator with tcgen05.ld (warp w owns TMEM lanes 32w..32w+31 = output
// features) and run the epilogue. Split-K over gridDim.y keeps enough CTAs
// in flight to stream the weights at HBM speed.
//
// k_gemm_simt: CUDA-core tiled GEMM with the same epilogues, for float32
// models (tcgen05 has no exact float32 mode) and as a second GPU path.
//
// Epilogues of the bf16 decode path (cluster epilogues): the S split-K CTAs
// of one 128-feature tile are launched as a (1, S, 1) thread-block cluster.
// Each stages its partial tile in shared memory; after a cluster barrier
// every CTA sums a 1/S share of the tile over the cluster through distributed
// shared memory (fixed order, so results are deterministic) and finishes it:
// residual add + scatter into the float32 stream H[idx[row]] (Eq. 7, one
// writer per element), RoPE on q and k at the token's original position with
// k and v appended to its loop-r page (Eq. 9, 11), or silu(gate) * up
// (SwiGLU; gate and up rows interleave per 64-feature tile so one tile holds
// both halves). No partial sum leaves the chip and no separate kernel runs.
//
// Other epilogues (SIMT path, prefill, LM head): split-K partial sums to a
// buffer consumed by k_rope_append / k_swiglu, atomic residual add + scatter,
// or a plain float32 store (logits).
#include "tlf_internal.cuh"

namespace tlf {

__device__ __forceinline__ void gemm_write(const GemmArgs& a, int split, int row, int col, float v) {
  if (a.epi == EPI_PARTIAL) {
    a.out[((size_t)split * a.max_rows + row) * a.N + col] = v;
  } else if (a.epi == EPI_RESID) {
    const int r = a.idx ? a.idx[row] : row;
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
constexpr int TC_STAGES = 4;

template <int NT>
constexpr int tc_smem_bytes() {
  return 1024 /*align slack*/ + TC_STAGES * (TC_BM * TC_BK * 2 + NT * TC_BK * 2) + 256 /*barriers, tmem slot*/;
}

// Second half of a cluster epilogue. Every CTA of the cluster has staged its
// fp32 partial tile [128 features][NT + 1] at `red`; this CTA sums the partners'
// tiles over its share of the token columns through distributed shared memory
// and finishes them according to the mode.
constexpr int CL_MAX = 8;  // largest cluster (split-K factor) of the cluster epilogues

// Sums over the cluster of the staged values at feature f, columns c..c+3
// (columns >= c1 give 0). All partner loads of the four columns are issued
// before any is used.
__device__ __forceinline__ void cluster_sum4(const uint32_t* pb, int S, int f, int c, int c1, float out[4]) {
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

template <int NT>
__device__ void cluster_epilogue(const GemmArgs& a, float* red, int* colinfo, int m0, int n, int tok0) {
  const int S = a.splits;
  const int rank = (int)cluster_ctarank();
  const int per = (n + S - 1) / S;
  const int c0 = rank * per, c1 = min(n, c0 + per);
  const int tid = threadIdx.x;
  uint32_t pb[CL_MAX];
  const uint32_t base = smem_u32(red);
#pragma unroll
  for (int p = 0; p < CL_MAX; ++p) pb[p] = (p < S) ? dsmem_map(base, (uint32_t)p) : 0u;

  if (a.epi == EPI_CL_RESID) {
    const int col = m0 + tid;
    if (col < a.N)
      for (int c = c0; c < c1; c += 4) {
        float sm[4];
        cluster_sum4(pb, S, tid, c, c1, sm);
#pragma unroll
        for (int q = 0; q < 4; ++q)
          if (c + q < c1) {
            const int row = a.idx ? a.idx[tok0 + c + q] : tok0 + c + q;
            atomicAdd(a.resid + (size_t)row * a.ldr + col, sm[q]);  // the only writer of this element
          }
      }
    return;
  }
  if (a.epi == EPI_CL_SWIGLU) {
    const int gf = (m0 >> 1) + tid;  // 64 gate rows then 64 up rows per 128-row tile
    if (tid < 64 && gf < a.md.ff)
      for (int c = c0; c < c1; c += 4) {
        float g[4], u[4];
        cluster_sum4(pb, S, tid, c, c1, g);
        cluster_sum4(pb, S, tid + 64, c, c1, u);
#pragma unroll
        for (int q = 0; q < 4; ++q)
          if (c + q < c1)
            reinterpret_cast<bf16*>(a.U)[(size_t)(tok0 + c + q) * a.md.ff + gf] =
                __float2bfloat16_rn(g[q] / (1.f + expf(-g[q])) * u[q]);
      }
    return;
  }
  // EPI_CL_QKV: column c is token k = c of A_r
  const ModelDims& md = a.md;
  const StepDev& s = a.s;
  const int ps = md.page_size, hd = md.hd, half = hd / 2;
  int* ci_pos = colinfo;
  int* ci_page = colinfo + NT;
  int* ci_off = colinfo + 2 * NT;
  for (int t = tid; t < c1 - c0; t += blockDim.x) {
    const int row = tok0 + c0 + t;
    int slot, L, pos;
    if (a.row_cslot) {  // prefill: per-row sequence slot, cache slot and position from the plan
      slot = a.row_slot[row];
      L = a.row_cslot[row];
      pos = a.row_pos[row];
    } else {            // decode: the token appends at the end of its loop-r cache
      slot = s.slots[s.idx[a.r * md.max_batch + row]];
      L = s.len[slot * md.M + a.r];
      pos = s.len[slot * md.M];  // every token runs loop 1: its length is the token count
    }
    int page = s.page_table[((size_t)slot * md.M + a.r) * md.max_pages + L / ps];
    if (page < 0 || page >= md.n_pages) {
      atomicOr(s.err, DEVERR_INDEX);
      page = -1;
    }
    ci_pos[t] = pos;
    ci_page[t] = page;
    ci_off[t] = L % ps;
    if (a.j == 0 && page >= 0) s.pos_table[(size_t)page * ps + L % ps] = pos;
  }
  __syncthreads();
  const int gfeat = m0 + tid;
  if (gfeat >= md.qkv_dim) return;
  const double two_pi = 6.283185307179586476925286766559;
  bf16* pool = reinterpret_cast<bf16*>(s.pool);
  if (gfeat < md.q_dim + md.kv_dim) {
    const bool is_q = gfeat < md.q_dim;
    const int fr = is_q ? gfeat : gfeat - md.q_dim;
    const int h = fr / hd, i = fr % hd;
    if (i >= half) return;  // the lower lane of the rotary pair handles both
    const double freq = a.inv_freq[i];
    for (int c = c0; c < c1; c += 4) {
      float x0[4], x1[4];
      cluster_sum4(pb, S, tid, c, c1, x0);
      cluster_sum4(pb, S, tid + half, c, c1, x1);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int cc = c + q;
        if (cc >= c1) break;
        double ang = (double)ci_pos[cc - c0] * freq;
        ang -= two_pi * rint(ang / two_pi);
        float sn, cs;
        sincosf((float)ang, &sn, &cs);
        const float r0 = x0[q] * cs - x1[q] * sn, r1 = x0[q] * sn + x1[q] * cs;
        if (is_q) {
          float* qo = a.Q + ((size_t)(tok0 + cc) * md.Hq + h) * hd;
          qo[i] = r0;
          qo[i + half] = r1;
        } else if (ci_page[cc - c0] >= 0) {
          bf16* kp = pool + (size_t)ci_page[cc - c0] * md.page_elems +
                     ((size_t)(a.j * 2 + 0) * md.Hkv + h) * ps * hd + (size_t)ci_off[cc - c0] * hd;
          kp[i] = __float2bfloat16_rn(r0);
          kp[i + half] = __float2bfloat16_rn(r1);
        }
      }
    }
  } else {
    const int fr = gfeat - md.q_dim - md.kv_dim;
    const int h = fr / hd, i = fr % hd;
    for (int c = c0; c < c1; c += 4) {
      float x[4];
      cluster_sum4(pb, S, tid, c, c1, x);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int cc = c + q;
        if (cc < c1 && ci_page[cc - c0] >= 0) {
          bf16* vp = pool + (size_t)ci_page[cc - c0] * md.page_elems +
                     ((size_t)(a.j * 2 + 1) * md.Hkv + h) * ps * hd + (size_t)ci_off[cc - c0] * hd;
          vp[i] = __float2bfloat16_rn(x[q]);
        }
      }
    }
  }
}

template <int NT>
__global__ void __launch_bounds__(128) k_gemm_tc(const __grid_constant__ CUtensorMap mapW,
                                                 const __grid_constant__ CUtensorMap mapX, GemmArgs a) {
  constexpr int A_BYTES = TC_BM * TC_BK * 2;
  constexpr int B_BYTES = NT * TC_BK * 2;
  constexpr uint32_t TMEM_COLS = NT < 32 ? 32 : NT;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + TC_STAGES * A_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sB + TC_STAGES * B_BYTES);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * TC_STAGES + 1);

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
    for (int i = 0; i < TC_STAGES; ++i) {
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
    const int pre = nk < TC_STAGES ? nk : TC_STAGES;
    for (int i = 0; i < pre; ++i) {
      mbar_arrive_expect_tx(full(i), A_BYTES + B_BYTES);
      tma_load_2d(smem_u32(sA + i * A_BYTES), &mapW, (kb0 + i) * TC_BK, m0, full(i));
    }
    pdl_wait();
    pdl_trigger();
    for (int i = 0; i < pre; ++i) tma_load_2d(smem_u32(sB + i * B_BYTES), &mapX, (kb0 + i) * TC_BK, tok0, full(i));
    for (int i = pre; i < nk; ++i) {
      const int st = i % TC_STAGES;
      const uint32_t ph = (uint32_t)(i / TC_STAGES) & 1u;
      if (!mbar_wait(empty(st), ph ^ 1u, a.err)) break;
      mbar_arrive_expect_tx(full(st), A_BYTES + B_BYTES);
      const int kx = (kb0 + i) * TC_BK;
      tma_load_2d(smem_u32(sA + st * A_BYTES), &mapW, kx, m0, full(st));
      tma_load_2d(smem_u32(sB + st * B_BYTES), &mapX, kx, tok0, full(st));
    }
  } else {
    pdl_wait();
    pdl_trigger();
  }
  if (nk > 0) {
    if (warp == 1 && lane == 0) {
      // MMA issuer
      const uint32_t idesc = idesc_bf16_f32(TC_BM, ncols);
      for (int i = 0; i < nk; ++i) {
        const int st = i % TC_STAGES;
        const uint32_t ph = (uint32_t)(i / TC_STAGES) & 1u;
        if (!mbar_wait(full(st), ph, a.err)) break;
        tc_fence_after();
        const uint64_t da = smem_desc_sw128(smem_u32(sA + st * A_BYTES));
        const uint64_t db = smem_desc_sw128(smem_u32(sB + st * B_BYTES));
#pragma unroll
        for (int k = 0; k < TC_BK / 16; ++k)  // +32 bytes per K step of 16 bf16 (encoded >> 4)
          tc_mma_f16(tmem, da + 2 * k, db + 2 * k, idesc, (i > 0 || k > 0) ? 1u : 0u);
        tc_commit(empty(st));
      }
      tc_commit(done);
    }
  }
  __syncwarp();

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
    int* colinfo = reinterpret_cast<int*>(red + 128 * NT);
    const int f = warp * 32 + lane;
    for (int c0 = 0; c0 < ncols; c0 += 16) {
      float v[16];
      if (ok && nk > 0) {
        tmem_ld_16(tmem + ((uint32_t)(warp * 32) << 16) + (uint32_t)c0, v);
      } else {
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] = 0.f;
      }
#pragma unroll
      for (int i = 0; i < 16; ++i) red[(c0 + i) * 128 + f] = v[i];
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tmem, TMEM_COLS);
    cluster_sync_all();  // every partner's tile is staged
    cluster_epilogue<NT>(a, red, colinfo, m0, n, tok0);
    __syncwarp();
    cluster_sync_all();  // partners have finished reading this CTA's tile
    return;
  }
  if (ok) {
    const int col = m0 + warp * 32 + lane;
    for (int c0 = 0; c0 < ncols; c0 += 16) {
      float v[16];
      if (nk > 0) {
        tmem_ld_16(tmem + ((uint32_t)(warp * 32) << 16) + (uint32_t)c0, v);
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

int gemm_tc_max_nt() { return 256; }

template <int NT>
static void launch_tc_nt(const CUtensorMap* mapW, const CUtensorMap* mapX, const GemmArgs& a, cudaStream_t st) {
  static bool attr_set = false;
  constexpr int smem = tc_smem_bytes<NT>();
  if (!attr_set) {
    cudaFuncSetAttribute(k_gemm_tc<NT>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    attr_set = true;
  }
  dim3 grid((a.N + TC_BM - 1) / TC_BM, a.splits, a.tok_tiles > 0 ? a.tok_tiles : 1);
  if (a.epi < EPI_CL_RESID) {
    launch_k(k_gemm_tc<NT>, grid, 128, smem, st, *mapW, *mapX, a);
    return;
  }
  // cluster epilogue: the splits of one tile form a (1, splits, 1) cluster
  static bool nonportable = false;
  if (a.splits > 8 && !nonportable) {
    cudaFuncSetAttribute(k_gemm_tc<NT>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    nonportable = true;
  }
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
  cudaLaunchKernelEx(&cfg, k_gemm_tc<NT>, *mapW, *mapX, a);
}

void launch_gemm_tc(const CUtensorMap* mapW, const CUtensorMap* mapX, int nt_max, const GemmArgs& a,
                    cudaStream_t st) {
  switch (nt_max) {
    case 16: launch_tc_nt<16>(mapW, mapX, a, st); break;
    case 32: launch_tc_nt<32>(mapW, mapX, a, st); break;
    case 64: launch_tc_nt<64>(mapW, mapX, a, st); break;
    case 128: launch_tc_nt<128>(mapW, mapX, a, st); break;
    default: launch_tc_nt<256>(mapW, mapX, a, st); break;
  }
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
