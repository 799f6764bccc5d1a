// Row-wise kernels of the decode step.
//
// k_norm_rows    gather + RMSNorm: X[k] = RMSNorm(H[idx[k]]) * gain for the
//                rows of the active set (Eq. 6 followed by the pre-norm); with
//                time/step conditioning the gain is scaled by (1 + gamma). In
//                split mode it writes H * gain unscaled plus the per-tile sums
//                of squares, and the consuming GEMM applies the factor.
// k_rope_table   (cos, sin) of every position x rotary frequency, built once.
// k_rope_append  sums the split-K partials of the fused QKV projection (Eq. 9),
//                rotates q and k at the token's original position, keeps q for
//                the attention kernel and appends k, v to the token's slot of
//                the loop-r page of its sequence (Eq. 11; the slot is the
//                loop-r cache length, so positions stay in increasing order).
// k_swiglu       sums gate/up partials and applies silu(g) * u.
// k_final        final RMSNorm of every row for the LM head, and the cache
//                length update len[seq][r] += 1 for r < m.
// k_scatter_cache writes a restored cache snapshot into pages.
#include "tlf_internal.cuh"

namespace tlf {

__device__ __forceinline__ float block_sum(float v) {
  __shared__ float ws[32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  v = warp_sum(v);
  if (lane == 0) ws[warp] = v;
  __syncthreads();
  float t = (lane < nw) ? ws[lane] : 0.f;
  t = warp_sum(t);
  __syncthreads();
  return t;
}

template <typename T>
__global__ void __launch_bounds__(256) k_norm_rows(const float* __restrict__ H, int ldh, const int* __restrict__ idx,
                                                   const int* __restrict__ n_dev, int n_host,
                                                   const float* __restrict__ gain, int d, float eps,
                                                   T* __restrict__ X, int ldx, CondArgs cg,
                                                   float* __restrict__ ss_out, int ldss, T* __restrict__ X_lo) {
  pdl_wait();
  pdl_trigger();
  const int k = blockIdx.x;
  const int n = n_dev ? *n_dev : n_host;
  if (k >= n) return;
  const int src = idx ? idx[k] : k;
  // the row (d <= 8192, a multiple of 64) is read once into registers, 16 bytes per load
  const float4* h4 = reinterpret_cast<const float4*>(H + (size_t)src * ldh);
  const float4* g4 = reinterpret_cast<const float4*>(gain);
  const int d4 = d / 4;
  float4 v[8];
  float ss = 0.f;
#pragma unroll
  for (int c = 0; c < 8; ++c) {
    const int i = threadIdx.x + c * blockDim.x;
    float t = 0.f;
    if (i < d4) {
      v[c] = h4[i];
      t = v[c].x * v[c].x + v[c].y * v[c].y + v[c].z * v[c].z + v[c].w * v[c].w;
    }
    if (ss_out) {
      // split norm: warp w of pass c holds features [128 (8c + w), +128), one tile of the partial sums
      t = warp_sum(t);
      if ((threadIdx.x & 31) == 0 && 4 * (c * blockDim.x + (threadIdx.x & ~31)) < d)
        ss_out[(size_t)k * ldss + c * (blockDim.x >> 5) + (threadIdx.x >> 5)] = t;
    }
    ss += t;
  }
  // split norm: the operand is written unscaled and the consumer applies the factor
  const float inv = ss_out ? 1.f : rsqrtf(block_sum(ss) / (float)d + eps);
  T* xr = X + (size_t)k * ldx;
  // time/step conditioning: the gain is scaled by (1 + gamma) of the row's (depth, loop)
  const float4* c4 = cg.mod ? reinterpret_cast<const float4*>(cond_row(cg, src)) : nullptr;
#pragma unroll
  for (int c = 0; c < 8; ++c) {
    const int i = threadIdx.x + c * blockDim.x;
    if (i < d4) {
      float4 g = g4[i];
      if (c4) {
        const float4 y = c4[i];
        g = make_float4(g.x * (1.f + y.x), g.y * (1.f + y.y), g.z * (1.f + y.z), g.w * (1.f + y.w));
      }
      const float y[4] = {v[c].x * inv * g.x, v[c].y * inv * g.y, v[c].z * inv * g.z, v[c].w * inv * g.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const T hi = from_f32<T>(y[e]);
        xr[4 * i + e] = hi;
        if (X_lo) X_lo[(size_t)k * ldx + 4 * i + e] = from_f32<T>(y[e] - to_f32(hi));  // two-term operand
      }
    }
  }
}

void launch_norm_rows(int dtype, const float* H, int ldh, const int* idx, const int* n_dev, int n_host, int rows_max,
                      const float* gain, int d, float eps, void* X, int ldx, cudaStream_t st, const CondArgs& gamma,
                      float* ss_out, void* X_lo) {
  if (rows_max <= 0) return;
  if (dtype == 1)
    launch_k(k_norm_rows<bf16>, rows_max, 256, 0, st, H, ldh, idx, n_dev, n_host, gain, d, eps, (bf16*)X, ldx, gamma,
             ss_out, split_norm_ldss(d), (bf16*)X_lo);
  else
    launch_k(k_norm_rows<float>, rows_max, 256, 0, st, H, ldh, idx, n_dev, n_host, gain, d, eps, (float*)X, ldx,
             gamma, ss_out, split_norm_ldss(d), (float*)nullptr);
}

// Rotary table: table[p][i] = (cos, sin)(p * theta_i), the angle formed and
// reduced in float64 and rounded once to float32 (Eq. 11 positions, R4 reading).
__global__ void k_rope_table(int max_pos, int half, const double* __restrict__ inv_freq, float2* __restrict__ table) {
  const double two_pi = 6.283185307179586476925286766559;
  const size_t n = (size_t)max_pos * half;
  for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n; e += (size_t)gridDim.x * blockDim.x) {
    const int p = (int)(e / half), i = (int)(e % half);
    double ang = (double)p * inv_freq[i];
    ang -= two_pi * rint(ang / two_pi);
    double sn, cs;
    sincos(ang, &sn, &cs);
    table[e] = make_float2((float)cs, (float)sn);
  }
}

void launch_rope_table(const ModelDims& md, const double* inv_freq, float2* table, cudaStream_t st) {
  k_rope_table<<<1024, 256, 0, st>>>(md.max_pos, md.hd / 2, inv_freq, table);
}

template <typename T>
__global__ void __launch_bounds__(256) k_rope_append(ModelDims md, StepDev s, int r, int j,
                                                     const float* __restrict__ part, int splits, float* __restrict__ Q,
                                                     const float2* __restrict__ rope) {
  pdl_wait();
  pdl_trigger();
  const int k = blockIdx.x;
  if (k >= s.n[r]) return;
  const int hd2 = md.hd / 2;
  const int n_pairs = (md.Hq + md.Hkv) * hd2;   // rotated q and k pairs, then v elements
  const int t = blockIdx.y * blockDim.x + threadIdx.x;
  if (t >= n_pairs + md.Hkv * md.hd) return;
  // page, slot and position of the token's new loop-r entry, from the plan kernel
  const int4 ri = s.rowinfo[r * md.max_batch + k];
  const int page = ri.x, off = ri.y, pos = ri.z;  // page -1: q only (no append target)
  const int ps = md.page_size, hd = md.hd, half = hd / 2;
  T* pg = reinterpret_cast<T*>(s.pool) + (size_t)(page < 0 ? 0 : page) * md.page_elems;
  const size_t pstride = (size_t)md.max_batch * md.qkv_dim;
  const float* prow = part + (size_t)k * md.qkv_dim;

  if (t < n_pairs) {
    // q heads then k heads: rotate pair (i, i + hd/2) by pos * theta_i
    const int h = t / half, i = t % half;
    const int c0 = h * hd + i, c1 = c0 + half;  // k columns follow the q columns
    float a = 0.f, c = 0.f;
    for (int sp = 0; sp < splits; ++sp) {
      a += prow[sp * pstride + c0];
      c += prow[sp * pstride + c1];
    }
    const float2 csn = rope[(size_t)pos * half + i];
    const float ra = a * csn.x - c * csn.y, rc = a * csn.y + c * csn.x;
    if (h < md.Hq) {
      float* qo = Q + ((size_t)k * md.Hq + h) * hd;
      qo[i] = ra;
      qo[i + half] = rc;
    } else if (page >= 0) {
      T* kp = pg + ((size_t)(j * 2 + 0) * md.Hkv + (h - md.Hq)) * ps * hd + (size_t)off * hd;
      kp[i] = from_f32<T>(ra);
      kp[i + half] = from_f32<T>(rc);
    }
  } else if (page >= 0) {
    const int tv = t - n_pairs;
    const int h = tv / hd, e = tv % hd;
    const int col = md.q_dim + md.kv_dim + tv;
    float a = 0.f;
    for (int sp = 0; sp < splits; ++sp) a += prow[sp * pstride + col];
    T* vp = pg + ((size_t)(j * 2 + 1) * md.Hkv + h) * ps * hd + (size_t)off * hd;
    vp[e] = from_f32<T>(a);
  }
}

void launch_rope_append(const ModelDims& md, const StepDev& s, int r, int j, const float* part, int splits, float* Q,
                        const float2* rope, cudaStream_t st) {
  const int work = (md.Hq + md.Hkv) * (md.hd / 2) + md.Hkv * md.hd;
  dim3 grid(md.max_batch, (work + 127) / 128);
  if (md.dtype == 1)
    launch_k(k_rope_append<bf16>, grid, 128, 0, st, md, s, r, j, part, splits, Q, rope);
  else
    launch_k(k_rope_append<float>, grid, 128, 0, st, md, s, r, j, part, splits, Q, rope);
}

template <typename T>
__global__ void __launch_bounds__(256) k_swiglu(const float* __restrict__ part, int splits, int max_rows,
                                                const int* __restrict__ n_dev, int ff, T* __restrict__ U) {
  pdl_wait();
  pdl_trigger();
  const int k = blockIdx.y;
  if (k >= *n_dev) return;
  const size_t N = 2 * (size_t)ff;
  for (int f = blockIdx.x * blockDim.x + threadIdx.x; f < ff; f += gridDim.x * blockDim.x) {
    float g = 0.f, u = 0.f;
    for (int sp = 0; sp < splits; ++sp) {
      const float* p = part + ((size_t)sp * max_rows + k) * N;
      g += p[f];
      u += p[ff + f];
    }
    U[(size_t)k * ff + f] = from_f32<T>(g / (1.f + expf(-g)) * u);
  }
}

void launch_swiglu(int dtype, const float* part, int splits, int max_rows, const int* n_dev, int ff, void* U,
                   cudaStream_t st) {
  dim3 grid((ff + 255) / 256, max_rows);
  if (dtype == 1)
    launch_k(k_swiglu<bf16>, grid, 256, 0, st, part, splits, max_rows, n_dev, ff, (bf16*)U);
  else
    launch_k(k_swiglu<float>, grid, 256, 0, st, part, splits, max_rows, n_dev, ff, (float*)U);
}

template <typename T>
__global__ void __launch_bounds__(256) k_final(ModelDims md, StepDev s, const float* __restrict__ gain,
                                               T* __restrict__ Xf) {
  pdl_wait();
  pdl_trigger();
  const int b = blockIdx.x;
  // the row (d <= 8192, a multiple of 64) is read once into registers, 16 bytes per load
  const float4* h4 = reinterpret_cast<const float4*>(s.H + (size_t)b * md.d);
  const float4* g4 = reinterpret_cast<const float4*>(gain);
  const int d4 = md.d / 4;
  float4 v[8];
  float ss = 0.f;
#pragma unroll
  for (int c = 0; c < 8; ++c) {
    const int i = threadIdx.x + c * blockDim.x;
    if (i < d4) {
      v[c] = h4[i];
      ss += v[c].x * v[c].x + v[c].y * v[c].y + v[c].z * v[c].z + v[c].w * v[c].w;
    }
  }
  ss = block_sum(ss);
  const float inv = rsqrtf(ss / (float)md.d + md.eps);
  T* xr = Xf + (size_t)b * md.d;
#pragma unroll
  for (int c = 0; c < 8; ++c) {
    const int i = threadIdx.x + c * blockDim.x;
    if (i < d4) {
      const float4 g = g4[i];
      xr[4 * i + 0] = from_f32<T>(v[c].x * inv * g.x);
      xr[4 * i + 1] = from_f32<T>(v[c].y * inv * g.y);
      xr[4 * i + 2] = from_f32<T>(v[c].z * inv * g.z);
      xr[4 * i + 3] = from_f32<T>(v[c].w * inv * g.w);
    }
  }
  if (threadIdx.x < md.M) {
    // every loop cache the token wrote to grows by one (all of them without recursion-wise caches,
    // where the loops it skipped hold a masked slot)
    const int r = threadIdx.x;
    if (r < s.m[b] || md.ablation == TLF_ABLATION_DENSE_CACHE) s.len[s.slots[b] * md.M + r] += 1;
  }
}

void launch_final(const ModelDims& md, const StepDev& s, int B, const float* gain, void* Xf, cudaStream_t st) {
  if (md.dtype == 1)
    launch_k(k_final<bf16>, B, 256, 0, st, md, s, gain, (bf16*)Xf);
  else
    launch_k(k_final<float>, B, 256, 0, st, md, s, gain, (float*)Xf);
}

// Snapshot entries e < n of loop r: src layout [n][J][Hkv][hd] for k and v.
template <typename T>
__global__ void k_scatter_cache(ModelDims md, int slot, int r, int n, const T* __restrict__ k, const T* __restrict__ v,
                                const int* __restrict__ positions, const int* __restrict__ page_table, T* pool,
                                int* pos_table) {
  const int e = blockIdx.x;
  if (e >= n) return;
  const int ps = md.page_size, hd = md.hd;
  const int page = page_table[((size_t)slot * md.M + r) * md.max_pages + e / ps];
  if (page < 0 || page >= md.n_pages) return;
  const int off = e % ps;
  T* pg = pool + (size_t)page * md.page_elems;
  const int per = md.J * md.Hkv * hd;
  for (int t = threadIdx.x; t < per; t += blockDim.x) {
    const int jj = t / (md.Hkv * hd), rem = t % (md.Hkv * hd), h = rem / hd, i = rem % hd;
    pg[((size_t)(jj * 2 + 0) * md.Hkv + h) * ps * hd + (size_t)off * hd + i] = k[(size_t)e * per + t];
    pg[((size_t)(jj * 2 + 1) * md.Hkv + h) * ps * hd + (size_t)off * hd + i] = v[(size_t)e * per + t];
  }
  if (threadIdx.x == 0) pos_table[(size_t)page * ps + off] = positions[e];
}

// K/V of entries e < n of loop r filled with a counter-based pattern: value =
// (h(x) mod 256 - 128) / 64 for x the element's index in the pool, with h the
// 32-bit integer finaliser of MurmurHash3 (multiples of 1/64 in [-2, 2),
// exact in bf16). Used to restore long caches whose values do not matter.
__device__ __forceinline__ uint32_t fmix32(uint32_t h) {
  h ^= h >> 16;
  h *= 0x85ebca6bu;
  h ^= h >> 13;
  h *= 0xc2b2ae35u;
  h ^= h >> 16;
  return h;
}

template <typename T>
__global__ void k_fill_cache(ModelDims md, int slot, int r, int n, const int* __restrict__ positions,
                             const int* __restrict__ page_table, T* pool, int* pos_table) {
  const int e = blockIdx.x;
  if (e >= n) return;
  const int ps = md.page_size, hd = md.hd;
  const int page = page_table[((size_t)slot * md.M + r) * md.max_pages + e / ps];
  if (page < 0 || page >= md.n_pages) return;
  const int off = e % ps;
  T* pg = pool + (size_t)page * md.page_elems;
  const int per = md.J * md.Hkv * hd;
  for (int t = threadIdx.x; t < 2 * per; t += blockDim.x) {
    const int kv = t / per, rem = t % per;
    const int jj = rem / (md.Hkv * hd), rem2 = rem % (md.Hkv * hd), h = rem2 / hd, i = rem2 % hd;
    const size_t idx = ((size_t)(jj * 2 + kv) * md.Hkv + h) * ps * hd + (size_t)off * hd + i;
    const uint32_t x = fmix32((uint32_t)((size_t)page * md.page_elems + idx));
    pg[idx] = from_f32<T>((float)((int)(x & 255u) - 128) / 64.f);
  }
  if (threadIdx.x == 0) pos_table[(size_t)page * ps + off] = positions[e];
}

void launch_fill_cache(const ModelDims& md, int slot, int r, int n, const int* positions, const int* page_table,
                       void* pool, int* pos_table, cudaStream_t st) {
  if (n <= 0) return;
  if (md.dtype == 1)
    k_fill_cache<bf16><<<n, 256, 0, st>>>(md, slot, r, n, positions, page_table, (bf16*)pool, pos_table);
  else
    k_fill_cache<float><<<n, 256, 0, st>>>(md, slot, r, n, positions, page_table, (float*)pool, pos_table);
}

void launch_scatter_cache(const ModelDims& md, int slot, int r, int n, const void* k, const void* v,
                          const int* positions, const int* page_table, void* pool, int* pos_table, cudaStream_t st) {
  if (n <= 0) return;
  if (md.dtype == 1)
    k_scatter_cache<bf16><<<n, 256, 0, st>>>(md, slot, r, n, (const bf16*)k, (const bf16*)v, positions, page_table,
                                             (bf16*)pool, pos_table);
  else
    k_scatter_cache<float><<<n, 256, 0, st>>>(md, slot, r, n, (const float*)k, (const float*)v, positions,
                                              page_table, (float*)pool, pos_table);
}

}  // namespace tlf
