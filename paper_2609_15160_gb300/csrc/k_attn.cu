// Recursion-wise decode attention (T-LoopFormer Sec. 3.3, Eq. 10).
//
// The query of a token at loop r, layer j attends only to cache (r, j) of its
// sequence. That cache holds exactly the tokens that ran loop r (Eq. 11), in
// position order, so the validity mask mu^(r) of Eq. 10 is realised by
// storage and the kernel reads no masked slots. The token's own entry was
// appended before this kernel runs, so the key count is len + 1.
//
// Split-K flash decoding: the plan kernel cut every (token, kv head) key
// range into chunks of `chunk` keys; a persistent grid walks the flat list of
// (token, kv head, chunk) items. For an item, thread 0 streams the chunk's
// pages (64 keys each; K and V of one kv head are contiguous 16-byte-aligned
// segments of a page) into an NST-deep shared-memory ring with 1-D bulk TMA
// copies that complete on mbarriers. Eight warps split each page; within a
// warp, LPK lanes share a key (each lane holds 16 bytes of it), scores are
// reduced with xor shuffles, and every lane group keeps an online-softmax
// state (running max, sum, output slice) in float32 for the G query heads of
// the kv head (grouped-query attention). The CTA merges its warps and writes
// one (max, sum, output) partial per query head; k_attn_combine merges the
// chunks of a token. Scores are kept in base 2 (q is pre-scaled by
// log2(e)/sqrt(hd)).
#include "tlf_internal.cuh"

namespace tlf {

constexpr int ATT_PS = 64;     // keys per page (the only page size the library accepts)
constexpr int ATT_WARPS = 8;

template <typename T, int HD>
struct AttnShape {
  static constexpr int VEC = 16 / (int)sizeof(T);   // elements per lane per key
  static constexpr int LPK = HD / VEC;              // lanes per key
  static constexpr int KPW = 32 / LPK;              // keys per warp step
  static constexpr int KEYS_PER_WARP = ATT_PS / ATT_WARPS;
  static constexpr int STEPS = KEYS_PER_WARP / KPW;
  static constexpr int SEG_BYTES = ATT_PS * HD * (int)sizeof(T);       // one page of K (or V) of one head
  static constexpr int STAGE_BYTES = 2 * SEG_BYTES;
  static constexpr int NST = (98304 / STAGE_BYTES) < 2 ? 2 : ((98304 / STAGE_BYTES) > 8 ? 8 : (98304 / STAGE_BYTES));
  static_assert(LPK >= 1 && LPK <= 32 && (32 % LPK) == 0, "head_dim / vector width mismatch");
  static_assert(STEPS >= 1, "page too small for the warp split");
};

template <typename T, int HD, int G>
constexpr int attn_smem_bytes() {
  using S = AttnShape<T, HD>;
  return 128 + S::NST * S::STAGE_BYTES + ATT_WARPS * G * (HD + 2) * 4 + 16 * 8;
}

template <typename T, int HD, int G>
__global__ void __launch_bounds__(256) k_attn_decode(ModelDims md, StepDev s, int r, int j, const float* __restrict__ Q,
                                                     float* __restrict__ part_o, float* __restrict__ part_ml) {
  using S = AttnShape<T, HD>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 127) & ~uintptr_t(127));
  uint8_t* ring = smem;                                                   // [NST][K seg | V seg]
  float* red = reinterpret_cast<float*>(ring + S::NST * S::STAGE_BYTES);  // [warps][G][HD + 2]
  uint64_t* bars = reinterpret_cast<uint64_t*>(red + ATT_WARPS * G * (HD + 2));

  pdl_wait();
  pdl_trigger();
  const int n_r = s.n[r];
  const int items = s.item_base[r * (md.max_batch + 1) + n_r];
  if ((int)blockIdx.x >= items) return;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int grp = lane / S::LPK, part = lane % S::LPK;
  const int chunk = s.chunk[r];
  const int M = md.M, Hkv = md.Hkv;
  const float scale = 1.4426950408889634f * rsqrtf((float)HD);

  if (tid == 0) {
    for (int i = 0; i < S::NST; ++i) mbar_init(smem_u32(&bars[i]), 1);
    fence_barrier_init();
  }
  __syncthreads();

  uint32_t gp = 0;  // pages consumed by this CTA so far (ring position / phase)
  for (int item = blockIdx.x; item < items; item += gridDim.x) {
    // item -> (token k, kv head, chunk c)
    const int* base = s.item_base + r * (md.max_batch + 1);
    int lo = 0, hi = n_r;  // largest k with base[k] <= item
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (base[mid] <= item) lo = mid; else hi = mid;
    }
    const int k = lo;
    const int nc = s.nch[r * md.max_batch + k];
    const int local = item - base[k];
    const int kvh = local / nc, c = local % nc;
    const int b = s.idx[r * md.max_batch + k];
    const int slot = s.slots[b];
    const int L = s.len[slot * M + r] + 1;
    const int key0 = c * chunk;
    const int key1 = min(L, key0 + chunk);
    const int npages = (key1 - key0 + ATT_PS - 1) / ATT_PS;
    const int* ptab = s.page_table + ((size_t)slot * M + r) * md.max_pages;

    auto issue = [&](int pi) {
      const int kp = key0 + pi * ATT_PS;
      const int valid = min(ATT_PS, key1 - kp);
      const int page = ptab[kp / ATT_PS];
      const int st = (int)((gp + pi) % S::NST);
      const uint32_t bar = smem_u32(&bars[st]);
      if (page < 0 || page >= md.n_pages) {
        atomicOr(s.err, DEVERR_INDEX);
        mbar_arrive(bar);  // complete the phase without data
        return;
      }
      const T* pg = reinterpret_cast<const T*>(s.pool) + (size_t)page * md.page_elems;
      const T* kseg = pg + ((size_t)(j * 2 + 0) * Hkv + kvh) * ATT_PS * HD;
      const T* vseg = pg + ((size_t)(j * 2 + 1) * Hkv + kvh) * ATT_PS * HD;
      const uint32_t bytes = (uint32_t)(valid * HD * sizeof(T));
      uint8_t* dst = ring + st * S::STAGE_BYTES;
      mbar_arrive_expect_tx(bar, 2 * bytes);
      bulk_g2s(smem_u32(dst), kseg, bytes, bar);
      bulk_g2s(smem_u32(dst + S::SEG_BYTES), vseg, bytes, bar);
    };

    if (tid == 0) {
      const int pre = min(npages, S::NST);
      for (int pi = 0; pi < pre; ++pi) issue(pi);
    }

    // this lane's 16-byte slice of the G queries, pre-scaled to base 2
    float q[G][S::VEC];
    const float* qrow = Q + (size_t)k * md.Hq * HD;
#pragma unroll
    for (int g = 0; g < G; ++g)
#pragma unroll
      for (int e = 0; e < S::VEC; ++e) q[g][e] = qrow[(kvh * G + g) * HD + part * S::VEC + e] * scale;

    float run_m[G], run_l[G], acc[G][S::VEC];
#pragma unroll
    for (int g = 0; g < G; ++g) {
      run_m[g] = -INFINITY;
      run_l[g] = 0.f;
#pragma unroll
      for (int e = 0; e < S::VEC; ++e) acc[g][e] = 0.f;
    }

    for (int pi = 0; pi < npages; ++pi) {
      const int st = (int)((gp + pi) % S::NST);
      const uint32_t ph = ((gp + pi) / S::NST) & 1u;
      const bool ok = mbar_wait(smem_u32(&bars[st]), ph, s.err);
      const int valid = min(ATT_PS, key1 - (key0 + pi * ATT_PS));
      const T* sk = reinterpret_cast<const T*>(ring + st * S::STAGE_BYTES);
      const T* sv = reinterpret_cast<const T*>(ring + st * S::STAGE_BYTES + S::SEG_BYTES);

      // scores of this warp's keys of the page
      float sc[S::STEPS][G];
#pragma unroll
      for (int t = 0; t < S::STEPS; ++t) {
        const int key = warp * S::KEYS_PER_WARP + t * S::KPW + grp;
        float kv[S::VEC];
        if (key < valid) Vec16<T>::load(sk + key * HD + part * S::VEC, kv);
        else {
#pragma unroll
          for (int e = 0; e < S::VEC; ++e) kv[e] = 0.f;
        }
#pragma unroll
        for (int g = 0; g < G; ++g) {
          float d = 0.f;
#pragma unroll
          for (int e = 0; e < S::VEC; ++e) d = fmaf(q[g][e], kv[e], d);
#pragma unroll
          for (int o = S::LPK / 2; o > 0; o >>= 1) d += __shfl_xor_sync(0xffffffffu, d, o);
          sc[t][g] = (key < valid) ? d : -INFINITY;
        }
      }
      // running max over the warp (all lane groups)
#pragma unroll
      for (int g = 0; g < G; ++g) {
        float pm = sc[0][g];
#pragma unroll
        for (int t = 1; t < S::STEPS; ++t) pm = fmaxf(pm, sc[t][g]);
#pragma unroll
        for (int o = S::LPK; o < 32; o <<= 1) pm = fmaxf(pm, __shfl_xor_sync(0xffffffffu, pm, o));
        if (pm > run_m[g]) {
          const float cr = exp2f(run_m[g] - pm);  // 0 when run_m was -inf
          run_l[g] *= cr;
#pragma unroll
          for (int e = 0; e < S::VEC; ++e) acc[g][e] *= cr;
          run_m[g] = pm;
        }
      }
      // probabilities and P.V for this lane group's keys
#pragma unroll
      for (int t = 0; t < S::STEPS; ++t) {
        const int key = warp * S::KEYS_PER_WARP + t * S::KPW + grp;
        if (key < valid) {
          float vv[S::VEC];
          Vec16<T>::load(sv + key * HD + part * S::VEC, vv);
#pragma unroll
          for (int g = 0; g < G; ++g) {
            const float p = exp2f(sc[t][g] - run_m[g]);
            run_l[g] += p;
#pragma unroll
            for (int e = 0; e < S::VEC; ++e) acc[g][e] = fmaf(p, vv[e], acc[g][e]);
          }
        }
      }
      // every warp is done with stage st; a timed-out wait ends the CTA uniformly
      if (__syncthreads_or(!ok)) return;
      if (tid == 0 && pi + S::NST < npages) {
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        issue(pi + S::NST);
      }
    }
    gp += (uint32_t)npages;

    // merge the lane groups of the warp (same running max inside a warp)
#pragma unroll
    for (int g = 0; g < G; ++g) {
#pragma unroll
      for (int o = S::LPK; o < 32; o <<= 1) {
        run_l[g] += __shfl_xor_sync(0xffffffffu, run_l[g], o);
#pragma unroll
        for (int e = 0; e < S::VEC; ++e) acc[g][e] += __shfl_xor_sync(0xffffffffu, acc[g][e], o);
      }
    }
    if (grp == 0) {
#pragma unroll
      for (int g = 0; g < G; ++g) {
        float* rw = red + (warp * G + g) * (HD + 2);
#pragma unroll
        for (int e = 0; e < S::VEC; ++e) rw[part * S::VEC + e] = acc[g][e];
        if (part == 0) {
          rw[HD] = run_m[g];
          rw[HD + 1] = run_l[g];
        }
      }
    }
    __syncthreads();
    // merge the warps and write this chunk's partial
    for (int t = tid; t < G * HD; t += blockDim.x) {
      const int g = t / HD, e = t % HD;
      float mx = -INFINITY;
#pragma unroll
      for (int w = 0; w < ATT_WARPS; ++w) mx = fmaxf(mx, red[(w * G + g) * (HD + 2) + HD]);
      float o = 0.f, l = 0.f;
#pragma unroll
      for (int w = 0; w < ATT_WARPS; ++w) {
        const float* rw = red + (w * G + g) * (HD + 2);
        const float f = (rw[HD] == -INFINITY) ? 0.f : exp2f(rw[HD] - mx);
        o = fmaf(f, rw[e], o);
        l = fmaf(f, rw[HD + 1], l);
      }
      part_o[((size_t)item * G + g) * HD + e] = o;
      if (e == 0) {
        part_ml[((size_t)item * G + g) * 2 + 0] = mx;
        part_ml[((size_t)item * G + g) * 2 + 1] = l;
      }
    }
    __syncthreads();
  }
}

// One CTA per (token, query head): softmax-weighted merge of the chunk partials.
template <typename T, int HD, int G>
__global__ void __launch_bounds__(128) k_attn_combine(ModelDims md, StepDev s, int r, const float* __restrict__ part_o,
                                                      const float* __restrict__ part_ml, T* __restrict__ O) {
  pdl_wait();
  pdl_trigger();
  const int k = blockIdx.x, h = blockIdx.y;
  if (k >= s.n[r]) return;
  const int kvh = h / G, g = h % G;
  const int nc = s.nch[r * md.max_batch + k];
  const int first = s.item_base[r * (md.max_batch + 1) + k] + kvh * nc;
  float mx = -INFINITY;
  for (int c = 0; c < nc; ++c) mx = fmaxf(mx, part_ml[((size_t)(first + c) * G + g) * 2]);
  for (int e = threadIdx.x; e < HD; e += blockDim.x) {
    float o = 0.f, l = 0.f;
    for (int c = 0; c < nc; ++c) {
      const size_t it = (size_t)(first + c) * G + g;
      const float f = exp2f(part_ml[it * 2] - mx);
      o = fmaf(f, part_o[it * HD + e], o);
      l = fmaf(f, part_ml[it * 2 + 1], l);
    }
    O[(size_t)k * md.q_dim + h * HD + e] = from_f32<T>(o / l);
  }
}

template <typename T, int HD, int G>
static void attn_launch(const ModelDims& md, const StepDev& s, int r, int j, const float* Q, float* po, float* pml,
                        int grid, cudaStream_t st) {
  static bool attr = false;
  constexpr int smem = attn_smem_bytes<T, HD, G>();
  if (!attr) {
    cudaFuncSetAttribute(k_attn_decode<T, HD, G>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    attr = true;
  }
  launch_k(k_attn_decode<T, HD, G>, grid, 32 * ATT_WARPS, smem, st, md, s, r, j, Q, po, pml);
}

template <typename T, int HD, int G>
static void combine_launch(const ModelDims& md, const StepDev& s, int r, const float* po, const float* pml, void* O,
                           cudaStream_t st) {
  dim3 grid(md.max_batch, md.Hq);
  launch_k(k_attn_combine<T, HD, G>, grid, HD < 128 ? HD : 128, 0, st, md, s, r, po, pml, (T*)O);
}

#define TLF_ATTN_DISPATCH(FN, ...)                                                              \
  do {                                                                                          \
    const int G_ = md.Hq / md.Hkv;                                                              \
    if (md.dtype == 1) {                                                                        \
      if (md.hd == 128 && G_ == 1) FN<bf16, 128, 1>(__VA_ARGS__);                               \
      else if (md.hd == 128 && G_ == 2) FN<bf16, 128, 2>(__VA_ARGS__);                          \
      else if (md.hd == 128 && G_ == 4) FN<bf16, 128, 4>(__VA_ARGS__);                          \
      else if (md.hd == 64 && G_ == 1) FN<bf16, 64, 1>(__VA_ARGS__);                            \
      else if (md.hd == 64 && G_ == 2) FN<bf16, 64, 2>(__VA_ARGS__);                            \
      else if (md.hd == 64 && G_ == 4) FN<bf16, 64, 4>(__VA_ARGS__);                            \
      else if (md.hd == 32 && G_ == 1) FN<bf16, 32, 1>(__VA_ARGS__);                            \
      else FN<bf16, 32, 2>(__VA_ARGS__);                                                        \
    } else {                                                                                    \
      if (md.hd == 128 && G_ == 1) FN<float, 128, 1>(__VA_ARGS__);                              \
      else if (md.hd == 128 && G_ == 2) FN<float, 128, 2>(__VA_ARGS__);                         \
      else if (md.hd == 64 && G_ == 1) FN<float, 64, 1>(__VA_ARGS__);                           \
      else if (md.hd == 64 && G_ == 2) FN<float, 64, 2>(__VA_ARGS__);                           \
      else if (md.hd == 32 && G_ == 1) FN<float, 32, 1>(__VA_ARGS__);                           \
      else if (md.hd == 32 && G_ == 2) FN<float, 32, 2>(__VA_ARGS__);                           \
      else if (md.hd == 16 && G_ == 1) FN<float, 16, 1>(__VA_ARGS__);                           \
      else FN<float, 16, 2>(__VA_ARGS__);                                                       \
    }                                                                                           \
  } while (0)

void launch_attn_decode(const ModelDims& md, const StepDev& s, int r, int j, const float* Q, float* part_o,
                        float* part_ml, int grid, cudaStream_t st) {
  TLF_ATTN_DISPATCH(attn_launch, md, s, r, j, Q, part_o, part_ml, grid, st);
}

void launch_attn_combine(const ModelDims& md, const StepDev& s, int r, const float* part_o, const float* part_ml,
                         void* O, cudaStream_t st) {
  TLF_ATTN_DISPATCH(combine_launch, md, s, r, part_o, part_ml, O, st);
}

// Resident CTAs: two per SM fit the ~104 KB ring of the largest head size.
int attn_decode_grid(const ModelDims& md, int num_sms) { return 2 * num_sms; }

}  // namespace tlf
