// Recursion-wise decode attention (T-LoopFormer Sec. 3.3, Eq. 10).
//
// The query of a token at loop r, layer j attends only to cache (r, j) of its
// sequence. That cache holds exactly the tokens that ran loop r (Eq. 11), in
// position order, so the validity mask mu^(r) of Eq. 10 is realised by
// storage and the kernel reads no masked slots. The token's own entry was
// appended before this kernel runs, so the key count is len + 1.
//
// Without recursion-wise caches (the dense-cache ablation, MASKED) every loop
// cache holds a slot per position and slots of tokens that exited earlier are
// masked (position -1): the kernel then also copies each page's positions and
// skips masked keys, reading the masked slots' K/V as the ablation requires.
//
// Work split (stream-K over pages): an item is one (token, kv head); its keys
// live in ceil((len+1)/64) pages. The plan kernel lays all items' pages out in
// one flat order; CTA c of the persistent grid takes the contiguous page range
// [c*per, (c+1)*per), so every CTA streams the same number of pages whatever
// the lengths, and streams them without draining its pipeline at item
// boundaries. A producer warp copies the K and V segments of each page (64
// keys of one kv head, contiguous and 16-byte aligned) into an NST-deep
// shared-memory ring with 1-D bulk TMA copies that complete on mbarriers. The
// copies carry an L2 evict-first hint: each page is read once per launch, and the
// hint keeps the step's small reused buffers resident in L2. The
// eight consumer warps split every page, release the stage on a per-stage
// mbarrier, and keep an online-softmax state (running max, sum, output slice)
// in float32 for the G query heads of the kv head (grouped-query attention),
// with LPK lanes sharing a key (16 bytes each) and xor-shuffle reductions.
// Scores are in base 2 (q pre-scaled by log2(e)/sqrt(hd)).
//
// When a CTA finishes its part of an item it merges its warps. An item that
// lies inside one CTA's range is written out directly. Otherwise each
// contributing CTA stores a partial (max, sum, output) and takes a ticket with
// an atomic counter, and the CTA that takes the last ticket merges the
// partials and writes the output (no CTA ever waits for another). On the
// tcgen05 decode path the output also gets its lo plane, bf16(o - bf16(o)): the
// output projection then takes a two-term operand.
#include <type_traits>

#include "tlf_internal.cuh"

namespace tlf {

constexpr int ATT_PS = 64;     // keys per page (the only page size the library accepts)
constexpr int ATT_WARPS = 8;   // consumer warps
constexpr int ATT_THREADS = 32 * (ATT_WARPS + 1);

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

// MASKED (the dense-cache ablation): each stage also holds the page's 64 positions, -1 = masked slot.
template <typename T, int HD, int G, bool MASKED>
constexpr int attn_smem_bytes() {
  using S = AttnShape<T, HD>;
  return 128 + S::NST * S::STAGE_BYTES + ATT_WARPS * G * (HD + 2) * 4 + (MASKED ? S::NST * ATT_PS * 4 : 0) +
         2 * S::NST * 8 + 16;
}

__device__ __forceinline__ void consumer_sync() {
  asm volatile("bar.sync 1, %0;" ::"n"(32 * ATT_WARPS) : "memory");
}

template <typename T, int HD, int G, bool MASKED>
__global__ void __launch_bounds__(ATT_THREADS) k_attn_decode(ModelDims md, StepDev s, int r, int j,
                                                             const float* __restrict__ Q, float* __restrict__ part,
                                                             T* __restrict__ O, int* __restrict__ cnt, bool o_lo) {
  using S = AttnShape<T, HD>;
  // output element (token k, query head hq, dim e); with o_lo also the lo plane of the
  // projection's two-term operand (bf16 of the rounding remainder, max_batch rows down)
  auto store_o = [&](int k, int hq, int e, float val) {
    const size_t at = (size_t)k * md.q_dim + (size_t)hq * HD + e;
    const T hi = from_f32<T>(val);
    O[at] = hi;
    if (o_lo) O[(size_t)md.max_batch * md.q_dim + at] = from_f32<T>(val - to_f32(hi));
  };
  constexpr int PSZ = G * (HD + 2);  // floats of one partial: per head, HD outputs then max and sum
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 127) & ~uintptr_t(127));
  uint8_t* ring = smem;                                                   // [NST][K seg | V seg]
  float* red = reinterpret_cast<float*>(ring + S::NST * S::STAGE_BYTES);  // [warps][G][HD + 2]
  int* mring = reinterpret_cast<int*>(red + ATT_WARPS * PSZ);              // [NST][64] positions (MASKED)
  uint64_t* full = reinterpret_cast<uint64_t*>(mring + (MASKED ? S::NST * ATT_PS : 0));
  uint64_t* empty = full + S::NST;
  int* flag = reinterpret_cast<int*>(empty + S::NST);
  volatile int* abort_flag = flag + 1;  // set when a bounded wait runs out: later waits are skipped

  pdl_wait();
  pdl_trigger();
  const int maxB = md.max_batch, M = md.M, Hkv = md.Hkv;
  const int n_r = s.n[r];
  const int* pbase = s.item_base + r * (maxB + 1);  // first flat page of each token's items
  const int* nkeys = s.nch + r * maxB;               // keys of each of the token's items (plan kernel)
  auto pages_of = [&](int kk) { return (nkeys[kk] + ATT_PS - 1) / ATT_PS; };
  const int total = (n_r > 0) ? pbase[n_r] : 0;
  const int per = (total + gridDim.x - 1) / gridDim.x;
  const int p0 = blockIdx.x * per;
  if (p0 >= total) return;
  const int p1 = min(total, p0 + per);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    for (int i = 0; i < S::NST; ++i) {
      mbar_init(smem_u32(&full[i]), 1);
      mbar_init(smem_u32(&empty[i]), ATT_WARPS);
    }
    *abort_flag = 0;
    fence_barrier_init();
  }
  __syncthreads();

  // (token, kv head, page) of flat page p: the largest k with pbase[k] <= p, found by the warp
  // with independent loads (32 entries of pbase a round) and a ballot
  auto locate = [&](int p, int& k, int& h, int& g) {
    int kk = 0;
    for (int b = 0; b < n_r; b += 32) {
      const int i = b + lane;
      const unsigned le = __ballot_sync(0xffffffffu, i < n_r && pbase[i] <= p);
      if (le) kk = b + 31 - __clz((int)le);
      if (le != 0xffffffffu) break;  // pbase is non-decreasing: no later entry is <= p
    }
    k = kk;
    const int off = p - pbase[k], np = pages_of(k);
    h = off / np;
    g = off % np;
  };

  if (warp == ATT_WARPS) {
    // ---------------- producer warp ----------------
    int k, h, g;
    locate(p0, k, h, g);  // the whole warp (ballot)
    if (lane == 0) {
      const uint64_t kv_policy = l2_policy_evict_first();  // pages are read once per launch
      int slot = s.slots[s.idx[r * maxB + k]];
      int L = nkeys[k];
      for (int p = p0; p < p1; ++p) {
        const int i = p - p0, st = i % S::NST;
        if (i >= S::NST && (*abort_flag || !mbar_wait(smem_u32(&empty[st]), ((i / S::NST) - 1) & 1, s.err))) {
          *abort_flag = 1;
          break;
        }
        const uint32_t bar = smem_u32(&full[st]);
        const int page = s.page_table[((size_t)slot * M + r) * md.max_pages + g];
        const int valid = min(ATT_PS, L - g * ATT_PS);
        if (page < 0 || page >= md.n_pages || valid <= 0) {
          atomicOr(s.err, DEVERR_INDEX);
          mbar_arrive(bar);  // complete the phase without data
        } else {
          const T* pg = reinterpret_cast<const T*>(s.pool) + (size_t)page * md.page_elems;
          const uint32_t bytes = (uint32_t)(valid * HD * sizeof(T));
          uint8_t* dst = ring + st * S::STAGE_BYTES;
          mbar_arrive_expect_tx(bar, 2 * bytes + (MASKED ? ATT_PS * 4 : 0));
          if (MASKED) bulk_g2s(smem_u32(mring + st * ATT_PS), s.pos_table + (size_t)page * ATT_PS, ATT_PS * 4, bar);
          bulk_g2s_hint(smem_u32(dst), pg + ((size_t)(j * 2 + 0) * Hkv + h) * ATT_PS * HD, bytes, bar, kv_policy);
          bulk_g2s_hint(smem_u32(dst + S::SEG_BYTES), pg + ((size_t)(j * 2 + 1) * Hkv + h) * ATT_PS * HD, bytes, bar,
                        kv_policy);
        }
        if (++g == pages_of(k)) {
          g = 0;
          if (++h == Hkv) {
            h = 0;
            do {
              ++k;
            } while (k < n_r && nkeys[k] == 0);  // rows with no keys have no pages (no gather)
            if (k < n_r) {
              slot = s.slots[s.idx[r * maxB + k]];
              L = nkeys[k];
            }
          }
        }
      }
    }
    return;
  }

  // ---------------- consumer warps ----------------
  const int grp = lane / S::LPK, part_lane = lane % S::LPK;
  const float scale = 1.4426950408889634f * rsqrtf((float)HD);
  int k, h, g;
  locate(p0, k, h, g);
  int L = 0;
  float q[G][S::VEC];
  float run_m[G], run_l[G], acc[G][S::VEC];
  auto begin_item = [&]() {
    L = nkeys[k];
    const float* qrow = Q + (size_t)k * md.Hq * HD;
#pragma unroll
    for (int gg = 0; gg < G; ++gg) {
#pragma unroll
      for (int e = 0; e < S::VEC; ++e) q[gg][e] = qrow[(h * G + gg) * HD + part_lane * S::VEC + e] * scale;
      run_m[gg] = -INFINITY;
      run_l[gg] = 0.f;
#pragma unroll
      for (int e = 0; e < S::VEC; ++e) acc[gg][e] = 0.f;
    }
  };
  begin_item();

  for (int p = p0; p < p1; ++p) {
    const int i = p - p0, st = i % S::NST;
    // a wait that runs out records the error word; the page is then computed on stale data
    if (!*abort_flag && !mbar_wait(smem_u32(&full[st]), (i / S::NST) & 1, s.err)) *abort_flag = 1;
    const int valid = min(ATT_PS, L - g * ATT_PS);
    const T* sk = reinterpret_cast<const T*>(ring + st * S::STAGE_BYTES);
    const T* sv = reinterpret_cast<const T*>(ring + st * S::STAGE_BYTES + S::SEG_BYTES);
    const int* smask = mring + st * ATT_PS;
    // key slot usable: inside the cache and, for a full-length cache, not masked (mu^(r) of Eq. 10)
    auto usable = [&](int key) { return key < valid && (!MASKED || smask[key] >= 0); };

    float sc[S::STEPS][G];
#pragma unroll
    for (int t = 0; t < S::STEPS; ++t) {
      const int key = warp * S::KEYS_PER_WARP + t * S::KPW + grp;
      float kv[S::VEC];
      const bool use = usable(key);
      if (use) {
        Vec16<T>::load(sk + key * HD + part_lane * S::VEC, kv);
      } else {
#pragma unroll
        for (int e = 0; e < S::VEC; ++e) kv[e] = 0.f;
      }
#pragma unroll
      for (int gg = 0; gg < G; ++gg) {
        float d = 0.f;
#pragma unroll
        for (int e = 0; e < S::VEC; ++e) d = fmaf(q[gg][e], kv[e], d);
#pragma unroll
        for (int o = S::LPK / 2; o > 0; o >>= 1) d += __shfl_xor_sync(0xffffffffu, d, o);
        sc[t][gg] = use ? d : -INFINITY;
      }
    }
#pragma unroll
    for (int gg = 0; gg < G; ++gg) {
      float pm = sc[0][gg];
#pragma unroll
      for (int t = 1; t < S::STEPS; ++t) pm = fmaxf(pm, sc[t][gg]);
#pragma unroll
      for (int o = S::LPK; o < 32; o <<= 1) pm = fmaxf(pm, __shfl_xor_sync(0xffffffffu, pm, o));
      if (pm > run_m[gg]) {
        const float cr = exp2f(run_m[gg] - pm);  // 0 when run_m was -inf
        run_l[gg] *= cr;
#pragma unroll
        for (int e = 0; e < S::VEC; ++e) acc[gg][e] *= cr;
        run_m[gg] = pm;
      }
    }
#pragma unroll
    for (int t = 0; t < S::STEPS; ++t) {
      const int key = warp * S::KEYS_PER_WARP + t * S::KPW + grp;
      if (usable(key)) {
        float vv[S::VEC];
        Vec16<T>::load(sv + key * HD + part_lane * S::VEC, vv);
#pragma unroll
        for (int gg = 0; gg < G; ++gg) {
          const float pr = exp2f(sc[t][gg] - run_m[gg]);
          run_l[gg] += pr;
#pragma unroll
          for (int e = 0; e < S::VEC; ++e) acc[gg][e] = fmaf(pr, vv[e], acc[gg][e]);
        }
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(smem_u32(&empty[st]));

    const bool item_end = (g + 1 == pages_of(k));
    if (item_end || p + 1 == p1) {
      // ---- this CTA's part of item (k, h) is done: merge the lane groups, then the warps ----
#pragma unroll
      for (int gg = 0; gg < G; ++gg) {
#pragma unroll
        for (int o = S::LPK; o < 32; o <<= 1) {
          run_l[gg] += __shfl_xor_sync(0xffffffffu, run_l[gg], o);
#pragma unroll
          for (int e = 0; e < S::VEC; ++e) acc[gg][e] += __shfl_xor_sync(0xffffffffu, acc[gg][e], o);
        }
      }
      if (grp == 0) {
#pragma unroll
        for (int gg = 0; gg < G; ++gg) {
          float* rw = red + (warp * G + gg) * (HD + 2);
#pragma unroll
          for (int e = 0; e < S::VEC; ++e) rw[part_lane * S::VEC + e] = acc[gg][e];
          if (part_lane == 0) {
            rw[HD] = run_m[gg];
            rw[HD + 1] = run_l[gg];
          }
        }
      }
      consumer_sync();
      const int np = pages_of(k);
      const int item = k * Hkv + h;
      const int first = pbase[k] + h * np;
      const int c_first = first / per, c_last = (first + np - 1) / per;
      float* my = part + (size_t)(item + blockIdx.x) * PSZ;
      const int nparts = c_last - c_first + 1;
      // merged state of this CTA's warps: thread t owns (head gg, dim e)
      for (int t = tid; t < G * HD; t += 32 * ATT_WARPS) {
        const int gg = t / HD, e = t % HD;
        float mx = -INFINITY;
#pragma unroll
        for (int w = 0; w < ATT_WARPS; ++w) mx = fmaxf(mx, red[(w * G + gg) * (HD + 2) + HD]);
        float o = 0.f, l = 0.f;
#pragma unroll
        for (int w = 0; w < ATT_WARPS; ++w) {
          const float* rw = red + (w * G + gg) * (HD + 2);
          const float f = (rw[HD] == -INFINITY) ? 0.f : exp2f(rw[HD] - mx);
          o = fmaf(f, rw[e], o);
          l = fmaf(f, rw[HD + 1], l);
        }
        if (nparts == 1) {
          store_o(k, h * G + gg, e, o / l);
        } else {
          my[gg * (HD + 2) + e] = o;
          if (e == 0) {
            my[gg * (HD + 2) + HD] = mx;
            my[gg * (HD + 2) + HD + 1] = l;
          }
        }
      }
      if (nparts > 1) {
        __threadfence();
        consumer_sync();
        if (tid == 0) {
          const int ticket = atomicAdd(cnt + item, 1);
          *flag = (ticket == nparts - 1);
        }
        consumer_sync();
        if (*flag) {
          // last contributor: merge the partials of CTAs c_first..c_last
          __threadfence();
          for (int t = tid; t < G * HD; t += 32 * ATT_WARPS) {
            const int gg = t / HD, e = t % HD;
            float mx = -INFINITY;
            for (int c = c_first; c <= c_last; ++c)
              mx = fmaxf(mx, __ldcg(part + (size_t)(item + c) * PSZ + gg * (HD + 2) + HD));
            float o = 0.f, l = 0.f;
            for (int c = c_first; c <= c_last; ++c) {
              const float* pp = part + (size_t)(item + c) * PSZ + gg * (HD + 2);
              const float f = exp2f(__ldcg(pp + HD) - mx);
              o = fmaf(f, __ldcg(pp + e), o);
              l = fmaf(f, __ldcg(pp + HD + 1), l);
            }
            store_o(k, h * G + gg, e, o / l);
          }
          if (tid == 0) cnt[item] = 0;  // ready for the next launch
        }
      }
      consumer_sync();  // `red` and `flag` are reused by the next item
      if (p + 1 < p1) {
        g = 0;
        if (++h == Hkv) {
          h = 0;
          do {
            ++k;
          } while (k < n_r && nkeys[k] == 0);
        }
        begin_item();
      }
    } else {
      ++g;
    }
  }
}

template <typename T, int HD, int G, bool MASKED>
static void attn_launch_v(const ModelDims& md, const StepDev& s, int r, int j, const float* Q, float* part, void* O,
                          int* cnt, int grid, cudaStream_t st, bool o_lo) {
  constexpr int smem = attn_smem_bytes<T, HD, G, MASKED>();
  (void)ensure_kernel_attrs((const void*)k_attn_decode<T, HD, G, MASKED>, smem);  // a failure shows at launch
  launch_k(k_attn_decode<T, HD, G, MASKED>, grid, ATT_THREADS, smem, st, md, s, r, j, Q, part, (T*)O, cnt, o_lo);
}

template <typename T, int HD, int G>
static void attn_launch(const ModelDims& md, const StepDev& s, int r, int j, const float* Q, float* part, void* O,
                        int* cnt, int grid, cudaStream_t st, bool o_lo) {
  o_lo = o_lo && std::is_same<T, bf16>::value;
  if constexpr (std::is_same<T, bf16>::value) {
    if (md.ablation == TLF_ABLATION_DENSE_CACHE) {
      attn_launch_v<T, HD, G, true>(md, s, r, j, Q, part, O, cnt, grid, st, o_lo);
      return;
    }
  }
  attn_launch_v<T, HD, G, false>(md, s, r, j, Q, part, O, cnt, grid, st, o_lo);
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

void launch_attn_decode(const ModelDims& md, const StepDev& s, int r, int j, const float* Q, float* part, void* O,
                        int* cnt, int grid, cudaStream_t st, bool o_lo) {
  TLF_ATTN_DISPATCH(attn_launch, md, s, r, j, Q, part, O, cnt, grid, st, o_lo);
}

// Resident CTAs: two per SM fit the ~104 KB ring of the largest head size.
int attn_decode_grid(const ModelDims& md, int num_sms) { return 2 * num_sms; }

// Floats of partial results one launch may write: one partial slot per (item + CTA) index.
size_t attn_partial_floats(const ModelDims& md, int grid) {
  const int G = md.Hq / md.Hkv;
  return ((size_t)md.max_batch * md.Hkv + grid) * G * (md.hd + 2);
}

}  // namespace tlf
