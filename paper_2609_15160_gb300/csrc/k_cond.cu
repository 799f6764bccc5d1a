// Time/step conditioning table (T-LoopFormer Sec. 3.1, App. A), built once per context.
//
// A token of depth m runs loop i (1..m) conditioned on the cumulative time
// t = (i-1)/m and the step Delta = 1/m (the uniform trajectory of its length).
// Each scalar x becomes 256 sinusoidal features [cos(x w_k), sin(x w_k)],
// w_k = 10000^(-(k-1)/128), then passes through its own two-layer SiLU MLP;
// the two embeddings add into c, and layer j's modulator maps SiLU(c)
// linearly to (alpha_msa, alpha_mlp, gamma_msa, gamma_mlp). With M loops
// there are M(M+1)/2 (depth, loop) pairs, so the whole conditioning is a table
// [J][M(M+1)/2][4][d] that the step reads per token (see CondArgs). The table
// is computed in float64 from the float32 weights and stored in float32;
// every dot product is one warp striding over the weight row (coalesced).
#include "tlf_internal.cuh"

namespace tlf {

constexpr int COND_F = 256;  // sinusoidal features per scalar

__device__ __forceinline__ double warp_sum_d(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ double silu_d(double x) { return x / (1.0 + exp(-x)); }

// (depth m, loop i) of pair index p, pairs ordered depth-major: p = m(m-1)/2 + (i-1)
__device__ __forceinline__ void pair_of(int p, int& m, int& i) {
  m = 1;
  int base = 0;
  while (base + m <= p) {
    base += m;
    ++m;
  }
  i = p - base + 1;
}

// hidden[p][which][u] = SiLU(w1[u] . f(x) + b1[u]); which 0: x = t, 1: x = Delta
__global__ void __launch_bounds__(256) k_cond_hidden(int d, const float* __restrict__ t_w1, const float* __restrict__ t_b1,
                                                     const float* __restrict__ dt_w1, const float* __restrict__ dt_b1,
                                                     double* __restrict__ hidden) {
  __shared__ double f[COND_F];
  const int p = blockIdx.x, which = blockIdx.y;
  int m, i;
  pair_of(p, m, i);
  const double x = which == 0 ? (double)(i - 1) / m : 1.0 / m;
  for (int k = threadIdx.x; k < COND_F / 2; k += blockDim.x) {
    const double w = exp(-(double)k / (COND_F / 2) * log(10000.0));
    f[2 * k] = cos(x * w);
    f[2 * k + 1] = sin(x * w);
  }
  __syncthreads();
  const float* w1 = which == 0 ? t_w1 : dt_w1;
  const float* b1 = which == 0 ? t_b1 : dt_b1;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
  for (int u = blockIdx.z * nw + warp; u < d; u += gridDim.z * nw) {
    double acc = 0.0;
    for (int k = lane; k < COND_F; k += 32) acc += (double)w1[(size_t)u * COND_F + k] * f[k];
    acc = warp_sum_d(acc);
    if (lane == 0) hidden[((size_t)p * 2 + which) * d + u] = silu_d(acc + b1[u]);
  }
}

// act[p][e] = SiLU(c_e), c = w2_t hidden_t + b2_t + w2_dt hidden_dt + b2_dt
__global__ void __launch_bounds__(256) k_cond_embed(int d, const float* __restrict__ t_w2, const float* __restrict__ t_b2,
                                                    const float* __restrict__ dt_w2, const float* __restrict__ dt_b2,
                                                    const double* __restrict__ hidden, double* __restrict__ act) {
  const int p = blockIdx.x;
  const double* ht = hidden + (size_t)p * 2 * d;
  const double* hdt = ht + d;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
  for (int e = blockIdx.y * nw + warp; e < d; e += gridDim.y * nw) {
    double c = 0.0;
    for (int u = lane; u < d; u += 32)
      c += (double)t_w2[(size_t)e * d + u] * ht[u] + (double)dt_w2[(size_t)e * d + u] * hdt[u];
    c = warp_sum_d(c);
    if (lane == 0) act[(size_t)p * d + e] = silu_d(c + (double)t_b2[e] + (double)dt_b2[e]);
  }
}

// table[j][p][o] = mod_w[j][o] . act[p] + mod_b[j][o], o < 4d
__global__ void __launch_bounds__(256) k_cond_mod(int d, int P, const float* __restrict__ mod_w,
                                                  const float* __restrict__ mod_b, const double* __restrict__ act,
                                                  float* __restrict__ table) {
  const int j = blockIdx.x / P, p = blockIdx.x % P;
  const double* a = act + (size_t)p * d;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
  for (int o = blockIdx.y * nw + warp; o < 4 * d; o += gridDim.y * nw) {
    const float* wr = mod_w + ((size_t)j * 4 * d + o) * d;
    double v = 0.0;
    for (int e = lane; e < d; e += 32) v += (double)wr[e] * a[e];
    v = warp_sum_d(v);
    if (lane == 0) table[((size_t)j * P + p) * 4 * d + o] = (float)(v + (double)mod_b[(size_t)j * 4 * d + o]);
  }
}

int build_cond_table(const ModelDims& md, const float* t_w1, const float* t_b1, const float* t_w2, const float* t_b2,
                     const float* dt_w1, const float* dt_b1, const float* dt_w2, const float* dt_b2,
                     const float* mod_w, const float* mod_b, float* table, cudaStream_t st) {
  const int d = md.d, P = md.M * (md.M + 1) / 2;
  double *hidden = nullptr, *act = nullptr;
  cudaError_t e = cudaMalloc(&hidden, (size_t)P * 2 * d * sizeof(double));
  if (e == cudaSuccess) e = cudaMalloc(&act, (size_t)P * d * sizeof(double));
  if (e == cudaSuccess) {
    k_cond_hidden<<<dim3(P, 2, 16), 256, 0, st>>>(d, t_w1, t_b1, dt_w1, dt_b1, hidden);
    k_cond_embed<<<dim3(P, 32), 256, 0, st>>>(d, t_w2, t_b2, dt_w2, dt_b2, hidden, act);
    k_cond_mod<<<dim3(md.J * P, 64), 256, 0, st>>>(d, P, mod_w, mod_b, act, table);
    e = cudaGetLastError();
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  }
  if (hidden) cudaFree(hidden);
  if (act) cudaFree(act);
  return (int)e;
}

}  // namespace tlf
