// Predictor distillation step (section "Cross-Modal Attention Distillation"): the batch loss
// mean_b D_KL(p*_b || p_hat_b) of Eq. 3's prediction against the teacher distribution that
// QCTS selected, and its gradient with respect to every predictor weight (the backward pass
// through Eq. 3's softmax-mean, RoPE, the projections and both MLPs).
//
// Everything is fp32 (the bf16 features and weights are decoded exactly): the gradient is
// checked against a float64 oracle, and the training step is off the inference path.  The
// contractions run on one tiled SIMT GEMM with either operand transposed (64 x 64 tiles,
// 4 x 4 outputs per thread, fixed summation order); the softmax, KL, RoPE and GELU steps
// and their derivatives are elementwise or row/column reductions in their own kernels, with
// fixed-order (deterministic) reductions.
#include <cmath>
#include <cstdint>

#include "kernels.h"
#include "ptx.cuh"

namespace mapk {
namespace {

constexpr int kGT = 64, kGK = 16;

// C[i, j] = alpha sum_k A(i, k) B(k, j) (+ C[i, j] when accumulate), row-major storage:
// A(i, k) = TA ? A[k lda + i] : A[i lda + k];  B(k, j) = TB ? B[j ldb + k] : B[k ldb + j].
template <bool TA, bool TB>
__global__ void __launch_bounds__(256) sgemm_kernel(int M, int N, int K, float alpha, const float* __restrict__ A,
                                                    long long lda, const float* __restrict__ B, long long ldb,
                                                    int accumulate, float* __restrict__ C, long long ldc) {
  __shared__ __align__(16) float As[kGK][kGT + 4];
  __shared__ __align__(16) float Bs[kGK][kGT + 4];
  pdl_enter();
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  const int i0 = blockIdx.x * kGT, j0 = blockIdx.y * kGT;   // rows along x: up to 2^31 - 1 tiles
  float acc[4][4];
#pragma unroll
  for (int r = 0; r < 4; ++r)
#pragma unroll
    for (int c = 0; c < 4; ++c) acc[r][c] = 0.f;
  for (int k0 = 0; k0 < K; k0 += kGK) {
#pragma unroll
    for (int e = threadIdx.x; e < kGT * kGK; e += 256) {
      // consecutive threads walk the operand's contiguous dimension
      const int ii = TA ? e % kGT : e / kGK, kk = TA ? e / kGT : e % kGK;
      const int gi = i0 + ii, gk = k0 + kk;
      float v = 0.f;
      if (gi < M && gk < K) v = TA ? A[static_cast<long long>(gk) * lda + gi] : A[static_cast<long long>(gi) * lda + gk];
      As[kk][ii] = v;
    }
#pragma unroll
    for (int e = threadIdx.x; e < kGT * kGK; e += 256) {
      const int jj = TB ? e / kGK : e % kGT, kk = TB ? e % kGK : e / kGT;
      const int gj = j0 + jj, gk = k0 + kk;
      float v = 0.f;
      if (gj < N && gk < K) v = TB ? B[static_cast<long long>(gj) * ldb + gk] : B[static_cast<long long>(gk) * ldb + gj];
      Bs[kk][jj] = v;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < kGK; ++kk) {
      const float4 a = *reinterpret_cast<const float4*>(&As[kk][ty * 4]);
      const float4 b = *reinterpret_cast<const float4*>(&Bs[kk][tx * 4]);
      const float av[4] = {a.x, a.y, a.z, a.w}, bv[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
      for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[r][c] = fmaf(av[r], bv[c], acc[r][c]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int r = 0; r < 4; ++r) {
    const int i = i0 + ty * 4 + r;
    if (i >= M) continue;
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int j = j0 + tx * 4 + c;
      if (j >= N) continue;
      float* o = C + static_cast<long long>(i) * ldc + j;
      *o = accumulate ? *o + alpha * acc[r][c] : alpha * acc[r][c];
    }
  }
}

__global__ void bf16_to_f32_kernel(const uint16_t* __restrict__ x, long long n, float* __restrict__ y) {
  pdl_enter();
  for (long long i = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; i < n;
       i += static_cast<long long>(gridDim.x) * blockDim.x)
    y[i] = __uint_as_float(static_cast<uint32_t>(x[i]) << 16);
}

__device__ __forceinline__ float gelu_f(float x) { return 0.5f * x * (1.0f + erff(x * 0.70710678118654752f)); }
// d/dx [x Phi(x)] = Phi(x) + x phi(x)
__device__ __forceinline__ float gelu_grad_f(float x) {
  const float Phi = 0.5f * (1.0f + erff(x * 0.70710678118654752f));
  const float phi = 0.39894228040143268f * expf(-0.5f * x * x);
  return Phi + x * phi;
}

// z[r, c] += b[c]; h[r, c] = GELU(z[r, c])
__global__ void bias_gelu_kernel(float* __restrict__ z, const float* __restrict__ b, long long rows, int cols,
                                 float* __restrict__ h) {
  pdl_enter();
  const long long n = rows * cols;
  for (long long i = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; i < n;
       i += static_cast<long long>(gridDim.x) * blockDim.x) {
    const float v = z[i] + b[i % cols];
    z[i] = v;
    h[i] = gelu_f(v);
  }
}

__global__ void bias_add_kernel(float* __restrict__ x, const float* __restrict__ b, long long rows, int cols) {
  pdl_enter();
  const long long n = rows * cols;
  for (long long i = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; i < n;
       i += static_cast<long long>(gridDim.x) * blockDim.x)
    x[i] += b[i % cols];
}

// RoPE on rows of width 2*half (rotate-half pairs (i, i + half)): forward y = R(a) x, or
// backward x' = R(-a) y'.  Row r sits at position pos[r] (pos != nullptr) or r % pos_mod;
// the (cos, sin) table is [half][ld], position-minor.
template <bool BACKWARD>
__global__ void rope_kernel(const float* __restrict__ x, long long rows, int half, const float2* __restrict__ tab,
                            int ld, const int32_t* __restrict__ pos, int pos_mod, float* __restrict__ y) {
  pdl_enter();
  const long long n = rows * half;
  for (long long t = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; t < n;
       t += static_cast<long long>(gridDim.x) * blockDim.x) {
    const long long r = t / half;
    const int i = static_cast<int>(t - r * half);
    const int p = pos ? pos[r] : static_cast<int>(r % pos_mod);
    const float2 cs = tab[static_cast<long long>(i) * ld + p];
    const float x1 = x[r * 2 * half + i], x2 = x[r * 2 * half + half + i];
    if (BACKWARD) {
      y[r * 2 * half + i] = x1 * cs.x + x2 * cs.y;
      y[r * 2 * half + half + i] = x2 * cs.x - x1 * cs.y;
    } else {
      y[r * 2 * half + i] = x1 * cs.x - x2 * cs.y;
      y[r * 2 * half + half + i] = x2 * cs.x + x1 * cs.y;
    }
  }
}

constexpr int kRowThreads = 256;

// Deterministic block sum (kRowThreads threads): warp trees, then warp 0 in order.
__device__ __forceinline__ float block_sum(float v, float* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
  __syncthreads();
  if (threadIdx.x == 0) {
    float s = red[0];
    for (int w = 1; w < kRowThreads / 32; ++w) s += red[w];
    red[kRowThreads / 32] = s;
  }
  __syncthreads();
  const float r = red[kRowThreads / 32];
  __syncthreads();
  return r;
}
__device__ __forceinline__ float block_max(float v, float* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
  __syncthreads();
  if (threadIdx.x == 0) {
    float s = red[0];
    for (int w = 1; w < kRowThreads / 32; ++w) s = fmaxf(s, red[w]);
    red[kRowThreads / 32] = s;
  }
  __syncthreads();
  const float r = red[kRowThreads / 32];
  __syncthreads();
  return r;
}

// One CTA per question row: logits row -> softmax over the N visual tokens, in place.
__global__ void __launch_bounds__(kRowThreads) row_softmax_kernel(float* __restrict__ L, int N) {
  __shared__ float red[kRowThreads / 32 + 1];
  pdl_enter();
  float* row = L + static_cast<long long>(blockIdx.x) * N;
  float m = -INFINITY;
  for (int n = threadIdx.x; n < N; n += kRowThreads) m = fmaxf(m, row[n]);
  m = block_max(m, red);
  float s = 0.f;
  for (int n = threadIdx.x; n < N; n += kRowThreads) s += expf(row[n] - m);
  s = block_sum(s, red);
  const float inv = 1.0f / s;
  for (int n = threadIdx.x; n < N; n += kRowThreads) row[n] = expf(row[n] - m) * inv;
}

// Per image b (grid.y) and column block: p_hat[n] = mean_m s[m, n]; g[n] = -p*[n] / (B p_hat[n]);
// the block's share of D_KL(p* || p_hat) goes to part[b * nblk + blockIdx.x].
__global__ void __launch_bounds__(kRowThreads) phat_kl_kernel(const float* __restrict__ S, const int32_t* __restrict__ qoff,
                                                              const float* __restrict__ teacher, int N, int B,
                                                              float* __restrict__ p_hat, float* __restrict__ g,
                                                              float* __restrict__ part) {
  __shared__ float red[kRowThreads / 32 + 1];
  pdl_enter();
  const int b = blockIdx.y;
  const int n = blockIdx.x * kRowThreads + threadIdx.x;
  const int o = qoff[b], M = qoff[b + 1] - o;
  float kl = 0.f;
  if (n < N) {
    const float* col = S + static_cast<long long>(o) * N + n;
    float acc = 0.f;
    for (int m = 0; m < M; ++m) acc += col[static_cast<long long>(m) * N];
    const float ph = acc / static_cast<float>(M);
    const float ps = teacher[static_cast<long long>(b) * N + n];
    p_hat[static_cast<long long>(b) * N + n] = ph;
    g[static_cast<long long>(b) * N + n] = -ps / (static_cast<float>(B) * ph);
    if (ps > 0.f) kl = ps * logf(ps / ph);
  }
  kl = block_sum(kl, red);
  if (threadIdx.x == 0) part[static_cast<long long>(b) * gridDim.x + blockIdx.x] = kl;
}

// loss = (1/B) sum over images and blocks of the partial divergences, in order.
__global__ void loss_reduce_kernel(const float* __restrict__ part, int n, int B, float* __restrict__ loss) {
  pdl_enter();
  if (threadIdx.x == 0 && blockIdx.x == 0) {
    float s = 0.f;
    for (int i = 0; i < n; ++i) s += part[i];
    *loss = s / static_cast<float>(B);
  }
}

// One CTA per question row m of image b (row_img[m]): softmax backward of the mean,
//   dl[m, n] = s[m, n] (g[n] - sum_n' s[m, n'] g[n']) / M_b, written over s.
__global__ void __launch_bounds__(kRowThreads) softmax_back_kernel(float* __restrict__ S, const int32_t* __restrict__ qoff,
                                                                   const int32_t* __restrict__ row_img,
                                                                   const float* __restrict__ g, int N) {
  __shared__ float red[kRowThreads / 32 + 1];
  pdl_enter();
  const long long m = blockIdx.x;
  const int b = row_img[m];
  const float inv_m = 1.0f / static_cast<float>(qoff[b + 1] - qoff[b]);
  float* row = S + m * N;
  const float* gb = g + static_cast<long long>(b) * N;
  float c = 0.f;
  for (int n = threadIdx.x; n < N; n += kRowThreads) c += row[n] * gb[n];
  c = block_sum(c, red);
  for (int n = threadIdx.x; n < N; n += kRowThreads) row[n] = row[n] * (gb[n] - c) * inv_m;
}

__global__ void gelu_back_kernel(float* __restrict__ dh, const float* __restrict__ z, long long n) {
  pdl_enter();
  for (long long i = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; i < n;
       i += static_cast<long long>(gridDim.x) * blockDim.x)
    dh[i] *= gelu_grad_f(z[i]);
}

// out[c] = sum_r X[r, c]: 32 columns per block, 8 row partitions, combined in order.
__global__ void __launch_bounds__(256) colsum_kernel(const float* __restrict__ X, long long rows, int cols,
                                                     float* __restrict__ out) {
  __shared__ float red[8][32];
  pdl_enter();
  const int c = blockIdx.x * 32 + threadIdx.x, y = threadIdx.y;
  float s = 0.f;
  if (c < cols)
    for (long long r = y; r < rows; r += 8) s += X[r * cols + c];
  red[y][threadIdx.x] = s;
  __syncthreads();
  if (y == 0 && c < cols) {
    float t = red[0][threadIdx.x];
    for (int i = 1; i < 8; ++i) t += red[i][threadIdx.x];
    out[c] = t;
  }
}

unsigned grid_for(long long n) {
  const long long b = (n + 255) / 256;
  return static_cast<unsigned>(b < 152 * 16 ? (b > 0 ? b : 1) : 152 * 16);
}

}  // namespace

cudaError_t launch_sgemm(bool ta, bool tb, int M, int N, int K, float alpha, const float* A, long long lda,
                         const float* B, long long ldb, bool accumulate, float* C, long long ldc, cudaStream_t st) {
  if (M <= 0 || N <= 0) return cudaSuccess;
  const dim3 grid((M + kGT - 1) / kGT, (N + kGT - 1) / kGT);
  if (grid.y > 65535) return cudaErrorInvalidValue;
  const int acc = accumulate ? 1 : 0;
  if (!ta && !tb) return launch_k(sgemm_kernel<false, false>, grid, dim3(256), 0, st, M, N, K, alpha, A, lda, B, ldb, acc, C, ldc);
  if (!ta && tb) return launch_k(sgemm_kernel<false, true>, grid, dim3(256), 0, st, M, N, K, alpha, A, lda, B, ldb, acc, C, ldc);
  if (ta && !tb) return launch_k(sgemm_kernel<true, false>, grid, dim3(256), 0, st, M, N, K, alpha, A, lda, B, ldb, acc, C, ldc);
  return launch_k(sgemm_kernel<true, true>, grid, dim3(256), 0, st, M, N, K, alpha, A, lda, B, ldb, acc, C, ldc);
}

cudaError_t launch_bf16_to_f32(const void* x, long long n, float* y, cudaStream_t st) {
  return launch_k(bf16_to_f32_kernel, dim3(grid_for(n)), dim3(256), 0, st, static_cast<const uint16_t*>(x), n, y);
}

cudaError_t launch_bias_gelu(float* z, const float* b, long long rows, int cols, float* h, cudaStream_t st) {
  return launch_k(bias_gelu_kernel, dim3(grid_for(rows * cols)), dim3(256), 0, st, z, b, rows, cols, h);
}

cudaError_t launch_bias_add(float* x, const float* b, long long rows, int cols, cudaStream_t st) {
  return launch_k(bias_add_kernel, dim3(grid_for(rows * cols)), dim3(256), 0, st, x, b, rows, cols);
}

cudaError_t launch_rope_f32(bool backward, const float* x, long long rows, int d, const float2* tab, int ld,
                            const int32_t* pos, int pos_mod, float* y, cudaStream_t st) {
  const int half = d / 2;
  if (backward)
    return launch_k(rope_kernel<true>, dim3(grid_for(rows * half)), dim3(256), 0, st, x, rows, half, tab, ld, pos,
                    pos_mod, y);
  return launch_k(rope_kernel<false>, dim3(grid_for(rows * half)), dim3(256), 0, st, x, rows, half, tab, ld, pos,
                  pos_mod, y);
}

cudaError_t launch_distill_loss_grad(float* S, long long total_m, const int32_t* qoff, const int32_t* row_img,
                                     const float* teacher, int B, int N, float* p_hat, float* g, float* part,
                                     float* loss, cudaStream_t st) {
  cudaError_t e = launch_k(row_softmax_kernel, dim3(static_cast<unsigned>(total_m)), dim3(kRowThreads), 0, st, S, N);
  if (e != cudaSuccess) return e;
  const int nblk = (N + kRowThreads - 1) / kRowThreads;
  e = launch_k(phat_kl_kernel, dim3(nblk, B), dim3(kRowThreads), 0, st, static_cast<const float*>(S), qoff, teacher,
               N, B, p_hat, g, part);
  if (e != cudaSuccess) return e;
  e = launch_k(loss_reduce_kernel, dim3(1), dim3(32), 0, st, static_cast<const float*>(part), nblk * B, B, loss);
  if (e != cudaSuccess) return e;
  return launch_k(softmax_back_kernel, dim3(static_cast<unsigned>(total_m)), dim3(kRowThreads), 0, st, S, qoff,
                  row_img, static_cast<const float*>(g), N);
}

cudaError_t launch_gelu_back(float* dh, const float* z, long long n, cudaStream_t st) {
  return launch_k(gelu_back_kernel, dim3(grid_for(n)), dim3(256), 0, st, dh, z, n);
}

cudaError_t launch_colsum(const float* X, long long rows, int cols, float* out, cudaStream_t st) {
  return launch_k(colsum_kernel, dim3((cols + 31) / 32), dim3(32, 8), 0, st, X, rows, cols, out);
}

}  // namespace mapk
