// Predictor distillation step (section "Cross-Modal Attention Distillation"): the batch loss
// mean_b D_KL(p*_b || p_hat_b) of Eq. 3's prediction against the teacher distribution that
// QCTS selected, and its gradient with respect to every predictor weight (the backward pass
// through Eq. 3's softmax-mean, RoPE, the projections and both MLPs).
//
// Activations and gradients are fp32 (the bf16 features and weights are decoded exactly): the
// gradient is checked against a float64 oracle.  The contractions run on the tcgen05 GEMM of
// gemm_tc.cu with split-bf16 operands: an fp32 operand x is staged as three bf16 terms hi, mid,
// lo (x to about 24 significant bits), a bf16 feature or weight as itself, and the product is
// formed from every term pair above 2^-24 (six for two fp32 operands, three against an exact
// bf16 one, one for two bf16 ones), accumulated in fp32 in TMEM.  The staging kernels also
// transpose, so that both operands are K-major whichever index the
// contraction runs over (tokens for the weight gradients).  The softmax, KL, RoPE and GELU
// steps and their derivatives are elementwise or row/column reductions in their own kernels,
// with fixed-order (deterministic) reductions.
#include <algorithm>
#include <cmath>
#include <cstdint>

#include <cuda_bf16.h>

#include "kernels.h"
#include "ptx.cuh"

namespace mapk {
namespace {

// Operand staging for the tensor-core GEMM.  Element (r, c) of the logical matrix X (r < rows,
// c < cols; X(r, c) = src[c * ld + r] when TRANS, else src[r * ld + c]; times alpha) is split into
// three bf16 terms, hi = bf16(x), mid = bf16(x - hi), lo = bf16(x - hi - mid) (x = hi + mid + lo
// to about 24 significant bits; both differences are exact in fp32), and each term is written to
// row r of dst (row stride ldd elements) at column off + c for every offset of its list (up to
// three, -1 = unused).  Columns cols .. kpad - 1 (kpad a multiple of 64) of each segment are
// written as zeros.  32 x 64 tiles through shared memory, so that the reads (along the source's
// contiguous index) and the writes (along c, two columns per thread) are both coalesced.  BF16:
// the source holds bf16 bit patterns.
struct SplitOffsets {
  int hi[3], mid[3], lo[3];
};

template <bool TRANS, bool BF16>
__global__ void __launch_bounds__(256) split_operand_kernel(const void* __restrict__ src, long long ld, int rows,
                                                            int cols, int kpad, float alpha,
                                                            uint16_t* __restrict__ dst, long long ldd,
                                                            SplitOffsets o) {
  __shared__ float t[64][33];                        // t[c - c0][r - r0]: 64 columns x 32 rows
  pdl_enter();
  const int c0 = blockIdx.x * 64, r0 = blockIdx.y * 32;
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  auto load = [&](long long i) -> float {
    if constexpr (BF16) return __uint_as_float(static_cast<uint32_t>(static_cast<const uint16_t*>(src)[i]) << 16);
    else return static_cast<const float*>(src)[i];
  };
  if (TRANS) {                                       // consecutive threads: consecutive r
#pragma unroll
    for (int i = ty; i < 64; i += 8) {
      const int r = r0 + tx, c = c0 + i;
      t[i][tx] = (r < rows && c < cols) ? load(static_cast<long long>(c) * ld + r) : 0.f;
    }
  } else {                                           // consecutive threads: consecutive c
#pragma unroll
    for (int i = ty; i < 32; i += 8)
#pragma unroll
      for (int h = 0; h < 64; h += 32) {
        const int r = r0 + i, c = c0 + h + tx;
        t[h + tx][i] = (r < rows && c < cols) ? load(static_cast<long long>(r) * ld + c) : 0.f;
      }
  }
  __syncthreads();
  // each thread writes two adjacent columns (4-byte stores: 128 bytes per warp and segment)
  const int c = c0 + 2 * tx;                         // kpad is a multiple of 64: c + 1 < kpad
#pragma unroll
  for (int i = ty; i < 32; i += 8) {
    const int r = r0 + i;
    if (r >= rows || c >= kpad) continue;
    uint32_t hv = 0, mv = 0, lv = 0;
#pragma unroll
    for (int u = 0; u < 2; ++u) {
      const float x = t[2 * tx + u][i] * alpha;
      const __nv_bfloat16 h = __float2bfloat16_rn(x);
      const float r1 = x - __bfloat162float(h);
      const __nv_bfloat16 m = __float2bfloat16_rn(r1);
      const __nv_bfloat16 l = __float2bfloat16_rn(r1 - __bfloat162float(m));
      hv |= static_cast<uint32_t>(__bfloat16_as_ushort(h)) << (16 * u);
      mv |= static_cast<uint32_t>(__bfloat16_as_ushort(m)) << (16 * u);
      lv |= static_cast<uint32_t>(__bfloat16_as_ushort(l)) << (16 * u);
    }
    uint16_t* row = dst + static_cast<long long>(r) * ldd + c;
#pragma unroll
    for (int j = 0; j < 3; ++j) {
      if (o.hi[j] >= 0) *reinterpret_cast<uint32_t*>(row + o.hi[j]) = hv;
      if (o.mid[j] >= 0) *reinterpret_cast<uint32_t*>(row + o.mid[j]) = mv;
      if (o.lo[j] >= 0) *reinterpret_cast<uint32_t*>(row + o.lo[j]) = lv;
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
__global__ void __launch_bounds__(kRowThreads) row_softmax_kernel(float* __restrict__ L, long long ld, int N) {
  __shared__ float red[kRowThreads / 32 + 1];
  pdl_enter();
  float* row = L + static_cast<long long>(blockIdx.x) * ld;
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
__global__ void __launch_bounds__(kRowThreads) phat_kl_kernel(const float* __restrict__ S, long long ld,
                                                              const int32_t* __restrict__ qoff,
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
    const float* col = S + static_cast<long long>(o) * ld + n;
    float acc = 0.f;
    for (int m = 0; m < M; ++m) acc += col[static_cast<long long>(m) * ld];
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
__global__ void __launch_bounds__(kRowThreads) softmax_back_kernel(float* __restrict__ S, long long ld,
                                                                   const int32_t* __restrict__ qoff,
                                                                   const int32_t* __restrict__ row_img,
                                                                   const float* __restrict__ g, int N) {
  __shared__ float red[kRowThreads / 32 + 1];
  pdl_enter();
  const long long m = blockIdx.x;
  const int b = row_img[m];
  const float inv_m = 1.0f / static_cast<float>(qoff[b + 1] - qoff[b]);
  float* row = S + m * ld;
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

// Column sums in two fixed-order passes: block (x, p) sums rows [p rows / P, (p+1) rows / P) of
// 32 columns (8 row phases combined in order) into part[p, c]; then out[c] = sum_p part[p, c].
constexpr int kColParts = 64;
__global__ void __launch_bounds__(256) colsum_part_kernel(const float* __restrict__ X, long long rows, int cols,
                                                          float* __restrict__ part) {
  __shared__ float red[8][32];
  pdl_enter();
  const int c = blockIdx.x * 32 + threadIdx.x, y = threadIdx.y, pidx = blockIdx.y;
  const long long r0 = rows * pidx / kColParts, r1 = rows * (pidx + 1) / kColParts;
  float s = 0.f;
  if (c < cols)
    for (long long r = r0 + y; r < r1; r += 8) s += X[r * cols + c];
  red[y][threadIdx.x] = s;
  __syncthreads();
  if (y == 0 && c < cols) {
    float t = red[0][threadIdx.x];
    for (int i = 1; i < 8; ++i) t += red[i][threadIdx.x];
    part[static_cast<long long>(pidx) * cols + c] = t;
  }
}

__global__ void colsum_final_kernel(const float* __restrict__ part, int cols, float* __restrict__ out) {
  pdl_enter();
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= cols) return;
  float s = 0.f;
  for (int p = 0; p < kColParts; ++p) s += part[static_cast<long long>(p) * cols + c];
  out[c] = s;
}

// C[i, j] = sum over the ks K slices of part[s * stride + i * ldp + j], in slice order.
__global__ void sum_slices_kernel(const float* __restrict__ part, int ks, long long stride, int M, int N,
                                  long long ldp, float* __restrict__ C, long long ldc) {
  pdl_enter();
  const long long t = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (t >= static_cast<long long>(M) * N) return;
  const long long i = t / N, j = t - i * N;
  const float* p = part + i * ldp + j;
  float s = 0.f;
  for (int k = 0; k < ks; ++k) s += p[k * stride];
  C[i * ldc + j] = s;
}

unsigned grid_for(long long n) {
  const long long b = (n + 255) / 256;
  return static_cast<unsigned>(b < 152 * 16 ? (b > 0 ? b : 1) : 152 * 16);
}

}  // namespace

namespace {

// Terms of the product a.b kept for each kind of operand pair (x = hi + mid + lo for an fp32
// operand, exact for a bf16 one): everything down to about 2^-24 relative, so the result is as
// good as an fp32 product accumulated in fp32.
//   bf16 . bf16 : a.b                                           1 product
//   fp32 . bf16 : lo.b + mid.b + hi.b                           3 products
//   fp32 . fp32 : mm + hl + lh + hm + mh + hh                   6 products (ml, lm, ll are below 2^-24)
// The staged operands are the matching segments side by side along K, so one GEMM with
// K' = (number of products) * Kp forms the sum.
struct TcPlan {
  int Kp, n;                // padded K, number of products (GEMM K = n Kp)
  int ka, kb;               // staged widths of A and B (Kp when that operand's K wraps)
  SplitOffsets a, b;
};

SplitOffsets no_offsets() {
  SplitOffsets o;
  for (int j = 0; j < 3; ++j) o.hi[j] = o.mid[j] = o.lo[j] = -1;
  return o;
}

// Segments are ordered smallest term first, so that the tensor cores' fp32 accumulator adds the
// small terms while it is still small and runs only the last Kp / 16 steps at full magnitude
// (their additions are where the accumulation error comes from).  An exact operand facing a
// split one is staged once and read three times through the GEMM's K wrap.
TcPlan tc_plan(int K, float alpha, bool a_bf16, bool b_bf16) {
  TcPlan p;
  p.Kp = ((K + 63) / 64) * 64;
  const int Kp = p.Kp;
  const bool a_split = !(a_bf16 && alpha == 1.0f), b_split = !b_bf16;
  p.a = no_offsets();
  p.b = no_offsets();
  if (!a_split && !b_split) {                       // a . b
    p.n = 1; p.ka = p.kb = Kp;
    p.a.hi[0] = 0;
    p.b.hi[0] = 0;
  } else if (a_split && !b_split) {                 // [lo | mid | hi] . [b] (wrapped)
    p.n = 3; p.ka = 3 * Kp; p.kb = Kp;
    p.a.lo[0] = 0; p.a.mid[0] = Kp; p.a.hi[0] = 2 * Kp;
    p.b.hi[0] = 0;
  } else if (!a_split && b_split) {                 // [a] (wrapped) . [lo | mid | hi]
    p.n = 3; p.ka = Kp; p.kb = 3 * Kp;
    p.a.hi[0] = 0;
    p.b.lo[0] = 0; p.b.mid[0] = Kp; p.b.hi[0] = 2 * Kp;
  } else {                                          // [m h l h m h] . [m l h m h h]
    p.n = 6; p.ka = p.kb = 6 * Kp;
    p.a.mid[0] = 0; p.a.hi[0] = Kp; p.a.lo[0] = 2 * Kp; p.a.hi[1] = 3 * Kp; p.a.mid[1] = 4 * Kp; p.a.hi[2] = 5 * Kp;
    p.b.mid[0] = 0; p.b.lo[0] = Kp; p.b.hi[0] = 2 * Kp; p.b.mid[1] = 3 * Kp; p.b.hi[1] = 4 * Kp; p.b.hi[2] = 5 * Kp;
  }
  return p;
}

// K slices for a GEMM whose output has too few tiles to fill the GPU (the weight gradients over
// the token index, the per-image query gradients): enough slices to give every SM (or 2-SM
// pair) a unit, each slice at least 16 K blocks deep.  Mirrors launch_gemm's choice of the
// 1-SM tile for an output of at most 128 x 128 and of 2-SM 256 x 256 tiles otherwise.
int tc_ksplit(int M, int N, int kprime, int num_sms) {
  const bool pair = !(M <= 128 && N <= 128);
  const int units = pair ? ((M + 127) / 128 + 1) / 2 * ((N + 255) / 256) : ((M + 127) / 128) * ((N + 127) / 128);
  const int slots = pair ? num_sms / 2 : num_sms;
  const int kbs = kprime / 64;
  if (units <= 0 || units * 2 > slots) return 1;
  int ks = std::min(slots / units, kbs / 16);
  return ks < 1 ? 1 : ks;
}

cudaError_t stage(const void* src, bool bf16, bool trans, long long ld, int rows, int cols, int kpad, float alpha,
                  uint16_t* dst, long long ldd, const SplitOffsets& o, cudaStream_t st) {
  const dim3 grid(kpad / 64, (rows + 31) / 32);
  if (grid.y > 65535u) return cudaErrorInvalidValue;
  if (trans) {
    if (bf16) return launch_k(split_operand_kernel<true, true>, grid, dim3(256), 0, st, src, ld, rows, cols, kpad, alpha, dst, ldd, o);
    return launch_k(split_operand_kernel<true, false>, grid, dim3(256), 0, st, src, ld, rows, cols, kpad, alpha, dst, ldd, o);
  }
  if (bf16) return launch_k(split_operand_kernel<false, true>, grid, dim3(256), 0, st, src, ld, rows, cols, kpad, alpha, dst, ldd, o);
  return launch_k(split_operand_kernel<false, false>, grid, dim3(256), 0, st, src, ld, rows, cols, kpad, alpha, dst, ldd, o);
}

}  // namespace

void tc_matmul_ws(int M, int N, int K, float alpha, bool a_bf16, bool b_bf16, int num_sms, size_t* a_elems,
                  size_t* b_elems, size_t* c_elems) {
  const TcPlan p = tc_plan(K, alpha, a_bf16, b_bf16);
  *a_elems = static_cast<size_t>(M) * p.ka;
  *b_elems = static_cast<size_t>(N) * p.kb;
  const int ks = tc_ksplit(M, N, p.n * p.Kp, num_sms);
  *c_elems = ks > 1 ? static_cast<size_t>(ks) * M * ((N + 3) / 4 * 4) : 0;
}

cudaError_t launch_tc_matmul(bool ta, bool tb, int M, int N, int K, float alpha, const void* A, bool a_bf16,
                             long long lda, const void* B, bool b_bf16, long long ldb, float* C, long long ldc,
                             void* wsA, void* wsB, float* wsC, int num_sms, int* status, long long wait_ns,
                             cudaStream_t st, long long* launches) {
  if (M <= 0 || N <= 0 || K <= 0) return cudaSuccess;
  const TcPlan p = tc_plan(K, alpha, a_bf16, b_bf16);
  const int kprime = p.n * p.Kp;
  // A_s(i, k) = A(i, k): a transposed read when ta.  B_s(j, k) = B(k, j): transposed unless tb.
  // A bf16 operand that is already K-major, dense, unscaled and 64-aligned in K is its own staged
  // form (the features and weights of the forward pass): it is read in place.
  auto in_place = [&](const void* x, bool bf16, bool kmajor, long long ld, float scale, int width) {
    return bf16 && kmajor && scale == 1.0f && K == p.Kp && ld == K && width == p.Kp &&
           (reinterpret_cast<uintptr_t>(x) & 15) == 0;
  };
  const void* As = A;
  const void* Bs = B;
  cudaError_t e = cudaSuccess;
  if (!in_place(A, a_bf16, !ta, lda, alpha, p.ka)) {
    As = wsA;
    if (launches) ++*launches;
    if ((e = stage(A, a_bf16, ta, lda, M, K, p.Kp, alpha, static_cast<uint16_t*>(wsA), p.ka, p.a, st)) != cudaSuccess)
      return e;
  }
  if (!in_place(B, b_bf16, tb, ldb, 1.0f, p.kb)) {
    Bs = wsB;
    if (launches) ++*launches;
    if ((e = stage(B, b_bf16, !tb, ldb, N, K, p.Kp, 1.0f, static_cast<uint16_t*>(wsB), p.kb, p.b, st)) != cudaSuccess)
      return e;
  }
  GemmDesc d{};
  d.A = As; d.a_rows_total = M; d.a_row_stride = 0;
  d.B = Bs; d.b_rows_total = N; d.b_row_stride = 0;
  d.M = M; d.N = N; d.K = kprime; d.batch = 1;
  d.epi = EPI_F32; d.status = status; d.wait_ns = wait_ns;
  if (p.ka < kprime) d.a_kwrap = p.ka;
  if (p.kb < kprime) d.b_kwrap = p.kb;
  const int ks = tc_ksplit(M, N, kprime, num_sms);
  if (launches) ++*launches;
  if (ks == 1) {
    d.C = C; d.ldc = ldc; d.c_batch_stride = 0;
    return launch_gemm(d, num_sms, st);
  }
  // K slices into wsC, then their sum in a fixed order
  const long long ldp = (N + 3) / 4 * 4;
  d.C = wsC; d.ldc = ldp; d.c_batch_stride = 0;
  d.ksplit = ks; d.c_split_stride = static_cast<long long>(M) * ldp;
  if ((e = launch_gemm(d, num_sms, st)) != cudaSuccess) return e;
  const long long total = static_cast<long long>(M) * N;
  if (launches) ++*launches;
  return launch_k(sum_slices_kernel, dim3(static_cast<unsigned>((total + 255) / 256)), dim3(256), 0, st,
                  static_cast<const float*>(wsC), ks, d.c_split_stride, M, N, ldp, C, ldc);
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

cudaError_t launch_distill_loss_grad(float* S, long long ld, long long total_m, const int32_t* qoff,
                                     const int32_t* row_img, const float* teacher, int B, int N, float* p_hat,
                                     float* g, float* part, float* loss, cudaStream_t st) {
  cudaError_t e = launch_k(row_softmax_kernel, dim3(static_cast<unsigned>(total_m)), dim3(kRowThreads), 0, st, S, ld, N);
  if (e != cudaSuccess) return e;
  const int nblk = (N + kRowThreads - 1) / kRowThreads;
  e = launch_k(phat_kl_kernel, dim3(nblk, B), dim3(kRowThreads), 0, st, static_cast<const float*>(S), ld, qoff,
               teacher, N, B, p_hat, g, part);
  if (e != cudaSuccess) return e;
  e = launch_k(loss_reduce_kernel, dim3(1), dim3(32), 0, st, static_cast<const float*>(part), nblk * B, B, loss);
  if (e != cudaSuccess) return e;
  return launch_k(softmax_back_kernel, dim3(static_cast<unsigned>(total_m)), dim3(kRowThreads), 0, st, S, ld, qoff,
                  row_img, static_cast<const float*>(g), N);
}

cudaError_t launch_gelu_back(float* dh, const float* z, long long n, cudaStream_t st) {
  return launch_k(gelu_back_kernel, dim3(grid_for(n)), dim3(256), 0, st, dh, z, n);
}

cudaError_t launch_colsum(const float* X, long long rows, int cols, float* part, float* out, cudaStream_t st) {
  cudaError_t e = launch_k(colsum_part_kernel, dim3((cols + 31) / 32, kColParts), dim3(32, 8), 0, st, X, rows, cols,
                           part);
  if (e != cudaSuccess) return e;
  return launch_k(colsum_final_kernel, dim3((cols + 255) / 256), dim3(256), 0, st, static_cast<const float*>(part),
                  cols, out);
}

}  // namespace mapk
