// Diversity-aware token selection, Eq. 4 (section "Inference-Time Token Pruning").
//
// The paper keeps an orthonormal basis B of the retained embeddings and picks
//   i_t = argmax_i p_hat_i * ||v_i - B B^T v_i||.
// Here B is never formed in D-space.  With G = V V^T, the coordinates of token i on the
// basis vectors are the rows of an incremental Cholesky factor:
//   e_beta[i] = (G[j_beta, i] - sum_{beta' < beta} e_beta'[j_beta] e_beta'[i]) / r_{j_beta},
//   r_i^2     = ||v_i||^2 - sum_beta e_beta[i]^2,
// where j_beta is the token that added basis vector beta and r_{j_beta} its residual at
// that time (the same quantities Gram-Schmidt would produce, in exact arithmetic).
//
// The greedy picks are sequential, but the Gram entries they need are dense products
// <v_i, v_j>, computed on the tensor cores in blocks.  Selection proceeds in rounds:
//   choose : active set A = the s candidates with the largest value bound U (a stale
//            value, or p_hat * ||v||^lambda for tokens never evaluated; values only shrink
//            as B grows, so U is always an upper bound); gather their rows and the rows of
//            new basis tokens into a compact buffer Vg.
//   gram   : G_blk = Vg[A] Vg[A u basis]^T on tcgen05 (gemm_tc.cu).
//   greedy : bring each A member's Cholesky coordinates up to date (exact values), then
//            pick while the best exact value in A beats the largest bound outside A (theta):
//            such a pick is the exact argmax over all candidates.  Each pick updates the
//            other A members.  Values are compared as the 64-bit key (value bits, ~index),
//            i.e. value descending, ties to the lower index.
// The first K0 picks (R0, top-K0 by p_hat) are forced, in p_hat order.  The result equals
// the eager fp32 greedy whatever s is; s only changes how much work is batched.
#include <algorithm>

#include "ptx.cuh"
#include "select.h"

namespace mapk {

namespace {

__device__ __forceinline__ uint64_t make_key(float v, int idx) {
  const float c = v > 0.f ? v : 0.f;            // values are >= 0: bit order = numeric order
  return (static_cast<uint64_t>(__float_as_uint(c)) << 32) | static_cast<uint64_t>(0xFFFFFFFFu - static_cast<uint32_t>(idx));
}
__device__ __forceinline__ int key_index(uint64_t key) {
  return static_cast<int>(0xFFFFFFFFu - static_cast<uint32_t>(key & 0xFFFFFFFFull));
}

__device__ __forceinline__ float sel_value(float p, float r2, float sq, float lam, float tau) {
  if (lam == 0.f) return p > 0.f ? p : 0.f;
  if (!(r2 > tau * sq) || !(r2 > 0.f)) return 0.f;
  const float v = lam == 1.f ? p * sqrtf(r2) : p * powf(r2, 0.5f * lam);
  return v > 0.f ? v : 0.f;
}

// k-th largest of n distinct keys in shared memory (1 <= k <= n), MSB-first radix select.
__device__ uint64_t block_kth_largest(const uint64_t* keys, int n, int k, uint32_t* hist, uint64_t* bc) {
  uint64_t prefix = 0, mask = 0;
  int want = k;
  for (int shift = 56; shift >= 0; shift -= 8) {
    for (int i = threadIdx.x; i < 256; i += blockDim.x) hist[i] = 0;
    __syncthreads();
    for (int i = threadIdx.x; i < n; i += blockDim.x) {
      const uint64_t key = keys[i];
      if ((key & mask) == prefix) atomicAdd(&hist[(key >> shift) & 255u], 1u);
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      int cum = 0, dsel = 0;
      for (int d = 255; d >= 0; --d) {
        const int h = static_cast<int>(hist[d]);
        if (cum + h >= want) { dsel = d; want -= cum; break; }
        cum += h;
      }
      bc[0] = static_cast<uint64_t>(dsel);
      bc[1] = static_cast<uint64_t>(want);
    }
    __syncthreads();
    prefix |= bc[0] << shift;
    mask |= 255ull << shift;
    want = static_cast<int>(bc[1]);
    __syncthreads();
  }
  return prefix;
}

// Sort n (<= cap, cap a power of two) keys descending in shared memory (bitonic).
__device__ void block_sort_desc(uint64_t* a, int n, int cap) {
  for (int i = n + threadIdx.x; i < cap; i += blockDim.x) a[i] = 0;
  __syncthreads();
  for (int size = 2; size <= cap; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = threadIdx.x; i < cap; i += blockDim.x) {
        const int j = i ^ stride;
        if (j > i) {
          const bool desc = (i & size) == 0;
          const uint64_t x = a[i], y = a[j];
          if (desc ? (x < y) : (x > y)) { a[i] = y; a[j] = x; }
        }
      }
      __syncthreads();
    }
  }
}

__device__ void block_sort_asc_i32(int32_t* a, int n, int cap) {
  for (int i = n + threadIdx.x; i < cap; i += blockDim.x) a[i] = 0x7FFFFFFF;
  __syncthreads();
  for (int size = 2; size <= cap; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = threadIdx.x; i < cap; i += blockDim.x) {
        const int j = i ^ stride;
        if (j > i) {
          const bool asc = (i & size) == 0;
          const int32_t x = a[i], y = a[j];
          if (asc ? (x > y) : (x < y)) { a[i] = y; a[j] = x; }
        }
      }
      __syncthreads();
    }
  }
}

__host__ __device__ inline int pow2_at_least(int n) {
  int c = 1;
  while (c < n) c <<= 1;
  return c;
}

// ------------------------------------------------------------------ init
// U = p_hat * ||v||^lambda, r2 = ||v||^2, nothing cached; R0 = top-K0 by p_hat in order.
__global__ void sel_init_kernel(SelState s) {
  extern __shared__ uint64_t sh64[];
  __shared__ uint32_t hist[256];
  __shared__ uint64_t bc[2];
  __shared__ int cnt;
  const int b = blockIdx.x;
  const long long base = static_cast<long long>(b) * s.N;
  for (int i = threadIdx.x; i < s.N; i += blockDim.x) {
    const float p = s.scores[base + i], sq = s.sqn[base + i];
    s.U[base + i] = sel_value(p, sq, sq, s.lambda, s.tau);
    s.r2[base + i] = sq;
    s.cstep[base + i] = 0;
    s.state[base + i] = 0;
    sh64[i] = make_key(p, i);
  }
  if (threadIdx.x == 0) {
    s.npicks[b] = 0; s.nbasis[b] = 0; s.nb_gathered[b] = 0; s.done[b] = 0; s.nlimit[b] = 0;
    cnt = 0;
  }
  __syncthreads();
  if (s.K0 > 0) {
    const uint64_t T = block_kth_largest(sh64, s.N, s.K0, hist, bc);
    uint64_t* sel = sh64 + s.N;
    for (int i = threadIdx.x; i < s.N; i += blockDim.x) {
      const uint64_t key = sh64[i];
      if (key >= T) sel[atomicAdd(&cnt, 1)] = key;
    }
    __syncthreads();
    block_sort_desc(sel, s.K0, pow2_at_least(s.K0));
    for (int i = threadIdx.x; i < s.K0; i += blockDim.x) s.r0[static_cast<long long>(b) * s.K + i] = key_index(sel[i]);
  }
}

// ------------------------------------------------------------------ choose
__global__ void sel_choose_kernel(SelState s) {
  extern __shared__ uint64_t sh64[];
  __shared__ uint32_t hist[256];
  __shared__ uint64_t bc[2];
  __shared__ int cnt, sh_mode, sh_na;
  __shared__ uint64_t sh_theta;
  const int b = blockIdx.x;
  const long long base = static_cast<long long>(b) * s.N;
  const int S = s.S, R = s.R;                // rows per image in Vg
  int32_t* aslot = s.aslot + static_cast<long long>(b) * S;
  if (s.done[b]) {
    if (threadIdx.x == 0) s.nlimit[b] = 0;
    return;
  }
  const int np = s.npicks[b], nb = s.nbasis[b];
  if (threadIdx.x == 0) cnt = 0;
  __syncthreads();
  if (np < s.K0) {
    // forced R0 chunk, in p_hat order
    const int na = min(S, s.K0 - np);
    for (int i = threadIdx.x; i < S; i += blockDim.x)
      aslot[i] = i < na ? s.r0[static_cast<long long>(b) * s.K + np + i] : -1;
    if (threadIdx.x == 0) { sh_mode = 1; sh_na = na; sh_theta = 0; }
  } else {
    int alive = 0;
    for (int i = threadIdx.x; i < s.N; i += blockDim.x) {
      const bool a = s.state[base + i] == 0;
      sh64[i] = a ? make_key(s.U[base + i], i) : 0ull;
      alive += a;
    }
    // count alive
    for (int o = 16; o > 0; o >>= 1) alive += __shfl_xor_sync(0xffffffffu, alive, o);
    if ((threadIdx.x & 31) == 0) atomicAdd(&cnt, alive);
    __syncthreads();
    const int n_alive = cnt;
    __syncthreads();
    if (threadIdx.x == 0) cnt = 0;
    __syncthreads();
    uint64_t T = 0;                            // keys > T form A; T = theta key (0: none outside)
    if (n_alive > S) T = block_kth_largest(sh64, s.N, S + 1, hist, bc);
    for (int i = threadIdx.x; i < s.N; i += blockDim.x) {
      const uint64_t key = sh64[i];
      if (key > T) aslot[atomicAdd(&cnt, 1)] = i;
    }
    __syncthreads();
    const int na = cnt;
    for (int i = na + threadIdx.x; i < S; i += blockDim.x) aslot[i] = -1;
    if (threadIdx.x == 0) { sh_mode = 0; sh_na = na; sh_theta = T; }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    s.mode[b] = sh_mode;
    s.theta[b] = sh_theta;
    s.nlimit[b] = S + nb;
  }
  // gather rows of A into Vg[b][0, S) and the new basis rows into Vg[b][S + nb_gathered, S + nb)
  const int vec = s.D / 8;
  const uint4* V = reinterpret_cast<const uint4*>(s.V) + base * vec;
  uint4* Vg = reinterpret_cast<uint4*>(s.Vg) + static_cast<long long>(b) * R * vec;
  const int na = sh_na;
  const int nbg = s.nb_gathered[b];
  const int rows = na + (nb - nbg);
  for (long long t = threadIdx.x; t < static_cast<long long>(rows) * vec; t += blockDim.x) {
    const int r = static_cast<int>(t / vec), c = static_cast<int>(t - static_cast<long long>(r) * vec);
    int src, dst;
    if (r < na) { src = aslot[r]; dst = r; }
    else { const int beta = nbg + (r - na); src = s.basis_tok[static_cast<long long>(b) * s.K + beta]; dst = S + beta; }
    Vg[static_cast<long long>(dst) * vec + c] = __ldg(V + static_cast<long long>(src) * vec + c);
  }
  __syncthreads();
  if (threadIdx.x == 0) s.nb_gathered[b] = nb;
}

// ------------------------------------------------------------------ greedy
// One CTA of S threads per image; thread = active slot.
__global__ void sel_greedy_kernel(SelState s) {
  __shared__ uint64_t wkey[32];
  __shared__ int sh_slot, sh_ext;
  __shared__ float sh_r2;
  const int b = blockIdx.x;
  if (s.done[b]) return;
  const int S = s.S, R = s.R;
  const long long base = static_cast<long long>(b) * s.N;
  const int slot = threadIdx.x;
  const int tok = s.aslot[static_cast<long long>(b) * S + slot];
  const float* Gr = s.G + (static_cast<long long>(b) * S + slot) * R;
  const int32_t* btok = s.basis_tok + static_cast<long long>(b) * s.K;
  const float* rnorm = s.rnorm + static_cast<long long>(b) * s.K;
  int nb = s.nbasis[b], np = s.npicks[b];
  const bool forced = s.mode[b] == 1;
  const uint64_t theta = s.theta[b];

  float* erow = tok >= 0 ? s.Ec + (base + tok) * s.K : nullptr;
  float r2 = 0.f, sq = 0.f, p = 0.f, val = 0.f;
  bool alive = false;
  if (tok >= 0) {
    r2 = s.r2[base + tok];
    sq = s.sqn[base + tok];
    p = s.scores[base + tok];
    alive = s.state[base + tok] == 0;
    // bring this token's coordinates up to date with the basis
    for (int beta = s.cstep[base + tok]; beta < nb; ++beta) {
      const float* L = s.Ec + (base + btok[beta]) * s.K;
      float acc = Gr[S + beta];
      for (int q = 0; q < beta; ++q) acc = fmaf(-L[q], erow[q], acc);
      const float e = acc / rnorm[beta];
      erow[beta] = e;
      r2 = fmaf(-e, e, r2);
    }
    val = sel_value(p, r2, sq, s.lambda, s.tau);
  }
  __syncthreads();

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nwarps = blockDim.x >> 5;
  for (int step = 0; np < s.K; ++step) {
    int jslot;
    if (forced) {
      jslot = step;
      if (jslot >= S) break;
      if (s.aslot[static_cast<long long>(b) * S + jslot] < 0) break;
    } else {
      uint64_t key = alive ? make_key(val, tok) : 0ull;
      for (int o = 16; o > 0; o >>= 1) {
        const uint64_t other = __shfl_xor_sync(0xffffffffu, key, o);
        key = other > key ? other : key;
      }
      if (lane == 0) wkey[warp] = key;
      __syncthreads();
      uint64_t best = 0;
      for (int w = 0; w < nwarps; ++w) best = wkey[w] > best ? wkey[w] : best;
      if (best == 0 || best <= theta) break;   // uniform: every thread computed the same best
      if (alive && make_key(val, tok) == best) sh_slot = slot;
      __syncthreads();
      jslot = sh_slot;
    }
    if (slot == jslot) {
      sh_r2 = r2;
      const int j = tok;
      sh_ext = (r2 > s.tau * sq) && (r2 > 0.f);
      s.state[base + j] = 1;
      s.picks[static_cast<long long>(b) * s.K + np] = j;
      alive = false;
      if (sh_ext) {
        s.basis_tok[static_cast<long long>(b) * s.K + nb] = j;
        s.rnorm[static_cast<long long>(b) * s.K + nb] = sqrtf(r2);
      }
    }
    __syncthreads();
    if (sh_ext) {
      const int jt = s.aslot[static_cast<long long>(b) * S + jslot];
      if (alive) {
        const float* L = s.Ec + (base + jt) * s.K;
        float acc = Gr[jslot];
        for (int q = 0; q < nb; ++q) acc = fmaf(-L[q], erow[q], acc);
        const float e = acc / sqrtf(sh_r2);
        erow[nb] = e;
        r2 = fmaf(-e, e, r2);
        val = sel_value(p, r2, sq, s.lambda, s.tau);
      }
      ++nb;
    }
    ++np;
    __syncthreads();
  }
  if (tok >= 0) {
    s.cstep[base + tok] = nb;
    s.r2[base + tok] = r2;
    s.U[base + tok] = val;
  }
  if (threadIdx.x == 0) {
    s.nbasis[b] = nb;
    s.npicks[b] = np;
    if (np >= s.K) { s.done[b] = 1; atomicAdd(s.done_count, 1); }
  }
}

// ------------------------------------------------------------------ outputs
// keep = picks sorted ascending; pick_order = picks.
__global__ void sel_finalize_kernel(const int32_t* picks, int K, int32_t* keep, int32_t* order) {
  extern __shared__ int32_t sh32[];
  const int b = blockIdx.x;
  const int32_t* p = picks + static_cast<long long>(b) * K;
  for (int i = threadIdx.x; i < K; i += blockDim.x) {
    sh32[i] = p[i];
    if (order) order[static_cast<long long>(b) * K + i] = p[i];
  }
  __syncthreads();
  block_sort_asc_i32(sh32, K, pow2_at_least(K));
  for (int i = threadIdx.x; i < K; i += blockDim.x) keep[static_cast<long long>(b) * K + i] = sh32[i];
}

// top-K by p_hat (lambda = 0 or K0 = K): R0 computed by sel_init is the whole answer.
__global__ void sel_copy_r0_kernel(const int32_t* r0, int K, int32_t* picks) {
  const int b = blockIdx.x;
  for (int i = threadIdx.x; i < K; i += blockDim.x)
    picks[static_cast<long long>(b) * K + i] = r0[static_cast<long long>(b) * K + i];
}

__global__ void sel_identity_kernel(int N, int32_t* keep, int32_t* order) {
  const int b = blockIdx.x;
  for (int i = threadIdx.x; i < N; i += blockDim.x) {
    keep[static_cast<long long>(b) * N + i] = i;
    if (order) order[static_cast<long long>(b) * N + i] = i;
  }
}

}  // namespace

size_t sel_init_smem(int N, int K0) { return (static_cast<size_t>(N) + pow2_at_least(std::max(K0, 1))) * 8; }
size_t sel_choose_smem(int N) { return static_cast<size_t>(N) * 8; }

cudaError_t launch_sel_init(const SelState& s, cudaStream_t st) {
  const size_t sm = sel_init_smem(s.N, s.K0);
  cudaError_t e = cudaFuncSetAttribute(sel_init_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(sm));
  if (e != cudaSuccess) return e;
  sel_init_kernel<<<s.B, 1024, sm, st>>>(s);
  return cudaGetLastError();
}

cudaError_t launch_sel_choose(const SelState& s, cudaStream_t st) {
  const size_t sm = sel_choose_smem(s.N);
  cudaError_t e = cudaFuncSetAttribute(sel_choose_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(sm));
  if (e != cudaSuccess) return e;
  sel_choose_kernel<<<s.B, 1024, sm, st>>>(s);
  return cudaGetLastError();
}

cudaError_t launch_sel_greedy(const SelState& s, cudaStream_t st) {
  sel_greedy_kernel<<<s.B, s.S, 0, st>>>(s);
  return cudaGetLastError();
}

cudaError_t launch_sel_finalize(const int32_t* picks, int B, int K, int32_t* keep, int32_t* order, cudaStream_t st) {
  const size_t sm = static_cast<size_t>(pow2_at_least(K)) * 4;
  sel_finalize_kernel<<<B, 1024, sm, st>>>(picks, K, keep, order);
  return cudaGetLastError();
}

cudaError_t launch_sel_copy_r0(const int32_t* r0, int B, int K, int32_t* picks, cudaStream_t st) {
  sel_copy_r0_kernel<<<B, 256, 0, st>>>(r0, K, picks);
  return cudaGetLastError();
}

cudaError_t launch_sel_identity(int B, int N, int32_t* keep, int32_t* order, cudaStream_t st) {
  sel_identity_kernel<<<B, 256, 0, st>>>(N, keep, order);
  return cudaGetLastError();
}

}  // namespace mapk
