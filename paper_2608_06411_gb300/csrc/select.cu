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
// <v_i, v_j>, computed on the tensor cores in blocks.
//   R0     : the first K0 picks (top-K0 by p_hat) are forced, in p_hat order; their basis is
//            the Cholesky factor of G[R0, R0] (sel_chol_kernel).  A tensor-core projection
//            of every token on that basis (gemm_tc.cu) then gives every candidate its exact
//            value.
// Later picks proceed in rounds:
//   choose : active set A = the s candidates with the largest value bound U (a stale
//            value, or p_hat * ||v||^lambda for tokens never evaluated; values only shrink
//            as B grows, so U is always an upper bound); gather their rows and the rows of
//            new basis tokens into a compact buffer Vg.
//   gram   : G_blk = Vg[A] Vg[A u new basis]^T on tcgen05 (gemm_tc.cu).
//   update : bring each A member's coordinates up to date (exact values).
//   resgram: replace G[A, A] by the Gram matrix of the residuals on the current basis, so
//            that the picks need only the coordinates added during the round.
//   greedy : pick while the best exact value in A beats the largest bound outside A (theta):
//            such a pick is the exact argmax over all candidates.  Each pick updates the
//            other A members.  Values are compared as the 64-bit key (value bits, ~index),
//            i.e. value descending, ties to the lower index; they are held squared
//            (p^2 rho^(2 lambda), same order, no square root).
// The result equals the eager fp32 greedy whatever s is; s only changes how much work is
// batched.
#include <algorithm>
#include <cstring>
#include <vector>

#include "kernels.h"
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

// The caller's buffers: through s.uptr when set (the cached loop graph was built for another
// call's pointers), else the fields themselves.
__device__ __forceinline__ const float* sel_scores(const SelState& s) {
  return s.uptr ? static_cast<const float*>(s.uptr[0]) : s.scores;
}
__device__ __forceinline__ const void* sel_features(const SelState& s) { return s.uptr ? s.uptr[1] : s.V; }

// Selection value, squared: p^2 * rho^(2 lambda) orders candidates like p * rho^lambda (both are
// >= 0) and needs no square root for lambda = 1.  rho^2 = r2 unless r2 <= tau ||v||^2 (then 0).
__device__ __forceinline__ float sel_value(float p, float r2, float sq, float lam, float tau) {
  if (!(p > 0.f)) return 0.f;
  if (lam == 0.f) return p * p;
  if (!(r2 > tau * sq) || !(r2 > 0.f)) return 0.f;
  const float v = lam == 1.f ? (p * p) * r2 : (p * p) * powf(r2, lam);
  return v > 0.f ? v : 0.f;
}

// k-th largest of n distinct 64-bit keys in shared memory (1 <= k <= n): MSB-first radix
// select, 8 bits per pass.  Lanes of a warp that hit the same bin add their count once
// (__match_any_sync), so bins shared by most keys (a common exponent) are not a
// serialisation point; one warp finds the bin with a shuffle scan.  As soon as the bin that
// holds the k-th key holds no other key, that key is the answer (usually after 2-3 passes).
// hist needs 256 entries, bc 4.
__device__ uint64_t block_kth_largest(const uint64_t* keys, int n, int k, uint32_t* hist, uint32_t* bc) {
  uint64_t prefix = 0, mask = 0;
  int want = k;
  const int lane = threadIdx.x & 31;
  for (int shift = 56; shift >= 0; shift -= 8) {
    for (int i = threadIdx.x; i < 256; i += blockDim.x) hist[i] = 0;
    __syncthreads();
    for (int i0 = 0; i0 < n; i0 += blockDim.x) {
      const int i = i0 + threadIdx.x;
      const bool in = i < n && (keys[i] & mask) == prefix;
      const uint32_t digit = in ? static_cast<uint32_t>((keys[i] >> shift) & 255u) : 256u;
      const unsigned active = __activemask();
      const unsigned peers = __match_any_sync(active, digit);
      if (in && lane == __ffs(peers) - 1) atomicAdd(&hist[digit], static_cast<uint32_t>(__popc(peers)));
    }
    __syncthreads();
    if (threadIdx.x < 32) {
      // lane l owns bins 255 - 8l .. 248 - 8l (descending); suffix counts from the top
      uint32_t c[8], tot = 0;
#pragma unroll
      for (int j = 0; j < 8; ++j) { c[j] = hist[255 - 8 * lane - j]; tot += c[j]; }
      uint32_t incl = tot;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t v = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += v;
      }
      uint32_t before = incl - tot;                 // keys in higher bins than this lane's
      const bool mine = before < static_cast<uint32_t>(want) && incl >= static_cast<uint32_t>(want);
      if (mine) {
        uint32_t cum = before;
        for (int j = 0; j < 8; ++j) {
          if (cum + c[j] >= static_cast<uint32_t>(want)) {
            bc[0] = 255 - 8 * lane - j;
            bc[1] = want - cum;
            bc[2] = c[j];                           // keys in that bin
            break;
          }
          cum += c[j];
        }
      }
    }
    __syncthreads();
    prefix |= static_cast<uint64_t>(bc[0]) << shift;
    mask |= 255ull << shift;
    want = static_cast<int>(bc[1]);
    if (bc[2] == 1u && shift > 0) {                 // uniform: the k-th key is the bin's only key
      __shared__ uint64_t found;
      for (int i = threadIdx.x; i < n; i += blockDim.x)
        if ((keys[i] & mask) == prefix) found = keys[i];
      __syncthreads();
      const uint64_t r = found;
      __syncthreads();
      return r;
    }
    __syncthreads();
  }
  return prefix;
}

// Sort `cap` (a power of two) keys descending in shared memory (bitonic network).
__device__ void block_sort_desc(uint64_t* a, int cap) {
  for (int size = 2; size <= cap; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = threadIdx.x; i < (cap >> 1); i += blockDim.x) {
        const int lo = (i / stride) * 2 * stride + (i % stride), hi = lo + stride;
        const bool desc = (lo & size) == 0;
        const uint64_t x = a[lo], y = a[hi];
        if (desc ? (x < y) : (x > y)) { a[lo] = y; a[hi] = x; }
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
      for (int i = threadIdx.x; i < (cap >> 1); i += blockDim.x) {
        const int lo = (i / stride) * 2 * stride + (i % stride), hi = lo + stride;
        const bool asc = (lo & size) == 0;
        const int32_t x = a[lo], y = a[hi];
        if (asc ? (x > y) : (x < y)) { a[lo] = y; a[hi] = x; }
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
// U = (p_hat * ||v||^lambda)^2, r2 = ||v||^2, nothing cached; R0 = top-K0 by p_hat, in order.
__global__ void __launch_bounds__(1024) sel_init_kernel(SelState s) {
  pdl_enter();
  extern __shared__ uint64_t sh64[];
  const int b = blockIdx.x;
  const long long base = static_cast<long long>(b) * s.N;
  __shared__ uint32_t hist[256], bc[4];
  __shared__ int cnt;
  const int nv = s.nvalid ? s.nvalid[b] : s.N;
  for (int i = threadIdx.x; i < s.N; i += blockDim.x) {
    if (i >= nv) {                       // padding: never a candidate, key below every token's
      s.U[base + i] = 0.f;
      s.r2[base + i] = 0.f;
      s.cstep[base + i] = 0;
      s.state[base + i] = 2;
      sh64[i] = 0ull;
      continue;
    }
    const float p = s.scores[base + i], sq = s.sqn ? s.sqn[base + i] : 0.f;
    s.U[base + i] = sel_value(p, sq, sq, s.lambda, s.tau);
    s.r2[base + i] = sq;
    s.cstep[base + i] = 0;
    s.state[base + i] = 0;
    sh64[i] = make_key(p, i);
  }
  if (b == 0 && threadIdx.x == 0) {   // counters of this selection (earlier readers have completed)
    if (s.bcount) { s.bcount[0] = 0; s.bcount[1] = 0; }
    if (s.done_count) *s.done_count = 0;
    if (s.uptr) { s.uptr[0] = s.scores; s.uptr[1] = s.V; }
  }
  if (threadIdx.x == 0) {
    s.npicks[b] = 0; s.nbasis[b] = 0; s.nb_gathered[b] = 0; s.done[b] = 0; s.nlimit[b] = 0;
    s.gb_lo[b] = 0; s.gb_hi[b] = 0; s.gbase[b] = 0;
    cnt = 0;
  }
  __syncthreads();
  if (s.K0 > 0) {
    const uint64_t T = block_kth_largest(sh64, s.N, s.K0, hist, bc);
    uint64_t* sel = sh64 + s.N;
    const int cap = pow2_at_least(s.K0);
    for (int i = threadIdx.x; i < s.N; i += blockDim.x)
      if (sh64[i] >= T) sel[atomicAdd(&cnt, 1)] = sh64[i];
    if (s.K0 <= static_cast<int>(blockDim.x)) {
      // The keys are distinct (each holds its token index), so a key's place in descending
      // order is the number of larger keys: one pass, no sorting network.
      __syncthreads();
      if (static_cast<int>(threadIdx.x) < s.K0) {
        const uint64_t x = sel[threadIdx.x];
        int rank = 0;
        for (int j = 0; j < s.K0; ++j) rank += sel[j] > x ? 1 : 0;
        s.r0[static_cast<long long>(b) * s.K + rank] = key_index(x);
      }
    } else {
      for (int i = s.K0 + threadIdx.x; i < cap; i += blockDim.x) sel[i] = 0ull;
      __syncthreads();
      block_sort_desc(sel, cap);
      for (int i = threadIdx.x; i < s.K0; i += blockDim.x) s.r0[static_cast<long long>(b) * s.K + i] = key_index(sel[i]);
    }
  }
}

// ------------------------------------------------------------------ choose
// Active set of the next round: the next R0 chunk (forced), else the S candidates with the
// largest bound U (value descending, ties to the lower index) and theta = the next key.
__global__ void __launch_bounds__(1024) sel_choose_kernel(SelState s) {
  pdl_enter();
  extern __shared__ uint64_t sh64[];
  const int b = blockIdx.x;
  const long long base = static_cast<long long>(b) * s.N;
  const int S = s.S;
  int32_t* aslot = s.aslot + static_cast<long long>(b) * S;
  if (s.blist && b == 0 && threadIdx.x == 0) s.bcount[s.bc_par ^ 1] = 0;
  if (s.done[b]) {
    if (threadIdx.x == 0) s.nlimit[b] = 0;
    return;
  }
  if (s.blist && threadIdx.x == 0) s.blist[atomicAdd(s.bcount + s.bc_par, 1)] = b;
  const int np = s.npicks[b], nb = s.nbasis[b];
  uint64_t theta = 0;
  int mode;
  if (np < s.K0) {
    const int na = min(S, s.K0 - np);
    for (int i = threadIdx.x; i < S; i += blockDim.x)
      aslot[i] = i < na ? s.r0[static_cast<long long>(b) * s.K + np + i] : -1;
    mode = 1;
  } else {
    __shared__ uint32_t hist[256], bc[4];
    __shared__ int cnt, n_alive;
    if (threadIdx.x == 0) { cnt = 0; n_alive = 0; }
    __syncthreads();
    int alive = 0;
    for (int i = threadIdx.x; i < s.N; i += blockDim.x) {
      const bool a = s.state[base + i] == 0;
      sh64[i] = a ? make_key(s.U[base + i], i) : 0ull;
      alive += a;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) alive += __shfl_xor_sync(0xffffffffu, alive, o);
    if ((threadIdx.x & 31) == 0 && alive) atomicAdd(&n_alive, alive);
    __syncthreads();
    // keys > theta form A; theta = the (S+1)-th largest key (0: nothing outside A)
    if (n_alive > S) theta = block_kth_largest(sh64, s.N, S + 1, hist, bc);
    for (int i = threadIdx.x; i < s.N; i += blockDim.x)
      if (sh64[i] > theta) aslot[atomicAdd(&cnt, 1)] = i;
    __syncthreads();
    for (int i = cnt + threadIdx.x; i < S; i += blockDim.x) aslot[i] = -1;
    mode = 0;
  }
  if (threadIdx.x == 0) {
    s.mode[b] = mode;
    s.theta[b] = theta;
    s.nlimit[b] = (mode == 1 && nb == s.gbase[b]) ? min(S, s.K0 - np) : S + nb - s.gbase[b];
    s.gb_lo[b] = s.nb_gathered[b];
    s.gb_hi[b] = nb;
    s.nb_gathered[b] = nb;
  }
}

// Copies the rows the Gram block needs into Vg: row r < S <- token aslot[r];
// row S + beta - gbase <- basis token beta for the basis vectors added since the last round.
// kGatherCtas CTAs per image, each walking every kGatherCtas-th row; finished images exit.
constexpr int kGatherCtas = 64;
constexpr int kGatherThreads = 128;

__global__ void __launch_bounds__(kGatherThreads) sel_gather_kernel(SelState s) {
  pdl_enter();
  const int b = blockIdx.y;
  if (s.done[b]) return;
  const int gb = s.gbase[b], lo = s.gb_lo[b], hi = s.gb_hi[b];
  const int vec = s.D / 8;
  for (int r = blockIdx.x; r < s.S + (hi - gb); r += kGatherCtas) {
    int src = -1;
    if (r < s.S) {
      src = s.aslot[static_cast<long long>(b) * s.S + r];
    } else {
      const int beta = r - s.S + gb;
      if (beta >= lo && beta < hi) src = s.basis_tok[static_cast<long long>(b) * s.K + beta];
    }
    if (src < 0) continue;                               // uniform in the CTA
    const uint4* __restrict__ V = reinterpret_cast<const uint4*>(sel_features(s)) + (static_cast<long long>(b) * s.N + src) * vec;
    uint4* __restrict__ dst = reinterpret_cast<uint4*>(s.Vg) + (static_cast<long long>(b) * s.R + r) * vec;
    // four 16-byte loads in flight per thread before their stores (V and Vg never overlap)
    int c = threadIdx.x;
    constexpr int T = kGatherThreads;
    for (; c + 3 * T < vec; c += 4 * T) {
      const uint4 x0 = __ldg(V + c), x1 = __ldg(V + c + T), x2 = __ldg(V + c + 2 * T), x3 = __ldg(V + c + 3 * T);
      dst[c] = x0;
      dst[c + T] = x1;
      dst[c + 2 * T] = x2;
      dst[c + 3 * T] = x3;
    }
    for (; c < vec; c += T) dst[c] = __ldg(V + c);
  }
}

// ------------------------------------------------------------------ coordinates
// Per-slot coordinate rows in shared memory have a pitch of 4 (mod 8) floats, so that eight
// lanes reading 16 bytes each from eight rows hit disjoint banks.
constexpr int kChunk = 32;
constexpr int kUpdSlots = 32;
constexpr int kRoundPitch = kRoundPicks + 4;

__host__ __device__ inline int coord_pitch(int KP) { return ((KP + 7) / 8) * 8 + 4; }

// ------------------------------------------------------------------ update
// Brings every active token's coordinates up to the current basis (nb vectors) by forward
// substitution before the picks:
//   e_beta[i] = (G[j_beta, i] - sum_{beta' < beta} e_beta'[j_beta] e_beta'[i]) / r_beta,
// 32 basis vectors (a chunk) at a time.  A CTA serves 32 slots, their coordinate rows in
// shared memory.  For a chunk starting at b0 the products with the coordinates before it,
// P[slot][row] = sum_{q < b0} e_q[slot] L[row][q] (L rows: the chunk's basis tokens' own
// coordinate rows), form a 32 x 32 x b0 matrix product: each warp takes every fourth
// 16-column block with 4 slots x 8 rows per thread (every loaded value feeds 4 or 8 FMAs).
// Warp 0 then adds the four partial products and solves the chunk's 32 x 32 triangle
// right-looking (lane = slot: each new coordinate is subtracted from the later ones at once,
// so a step waits for one FMA), while warps 1-3 copy the next chunk's L rows, triangle,
// Gram entries and basis norms into shared memory (cp.async), so that no chunk waits for a
// global load.  An image's slots spread over S / 32 CTAs.  Writes Ec, r2 and cstep = nb.
constexpr int kUpdWarps = 4;

__global__ void __launch_bounds__(kUpdSlots * kUpdWarps, 1) sel_update_kernel(SelState s) {
  pdl_enter();
  extern __shared__ __align__(16) float shu[];           // [32][P] slot rows, then [32][KP] L rows
  __shared__ float Lt[2][kChunk][kChunk + 1];            // a chunk's triangle L[i][b0 + q], q < i
  __shared__ float gsm[2][kUpdSlots][kChunk + 1];        // its Gram entries G[slot][b0 + i]
  __shared__ float rn[2][kChunk];                        // its basis norms
  __shared__ float part[kUpdWarps][kUpdSlots][kChunk + 1];
  __shared__ int tok_s[kUpdSlots], c0_s[kUpdSlots];
  const int b = blockIdx.y;
  if (s.done[b]) return;
  const int S = s.S, R = s.R, KP = s.KP, P = coord_pitch(KP);
  float* Lb = shu + kUpdSlots * P;
  const int nb = s.nbasis[b], gbase = s.gbase[b];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const long long base = static_cast<long long>(b) * s.N;
  if (threadIdx.x < kUpdSlots) {
    const int slot = blockIdx.x * kUpdSlots + threadIdx.x;
    const int tok = slot < S ? s.aslot[static_cast<long long>(b) * S + slot] : -1;
    tok_s[threadIdx.x] = tok;
    c0_s[threadIdx.x] = tok >= 0 ? min(s.cstep[base + tok], nb) : nb;
  }
  __syncthreads();
  int cmin = nb;                                     // fewest cached coordinates over the slots
  for (int i = 0; i < kUpdSlots; ++i) cmin = min(cmin, c0_s[i]);
  if (cmin >= nb) return;                            // uniform
  const int32_t* btok_g = s.basis_tok + static_cast<long long>(b) * s.K;
  const float* rnorm = s.rnorm + static_cast<long long>(b) * s.K;
  const float* Gb = s.G + (static_cast<long long>(b) * S + blockIdx.x * kUpdSlots) * R;
  // everything chunk c needs, copied by threads t0, t0 + stride, ... (one commit group)
  auto stage = [&](int c, int buf, int t0, int stride) {
    const int nch = min(nb, c + kChunk) - c, v4 = c / 4;
    for (int e = t0; e < nch * v4; e += stride) {    // L rows, columns [0, c)
      const int row = e / v4, q = (e - row * v4) * 4;
      cp_async16(Lb + row * KP + q, s.Ec + (base + __ldg(btok_g + c + row)) * KP + q);
    }
    for (int e = t0; e < nch * kChunk; e += stride) {   // the triangle: row i, columns c .. c + i - 1
      const int i = e / kChunk, q = e - i * kChunk;
      if (q < i) cp_async4(&Lt[buf][i][q], s.Ec + (base + __ldg(btok_g + c + i)) * KP + c + q);
    }
    for (int e = t0; e < kUpdSlots * nch; e += stride) {   // Gram entries of the slots that need them
      const int sl = e / nch, i = e - sl * nch;
      if (tok_s[sl] >= 0 && c + i >= c0_s[sl]) cp_async4(&gsm[buf][sl][i], Gb + static_cast<long long>(sl) * R + S + c + i - gbase);
    }
    for (int e = t0; e < nch; e += stride) cp_async4(&rn[buf][e], rnorm + c + e);
    cp_async_commit();
  };
  for (int r = warp; r < kUpdSlots; r += kUpdWarps) {   // cached coordinates [0, c0) of every slot
    const int tok = tok_s[r], c0 = c0_s[r];
    if (tok < 0) continue;
    const float* g = s.Ec + (base + tok) * KP;
    float* me = shu + r * P;
    for (int q = 4 * lane; q < c0; q += 128) cp_async16(me + q, g + q);
  }
  const int first = (cmin / kChunk) * kChunk;
  stage(first, 0, threadIdx.x, blockDim.x);
  const int mtok = tok_s[lane], mc0 = c0_s[lane];    // warp 0: this lane's slot
  float r2 = warp == 0 && mtok >= 0 ? s.r2[base + mtok] : 0.f;
  const int sg = lane >> 2, rg = lane & 3;           // products: slots 4 sg + 0..3, rows rg + 4 j
  int buf = 0;
  for (int b0 = first; b0 < nb; b0 += kChunk, buf ^= 1) {
    const int nch = min(nb, b0 + kChunk) - b0;
    cp_async_wait_all();                             // this chunk's copies (and the slot rows)
    __syncthreads();
    float acc[4][8];
#pragma unroll
    for (int u = 0; u < 4; ++u)
#pragma unroll
      for (int j = 0; j < 8; ++j) acc[u][j] = 0.f;
    for (int qa = 16 * warp; qa < b0; qa += 16 * kUpdWarps) {   // whole 16-column blocks (b0 % 32 == 0)
#pragma unroll
      for (int q4 = 0; q4 < 16; q4 += 4) {
        float4 m[4], l[8];
#pragma unroll
        for (int u = 0; u < 4; ++u) m[u] = *reinterpret_cast<const float4*>(shu + (4 * sg + u) * P + qa + q4);
#pragma unroll
        for (int j = 0; j < 8; ++j)
          l[j] = rg + 4 * j < nch ? *reinterpret_cast<const float4*>(Lb + (rg + 4 * j) * KP + qa + q4)
                                  : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int u = 0; u < 4; ++u)
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            float t = acc[u][j];
            t = fmaf(m[u].x, l[j].x, t);
            t = fmaf(m[u].y, l[j].y, t);
            t = fmaf(m[u].z, l[j].z, t);
            acc[u][j] = fmaf(m[u].w, l[j].w, t);
          }
      }
    }
#pragma unroll
    for (int u = 0; u < 4; ++u)
#pragma unroll
      for (int j = 0; j < 8; ++j) part[warp][4 * sg + u][rg + 4 * j] = acc[u][j];
    __syncthreads();                                 // products done: Lb is free
    if (warp != 0) {
      if (b0 + kChunk < nb) stage(b0 + kChunk, buf ^ 1, threadIdx.x - 32, blockDim.x - 32);
    } else if (mtok >= 0) {
      float* me = shu + lane * P;
      float av[kChunk];
#pragma unroll
      for (int i = 0; i < kChunk; ++i)
        av[i] = (i < nch && b0 + i >= mc0)
                    ? gsm[buf][lane][i] - ((part[0][lane][i] + part[1][lane][i]) + (part[2][lane][i] + part[3][lane][i]))
                    : 0.f;
#pragma unroll
      for (int i = 0; i < kChunk; ++i) {
        if (i < nch) {
          const int beta = b0 + i;
          float ei;
          if (beta >= mc0) {
            ei = av[i] / rn[buf][i];
            me[beta] = ei;
            r2 = fmaf(-ei, ei, r2);
          } else {
            ei = me[beta];
          }
#pragma unroll
          for (int j = i + 1; j < kChunk; ++j) av[j] = fmaf(-Lt[buf][j][i], ei, av[j]);
        }
      }
    }
    __syncthreads();                                 // this chunk's coordinates are written
  }
  if (warp == 0 && mtok >= 0 && mc0 < nb) {
    s.r2[base + mtok] = r2;
    s.cstep[base + mtok] = nb;
  }
  for (int r = warp; r < kUpdSlots; r += kUpdWarps) {   // new coordinates [c0, nb), a warp per row
    const int tok = tok_s[r], c0 = c0_s[r];
    if (tok < 0 || c0 >= nb) continue;
    float* g = s.Ec + (base + tok) * KP;
    const float* me = shu + r * P;
    for (int q = c0 + lane; q < nb; q += 32) g[q] = me[q];
  }
}

// ------------------------------------------------------------------ R0 basis
// The K0 forced picks (R0 in p_hat order) need no argmax: their basis is the Cholesky factor
// of the K0 x K0 Gram matrix G[R0, R0], column by column in pick order (right-looking, in
// shared memory).  Column t adds basis vector nb unless its residual is degenerate
// (r^2 <= tau ||v||^2); its entries below the diagonal are the later R0 tokens' coordinates
// e_nb.  Writes picks, state, basis, Ec rows, cstep and r2 of the R0 tokens.
constexpr int kCholThreads = kCholMax;

// Left-looking, one thread per R0 position u, G[R0, R0] and the coordinate rows in shared
// memory; one block barrier per basis vector.
__global__ void __launch_bounds__(kCholThreads, 1) sel_chol_kernel(SelState s) {
  pdl_enter();
  extern __shared__ __align__(16) float shc[];
  __shared__ float r2s[kCholMax], dg[kCholMax], dpick[kCholMax], ps[kCholMax];
  __shared__ int tk[kCholMax], mine_s[kCholMax], bidx[kCholMax];
  const int b = blockIdx.x;
  const int K0 = s.K0, ldg = (K0 + 3) & ~3, PL = coord_pitch(K0);
  float* Gs = shc;                                   // [K0][ldg]
  float* Ls = shc + K0 * ldg;                        // [K0][PL] coordinates, zeros past the valid ones
  const long long base = static_cast<long long>(b) * s.N;
  const float* Gb = s.G + static_cast<long long>(b) * s.S * s.R;
  {
    const int v4 = ldg / 4;                          // G rows are 16-byte aligned (R % 16 == 0)
    for (int i = threadIdx.x; i < K0 * v4; i += blockDim.x) {
      const int r = i / v4, c = (i - r * v4) * 4;
      cp_async16(Gs + r * ldg + c, Gb + static_cast<long long>(r) * s.R + c);
    }
  }
  for (int i = threadIdx.x; i < K0 * PL / 4; i += blockDim.x)
    reinterpret_cast<float4*>(Ls)[i] = make_float4(0.f, 0.f, 0.f, 0.f);
  cp_async_wait_all();
  const int u = threadIdx.x;
  if (u < K0) {
    tk[u] = s.r0[static_cast<long long>(b) * s.K + u];
    ps[u] = s.scores[base + tk[u]];
  }
  __syncthreads();
  float r2 = 0.f;
  if (u < K0) {
    r2 = Gs[u * ldg + u];
    r2s[u] = r2;
    dg[u] = r2;
  }
  __syncthreads();
  float* me = Ls + u * PL;
  int nb = 0;
  for (int t = 0; t < K0; ++t) {
    const float d = r2s[t], sq = dg[t];
    const bool ext = d > s.tau * sq && d > 0.f;
    if (u == t) {                                         // global writes wait for the end
      mine_s[t] = nb;
      dpick[t] = d;
      bidx[t] = ext ? nb : -1;
    }
    if (!ext) continue;                                   // uniform
    if (u > t && u < K0) {
      const float* lt = Ls + t * PL;
      const float rinv = 1.0f / sqrtf(d), gut = Gs[u * ldg + t];   // independent of the dot product
      float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
#pragma unroll 4
      for (int q = 0; q < nb; q += 4) {                   // rows are zero past nb
        const float4 x = *reinterpret_cast<const float4*>(lt + q);
        const float4 y = *reinterpret_cast<const float4*>(me + q);
        a0 = fmaf(x.x, y.x, a0);
        a1 = fmaf(x.y, y.y, a1);
        a2 = fmaf(x.z, y.z, a2);
        a3 = fmaf(x.w, y.w, a3);
      }
      const float e = (gut - ((a0 + a1) + (a2 + a3))) * rinv;
      me[nb] = e;
      r2 = fmaf(-e, e, r2);
      r2s[u] = r2;
    }
    __syncthreads();
    ++nb;
  }
  __syncthreads();
  if (u < K0) {
    const int tok = tk[u];
    const float d = dpick[u];
    s.picks[static_cast<long long>(b) * s.K + u] = tok;
    s.state[base + tok] = 1;
    s.cstep[base + tok] = mine_s[u];
    s.r2[base + tok] = d;
    s.U[base + tok] = sel_value(ps[u], d, dg[u], s.lambda, s.tau);
    if (bidx[u] >= 0) {
      s.basis_tok[static_cast<long long>(b) * s.K + bidx[u]] = tok;
      s.rnorm[static_cast<long long>(b) * s.K + bidx[u]] = sqrtf(d);
    }
  }
  // coordinate rows of the R0 tokens: e_beta for beta < (basis size at their pick)
  for (int i = threadIdx.x; i < K0 * PL; i += blockDim.x) {
    const int r = i / PL, q = i - r * PL;
    if (q < mine_s[r]) s.Ec[(base + tk[r]) * s.KP + q] = Ls[r * PL + q];
  }
  if (threadIdx.x == 0) {
    s.nbasis[b] = nb;
    s.npicks[b] = K0;
  }
}

// ------------------------------------------------------------------ residual Gram
// When a round's picks start, every active token's coordinates are current on the c0 basis
// vectors of the round (sel_update_kernel).  Over that basis the residual Gram matrix of
// the active set is
//   G'[i][k] = <v_i, v_k> - sum_{q < c0} e_q[i] e_q[k]   (the inner product of the residuals),
// and a pick then needs only the coordinates added during the round (sel_greedy_kernel).
// It replaces the A x A part of the Gram block in place.  One CTA of 64 threads per 32 x 32
// tile of the upper triangle (the matrix is symmetric: the mirrored tile is written from the
// same values), 4 x 4 outputs per thread; the coordinates are staged in 16-column chunks,
// transposed, in two shared buffers, the next chunk loaded during the products of the
// current one.  Small tiles keep several CTAs on every SM, so the chunk loop's latency is
// hidden, with few images (c0 is large) as with many.
constexpr int kRgTile = 32, kRgChunk = 16, kRgPad = kRgTile + 4, kRgThreads = 64;

__global__ void __launch_bounds__(kRgThreads) sel_resgram_kernel(SelState s) {
  pdl_enter();
  // two buffers of both operands' chunks; after the products, the output tile
  __shared__ __align__(16) float sbuf[4 * kRgChunk * kRgPad];
  static_assert(4 * kRgChunk * kRgPad >= kRgTile * (kRgTile + 1), "tile staging");
  float(*Ei)[kRgChunk][kRgPad] = reinterpret_cast<float(*)[kRgChunk][kRgPad]>(sbuf);
  float(*Ek)[kRgChunk][kRgPad] = reinterpret_cast<float(*)[kRgChunk][kRgPad]>(sbuf + 2 * kRgChunk * kRgPad);
  __shared__ int toki[kRgTile], tokk[kRgTile];
  const int b = blockIdx.y;
  if (s.done[b]) return;
  const int c0 = s.nbasis[b];
  if (c0 == 0) return;
  const int S = s.S, KP = s.KP;
  int t = blockIdx.x, ti = 0;
  const int T = S / kRgTile;
  while (t >= T - ti) { t -= T - ti; ++ti; }
  const int tk = ti + t;
  const int32_t* aslot = s.aslot + static_cast<long long>(b) * S;
  const int tid = threadIdx.x;
  if (tid < kRgTile) toki[tid] = aslot[ti * kRgTile + tid];
  else tokk[tid - kRgTile] = aslot[tk * kRgTile + tid - kRgTile];
  // a tile whose rows or columns are all empty slots writes nothing
  const bool any_i = __syncthreads_or(tid < kRgTile && toki[tid] >= 0);
  const bool any_k = __syncthreads_or(tid < kRgTile && tokk[tid] >= 0);
  if (!any_i || !any_k) return;
  const long long base = static_cast<long long>(b) * s.N;
  // staging: threads 0-31 the rows of the tile's row slots, 32-63 those of its column slots
  const int lr = tid & (kRgTile - 1);
  const int ltok = tid < kRgTile ? toki[lr] : tokk[lr];
  const float* row = ltok >= 0 ? s.Ec + (base + ltok) * KP : nullptr;
  float(*Eop)[kRgChunk][kRgPad] = tid < kRgTile ? Ei : Ek;
  auto load16 = [&](int q, float* x) {
#pragma unroll
    for (int j = 0; j < 16; ++j) x[j] = 0.f;
    if (!row) return;
    if (q + 16 <= c0) {
#pragma unroll
      for (int j = 0; j < 16; j += 4) {
        const float4 u = *reinterpret_cast<const float4*>(row + q + j);
        x[j] = u.x; x[j + 1] = u.y; x[j + 2] = u.z; x[j + 3] = u.w;
      }
    } else {
#pragma unroll
      for (int j = 0; j < 16; ++j)
        if (q + j < c0) x[j] = row[q + j];
    }
  };
  const int tx = tid & 7, ty = tid >> 3;             // outputs: rows ty*4 .. +3, columns tx*4 .. +3
  float acc[4][4];
#pragma unroll
  for (int r = 0; r < 4; ++r)
#pragma unroll
    for (int c = 0; c < 4; ++c) acc[r][c] = 0.f;
  float x[16];
  load16(0, x);
  int buf = 0;
#pragma unroll
  for (int j = 0; j < 16; ++j) Eop[0][j][lr] = x[j];
  __syncthreads();
  for (int q0 = 0; q0 < c0; q0 += kRgChunk, buf ^= 1) {
    const bool more = q0 + kRgChunk < c0;
    if (more) load16(q0 + kRgChunk, x);              // next chunk in flight during the products
#pragma unroll
    for (int q = 0; q < kRgChunk; ++q) {
      const float4 a = *reinterpret_cast<const float4*>(&Ei[buf][q][ty * 4]);
      const float4 c = *reinterpret_cast<const float4*>(&Ek[buf][q][tx * 4]);
      const float av[4] = {a.x, a.y, a.z, a.w}, cv[4] = {c.x, c.y, c.z, c.w};
#pragma unroll
      for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int cc = 0; cc < 4; ++cc) acc[r][cc] = fmaf(av[r], cv[cc], acc[r][cc]);
    }
    if (more) {                                      // the other buffer was last read a chunk ago
#pragma unroll
      for (int j = 0; j < 16; ++j) Eop[buf ^ 1][j][lr] = x[j];
    }
    __syncthreads();
  }
  // G' = G - acc through a shared tile, so that both the tile and its mirror are read and
  // written in whole rows (coalesced)
  float(*Tt)[kRgTile + 1] = reinterpret_cast<float(*)[kRgTile + 1]>(sbuf);
#pragma unroll
  for (int r = 0; r < 4; ++r)
#pragma unroll
    for (int cc = 0; cc < 4; ++cc) Tt[ty * 4 + r][tx * 4 + cc] = acc[r][cc];
  __syncthreads();
  float* Gb = s.G + static_cast<long long>(b) * S * s.R;
  constexpr int kRowsPer = kRgTile * kRgTile / kRgThreads;   // rows of the tile per thread
  {
    const int c = tid & (kRgTile - 1), r0 = tid / kRgTile;
    const bool okc = tokk[c] >= 0;
    float* g0 = Gb + static_cast<long long>(ti * kRgTile) * s.R + tk * kRgTile + c;
    float gv[kRowsPer];                              // every load in flight before the stores
#pragma unroll
    for (int m = 0; m < kRowsPer; ++m) {
      const int r = r0 + m * (kRgThreads / kRgTile);
      gv[m] = okc && toki[r] >= 0 ? g0[static_cast<long long>(r) * s.R] : 0.f;
    }
#pragma unroll
    for (int m = 0; m < kRowsPer; ++m) {
      const int r = r0 + m * (kRgThreads / kRgTile);
      if (okc && toki[r] >= 0) {
        const float v = gv[m] - Tt[r][c];
        g0[static_cast<long long>(r) * s.R] = v;
        Tt[r][c] = v;
      }
    }
    if (ti != tk) {
      __syncthreads();
      float* m0 = Gb + static_cast<long long>(tk * kRgTile) * s.R + ti * kRgTile + c;
#pragma unroll
      for (int m = 0; m < kRowsPer; ++m) {         // row r of the mirror: column r of the tile
        const int r = r0 + m * (kRgThreads / kRgTile);
        if (tokk[r] >= 0 && toki[c] >= 0) m0[static_cast<long long>(r) * s.R] = Tt[c][r];
      }
    }
  }
}

// ------------------------------------------------------------------ greedy
// One CTA of S threads per image; thread = active slot.  The A x A part of the Gram block
// holds the residual Gram matrix G' on the c0 basis vectors of the round (above), so a pick
// of slot j updates slot i with the coordinates added in this launch only:
//   e_new[i] = (G'[j][i] - sum_{c0 <= q < nb} e_q[j] e_q[i]) / r_j.
// Each slot keeps its round coordinates in a shared-memory row: its own side of the dot
// products, and the other side for every thread (16-byte broadcasts) when that slot wins.  The picks take one block barrier each: the winning slot is carried in the low bits
// of the key, and every slot's residual is published in shared memory, so all threads
// derive the basis update from the same values; the winner's G' entry is loaded while the
// dot product runs.  At most kRoundPicks picks per launch (the next round continues).

// key of a candidate inside the round: (value bits, 0xFFFF - token, slot); the upper 48
// bits order like make_key (value descending, lower token first).
__device__ __forceinline__ uint64_t theta48(uint64_t theta) {   // make_key -> upper 48 bits of the round key
  if (theta == 0) return 0;
  const uint32_t tok = static_cast<uint32_t>(key_index(theta));
  return ((theta >> 32) << 16) | (0xFFFFu - tok);
}

// Largest (hi, lo) pair over the warp, hi first: two warp reductions on 32-bit words.
__device__ __forceinline__ uint64_t warp_max_key(uint32_t hi, uint32_t lo) {
  const uint32_t h = __reduce_max_sync(0xffffffffu, hi);
  const uint32_t l = __reduce_max_sync(0xffffffffu, hi == h ? lo : 0u);
  return (static_cast<uint64_t>(h) << 32) | l;
}

__global__ void __launch_bounds__(kActiveSlots, 1) sel_greedy_kernel(SelState s) {
  pdl_enter();
  extern __shared__ __align__(16) float shf[];
  __shared__ uint64_t wkey[2][32];
  const int b = blockIdx.x;
  if (s.done[b]) return;
  const int S = s.S, R = s.R, KP = s.KP;
  float* r2s = shf;                                  // [S] published residuals
  float* sqs = r2s + S;                              // [S]
  int32_t* tks = reinterpret_cast<int32_t*>(sqs + S);   // [S] tokens of the slots
  int32_t* ends = tks + S;                           // [S] round coordinates of the slots at the end
  int32_t* pk_tok = ends + S;                        // [kRoundPicks] this launch's picks
  float* pk_r2 = reinterpret_cast<float*>(pk_tok + kRoundPicks);  // their residuals (-1: no basis vector)
  float* Er = pk_r2 + kRoundPicks;                   // [S][kRoundPitch] round coordinates
  const long long base = static_cast<long long>(b) * s.N;
  const int slot = threadIdx.x;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
  const int tok = s.aslot[static_cast<long long>(b) * S + slot];
  const float* Gb = s.G + static_cast<long long>(b) * S * R;
  int nb = s.nbasis[b], np = s.npicks[b];
  const int c0 = nb;
  const bool forced = s.mode[b] == 1;
  const uint64_t th48 = theta48(s.theta[b]);
  float* me = Er + slot * kRoundPitch;

  float r2 = 0.f, sq = 0.f, p = 0.f, val = 0.f;
  int mine = nb;                                     // valid coordinates at the end
  bool alive = false;
  if (tok >= 0) {
    p = sel_scores(s)[base + tok];
    alive = s.state[base + tok] == 0;
    if (s.cstep[base + tok] < nb) {                  // sel_update_kernel did not run
      atomicOr(s.status, ST_INTERNAL);
      alive = false;
    }
    r2 = s.r2[base + tok];
    sq = s.sqn[base + tok];
  }
  {
    // zero rows: the unrolled dot products read a winner's row up to the next multiple of 32
    float4* row4 = reinterpret_cast<float4*>(me);
    for (int q = 0; q < kRoundPitch / 4; ++q) row4[q] = make_float4(0.f, 0.f, 0.f, 0.f);
  }
  tks[slot] = tok;
  if (tok >= 0) val = sel_value(p, r2, sq, s.lambda, s.tau);
  r2s[slot] = r2;
  sqs[slot] = sq;
  __syncthreads();

  int nr = 0;                                        // round coordinates so far (uniform)
  for (int step = 0, buf = 0; np < s.K && step < kRoundPicks; ++step, buf ^= 1) {
    {
      const uint32_t vb = alive ? __float_as_uint(val > 0.f ? val : 0.f) : 0u;
      const uint32_t lo = alive ? ((0xFFFFu - static_cast<uint32_t>(tok)) << 16) | static_cast<uint32_t>(slot) : 0u;
      const uint64_t key = warp_max_key(vb, lo);
      if (lane == 0) wkey[buf][warp] = key;
    }
    __syncthreads();
    int jslot;
    if (forced) {
      jslot = step;
      if (jslot >= S || tks[jslot] < 0) break;
    } else {
      const uint64_t k = lane < nwarps ? wkey[buf][lane] : 0ull;
      const uint64_t best = warp_max_key(static_cast<uint32_t>(k >> 32), static_cast<uint32_t>(k));
      if (best == 0 || (best >> 16) <= th48) break;   // uniform
      jslot = static_cast<int>(best & 0xFFFFu);
    }
    const int jt = tks[jslot];
    const float r2j = r2s[jslot], sqj = sqs[jslot];
    const bool ext = (r2j > s.tau * sqj) && (r2j > 0.f);
    if (slot == jslot) {                             // global writes wait for the end
      alive = false;
      mine = nb;
      pk_tok[step] = jt;
      pk_r2[step] = ext ? r2j : -1.f;
    }
    if (ext) {
      if (alive) {
        const float gji = Gb[static_cast<long long>(jslot) * R + slot];   // in flight during the dot product
        const float rinv = 1.0f / sqrtf(r2j);
        const float* cj = Er + jslot * kRoundPitch;
        float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
        // 32 coordinates per branch, so that the loads of a block issue together; rows are
        // zero past the round's coordinates
#pragma unroll
        for (int blk = 0; blk < kRoundPicks / 32; ++blk) {
          if (32 * blk < nr) {
#pragma unroll
            for (int g = 8 * blk; g < 8 * blk + 8; ++g) {
              const float4 c = *reinterpret_cast<const float4*>(cj + 4 * g);
              const float4 m = *reinterpret_cast<const float4*>(me + 4 * g);
              a0 = fmaf(c.x, m.x, a0);
              a1 = fmaf(c.y, m.y, a1);
              a2 = fmaf(c.z, m.z, a2);
              a3 = fmaf(c.w, m.w, a3);
            }
          }
        }
        const float e = (gji - ((a0 + a1) + (a2 + a3))) * rinv;
        me[nr] = e;
        r2 = fmaf(-e, e, r2);
        val = sel_value(p, r2, sq, s.lambda, s.tau);
        r2s[slot] = r2;
      }
      ++nb;
      ++nr;
    }
    ++np;
  }
  // write back: this launch's picks, then the active tokens
  const int np0 = s.npicks[b], nb0 = s.nbasis[b];
  __syncthreads();
  if (threadIdx.x == 0) {
    int nbw = nb0;
    for (int i = 0; i < np - np0; ++i) {
      if (pk_r2[i] >= 0.f) {
        s.basis_tok[static_cast<long long>(b) * s.K + nbw] = pk_tok[i];
        s.rnorm[static_cast<long long>(b) * s.K + nbw] = sqrtf(pk_r2[i]);
        ++nbw;
      }
    }
  }
  for (int i = threadIdx.x; i < np - np0; i += blockDim.x) {
    s.picks[static_cast<long long>(b) * s.K + np0 + i] = pk_tok[i];
    s.state[base + pk_tok[i]] = 1;
  }
  if (tok >= 0) {
    if (alive) mine = nb;
    s.cstep[base + tok] = mine;
    s.r2[base + tok] = r2;
    s.U[base + tok] = val;
  }
  // coordinates [c0, mine) of every slot: its round row, one warp per row
  ends[slot] = tok >= 0 ? mine : c0;
  __syncthreads();
  for (int r = warp; r < S; r += nwarps) {
    const int t = tks[r], end = ends[r];
    if (t < 0) continue;
    float* g = s.Ec + (base + t) * KP;
    const float* src = Er + r * kRoundPitch;
    for (int q = c0 + lane; q < end; q += 32) g[q] = src[q - c0];
  }
  if (threadIdx.x == 0) {
    s.nbasis[b] = nb;
    s.npicks[b] = np;
    if (np >= s.K) { s.done[b] = 1; atomicAdd(s.done_count, 1); }
  }
}

// ------------------------------------------------------------------ projection set-up
// Gathers every basis row of the images to project (no active tokens) for the projection.
__global__ void sel_proj_prep_kernel(SelState s, int first) {
  pdl_enter();
  const int b = blockIdx.x;
  const int nb = s.nbasis[b];
  const bool go = first || (!s.done[b] && nb > s.gbase[b] && nb <= kReprojMax);
  if (s.blist && b == 0 && threadIdx.x == 0) s.bcount[s.bc_par ^ 1] = 0;
  if (!go) {
    if (threadIdx.x == 0) s.proj_lim[b] = 0;
    return;
  }
  for (int i = threadIdx.x; i < s.S; i += blockDim.x) s.aslot[static_cast<long long>(b) * s.S + i] = -1;
  if (threadIdx.x == 0) {
    if (s.blist) s.blist[atomicAdd(s.bcount + s.bc_par, 1)] = b;
    s.proj_lim[b] = kReprojMax;
    s.gbase[b] = 0;                                  // rows S + beta for the whole basis
    s.gb_lo[b] = 0;
    s.gb_hi[b] = nb;
    s.nb_gathered[b] = nb;
  }
}

__global__ void sel_proj_done_kernel(SelState s) {
  pdl_enter();
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b < s.B && s.proj_lim[b] > 0) {
    s.gbase[b] = s.nbasis[b];
    s.nb_gathered[b] = s.nbasis[b];
  }
}

// ------------------------------------------------------------------ outputs
// keep = picks sorted ascending; pick_order = picks.
__global__ void sel_finalize_kernel(const int32_t* picks, int K, int32_t* keep, int32_t* order) {
  pdl_enter();
  extern __shared__ int32_t sh32[];
  const int b = blockIdx.x;
  const int32_t* p = picks + static_cast<long long>(b) * K;
  for (int i = threadIdx.x; i < K; i += blockDim.x) {
    sh32[i] = p[i];
    if (order) order[static_cast<long long>(b) * K + i] = p[i];
  }
  __syncthreads();
  if (K <= static_cast<int>(blockDim.x)) {
    // place = number of smaller picks (equal ones, which a valid selection never has, by position)
    const int i = threadIdx.x;
    if (i < K) {
      const int32_t x = sh32[i];
      int rank = 0;
      for (int j = 0; j < K; ++j) {
        const int32_t y = sh32[j];
        rank += (y < x || (y == x && j < i)) ? 1 : 0;
      }
      keep[static_cast<long long>(b) * K + rank] = x;
    }
    return;
  }
  block_sort_asc_i32(sh32, K, pow2_at_least(K));
  for (int i = threadIdx.x; i < K; i += blockDim.x) keep[static_cast<long long>(b) * K + i] = sh32[i];
}

// top-K by p_hat (lambda = 0 or K0 = K): R0 computed by sel_init is the whole answer.
__global__ void sel_copy_r0_kernel(const int32_t* r0, int K, int32_t* picks) {
  pdl_enter();
  const int b = blockIdx.x;
  for (int i = threadIdx.x; i < K; i += blockDim.x)
    picks[static_cast<long long>(b) * K + i] = r0[static_cast<long long>(b) * K + i];
}

__global__ void sel_identity_kernel(int N, int32_t* keep, int32_t* order) {
  pdl_enter();
  const int b = blockIdx.x;
  for (int i = threadIdx.x; i < N; i += blockDim.x) {
    keep[static_cast<long long>(b) * N + i] = i;
    if (order) order[static_cast<long long>(b) * N + i] = i;
  }
}


// ------------------------------------------------------------------ device-side round loop
// First node of the loop graph: the WHILE body runs only if an image still selects.
__global__ void sel_loop_init_kernel(SelState s, cudaGraphConditionalHandle h, int32_t* iters) {
  if (threadIdx.x == 0) {
    *iters = 0;
    cudaGraphSetConditional(h, (*s.done_count < s.B && *s.status == 0) ? 1u : 0u);
  }
}

// Last node of the WHILE body: run another round while an image still selects, no kernel
// has reported an error and the iteration cap has not been reached (then ST_INTERNAL).  It
// also clears the image-list count the round's choose appended to (the Gram block has read
// it), so that the next iteration's choose starts from zero on the same counter.
__global__ void sel_loop_cond_kernel(SelState s, cudaGraphConditionalHandle h, int32_t* iters, int cap_iters,
                                     long long* iters_total) {
  if (threadIdx.x == 0) {
    s.bcount[s.bc_par] = 0;
    const int it = *iters + 1;
    *iters = it;
    *iters_total += 1;
    const bool pending = *s.done_count < s.B, err = *s.status != 0;
    if (pending && !err && it >= cap_iters) atomicOr(s.status, ST_INTERNAL);
    cudaGraphSetConditional(h, (pending && !err && it < cap_iters) ? 1u : 0u);
  }
}

}  // namespace

size_t sel_init_smem(int N, int K0) { return (static_cast<size_t>(N) + pow2_at_least(std::max(K0, 1))) * 8; }
size_t sel_choose_smem(int N) { return static_cast<size_t>(N) * 8; }
size_t sel_greedy_smem(int S) {
  return static_cast<size_t>(S) * 16 + static_cast<size_t>(kRoundPicks) * 8 +
         static_cast<size_t>(S) * kRoundPitch * 4;
}
size_t sel_chol_smem(int K0) {
  return (static_cast<size_t>(K0) * ((K0 + 3) & ~3) + static_cast<size_t>(K0) * coord_pitch(K0)) * 4;
}
size_t sel_update_smem(int KP) {
  return (static_cast<size_t>(kUpdSlots) * coord_pitch(KP) + static_cast<size_t>(kChunk) * KP) * 4;
}

cudaError_t launch_sel_init(const SelState& s, cudaStream_t st) {
  const size_t sm = sel_init_smem(s.N, s.K0);
  cudaError_t e = cudaFuncSetAttribute(sel_init_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(sm));
  if (e != cudaSuccess) return e;
  return launch_k(sel_init_kernel, dim3(s.B), dim3(1024), sm, st, s);
}

cudaError_t launch_sel_choose(const SelState& s, cudaStream_t st) {
  const size_t sm = sel_choose_smem(s.N);
  cudaError_t e = cudaFuncSetAttribute(sel_choose_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(sm));
  if (e != cudaSuccess) return e;
  if ((e = launch_k(sel_choose_kernel, dim3(s.B), dim3(1024), sm, st, s)) != cudaSuccess) return e;
  return launch_k(sel_gather_kernel, dim3(kGatherCtas, s.B), dim3(kGatherThreads), 0, st, s);
}

cudaError_t launch_sel_greedy(const SelState& s, cudaStream_t st) {
  if (s.S != kActiveSlots) return cudaErrorInvalidValue;
  const size_t um = sel_update_smem(s.KP);
  cudaError_t e = cudaFuncSetAttribute(sel_update_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(um));
  if (e != cudaSuccess) return e;
  e = launch_k(sel_update_kernel, dim3((s.S + kUpdSlots - 1) / kUpdSlots, s.B), dim3(kUpdSlots * kUpdWarps), um, st, s);
  if (e != cudaSuccess) return e;
  const int T = s.S / kRgTile;
  e = launch_k(sel_resgram_kernel, dim3(T * (T + 1) / 2, s.B), dim3(kRgThreads), 0, st, s);
  if (e != cudaSuccess) return e;
  const size_t sm = sel_greedy_smem(s.S);
  e = cudaFuncSetAttribute(sel_greedy_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(sm));
  if (e != cudaSuccess) return e;
  return launch_k(sel_greedy_kernel, dim3(s.B), dim3(s.S), sm, st, s);
}

cudaError_t launch_sel_chol(const SelState& s, cudaStream_t st) {
  if (s.K0 < 1 || s.K0 > kCholMax || s.K0 > s.S) return cudaErrorInvalidValue;
  const size_t sm = sel_chol_smem(s.K0);
  cudaError_t e = cudaFuncSetAttribute(sel_chol_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(sm));
  if (e != cudaSuccess) return e;
  return launch_k(sel_chol_kernel, dim3(s.B), dim3(kCholThreads), sm, st, s);
}

cudaError_t launch_sel_finalize(const int32_t* picks, int B, int K, int32_t* keep, int32_t* order, cudaStream_t st) {
  const size_t sm = static_cast<size_t>(pow2_at_least(K)) * 4;
  return launch_k(sel_finalize_kernel, dim3(B), dim3(1024), sm, st, picks, K, keep, order);
}

cudaError_t launch_sel_copy_r0(const int32_t* r0, int B, int K, int32_t* picks, cudaStream_t st) {
  return launch_k(sel_copy_r0_kernel, dim3(B), dim3(256), 0, st, r0, K, picks);
}

cudaError_t launch_sel_proj_prep(const SelState& s, bool first, cudaStream_t st) {
  return launch_k(sel_proj_prep_kernel, dim3(s.B), dim3(256), 0, st, s, first ? 1 : 0);
}

cudaError_t launch_sel_gather(const SelState& s, cudaStream_t st) {
  return launch_k(sel_gather_kernel, dim3(kGatherCtas, s.B), dim3(kGatherThreads), 0, st, s);
}

cudaError_t launch_sel_proj_done(const SelState& s, cudaStream_t st) {
  return launch_k(sel_proj_done_kernel, dim3((s.B + 127) / 128), dim3(128), 0, st, s);
}

cudaError_t launch_sel_identity(int B, int N, int32_t* keep, int32_t* order, cudaStream_t st) {
  return launch_k(sel_identity_kernel, dim3(B), dim3(256), 0, st, N, keep, order);
}

// ------------------------------------------------------------------ loop graph cache
struct SelLoopEntry {
  std::vector<long long> key;
  cudaGraph_t graph = nullptr;
  cudaGraphExec_t exec = nullptr;
};

struct SelLoopCache {
  std::vector<SelLoopEntry> entries;   // most recently used last
  cudaStream_t cap = nullptr;          // stream the loop body is captured on
};

namespace {
constexpr size_t kSelLoopCacheMax = 8;

void release_entry(SelLoopEntry& e) {
  if (e.exec) cudaGraphExecDestroy(e.exec);
  if (e.graph) cudaGraphDestroy(e.graph);
  e.exec = nullptr;
  e.graph = nullptr;
}

long long fbits(float f) {
  uint32_t u;
  std::memcpy(&u, &f, 4);
  return static_cast<long long>(u);
}
long long pbits(const void* p) { return static_cast<long long>(reinterpret_cast<uintptr_t>(p)); }

// Everything the captured kernels depend on, except the caller's scores and features (read
// through s.uptr).
std::vector<long long> loop_key(const SelState& s, const GemmDesc& g, int num_sms, int cap_iters, const int32_t* iters,
                                const long long* iters_total) {
  return {s.B, s.N, s.D, s.K, s.K0, s.S, s.R, s.KP, fbits(s.lambda), fbits(s.tau), pbits(s.sqn), pbits(s.U),
          pbits(s.r2), pbits(s.cstep), pbits(s.state), pbits(s.Ec), pbits(s.picks), pbits(s.r0), pbits(s.basis_tok),
          pbits(s.rnorm), pbits(s.npicks), pbits(s.nbasis), pbits(s.nb_gathered), pbits(s.done), pbits(s.mode),
          pbits(s.nlimit), pbits(s.gb_lo), pbits(s.gb_hi), pbits(s.gbase), pbits(s.theta), pbits(s.aslot),
          pbits(s.Vg), pbits(s.G), pbits(s.done_count), pbits(s.proj_lim), pbits(s.blist), pbits(s.bcount),
          s.bc_par, pbits(s.status), pbits(s.nvalid), pbits(s.uptr),
          pbits(g.A), g.a_rows_total, g.a_row_stride, pbits(g.B), g.b_rows_total, g.b_row_stride, g.M, g.N, g.K,
          g.batch, pbits(g.n_limit), pbits(g.C), g.ldc, g.c_batch_stride, g.epi, pbits(g.status), pbits(g.blist),
          g.wait_ns, num_sms, cap_iters, pbits(iters), pbits(iters_total)};
}

// Builds the graph: [test kernel] -> WHILE { choose + gather, Gram, update + residual Gram +
// greedy; test }.
cudaError_t build_loop(SelLoopCache* c, const SelState& s, const GemmDesc& gram, int num_sms, int cap_iters,
                       int32_t* iters, long long* iters_total, SelLoopEntry& out) {
  cudaError_t e = cudaSuccess;
  if (!c->cap && (e = cudaStreamCreateWithFlags(&c->cap, cudaStreamNonBlocking)) != cudaSuccess) return e;
  cudaGraph_t g = nullptr;
  if ((e = cudaGraphCreate(&g, 0)) != cudaSuccess) return e;
  auto fail = [&](cudaError_t err) {
    cudaGraphDestroy(g);
    return err;
  };
  cudaGraphConditionalHandle h;
  if ((e = cudaGraphConditionalHandleCreate(&h, g, 0, 0)) != cudaSuccess) return fail(e);
  SelState sc = s;
  void* init_args[] = {&sc, &h, &iters};
  cudaKernelNodeParams kp = {};
  kp.func = reinterpret_cast<void*>(sel_loop_init_kernel);
  kp.gridDim = dim3(1);
  kp.blockDim = dim3(32);
  kp.kernelParams = init_args;
  cudaGraphNode_t init_node;
  if ((e = cudaGraphAddKernelNode(&init_node, g, nullptr, 0, &kp)) != cudaSuccess) return fail(e);
  cudaGraphNodeParams cp = {};
  cp.type = cudaGraphNodeTypeConditional;
  cp.conditional.handle = h;
  cp.conditional.type = cudaGraphCondTypeWhile;
  cp.conditional.size = 1;
  cudaGraphNode_t loop_node;
  if ((e = cudaGraphAddNode(&loop_node, g, &init_node, nullptr, 1, &cp)) != cudaSuccess) return fail(e);
  cudaGraph_t body = cp.conditional.phGraph_out[0];
  if ((e = cudaStreamBeginCaptureToGraph(c->cap, body, nullptr, nullptr, 0, cudaStreamCaptureModeRelaxed)) !=
      cudaSuccess)
    return fail(e);
  pdl_disabled() = true;
  SelState r = s;
  {
    GemmDesc d = gram;
    d.bcount = r.bcount + r.bc_par;              // the count this round's choose appends to
    if ((e = launch_sel_choose(r, c->cap)) == cudaSuccess && (e = launch_gemm(d, num_sms, c->cap)) == cudaSuccess)
      e = launch_sel_greedy(r, c->cap);
  }
  if (e == cudaSuccess) e = launch_k(sel_loop_cond_kernel, dim3(1), dim3(32), 0, c->cap, r, h, iters, cap_iters, iters_total);
  pdl_disabled() = false;
  cudaGraph_t captured = nullptr;
  const cudaError_t e2 = cudaStreamEndCapture(c->cap, &captured);
  if (e == cudaSuccess) e = e2;
  if (e != cudaSuccess) return fail(e);
  cudaGraphExec_t x = nullptr;
  if ((e = cudaGraphInstantiate(&x, g, 0)) != cudaSuccess) return fail(e);
  out.graph = g;
  out.exec = x;
  return cudaSuccess;
}
}  // namespace

SelLoopCache* sel_loop_cache_create() { return new SelLoopCache(); }

void sel_loop_cache_destroy(SelLoopCache* c) {
  if (!c) return;
  for (auto& e : c->entries) release_entry(e);
  if (c->cap) cudaStreamDestroy(c->cap);
  delete c;
}

cudaError_t launch_sel_loop(SelLoopCache* c, const SelState& s, const GemmDesc& gram, int num_sms, int cap_iters,
                            int32_t* iters, long long* iters_total, cudaStream_t st) {
  if (!c || !s.uptr || !s.done_count || !iters || !iters_total || (s.bc_par & ~1)) return cudaErrorInvalidValue;
  std::vector<long long> key = loop_key(s, gram, num_sms, cap_iters, iters, iters_total);
  size_t hit = c->entries.size();
  for (size_t i = 0; i < c->entries.size(); ++i)
    if (c->entries[i].key == key) { hit = i; break; }
  if (hit == c->entries.size()) {
    SelLoopEntry ent;
    ent.key = std::move(key);
    const cudaError_t e = build_loop(c, s, gram, num_sms, cap_iters, iters, iters_total, ent);
    if (e != cudaSuccess) return e;
    if (c->entries.size() >= kSelLoopCacheMax) {
      release_entry(c->entries.front());
      c->entries.erase(c->entries.begin());
    }
    c->entries.push_back(std::move(ent));
  } else if (hit + 1 != c->entries.size()) {
    SelLoopEntry ent = std::move(c->entries[hit]);
    c->entries.erase(c->entries.begin() + static_cast<long>(hit));
    c->entries.push_back(std::move(ent));
  }
  return cudaGraphLaunch(c->entries.back().exec, st);
}

}  // namespace mapk
