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

// k-th largest of n distinct 64-bit keys in shared memory (1 <= k <= n): MSB-first radix
// select, 8 bits per pass.  Lanes of a warp that hit the same bin add their count once
// (__match_any_sync), so bins shared by most keys (a common exponent) are not a
// serialisation point; one warp finds the bin with a shuffle scan.
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
// U = p_hat * ||v||^lambda, r2 = ||v||^2, nothing cached; R0 = top-K0 by p_hat, in order.
__global__ void __launch_bounds__(1024) sel_init_kernel(SelState s) {
  extern __shared__ uint64_t sh64[];
  const int b = blockIdx.x;
  const long long base = static_cast<long long>(b) * s.N;
  __shared__ uint32_t hist[256], bc[2];
  __shared__ int cnt;
  for (int i = threadIdx.x; i < s.N; i += blockDim.x) {
    const float p = s.scores[base + i], sq = s.sqn ? s.sqn[base + i] : 0.f;
    s.U[base + i] = sel_value(p, sq, sq, s.lambda, s.tau);
    s.r2[base + i] = sq;
    s.cstep[base + i] = 0;
    s.state[base + i] = 0;
    sh64[i] = make_key(p, i);
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
    for (int i = s.K0 + threadIdx.x; i < cap; i += blockDim.x) sel[i] = 0ull;
    __syncthreads();
    block_sort_desc(sel, cap);
    for (int i = threadIdx.x; i < s.K0; i += blockDim.x) s.r0[static_cast<long long>(b) * s.K + i] = key_index(sel[i]);
  }
}

// ------------------------------------------------------------------ choose
// Active set of the next round: the next R0 chunk (forced), else the S candidates with the
// largest bound U (value descending, ties to the lower index) and theta = the next key.
__global__ void __launch_bounds__(1024) sel_choose_kernel(SelState s) {
  extern __shared__ uint64_t sh64[];
  const int b = blockIdx.x;
  const long long base = static_cast<long long>(b) * s.N;
  const int S = s.S;
  int32_t* aslot = s.aslot + static_cast<long long>(b) * S;
  if (s.done[b]) {
    if (threadIdx.x == 0) s.nlimit[b] = 0;
    return;
  }
  const int np = s.npicks[b], nb = s.nbasis[b];
  uint64_t theta = 0;
  int mode;
  if (np < s.K0) {
    const int na = min(S, s.K0 - np);
    for (int i = threadIdx.x; i < S; i += blockDim.x)
      aslot[i] = i < na ? s.r0[static_cast<long long>(b) * s.K + np + i] : -1;
    mode = 1;
  } else {
    __shared__ uint32_t hist[256], bc[2];
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
    s.nlimit[b] = S + nb - s.gbase[b];
    s.gb_lo[b] = s.nb_gathered[b];
    s.gb_hi[b] = nb;
    s.nb_gathered[b] = nb;
  }
}

// Copies the rows the Gram block needs into Vg: row r < S <- token aslot[r];
// row S + beta - gbase <- basis token beta for the basis vectors added since the last round.
// kGatherCtas CTAs per image, each walking every kGatherCtas-th row; finished images exit.
constexpr int kGatherCtas = 64;

__global__ void __launch_bounds__(128) sel_gather_kernel(SelState s) {
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
    const uint4* V = reinterpret_cast<const uint4*>(s.V) + (static_cast<long long>(b) * s.N + src) * vec;
    uint4* dst = reinterpret_cast<uint4*>(s.Vg) + (static_cast<long long>(b) * s.R + r) * vec;
    for (int c = threadIdx.x; c < vec; c += blockDim.x) dst[c] = __ldg(V + c);
  }
}

// ------------------------------------------------------------------ greedy
// One CTA of S threads per image; thread = active slot.
//
// The coordinates of the active tokens live in E during the round: shared memory laid out
// [KP][S] when it fits (SMEM = true), else the tokens' global cache rows.
// Phase 1 brings every active token's coordinates up to the current basis by forward
// substitution, 32 basis vectors at a time: the 32 rows of L (the basis tokens' own
// coordinate rows) are staged in shared memory and the 32 results accumulate in registers.
// Phase 2 makes the picks with one block barrier per pick: the winning slot is carried in
// the low bits of the key, and every slot's residual is published in shared memory, so
// all threads derive the basis update from the same values.  Phase 3 writes back.
constexpr int kChunk = 32;

template <bool SMEM>
struct Coords {
  float* Es;            // SMEM: [KP][S]
  float* Ec;            // global cache rows
  long long base;
  int S, KP;
  __device__ __forceinline__ float* at(int slot, int tok, int q) const {
    if constexpr (SMEM) return Es + static_cast<long long>(q) * S + slot;
    else return Ec + (base + tok) * KP + q;
  }
};

// key of a candidate inside the round: (value bits, 0xFFFF - token, slot); the upper 48
// bits order like make_key (value descending, lower token first).
__device__ __forceinline__ uint64_t slot_key(float v, int tok, int slot) {
  const float c = v > 0.f ? v : 0.f;
  return (static_cast<uint64_t>(__float_as_uint(c)) << 32) | (static_cast<uint64_t>(0xFFFFu - tok) << 16) |
         static_cast<uint64_t>(slot);
}
__device__ __forceinline__ uint64_t theta48(uint64_t theta) {   // make_key -> upper 48 bits of slot_key
  if (theta == 0) return 0;
  const uint32_t tok = static_cast<uint32_t>(key_index(theta));
  return ((theta >> 32) << 16) | (0xFFFFu - tok);
}

template <bool SMEM>
__global__ void __launch_bounds__(256, 1) sel_greedy_kernel(SelState s) {
  extern __shared__ __align__(16) float shf[];
  __shared__ uint64_t wkey[2][32];
  __shared__ float sh_rinv_chunk[kChunk];
  const int b = blockIdx.x;
  if (s.done[b]) return;
  const int S = s.S, R = s.R, KP = s.KP;
  float* Lc = shf;                                   // [kChunk][KP]
  float* r2s = shf + kChunk * KP;                    // [S] published residuals
  float* sqs = r2s + S;                              // [S]
  int32_t* tks = reinterpret_cast<int32_t*>(sqs + S);   // [S] tokens of the slots
  Coords<SMEM> E{reinterpret_cast<float*>(tks + S), s.Ec, static_cast<long long>(b) * s.N, S, KP};
  const long long base = E.base;
  const int slot = threadIdx.x;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
  const int tok = s.aslot[static_cast<long long>(b) * S + slot];
  const int32_t* btok = s.basis_tok + static_cast<long long>(b) * s.K;
  const float* rnorm = s.rnorm + static_cast<long long>(b) * s.K;
  const float* Gb = s.G + static_cast<long long>(b) * S * R;
  const float* Gr = Gb + static_cast<long long>(slot) * R;
  int nb = s.nbasis[b], np = s.npicks[b];
  const int gbase = s.gbase[b];
  const bool forced = s.mode[b] == 1;
  const uint64_t th48 = theta48(s.theta[b]);

  float r2 = 0.f, sq = 0.f, p = 0.f, val = 0.f;
  int c0 = nb, mine = nb;                            // cached coordinates; valid coordinates at the end
  bool alive = false;
  if (tok >= 0) {
    p = s.scores[base + tok];
    alive = s.state[base + tok] == 0;
    c0 = min(s.cstep[base + tok], nb);
    if (s.diag_sq && c0 == 0) {
      sq = r2 = Gr[slot];                            // <v, v> from the Gram block
    } else {
      r2 = s.r2[base + tok];
      sq = s.sqn[base + tok];
    }
    if constexpr (SMEM) {
      const float4* g = reinterpret_cast<const float4*>(s.Ec + (base + tok) * KP);
      int q = 0;
      for (; q + 16 <= c0; q += 16) {
        float4 v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) v[u] = g[q / 4 + u];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          *E.at(slot, tok, q + 4 * u) = v[u].x; *E.at(slot, tok, q + 4 * u + 1) = v[u].y;
          *E.at(slot, tok, q + 4 * u + 2) = v[u].z; *E.at(slot, tok, q + 4 * u + 3) = v[u].w;
        }
      }
      for (; q < c0; ++q) *E.at(slot, tok, q) = s.Ec[(base + tok) * KP + q];
    }
  }
  tks[slot] = tok;

  // ---- phase 1: forward substitution, chunk by chunk
  for (int b0 = 0; b0 < nb; b0 += kChunk) {
    const int b1 = min(nb, b0 + kChunk);
    __syncthreads();
    {
      const int KV = KP / 4, nvec = (b1 - b0) * KV;
      for (int t0 = threadIdx.x; t0 < nvec; t0 += 4 * blockDim.x) {
        float4 v[4];
        int qs[4], is[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int t = t0 + u * blockDim.x;
          is[u] = t / KV;
          qs[u] = (t - is[u] * KV) * 4;
          v[u] = t < nvec ? *reinterpret_cast<const float4*>(s.Ec + (base + btok[b0 + is[u]]) * KP + qs[u])
                          : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int t = t0 + u * blockDim.x;
          if (t < nvec) {
            const int lim = b0 + is[u];
            v[u].x = qs[u] < lim ? v[u].x : 0.f;
            v[u].y = qs[u] + 1 < lim ? v[u].y : 0.f;
            v[u].z = qs[u] + 2 < lim ? v[u].z : 0.f;
            v[u].w = qs[u] + 3 < lim ? v[u].w : 0.f;
            *reinterpret_cast<float4*>(Lc + is[u] * KP + qs[u]) = v[u];
          }
        }
      }
    }
    if (threadIdx.x < b1 - b0) sh_rinv_chunk[threadIdx.x] = 1.0f / rnorm[b0 + threadIdx.x];
    __syncthreads();
    if (tok < 0 || b1 <= c0) continue;
    float acc[kChunk], e[kChunk];
#pragma unroll
    for (int i = 0; i < kChunk; ++i) acc[i] = (b0 + i < b1 && b0 + i >= c0) ? Gr[S + b0 + i - gbase] : 0.f;
    for (int q = 0; q < b0; q += 4) {
      float4 eq;
      if constexpr (SMEM) {
        eq = make_float4(*E.at(slot, tok, q), *E.at(slot, tok, q + 1), *E.at(slot, tok, q + 2), *E.at(slot, tok, q + 3));
      } else {
        eq = *reinterpret_cast<const float4*>(E.at(slot, tok, q));
      }
#pragma unroll
      for (int i = 0; i < kChunk; ++i) {
        const float4 l = *reinterpret_cast<const float4*>(Lc + i * KP + q);
        acc[i] = fmaf(-l.x, eq.x, acc[i]);
        acc[i] = fmaf(-l.y, eq.y, acc[i]);
        acc[i] = fmaf(-l.z, eq.z, acc[i]);
        acc[i] = fmaf(-l.w, eq.w, acc[i]);
      }
    }
#pragma unroll
    for (int i = 0; i < kChunk; ++i) {
      const int beta = b0 + i;
      if (beta < b1) {
        if (beta >= c0) {
          float a = acc[i];
#pragma unroll
          for (int q = 0; q < i; ++q) a = fmaf(-Lc[i * KP + b0 + q], e[q], a);
          e[i] = a * sh_rinv_chunk[i];
          *E.at(slot, tok, beta) = e[i];
          r2 = fmaf(-e[i], e[i], r2);
        } else {
          e[i] = *E.at(slot, tok, beta);
        }
      }
    }
  }
  if (tok >= 0) val = sel_value(p, r2, sq, s.lambda, s.tau);
  r2s[slot] = r2;
  sqs[slot] = sq;

  // ---- phase 2: picks, one block barrier each
  for (int step = 0, buf = 0; np < s.K; ++step, buf ^= 1) {
    uint64_t key = alive ? slot_key(val, tok, slot) : 0ull;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const uint64_t other = __shfl_xor_sync(0xffffffffu, key, o);
      key = other > key ? other : key;
    }
    if (lane == 0) wkey[buf][warp] = key;
    __syncthreads();
    int jslot;
    if (forced) {
      jslot = step;
      if (jslot >= S || tks[jslot] < 0) break;
    } else {
      uint64_t best = lane < nwarps ? wkey[buf][lane] : 0ull;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const uint64_t other = __shfl_xor_sync(0xffffffffu, best, o);
        best = other > best ? other : best;
      }
      if (best == 0 || (best >> 16) <= th48) break;   // uniform
      jslot = static_cast<int>(best & 0xFFFFu);
    }
    const int jt = tks[jslot];
    const float r2j = r2s[jslot], sqj = sqs[jslot];
    const bool ext = (r2j > s.tau * sqj) && (r2j > 0.f);
    if (slot == jslot) {
      alive = false;
      mine = nb;
      s.state[base + jt] = 1;
      s.picks[static_cast<long long>(b) * s.K + np] = jt;
      if (ext) {
        s.basis_tok[static_cast<long long>(b) * s.K + nb] = jt;
        s.rnorm[static_cast<long long>(b) * s.K + nb] = sqrtf(r2j);
      }
    }
    if (ext) {
      if (alive) {
        const float rinv = 1.0f / sqrtf(r2j);
        float a0 = Gb[static_cast<long long>(jslot) * R + slot], a1 = 0.f, a2 = 0.f, a3 = 0.f;
        int q = 0;
        for (; q + 4 <= nb; q += 4) {
          a0 = fmaf(-*E.at(jslot, jt, q), *E.at(slot, tok, q), a0);
          a1 = fmaf(-*E.at(jslot, jt, q + 1), *E.at(slot, tok, q + 1), a1);
          a2 = fmaf(-*E.at(jslot, jt, q + 2), *E.at(slot, tok, q + 2), a2);
          a3 = fmaf(-*E.at(jslot, jt, q + 3), *E.at(slot, tok, q + 3), a3);
        }
        for (; q < nb; ++q) a0 = fmaf(-*E.at(jslot, jt, q), *E.at(slot, tok, q), a0);
        const float e = ((a0 + a1) + (a2 + a3)) * rinv;
        *E.at(slot, tok, nb) = e;
        r2 = fmaf(-e, e, r2);
        val = sel_value(p, r2, sq, s.lambda, s.tau);
        r2s[slot] = r2;
      }
      ++nb;
    }
    ++np;
  }
  // ---- phase 3: write back
  if (tok >= 0) {
    if (alive) mine = nb;
    if constexpr (SMEM) {
      float* g = s.Ec + (base + tok) * KP;
      for (int q = c0; q < mine; ++q) g[q] = *E.at(slot, tok, q);
    }
    s.cstep[base + tok] = mine;
    s.r2[base + tok] = r2;
    s.U[base + tok] = val;
  }
  if (threadIdx.x == 0) {
    s.nbasis[b] = nb;
    s.npicks[b] = np;
    if (np >= s.K) { s.done[b] = 1; atomicAdd(s.done_count, 1); }
  }
}

// ------------------------------------------------------------------ projection set-up
// After the R0 rounds: gather every R0 basis row (no active tokens) for the projection.
__global__ void sel_proj_prep_kernel(SelState s) {
  const int b = blockIdx.x;
  for (int i = threadIdx.x; i < s.S; i += blockDim.x) s.aslot[static_cast<long long>(b) * s.S + i] = -1;
  if (threadIdx.x == 0) {
    s.gb_lo[b] = s.nb_gathered[b];
    s.gb_hi[b] = s.nbasis[b];
    s.nb_gathered[b] = s.nbasis[b];
  }
}

__global__ void sel_proj_done_kernel(SelState s) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b < s.B) {
    s.gbase[b] = s.nbasis[b];
    s.nb_gathered[b] = s.nbasis[b];
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
size_t sel_greedy_smem(int KP, int S, bool* smem_coords) {
  const size_t lc = static_cast<size_t>(kChunk) * KP * 4 + static_cast<size_t>(S) * 12;
  const size_t es = static_cast<size_t>(KP) * S * 4;
  *smem_coords = lc + es <= 200 * 1024;
  return *smem_coords ? lc + es : lc;
}

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
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  sel_gather_kernel<<<dim3(kGatherCtas, s.B), 128, 0, st>>>(s);
  return cudaGetLastError();
}

cudaError_t launch_sel_greedy(const SelState& s, cudaStream_t st) {
  bool in_smem = false;
  const size_t sm = sel_greedy_smem(s.KP, s.S, &in_smem);
  cudaError_t e;
  if (in_smem) {
    e = cudaFuncSetAttribute(sel_greedy_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(sm));
    if (e != cudaSuccess) return e;
    sel_greedy_kernel<true><<<s.B, s.S, sm, st>>>(s);
  } else {
    e = cudaFuncSetAttribute(sel_greedy_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(sm));
    if (e != cudaSuccess) return e;
    sel_greedy_kernel<false><<<s.B, s.S, sm, st>>>(s);
  }
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

cudaError_t launch_sel_proj_prep(const SelState& s, cudaStream_t st) {
  sel_proj_prep_kernel<<<s.B, 256, 0, st>>>(s);
  return cudaGetLastError();
}

cudaError_t launch_sel_gather(const SelState& s, cudaStream_t st) {
  sel_gather_kernel<<<dim3(kGatherCtas, s.B), 128, 0, st>>>(s);
  return cudaGetLastError();
}

cudaError_t launch_sel_proj_done(const SelState& s, cudaStream_t st) {
  sel_proj_done_kernel<<<(s.B + 127) / 128, 128, 0, st>>>(s);
  return cudaGetLastError();
}

cudaError_t launch_sel_identity(int B, int N, int32_t* keep, int32_t* order, cudaStream_t st) {
  sel_identity_kernel<<<B, 256, 0, st>>>(N, keep, order);
  return cudaGetLastError();
}

}  // namespace mapk
