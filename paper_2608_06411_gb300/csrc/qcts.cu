// Question Contrastive Teacher Selection (section "Question Contrastive Teacher Selection",
// Eq. 1 and Eq. 2): from the text-to-vision attention maps of every language-model layer,
// for the sample's question and for the fixed reference question, the per-layer target
// distributions p^l and p_ref^l, their Jensen-Shannon divergence, and the teacher layer
// l* = argmax_l D_JS(p^l, p_ref^l).
//
// The work is one streaming read of the attention maps (hundreds of MB per sample for a
// 7B backbone), so it is HBM-bound; two launches:
//   1. qcts_colsum_kernel: Eq. 1 column sums.  A cluster of 8 CTAs splits the rows (head,
//      question token) of one (sample, layer, 512-column tile); each thread owns 8 adjacent
//      columns (one 16-byte load per row) and one of 4 row phases, with 8 rows in flight.
//      The 32 partial sums per column are added in a fixed order through distributed
//      shared memory (each CTA of the cluster finishes 1/8 of the columns), so results do
//      not depend on scheduling and no global scratch or atomics are needed.
//   2. qcts_finish_kernel: one CTA per (sample, layer): l1 normalisation of both aggregates
//      in place and the divergence; the last CTA of each sample to finish takes the argmax
//      over layers (ties to the lower layer) and copies p^{l*}.
#include <algorithm>
#include <cmath>
#include <cstdint>
#include <memory>
#include <new>

#include "../../include/map_gb300.h"
#include "ptx.cuh"

namespace mapk {
namespace {

constexpr int kThreads = 256;
constexpr int kColGroups = 64;                  // threads across the columns of a tile
constexpr int kPhases = kThreads / kColGroups;  // threads down the rows
constexpr int kCluster = 8;                     // CTAs splitting the rows of one tile
constexpr int kUnroll = 8;                      // rows in flight per thread
constexpr int kMaxSamples = 1024;               // samples per launch (kernel-parameter table)

struct QctsMeta {
  int b0, count;       // global index of the first sample of this launch, samples in it
  int L, H, N, m_ref;
  int32_t lens[kMaxSamples];
  long long row0[kMaxSamples];   // first row (of N elements) of each sample's question block
};

template <int VEC> struct Load;
template <> struct Load<8> {
  using T = uint4;
  static __device__ __forceinline__ T get(const uint16_t* p) { return __ldcs(reinterpret_cast<const uint4*>(p)); }
  static __device__ __forceinline__ void add(const T& u, float* acc) {
    acc[0] += __uint_as_float(u.x << 16);
    acc[1] += __uint_as_float(u.x & 0xFFFF0000u);
    acc[2] += __uint_as_float(u.y << 16);
    acc[3] += __uint_as_float(u.y & 0xFFFF0000u);
    acc[4] += __uint_as_float(u.z << 16);
    acc[5] += __uint_as_float(u.z & 0xFFFF0000u);
    acc[6] += __uint_as_float(u.w << 16);
    acc[7] += __uint_as_float(u.w & 0xFFFF0000u);
  }
};
template <> struct Load<2> {
  using T = unsigned int;
  static __device__ __forceinline__ T get(const uint16_t* p) {
    return __ldcs(reinterpret_cast<const unsigned int*>(p));
  }
  static __device__ __forceinline__ void add(const T& u, float* acc) {
    acc[0] += __uint_as_float(u << 16);
    acc[1] += __uint_as_float(u & 0xFFFF0000u);
  }
};
template <> struct Load<1> {
  using T = unsigned short;
  static __device__ __forceinline__ T get(const uint16_t* p) { return __ldcs(p); }
  static __device__ __forceinline__ void add(const T& u, float* acc) {
    acc[0] += __uint_as_float(static_cast<uint32_t>(u) << 16);
  }
};

// acc += rows p, p + stride, ... (n of them), kUnroll loads issued before their adds.
template <int VEC>
__device__ __forceinline__ void add_rows(const uint16_t* p, long long stride, long long n, float* acc) {
  using L = Load<VEC>;
  long long i = 0;
  for (; i + kUnroll <= n; i += kUnroll) {
    typename L::T x[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) x[u] = L::get(p + u * stride);
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) L::add(x[u], acc);
    p += kUnroll * stride;
  }
  for (; i < n; ++i, p += stride) L::add(L::get(p), acc);
}

__device__ __forceinline__ float ld_shared_cluster_f32(uint32_t addr) {
  float v;
  asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(addr) : "memory");
  return v;
}

// Eq. 1 for one (sample, layer, column tile): a[n] = 1/(H M) sum_{h, m} A[h, m, n] for the
// question (into a_out) and 1/(H M_ref) sum for the reference question (into aref_out).
// Grid (kCluster, column tiles, samples * L); cluster (kCluster, 1, 1).  No thread returns
// before the two cluster barriers.
template <int VEC>
__global__ void __launch_bounds__(kThreads, 3) qcts_colsum_kernel(const __grid_constant__ QctsMeta m,
                                                               const uint16_t* __restrict__ attn,
                                                               const uint16_t* __restrict__ ref,
                                                               float* __restrict__ a_out,
                                                               float* __restrict__ aref_out,
                                                               int32_t* __restrict__ teacher) {
  constexpr int W = kColGroups * VEC;       // columns per tile
  constexpr int kPer = W / kCluster;        // columns each CTA finishes
  __shared__ float part[2][kPhases][W];
  pdl_enter();
  const int rank = static_cast<int>(cluster_ctarank());
  const int tile = blockIdx.y;
  const int bl = blockIdx.z / m.L, l = blockIdx.z - bl * m.L;
  const long long b = m.b0 + bl;
  const int N = m.N;
  const int cg = threadIdx.x % kColGroups, ph = threadIdx.x / kColGroups;
  const long long col = static_cast<long long>(tile) * W + cg * VEC;
  if (rank == 0 && tile == 0 && l == 0 && threadIdx.x == 0) teacher[b] = 0;   // finish-kernel counter

  float acc_q[VEC], acc_r[VEC];
#pragma unroll
  for (int v = 0; v < VEC; ++v) acc_q[v] = acc_r[v] = 0.f;
  if (col < N) {   // N % VEC == 0: the whole group is inside the row
    const long long Rq = static_cast<long long>(m.H) * m.lens[bl];
    const long long q_begin = Rq * rank / kCluster, q_end = Rq * (rank + 1) / kCluster;
    const long long nq = q_end - q_begin - ph > 0 ? (q_end - q_begin - ph + kPhases - 1) / kPhases : 0;
    const uint16_t* pq = attn + (m.row0[bl] + l * Rq + q_begin + ph) * N + col;
    add_rows<VEC>(pq, static_cast<long long>(kPhases) * N, nq, acc_q);

    const long long Rr = static_cast<long long>(m.H) * m.m_ref;
    const long long r_begin = Rr * rank / kCluster, r_end = Rr * (rank + 1) / kCluster;
    const long long nr = r_end - r_begin - ph > 0 ? (r_end - r_begin - ph + kPhases - 1) / kPhases : 0;
    const uint16_t* pr = ref + ((b * m.L + l) * Rr + r_begin + ph) * N + col;
    add_rows<VEC>(pr, static_cast<long long>(kPhases) * N, nr, acc_r);
  }
#pragma unroll
  for (int v = 0; v < VEC; ++v) {
    part[0][ph][cg * VEC + v] = acc_q[v];
    part[1][ph][cg * VEC + v] = acc_r[v];
  }
  cluster_sync();   // every CTA's partials are written

  const int Mb = m.lens[bl];
  const float scale_q = Mb > 0 ? 1.0f / (static_cast<float>(m.H) * static_cast<float>(Mb)) : 0.f;
  const float scale_r = 1.0f / (static_cast<float>(m.H) * static_cast<float>(m.m_ref));
  for (int i = threadIdx.x; i < 2 * kPer; i += kThreads) {
    const int which = i / kPer;
    const int c = rank * kPer + (i - which * kPer);
    float s = 0.f;
    for (int src = 0; src < kCluster; ++src) {
#pragma unroll
      for (int p = 0; p < kPhases; ++p) s += ld_shared_cluster_f32(mapa_u32(&part[which][p][c], src));
    }
    const long long gcol = static_cast<long long>(tile) * W + c;
    if (gcol < N) {
      float* out = which ? aref_out : a_out;
      out[(b * m.L + l) * N + gcol] = s * (which ? scale_r : scale_q);
    }
  }
  cluster_sync();   // no CTA leaves while a peer may still read its shared memory
}

// Deterministic block sum of two values (256 threads): warp trees, then warp 0 in order.
__device__ __forceinline__ float2 block_sum2(float x, float y, float2* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    x += __shfl_xor_sync(0xffffffffu, x, o);
    y += __shfl_xor_sync(0xffffffffu, y, o);
  }
  const int w = threadIdx.x >> 5;
  if ((threadIdx.x & 31) == 0) red[w] = make_float2(x, y);
  __syncthreads();
  if (threadIdx.x == 0) {
    float2 s = red[0];
    for (int i = 1; i < kThreads / 32; ++i) {
      s.x += red[i].x;
      s.y += red[i].y;
    }
    red[kThreads / 32] = s;
  }
  __syncthreads();
  const float2 r = red[kThreads / 32];
  __syncthreads();   // red may be reused
  return r;
}

// phi(d) = (1 + d) ln(1 + d) + (1 - d) ln(1 - d) >= 0, so that with m = (p + q)/2 and
// d = (p - q)/(p + q):  p ln(p/m) + q ln(q/m) = m phi(d).  For |d| < 1/4 the even power
// series phi(d) = sum_k d^(2k) / (k (2k - 1)) (six terms, truncation below 1e-9 relative)
// avoids the cancellation of the two logarithms when p is close to q.
__device__ __forceinline__ float js_phi(float d) {
  const float u = d * d;
  if (u < 0.0625f) {
    return u * (1.0f + u * (1.0f / 6.0f + u * (1.0f / 15.0f + u * (1.0f / 28.0f + u * (1.0f / 45.0f + u * (1.0f / 66.0f))))));
  }
  const float a = (1.0f + d) * log1pf(d);
  const float c = (1.0f - d) > 0.f ? (1.0f - d) * log1pf(-d) : 0.f;
  return a + c;
}

__device__ __forceinline__ float js_term(float pn, float qn) {
  const float t = pn + qn;
  return t > 0.f ? 0.5f * t * js_phi((pn - qn) / t) : 0.f;
}

// One CTA per (sample, layer): p = a / sum(a) (uniform when the sum is zero) for the
// question and the reference, written in place, and js = D_JS(p, p_ref) in nats.  The last
// CTA of a sample to finish (counted in teacher[b], zeroed by the column-sum kernel) takes
// l* = argmax_l js (ties to the lower layer), writes it over the count and copies p^{l*} to
// teacher_p.  V4: N % 4 == 0 and 16-byte aligned rows (float4 accesses).
template <bool V4>
__global__ void __launch_bounds__(kThreads) qcts_finish_kernel(int L, int N, int b0, float* __restrict__ p,
                                                               float* __restrict__ pref, float* __restrict__ js,
                                                               int32_t* __restrict__ teacher,
                                                               float* __restrict__ teacher_p) {
  __shared__ float2 red[kThreads / 32 + 1];
  __shared__ int last;
  pdl_enter();
  const long long b = b0 + blockIdx.y;
  const long long row = b * L + blockIdx.x;
  float* a = p + row * N;
  float* r = pref + row * N;
  const float inv_n = 1.0f / static_cast<float>(N);
  float acc = 0.f;
  if (V4) {
    const int n4 = N / 4;
    float4* a4 = reinterpret_cast<float4*>(a);
    float4* r4 = reinterpret_cast<float4*>(r);
    float sa = 0.f, sr = 0.f;
    for (int i = threadIdx.x; i < n4; i += kThreads) {
      const float4 x = a4[i], y = r4[i];
      sa += (x.x + x.y) + (x.z + x.w);
      sr += (y.x + y.y) + (y.z + y.w);
    }
    const float2 s = block_sum2(sa, sr, red);
    const bool ua = !(s.x > 0.f), ur = !(s.y > 0.f);
    for (int i = threadIdx.x; i < n4; i += kThreads) {
      const float4 x = a4[i], y = r4[i];
      const float4 pn = ua ? make_float4(inv_n, inv_n, inv_n, inv_n)
                           : make_float4(x.x / s.x, x.y / s.x, x.z / s.x, x.w / s.x);
      const float4 qn = ur ? make_float4(inv_n, inv_n, inv_n, inv_n)
                           : make_float4(y.x / s.y, y.y / s.y, y.z / s.y, y.w / s.y);
      a4[i] = pn;
      r4[i] = qn;
      acc += (js_term(pn.x, qn.x) + js_term(pn.y, qn.y)) + (js_term(pn.z, qn.z) + js_term(pn.w, qn.w));
    }
  } else {
    float sa = 0.f, sr = 0.f;
    for (int n = threadIdx.x; n < N; n += kThreads) {
      sa += a[n];
      sr += r[n];
    }
    const float2 s = block_sum2(sa, sr, red);
    const bool ua = !(s.x > 0.f), ur = !(s.y > 0.f);
    for (int n = threadIdx.x; n < N; n += kThreads) {
      const float pn = ua ? inv_n : a[n] / s.x;
      const float qn = ur ? inv_n : r[n] / s.y;
      a[n] = pn;
      r[n] = qn;
      acc += js_term(pn, qn);
    }
  }
  __threadfence();   // this thread's p, p_ref writes are visible before the sample's count moves
  const float2 tot = block_sum2(acc, 0.f, red);
  if (threadIdx.x == 0) {
    js[row] = 0.5f * tot.x;
    __threadfence();
    last = atomicAdd(teacher + b, 1) == L - 1;
  }
  __syncthreads();
  if (!last) return;
  __threadfence();
  __shared__ int best_l;
  if (threadIdx.x < 32) {
    float bv = -INFINITY;
    int bi = 0x7fffffff;
    for (int l = threadIdx.x; l < L; l += 32) {
      const float v = __ldcg(js + b * L + l);
      if (v > bv) {   // l increases within a lane: a later equal value never wins
        bv = v;
        bi = l;
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
      const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
      if (ov > bv || (ov == bv && oi < bi)) {
        bv = ov;
        bi = oi;
      }
    }
    if (threadIdx.x == 0) {
      best_l = bi < L ? bi : 0;
      teacher[b] = best_l;
    }
  }
  __syncthreads();
  if (teacher_p != nullptr) {
    const float* src = p + (b * L + best_l) * N;
    for (int n = threadIdx.x; n < N; n += kThreads) teacher_p[b * N + n] = __ldcg(src + n);
  }
}

template <typename... KParams, typename... Args>
cudaError_t launch_cluster(void (*kern)(KParams...), dim3 grid, dim3 block, unsigned cx, cudaStream_t st,
                           Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = 0;
  cfg.stream = st;
  cudaLaunchAttribute at[2];
  at[0].id = cudaLaunchAttributeClusterDimension;
  at[0].val.clusterDim.x = cx;
  at[0].val.clusterDim.y = 1;
  at[0].val.clusterDim.z = 1;
  at[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...);
}

template <int VEC>
cudaError_t launch_colsum(const QctsMeta& m, const void* attn, const void* ref, float* p, float* pref,
                          int32_t* teacher, cudaStream_t st) {
  constexpr int W = kColGroups * VEC;
  const dim3 grid(kCluster, (m.N + W - 1) / W, m.count * m.L);
  return launch_cluster(qcts_colsum_kernel<VEC>, grid, dim3(kThreads), kCluster, st, m,
                        static_cast<const uint16_t*>(attn), static_cast<const uint16_t*>(ref), p, pref, teacher);
}

}  // namespace
}  // namespace mapk

extern "C" int map_qcts(const void* attn, const int32_t* lens, const void* attn_ref, int M_ref, int B, int L, int H,
                        int N, float* p, float* p_ref, float* js, int32_t* teacher, float* teacher_p, void* stream) {
  using namespace mapk;
  if (!attn || !lens || !attn_ref || !p || !p_ref || !js || !teacher) return MAP_EINVAL;
  if (B < 1 || L < 1 || H < 1 || N < 1 || M_ref < 1) return MAP_EINVAL;
  if (L > 65535 || (static_cast<long long>(N) + kColGroups - 1) / kColGroups > 65535) return MAP_EUNSUPPORTED;
  for (int b = 0; b < B; ++b)
    if (lens[b] < 0) return MAP_EINVAL;
  const uintptr_t ua = reinterpret_cast<uintptr_t>(attn), ur = reinterpret_cast<uintptr_t>(attn_ref);
  if ((ua | ur) & 1u) return MAP_EINVAL;
  int vec = 1;
  if (N % 8 == 0 && ((ua | ur) & 15u) == 0) vec = 8;
  else if (N % 2 == 0 && ((ua | ur) & 3u) == 0) vec = 2;
  const bool v4 = N % 4 == 0 && ((reinterpret_cast<uintptr_t>(p) | reinterpret_cast<uintptr_t>(p_ref)) & 15u) == 0;
  cudaStream_t st = static_cast<cudaStream_t>(stream);

  // samples per launch: the parameter table and gridDim.z = samples * L
  const int per_launch = std::max(1, std::min(kMaxSamples, 65535 / L));
  std::unique_ptr<QctsMeta> mp(new (std::nothrow) QctsMeta);   // ~12 KB, copied into the launch parameters
  if (!mp) return MAP_ENOMEM;
  QctsMeta& m = *mp;
  long long row = 0;
  for (int b0 = 0; b0 < B; b0 += per_launch) {
    m.b0 = b0;
    m.count = std::min(per_launch, B - b0);
    m.L = L;
    m.H = H;
    m.N = N;
    m.m_ref = M_ref;
    for (int i = 0; i < m.count; ++i) {
      m.lens[i] = lens[b0 + i];
      m.row0[i] = row;
      row += static_cast<long long>(L) * H * lens[b0 + i];
    }
    cudaError_t e = vec == 8 ? launch_colsum<8>(m, attn, attn_ref, p, p_ref, teacher, st)
                  : vec == 2 ? launch_colsum<2>(m, attn, attn_ref, p, p_ref, teacher, st)
                             : launch_colsum<1>(m, attn, attn_ref, p, p_ref, teacher, st);
    if (e == cudaSuccess)
      e = v4 ? launch_k(qcts_finish_kernel<true>, dim3(L, m.count), dim3(kThreads), 0, st, L, N, b0, p, p_ref, js,
                        teacher, teacher_p)
             : launch_k(qcts_finish_kernel<false>, dim3(L, m.count), dim3(kThreads), 0, st, L, N, b0, p, p_ref,
                        js, teacher, teacher_p);
    if (e != cudaSuccess) {
      cudaGetLastError();
      return e == cudaErrorInvalidValue ? MAP_EINVAL : MAP_ECUDA;
    }
  }
  return MAP_OK;
}
