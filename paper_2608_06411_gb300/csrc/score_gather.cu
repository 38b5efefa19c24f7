// Eq. 3 softmax-mean scores, squared row norms, and the compaction gather.
#include <algorithm>

#include "kernels.h"
#include "ptx.cuh"

namespace mapk {

namespace {

// ------------------------------------------------------------------ squared norms
// One warp per row; 16-byte loads; fp32 accumulation in a fixed order.
__global__ void row_sqnorm_kernel(const uint4* __restrict__ x, long long rows, int vec_per_row,
                                  float* __restrict__ out) {
  const long long row = static_cast<long long>(blockIdx.x) * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= rows) return;
  const uint4* p = x + row * vec_per_row;
  float acc = 0.f;
  for (int v = lane; v < vec_per_row; v += 32) {
    const uint4 u = __ldg(p + v);
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float lo = __uint_as_float(w[i] << 16), hi = __uint_as_float(w[i] & 0xFFFF0000u);
      acc = fmaf(lo, lo, acc);
      acc = fmaf(hi, hi, acc);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if (lane == 0) out[row] = acc;
}

// ------------------------------------------------------------------ gather
// out[b, j, :] = V[b, idx[b, j], :]; one CTA per output row, uint4 copies.
__global__ void gather_rows_kernel(const uint4* __restrict__ V, const int32_t* __restrict__ idx, int N, int k,
                                   int vec_per_row, uint4* __restrict__ out, int* status) {
  const long long r = blockIdx.x;           // b * k + j
  const long long b = r / k;
  const int src = __ldg(idx + r);
  if (src < 0 || src >= N) {
    if (threadIdx.x == 0) atomicOr(status, ST_BADINDEX);
    return;
  }
  const uint4* s = V + (b * N + src) * vec_per_row;
  uint4* d = out + r * vec_per_row;
  for (int v = threadIdx.x; v < vec_per_row; v += blockDim.x) d[v] = __ldg(s + v);
}

// ------------------------------------------------------------------ Eq. 3
// Pass 1: per query m and key split, running max / sum of exp over the split's keys.
// Thread = one query (q_m in registers); keys staged through shared memory in tiles.
template <int DP>
__global__ void __launch_bounds__(128) score_stats_kernel(const float* __restrict__ q, const float* __restrict__ k,
                                                          const int* __restrict__ q_off, int N, int nsplit,
                                                          float scale, float2* __restrict__ stats) {
  constexpr int KT = 32;
  __shared__ float4 ks[KT * DP / 4];
  const int b = blockIdx.z, split = blockIdx.y;
  const int m0 = q_off[b], M = q_off[b + 1] - m0;
  const int m = blockIdx.x * 128 + threadIdx.x;
  if (blockIdx.x * 128 >= M) return;
  const bool active = m < M;
  float qr[DP];
  {
    const float4* qp = reinterpret_cast<const float4*>(q + static_cast<long long>(m0 + (active ? m : 0)) * DP);
#pragma unroll
    for (int i = 0; i < DP / 4; ++i) {
      const float4 v = __ldg(qp + i);
      qr[4 * i] = v.x * scale; qr[4 * i + 1] = v.y * scale; qr[4 * i + 2] = v.z * scale; qr[4 * i + 3] = v.w * scale;
    }
  }
  const int per = (N + nsplit - 1) / nsplit;
  const int n_beg = split * per, n_end = min(N, n_beg + per);
  float mx = -INFINITY, sm = 0.f;
  const float4* kb = reinterpret_cast<const float4*>(k + static_cast<long long>(b) * N * DP);
  for (int t0 = n_beg; t0 < n_end; t0 += KT) {
    const int cnt = min(KT, n_end - t0);
    __syncthreads();
    for (int i = threadIdx.x; i < cnt * DP / 4; i += 128) ks[i] = __ldg(kb + static_cast<long long>(t0) * (DP / 4) + i);
    __syncthreads();
    for (int j = 0; j < cnt; ++j) {
      float l0 = 0.f, l1 = 0.f, l2 = 0.f, l3 = 0.f;
#pragma unroll
      for (int i = 0; i < DP / 4; ++i) {
        const float4 kv = ks[j * (DP / 4) + i];
        l0 = fmaf(qr[4 * i], kv.x, l0);
        l1 = fmaf(qr[4 * i + 1], kv.y, l1);
        l2 = fmaf(qr[4 * i + 2], kv.z, l2);
        l3 = fmaf(qr[4 * i + 3], kv.w, l3);
      }
      const float l = (l0 + l1) + (l2 + l3);
      if (l > mx) { sm = sm * expf(mx - l) + 1.f; mx = l; }
      else sm += expf(l - mx);
    }
  }
  if (active) stats[static_cast<long long>(m0 + m) * nsplit + split] = make_float2(mx, sm);
}

// Pass 2: thread = one key n (k_n in registers); loops over the image's queries with
// their combined (max, 1/sum) and accumulates p_hat_n = (1/M) sum_m exp(l_mn - max_m) / sum_m.
template <int DP>
__global__ void __launch_bounds__(128) score_mean_kernel(const float* __restrict__ q, const float* __restrict__ k,
                                                         const int* __restrict__ q_off, int N, int nsplit,
                                                         float scale, const float2* __restrict__ stats,
                                                         float* __restrict__ scores) {
  constexpr int QT = 32;
  __shared__ float4 qs[QT * DP / 4];
  __shared__ float2 qn[QT];          // (max_m, 1 / sum_m)
  const int b = blockIdx.y;
  const int n = blockIdx.x * 128 + threadIdx.x;
  const bool active = n < N;
  const int m0 = q_off[b], M = q_off[b + 1] - m0;
  float kr[DP];
  {
    const float4* kp = reinterpret_cast<const float4*>(k + (static_cast<long long>(b) * N + (active ? n : 0)) * DP);
#pragma unroll
    for (int i = 0; i < DP / 4; ++i) {
      const float4 v = __ldg(kp + i);
      kr[4 * i] = v.x; kr[4 * i + 1] = v.y; kr[4 * i + 2] = v.z; kr[4 * i + 3] = v.w;
    }
  }
  float acc = 0.f;
  for (int t0 = 0; t0 < M; t0 += QT) {
    const int cnt = min(QT, M - t0);
    __syncthreads();
    const float4* qp = reinterpret_cast<const float4*>(q + static_cast<long long>(m0 + t0) * DP);
    for (int i = threadIdx.x; i < cnt * DP / 4; i += 128) {
      float4 v = __ldg(qp + i);
      v.x *= scale; v.y *= scale; v.z *= scale; v.w *= scale;
      qs[i] = v;
    }
    if (threadIdx.x < cnt) {
      const float2* st = stats + static_cast<long long>(m0 + t0 + threadIdx.x) * nsplit;
      float mx = -INFINITY;
      for (int s = 0; s < nsplit; ++s) mx = fmaxf(mx, st[s].x);
      float sm = 0.f;
      for (int s = 0; s < nsplit; ++s) {
        const float2 v = st[s];
        if (v.y > 0.f) sm += v.y * expf(v.x - mx);
      }
      qn[threadIdx.x] = make_float2(mx, 1.f / sm);
    }
    __syncthreads();
    for (int j = 0; j < cnt; ++j) {
      float l0 = 0.f, l1 = 0.f, l2 = 0.f, l3 = 0.f;
#pragma unroll
      for (int i = 0; i < DP / 4; ++i) {
        const float4 qv = qs[j * (DP / 4) + i];
        l0 = fmaf(qv.x, kr[4 * i], l0);
        l1 = fmaf(qv.y, kr[4 * i + 1], l1);
        l2 = fmaf(qv.z, kr[4 * i + 2], l2);
        l3 = fmaf(qv.w, kr[4 * i + 3], l3);
      }
      const float l = (l0 + l1) + (l2 + l3);
      const float2 st = qn[j];
      acc += expf(l - st.x) * st.y;
    }
  }
  if (active) scores[static_cast<long long>(b) * N + n] = acc / static_cast<float>(M);
}

}  // namespace

cudaError_t launch_row_sqnorm(const void* x, long long rows, int D, float* out, cudaStream_t st) {
  if (rows <= 0) return cudaSuccess;
  if (D % 8 != 0) return cudaErrorInvalidValue;
  const int warps = 8;
  const long long blocks = (rows + warps - 1) / warps;
  row_sqnorm_kernel<<<static_cast<unsigned>(blocks), warps * 32, 0, st>>>(static_cast<const uint4*>(x), rows, D / 8,
                                                                          out);
  return cudaGetLastError();
}

cudaError_t launch_gather(const void* V, const int32_t* idx, int B, int N, int k, int D, void* out, int* status,
                          cudaStream_t st) {
  if (B <= 0 || k <= 0) return cudaSuccess;
  if (D % 8 != 0) return cudaErrorInvalidValue;
  const long long rows = static_cast<long long>(B) * k;
  gather_rows_kernel<<<static_cast<unsigned>(rows), 128, 0, st>>>(static_cast<const uint4*>(V), idx, N, k, D / 8,
                                                                   static_cast<uint4*>(out), status);
  return cudaGetLastError();
}

cudaError_t launch_scores(const ScoreDesc& d, cudaStream_t st) {
  const float scale = 1.0f / sqrtf(static_cast<float>(d.dp));
  dim3 g1((d.max_m + 127) / 128, d.nsplit, d.B);
  dim3 g2((d.N + 127) / 128, d.B);
  const float2* stats = reinterpret_cast<const float2*>(d.stats);
  if (d.dp == 128) {
    score_stats_kernel<128><<<g1, 128, 0, st>>>(d.q, d.k, d.q_off, d.N, d.nsplit, scale,
                                                reinterpret_cast<float2*>(d.stats));
    score_mean_kernel<128><<<g2, 128, 0, st>>>(d.q, d.k, d.q_off, d.N, d.nsplit, scale, stats, d.scores);
  } else if (d.dp == 64) {
    score_stats_kernel<64><<<g1, 128, 0, st>>>(d.q, d.k, d.q_off, d.N, d.nsplit, scale,
                                               reinterpret_cast<float2*>(d.stats));
    score_mean_kernel<64><<<g2, 128, 0, st>>>(d.q, d.k, d.q_off, d.N, d.nsplit, scale, stats, d.scores);
  } else {
    return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace mapk
