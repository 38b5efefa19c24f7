// Eq. 3 softmax statistics combine, weight folding, squared row norms, and the compaction gather.
#include <algorithm>

#include "kernels.h"
#include "ptx.cuh"

namespace mapk {

namespace {

// ------------------------------------------------------------------ squared norms
// One warp per row; 16-byte loads; fp32 accumulation in a fixed order.
__global__ void row_sqnorm_kernel(const uint4* __restrict__ x, long long rows, int vec_per_row,
                                  float* __restrict__ out) {
  pdl_enter();
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
  pdl_enter();
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

// (max, sum) partials of one column over all slabs -> (max + ln sum, 1/sum).  A block covers 32
// columns (threadIdx.x, coalesced) with kCombY threads per column splitting the slabs; the
// kCombY partial maxima and sums are combined in a fixed order in shared memory.
constexpr int kCombY = 8;
__global__ void __launch_bounds__(32 * kCombY) stats_combine_kernel(const float2* __restrict__ part, int nparts,
                                                                    int ld, const int* __restrict__ lens,
                                                                    float2* __restrict__ fin) {
  __shared__ float red[kCombY][32];
  pdl_enter();
  const int b = blockIdx.y, x = threadIdx.x, y = threadIdx.y, col = blockIdx.x * 32 + x;
  const bool on = col < lens[b];
  const float2* p = part + static_cast<long long>(b) * nparts * ld + col;
  float m = -INFINITY;
  if (on)
    for (int i = y; i < nparts; i += kCombY) m = fmaxf(m, p[static_cast<long long>(i) * ld].x);
  red[y][x] = m;
  __syncthreads();
  m = red[0][x];
#pragma unroll
  for (int j = 1; j < kCombY; ++j) m = fmaxf(m, red[j][x]);
  __syncthreads();
  float sum = 0.f;
  if (on)
    for (int i = y; i < nparts; i += kCombY) {
      const float2 v = p[static_cast<long long>(i) * ld];
      if (v.y > 0.f) sum += v.y * expf(v.x - m);
    }
  red[y][x] = sum;
  __syncthreads();
  if (y == 0 && on) {
    float s = red[0][x];
#pragma unroll
    for (int j = 1; j < kCombY; ++j) s += red[j][x];
    // one log-normaliser per column: exp(l - m) / s = exp(l - (m + ln s))
    fin[static_cast<long long>(b) * ld + col] = make_float2(m + logf(s), 1.0f / s);
  }
}

__global__ void sum_tiles_kernel(const float* __restrict__ part, int N, int n_tiles, long long total,
                                 float* __restrict__ scores) {
  pdl_enter();
  const long long i = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (i >= total) return;
  const long long b = i / N, n = i - b * N;
  float s = 0.f;
  for (int t = 0; t < n_tiles; ++t) s += part[(b * n_tiles + t) * N + n];
  scores[i] = s;
}

// out[p, i] (three bf16 segments) = sum_j Wp[p, j] W2[j, i]; thread = (p, i), fp64 sums.
__global__ void fold_weights_kernel(const __nv_bfloat16* __restrict__ Wp, const __nv_bfloat16* __restrict__ W2,
                                    const __nv_bfloat16* __restrict__ b2, int dp, int Dh,
                                    __nv_bfloat16* __restrict__ out, float* __restrict__ bias_out) {
  pdl_enter();
  const int i = blockIdx.x * blockDim.x + threadIdx.x, p = blockIdx.y;
  if (i < Dh) {
    double acc = 0.0;
    for (int j = 0; j < Dh; ++j)
      acc += static_cast<double>(__bfloat162float(Wp[static_cast<long long>(p) * Dh + j])) *
             static_cast<double>(__bfloat162float(W2[static_cast<long long>(j) * Dh + i]));
    const __nv_bfloat16 hi = __float2bfloat16_rn(static_cast<float>(acc));
    const __nv_bfloat16 lo = __float2bfloat16_rn(static_cast<float>(acc - static_cast<double>(__bfloat162float(hi))));
    __nv_bfloat16* row = out + static_cast<long long>(p) * 3 * Dh;
    row[i] = hi;
    row[Dh + i] = hi;
    row[2 * Dh + i] = lo;
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    double acc = 0.0;
    for (int j = 0; j < Dh; ++j)
      acc += static_cast<double>(__bfloat162float(Wp[static_cast<long long>(p) * Dh + j])) *
             static_cast<double>(__bfloat162float(b2[j]));
    bias_out[p] = static_cast<float>(acc);
  }
}

constexpr int kMetaImages = 1024;
struct MetaChunk {
  int b0, count, N, last, has_nv;
  int32_t lens[kMetaImages];
  int32_t offs[kMetaImages];
  int32_t nv[kMetaImages];       // valid visual tokens per image (has_nv), else N
};

// One CTA per image of the chunk.
__global__ void query_meta_kernel(const __grid_constant__ MetaChunk m, int32_t* __restrict__ off,
                                  int32_t* __restrict__ len, int32_t* __restrict__ pos,
                                  int32_t* __restrict__ nvalid) {
  pdl_enter();
  const int i = blockIdx.x, b = m.b0 + i;
  const int o = m.offs[i], l = m.lens[i];
  const int n = m.has_nv ? m.nv[i] : m.N;
  if (threadIdx.x == 0) {
    off[b] = o;
    len[b] = l;
    if (nvalid) nvalid[b] = n;
    if (m.last && i == m.count - 1) off[b + 1] = o + l;
  }
  for (int t = threadIdx.x; t < l; t += blockDim.x) pos[o + t] = n + t;
}

constexpr int kPutInts = 2048;
struct IntChunk {
  int n;
  int32_t v[kPutInts];
};

__global__ void put_ints_kernel(const __grid_constant__ IntChunk c, int32_t* __restrict__ dst) {
  pdl_enter();
  for (int i = threadIdx.x; i < c.n; i += blockDim.x) dst[i] = c.v[i];
}

constexpr int kAsmImages = 512;
struct AssembleChunk {
  int b0, count, N, k, pos_offset;
  int32_t lens[kAsmImages];
  int32_t nv[kAsmImages];           // valid visual tokens per image (N without padding)
  long long text_row[kAsmImages];   // first question row of each image in text_feats
  long long seq_row[kAsmImages];    // first row of each image's output sequence
};

// Hand-off sequence: row j of image b is kept token keep[b, j] (j < k) or question token
// j - k; one CTA per output row (grid: rows of the longest sequence in the chunk x images).
__global__ void assemble_kernel(const __grid_constant__ AssembleChunk m, const uint4* __restrict__ V,
                                const int32_t* __restrict__ idx, const uint4* __restrict__ T, int vec_per_row,
                                uint4* __restrict__ seq, int32_t* __restrict__ pos, int* status) {
  pdl_enter();
  const int i = blockIdx.y, j = blockIdx.x;
  const long long b = m.b0 + i;
  if (j >= m.k + m.lens[i]) return;
  const long long r = m.seq_row[i] + j;
  const int nv = m.nv[i];
  const uint4* src;
  int p;
  if (j < m.k) {
    const int t = __ldg(idx + b * m.k + j);
    if (t < 0 || t >= nv) {
      if (threadIdx.x == 0) {
        atomicOr(status, ST_BADINDEX);
        pos[r] = -1;
      }
      return;
    }
    src = V + (b * m.N + t) * vec_per_row;
    p = t;
  } else {
    src = T + (m.text_row[i] + (j - m.k)) * vec_per_row;
    p = nv + (j - m.k);
  }
  if (threadIdx.x == 0) pos[r] = p + m.pos_offset;
  uint4* d = seq + r * vec_per_row;
  for (int v = threadIdx.x; v < vec_per_row; v += blockDim.x) d[v] = __ldg(src + v);
}

__global__ void flags_to_host_kernel(const int32_t* a, const int* b, volatile int32_t* ah, volatile int* bh) {
  pdl_enter();
  *ah = *a;
  *bh = *b;
}

}  // namespace

cudaError_t launch_put_ints(const int32_t* host, int n, int32_t* dst, cudaStream_t st) {
  for (int i0 = 0; i0 < n; i0 += kPutInts) {
    IntChunk c;
    c.n = n - i0 < kPutInts ? n - i0 : kPutInts;
    for (int i = 0; i < c.n; ++i) c.v[i] = host[i0 + i];
    const cudaError_t e = launch_k(put_ints_kernel, dim3(1), dim3(256), 0, st, c, dst + i0);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

cudaError_t launch_query_meta(const int32_t* lens, const long long* offs, int B, int N, int32_t* off, int32_t* len,
                              int32_t* pos, const int32_t* nv, int32_t* nvalid, cudaStream_t st) {
  for (int b0 = 0; b0 < B; b0 += kMetaImages) {
    MetaChunk m;
    m.b0 = b0;
    m.count = B - b0 < kMetaImages ? B - b0 : kMetaImages;
    m.N = N;
    m.last = b0 + m.count == B;
    m.has_nv = nv != nullptr;
    for (int i = 0; i < m.count; ++i) {
      m.lens[i] = lens[b0 + i];
      m.offs[i] = static_cast<int32_t>(offs[b0 + i]);
      m.nv[i] = nv ? nv[b0 + i] : N;
    }
    const cudaError_t e = launch_k(query_meta_kernel, dim3(m.count), dim3(128), 0, st, m, off, len, pos, nvalid);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

cudaError_t launch_assemble(const void* V, const int32_t* idx, const void* T, const int32_t* lens, const int32_t* nv,
                            int B, int N, int k, int D, int pos_offset, void* seq, int32_t* pos, int* status,
                            cudaStream_t st) {
  if (D % 8 != 0) return cudaErrorInvalidValue;
  long long trow = 0, srow = 0;
  for (int b0 = 0; b0 < B; b0 += kAsmImages) {
    AssembleChunk m;
    m.b0 = b0;
    m.count = B - b0 < kAsmImages ? B - b0 : kAsmImages;
    m.N = N;
    m.k = k;
    m.pos_offset = pos_offset;
    int max_rows = 0;
    for (int i = 0; i < m.count; ++i) {
      m.lens[i] = lens[b0 + i];
      m.nv[i] = nv ? nv[b0 + i] : N;
      m.text_row[i] = trow;
      m.seq_row[i] = srow;
      trow += lens[b0 + i];
      srow += k + lens[b0 + i];
      max_rows = std::max(max_rows, k + lens[b0 + i]);
    }
    if (max_rows == 0) continue;
    const cudaError_t e = launch_k(assemble_kernel, dim3(max_rows, m.count), dim3(128), 0, st, m,
                                   static_cast<const uint4*>(V), idx, static_cast<const uint4*>(T), D / 8,
                                   static_cast<uint4*>(seq), pos, status);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

cudaError_t launch_flags_to_host(const int32_t* a, const int* b, int32_t* a_host_dev, int* b_host_dev, cudaStream_t st) {
  return launch_k(flags_to_host_kernel, dim3(1), dim3(1), 0, st, a, b, static_cast<volatile int32_t*>(a_host_dev),
                  static_cast<volatile int*>(b_host_dev));
}

cudaError_t launch_fold_weights(const void* Wp, const void* W2, const void* b2, int dp, int Dh, void* out,
                                float* bias_out, cudaStream_t st) {
  if (dp <= 0 || Dh <= 0) return cudaErrorInvalidValue;
  return launch_k(fold_weights_kernel, dim3((Dh + 127) / 128, dp), dim3(128), 0, st,
                  static_cast<const __nv_bfloat16*>(Wp), static_cast<const __nv_bfloat16*>(W2),
                  static_cast<const __nv_bfloat16*>(b2), dp, Dh, static_cast<__nv_bfloat16*>(out), bias_out);
}

cudaError_t launch_stats_combine(const float2* part, int B, int nparts, int ld, const int* lens, float2* fin,
                                 cudaStream_t st) {
  dim3 g((ld + 31) / 32, B);
  return launch_k(stats_combine_kernel, g, dim3(32, kCombY), 0, st, part, nparts, ld, lens, fin);
}

cudaError_t launch_row_sqnorm(const void* x, long long rows, int D, float* out, cudaStream_t st) {
  if (rows <= 0) return cudaSuccess;
  if (D % 8 != 0) return cudaErrorInvalidValue;
  const int warps = 8;
  const long long blocks = (rows + warps - 1) / warps;
  return launch_k(row_sqnorm_kernel, dim3(static_cast<unsigned>(blocks)), dim3(warps * 32), 0, st,
                  static_cast<const uint4*>(x), rows, D / 8, out);
}

cudaError_t launch_gather(const void* V, const int32_t* idx, int B, int N, int k, int D, void* out, int* status,
                          cudaStream_t st) {
  if (B <= 0 || k <= 0) return cudaSuccess;
  if (D % 8 != 0) return cudaErrorInvalidValue;
  const long long rows = static_cast<long long>(B) * k;
  return launch_k(gather_rows_kernel, dim3(static_cast<unsigned>(rows)), dim3(128), 0, st,
                  static_cast<const uint4*>(V), idx, N, k, D / 8, static_cast<uint4*>(out), status);
}

cudaError_t launch_sum_tiles(const float* part, int B, int N, int n_tiles, float* scores, cudaStream_t st) {
  const long long total = static_cast<long long>(B) * N;
  return launch_k(sum_tiles_kernel, dim3(static_cast<unsigned>((total + 255) / 256)), dim3(256), 0, st, part, N,
                  n_tiles, total, scores);
}

}  // namespace mapk
