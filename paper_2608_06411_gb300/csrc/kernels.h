// Host-side launchers of the CUDA kernels (internal to libmap_gb300).
#pragma once
#include <cstdint>
#include <cuda_runtime.h>

namespace mapk {

// *_SPLIT epilogues store an fp32 activation x as two bf16 halves, hi = bf16(x) at
// column c and lo = bf16(x - hi) at column N + c of a [rows, 2N] buffer, so that the next
// layer can consume ~16 significant bits through a bf16 GEMM: [hi | lo] @ [W | W]^T.
enum Epi { EPI_GELU_BF16 = 0, EPI_BIAS_BF16 = 1, EPI_ROPE_F32 = 2, EPI_F32 = 3, EPI_GELU_SPLIT = 4,
           EPI_BIAS_SPLIT = 5 };

// Batched C = epi(A @ B^T): A rows [batch][a_row_stride] x K, B rows [batch][b_row_stride] x K
// (both bf16, K contiguous, tightly packed 2D arrays of a_rows_total / b_rows_total rows).
struct GemmDesc {
  const void* A; long long a_rows_total; int a_row_stride;
  const void* B; long long b_rows_total; int b_row_stride;
  int M, N, K, batch;
  const int* n_limit;                   // per-batch output-column limit (device) or nullptr
  void* C; long long ldc; long long c_batch_stride;   // elements
  const void* bias;                     // bf16 [N] or nullptr
  const float2* rope; int rope_half;    // (cos, sin) table [pos][rope_half]
  const int* pos; int pos_mod;          // per-row positions (device) or row % pos_mod
  int epi;
  int* status;
};

// Returns cudaSuccess, or an error for an unsupported shape (cudaErrorInvalidValue).
cudaError_t launch_gemm(const GemmDesc& d, int num_sms, cudaStream_t st);

// Squared row norms of bf16 rows: out[r] = sum_d x[r, d]^2 (fp32).
cudaError_t launch_row_sqnorm(const void* x, long long rows, int D, float* out, cudaStream_t st);

// Eq. 3 softmax statistics and mean (q [sum M, dp], k [B*N, dp] fp32).
struct ScoreDesc {
  const float* q; const float* k;
  const int* q_off;       // [B+1] device row offsets of each image's queries
  int B, N, dp, max_m;
  float* stats;           // workspace [sum M][nsplit][2]
  int nsplit;
  float* scores;          // [B, N]
  int* status;
};
cudaError_t launch_scores(const ScoreDesc& d, cudaStream_t st);

// Gather rows: out[b, j, :] = V[b, idx[b, j], :].
cudaError_t launch_gather(const void* V, const int32_t* idx, int B, int N, int k, int D, void* out,
                          int* status, cudaStream_t st);

}  // namespace mapk
