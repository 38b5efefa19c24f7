// Host-side launchers of the CUDA kernels (internal to libmap_gb300).
#pragma once
#include <cstdint>
#include <cuda_runtime.h>

namespace mapk {

// *_SPLIT epilogues store an fp32 activation x as two bf16 halves, hi = bf16(x) at
// column c and lo = bf16(x - hi) at column N + c of a [rows, 2N] buffer, so that the next
// layer can consume ~16 significant bits through a bf16 GEMM: [hi | lo] @ [W | W]^T.
// EPI_ROPE_SPLIT3 applies RoPE (and `scale`) and stores the vector as three bf16
// segments, [hi | lo | hi] (split_kind 0, keys) or [hi | hi | lo] (split_kind 1, queries),
// so that one bf16 GEMM with K = 3 dp gives q.k to about 16 significant bits; it can also
// store the fp32 vector to `aux`.
// EPI_SM_STATS / EPI_SM_MEAN are the two passes of Eq. 3 over a logits tile (rows =
// visual tokens, columns = question tokens): per-column max / sum of exp over each
// 32-row slab, then per-row mean over columns of exp(l - max) / sum.
// EPI_PROJECT: rows = visual tokens, columns = the R0 basis tokens' rows (Gram entries
// <v_n, v_r>); the epilogue solves for the tokens' Cholesky coordinates against the R0
// basis (L staged in shared memory); ||v_n||^2 is the diagonal of an A A^T product that the
// MMA thread accumulates from the same shared-memory tiles.  It writes the exact residual,
// value and coordinate cache of every candidate token (see select.cu).
enum Epi { EPI_GELU_BF16 = 0, EPI_BIAS_BF16 = 1, EPI_ROPE_F32 = 2, EPI_F32 = 3, EPI_GELU_SPLIT = 4,
           EPI_BIAS_SPLIT = 5, EPI_ROPE_SPLIT3 = 6, EPI_SM_STATS = 7, EPI_SM_MEAN = 8, EPI_PROJECT = 9 };

// Inputs and outputs of the EPI_PROJECT epilogue (device pointers).
struct ProjArgs {
  const uint8_t* state;        // [B, N] 0 = candidate
  const float* scores;         // [B, N] p_hat
  float* Ec; int KP;           // coordinate cache rows [B, N, KP]
  const int32_t* basis_tok;    // [B, Kcap]
  const float* rnorm;          // [B, Kcap]
  const int32_t* nbasis;       // [B] basis size after R0 (<= 128)
  int Kcap;
  float lambda, tau;
  float* r2; float* U; float* sqn; int32_t* cstep;   // [B, N] outputs
};

// Batched C = epi(A @ B^T): A rows [batch][a_row_stride] x K, B rows [batch][b_row_stride] x K
// (both bf16, K contiguous, tightly packed 2D arrays of a_rows_total / b_rows_total rows).
struct GemmDesc {
  const void* A; long long a_rows_total; int a_row_stride;
  const void* B; long long b_rows_total; int b_row_stride;
  int M, N, K, batch;
  const int* n_limit;                   // per-batch output-column limit (device) or nullptr
  void* C; long long ldc; long long c_batch_stride;   // elements
  const void* bias;                     // bf16 [N] or nullptr
  const float2* rope; int rope_half;    // (cos, sin) table [rope_half][rope_ld]: position-minor, so
  int rope_ld = 0;                      // lanes (consecutive rows) read consecutive entries
  const int* pos; int pos_mod;          // per-row positions (device) or row % pos_mod
  int epi;
  int* status;
  // EPI_ROPE_SPLIT3
  int split_kind = 0; float scale = 1.f; float* aux = nullptr;
  // batched B rows at per-batch offsets (device) instead of b * b_row_stride
  const int* b_off = nullptr;
  // EPI_SM_STATS: partial (max, sum) per 32-row slab [batch][m_tiles * 4][stat_ld] (float2)
  // EPI_SM_MEAN:  final (max + ln sum, 1/sum) per column [batch][stat_ld]; output C = scores
  //               [batch][M] when one column tile covers all columns
  float2* stats = nullptr; int stat_ld = 0;
  const int* col_count = nullptr;       // per-batch number of valid columns (M_b)
  // B rows at b * b_row_stride + b_base
  int b_base = 0;
  ProjArgs proj{};
  // A has a_kwrap columns; its K coordinate wraps (k mod a_kwrap), so a K-segment of A can
  // be read twice against different B segments (0: A has K columns)
  int a_kwrap = 0;
  // B has b_kwrap columns and its K coordinate wraps likewise (0: B has K columns)
  int b_kwrap = 0;
  // split3 = 1 (with K = 3 Dh, A = [hi | lo] and B = [W_hi | W_hi | W_lo]): K blocks are taken
  // as (hi_j, W_hi_j), (hi_j, W_lo_j) for every j, then (lo_j, W_hi_j), so each block of A_hi
  // is read twice back to back (the second time from L2)
  int split3 = 0;
  const float* biasf = nullptr;         // EPI_ROPE_SPLIT3: fp32 bias [N] added before RoPE
  // Batch entries to process (device): blist[0 .. *bcount) instead of 0 .. batch-1, so that a
  // launch over a few active images spreads their tiles over all SMs (grid sized for batch)
  const int* blist = nullptr; const int* bcount = nullptr;
  // Per-batch number of valid A rows (device) or nullptr: rows at or past it are treated as
  // absent (EPI_SM_STATS: excluded from the column statistics; EPI_SM_MEAN: output 0)
  const int* m_limit = nullptr;
  // Limit (ns) of the producer / MMA / epilogue waits; 0 = the default 2 s.  The waits that
  // let in-flight copies and MMAs land before an aborting CTA exits keep the default.
  long long wait_ns = 0;
  // A and B are the same matrix (same pointer, rows and strides, no K wrap): a tile whose B
  // rows are its A rows (the diagonal tile of a Gram block) loads them once and the MMA reads
  // the A stage as B
  int sym = 0;
  // Units ordered column tile first (then batch entry, K slice, row tile): with n_limit
  // skipping whole column tiles of some entries, the other units stay spread over all CTAs
  int n_outer = 0;
  // EPI_F32 split-K: ksplit K slices, each unit one slice of a tile, slice s writing its partial
  // sum at C + s * c_split_stride (elements, a multiple of 4); the caller adds the slices
  int ksplit = 1; long long c_split_stride = 0;
};

// Returns cudaSuccess, or an error for an unsupported shape (cudaErrorInvalidValue).
cudaError_t launch_gemm(const GemmDesc& d, int num_sms, cudaStream_t st);

// Folds a projection after a linear layer into one matrix: W = Wp W2 ([dp, Dh] = [dp, Dh] x
// [Dh, Dh]) and bias = Wp b2, accumulated in fp64 from the bf16 inputs.  W is stored as the
// bf16 rows [hi | hi | lo] ([dp, 3 Dh], hi = bf16(W), lo = bf16(W - hi)) for activations laid
// out [hi | lo] and read with the K-wrap [hi | lo | hi]; bias in fp32.
cudaError_t launch_fold_weights(const void* Wp, const void* W2, const void* b2, int dp, int Dh, void* out,
                                float* bias_out, cudaStream_t st);

// Per-image question metadata written on the device from values passed as kernel parameters
// (no host-to-device copy, so nothing queues behind bulk input copies on the copy engines):
// off[b] = first query row of image b (off[B] = total), len[b], pos[row] = N + m for the
// m-th question token of its image.  lens has B entries; offs are their exclusive prefix sums.
// With nv (host, B entries: valid visual tokens per image) the positions are nv[b] + m and
// nvalid[b] = nv[b] is written too (nvalid may be nullptr).
cudaError_t launch_query_meta(const int32_t* lens, const long long* offs, int B, int N, int32_t* off, int32_t* len,
                              int32_t* pos, const int32_t* nv, int32_t* nvalid, cudaStream_t st);
// dst[0 .. n) = host[0 .. n), passed as kernel parameters (no copy engine).
cudaError_t launch_put_ints(const int32_t* host, int n, int32_t* dst, cudaStream_t st);
// Copies two device ints into host-mapped memory (device aliases of pinned host words).
cudaError_t launch_flags_to_host(const int32_t* a, const int* b, int32_t* a_host_dev, int* b_host_dev, cudaStream_t st);

// Squared row norms of bf16 rows: out[r] = sum_d x[r, d]^2 (fp32).
cudaError_t launch_row_sqnorm(const void* x, long long rows, int D, float* out, cudaStream_t st);

// scores[b, n] = sum_t part[b, t, n] over n_tiles column-tile partial means.
cudaError_t launch_sum_tiles(const float* part, int B, int N, int n_tiles, float* scores, cudaStream_t st);

// Combines the per-slab softmax statistics into (max + ln sum, 1/sum) per question token:
// part [B][nparts][ld] -> fin [B][ld], columns < lens[b].
cudaError_t launch_stats_combine(const float2* part, int B, int nparts, int ld, const int* lens, float2* fin,
                                 cudaStream_t st);

// Gather rows: out[b, j, :] = V[b, idx[b, j], :].
cudaError_t launch_gather(const void* V, const int32_t* idx, int B, int N, int k, int D, void* out,
                          int* status, cudaStream_t st);

// Hand-off sequence per image: the kept rows V[b, idx[b, j]] (j < k), then the image's
// lens[b] question rows of T (packed in image order); pos = the kept index or n_b + m, plus
// pos_offset, with n_b = nv[b] (host; nullptr: N).  Indices outside [0, n_b) are not copied:
// pos = -1 and ST_BADINDEX in *status.
cudaError_t launch_assemble(const void* V, const int32_t* idx, const void* T, const int32_t* lens, const int32_t* nv,
                            int B, int N, int k, int D, int pos_offset, void* seq, int32_t* pos, int* status,
                            cudaStream_t st);

// ------------------------------------------------------------------ distillation step (fp32)
// C[i, j] = alpha sum_k A(i, k) B(k, j) on the tcgen05 GEMM, fp32 in (or bf16: a_bf16 / b_bf16)
// and fp32 out; row-major, A(i, k) = ta ? A[k lda + i] : A[i lda + k], B(k, j) = tb ? B[j ldb + k]
// : B[k ldb + j].  fp32 operands are staged as three bf16 terms (split-bf16 products to fp32
// accuracy, see distill.cu) in wsA / wsB, of at least the element counts tc_matmul_ws returns; C must be
// 16-byte aligned with ldc % 4 == 0.  Deterministic (fixed summation order).
// wsC: K-slice partial sums when the output has too few tiles to fill the GPU.  A bf16 operand
// that is K-major, dense and 64-aligned is read in place.  *launches (if given) counts the
// kernels launched.
void tc_matmul_ws(int M, int N, int K, float alpha, bool a_bf16, bool b_bf16, int num_sms, size_t* a_elems,
                  size_t* b_elems, size_t* c_elems);
cudaError_t launch_tc_matmul(bool ta, bool tb, int M, int N, int K, float alpha, const void* A, bool a_bf16,
                             long long lda, const void* B, bool b_bf16, long long ldb, float* C, long long ldc,
                             void* wsA, void* wsB, float* wsC, int num_sms, int* status, long long wait_ns,
                             cudaStream_t st, long long* launches);
cudaError_t launch_bf16_to_f32(const void* x, long long n, float* y, cudaStream_t st);
// z += b (per column); h = GELU(z)
cudaError_t launch_bias_gelu(float* z, const float* b, long long rows, int cols, float* h, cudaStream_t st);
cudaError_t launch_bias_add(float* x, const float* b, long long rows, int cols, cudaStream_t st);
// RoPE (or its transpose when backward) on [rows, d] fp32 rows; positions pos[r] or r % pos_mod.
cudaError_t launch_rope_f32(bool backward, const float* x, long long rows, int d, const float2* tab, int ld,
                            const int32_t* pos, int pos_mod, float* y, cudaStream_t st);
// S [total_m, N] logits of all images' question rows (row stride ld; image b: rows qoff[b] ..
// qoff[b+1]) -> softmax, p_hat [B, N], g = dL/dp_hat, *loss = mean_b D_KL(teacher_b || p_hat_b),
// then S is overwritten with dL/dlogits.  row_img [total_m]: image of each row; part: B * ceil(N/256)
// floats.
cudaError_t launch_distill_loss_grad(float* S, long long ld, long long total_m, const int32_t* qoff,
                                     const int32_t* row_img, const float* teacher, int B, int N, float* p_hat,
                                     float* g, float* part, float* loss, cudaStream_t st);
// dh *= GELU'(z)
cudaError_t launch_gelu_back(float* dh, const float* z, long long n, cudaStream_t st);
// out[c] = sum_r X[r, c], in a fixed order; part: 64 * cols floats of workspace
cudaError_t launch_colsum(const float* X, long long rows, int cols, float* part, float* out, cudaStream_t st);

}  // namespace mapk
