// Selection state and launchers (internal to libmap_gb300); see select.cu.
#pragma once
#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

namespace mapk {

constexpr int kCholMax = 128;     // largest R0 factored by sel_chol_kernel

struct SelState {
  int B, N, D, K, K0, S;          // S = active-set size (Gram block rows)
  int R;                          // rows per image in Vg = row stride of G (>= S + K, multiple of 16)
  int KP;                         // row stride of Ec (>= K, multiple of 4)
  float lambda, tau;
  const float* scores;            // [B, N] p_hat
  const void* V;                  // [B, N, D] bf16
  const float* sqn;               // [B, N] ||v||^2
  float* U;                       // [B, N] squared value bound / exact squared value (sel_value)
  float* r2;                      // [B, N] residual^2 as of cstep
  int32_t* cstep;                 // [B, N] basis coordinates cached
  uint8_t* state;                 // [B, N] 0 candidate, 1 retained, 2 padding (never a candidate)
  float* Ec;                      // [B, N, KP] cached coordinates e_beta[i]
  int32_t* picks;                 // [B, K] pick order
  int32_t* r0;                    // [B, K] R0 in p_hat order (first K0 used)
  int32_t* basis_tok;             // [B, K] token that added basis vector beta
  float* rnorm;                   // [B, K] its residual norm at that time
  int32_t* npicks; int32_t* nbasis; int32_t* nb_gathered; int32_t* done; int32_t* mode;
  int32_t* nlimit;                // [B] Gram block columns (S + nbasis), 0 when done
  int32_t* gb_lo; int32_t* gb_hi;  // [B] basis rows to gather this round
  int32_t* gbase;                 // [B] first basis vector whose row is in Vg (row S + beta - gbase);
                                  // after the R0 projection every candidate's coordinates on the
                                  // R0 basis are cached, so those columns are not recomputed
  uint64_t* theta;                // [B] key of the best candidate outside A (0: none)
  int32_t* aslot;                 // [B, S] active tokens (-1 empty)
  void* Vg;                       // [B, R, D] bf16 gathered rows
  float* G;                       // [B, S, R] Gram block
  int32_t* done_count;            // images finished
  int32_t* proj_lim;              // [B] basis columns the projection GEMM computes (0: image skipped)
  // Images the next Gram / projection GEMM processes (optional): blist[0 .. bcount[bc_par]).
  // A list producer (choose, projection prep) appends through bcount[bc_par] and zeroes
  // bcount[bc_par ^ 1] for the next producer, so no separate reset precedes it; the host
  // flips bc_par after each producer's consumer.
  int32_t* blist; int32_t* bcount; int bc_par;
  int* status;
  const int32_t* nvalid;          // [B] valid tokens per image (nullptr: all N); the rest are padding
  // Optional device array {scores, V}, written by sel_init from the two fields above: the
  // kernels of the cached selection-loop graph read the caller's buffers through it, so one
  // graph serves every call of the same shape.
  const void** uptr;
};

size_t sel_init_smem(int N, int K0);
size_t sel_choose_smem(int N);
// Active-set size (Gram block rows, threads of the greedy CTA) and the most picks one greedy
// launch makes (their coordinates are held in registers; the next round continues).
constexpr int kActiveSlots = 256;
constexpr int kRoundPicks = 128;
size_t sel_greedy_smem(int S);
cudaError_t launch_sel_init(const SelState& s, cudaStream_t st);
cudaError_t launch_sel_choose(const SelState& s, cudaStream_t st);
// sel_update_kernel (coordinates of the active tokens up to the current basis), the residual
// Gram matrix of the active set on that basis, then the picks.
cudaError_t launch_sel_greedy(const SelState& s, cudaStream_t st);
// The K0 forced R0 picks from the Gram block G[R0, R0] of a forced round (K0 <= kCholMax, <= S).
cudaError_t launch_sel_chol(const SelState& s, cudaStream_t st);
cudaError_t launch_sel_finalize(const int32_t* picks, int B, int K, int32_t* keep, int32_t* order, cudaStream_t st);
cudaError_t launch_sel_copy_r0(const int32_t* r0, int B, int K, int32_t* picks, cudaStream_t st);
cudaError_t launch_sel_identity(int B, int N, int32_t* keep, int32_t* order, cudaStream_t st);
// Queues basis rows for gathering into Vg (rows S + beta) ahead of a projection of every
// candidate on the whole basis: first = the R0 basis of every image; otherwise (after a
// greedy round) the basis of each image still selecting whose basis has grown and has at
// most kReprojMax vectors, other images are skipped (proj_lim 0).
constexpr int kReprojMax = 128;
cudaError_t launch_sel_proj_prep(const SelState& s, bool first, cudaStream_t st);
cudaError_t launch_sel_gather(const SelState& s, cudaStream_t st);
// After a projection: the projected images' later Gram blocks start past their basis.
cudaError_t launch_sel_proj_done(const SelState& s, cudaStream_t st);

// ------------------------------------------------------------------ device-side round loop
// The selection rounds after the first ones run as a CUDA graph: a kernel node that tests
// whether any image still selects, then a WHILE conditional node whose body is one round
// (choose + gather, Gram block, coordinate update + residual Gram + greedy picks) followed by
// the same test.
// The host never waits for the rounds.  Graphs are cached per shape and workspace.
struct GemmDesc;
struct SelLoopCache;
SelLoopCache* sel_loop_cache_create();
void sel_loop_cache_destroy(SelLoopCache* c);
// iters: device int (this call's loop iterations); iters_total: device counter of every loop
// iteration run so far (for launch counts).  After cap_iters iterations with images still
// selecting the loop stops and sets ST_INTERNAL.
cudaError_t launch_sel_loop(SelLoopCache* cache, const SelState& s, const GemmDesc& gram, int num_sms, int cap_iters,
                            int32_t* iters, long long* iters_total, cudaStream_t st);
constexpr int kSelLoopKernelsPerIter = 7;

}  // namespace mapk
