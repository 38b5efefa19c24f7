// Persistent tcgen05 GEMM for sm_103a:  C = epilogue(A @ B^T), A [M, K], B [N, K] bf16.
//
// Used for every dense contraction of the pruning path: the predictor layers f_V, f_T
// (Linear -> GELU -> Linear), the W_K / W_Q projections with RoPE fused into the
// epilogue (section "Cross-Modal Attention Distillation"), and the Gram blocks
// <v_i, v_j> that the diversity term of Eq. 4 needs.
//
// Structure (one CTA per SM, 6 warps):
//   warp 0      one thread issues TMA loads of 128x64 (A) and BNx64 (B) bf16 tiles, 128-byte
//               swizzled, into a STAGES-deep shared-memory ring (mbarrier full/empty).
//   warp 1      allocates TMEM (2 accumulators x BN fp32 columns); one thread issues
//               tcgen05.mma (M=128, N=BN, K=16) x 4 per stage and commits to mbarriers.
//   CG2 (the BN = 256 predictor layers): 2-CTA clusters run 2-SM MMAs (cta_group::2,
//               M = 256): each CTA loads its 128 A rows and half of the B tile, both
//               complete on the leader's full barrier, the leader's thread issues the MMAs and
//               its commits release the stage and the accumulator in both CTAs.
//   warps 2-5   epilogue: tcgen05.ld the accumulator (one TMEM lane = one output row per
//               thread), apply bias / GELU / RoPE, store (bf16, bf16 hi/lo pair, or fp32);
//               release the accumulator so the
//               MMA warp can start the tile after next while this one drains.
//   EPI_PROJECT: the MMA thread also accumulates A A^T (N = 128) of every stage into a second
//               TMEM accumulator, whose diagonal is ||row||^2.
// All waits are bounded (ptx.cuh); a timeout sets ST_TIMEOUT and every role drains and exits.
#include <algorithm>
#include <cstdio>
#include <cudaTypedefs.h>

#include "kernels.h"
#include "ptx.cuh"

namespace mapk {

namespace {

constexpr int kBM = 128;
constexpr int kBK = 64;

struct KArgs {
  int M, N, K, batch, a_row_stride, b_row_stride;
  const int* n_limit;
  void* C; long long ldc; long long c_batch_stride;
  const __nv_bfloat16* bias;
  const float2* rope; int rope_half; int rope_ld;
  const int* pos; int pos_mod;
  int* status;
  int split_kind; float scale; float* aux;
  const int* b_off;
  float2* stats; int stat_ld;
  const int* col_count;
  int b_base;
  ProjArgs proj;
  int a_kwrap, b_kwrap;
  int split3;
  const float* biasf;
  const int* blist; const int* bcount;
  const int* m_limit;
  unsigned long long wait_ns;   // limit of the role waits (the drain waits keep kWaitLimitNs)
  int ksplit; long long c_split_stride;   // EPI_F32 split-K: partial sums per K slice
  int sym;                                 // B is A: the diagonal tile reads its A stage as B
  int n_outer;                             // unit order: column tiles outermost
};

__device__ __forceinline__ float gelu_erf(float x) {
  return 0.5f * x * (1.0f + erff(x * 0.70710678118654752f));
}

__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
  __nv_bfloat162 h = __floats2bfloat162_rn(a, b);   // .x = a (low half), .y = b
  return *reinterpret_cast<uint32_t*>(&h);
}

constexpr int kProjMaxBasis = 128;             // EPI_PROJECT: R0 basis size supported

template <int BN, int STAGES, int EPI, bool CG2>
struct Smem {
  static constexpr bool PROJ = EPI == EPI_PROJECT;
  static constexpr uint32_t A_BYTES = kBM * kBK * 2;
  static constexpr uint32_t B_BYTES = (CG2 ? BN / 2 : BN) * kBK * 2;   // CG2: this CTA's half
  static constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr uint32_t TILES = STAGES * STAGE_BYTES;
  static constexpr uint32_t BARS = (2 * STAGES + 5 + (PROJ ? 1 : 0)) * 8;
  // per-warp 32x32 transposes (EPI_SM_STATS) or 32 column normalisers (EPI_SM_MEAN)
  static constexpr uint32_t XPOSE = EPI == EPI_SM_STATS ? 4 * 32 * 33 * 4 : (EPI == EPI_SM_MEAN ? 4 * 32 * 4 : 0);
  // bf16 outputs written by TMA box stores from per-warp staging: hi/lo split epilogues use two
  // buffers of (hi, lo) 32x32 boxes, EPI_ROPE_SPLIT3 (BN = 128) one buffer of (hi, lo) x 2 halves
  static constexpr bool TSTORE_ROPE = EPI == EPI_ROPE_SPLIT3 && BN == 128;
  static constexpr bool TSTORE = EPI == EPI_GELU_SPLIT || EPI == EPI_BIAS_SPLIT || TSTORE_ROPE;
  static constexpr uint32_t STG = TSTORE ? 4 * 4 * 32 * 32 * 2 : 0;
  static constexpr uint32_t LSM = PROJ ? BN * BN * 4 : 0;       // L rows of the basis (pitch BN)
  static constexpr uint32_t PEXTRA = PROJ ? BN * 4 : 0;          // 1/r of the basis
  static constexpr uint32_t TOTAL = 1024 + TILES + STG + BARS + 16 + XPOSE + LSM + PEXTRA;
  static constexpr uint32_t TMEM_COLS = PROJ ? (2 * BN + 2 * kBM <= 256 ? 256u : 512u) : 2 * BN;   // + A A^T
  static constexpr int THREADS = 192;
};

// Selection value, squared: p^2 * rho^(2 lambda) orders candidates like p * rho^lambda (both are
// >= 0) and needs no square root for lambda = 1.  rho^2 = r2 unless r2 <= tau ||v||^2 (then 0).
__device__ __forceinline__ float proj_value(float p, float r2, float sq, float lam, float tau) {
  if (!(p > 0.f)) return 0.f;
  if (lam == 0.f) return p * p;
  if (!(r2 > tau * sq) || !(r2 > 0.f)) return 0.f;
  const float v = lam == 1.f ? (p * p) * r2 : (p * p) * powf(r2, lam);
  return v > 0.f ? v : 0.f;
}

struct TileCoord { int b, m_blk, n_blk, ks; bool skip; };

// Work unit t -> tile.  With PAIR the unit is a pair of vertically adjacent M tiles with the
// same N tile, processed by the two CTAs of a cluster (rank 0 the upper, rank 1 the lower).
// With split-K (ksplit > 1) a unit is also one K slice ks of its tile.
template <bool PAIR>
__device__ __forceinline__ TileCoord tile_coord(const KArgs& a, int t, int nbatch, int m_units, int n_tiles, int BN,
                                                uint32_t crank) {
  TileCoord c;
  int mu;
  if (a.n_outer) {
    // column tiles outermost: the units of one column tile of every batch entry are
    // consecutive, so that when whole column tiles are skipped (n_limit) the remaining units
    // still spread over all CTAs
    const int per_n = nbatch * m_units * a.ksplit;
    c.n_blk = t / per_n;
    int rem = t - c.n_blk * per_n;
    c.b = rem / (m_units * a.ksplit);
    rem -= c.b * (m_units * a.ksplit);
    c.ks = rem / m_units;
    mu = rem - c.ks * m_units;
  } else {
    const int tiles = m_units * n_tiles;
    const int per = tiles * a.ksplit;
    c.b = t / per;
    int rem = t - c.b * per;
    c.ks = rem / tiles;
    rem -= c.ks * tiles;
    mu = rem / n_tiles;
    c.n_blk = rem - mu * n_tiles;
  }
  if (a.blist) c.b = __ldg(a.blist + c.b);
  c.m_blk = PAIR ? 2 * mu + static_cast<int>(crank) : mu;
  int lim = a.n_limit ? min(a.N, __ldg(a.n_limit + c.b)) : a.N;
  c.skip = c.n_blk * BN >= lim;
  return c;
}

template <int BN, int STAGES, int EPI, bool CG2>
__global__ void __launch_bounds__(Smem<BN, STAGES, EPI, CG2>::THREADS, 1)
gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
               const __grid_constant__ CUtensorMap tmC, KArgs a) {
  using S = Smem<BN, STAGES, EPI, CG2>;
  constexpr bool PAIR = CG2;
  constexpr uint32_t IDESC = idesc_bf16(CG2 ? 2 * kBM : kBM, BN);
  const uint32_t crank = PAIR ? cluster_ctarank() : 0u;
  const int unit0 = PAIR ? static_cast<int>(blockIdx.x >> 1) : static_cast<int>(blockIdx.x);
  const int units_step = PAIR ? static_cast<int>(gridDim.x >> 1) : static_cast<int>(gridDim.x);
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + STAGES * S::A_BYTES;
  uint8_t* stg = smem + S::TILES;                // TSTORE staging boxes (1024-aligned)
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + S::TILES + S::STG);
  uint64_t* empty = full + STAGES;
  uint64_t* tfull = empty + STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1 + (S::PROJ ? 1 : 0));
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  uint64_t* egsync = drain + 1;                  // EPI_PROJECT: epilogue warps' group barrier
  float* xpose = reinterpret_cast<float*>(smem + S::TILES + S::STG + S::BARS + 16);
  float* Lsm = xpose + S::XPOSE / 4;
  float* rinv_sm = Lsm + S::LSM / 4;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) { mbar_init(&full[s], 1); mbar_init(&empty[s], 1); }
    // tempty: one arrive per epilogue warp (of both CTAs with CG2, on the leader's barrier)
    for (int i = 0; i < 2; ++i) { mbar_init(&tfull[i], 1); mbar_init(&tempty[i], CG2 ? 8 : 4); }
    mbar_init(drain, 1);
    if constexpr (S::PROJ) {
      mbar_init(egsync, 128);
    }
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) { tma_prefetch_desc(&tmA); tma_prefetch_desc(&tmB); }
  pdl_enter();                                    // inputs below come from the previous kernel
  if (warp == 1) {
    if constexpr (CG2) { tmem_alloc_cg2(tmem_slot, S::TMEM_COLS); tmem_relinquish_cg2(); }
    else { tmem_alloc(tmem_slot, S::TMEM_COLS); tmem_relinquish(); }
  }
  if constexpr (PAIR) cluster_sync();             // peer barriers initialised before any remote arrive
  else __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  const int m_tiles = (a.M + kBM - 1) / kBM;
  const int m_units = PAIR ? (m_tiles + 1) / 2 : m_tiles;
  const int n_tiles = (a.N + BN - 1) / BN;
  const int nbatch = a.blist ? min(a.batch, *a.bcount) : a.batch;
  const int total = nbatch * m_units * n_tiles * a.ksplit;
  const int KB = a.K / kBK;
  // K blocks of a unit's slice (the whole K without split-K)
  auto kb_range = [&](const TileCoord& c, int& kb0, int& kb1) {
    kb0 = c.ks * KB / a.ksplit;
    kb1 = (c.ks + 1) * KB / a.ksplit;
  };
  // K block kb -> (A column, B column)
  auto kcols = [&](int kb, int& ac, int& bc) {
    if (a.split3) {
      const int nbk = KB / 3;
      if (kb < 2 * nbk) {
        const int j = kb >> 1;
        ac = j * kBK;
        bc = (kb & 1) ? (2 * nbk + j) * kBK : j * kBK;
      } else {
        ac = bc = (kb - nbk) * kBK;
      }
    } else {
      ac = a.a_kwrap > 0 ? (kb * kBK) % a.a_kwrap : kb * kBK;
      bc = a.b_kwrap > 0 ? (kb * kBK) % a.b_kwrap : kb * kBK;
    }
  };

  // With a.sym, a tile whose B rows (this CTA's half of them with 2-SM pairs) are its A rows
  // loads them once: the same stage layout serves as both operands (BN / 2 or BN == kBM rows).
  // Both CTAs of a pair and all roles reach the same answer (the row offsets cancel).
  auto b_is_a = [&](const TileCoord& c) {
    if (!a.sym || (CG2 ? BN / 2 : BN) != kBM) return false;
    const int arow = c.b * a.a_row_stride + c.m_blk * kBM;
    const int brow = c.b * a.b_row_stride + a.b_base + c.n_blk * BN + (CG2 ? static_cast<int>(crank) * (BN / 2) : 0);
    return arow == brow;
  };

  // Producer: parity of the last load issued into each stage (-1: none), for the drain below.
  int last_par[STAGES];
#pragma unroll
  for (int s = 0; s < STAGES; ++s) last_par[s] = -1;
  if (warp == 0) {
    if (lane == 0) {
      // ---------------------------------------------------------------- TMA producer
      uint32_t stage = 0, phase = 0;
      bool ok = true;
      for (int t = unit0; t < total && ok; t += units_step) {
        TileCoord c = tile_coord<PAIR>(a, t, nbatch, m_units, n_tiles, BN, crank);
        if (c.skip) continue;
        const int arow = c.b * a.a_row_stride + c.m_blk * kBM;
        const int brow = (a.b_off ? __ldg(a.b_off + c.b) : c.b * a.b_row_stride + a.b_base) + c.n_blk * BN;
        const bool alias = b_is_a(c);
        const int kstep = alias ? 2 : 1;           // alias: two K blocks per stage (A and B buffers)
        int kb0, kb1;
        kb_range(c, kb0, kb1);
        for (int kb = kb0; kb < kb1; kb += kstep) {
          if (!mbar_wait(&empty[stage], phase ^ 1, a.status, abort_flag, a.wait_ns)) { ok = false; break; }
          int ac, bc;
          kcols(kb, ac, bc);
          if (alias) {
            // K block kb into the A buffer, kb + 1 (when in range) into the B buffer; no kwrap
            const int n2 = kb + 1 < kb1 ? 2 : 1;
            if constexpr (CG2) {
              if (crank == 0) mbar_arrive_expect_tx(&full[stage], 2 * n2 * S::A_BYTES);
              const uint32_t fb = mapa_u32(&full[stage], 0);
              tma_load_2d_cg2(sA + stage * S::A_BYTES, &tmA, fb, ac, arow);
              if (n2 == 2) tma_load_2d_cg2(sB + stage * S::B_BYTES, &tmA, fb, ac + kBK, arow);
            } else {
              mbar_arrive_expect_tx(&full[stage], n2 * S::A_BYTES);
              tma_load_2d(sA + stage * S::A_BYTES, &tmA, &full[stage], ac, arow);
              if (n2 == 2) tma_load_2d(sB + stage * S::B_BYTES, &tmA, &full[stage], ac + kBK, arow);
            }
          } else if constexpr (CG2) {
            // both CTAs' copies complete on the leader's full barrier, which expects them all
            if (crank == 0) mbar_arrive_expect_tx(&full[stage], 2 * S::STAGE_BYTES);
            const uint32_t fb = mapa_u32(&full[stage], 0);
            tma_load_2d_cg2(sA + stage * S::A_BYTES, &tmA, fb, ac, arow);
            tma_load_2d_cg2(sB + stage * S::B_BYTES, &tmB, fb, bc, brow + static_cast<int>(crank) * (BN / 2));
          } else {
            mbar_arrive_expect_tx(&full[stage], S::STAGE_BYTES);
            tma_load_2d(sA + stage * S::A_BYTES, &tmA, &full[stage], ac, arow);
            tma_load_2d(sB + stage * S::B_BYTES, &tmB, &full[stage], bc, brow);
          }
          last_par[stage] = static_cast<int>(phase);
          if (++stage == STAGES) { stage = 0; phase ^= 1; }
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0 && crank == 0) {
      // ---------------------------------------------------------------- MMA issuer (CG2: leader)
      uint32_t stage = 0, phase = 0, acc = 0, acc_phase = 0;
      bool issued = false, ok = true;
      for (int t = unit0; t < total && ok; t += units_step) {
        TileCoord c = tile_coord<PAIR>(a, t, nbatch, m_units, n_tiles, BN, crank);
        if (c.skip) continue;
        if (!mbar_wait(&tempty[acc], acc_phase ^ 1, a.status, abort_flag, a.wait_ns)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * BN;
        const bool alias = b_is_a(c);
        const int kstep = alias ? 2 : 1;
        int kb0, kb1;
        kb_range(c, kb0, kb1);
        for (int kb = kb0; kb < kb1; kb += kstep) {
          if (!mbar_wait(&full[stage], phase, a.status, abort_flag, a.wait_ns)) { ok = false; break; }
          tc_fence_after();
          const uint32_t a0 = smem_u32(sA + stage * S::A_BYTES);
          const uint32_t b0 = alias ? a0 : smem_u32(sB + stage * S::B_BYTES);
          if (alias) {
            // each buffer is both operands of its K block (the tile's B rows are its A rows)
            const uint32_t a1 = smem_u32(sB + stage * S::B_BYTES);
            const int n2 = kb + 1 < kb1 ? 2 : 1;
            for (int h = 0; h < n2; ++h) {
              const uint32_t x = h == 0 ? a0 : a1;
#pragma unroll
              for (int k = 0; k < kBK / 16; ++k) {
                const uint32_t acc_on = (kb != kb0 || h != 0 || k != 0);
                if constexpr (CG2) umma_bf16_cg2(d_tmem, desc_sw128(x + k * 32), desc_sw128(x + k * 32), IDESC, acc_on);
                else umma_bf16(d_tmem, desc_sw128(x + k * 32), desc_sw128(x + k * 32), IDESC, acc_on);
              }
            }
            if constexpr (CG2) umma_commit_cg2_mc(&empty[stage], static_cast<uint16_t>(3));
            else umma_commit(&empty[stage]);
          } else if constexpr (CG2) {
#pragma unroll
            for (int k = 0; k < kBK / 16; ++k)
              umma_bf16_cg2(d_tmem, desc_sw128(a0 + k * 32), desc_sw128(b0 + k * 32), IDESC, (kb != kb0 || k != 0));
            umma_commit_cg2_mc(&empty[stage], static_cast<uint16_t>(3));
          } else {
#pragma unroll
            for (int k = 0; k < kBK / 16; ++k)
              umma_bf16(d_tmem, desc_sw128(a0 + k * 32), desc_sw128(b0 + k * 32), IDESC, (kb != kb0 || k != 0));
            if constexpr (S::PROJ) {   // A A^T: its diagonal is ||row||^2
              const uint32_t n_tmem = tmem_base + 2 * BN + acc * kBM;
#pragma unroll
              for (int k = 0; k < kBK / 16; ++k)
                umma_bf16(n_tmem, desc_sw128(a0 + k * 32), desc_sw128(a0 + k * 32), idesc_bf16(kBM, kBM),
                          (kb != kb0 || k != 0));
            }
            umma_commit(&empty[stage]);
          }
          issued = true;
          if (++stage == STAGES) { stage = 0; phase ^= 1; }
        }
        if (!ok) break;
        if constexpr (CG2) umma_commit_cg2_mc(&tfull[acc], static_cast<uint16_t>(3));
        else umma_commit(&tfull[acc]);
        acc ^= 1;
        if (acc == 0) acc_phase ^= 1;
      }
      if (issued) {   // every MMA of this CTA has completed before TMEM is released
        if constexpr (CG2) umma_commit_cg2(drain);
        else umma_commit(drain);
        mbar_wait(drain, 0, a.status, nullptr);
      }
    }
    __syncwarp();
  } else if (warp < 6) {
    // ------------------------------------------------------------------ epilogue
    const int lane_grp = warp & 3;                 // TMEM lanes this warp may access
    const int r_in_tile = lane_grp * 32 + lane;
    uint32_t acc = 0, acc_phase = 0;
    int staged_b = -1;                             // EPI_PROJECT: image whose L is in shared memory
    uint32_t eg_phase = 0;
    bool eg_ok = true;
    for (int t = unit0; t < total && eg_ok; t += units_step) {
      TileCoord c = tile_coord<PAIR>(a, t, nbatch, m_units, n_tiles, BN, crank);
      if (c.skip) continue;
      if constexpr (S::PROJ) {
        if (c.b != staged_b) {                     // stage L and 1/r of this image's R0 basis
          // group barrier of the 128 epilogue threads (bounded, unlike a named barrier)
          mbar_arrive(egsync);
          if (!mbar_wait(egsync, eg_phase, a.status, abort_flag, a.wait_ns)) { eg_ok = false; break; }
          eg_phase ^= 1;
          const ProjArgs& pj = a.proj;
          const int nb0 = min(BN, __ldg(pj.nbasis + c.b));
          const long long ibase = static_cast<long long>(c.b) * a.M;
          const int KV = BN / 4;
          for (int t4 = threadIdx.x - 64; t4 < nb0 * KV; t4 += 128) {
            const int i = t4 / KV, q = (t4 - i * KV) * 4;
            float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
            if (q < i) {
              const int tk = __ldg(pj.basis_tok + static_cast<long long>(c.b) * pj.Kcap + i);
              const float* row = pj.Ec + (ibase + tk) * pj.KP + q;
              v.x = row[0];
              v.y = q + 1 < i ? row[1] : 0.f;
              v.z = q + 2 < i ? row[2] : 0.f;
              v.w = q + 3 < i ? row[3] : 0.f;
            }
            *reinterpret_cast<float4*>(Lsm + i * BN + q) = v;
          }
          for (int i = threadIdx.x - 64; i < nb0; i += 128)
            rinv_sm[i] = 1.0f / __ldg(pj.rnorm + static_cast<long long>(c.b) * pj.Kcap + i);
          mbar_arrive(egsync);
          if (!mbar_wait(egsync, eg_phase, a.status, abort_flag, a.wait_ns)) { eg_ok = false; break; }
          eg_phase ^= 1;
          staged_b = c.b;
        }
      }
      if (!mbar_wait(&tfull[acc], acc_phase, a.status, abort_flag, a.wait_ns)) break;
      tc_fence_after();
      const int row = c.m_blk * kBM + r_in_tile;
      const bool row_ok = row < (a.m_limit ? min(a.M, __ldg(a.m_limit + c.b)) : a.M);
      const int lim = a.n_limit ? min(a.N, __ldg(a.n_limit + c.b)) : a.N;
      const int col0 = c.n_blk * BN;
      const uint32_t tbase = tmem_base + (static_cast<uint32_t>(lane_grp * 32) << 16) + acc * BN;
      const long long crow = static_cast<long long>(c.b) * a.c_batch_stride + static_cast<long long>(row) * a.ldc;

      if constexpr (EPI == EPI_ROPE_F32) {
        // BN == dp: the whole row is in this tile; rotate pairs (i, i + dp/2).
        constexpr int HALF = BN / 2;
        float* out = reinterpret_cast<float*>(a.C) + crow;
        int pos = 0;
        if (row_ok) pos = a.pos ? __ldg(a.pos + row) : row % a.pos_mod;
        const float2* rt = a.rope + pos;
#pragma unroll 1
        for (int ch = 0; ch < HALF / 32; ++ch) {
          uint32_t r1[32], r2[32];
          tmem_ld32(tbase + ch * 32, r1);
          tmem_ld32(tbase + HALF + ch * 32, r2);
          if (row_ok) {
#pragma unroll
            for (int j = 0; j < 32; j += 4) {
              float o1[4], o2[4];
#pragma unroll
              for (int u = 0; u < 4; ++u) {
                const float2 cs = __ldg(rt + static_cast<long long>(ch * 32 + j + u) * a.rope_ld);
                const float x1 = __uint_as_float(r1[j + u]), x2 = __uint_as_float(r2[j + u]);
                o1[u] = x1 * cs.x - x2 * cs.y;
                o2[u] = x2 * cs.x + x1 * cs.y;
              }
              *reinterpret_cast<float4*>(out + ch * 32 + j) = make_float4(o1[0], o1[1], o1[2], o1[3]);
              *reinterpret_cast<float4*>(out + HALF + ch * 32 + j) = make_float4(o2[0], o2[1], o2[2], o2[3]);
            }
          }
        }
      } else if constexpr (S::TSTORE_ROPE) {
        // BN == dp = 128; x = RoPE(acc + bias) * scale as bf16 (hi, lo) segments, staged per warp
        // in shared memory and written by TMA box stores (rows past M are clipped)
        constexpr int HALF = BN / 2;
        float* aux = (a.aux && row_ok) ? a.aux + static_cast<long long>(row) * BN : nullptr;
        int pos = 0;
        if (row_ok) pos = a.pos ? __ldg(a.pos + row) : row % a.pos_mod;
        const float2* rt = a.rope + pos;
        const int seg_lo = a.split_kind == 0 ? 1 : 2;   // keys [hi, lo, hi], queries [hi, hi, lo]
        const int ew = warp - 2;
        const int y = c.b * a.a_row_stride + c.m_blk * kBM + lane_grp * 32;
        uint8_t* sb = stg + ew * 8192;                 // [hi1 | lo1 | hi2 | lo2], 32 rows x 64 B each
#pragma unroll 1
        for (int ch = 0; ch < HALF / 32; ++ch) {
          uint32_t r1[32], r2[32];
          tmem_ld32(tbase + ch * 32, r1);
          tmem_ld32(tbase + HALF + ch * 32, r2);
          if (lane == 0) bulk_wait_group_read<0>();    // the previous chunk's stores have read sb
          __syncwarp();
#pragma unroll
          for (int j = 0; j < 32; j += 8) {
            float o1[8], o2[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
              const float2 cs = __ldg(rt + static_cast<long long>(ch * 32 + j + u) * a.rope_ld);
              float x1 = __uint_as_float(r1[j + u]), x2 = __uint_as_float(r2[j + u]);
              if (a.biasf) {
                x1 += __ldg(a.biasf + ch * 32 + j + u);
                x2 += __ldg(a.biasf + HALF + ch * 32 + j + u);
              }
              o1[u] = x1 * cs.x - x2 * cs.y;
              o2[u] = x2 * cs.x + x1 * cs.y;
            }
            if (aux) {
#pragma unroll
              for (int u = 0; u < 8; u += 4) {
                *reinterpret_cast<float4*>(aux + ch * 32 + j + u) = make_float4(o1[u], o1[u + 1], o1[u + 2], o1[u + 3]);
                *reinterpret_cast<float4*>(aux + HALF + ch * 32 + j + u) =
                    make_float4(o2[u], o2[u + 1], o2[u + 2], o2[u + 3]);
              }
            }
#pragma unroll
            for (int u = 0; u < 8; ++u) { o1[u] *= a.scale; o2[u] *= a.scale; }
            uint32_t h1[4], l1[4], h2[4], l2[4];
#pragma unroll
            for (int u = 0; u < 8; u += 2) {
              const __nv_bfloat162 a1 = __floats2bfloat162_rn(o1[u], o1[u + 1]);
              const __nv_bfloat162 a2 = __floats2bfloat162_rn(o2[u], o2[u + 1]);
              h1[u / 2] = *reinterpret_cast<const uint32_t*>(&a1);
              h2[u / 2] = *reinterpret_cast<const uint32_t*>(&a2);
              l1[u / 2] = pack_bf16(o1[u] - __bfloat162float(a1.x), o1[u + 1] - __bfloat162float(a1.y));
              l2[u / 2] = pack_bf16(o2[u] - __bfloat162float(a2.x), o2[u + 1] - __bfloat162float(a2.y));
            }
            uint8_t* rowp = sb + lane * 64 + ((j / 8) ^ ((lane >> 1) & 3)) * 16;   // 64-byte swizzle
            *reinterpret_cast<uint4*>(rowp) = make_uint4(h1[0], h1[1], h1[2], h1[3]);
            *reinterpret_cast<uint4*>(rowp + 2048) = make_uint4(l1[0], l1[1], l1[2], l1[3]);
            *reinterpret_cast<uint4*>(rowp + 4096) = make_uint4(h2[0], h2[1], h2[2], h2[3]);
            *reinterpret_cast<uint4*>(rowp + 6144) = make_uint4(l2[0], l2[1], l2[2], l2[3]);
          }
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) {
#pragma unroll
            for (int sg = 0; sg < 3; ++sg) {
              const int x = sg * BN + ch * 32;
              tma_store_2d(&tmC, sb + (sg == seg_lo ? 2048 : 0), x, y);
              tma_store_2d(&tmC, sb + (sg == seg_lo ? 6144 : 4096), x + HALF, y);
            }
            bulk_commit_group();
          }
        }
      } else if constexpr (EPI == EPI_ROPE_SPLIT3) {
        // BN == dp; x = RoPE(acc) * scale, stored as bf16 (hi, lo) segments
        constexpr int HALF = BN / 2;
        __nv_bfloat16* out = reinterpret_cast<__nv_bfloat16*>(a.C) + crow;
        float* aux = a.aux ? a.aux + static_cast<long long>(row) * BN : nullptr;
        int pos = 0;
        if (row_ok) pos = a.pos ? __ldg(a.pos + row) : row % a.pos_mod;
        const float2* rt = a.rope + pos;
        // segment order: keys [hi, lo, hi], queries [hi, hi, lo]
        const int seg_lo = a.split_kind == 0 ? 1 : 2;
#pragma unroll 1
        for (int ch = 0; ch < HALF / 32; ++ch) {
          uint32_t r1[32], r2[32];
          tmem_ld32(tbase + ch * 32, r1);
          tmem_ld32(tbase + HALF + ch * 32, r2);
          if (row_ok) {
#pragma unroll
            for (int j = 0; j < 32; j += 8) {
              float o1[8], o2[8];
#pragma unroll
              for (int u = 0; u < 8; ++u) {
                const float2 cs = __ldg(rt + static_cast<long long>(ch * 32 + j + u) * a.rope_ld);
                float x1 = __uint_as_float(r1[j + u]), x2 = __uint_as_float(r2[j + u]);
                if (a.biasf) {
                  x1 += __ldg(a.biasf + ch * 32 + j + u);
                  x2 += __ldg(a.biasf + HALF + ch * 32 + j + u);
                }
                o1[u] = x1 * cs.x - x2 * cs.y;
                o2[u] = x2 * cs.x + x1 * cs.y;
              }
              if (aux) {
#pragma unroll
                for (int u = 0; u < 8; u += 4) {
                  *reinterpret_cast<float4*>(aux + ch * 32 + j + u) = make_float4(o1[u], o1[u + 1], o1[u + 2], o1[u + 3]);
                  *reinterpret_cast<float4*>(aux + HALF + ch * 32 + j + u) =
                      make_float4(o2[u], o2[u + 1], o2[u + 2], o2[u + 3]);
                }
              }
#pragma unroll
              for (int u = 0; u < 8; ++u) { o1[u] *= a.scale; o2[u] *= a.scale; }
              uint32_t h1[4], l1[4], h2[4], l2[4];
#pragma unroll
              for (int u = 0; u < 8; u += 2) {
                const __nv_bfloat162 a1 = __floats2bfloat162_rn(o1[u], o1[u + 1]);
                const __nv_bfloat162 a2 = __floats2bfloat162_rn(o2[u], o2[u + 1]);
                h1[u / 2] = *reinterpret_cast<const uint32_t*>(&a1);
                h2[u / 2] = *reinterpret_cast<const uint32_t*>(&a2);
                l1[u / 2] = pack_bf16(o1[u] - __bfloat162float(a1.x), o1[u + 1] - __bfloat162float(a1.y));
                l2[u / 2] = pack_bf16(o2[u] - __bfloat162float(a2.x), o2[u + 1] - __bfloat162float(a2.y));
              }
              const uint4 H1 = make_uint4(h1[0], h1[1], h1[2], h1[3]), L1 = make_uint4(l1[0], l1[1], l1[2], l1[3]);
              const uint4 H2 = make_uint4(h2[0], h2[1], h2[2], h2[3]), L2 = make_uint4(l2[0], l2[1], l2[2], l2[3]);
#pragma unroll
              for (int sg = 0; sg < 3; ++sg) {
                __nv_bfloat16* o = out + sg * BN + ch * 32 + j;
                *reinterpret_cast<uint4*>(o) = sg == seg_lo ? L1 : H1;
                *reinterpret_cast<uint4*>(o + HALF) = sg == seg_lo ? L2 : H2;
              }
            }
          }
        }
      } else if constexpr (EPI == EPI_SM_STATS) {
        // column max / sum of exp over this warp's 32 rows (rows past M count as -inf):
        // the 32x32 chunk is transposed through shared memory, lane j reduces column j.
        float2* part = a.stats + (static_cast<long long>(c.b) * m_tiles * 4 + c.m_blk * 4 + lane_grp) * a.stat_ld;
        const int ncol = a.col_count ? min(lim, __ldg(a.col_count + c.b)) : lim;
        float* tr = xpose + (warp - 2) * 32 * 33;
#pragma unroll 1
        for (int ch = 0; ch < BN / 32; ++ch) {
          uint32_t r[32];
          tmem_ld32(tbase + ch * 32, r);
          const int cbase = col0 + ch * 32;
          if (cbase >= ncol) continue;                    // uniform in the warp
#pragma unroll
          for (int j = 0; j < 32; ++j) tr[lane * 33 + j] = row_ok ? __uint_as_float(r[j]) : -INFINITY;
          __syncwarp();
          float m = -INFINITY;
#pragma unroll
          for (int i = 0; i < 32; ++i) m = fmaxf(m, tr[i * 33 + lane]);
          float sum = 0.f;
          if (m != -INFINITY) {
#pragma unroll
            for (int i = 0; i < 32; ++i) sum += __expf(tr[i * 33 + lane] - m);
          }
          __syncwarp();
          if (cbase + lane < ncol) part[cbase + lane] = make_float2(m, sum);
        }
      } else if constexpr (EPI == EPI_SM_MEAN) {
        // p_hat[row] = (1/M_b) sum_col exp(l - c_col), c_col = max_col + ln(sum_col): each chunk's
        // 32 column normalisers are loaded once (lane j: column j) into this warp's shared row
        // and read back as broadcasts
        const int ncol = a.col_count ? min(lim, __ldg(a.col_count + c.b)) : lim;
        const float2* fin = a.stats + static_cast<long long>(c.b) * a.stat_ld;
        float* cn = xpose + (warp - 2) * 32;
        float acc_p = 0.f;
#pragma unroll 1
        for (int ch = 0; ch < BN / 32; ++ch) {
          uint32_t r[32];
          tmem_ld32(tbase + ch * 32, r);
          const int cbase = col0 + ch * 32;
          if (cbase >= ncol) continue;                    // uniform in the warp
          __syncwarp();                                   // the previous chunk's reads are done
          cn[lane] = cbase + lane < ncol ? __ldg(fin + cbase + lane).x : INFINITY;   // exp(-inf) = 0
          __syncwarp();
#pragma unroll
          for (int j = 0; j < 32; ++j) acc_p += __expf(__uint_as_float(r[j]) - cn[j]);
        }
        if (row < a.M) {   // rows past the image's valid tokens (m_limit) get 0
          float* out = reinterpret_cast<float*>(a.C) + static_cast<long long>(c.b) * a.c_batch_stride;
          out[static_cast<long long>(c.n_blk) * a.M + row] =
              row_ok ? acc_p / static_cast<float>(ncol > 0 ? ncol : 1) : 0.f;
        }
      } else if constexpr (EPI == EPI_PROJECT) {
        // Cholesky coordinates of token `row` on the R0 basis by forward substitution,
        // 32 basis vectors at a time: e_beta = (g_beta - sum_{q<beta} L[beta][q] e_q) / r_beta.
        // Each finished chunk of e replaces its g columns in TMEM, where later chunks read it.
        const ProjArgs& pj = a.proj;
        const int nb0 = min(BN, __ldg(pj.nbasis + c.b));
        const long long tok = static_cast<long long>(c.b) * a.M + row;
        const bool alive = row_ok && __ldg(pj.state + tok) == 0;
        float* erow = pj.Ec + tok * pj.KP;
        float sq = 0.f;
        {
          uint32_t dg[32];
          tmem_ld32(tmem_base + (static_cast<uint32_t>(lane_grp * 32) << 16) + 2 * BN + acc * kBM + lane_grp * 32, dg);
#pragma unroll
          for (int j = 0; j < 32; ++j) sq = j == lane ? __uint_as_float(dg[j]) : sq;
        }
        float r2 = sq;
#pragma unroll 1
        for (int b0 = 0; b0 < nb0; b0 += 32) {
          float accv[32];
          {
            uint32_t g[32];
            tmem_ld32(tbase + b0, g);
#pragma unroll
            for (int i = 0; i < 32; ++i) accv[i] = __uint_as_float(g[i]);
          }
          const int b1 = min(nb0, b0 + 32);
          const bool full32 = b1 - b0 > 16;             // uniform: rows 16..31 of this chunk exist
#pragma unroll 1
          for (int qc = 0; qc < b0; qc += 8) {
            uint32_t ep[8];
            tmem_ld8(tbase + qc, ep);
            if (alive) {
#pragma unroll
              for (int qq = 0; qq < 8; qq += 4) {
#pragma unroll
                for (int i = 0; i < 16; ++i) {
                  const float4 l = *reinterpret_cast<const float4*>(Lsm + (b0 + i) * BN + qc + qq);
                  accv[i] = fmaf(-l.x, __uint_as_float(ep[qq]), accv[i]);
                  accv[i] = fmaf(-l.y, __uint_as_float(ep[qq + 1]), accv[i]);
                  accv[i] = fmaf(-l.z, __uint_as_float(ep[qq + 2]), accv[i]);
                  accv[i] = fmaf(-l.w, __uint_as_float(ep[qq + 3]), accv[i]);
                }
                if (full32) {
#pragma unroll
                  for (int i = 16; i < 32; ++i) {
                    const float4 l = *reinterpret_cast<const float4*>(Lsm + (b0 + i) * BN + qc + qq);
                    accv[i] = fmaf(-l.x, __uint_as_float(ep[qq]), accv[i]);
                    accv[i] = fmaf(-l.y, __uint_as_float(ep[qq + 1]), accv[i]);
                    accv[i] = fmaf(-l.z, __uint_as_float(ep[qq + 2]), accv[i]);
                    accv[i] = fmaf(-l.w, __uint_as_float(ep[qq + 3]), accv[i]);
                  }
                }
              }
            }
          }
          // the triangle, in place: accv[i] becomes e_{b0+i}
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            float v = 0.f;
            if (alive && b0 + i < b1) {
              v = accv[i];
#pragma unroll
              for (int q = 0; q < i; ++q) v = fmaf(-Lsm[(b0 + i) * BN + b0 + q], accv[q], v);
              v *= rinv_sm[b0 + i];
              r2 = fmaf(-v, v, r2);
            }
            accv[i] = v;
          }
          if (alive) {
#pragma unroll
            for (int i = 0; i < 32; i += 4)
              if (b0 + i + 4 <= b1)
                *reinterpret_cast<float4*>(erow + b0 + i) = make_float4(accv[i], accv[i + 1], accv[i + 2], accv[i + 3]);
              else
                for (int u = i; u < b1 - b0 && u < i + 4; ++u) erow[b0 + u] = accv[u];
          }
          if (b0 + 32 < nb0) {
            uint32_t eb[32];
#pragma unroll
            for (int i = 0; i < 32; ++i) eb[i] = __float_as_uint(accv[i]);
            tmem_st32(tbase + b0, eb);
          }
        }
        if (alive) {
          pj.r2[tok] = r2;
          pj.sqn[tok] = sq;
          pj.U[tok] = proj_value(__ldg(pj.scores + tok), r2, sq, pj.lambda, pj.tau);
          pj.cstep[tok] = nb0;
        }
      } else if constexpr (EPI == EPI_F32) {
        float* out = reinterpret_cast<float*>(a.C) + crow + col0 + c.ks * a.c_split_stride;
#pragma unroll 1
        for (int ch = 0; ch < BN / 32; ++ch) {
          uint32_t r[32];
          tmem_ld32(tbase + ch * 32, r);
          const int cbase = col0 + ch * 32;
          if (row_ok && cbase < lim) {
            if (cbase + 32 <= lim) {
#pragma unroll
              for (int j = 0; j < 32; j += 4)
                *reinterpret_cast<float4*>(out + ch * 32 + j) =
                    make_float4(__uint_as_float(r[j]), __uint_as_float(r[j + 1]), __uint_as_float(r[j + 2]),
                                __uint_as_float(r[j + 3]));
            } else {
#pragma unroll
              for (int j = 0; j < 32; ++j)
                if (cbase + j < lim) out[ch * 32 + j] = __uint_as_float(r[j]);
            }
          }
        }
      } else if constexpr (S::TSTORE) {
        // (hi, lo) of each 32x32 chunk go through shared memory to two TMA box stores
        // (coalesced, asynchronous); buffers alternate, reused once their store has read them
        const int ew = warp - 2;
        const int y = c.b * a.a_row_stride + c.m_blk * kBM + lane_grp * 32;   // first row of this warp
#pragma unroll 1
        for (int ch = 0; ch < BN / 32; ++ch) {
          uint32_t r[32];
          tmem_ld32(tbase + ch * 32, r);
          const int cbase = col0 + ch * 32;
          uint8_t* hb = stg + (ew * 2 + (ch & 1)) * 4096;     // [hi 32x32 | lo 32x32] bf16
          if (lane == 0) bulk_wait_group_read<1>();      // this buffer's previous store has read it
          __syncwarp();
          uint32_t pk[16], pl[16];
#pragma unroll
          for (int j = 0; j < 32; j += 2) {
            float x0 = __uint_as_float(r[j]), x1 = __uint_as_float(r[j + 1]);
            if (a.bias) {
              const __nv_bfloat162 bb = __ldg(reinterpret_cast<const __nv_bfloat162*>(a.bias + cbase + j));
              x0 += __bfloat162float(bb.x);
              x1 += __bfloat162float(bb.y);
            }
            if constexpr (EPI == EPI_GELU_SPLIT) { x0 = gelu_erf(x0); x1 = gelu_erf(x1); }
            const __nv_bfloat162 hi = __floats2bfloat162_rn(x0, x1);
            pk[j / 2] = *reinterpret_cast<const uint32_t*>(&hi);
            pl[j / 2] = pack_bf16(x0 - __bfloat162float(hi.x), x1 - __bfloat162float(hi.y));
          }
          // 64-byte swizzle: 16-byte unit v of row r sits at unit v ^ ((r >> 1) & 3), so the
          // eight rows of a quarter warp hit distinct banks
          uint4* oh = reinterpret_cast<uint4*>(hb + lane * 64);
          uint4* ol = reinterpret_cast<uint4*>(hb + 2048 + lane * 64);
          const int sw = (lane >> 1) & 3;
#pragma unroll
          for (int v = 0; v < 4; ++v) {
            oh[v ^ sw] = make_uint4(pk[4 * v], pk[4 * v + 1], pk[4 * v + 2], pk[4 * v + 3]);
            ol[v ^ sw] = make_uint4(pl[4 * v], pl[4 * v + 1], pl[4 * v + 2], pl[4 * v + 3]);
          }
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0 && cbase < lim) {                  // rows past M are clipped by the store
            tma_store_2d(&tmC, hb, cbase, y);
            tma_store_2d(&tmC, hb + 2048, a.N + cbase, y);
            bulk_commit_group();
          }
        }
      } else {
        __nv_bfloat16* out = reinterpret_cast<__nv_bfloat16*>(a.C) + crow + col0;
#pragma unroll 1
        for (int ch = 0; ch < BN / 32; ++ch) {
          uint32_t r[32];
          tmem_ld32(tbase + ch * 32, r);
          const int cbase = col0 + ch * 32;
          if (row_ok && cbase < lim) {
            constexpr bool SPLIT = EPI == EPI_GELU_SPLIT || EPI == EPI_BIAS_SPLIT;
            uint32_t pk[16], pl[16];
#pragma unroll
            for (int j = 0; j < 32; j += 2) {
              float x0 = __uint_as_float(r[j]), x1 = __uint_as_float(r[j + 1]);
              if (a.bias) {
                const __nv_bfloat162 bb = __ldg(reinterpret_cast<const __nv_bfloat162*>(a.bias + cbase + j));
                x0 += __bfloat162float(bb.x);
                x1 += __bfloat162float(bb.y);
              }
              if constexpr (EPI == EPI_GELU_BF16 || EPI == EPI_GELU_SPLIT) { x0 = gelu_erf(x0); x1 = gelu_erf(x1); }
              const __nv_bfloat162 hi = __floats2bfloat162_rn(x0, x1);
              pk[j / 2] = *reinterpret_cast<const uint32_t*>(&hi);
              if constexpr (SPLIT) pl[j / 2] = pack_bf16(x0 - __bfloat162float(hi.x), x1 - __bfloat162float(hi.y));
            }
            uint4* o = reinterpret_cast<uint4*>(out + ch * 32);
#pragma unroll
            for (int v = 0; v < 4; ++v) o[v] = make_uint4(pk[4 * v], pk[4 * v + 1], pk[4 * v + 2], pk[4 * v + 3]);
            if constexpr (SPLIT) {
              uint4* ol = reinterpret_cast<uint4*>(out + a.N + ch * 32);
#pragma unroll
              for (int v = 0; v < 4; ++v) ol[v] = make_uint4(pl[4 * v], pl[4 * v + 1], pl[4 * v + 2], pl[4 * v + 3]);
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if constexpr (CG2) mbar_arrive_cluster(mapa_u32(&tempty[acc], 0));
        else mbar_arrive(&tempty[acc]);
      }
      acc ^= 1;
      if (acc == 0) acc_phase ^= 1;
    }
    if constexpr (S::TSTORE) {
      if (lane == 0) bulk_wait_group_all();              // every box store has completed
      __syncwarp();
    }
  }
  // Every role of this CTA has left its loop.  If one gave up (a bounded wait ran out), loads
  // may still be in flight that no MMA waited for: let them land before the CTA exits.  With
  // 2-SM pairs both CTAs' loads complete on the leader's barriers, which the leader drains.
  __syncthreads();
  if (*abort_flag && warp == 0 && lane == 0 && crank == 0) {
    for (int s = 0; s < STAGES; ++s)
      if (last_par[s] >= 0) mbar_wait(&full[s], static_cast<uint32_t>(last_par[s]), a.status, nullptr);
  }
  if constexpr (PAIR) cluster_sync();             // no commit or remote arrive still in flight
  else __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    if constexpr (CG2) tmem_dealloc_cg2(tmem_base, S::TMEM_COLS);
    else tmem_dealloc(tmem_base, S::TMEM_COLS);
  }
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

// 2D bf16 tensor map over [rows, K] (K contiguous), box 64 x box_rows, 128-byte swizzle.
bool make_map(CUtensorMap* m, const void* base, long long rows, int K, int box_rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(K) * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(kBK), static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

template <int BN, int STAGES, int EPI, bool PAIR = false>
cudaError_t run(const GemmDesc& d, const KArgs& ka, int num_sms, cudaStream_t st) {
  using S = Smem<BN, STAGES, EPI, PAIR>;
  CUtensorMap ta, tb;
  if (!make_map(&ta, d.A, d.a_rows_total, d.a_kwrap > 0 ? d.a_kwrap : d.K, kBM)) return cudaErrorInvalidValue;
  if (!make_map(&tb, d.B, d.b_rows_total, d.b_kwrap > 0 ? d.b_kwrap : d.K, PAIR ? BN / 2 : BN))
    return cudaErrorInvalidValue;
  CUtensorMap tc = ta;
  if constexpr (S::TSTORE) {       // output [rows, ldc] bf16, 32x32 boxes, 64-byte swizzle
    // box stores clip at a_rows_total, which is the row bound M only for one flat batch
    if (d.batch != 1 || d.a_rows_total != d.M) return cudaErrorInvalidValue;
    auto fn = encode_fn();
    if (!fn) return cudaErrorInvalidValue;
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(d.ldc), static_cast<cuuint64_t>(d.a_rows_total)};
    cuuint64_t strides[1] = {static_cast<cuuint64_t>(d.ldc) * 2};
    cuuint32_t box[2] = {32, 32};
    cuuint32_t estr[2] = {1, 1};
    if (fn(&tc, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, d.C, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
           CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) !=
        CUDA_SUCCESS)
      return cudaErrorInvalidValue;
  }
  auto kern = gemm_tc_kernel<BN, STAGES, EPI, PAIR>;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, S::TOTAL);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  const int m_tiles = (d.M + kBM - 1) / kBM, n_tiles = (d.N + BN - 1) / BN;
  if (PAIR) {
    const int units = d.batch * ((m_tiles + 1) / 2) * n_tiles * ka.ksplit;
    if (units == 0) return cudaSuccess;
    const int grid = 2 * std::max(1, std::min(units, num_sms / 2));
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(S::THREADS);
    cfg.dynamicSmemBytes = S::TOTAL;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = pdl_disabled() ? 0 : 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, kern, ta, tb, tc, ka);
  }
  const int tiles = d.batch * m_tiles * n_tiles * ka.ksplit;
  if (tiles == 0) return cudaSuccess;
  const int grid = std::max(1, std::min(tiles, num_sms));
  return launch_k(kern, dim3(grid), dim3(S::THREADS), S::TOTAL, st, ta, tb, tc, ka);
}

}  // namespace

cudaError_t launch_gemm(const GemmDesc& d, int num_sms, cudaStream_t st) {
  if (d.K <= 0 || d.K % kBK != 0 || d.M < 0 || d.N <= 0 || d.batch <= 0) return cudaErrorInvalidValue;
  if (d.a_kwrap < 0 || d.a_kwrap % kBK != 0 || d.a_kwrap > d.K) return cudaErrorInvalidValue;
  if (d.b_kwrap < 0 || d.b_kwrap % kBK != 0 || d.b_kwrap > d.K || (d.b_kwrap > 0 && d.split3))
    return cudaErrorInvalidValue;
  if (d.split3 && (d.K % (3 * kBK) != 0 || d.a_kwrap != 2 * (d.K / 3))) return cudaErrorInvalidValue;
  if ((reinterpret_cast<uintptr_t>(d.A) | reinterpret_cast<uintptr_t>(d.B)) & 15) return cudaErrorInvalidValue;
  if (d.M == 0) return cudaSuccess;
  // every output row and column block is written with 16-byte vector stores
  const bool scalar_out = d.epi == EPI_SM_STATS || d.epi == EPI_SM_MEAN;   // float / float2 stores
  const bool f32 = d.epi == EPI_F32 || d.epi == EPI_ROPE_F32;
  const long long vec = f32 ? 4 : 8;
  if (d.epi == EPI_PROJECT) {      // writes through ProjArgs only (float4 reads of Ec rows)
    if (d.proj.KP % 4 != 0 || !d.proj.Ec || (reinterpret_cast<uintptr_t>(d.proj.Ec) & 15)) return cudaErrorInvalidValue;
  } else if (!scalar_out &&
             (d.ldc % vec != 0 || d.c_batch_stride % vec != 0 || (reinterpret_cast<uintptr_t>(d.C) & 15))) {
    return cudaErrorInvalidValue;
  }
  if (scalar_out && (!d.stats || (reinterpret_cast<uintptr_t>(d.stats) & 7) || (reinterpret_cast<uintptr_t>(d.C) & 3)))
    return cudaErrorInvalidValue;
  if ((d.epi == EPI_GELU_SPLIT || d.epi == EPI_BIAS_SPLIT) && d.ldc < 2LL * d.N) return cudaErrorInvalidValue;
  KArgs ka;
  ka.M = d.M; ka.N = d.N; ka.K = d.K; ka.batch = d.batch;
  ka.a_row_stride = d.a_row_stride; ka.b_row_stride = d.b_row_stride;
  ka.n_limit = d.n_limit; ka.C = d.C; ka.ldc = d.ldc; ka.c_batch_stride = d.c_batch_stride;
  ka.bias = static_cast<const __nv_bfloat16*>(d.bias);
  ka.rope = d.rope; ka.rope_half = d.rope_half; ka.rope_ld = d.rope_ld; ka.pos = d.pos; ka.pos_mod = d.pos_mod > 0 ? d.pos_mod : 1;
  ka.status = d.status;
  ka.split_kind = d.split_kind; ka.scale = d.scale; ka.aux = d.aux; ka.b_off = d.b_off;
  ka.stats = d.stats; ka.stat_ld = d.stat_ld; ka.col_count = d.col_count;
  ka.b_base = d.b_base; ka.proj = d.proj;
  ka.a_kwrap = d.a_kwrap; ka.b_kwrap = d.b_kwrap; ka.biasf = d.biasf; ka.split3 = d.split3;
  ka.blist = d.blist; ka.bcount = d.blist ? d.bcount : nullptr;
  ka.m_limit = d.m_limit;
  ka.wait_ns = d.wait_ns > 0 ? static_cast<unsigned long long>(d.wait_ns) : kWaitLimitNs;
  // split-K: fp32 partial tiles only, every slice at least one K block
  if (d.ksplit < 1 || (d.ksplit > 1 && (d.epi != EPI_F32 || d.ksplit > d.K / kBK || d.c_split_stride % 4 != 0)))
    return cudaErrorInvalidValue;
  ka.ksplit = d.ksplit; ka.c_split_stride = d.c_split_stride;
  if (d.blist && !d.bcount) return cudaErrorInvalidValue;
  if (d.sym && (d.A != d.B || d.a_row_stride != d.b_row_stride || d.a_rows_total != d.b_rows_total || d.b_off ||
                d.a_kwrap || d.b_kwrap || d.split3))
    return cudaErrorInvalidValue;
  ka.sym = d.sym;
  ka.n_outer = d.n_outer;
  switch (d.epi) {
    case EPI_GELU_BF16:
      if (d.N % 256 == 0) return run<256, 4, EPI_GELU_BF16>(d, ka, num_sms, st);
      if (d.N % 64 == 0) return run<64, 8, EPI_GELU_BF16>(d, ka, num_sms, st);
      return cudaErrorInvalidValue;
    case EPI_BIAS_BF16:
      if (d.N % 256 == 0) return run<256, 4, EPI_BIAS_BF16>(d, ka, num_sms, st);
      if (d.N % 64 == 0) return run<64, 8, EPI_BIAS_BF16>(d, ka, num_sms, st);
      return cudaErrorInvalidValue;
    case EPI_ROPE_F32:
      if (d.N == 64) return run<64, 8, EPI_ROPE_F32>(d, ka, num_sms, st);
      if (d.N == 128) return run<128, 6, EPI_ROPE_F32>(d, ka, num_sms, st);
      if (d.N == 256) return run<256, 4, EPI_ROPE_F32>(d, ka, num_sms, st);
      return cudaErrorInvalidValue;
    case EPI_GELU_SPLIT:
      if (d.N % 256 == 0) return run<256, 6, EPI_GELU_SPLIT, true>(d, ka, num_sms, st);
      if (d.N % 64 == 0) return run<64, 8, EPI_GELU_SPLIT>(d, ka, num_sms, st);
      return cudaErrorInvalidValue;
    case EPI_BIAS_SPLIT:
      if (d.N % 256 == 0) return run<256, 6, EPI_BIAS_SPLIT, true>(d, ka, num_sms, st);
      if (d.N % 64 == 0) return run<64, 8, EPI_BIAS_SPLIT>(d, ka, num_sms, st);
      return cudaErrorInvalidValue;
    case EPI_ROPE_SPLIT3:   // dp = 128: 2-SM pairs share the B tile (each CTA loads 64 of its rows)
      if (d.N == 64) return run<64, 8, EPI_ROPE_SPLIT3>(d, ka, num_sms, st);
      if (d.N == 128) return run<128, 8, EPI_ROPE_SPLIT3, true>(d, ka, num_sms, st);
      return cudaErrorInvalidValue;
    case EPI_SM_STATS:
      return run<256, 4, EPI_SM_STATS>(d, ka, num_sms, st);
    case EPI_SM_MEAN:
      return run<256, 4, EPI_SM_MEAN>(d, ka, num_sms, st);
    case EPI_PROJECT:
      if (d.N > kProjMaxBasis || d.batch < 1) return cudaErrorInvalidValue;
      if (d.N <= 96) return run<96, 6, EPI_PROJECT>(d, ka, num_sms, st);
      return run<128, 5, EPI_PROJECT>(d, ka, num_sms, st);
    case EPI_F32:   // Gram blocks: one 256 x 256 pair tile per image and 256 columns
      if (d.M <= kBM && d.N <= 128) return run<128, 6, EPI_F32>(d, ka, num_sms, st);   // G[R0, R0]
      return run<256, 6, EPI_F32, true>(d, ka, num_sms, st);
    default:
      return cudaErrorInvalidValue;
  }
}

}  // namespace mapk
