// C ABI of libmap_gb300 (include/map_gb300.h): context, workspace, argument checks and
// the orchestration of the kernels for score (Eq. 3), select (Eq. 4) and gather.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <new>
#include <vector>

#include "../../include/map_gb300.h"
#include "kernels.h"
#include "ptx.cuh"
#include "select.h"

using mapk::GemmDesc;

namespace {

constexpr int kMaxKDiverse = 768;   // k limit when the diversity term is on (the coordinate update
                                    // stages 32 slot rows and 32 basis rows of k floats in shared memory)
constexpr int kProjMaxBasis = 128;  // basis vectors one projection pass takes
constexpr int kMaxK = 4096;
constexpr int kMaxN = 16384;

struct DevBuf {
  void* p = nullptr;
  size_t cap = 0;
};

struct TimedPair { cudaEvent_t a, b; int id; };

}  // namespace

struct map_ctx {
  map_config cfg{};
  int device = 0, num_sms = 148;
  void* w[10] = {};                 // wT1 bT1 wT2 bT2 wQ wV1 bV1 wV2 bV2 wK (device bf16)
  // W_Q f_T layer 2 and W_K f_V layer 2 folded (no nonlinearity between them): bf16 rows
  // [hi | hi | lo] of W_Q W_T2 / W_K W_V2 ([dp, 3 Dh]) and fp32 biases W_Q b_T2 / W_K b_V2
  void* wqt = nullptr; void* wkv = nullptr; float* bqt = nullptr; float* bkv = nullptr;
  DevBuf rope;  int rope_rows = 0;
  DevBuf h1, kb, th1, qb, stats, qoff, post, sqn, pmean, snv, dist, dsa, dsb, dsc;
  // selection
  DevBuf sU, sr2, scstep, sstate, sEc, spicks, sr0, sbt, srn, ssmall, stheta, saslot, sVg, sG;
  // map_prune staging
  DevBuf pvis, ptext, pout, pkeep, pscores;
  int* status = nullptr;            // device status word
  int* h_status = nullptr;          // pinned, mapped
  int32_t* h_done = nullptr;        // pinned, mapped
  int* h_status_dev = nullptr; int32_t* h_done_dev = nullptr;   // their device aliases
  cudaStream_t s_in = nullptr, s_out = nullptr;   // map_prune copy streams (host buffers)
  cudaStream_t s_aux = nullptr;     // question branch of the predictor, concurrent with the visual one
  cudaEvent_t ev_fork = nullptr, ev_join = nullptr;
  bool timing = false;
  std::vector<TimedPair> pairs;
  std::vector<cudaEvent_t> free_events;
  double t_ms[MAP_K_NUM] = {};
  long long t_n[MAP_K_NUM] = {};
  map_counters counters{};
  int deferred = MAP_OK;
  long long wait_ns = 0;            // GEMM role-wait limit (0: the kernels' default)
  mapk::SelLoopCache* loops = nullptr;   // cached graphs of the selection's device-side round loop
  long long* loop_iters_total = nullptr; // device: loop iterations run so far (one round each)
};

namespace {

int cuda_err(cudaError_t e) { return e == cudaSuccess ? MAP_OK : (e == cudaErrorMemoryAllocation ? MAP_ENOMEM : MAP_ECUDA); }

#define MAP_TRY(expr)                      \
  do {                                     \
    int _rc = (expr);                      \
    if (_rc != MAP_OK) return _rc;         \
  } while (0)
#define CU_TRY(expr) MAP_TRY(cuda_err(expr))

int ensure(DevBuf& b, size_t bytes) {
  if (bytes <= b.cap) return MAP_OK;
  if (b.p) {
    cudaError_t e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return MAP_ECUDA;
    cudaFree(b.p);
    b.p = nullptr;
    b.cap = 0;
  }
  size_t want = bytes + bytes / 8 + 256;
  if (cudaMalloc(&b.p, want) != cudaSuccess) {
    cudaGetLastError();
    return MAP_ENOMEM;
  }
  b.cap = want;
  return MAP_OK;
}

void release(DevBuf& b) {
  if (b.p) cudaFree(b.p);
  b.p = nullptr;
  b.cap = 0;
}

cudaEvent_t take_event(map_ctx* c) {
  if (!c->free_events.empty()) {
    cudaEvent_t e = c->free_events.back();
    c->free_events.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  cudaEventCreate(&e);
  return e;
}

// Brackets a launch with CUDA events when timing is on.
struct Timed {
  map_ctx* c; cudaStream_t st; int id; cudaEvent_t a = nullptr;
  Timed(map_ctx* c_, cudaStream_t st_, int id_) : c(c_), st(st_), id(id_) {
    if (c->timing) { a = take_event(c); cudaEventRecord(a, st); }
  }
  ~Timed() {
    if (a) {
      cudaEvent_t b = take_event(c);
      cudaEventRecord(b, st);
      c->pairs.push_back({a, b, id});
    }
  }
};

int dev_status_error(int st) {
  if (st & mapk::ST_TIMEOUT) return MAP_ETIMEOUT;
  if (st) return MAP_EINTERNAL;
  return MAP_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

int check_config(const map_config* c) {
  if (!c) return MAP_EINVAL;
  if (c->D <= 0 || c->D % 64 != 0) return MAP_EINVAL;
  if (c->Dh <= 0 || c->Dh % 256 != 0) return MAP_EINVAL;
  if (c->dp != 64 && c->dp != 128) return MAP_EINVAL;
  if (!(c->rope_theta > 0.f)) return MAP_EINVAL;
  if (!(c->lambda >= 0.f) || !(c->tau >= 0.f) || !(c->k0_frac >= 0.f)) return MAP_EINVAL;
  return MAP_OK;
}

int resolve_k0(const map_config& c, int K) {
  long long k0 = c.k0_abs >= 0 ? c.k0_abs : static_cast<long long>(std::floor(static_cast<double>(c.k0_frac) * K));
  if (k0 < 0) k0 = 0;
  if (k0 > K) k0 = K;
  return static_cast<int>(k0);
}

// RoPE table (cos, sin) of pos * theta^(-2i/dp), i < dp/2, for pos < rows; computed in
// double on the host, stored as float.
int ensure_rope(map_ctx* c, int rows_needed) {
  if (rows_needed <= c->rope_rows) return MAP_OK;
  const int rows = ((rows_needed + 1023) / 1024) * 1024;
  const int half = c->cfg.dp / 2;
  std::vector<float2> tab(static_cast<size_t>(rows) * half);
  for (int p = 0; p < rows; ++p)
    for (int i = 0; i < half; ++i) {
      const double f = std::pow(static_cast<double>(c->cfg.rope_theta), -2.0 * i / c->cfg.dp);
      const double a = p * f;
      tab[static_cast<size_t>(i) * rows + p] = make_float2(static_cast<float>(std::cos(a)), static_cast<float>(std::sin(a)));
    }
  MAP_TRY(ensure(c->rope, tab.size() * sizeof(float2)));
  CU_TRY(cudaMemcpy(c->rope.p, tab.data(), tab.size() * sizeof(float2), cudaMemcpyHostToDevice));
  c->rope_rows = rows;
  return MAP_OK;
}


int gemm(map_ctx* c, const GemmDesc& d, cudaStream_t st) {
  ++c->counters.launches;
  GemmDesc dd = d;
  dd.wait_ns = c->wait_ns;
  cudaError_t e = mapk::launch_gemm(dd, c->num_sms, st);
  if (e == cudaErrorInvalidValue) return MAP_EUNSUPPORTED;
  return cuda_err(e);
}

GemmDesc linear_desc(map_ctx* c, const void* x, long long rows, int K, const void* w, int Nout, const void* bias,
                     void* y, int epi) {
  GemmDesc d{};
  d.A = x; d.a_rows_total = rows; d.a_row_stride = 0;
  d.B = w; d.b_rows_total = Nout; d.b_row_stride = 0;
  d.M = static_cast<int>(rows); d.N = Nout; d.K = K; d.batch = 1;
  d.n_limit = nullptr; d.C = y; d.ldc = Nout; d.c_batch_stride = 0;
  d.bias = bias; d.rope = nullptr; d.rope_half = c->cfg.dp / 2; d.pos = nullptr; d.pos_mod = 1;
  d.epi = epi; d.status = c->status;
  return d;
}

// Predictor for one modality (Eq. 3): x [rows, D] -> RoPE(Wp f(x)) * scale [rows, dp] with
// f = Linear -> GELU -> Linear, stored as three bf16 segments [rows, 3 dp] (split_kind 0:
// hi|lo|hi, 1: hi|hi|lo) and, if aux is given, as fp32 too.  The hidden activation
// h1 = GELU(W1 x + b1) is kept as a bf16 hi/lo pair [rows, 2 Dh] (about 16 significant bits);
// the second layer and the projection are one folded matrix Wf = Wp W2 with bias Wp b2.
int predictor_branch(map_ctx* c, const void* x, long long rows, const void* w1, const void* b1, const void* wf,
                     const float* bf, DevBuf& h1, void* out3, int split_kind, float scale, float* aux,
                     const int* pos, int pos_mod, cudaStream_t st, int tid_l1, int tid_p) {
  const map_config& g = c->cfg;
  MAP_TRY(ensure(h1, static_cast<size_t>(rows) * g.Dh * 4));
  {
    Timed t(c, st, tid_l1);
    GemmDesc d = linear_desc(c, x, rows, g.D, w1, g.Dh, b1, h1.p, mapk::EPI_GELU_SPLIT);
    d.ldc = 2LL * g.Dh;
    MAP_TRY(gemm(c, d, st));
  }
  {
    // K = 3 Dh: h_hi Wf_hi + h_hi Wf_lo + h_lo Wf_hi, A = [hi | lo] against
    // [Wf_hi | Wf_hi | Wf_lo], each block of h_hi used twice in a row (split3 K order)
    Timed t(c, st, tid_p);
    GemmDesc d = linear_desc(c, h1.p, rows, 3 * g.Dh, wf, g.dp, nullptr, out3, mapk::EPI_ROPE_SPLIT3);
    d.a_kwrap = 2 * g.Dh;
    d.split3 = 1;
    d.biasf = bf;
    d.ldc = 3LL * g.dp;
    d.rope = static_cast<const float2*>(c->rope.p);
    d.rope_ld = c->rope_rows;
    d.pos = g.rope_on ? pos : nullptr;      // without RoPE every position is 0: cos 1, sin 0
    d.pos_mod = g.rope_on ? pos_mod : 1;
    d.split_kind = split_kind;
    d.scale = scale;
    d.aux = aux;
    MAP_TRY(gemm(c, d, st));
  }
  return MAP_OK;
}

// nv (host, B entries, or nullptr = every image has N tokens): valid visual tokens per image;
// rows at or past nv[b] are padding, excluded from Eq. 3 (their score is 0).
int score_impl(map_ctx* c, const void* text, const void* vis, const int32_t* lens, const int32_t* nv, int B, int N,
               float* scores, float* q_out, float* k_out, cudaStream_t st) {
  if (!c || !text || !vis || !lens || !scores) return MAP_EINVAL;
  if (B < 1 || N < 1) return MAP_EINVAL;
  if (nv)
    for (int b = 0; b < B; ++b)
      if (nv[b] < 1 || nv[b] > N) return MAP_EINVAL;
  if (!aligned16(text) || !aligned16(vis)) return MAP_EINVAL;
  long long total_m = 0;
  int max_m = 0;
  for (int b = 0; b < B; ++b) {
    if (lens[b] < 1) return MAP_EINVAL;
    total_m += lens[b];
    max_m = lens[b] > max_m ? lens[b] : max_m;
  }
  if (total_m > (1ll << 30) || static_cast<long long>(B) * N > (1ll << 30)) return MAP_EUNSUPPORTED;
  const map_config& g = c->cfg;
  CU_TRY(cudaSetDevice(c->device));
  MAP_TRY(ensure_rope(c, g.rope_on ? N + max_m + 1 : 1));
  // per-image query offsets, lengths and question-token positions N + m, written on the device
  const size_t off_bytes = static_cast<size_t>(B + 1) * 4, len_bytes = static_cast<size_t>(B) * 4;
  const size_t pos_bytes = static_cast<size_t>(total_m) * 4;
  MAP_TRY(ensure(c->qoff, off_bytes + 2 * len_bytes));
  MAP_TRY(ensure(c->post, pos_bytes));
  {
    std::vector<long long> offs(B);
    long long acc = 0;
    for (int b = 0; b < B; ++b) { offs[b] = acc; acc += lens[b]; }
    int32_t* qo = static_cast<int32_t*>(c->qoff.p);
    CU_TRY(mapk::launch_query_meta(lens, offs.data(), B, N, qo, qo + (B + 1), static_cast<int32_t*>(c->post.p), nv,
                                   nv ? qo + (2 * B + 1) : nullptr, st));
    c->counters.launches += (B + 1023) / 1024;
  }
  const int* d_off = static_cast<const int*>(c->qoff.p);
  const int* d_len = d_off + (B + 1);
  const int* d_nv = nv ? d_off + (2 * B + 1) : nullptr;

  const long long vrows = static_cast<long long>(B) * N;
  const int dp3 = 3 * g.dp;
  MAP_TRY(ensure(c->kb, static_cast<size_t>(vrows) * dp3 * 2));
  MAP_TRY(ensure(c->qb, static_cast<size_t>(total_m) * dp3 * 2));
  // The two branches are independent until Eq. 3: the question branch runs on a second stream
  // (it fills SMs that a small batch's visual GEMMs leave idle), joined before the logits.
  if (!c->s_aux) CU_TRY(cudaStreamCreateWithFlags(&c->s_aux, cudaStreamNonBlocking));
  if (!c->ev_fork) CU_TRY(cudaEventCreateWithFlags(&c->ev_fork, cudaEventDisableTiming));
  if (!c->ev_join) CU_TRY(cudaEventCreateWithFlags(&c->ev_join, cudaEventDisableTiming));
  CU_TRY(cudaEventRecord(c->ev_fork, st));
  CU_TRY(cudaStreamWaitEvent(c->s_aux, c->ev_fork, 0));
  MAP_TRY(predictor_branch(c, text, total_m, c->w[0], c->w[1], c->wqt, c->bqt, c->th1, c->qb.p, 1,
                           1.0f / std::sqrt(static_cast<float>(g.dp)), q_out, static_cast<const int*>(c->post.p), 1,
                           c->s_aux, MAP_K_GEMM_TEXT, MAP_K_GEMM_TEXT));
  CU_TRY(cudaEventRecord(c->ev_join, c->s_aux));
  MAP_TRY(predictor_branch(c, vis, vrows, c->w[5], c->w[6], c->wkv, c->bkv, c->h1, c->kb.p, 0, 1.0f, k_out, nullptr,
                           N, st, MAP_K_GEMM_FV1, MAP_K_GEMM_WK));
  CU_TRY(cudaStreamWaitEvent(st, c->ev_join, 0));
  // Eq. 3 on the tensor cores: logits tile [visual tokens x question tokens] of one image,
  // pass 1 -> per-slab column (max, sum exp), combine -> max + ln(sum), pass 2 -> mean.
  const int m_tiles = (N + 127) / 128, nparts = 4 * m_tiles;
  const int ld = ((max_m + 3) / 4) * 4;
  const int n_tiles = (max_m + 255) / 256;
  MAP_TRY(ensure(c->stats, static_cast<size_t>(B) * (nparts + 1) * ld * 8));
  float2* part = static_cast<float2*>(c->stats.p);
  float2* fin = part + static_cast<size_t>(B) * nparts * ld;
  GemmDesc d{};
  d.A = c->kb.p; d.a_rows_total = vrows; d.a_row_stride = N;
  d.B = c->qb.p; d.b_rows_total = total_m; d.b_row_stride = 0; d.b_off = d_off;
  d.M = N; d.N = max_m; d.K = dp3; d.batch = B; d.n_limit = d_len; d.col_count = d_len;
  d.m_limit = d_nv;
  d.status = c->status;
  float* mean_out = scores;
  if (n_tiles > 1) {
    MAP_TRY(ensure(c->pmean, static_cast<size_t>(vrows) * n_tiles * 4));
    mean_out = static_cast<float*>(c->pmean.p);
  }
  {
    Timed t(c, st, MAP_K_SCORES);
    d.epi = mapk::EPI_SM_STATS; d.stats = part; d.stat_ld = ld;
    d.C = part; d.ldc = 4; d.c_batch_stride = 0;
    MAP_TRY(gemm(c, d, st));
    ++c->counters.launches;
    CU_TRY(mapk::launch_stats_combine(part, B, nparts, ld, d_len, fin, st));
    d.epi = mapk::EPI_SM_MEAN; d.stats = fin;
    d.C = mean_out; d.ldc = 4; d.c_batch_stride = static_cast<long long>(N) * n_tiles;
    MAP_TRY(gemm(c, d, st));
    if (n_tiles > 1) {
      ++c->counters.launches;
      CU_TRY(mapk::launch_sum_tiles(mean_out, B, N, n_tiles, scores, st));
    }
  }
  return MAP_OK;
}

template <typename T>
T* carve(char*& p, size_t n) {
  T* r = reinterpret_cast<T*>(p);
  p += ((n * sizeof(T) + 255) / 256) * 256;
  return r;
}

// nv as for score_impl: tokens at or past nv[b] are never retained (K <= every nv[b]).
int select_impl(map_ctx* c, const float* scores, const void* vis, const int32_t* nv, int B, int N, int K,
                int32_t* keep, int32_t* order, cudaStream_t st) {
  if (!c || !scores || !vis) return MAP_EINVAL;
  if (B < 1 || N < 1 || K < 0 || K > N) return MAP_EINVAL;
  if (nv)
    for (int b = 0; b < B; ++b)
      if (nv[b] < 1 || nv[b] > N || K > nv[b]) return MAP_EINVAL;
  if (K == 0) return MAP_OK;
  if (!keep) return MAP_EINVAL;
  if (K > kMaxK || N > kMaxN) return MAP_EUNSUPPORTED;
  if (!aligned16(vis)) return MAP_EINVAL;
  CU_TRY(cudaSetDevice(c->device));
  Timed timed(c, st, MAP_K_SELECT);
  if (K == N) {
    ++c->counters.launches;
    CU_TRY(mapk::launch_sel_identity(B, N, keep, order, st));
    return MAP_OK;
  }
  const map_config& g = c->cfg;
  int K0 = resolve_k0(g, K);
  if (g.lambda == 0.f) K0 = K;        // values are p_hat alone: plain top-K
  if (K0 < K && K > kMaxKDiverse) return MAP_EUNSUPPORTED;
  const long long BN = static_cast<long long>(B) * N;
  const int S = mapk::kActiveSlots, R = ((S + K + 15) / 16) * 16;   // row stride of Vg and G (16-byte rows)

  mapk::SelState s{};
  const int KP = ((K + 3) / 4) * 4;
  s.B = B; s.N = N; s.D = g.D; s.K = K; s.K0 = K0; s.S = S; s.R = R; s.KP = KP;
  s.lambda = g.lambda; s.tau = g.tau;
  s.scores = scores; s.V = vis; s.status = c->status;
  if (nv) {                                      // valid tokens per image, on the device
    MAP_TRY(ensure(c->snv, static_cast<size_t>(B) * 4));
    c->counters.launches += (B + 2047) / 2048;
    CU_TRY(mapk::launch_put_ints(nv, B, static_cast<int32_t*>(c->snv.p), st));
    s.nvalid = static_cast<const int32_t*>(c->snv.p);
  }
  // per-token arrays
  MAP_TRY(ensure(c->sqn, BN * 4));
  MAP_TRY(ensure(c->sU, BN * 4));
  MAP_TRY(ensure(c->sr2, BN * 4));
  MAP_TRY(ensure(c->scstep, BN * 4));
  MAP_TRY(ensure(c->sstate, BN));
  MAP_TRY(ensure(c->spicks, static_cast<size_t>(B) * K * 4));
  MAP_TRY(ensure(c->sr0, static_cast<size_t>(B) * K * 4));
  MAP_TRY(ensure(c->sbt, static_cast<size_t>(B) * K * 4));
  MAP_TRY(ensure(c->srn, static_cast<size_t>(B) * K * 4));
  MAP_TRY(ensure(c->ssmall, static_cast<size_t>(B) * 4 * 16 + 24 * 256));
  static_assert(mapk::kReprojMax <= kProjMaxBasis, "re-projection basis limit");
  MAP_TRY(ensure(c->stheta, static_cast<size_t>(B) * 8));
  MAP_TRY(ensure(c->saslot, static_cast<size_t>(B) * S * 4));
  s.sqn = static_cast<float*>(c->sqn.p);
  s.U = static_cast<float*>(c->sU.p);
  s.r2 = static_cast<float*>(c->sr2.p);
  s.cstep = static_cast<int32_t*>(c->scstep.p);
  s.state = static_cast<uint8_t*>(c->sstate.p);
  s.picks = static_cast<int32_t*>(c->spicks.p);
  s.r0 = static_cast<int32_t*>(c->sr0.p);
  s.basis_tok = static_cast<int32_t*>(c->sbt.p);
  s.rnorm = static_cast<float*>(c->srn.p);
  char* sm = static_cast<char*>(c->ssmall.p);
  s.npicks = carve<int32_t>(sm, B);
  s.nbasis = carve<int32_t>(sm, B);
  s.nb_gathered = carve<int32_t>(sm, B);
  s.done = carve<int32_t>(sm, B);
  s.mode = carve<int32_t>(sm, B);
  s.nlimit = carve<int32_t>(sm, B);
  s.gb_lo = carve<int32_t>(sm, B);
  s.gb_hi = carve<int32_t>(sm, B);
  s.gbase = carve<int32_t>(sm, B);
  s.proj_lim = carve<int32_t>(sm, B);
  s.blist = carve<int32_t>(sm, B);
  s.bcount = carve<int32_t>(sm, 2);
  s.done_count = carve<int32_t>(sm, 1);
  s.uptr = carve<const void*>(sm, 2);
  int32_t* loop_iters = carve<int32_t>(sm, 1);
  s.theta = static_cast<uint64_t*>(c->stheta.p);
  s.aslot = static_cast<int32_t*>(c->saslot.p);

  // With 0 < K0 < K, one tensor-core pass over V after the first R0 tokens gives every
  // candidate its exact value on their basis (and ||v||^2); otherwise values start from
  // p_hat * ||v||^lambda.  The first K0c <= min(128, S) tokens of R0 are factored before the pass;
  // the rest of R0 is retained in the rounds after it, as forced picks, and every
  // value the pass gave stays a valid upper bound (values only shrink as the basis grows).
  const int K0c = std::min({K0, mapk::kCholMax, S});
  const bool project = K0 > 0 && K0 < K;
  if (K0 < K && !project) {
    ++c->counters.launches;
    CU_TRY(mapk::launch_row_sqnorm(vis, BN, g.D, static_cast<float*>(c->sqn.p), st));
  } else if (K0 >= K) {
    CU_TRY(cudaMemsetAsync(c->sqn.p, 0, BN * 4, st));
  }
  ++c->counters.launches;
  {
    mapk::SelState si = s;
    if (project) si.sqn = nullptr;     // written by the projection
    CU_TRY(mapk::launch_sel_init(si, st));
  }
  if (K0 < K) {
    MAP_TRY(ensure(c->sEc, static_cast<size_t>(BN) * KP * 4));
    MAP_TRY(ensure(c->sVg, static_cast<size_t>(B) * R * g.D * 2));
    MAP_TRY(ensure(c->sG, static_cast<size_t>(B) * S * R * 4));
    s.Ec = static_cast<float*>(c->sEc.p);
    s.Vg = c->sVg.p;
    s.G = static_cast<float*>(c->sG.p);
    GemmDesc d{};
    d.A = s.Vg; d.a_rows_total = static_cast<long long>(B) * R; d.a_row_stride = R;
    d.B = s.Vg; d.b_rows_total = static_cast<long long>(B) * R; d.b_row_stride = R;
    d.M = S; d.N = R; d.K = g.D; d.batch = B; d.n_limit = s.nlimit;
    d.C = s.G; d.ldc = R; d.c_batch_stride = static_cast<long long>(S) * R;
    d.epi = mapk::EPI_F32; d.status = c->status;
    d.sym = 1;                                   // A x A tiles load their rows once
    d.n_outer = 1;                               // the basis columns are often skipped
    d.blist = s.blist;                           // images still selecting (built by choose)
    // the GEMM after a list producer reads the count that producer appended through
    auto take_list = [&](GemmDesc& g) { g.bcount = s.bcount + s.bc_par; s.bc_par ^= 1; };
    // Rounds: every round picks or makes S stale bounds exact, so at most ceil(N / S) rounds
    // without a pick come before each pick; one more per kRoundPicks picks of a launch.
    const long long cap = static_cast<long long>(K) * ((N + S - 1) / S + 1) +
                          (K + mapk::kRoundPicks - 1) / mapk::kRoundPicks + 64;
    if (project) {
      // R0: gather its rows, G[R0, R0] on the tensor cores, then its Cholesky factor.
      c->counters.launches += 3;
      CU_TRY(mapk::launch_sel_choose(s, st));
      {
        GemmDesc d0 = d;              // only the K0c x K0c corner of the block
        d0.M = K0c; d0.N = K0c;
        take_list(d0);
        MAP_TRY(gemm(c, d0, st));
      }
      {
        mapk::SelState sc = s;        // the first K0c tokens of R0
        sc.K0 = K0c;
        CU_TRY(mapk::launch_sel_chol(sc, st));
      }
      ++c->counters.select_rounds;
      // every candidate's exact value: one tensor-core pass over V against the R0 basis
      GemmDesc pd{};
      pd.A = vis; pd.a_rows_total = BN; pd.a_row_stride = N;
      pd.B = s.Vg; pd.b_rows_total = static_cast<long long>(B) * R; pd.b_row_stride = R; pd.b_base = S;
      pd.M = N; pd.N = kProjMaxBasis; pd.K = g.D; pd.batch = B; pd.n_limit = s.proj_lim;
      pd.blist = s.blist;                         // images to project (built by proj_prep)
      pd.C = nullptr; pd.ldc = 0; pd.c_batch_stride = 0;
      pd.epi = mapk::EPI_PROJECT; pd.status = c->status;
      pd.proj.state = s.state; pd.proj.scores = scores; pd.proj.Ec = s.Ec; pd.proj.KP = KP;
      pd.proj.basis_tok = s.basis_tok; pd.proj.rnorm = s.rnorm; pd.proj.nbasis = s.nbasis; pd.proj.Kcap = K;
      pd.proj.lambda = g.lambda; pd.proj.tau = g.tau;
      pd.proj.r2 = s.r2; pd.proj.U = s.U; pd.proj.sqn = static_cast<float*>(c->sqn.p); pd.proj.cstep = s.cstep;
      auto project_all = [&](bool first) -> int {
        c->counters.launches += 3;
        CU_TRY(mapk::launch_sel_proj_prep(s, first, st));
        CU_TRY(mapk::launch_sel_gather(s, st));
        take_list(pd);
        MAP_TRY(gemm(c, pd, st));
        CU_TRY(mapk::launch_sel_proj_done(s, st));
        return MAP_OK;
      };
      pd.N = K0c <= 96 ? 96 : kProjMaxBasis;   // basis columns the R0 projection needs
      MAP_TRY(project_all(true));
      pd.N = kProjMaxBasis;
      // one round (greedy, or the rest of R0 when K0 > K0c), then the images still selecting are
      // projected again on their whole basis (when it has at most kReprojMax vectors): exact
      // values for every candidate make the next active set the true top S
      c->counters.launches += 5;
      CU_TRY(mapk::launch_sel_choose(s, st));
      take_list(d);
      MAP_TRY(gemm(c, d, st));
      CU_TRY(mapk::launch_sel_greedy(s, st));
      ++c->counters.select_rounds;
      MAP_TRY(project_all(false));
    }
    // The remaining rounds run as a device-side loop (a CUDA graph whose WHILE node repeats a
    // round while an image still selects): the host never waits for them.
    if (!c->loops) c->loops = mapk::sel_loop_cache_create();
    if (!c->loops) return MAP_ENOMEM;
    GemmDesc dl = d;
    dl.wait_ns = c->wait_ns;
    ++c->counters.launches;            // the test kernel ahead of the loop; iterations are counted on the device
    CU_TRY(mapk::launch_sel_loop(c->loops, s, dl, c->num_sms, static_cast<int>(cap), loop_iters,
                                 c->loop_iters_total, st));
  } else {
    ++c->counters.launches;
    CU_TRY(mapk::launch_sel_copy_r0(s.r0, B, K, s.picks, st));
  }
  ++c->counters.launches;
  CU_TRY(mapk::launch_sel_finalize(s.picks, B, K, keep, order, st));
  return MAP_OK;
}

int gather_impl(map_ctx* c, const void* vis, const int32_t* keep, int B, int N, int K, void* out, cudaStream_t st) {
  if (!c || !vis) return MAP_EINVAL;
  if (B < 1 || N < 1 || K < 0) return MAP_EINVAL;
  if (K == 0) return MAP_OK;
  if (!keep || !out) return MAP_EINVAL;
  if (!aligned16(vis) || !aligned16(out)) return MAP_EINVAL;
  CU_TRY(cudaSetDevice(c->device));
  Timed t(c, st, MAP_K_GATHER);
  ++c->counters.launches;
  CU_TRY(mapk::launch_gather(vis, keep, B, N, K, c->cfg.D, out, c->status, st));
  return MAP_OK;
}

int assemble_impl(map_ctx* ctx, const void* vis_feats, const int32_t* keep_idx, const void* text_feats,
                  const int32_t* lens, const int32_t* nv, int B, int N, int k, int pos_offset, void* seq,
                  int32_t* pos_ids, cudaStream_t st) {
  if (!ctx || !vis_feats || !text_feats || !lens) return MAP_EINVAL;
  if (B < 1 || N < 1 || k < 0 || k > N) return MAP_EINVAL;
  long long rows = 0;
  for (int b = 0; b < B; ++b) {
    if (lens[b] < 0) return MAP_EINVAL;
    if (nv && (nv[b] < 1 || nv[b] > N || k > nv[b])) return MAP_EINVAL;
    rows += k + lens[b];
  }
  if (rows == 0) return MAP_OK;
  if (!seq || !pos_ids || (k > 0 && !keep_idx)) return MAP_EINVAL;
  if (!aligned16(vis_feats) || !aligned16(text_feats) || !aligned16(seq)) return MAP_EINVAL;
  CU_TRY(cudaSetDevice(ctx->device));
  ++ctx->counters.launches;
  CU_TRY(mapk::launch_assemble(vis_feats, keep_idx, text_feats, lens, nv, B, N, k, ctx->cfg.D, pos_offset, seq,
                               pos_ids, ctx->status, st));
  return MAP_OK;
}

bool is_device_ptr(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged;
}

}  // namespace

// Read-only view of a context for other translation units of the library.
namespace mapk {
struct CtxView {
  const map_config* cfg;
  int device, num_sms;
  int* status;
  int32_t* h_done;
  long long* launches;
  long long* rounds;
  int* h_status;
  int32_t* h_done_dev;
  int* h_status_dev;
  int* deferred;
};
CtxView ctx_view(map_ctx* c) {
  return CtxView{&c->cfg, c->device, c->num_sms, c->status, c->h_done, &c->counters.launches,
                 &c->counters.select_rounds, c->h_status, c->h_done_dev, c->h_status_dev, &c->deferred};
}
}  // namespace mapk

extern "C" {

int map_config_default(map_config* cfg) {
  if (!cfg) return MAP_EINVAL;
  cfg->D = 4096; cfg->Dh = 1024; cfg->dp = 128;
  cfg->rope_theta = 10000.f; cfg->rope_on = 1;
  cfg->k0_frac = 0.5f; cfg->k0_abs = -1;
  cfg->lambda = 1.0f; cfg->tau = 1e-5f;
  return MAP_OK;
}

int map_init(const map_config* cfg, const map_weights* w, map_ctx** out) {
  if (!out) return MAP_EINVAL;
  *out = nullptr;
  if (check_config(cfg) != MAP_OK || !w) return MAP_EINVAL;
  const void* src[10] = {w->wT1, w->bT1, w->wT2, w->bT2, w->wQ, w->wV1, w->bV1, w->wV2, w->bV2, w->wK};
  for (const void* p : src)
    if (!p) return MAP_EINVAL;
  map_ctx* c = new (std::nothrow) map_ctx();
  if (!c) return MAP_ENOMEM;
  c->cfg = *cfg;
  int rc = MAP_OK;
  do {
    if (cudaGetDevice(&c->device) != cudaSuccess) { rc = MAP_ECUDA; break; }
    if (cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, c->device) != cudaSuccess) { rc = MAP_ECUDA; break; }
    const size_t D = cfg->D, Dh = cfg->Dh, dp = cfg->dp;
    const size_t rows[10] = {Dh, 1, Dh, 1, dp, Dh, 1, Dh, 1, dp};
    const size_t cols[10] = {D, Dh, Dh, Dh, Dh, D, Dh, Dh, Dh, Dh};
    for (int i = 0; i < 10 && rc == MAP_OK; ++i) {
      if (cudaMalloc(&c->w[i], rows[i] * cols[i] * 2) != cudaSuccess) { rc = MAP_ENOMEM; break; }
      if (cudaMemcpy(c->w[i], src[i], rows[i] * cols[i] * 2, cudaMemcpyDefault) != cudaSuccess) rc = MAP_ECUDA;
    }
    if (rc != MAP_OK) break;
    // The projections follow the second MLP layers with nothing in between: fold them.
    if (cudaMalloc(&c->wqt, dp * 3 * Dh * 2) != cudaSuccess || cudaMalloc(&c->wkv, dp * 3 * Dh * 2) != cudaSuccess ||
        cudaMalloc(reinterpret_cast<void**>(&c->bqt), dp * 4) != cudaSuccess ||
        cudaMalloc(reinterpret_cast<void**>(&c->bkv), dp * 4) != cudaSuccess) {
      rc = MAP_ENOMEM;
      break;
    }
    if (mapk::launch_fold_weights(c->w[4], c->w[2], c->w[3], static_cast<int>(dp), static_cast<int>(Dh), c->wqt,
                                  c->bqt, nullptr) != cudaSuccess ||
        mapk::launch_fold_weights(c->w[9], c->w[7], c->w[8], static_cast<int>(dp), static_cast<int>(Dh), c->wkv,
                                  c->bkv, nullptr) != cudaSuccess ||
        cudaDeviceSynchronize() != cudaSuccess) {
      rc = MAP_ECUDA;
      break;
    }
    if (cudaMalloc(reinterpret_cast<void**>(&c->loop_iters_total), sizeof(long long)) != cudaSuccess) {
      rc = MAP_ENOMEM;
      break;
    }
    if (cudaMemset(c->loop_iters_total, 0, sizeof(long long)) != cudaSuccess) { rc = MAP_ECUDA; break; }
    if (cudaMalloc(&c->status, sizeof(int)) != cudaSuccess) { rc = MAP_ENOMEM; break; }
    if (cudaMemset(c->status, 0, sizeof(int)) != cudaSuccess) { rc = MAP_ECUDA; break; }
    if (cudaHostAlloc(&c->h_status, sizeof(int), cudaHostAllocMapped) != cudaSuccess) { rc = MAP_ENOMEM; break; }
    if (cudaHostAlloc(&c->h_done, sizeof(int32_t), cudaHostAllocMapped) != cudaSuccess) { rc = MAP_ENOMEM; break; }
    if (cudaHostGetDevicePointer(reinterpret_cast<void**>(&c->h_status_dev), c->h_status, 0) != cudaSuccess ||
        cudaHostGetDevicePointer(reinterpret_cast<void**>(&c->h_done_dev), c->h_done, 0) != cudaSuccess) {
      rc = MAP_ECUDA;
      break;
    }
  } while (false);
  if (rc != MAP_OK) {
    cudaGetLastError();
    map_destroy(c);
    return rc;
  }
  *out = c;
  return MAP_OK;
}

int map_score(map_ctx* ctx, const void* text_feats, const void* vis_feats, const int32_t* lens, int B, int N,
              float* scores, void* stream) {
  return score_impl(ctx, text_feats, vis_feats, lens, nullptr, B, N, scores, nullptr, nullptr,
                    static_cast<cudaStream_t>(stream));
}

int map_score_debug(map_ctx* ctx, const void* text_feats, const void* vis_feats, const int32_t* lens, int B, int N,
                    float* scores, float* q_out, float* k_out, void* stream) {
  return score_impl(ctx, text_feats, vis_feats, lens, nullptr, B, N, scores, q_out, k_out,
                    static_cast<cudaStream_t>(stream));
}

int map_select(map_ctx* ctx, const float* scores, const void* vis_feats, int B, int N, int k, int32_t* keep_idx,
               int32_t* pick_order, void* stream) {
  return select_impl(ctx, scores, vis_feats, nullptr, B, N, k, keep_idx, pick_order,
                     static_cast<cudaStream_t>(stream));
}

int map_gather(map_ctx* ctx, const void* vis_feats, const int32_t* keep_idx, int B, int N, int k, void* out,
               void* stream) {
  return gather_impl(ctx, vis_feats, keep_idx, B, N, k, out, static_cast<cudaStream_t>(stream));
}

int map_assemble(map_ctx* ctx, const void* vis_feats, const int32_t* keep_idx, const void* text_feats,
                 const int32_t* lens, int B, int N, int k, int pos_offset, void* seq, int32_t* pos_ids,
                 void* stream) {
  return assemble_impl(ctx, vis_feats, keep_idx, text_feats, lens, nullptr, B, N, k, pos_offset, seq, pos_ids,
                       static_cast<cudaStream_t>(stream));
}

int map_assemble_ragged(map_ctx* ctx, const void* vis_feats, const int32_t* keep_idx, const void* text_feats,
                        const int32_t* lens, const int32_t* n_valid, int B, int N, int k, int pos_offset, void* seq,
                        int32_t* pos_ids, void* stream) {
  if (!n_valid) return MAP_EINVAL;
  return assemble_impl(ctx, vis_feats, keep_idx, text_feats, lens, n_valid, B, N, k, pos_offset, seq, pos_ids,
                       static_cast<cudaStream_t>(stream));
}

}  // extern "C"

namespace {
int prune_impl(map_ctx* ctx, const void* text_feats, const void* vis_feats, const int32_t* lens, const int32_t* nv,
               int B, int N, int k, void* out, int32_t* keep_idx, float* scores, void* stream) {
  if (!ctx || !text_feats || !vis_feats || !lens || !out || !keep_idx) return MAP_EINVAL;
  if (B < 1 || N < 1 || k < 0 || k > N) return MAP_EINVAL;
  if (nv)
    for (int b = 0; b < B; ++b)
      if (nv[b] < 1 || nv[b] > N || k > nv[b]) return MAP_EINVAL;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  map_ctx* c = ctx;
  CU_TRY(cudaSetDevice(c->device));
  long long total_m = 0;
  for (int b = 0; b < B; ++b) {
    if (lens[b] < 1) return MAP_EINVAL;
    total_m += lens[b];
  }
  const size_t D = c->cfg.D;
  const size_t vis_bytes = static_cast<size_t>(B) * N * D * 2, text_bytes = static_cast<size_t>(total_m) * D * 2;
  const size_t out_bytes = static_cast<size_t>(B) * k * D * 2, keep_bytes = static_cast<size_t>(B) * k * 4;
  const size_t sc_bytes = static_cast<size_t>(B) * N * 4;
  const bool dv = is_device_ptr(vis_feats), dt = is_device_ptr(text_feats), dout = is_device_ptr(out);
  const bool dkeep = is_device_ptr(keep_idx), dsc = scores ? is_device_ptr(scores) : true;
  const void* v = vis_feats;
  const void* t = text_feats;
  if (!dv) { MAP_TRY(ensure(c->pvis, vis_bytes)); v = c->pvis.p; }
  if (!dt) { MAP_TRY(ensure(c->ptext, text_bytes)); t = c->ptext.p; }
  void* o = out;
  int32_t* kp = keep_idx;
  float* sp = scores;
  if (!dout) { MAP_TRY(ensure(c->pout, out_bytes)); o = c->pout.p; }
  if (!dkeep) { MAP_TRY(ensure(c->pkeep, keep_bytes)); kp = static_cast<int32_t*>(c->pkeep.p); }
  if (!dsc || !scores) { MAP_TRY(ensure(c->pscores, sc_bytes)); sp = static_cast<float*>(c->pscores.p); }
  const bool host_io = !dv || !dt || !dout || !dkeep || (scores && !dsc);

  // With host buffers the batch runs as a pipeline of image chunks: chunk i+1 is copied in
  // (stream s_in) while chunk i is scored, selected and gathered (the caller's stream) and
  // chunk i-1 is copied out (stream s_out).  Results equal the one-shot path.
  const int nchunk = host_io ? std::min(B, 4) : 1;
  if (nchunk > 1) {
    if (!c->s_in) CU_TRY(cudaStreamCreateWithFlags(&c->s_in, cudaStreamNonBlocking));
    if (!c->s_out) CU_TRY(cudaStreamCreateWithFlags(&c->s_out, cudaStreamNonBlocking));
  }
  std::vector<long long> toff(B + 1, 0);
  for (int b = 0; b < B; ++b) toff[b + 1] = toff[b] + lens[b];
  cudaStream_t si = nchunk > 1 ? c->s_in : st, so = nchunk > 1 ? c->s_out : st;
  std::vector<cudaEvent_t> evs;
  auto ev = [&]() { cudaEvent_t e = take_event(c); evs.push_back(e); return e; };
  auto finish = [&](int rc) {
    for (cudaEvent_t e : evs) c->free_events.push_back(e);
    return rc;
  };
  if (nchunk > 1) {                         // buffers reused from earlier work on the caller's stream
    cudaEvent_t e0 = ev();
    if (cudaEventRecord(e0, st) != cudaSuccess || cudaStreamWaitEvent(si, e0, 0) != cudaSuccess ||
        cudaStreamWaitEvent(so, e0, 0) != cudaSuccess)
      return finish(MAP_ECUDA);
  }
  std::vector<cudaEvent_t> ev_in(nchunk);
  // Chunk boundaries, weights 3 : 3 : ... : 1.  The copy engine idles from the end of the last
  // copy-in until the call returns, i.e. while the last chunk is scored, selected, gathered and
  // copied out, so the last chunk is the small one; the others stay copy-bound.
  std::vector<int> cb(nchunk + 1, 0);
  {
    const int wsum = 3 * (nchunk - 1) + 1;
    for (int i = 1; i < nchunk; ++i) {
      const int v = static_cast<int>(static_cast<long long>(B) * 3 * i / wsum);
      cb[i] = std::min(std::max(v, cb[i - 1] + 1), B - (nchunk - i));
    }
    cb[nchunk] = B;
  }
  auto chunk = [&](int i, int& b0, int& b1) { b0 = cb[i]; b1 = cb[i + 1]; };
  for (int i = 0; i < nchunk; ++i) {
    int b0, b1;
    chunk(i, b0, b1);
    const size_t vo = static_cast<size_t>(b0) * N * D * 2, vn = static_cast<size_t>(b1 - b0) * N * D * 2;
    const size_t to = static_cast<size_t>(toff[b0]) * D * 2, tn = static_cast<size_t>(toff[b1] - toff[b0]) * D * 2;
    if (!dv && cudaMemcpyAsync(static_cast<char*>(c->pvis.p) + vo, static_cast<const char*>(vis_feats) + vo, vn,
                               cudaMemcpyHostToDevice, si) != cudaSuccess)
      return finish(MAP_ECUDA);
    if (!dt && cudaMemcpyAsync(static_cast<char*>(c->ptext.p) + to, static_cast<const char*>(text_feats) + to, tn,
                               cudaMemcpyHostToDevice, si) != cudaSuccess)
      return finish(MAP_ECUDA);
    ev_in[i] = ev();
    if (cudaEventRecord(ev_in[i], si) != cudaSuccess) return finish(MAP_ECUDA);
  }
  for (int i = 0; i < nchunk; ++i) {
    int b0, b1;
    chunk(i, b0, b1);
    const int Bc = b1 - b0;
    if (cudaStreamWaitEvent(st, ev_in[i], 0) != cudaSuccess) return finish(MAP_ECUDA);
    const void* vc = static_cast<const char*>(v) + static_cast<size_t>(b0) * N * D * 2;
    const void* tc = static_cast<const char*>(t) + static_cast<size_t>(toff[b0]) * D * 2;
    float* spc = sp + static_cast<size_t>(b0) * N;
    int32_t* kpc = kp + static_cast<size_t>(b0) * k;
    void* oc = static_cast<char*>(o) + static_cast<size_t>(b0) * k * D * 2;
    const int32_t* nvc = nv ? nv + b0 : nullptr;
    int rc = score_impl(c, tc, vc, lens + b0, nvc, Bc, N, spc, nullptr, nullptr, st);
    if (rc == MAP_OK) rc = select_impl(c, spc, vc, nvc, Bc, N, k, kpc, nullptr, st);
    if (rc == MAP_OK) rc = gather_impl(c, vc, kpc, Bc, N, k, oc, st);
    if (rc != MAP_OK) return finish(rc);
    if (host_io) {
      cudaEvent_t ed = ev();
      if (cudaEventRecord(ed, st) != cudaSuccess || cudaStreamWaitEvent(so, ed, 0) != cudaSuccess) return finish(MAP_ECUDA);
      const size_t oo = static_cast<size_t>(b0) * k * D * 2, on = static_cast<size_t>(Bc) * k * D * 2;
      const size_t ko = static_cast<size_t>(b0) * k * 4, kn = static_cast<size_t>(Bc) * k * 4;
      const size_t so_ = static_cast<size_t>(b0) * N * 4, sn = static_cast<size_t>(Bc) * N * 4;
      if (!dout && on && cudaMemcpyAsync(static_cast<char*>(out) + oo, static_cast<char*>(o) + oo, on,
                                         cudaMemcpyDeviceToHost, so) != cudaSuccess)
        return finish(MAP_ECUDA);
      if (!dkeep && kn && cudaMemcpyAsync(reinterpret_cast<char*>(keep_idx) + ko, reinterpret_cast<char*>(kp) + ko, kn,
                                          cudaMemcpyDeviceToHost, so) != cudaSuccess)
        return finish(MAP_ECUDA);
      if (scores && !dsc && cudaMemcpyAsync(reinterpret_cast<char*>(scores) + so_, reinterpret_cast<char*>(sp) + so_,
                                            sn, cudaMemcpyDeviceToHost, so) != cudaSuccess)
        return finish(MAP_ECUDA);
    }
  }
  if (host_io) {
    if (nchunk > 1) {
      cudaEvent_t ee = ev();
      if (cudaEventRecord(ee, so) != cudaSuccess || cudaStreamWaitEvent(st, ee, 0) != cudaSuccess) return finish(MAP_ECUDA);
    }
    if (cudaStreamSynchronize(st) != cudaSuccess) return finish(MAP_ECUDA);
  }
  return finish(MAP_OK);
}
}  // namespace

extern "C" {

int map_prune(map_ctx* ctx, const void* text_feats, const void* vis_feats, const int32_t* lens, int B, int N, int k,
              void* out, int32_t* keep_idx, float* scores, void* stream) {
  return prune_impl(ctx, text_feats, vis_feats, lens, nullptr, B, N, k, out, keep_idx, scores, stream);
}

int map_prune_ragged(map_ctx* ctx, const void* text_feats, const void* vis_feats, const int32_t* lens,
                     const int32_t* n_valid, int B, int N, int k, void* out, int32_t* keep_idx, float* scores,
                     void* stream) {
  if (!n_valid) return MAP_EINVAL;
  return prune_impl(ctx, text_feats, vis_feats, lens, n_valid, B, N, k, out, keep_idx, scores, stream);
}

int map_score_ragged(map_ctx* ctx, const void* text_feats, const void* vis_feats, const int32_t* lens,
                     const int32_t* n_valid, int B, int N, float* scores, void* stream) {
  if (!n_valid) return MAP_EINVAL;
  return score_impl(ctx, text_feats, vis_feats, lens, n_valid, B, N, scores, nullptr, nullptr,
                    static_cast<cudaStream_t>(stream));
}

int map_select_ragged(map_ctx* ctx, const float* scores, const void* vis_feats, const int32_t* n_valid, int B, int N,
                      int k, int32_t* keep_idx, int32_t* pick_order, void* stream) {
  if (!n_valid) return MAP_EINVAL;
  return select_impl(ctx, scores, vis_feats, n_valid, B, N, k, keep_idx, pick_order,
                     static_cast<cudaStream_t>(stream));
}

int map_distill_grad(map_ctx* ctx, const void* text_feats, const void* vis_feats, const int32_t* lens,
                     const float* teacher, int B, int N, float* loss, const map_grads* grads, void* stream) {
  if (!ctx || !text_feats || !vis_feats || !lens || !teacher || !loss || !grads) return MAP_EINVAL;
  float* gout[10] = {grads->wT1, grads->bT1, grads->wT2, grads->bT2, grads->wQ,
                     grads->wV1, grads->bV1, grads->wV2, grads->bV2, grads->wK};
  for (float* p : gout)
    if (!p) return MAP_EINVAL;
  if (B < 1 || N < 1) return MAP_EINVAL;
  long long total_m = 0;
  int max_m = 0;
  for (int b = 0; b < B; ++b) {
    if (lens[b] < 1) return MAP_EINVAL;
    total_m += lens[b];
    max_m = std::max(max_m, static_cast<int>(lens[b]));
  }
  if (total_m > (1ll << 24) || static_cast<long long>(B) * N > (1ll << 24)) return MAP_EUNSUPPORTED;
  map_ctx* c = ctx;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const map_config& g = c->cfg;
  const long long D = g.D, Dh = g.Dh, dp = g.dp, Tv = static_cast<long long>(B) * N, Tt = total_m;
  CU_TRY(cudaSetDevice(c->device));
  MAP_TRY(ensure_rope(c, g.rope_on ? N + max_m + 1 : 1));
  // question offsets and positions N + m (as for map_score), image of every question row
  MAP_TRY(ensure(c->qoff, static_cast<size_t>(3 * B + 1) * 4));
  MAP_TRY(ensure(c->post, static_cast<size_t>(total_m) * 4));
  std::vector<long long> offs(B);
  std::vector<int32_t> row_img(static_cast<size_t>(total_m));
  {
    long long acc = 0;
    for (int b = 0; b < B; ++b) {
      offs[b] = acc;
      for (int m = 0; m < lens[b]; ++m) row_img[static_cast<size_t>(acc + m)] = b;
      acc += lens[b];
    }
  }
  int32_t* qo = static_cast<int32_t*>(c->qoff.p);
  int32_t* post = static_cast<int32_t*>(c->post.p);
  CU_TRY(mapk::launch_query_meta(lens, offs.data(), B, N, qo, qo + (B + 1), post, nullptr, nullptr, st));
  // fp32 workspace (the features and weights stay bf16: the tensor-core GEMMs read them as exact
  // operands; only the biases are needed in fp32)
  const int nblk = (N + 255) / 256;
  const long long Np = (N + 3) / 4 * 4;              // logits row stride: 16-byte aligned rows
  const int bias_idx[4] = {1, 3, 6, 8};
  const long long floats = 4 * Dh + 5 * (Tv + Tt) * Dh + 4 * (Tv + Tt) * dp + Tt * Np + 2LL * B * N +
                           static_cast<long long>(B) * nblk + total_m + 64 * Dh + 64 * 16;
  MAP_TRY(ensure(c->dist, static_cast<size_t>(floats) * 4));
  float* base = static_cast<float*>(c->dist.p);
  auto take = [&](long long n) { float* p = base; base += ((n + 15) / 16) * 16; return p; };
  float* Wb[10] = {};
  for (int i : bias_idx) Wb[i] = take(Dh);
  float *z1v = take(Tv * Dh), *h1v = take(Tv * Dh), *h2v = take(Tv * Dh), *dh2v = take(Tv * Dh), *dh1v = take(Tv * Dh);
  float *z1t = take(Tt * Dh), *h1t = take(Tt * Dh), *h2t = take(Tt * Dh), *dh2t = take(Tt * Dh), *dh1t = take(Tt * Dh);
  float *kp = take(Tv * dp), *kk = take(Tv * dp), *dk = take(Tv * dp), *dkp = take(Tv * dp);
  float *qp = take(Tt * dp), *qq = take(Tt * dp), *dq = take(Tt * dp), *dqp = take(Tt * dp);
  float* S = take(Tt * Np);
  float *p_hat = take(static_cast<long long>(B) * N), *gb = take(static_cast<long long>(B) * N);
  float* part = take(static_cast<long long>(B) * nblk);
  int32_t* d_row_img = reinterpret_cast<int32_t*>(take(total_m));
  float* colpart = take(64 * Dh);                    // partial column sums of the bias gradients
  const float rs = 1.0f / std::sqrt(static_cast<float>(dp));
  // Every contraction of the step, in order: C = alpha A(M x K) B(K x N) with A(i, k) = ta ? A[k lda
  // + i] : A[i lda + k], B(k, j) = tb ? B[j ldb + k] : B[k ldb + j]; bf16 operands are exact.
  struct Mm { bool ta, tb; long long M, N, K; float alpha; const void* A; bool abf; long long lda;
              const void* Bm; bool bbf; long long ldb; float* C; long long ldc; };
  std::vector<Mm> fwd, mid, bwd;
  auto branch_fwd = [&](const void* X, long long T, int i1, float* z1, float* h1, float* h2, int ip, float* pre) {
    fwd.push_back({false, true, T, Dh, D, 1.f, X, true, D, c->w[i1], true, D, z1, Dh});
    fwd.push_back({false, true, T, Dh, Dh, 1.f, h1, false, Dh, c->w[i1 + 2], true, Dh, h2, Dh});
    fwd.push_back({false, true, T, dp, Dh, 1.f, h2, false, Dh, c->w[ip], true, Dh, pre, dp});
  };
  branch_fwd(vis_feats, Tv, 5, z1v, h1v, h2v, 9, kp);
  branch_fwd(text_feats, Tt, 0, z1t, h1t, h2t, 4, qp);
  for (int b = 0; b < B; ++b)     // Eq. 3 logits per image, then (after the loss) dq and dk
    mid.push_back({false, true, lens[b], N, dp, rs, qq + offs[b] * dp, false, dp, kk + b * N * dp, false, dp,
                   S + offs[b] * Np, Np});
  for (int b = 0; b < B; ++b) {
    mid.push_back({false, false, lens[b], dp, N, rs, S + offs[b] * Np, false, Np, kk + b * N * dp, false, dp,
                   dq + offs[b] * dp, dp});
    mid.push_back({true, false, N, dp, lens[b], rs, S + offs[b] * Np, false, Np, qq + offs[b] * dp, false, dp,
                   dk + b * N * dp, dp});
  }
  auto branch_bwd = [&](long long T, float* dpre, const void* X, int i1, const float* h1, const float* h2, float* dh2,
                        float* dh1, int ip) {
    bwd.push_back({true, false, dp, Dh, T, 1.f, dpre, false, dp, h2, false, Dh, gout[ip], Dh});
    bwd.push_back({false, false, T, Dh, dp, 1.f, dpre, false, dp, c->w[ip], true, Dh, dh2, Dh});
    bwd.push_back({true, false, Dh, Dh, T, 1.f, dh2, false, Dh, h1, false, Dh, gout[i1 + 2], Dh});
    bwd.push_back({false, false, T, Dh, Dh, 1.f, dh2, false, Dh, c->w[i1 + 2], true, Dh, dh1, Dh});
    bwd.push_back({true, false, Dh, D, T, 1.f, dh1, false, Dh, X, true, D, gout[i1], D});
  };
  branch_bwd(Tv, dkp, vis_feats, 5, h1v, h2v, dh2v, dh1v, 9);
  branch_bwd(Tt, dqp, text_feats, 0, h1t, h2t, dh2t, dh1t, 4);
  // staging buffers for the split-bf16 operands: the largest any contraction needs
  size_t wa = 0, wb = 0, wc = 0;
  for (const auto* list : {&fwd, &mid, &bwd})
    for (const Mm& m : *list) {
      size_t a = 0, bb = 0, cc = 0;
      mapk::tc_matmul_ws(static_cast<int>(m.M), static_cast<int>(m.N), static_cast<int>(m.K), m.alpha, m.abf, m.bbf,
                         c->num_sms, &a, &bb, &cc);
      wa = std::max(wa, a);
      wb = std::max(wb, bb);
      wc = std::max(wc, cc);
    }
  MAP_TRY(ensure(c->dsa, wa * 2));
  MAP_TRY(ensure(c->dsb, wb * 2));
  MAP_TRY(ensure(c->dsc, std::max<size_t>(wc, 4) * 4));
  long long mm_launches = 0;
  auto run_mm = [&](const Mm& m) -> int {
    cudaError_t e = mapk::launch_tc_matmul(m.ta, m.tb, static_cast<int>(m.M), static_cast<int>(m.N),
                                           static_cast<int>(m.K), m.alpha, m.A, m.abf, m.lda, m.Bm, m.bbf, m.ldb,
                                           m.C, m.ldc, c->dsa.p, c->dsb.p, static_cast<float*>(c->dsc.p), c->num_sms,
                                           c->status, c->wait_ns, st, &mm_launches);
    if (e == cudaErrorInvalidValue) return MAP_EUNSUPPORTED;
    return cuda_err(e);
  };
  CU_TRY(mapk::launch_put_ints(row_img.data(), static_cast<int>(total_m), d_row_img, st));
  for (int i : bias_idx) CU_TRY(mapk::launch_bf16_to_f32(c->w[i], Dh, Wb[i], st));
  const float2* tab = static_cast<const float2*>(c->rope.p);
  // forward: z1 = X W1^T + b1, h1 = GELU(z1), h2 = h1 W2^T + b2, projection, RoPE
  auto fwd_tail = [&](int j, long long T, int i1, float* z1, float* h1, float* h2, float* pre, float* post_rope,
                      const int32_t* pos, int pos_mod) -> int {
    MAP_TRY(run_mm(fwd[j]));
    CU_TRY(mapk::launch_bias_gelu(z1, Wb[i1 + 1], T, Dh, h1, st));
    MAP_TRY(run_mm(fwd[j + 1]));
    CU_TRY(mapk::launch_bias_add(h2, Wb[i1 + 3], T, Dh, st));
    MAP_TRY(run_mm(fwd[j + 2]));
    CU_TRY(mapk::launch_rope_f32(false, pre, T, dp, tab, c->rope_rows, pos, pos_mod, post_rope, st));
    return MAP_OK;
  };
  MAP_TRY(fwd_tail(0, Tv, 5, z1v, h1v, h2v, kp, kk, nullptr, g.rope_on ? N : 1));
  MAP_TRY(fwd_tail(3, Tt, 0, z1t, h1t, h2t, qp, qq, g.rope_on ? post : nullptr, 1));
  // Eq. 3 logits per image, softmax, KL, and dL/dlogits
  for (int b = 0; b < B; ++b) MAP_TRY(run_mm(mid[b]));
  CU_TRY(mapk::launch_distill_loss_grad(S, Np, total_m, qo, d_row_img, teacher, B, N, p_hat, gb, part, loss, st));
  for (size_t j = B; j < mid.size(); ++j) MAP_TRY(run_mm(mid[j]));
  // backward through RoPE, the projection and the MLP of each branch
  auto bwd_tail = [&](int j, float* dpost, long long T, const int32_t* pos, int pos_mod, float* dpre, const float* z1,
                      float* dh2, float* dh1, int i1) -> int {
    CU_TRY(mapk::launch_rope_f32(true, dpost, T, dp, tab, c->rope_rows, pos, pos_mod, dpre, st));
    MAP_TRY(run_mm(bwd[j]));                         // dW_p
    MAP_TRY(run_mm(bwd[j + 1]));                     // dh2
    MAP_TRY(run_mm(bwd[j + 2]));                     // dW2
    CU_TRY(mapk::launch_colsum(dh2, T, Dh, colpart, gout[i1 + 3], st));
    MAP_TRY(run_mm(bwd[j + 3]));                     // dh1
    CU_TRY(mapk::launch_gelu_back(dh1, z1, T * Dh, st));
    MAP_TRY(run_mm(bwd[j + 4]));                     // dW1
    CU_TRY(mapk::launch_colsum(dh1, T, Dh, colpart, gout[i1 + 1], st));
    return MAP_OK;
  };
  MAP_TRY(bwd_tail(0, dk, Tv, nullptr, g.rope_on ? N : 1, dkp, z1v, dh2v, dh1v, 5));
  MAP_TRY(bwd_tail(5, dq, Tt, g.rope_on ? post : nullptr, 1, dqp, z1t, dh2t, dh1t, 0));
  // query metadata, question-row images, 4 bias conversions, the contractions (the GEMM, its
  // operand stagings and the sum of its K slices, as counted by the launcher), 2 x 3 forward
  // elementwise, 4 loss / softmax-backward kernels, 2 x 6 backward elementwise (RoPE transpose,
  // GELU', two column sums of two launches each)
  c->counters.launches += (B + 1023) / 1024 + (total_m + 2047) / 2048 + 4 + mm_launches + 6 + 4 + 12;
  return MAP_OK;
}

int map_status(map_ctx* ctx, void* stream) {
  if (!ctx) return MAP_EINVAL;
  if (cudaSetDevice(ctx->device) != cudaSuccess) return MAP_ECUDA;
  cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return MAP_ECUDA;
  if (cudaMemcpy(ctx->h_status, ctx->status, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess) return MAP_ECUDA;
  int rc = dev_status_error(*ctx->h_status);
  if (*ctx->h_status) cudaMemset(ctx->status, 0, sizeof(int));
  if (rc == MAP_OK && ctx->deferred != MAP_OK) rc = ctx->deferred;
  ctx->deferred = MAP_OK;
  e = cudaGetLastError();
  if (rc == MAP_OK && e != cudaSuccess) rc = MAP_ECUDA;
  return rc;
}

void map_destroy(map_ctx* ctx) {
  if (!ctx) return;
  cudaSetDevice(ctx->device);
  cudaDeviceSynchronize();
  for (void*& p : ctx->w)
    if (p) cudaFree(p);
  for (void* p : {ctx->wqt, ctx->wkv, static_cast<void*>(ctx->bqt), static_cast<void*>(ctx->bkv)})
    if (p) cudaFree(p);
  DevBuf* bufs[] = {&ctx->rope, &ctx->h1, &ctx->kb, &ctx->th1, &ctx->qb, &ctx->stats,
                    &ctx->qoff, &ctx->post, &ctx->sqn, &ctx->pmean, &ctx->snv, &ctx->dist, &ctx->dsa, &ctx->dsb, &ctx->dsc, &ctx->sU, &ctx->sr2, &ctx->scstep, &ctx->sstate,
                    &ctx->sEc, &ctx->spicks, &ctx->sr0, &ctx->sbt, &ctx->srn, &ctx->ssmall, &ctx->stheta,
                    &ctx->saslot, &ctx->sVg, &ctx->sG, &ctx->pvis, &ctx->ptext, &ctx->pout, &ctx->pkeep,
                    &ctx->pscores};
  for (DevBuf* b : bufs) release(*b);
  if (ctx->status) cudaFree(ctx->status);
  if (ctx->loop_iters_total) cudaFree(ctx->loop_iters_total);
  mapk::sel_loop_cache_destroy(ctx->loops);
  if (ctx->h_status) cudaFreeHost(ctx->h_status);
  if (ctx->h_done) cudaFreeHost(ctx->h_done);
  if (ctx->s_in) cudaStreamDestroy(ctx->s_in);
  if (ctx->s_out) cudaStreamDestroy(ctx->s_out);
  if (ctx->s_aux) cudaStreamDestroy(ctx->s_aux);
  if (ctx->ev_fork) cudaEventDestroy(ctx->ev_fork);
  if (ctx->ev_join) cudaEventDestroy(ctx->ev_join);
  for (auto& pr : ctx->pairs) { cudaEventDestroy(pr.a); cudaEventDestroy(pr.b); }
  for (auto e : ctx->free_events) cudaEventDestroy(e);
  delete ctx;
}

const char* map_strerror(int code) {
  switch (code) {
    case MAP_OK: return "ok";
    case MAP_EINVAL: return "invalid argument";
    case MAP_ENOMEM: return "out of memory";
    case MAP_ECUDA: return "CUDA error";
    case MAP_ETIMEOUT: return "device-side wait timed out";
    case MAP_EUNSUPPORTED: return "unsupported shape";
    case MAP_EINTERNAL: return "device-side consistency check failed";
    default: return "unknown error";
  }
}

int map_get_counters(map_ctx* ctx, map_counters* out) {
  if (!ctx || !out) return MAP_EINVAL;
  *out = ctx->counters;
  long long iters = 0;   // iterations of the device-side selection loop (completed work)
  if (cudaSetDevice(ctx->device) != cudaSuccess ||
      cudaMemcpy(&iters, ctx->loop_iters_total, sizeof(iters), cudaMemcpyDeviceToHost) != cudaSuccess)
    return MAP_ECUDA;
  out->launches += mapk::kSelLoopKernelsPerIter * iters;
  out->select_rounds += iters;
  return MAP_OK;
}

int map_set_wait_limit(map_ctx* ctx, long long ns) {
  if (!ctx) return MAP_EINVAL;
  ctx->wait_ns = ns > 0 ? ns : 0;
  return MAP_OK;
}

int map_set_timing(map_ctx* ctx, int enable) {
  if (!ctx) return MAP_EINVAL;
  ctx->timing = enable != 0;
  return MAP_OK;
}

int map_read_timing(map_ctx* ctx, int id, double* total_ms, long long* count) {
  if (!ctx || id < 0 || id >= MAP_K_NUM || !total_ms || !count) return MAP_EINVAL;
  if (cudaDeviceSynchronize() != cudaSuccess) return MAP_ECUDA;
  for (auto& pr : ctx->pairs) {
    float ms = 0.f;
    cudaEventElapsedTime(&ms, pr.a, pr.b);
    ctx->t_ms[pr.id] += ms;
    ctx->t_n[pr.id] += 1;
    ctx->free_events.push_back(pr.a);
    ctx->free_events.push_back(pr.b);
  }
  ctx->pairs.clear();
  *total_ms = ctx->t_ms[id];
  *count = ctx->t_n[id];
  ctx->t_ms[id] = 0;
  ctx->t_n[id] = 0;
  return MAP_OK;
}

int map_linear(map_ctx* ctx, const void* x, const void* w, const void* b, int M, int K, int Nout, int epi, void* y,
               void* stream) {
  if (!ctx || !x || !w || !y || M < 0 || K <= 0 || Nout <= 0) return MAP_EINVAL;
  if (epi != mapk::EPI_GELU_BF16 && epi != mapk::EPI_BIAS_BF16 && epi != mapk::EPI_F32) return MAP_EINVAL;
  if (K % 64 != 0 || Nout % 64 != 0) return MAP_EUNSUPPORTED;
  if (!aligned16(x) || !aligned16(w) || !aligned16(y)) return MAP_EINVAL;
  if (cudaSetDevice(ctx->device) != cudaSuccess) return MAP_ECUDA;
  GemmDesc d = linear_desc(ctx, x, M, K, w, Nout, epi == mapk::EPI_F32 ? nullptr : b, y, epi);
  return gemm(ctx, d, static_cast<cudaStream_t>(stream));
}

}  // extern "C"
