// map_select_noalloc: the diversity-aware selection with no memory allocation in the call.
//
// Some callers cannot allocate device memory while they prune: code that runs inside
// another framework's caching pool or under a fixed device-memory budget (a cudaMalloc
// would take memory the budget does not have, or fail), and latency-bound serving paths
// that must not stall on the allocator (cudaMalloc / cudaFree may synchronise the device).
// map_select grows workspace owned by the context on demand; this entry point instead
// carves every buffer it needs from one file-scope device array of kNoAllocScratchBytes,
// which each GPU that loads this part of the library holds until the process exits.
//
// The array's device address is looked up once per device (cudaGetSymbolAddress, with
// that device current) by the first call made on that device; make that first call
// before any stream capture.  Every call shares the array and leaves its contents
// behind: the completion counter is cleared at the start of each call, everything else
// is written before it is read.  Calls whose work overlaps on the GPU (two streams, two
// host threads) race on the array and must be serialised by the caller.
//
// It runs the selection without the tensor-core projection pass that map_select uses
// when |R0| <= 128: every candidate starts from the bound p_hat * ||v||^lambda and the
// rounds of active sets (Gram blocks, coordinate updates, greedy picks) do the rest.
// The picks are the same exact greedy picks; only the number of rounds differs.
#include <cmath>
#include <mutex>

#include "../../include/map_gb300.h"
#include "kernels.h"
#include "ptx.cuh"
#include "select.h"

namespace mapk {
struct CtxView {
  const map_config* cfg;
  int device, num_sms;
  int* status;
  int32_t* h_done;
  long long* launches;
  long long* rounds;
  int* h_status;                     // host-mapped words and their device aliases
  int32_t* h_done_dev;
  int* h_status_dev;
  int* deferred;                     // error reported by the next map_status
};
CtxView ctx_view(map_ctx* c);
}  // namespace mapk

namespace {

constexpr size_t kNoAllocScratchBytes = MAP_NOALLOC_SCRATCH_BYTES;
constexpr int kSelS = mapk::kActiveSlots;
constexpr int kMaxDevices = 64;
constexpr int kMaxN = 16384;
constexpr int kMaxK = 4096;          // plain top-k
constexpr int kMaxKDiverse = 768;    // with the diversity term (as map_select)

static __device__ __align__(256) unsigned char g_scratch[kNoAllocScratchBytes];

std::mutex g_mu;
void* g_scratch_ptr[kMaxDevices] = {};

// Device address of g_scratch for the current device (looked up once per device).
int scratch_for_device(int dev, void** out) {
  if (dev < 0 || dev >= kMaxDevices) return MAP_EUNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_scratch_ptr[dev]) {
    void* p = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&p, g_scratch);
    if (e != cudaSuccess || p == nullptr) {
      cudaGetLastError();
      return MAP_ECUDA;
    }
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
  return MAP_OK;
}

// Bump allocator over the scratch array (256-byte aligned pieces).
struct Carver {
  char* base;
  size_t used = 0, cap;
  template <typename T>
  T* take(size_t n) {
    T* r = reinterpret_cast<T*>(base + used);
    used += ((n * sizeof(T) + 255) / 256) * 256;
    return r;
  }
  bool ok() const { return used <= cap; }
};

int k0_of(const map_config& c, int K) {
  long long k0 = c.k0_abs >= 0 ? c.k0_abs : static_cast<long long>(std::floor(static_cast<double>(c.k0_frac) * K));
  return static_cast<int>(k0 < 0 ? 0 : (k0 > K ? K : k0));
}

int rc_of(cudaError_t e) { return e == cudaSuccess ? MAP_OK : MAP_ECUDA; }

}  // namespace

extern "C" int map_select_noalloc(map_ctx* ctx, const float* scores, const void* vis_feats, int B, int N, int k,
                                  int32_t* keep_idx, int32_t* pick_order, void* stream) {
  if (!ctx || !scores || !vis_feats) return MAP_EINVAL;
  if (B < 1 || N < 1 || k < 0 || k > N) return MAP_EINVAL;
  if (k == 0) return MAP_OK;
  if (!keep_idx) return MAP_EINVAL;
  if ((reinterpret_cast<uintptr_t>(vis_feats) & 15) != 0) return MAP_EINVAL;
  if (N > kMaxN || k > kMaxK) return MAP_EUNSUPPORTED;
  mapk::CtxView v = mapk::ctx_view(ctx);
  const map_config& g = *v.cfg;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (cudaSetDevice(v.device) != cudaSuccess) return MAP_ECUDA;
  void* base = nullptr;
  int rc = scratch_for_device(v.device, &base);
  if (rc != MAP_OK) return rc;

  if (k == N) {
    ++*v.launches;
    return rc_of(mapk::launch_sel_identity(B, N, keep_idx, pick_order, st));
  }
  int K0 = k0_of(g, k);
  if (g.lambda == 0.f) K0 = k;
  if (K0 < k && k > kMaxKDiverse) return MAP_EUNSUPPORTED;
  const int K = k, S = kSelS, R = ((kSelS + K + 15) / 16) * 16, KP = ((K + 3) / 4) * 4;
  const long long BN = static_cast<long long>(B) * N;

  Carver cv{static_cast<char*>(base), 0, kNoAllocScratchBytes};
  mapk::SelState s{};
  s.B = B; s.N = N; s.D = g.D; s.K = K; s.K0 = K0; s.S = S; s.R = R; s.KP = KP;
  s.lambda = g.lambda; s.tau = g.tau;
  s.scores = scores; s.V = vis_feats; s.status = v.status;
  float* sqn = cv.take<float>(BN);
  s.sqn = sqn;
  s.U = cv.take<float>(BN);
  s.r2 = cv.take<float>(BN);
  s.cstep = cv.take<int32_t>(BN);
  s.state = cv.take<uint8_t>(BN);
  s.picks = cv.take<int32_t>(static_cast<size_t>(B) * K);
  s.r0 = cv.take<int32_t>(static_cast<size_t>(B) * K);
  s.basis_tok = cv.take<int32_t>(static_cast<size_t>(B) * K);
  s.rnorm = cv.take<float>(static_cast<size_t>(B) * K);
  s.npicks = cv.take<int32_t>(B);
  s.nbasis = cv.take<int32_t>(B);
  s.nb_gathered = cv.take<int32_t>(B);
  s.done = cv.take<int32_t>(B);
  s.mode = cv.take<int32_t>(B);
  s.nlimit = cv.take<int32_t>(B);
  s.gb_lo = cv.take<int32_t>(B);
  s.gb_hi = cv.take<int32_t>(B);
  s.gbase = cv.take<int32_t>(B);
  s.done_count = cv.take<int32_t>(1);
  s.theta = cv.take<uint64_t>(B);
  s.aslot = cv.take<int32_t>(static_cast<size_t>(B) * S);
  if (K0 < K) {
    s.Ec = cv.take<float>(static_cast<size_t>(BN) * KP);
    s.Vg = cv.take<uint16_t>(static_cast<size_t>(B) * R * g.D);
    s.G = cv.take<float>(static_cast<size_t>(B) * S * R);
  }
  if (!cv.ok()) return MAP_EUNSUPPORTED;      // workspace larger than the static array

  if (K0 < K) {
    ++*v.launches;
    rc = rc_of(mapk::launch_row_sqnorm(vis_feats, BN, g.D, sqn, st));
  } else {
    rc = rc_of(cudaMemsetAsync(sqn, 0, BN * 4, st));
  }
  if (rc != MAP_OK) return rc;
  ++*v.launches;
  if ((rc = rc_of(mapk::launch_sel_init(s, st))) != MAP_OK) return rc;
  if (K0 < K) {                   // sel_init has zeroed done_count
    mapk::GemmDesc d{};
    d.A = s.Vg; d.a_rows_total = static_cast<long long>(B) * R; d.a_row_stride = R;
    d.B = s.Vg; d.b_rows_total = static_cast<long long>(B) * R; d.b_row_stride = R;
    d.M = S; d.N = R; d.K = g.D; d.batch = B; d.n_limit = s.nlimit;
    d.C = s.G; d.ldc = R; d.c_batch_stride = static_cast<long long>(S) * R;
    d.epi = mapk::EPI_F32; d.status = v.status;
    d.sym = 1;                                   // A x A tiles load their rows once
    d.n_outer = 1;                               // the basis columns are often skipped
    // every round picks or makes S stale bounds exact: at most ceil(N / S) rounds without a
    // pick come before each pick
    const long long cap = static_cast<long long>(K) * ((N + S - 1) / S + 1) +
                          (K + mapk::kRoundPicks - 1) / mapk::kRoundPicks + 64;
    long long rounds = 0;
    int burst = (K0 + mapk::kRoundPicks - 1) / mapk::kRoundPicks + 6;
    for (;;) {
      for (int r = 0; r < burst; ++r) {
        *v.launches += 6;
        if ((rc = rc_of(mapk::launch_sel_choose(s, st))) != MAP_OK) return rc;
        cudaError_t e = mapk::launch_gemm(d, v.num_sms, st);
        if (e == cudaErrorInvalidValue) return MAP_EUNSUPPORTED;
        if ((rc = rc_of(e)) != MAP_OK) return rc;
        if ((rc = rc_of(mapk::launch_sel_greedy(s, st))) != MAP_OK) return rc;
      }
      rounds += burst;
      *v.rounds += burst;
      // completion and device status through host-mapped words (no copy engine)
      ++*v.launches;
      if ((rc = rc_of(mapk::launch_flags_to_host(s.done_count, v.status, v.h_done_dev, v.h_status_dev, st))) != MAP_OK)
        return rc;
      if ((rc = rc_of(cudaStreamSynchronize(st))) != MAP_OK) return rc;
      if (*v.h_done >= B) break;
      if (*v.h_status) {              // a kernel gave up (bounded wait) or saw a bad index: stop here
        *v.deferred = (*v.h_status & mapk::ST_TIMEOUT) ? MAP_ETIMEOUT : MAP_EINTERNAL;
        return *v.deferred;
      }
      if (rounds > cap) {
        *v.deferred = MAP_EINTERNAL;
        return MAP_EINTERNAL;
      }
      burst = 2;
    }
  } else {
    ++*v.launches;
    if ((rc = rc_of(mapk::launch_sel_copy_r0(s.r0, B, K, s.picks, st))) != MAP_OK) return rc;
  }
  ++*v.launches;
  return rc_of(mapk::launch_sel_finalize(s.picks, B, K, keep_idx, pick_order, st));
}
