// C ABI of the BCMT token mixer: argument validation, workspace layout, and
// the launch sequence of the forward (Sec. 3.2-3.8) and backward passes on the
// caller's stream.  No device memory is allocated per call.
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <algorithm>
#include <array>
#include <memory>
#include <mutex>
#include <string>
#include <vector>

#include "../../include/bcmt.h"
#include "../../include/bcmt_testing.h"
#include "common.cuh"
#include "internal.h"
#include "tc.cuh"

namespace bcmt {

// Device status word: kernels OR kStatus* bits into it when a bounded wait
// expires.  Module-scope, one per device; its device address is looked up
// once per device.
__device__ unsigned g_status_word;

namespace {

thread_local std::string g_last_error;

bcmt_status fail(bcmt_status code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return code;
}

unsigned* status_ptr() {
  static std::mutex mu;
  static std::vector<unsigned*> per_dev;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return nullptr;
  std::lock_guard<std::mutex> lk(mu);
  if ((int)per_dev.size() <= dev) per_dev.resize(dev + 1, nullptr);
  if (!per_dev[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_status_word) != cudaSuccess) return nullptr;
    per_dev[dev] = static_cast<unsigned*>(p);
  }
  return per_dev[dev];
}

// Side streams per device for work that runs beside the layer's critical
// chain (the memory gradient and the small weight gradients of the backward
// pass): forked from and joined back into the caller's stream with events,
// so the branches can also be captured into a CUDA graph.  The critical chain
// itself stays on the caller's stream, so that consecutive calls (forward,
// then backward) chain by programmatic dependent launch; its launches carry
// the device's highest stream priority as a launch attribute, the side
// streams the lowest, so that when both have CTAs waiting the block scheduler
// places the critical ones first.  Streams and events are host-side objects:
// no device memory.
constexpr int kSideEvents = 16;
struct SideStream {
  cudaStream_t side = nullptr, side2 = nullptr;
  int greatest = 0;  // the device's highest stream priority
  cudaEvent_t ev[kSideEvents] = {};
  std::mutex mu;  // one call at a time may use the streams' events
};

SideStream* side_stream() {
  static std::mutex mu;
  static std::vector<SideStream*> per_dev;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return nullptr;
  std::lock_guard<std::mutex> lk(mu);
  if ((int)per_dev.size() <= dev) per_dev.resize(dev + 1, nullptr);
  if (!per_dev[dev]) {
    SideStream* ss = new SideStream();
    int least = 0, greatest = 0;
    bool ok = cudaDeviceGetStreamPriorityRange(&least, &greatest) == cudaSuccess &&
              cudaStreamCreateWithPriority(&ss->side, cudaStreamNonBlocking, least) == cudaSuccess &&
              cudaStreamCreateWithPriority(&ss->side2, cudaStreamNonBlocking, least) == cudaSuccess;
    ss->greatest = greatest;
    for (int i = 0; i < kSideEvents && ok; ++i)
      ok = cudaEventCreateWithFlags(&ss->ev[i], cudaEventDisableTiming) == cudaSuccess;
    if (!ok) {
      delete ss;  // fall back to the caller's stream alone
      return nullptr;
    }
    per_dev[dev] = ss;
  }
  return per_dev[dev];
}

// Fork/join of one call: the critical chain runs on the caller's stream at
// the highest priority; the side streams fork from it at point() / point2(),
// and on destruction (every return path) they are joined back into it.
// Plain event record/wait, so a CUDA graph capture of the caller's stream
// captures every branch.  Without a SideStream everything stays on the
// caller's stream at its own priority.
struct Fork {
  SideStream* ss;
  cudaStream_t user;
  int next = 0;
  bool forked = false, forked2 = false;
  PriorityOverride saved;
  Fork(SideStream* s, cudaStream_t u) : ss(s), user(u) {
    if (!ss) return;
    ss->mu.lock();
    saved = priority_override();
    priority_override() = PriorityOverride{true, user, ss->greatest};
  }
  cudaStream_t main() const { return user; }
  cudaStream_t side() const { return ss ? ss->side : user; }
  cudaStream_t side2() const { return ss ? ss->side2 : user; }
  // the side stream waits for everything enqueued on the critical chain so far
  bool point() {
    if (!ss || next >= kSideEvents - 3) return false;
    cudaEventRecord(ss->ev[next], user);
    cudaStreamWaitEvent(ss->side, ss->ev[next], 0);
    ++next;
    forked = true;
    return true;
  }
  // the same for the second side stream
  bool point2() {
    if (!ss || next >= kSideEvents - 3) return false;
    cudaEventRecord(ss->ev[next], user);
    cudaStreamWaitEvent(ss->side2, ss->ev[next], 0);
    ++next;
    forked2 = true;
    return true;
  }
  // records what the side stream has been given so far; wait_mark(m) later
  // makes the critical chain wait for exactly that
  int mark() {
    if (!ss || !forked || next >= kSideEvents - 3) return -1;
    cudaEventRecord(ss->ev[next], ss->side);
    return next++;
  }
  void wait_mark(int m) {
    if (ss && m >= 0) cudaStreamWaitEvent(user, ss->ev[m], 0);
  }
  ~Fork() {
    if (!ss) return;
    if (forked2) {
      cudaEventRecord(ss->ev[kSideEvents - 3], ss->side2);
      cudaStreamWaitEvent(user, ss->ev[kSideEvents - 3], 0);
    }
    if (forked) {
      cudaEventRecord(ss->ev[kSideEvents - 2], ss->side);
      cudaStreamWaitEvent(user, ss->ev[kSideEvents - 2], 0);
    }
    priority_override() = saved;
    ss->mu.unlock();
  }
};

// Tensor-core paths of the layer (switchable only through bcmt_testing.h).
bool g_use_tc_gemm = true;
bool g_use_tc_attn = true;

// ------------------------------------------------------------------ profiling
struct ProfRec {
  const char* name;
  cudaEvent_t a, b;
};
std::mutex g_prof_mu;
std::vector<ProfRec> g_prof_recs;
std::vector<cudaEvent_t> g_prof_pool;
size_t g_prof_pool_used = 0;
constexpr size_t kProfMaxRecs = 1 << 16;

cudaEvent_t prof_event() {
  if (g_prof_pool_used == g_prof_pool.size()) {
    cudaEvent_t e;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    g_prof_pool.push_back(e);
  }
  return g_prof_pool[g_prof_pool_used++];
}

struct Prof {
  bool on;
  cudaStream_t s;
  cudaEvent_t a = nullptr;
  const char* name = nullptr;
  void begin(const char* n) {
    if (!on) return;
    std::lock_guard<std::mutex> lk(g_prof_mu);
    if (g_prof_recs.size() >= kProfMaxRecs) return;
    name = n;
    a = prof_event();
    if (a) cudaEventRecord(a, s);
  }
  void end(const char* n) {
    if (!on || !a) return;
    std::lock_guard<std::mutex> lk(g_prof_mu);
    cudaEvent_t b = prof_event();
    if (!b) return;
    cudaEventRecord(b, s);
    g_prof_recs.push_back({n ? n : name, a, b});
    a = nullptr;
  }
};

// ---------------------------------------------------------------- validation
bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

bcmt_status check_params(const bcmt_params* p) {
  if (!p) return fail(BCMT_ERR_ARG, "params is NULL");
  if (p->B < 1 || p->T < 1 || p->D < 1 || p->H < 1 || p->L < 1)
    return fail(BCMT_ERR_SHAPE, "B, T, D, H, L must be >= 1 (got %d %d %d %d %d)", p->B, p->T,
                p->D, p->H, p->L);
  if (p->dtype != BCMT_F32 && p->dtype != BCMT_BF16)
    return fail(BCMT_ERR_ARG, "dtype must be BCMT_F32 or BCMT_BF16 (got %d)", p->dtype);
  if (p->D % 64 != 0) return fail(BCMT_ERR_SHAPE, "D = %d is not a multiple of 64", p->D);
  if (p->D % p->H != 0) return fail(BCMT_ERR_SHAPE, "D = %d is not divisible by H = %d", p->D, p->H);
  const int dh = p->D / p->H;
  if (dh % 8 != 0 || dh > 128)
    return fail(BCMT_ERR_SHAPE, "head width D/H = %d must be a multiple of 8 and <= 128", dh);
  if (p->L > 1024) return fail(BCMT_ERR_UNSUPPORTED, "block size L = %d > 1024", p->L);
  if ((long long)p->B * p->T > (1ll << 30))
    return fail(BCMT_ERR_SHAPE, "B*T = %lld tokens is too large", (long long)p->B * p->T);
  if (p->flags & ~(unsigned)(BCMT_FLAG_HONLY | BCMT_FLAG_CHECK | BCMT_FLAG_PROFILE))
    return fail(BCMT_ERR_ARG, "unknown flag bits 0x%x", p->flags);
  return BCMT_OK;
}

bcmt_status check_ptr(const void* ptr, const char* name) {
  if (!ptr) return fail(BCMT_ERR_ARG, "%s is NULL", name);
  if (!aligned16(ptr)) return fail(BCMT_ERR_ALIGN, "%s is not 16-byte aligned", name);
  return BCMT_OK;
}

#define BCMT_TRY(expr)                  \
  do {                                  \
    bcmt_status _s = (expr);            \
    if (_s != BCMT_OK) return _s;       \
  } while (0)

// ----------------------------------------------------------- workspace layout
size_t al256(size_t x) { return (x + 255) & ~size_t(255); }

struct Geometry {
  int B, T, D, H, L, Nb, dh, es;
  long n;  // tokens B*T
  bool honly, from_x;
  int dtype;
  explicit Geometry(const bcmt_params* p)
      : B(p->B), T(p->T), D(p->D), H(p->H), L(p->L), Nb((p->T + p->L - 1) / p->L), dh(p->D / p->H),
        es(p->dtype == BCMT_BF16 ? 2 : 4), n((long)p->B * p->T),
        honly((p->flags & BCMT_FLAG_HONLY) != 0), from_x(p->input_is_x != 0), dtype(p->dtype) {}
};

int device_sms() {
  static int n = 0;
  if (!n) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 2)
      n = 148;
  }
  return n;
}

// Weight gradients dW[M,N] = A^T B over K = tokens run on the CTA-pair GEMM
// (256 x 256 tiles) when both sides are multiples of 256, else on 128-wide
// tiles, with K split into ranges of at least 8 slices.  A large product
// (at least 8 pair tiles: dW_qkv, the step's last GEMM) is split to fill one
// round of CTA pairs; the D x D ones are split to about 50 pairs (at most 12
// splits), leaving SMs to the critical path beside them.
bool dw_pair(int dtype, int M, int N) {
  return dtype == BCMT_BF16 && g_use_tc_gemm && M % 256 == 0 && N % 256 == 0;
}
int dw_splits(int dtype, int M, int N, long K, int max_pairs = 0) {
  const int nkb = (int)((K + 63) / 64);
  int target, tiles;
  if (dw_pair(dtype, M, N)) {
    tiles = (M / 256) * (N / 256);
    target = tiles >= 8 ? device_sms() / 2 : std::min(50, 12 * tiles);
    if (max_pairs > 0) target = std::min(target, max_pairs);
  } else {
    tiles = ((M + 127) / 128) * ((N + 127) / 128);
    target = 100;
  }
  int s = std::max(1, target / std::max(1, tiles));
  return std::max(1, std::min(s, nkb / 8));
}

// The backward pass's last products -- dX = dQKV W_QKV^T and the K-split
// weight gradients dW_QKV = X^T dQKV, dW_g = H^T dU (when the gate exists)
// and dW_O = Hhat^T dH -- share one CTA-pair launch when they fit its
// 256 x 256 tiles (bf16, D a multiple of 256).  The weight gradients then
// leave the side streams, where they slowed the critical kernels beside them.
bool tail_grouped(const Geometry& g) {
  return g.from_x && dw_pair(g.dtype, g.D, 3 * g.D) && gemm_tc_available() && g.n >= 256;
}
// K splits of the weight gradients in that launch (in launch order: dW_QKV,
// dW_g, dW_O; 0 = absent): the counts for which the launch, scheduled longest
// item first onto the least loaded SM pair (gemm_tc_pair_group), followed by
// the reduction of the partials, finishes first.  Unit: one 64-deep K slice
// of a 256 x 256 tile (8.4 MFLOP, about 0.45 us on a pair); each item costs
// its slices plus a fixed overhead for pipeline fill and epilogue, and each
// split of an M x N product adds the reduction's reading of M*N fp32
// partials at about 3 MB per unit.  Up to 16 splits each; ties go to fewer
// splits.  Cached per shape: the search runs once.
struct TailPlan {
  int s[3] = {1, 0, 0};
};
TailPlan tail_plan(const Geometry& g) {
  const int pairs = std::max(1, device_sms() / 2);
  const int D = g.D, n = (int)g.n;
  const int nkb = (int)((g.n + 63) / 64);
  const bool gate = !g.honly;
  const double out_units[3] = {3.0 * D * D * 4.0 / 3.0e6, (double)D * D * 4.0 / 3.0e6,
                               (double)D * D * 4.0 / 3.0e6};
  static std::mutex mu;
  static std::vector<std::pair<std::array<long, 4>, TailPlan>> cache;
  const std::array<long, 4> key{pairs, (long)g.n, (long)D, (long)g.honly};
  std::lock_guard<std::mutex> lock(mu);
  for (const auto& c : cache)
    if (c.first == key) return c.second;
  const int smax = std::min(16, std::max(1, nkb / 8));
  TailPlan best;
  double best_t = -1.0;
  for (int a = 1; a <= smax; ++a)
    for (int b = gate ? 1 : 0; b <= (gate ? smax : 0); ++b)
      for (int c = 1; c <= smax; ++c) {
        // the weight products in launch order (dW_QKV, dW_g when present, dW_O)
        int Mw[3], Nw[3], Kw[3], sw[3], nw = 0;
        const int sp[3] = {a, b, c};
        const int Ns[3] = {3 * D, D, D};
        double red = 0.0;
        for (int w = 0; w < 3; ++w) {
          if (w == 1 && !gate) continue;
          Mw[nw] = D;
          Nw[nw] = Ns[w];
          Kw[nw] = n;
          sw[nw] = sp[w];
          red += effective_splits(n, sp[w]) * out_units[w];
          ++nw;
        }
        const long ms = tc2_group_makespan(n, D, 3 * D, Mw, Nw, Kw, sw, nw, pairs);
        if (ms < 0) continue;
        const double t_end = (double)ms + red;
        if (best_t < 0 || t_end < best_t) {
          best_t = t_end;
          best.s[0] = a;
          best.s[1] = b;
          best.s[2] = c;
        }
      }
  cache.emplace_back(key, best);
  return best;
}
int dqkv_splits(const Geometry& g) {
  return tail_grouped(g) ? tail_plan(g).s[0] : dw_splits(g.dtype, g.D, 3 * g.D, g.n);
}

// K splits of the memory projections P = M W_m and dM = dP W_m^T ([B*Nb, D]
// x [D, D]): a few hundred rows make one tile row, so splitting K spreads
// the operand bytes over more SMs (each CTA of the unsplit product streams
// all of M); the consumers sum the fp32 partials as they read them.  dM runs
// beside dH = dY + dU W_g^T, which holds most SMs: two splits, so that its
// CTAs fit in the SMs left over.
// The forward memory scan and its D x D projection in one launch
// (memory_proj_fwd, warp-level mma) when the shape is small enough; else the
// scan kernel and the tcgen05 projection.
bool mem_fused(const Geometry& g) {
  return !g.honly && g_use_tc_gemm && memory_proj_fits(g.dtype, g.B, g.Nb, g.D);
}
// fp32 partials of P = M W_m that the memory row's readers sum (one when the
// fused kernel computes P whole)
int mem_splits(const Geometry& g) { return mem_fused(g) ? 1 : effective_splits(g.D, 4); }
int dm_splits(const Geometry& g) { return effective_splits(g.D, 2); }

// The forward's output projection and gate share one product,
// Concat [W_O | W_O W_g] (bf16 tensor-core path): H W_g = Concat (W_O W_g).
// The weight product W_O W_g rides in the Q/K/V projection's launch when that
// runs on the single-CTA kernel, else it is a launch of its own before it.
bool fused_gate(const Geometry& g) {
  return !g.honly && g.dtype == BCMT_BF16 && g_use_tc_gemm && gemm_tc_available();
}

struct FwdWs {
  char *qkv, *hhat, *hloc, *G, *Mb, *wog;
  float *lse, *alpha, *S, *M, *Z, *Zinv, *C, *spart;
  size_t bytes;
};

FwdWs fwd_layout(const Geometry& g, void* base) {
  FwdWs w;
  char* p = static_cast<char*>(base);
  size_t off = 0;
  auto take = [&](size_t bytes) {
    char* r = p ? p + off : nullptr;
    off += al256(bytes);
    return r;
  };
  w.qkv = g.from_x ? take((size_t)g.n * 3 * g.D * g.es) : nullptr;
  w.lse = reinterpret_cast<float*>(take((size_t)g.B * g.H * g.T * 4));
  w.hhat = take((size_t)g.n * g.D * g.es);
  if (!g.honly) {
    w.hloc = take((size_t)g.n * g.D * g.es);
    w.alpha = reinterpret_cast<float*>(take((size_t)g.n * 4));
    // partial pooling scores: one per token and 4-column run at most
    w.spart = reinterpret_cast<float*>(take((size_t)g.n * (g.D / 4) * 4));
    w.S = reinterpret_cast<float*>(take((size_t)g.B * g.Nb * g.D * 4));
    w.M = reinterpret_cast<float*>(take((size_t)g.B * g.Nb * g.D * 4));
    // M in the storage dtype: the A operand of the memory projection (and of dW_m)
    w.Mb = g.dtype == BCMT_BF16 ? take((size_t)g.B * g.Nb * g.D * 2) : reinterpret_cast<char*>(w.M);
    w.Z = reinterpret_cast<float*>(take((size_t)g.Nb * g.D * 4));
    w.Zinv = reinterpret_cast<float*>(take((size_t)g.Nb * g.D * 4));
    // the K-split partials of P = M W_m (the memory rows C, before the shift)
    w.C = reinterpret_cast<float*>(take((size_t)mem_splits(g) * g.B * g.Nb * g.D * 4));
    w.G = take((size_t)g.n * g.D * g.es);
    // W_O W_g [D, D]: the B operand of the gate columns of the fused projection
    w.wog = fused_gate(g) ? take((size_t)g.D * g.D * g.es) : nullptr;
  } else {
    w.wog = nullptr;
    w.hloc = w.G = w.Mb = nullptr;
    w.alpha = w.S = w.M = w.Z = w.Zinv = w.C = w.spart = nullptr;
  }
  w.bytes = off;
  return w;
}

struct BwdWs {
  char *dU, *dH, *dHhat, *dqkv, *dPb;
  float *dP, *dM, *dS, *ds, *dwp_part, *da_part, *Drow, *part, *part_o, *part_qkv;
  size_t bytes;
};

BwdWs bwd_layout(const Geometry& g, void* base) {
  BwdWs w;
  char* p = static_cast<char*>(base);
  size_t off = 0;
  auto take = [&](size_t bytes) {
    char* r = p ? p + off : nullptr;
    off += al256(bytes);
    return r;
  };
  if (!g.honly) {
    w.dU = take((size_t)g.n * g.D * g.es);
    w.dH = take((size_t)g.n * g.D * g.es);
    w.dP = reinterpret_cast<float*>(take((size_t)g.B * g.Nb * g.D * 4));
    w.dPb = g.dtype == BCMT_BF16 ? take((size_t)g.B * g.Nb * g.D * 2) : reinterpret_cast<char*>(w.dP);
    w.dM = reinterpret_cast<float*>(take((size_t)dm_splits(g) * g.B * g.Nb * g.D * 4));
    w.dS = reinterpret_cast<float*>(take((size_t)g.B * g.Nb * g.D * 4));
    w.ds = reinterpret_cast<float*>(take((size_t)g.n * 4));
    w.dwp_part = reinterpret_cast<float*>(
        take((size_t)g.B * g.Nb * summary_bwd_chunks(g.dtype, g.L, g.D) * g.D * 4));
    w.da_part = reinterpret_cast<float*>(take((size_t)g.B * g.D * 4));
  } else {
    w.dU = w.dH = w.dPb = nullptr;
    w.dP = w.dM = w.dS = w.ds = w.dwp_part = w.da_part = nullptr;
  }
  w.dHhat = take((size_t)g.n * g.D * g.es);
  w.dqkv = g.from_x ? take((size_t)g.n * 3 * g.D * g.es) : nullptr;
  w.Drow = reinterpret_cast<float*>(take((size_t)g.B * g.H * g.T * 4));
  const bool grouped = tail_grouped(g);
  const TailPlan tp = grouped ? tail_plan(g) : TailPlan();
  size_t part = (size_t)(grouped ? std::max(1, tp.s[1]) : dw_splits(g.dtype, g.D, g.D, g.n)) *
                g.D * g.D * 4;
  if (g.from_x && !grouped)
    part = std::max(part, (size_t)dqkv_splits(g) * g.D * 3 * g.D * 4);
  w.part = reinterpret_cast<float*>(take(part));
  // dW_QKV's partials: on the side stream after dW_g they reuse dW_g's
  // buffer; in the grouped launch, which also computes dW_g, they get their
  // own
  w.part_qkv = grouped ? reinterpret_cast<float*>(take((size_t)dqkv_splits(g) * g.D * 3 * g.D * 4))
                       : w.part;
  // dW_O's K-split partials: its product runs on the critical stream (or the
  // second side stream) while the side stream may still be reducing dW_g's
  w.part_o = reinterpret_cast<float*>(
      take((size_t)(grouped ? tp.s[2] : dw_splits(g.dtype, g.D, g.D, g.n)) * g.D * g.D * 4));
  w.bytes = off;
  return w;
}

bcmt_status cuda_fail(cudaError_t e, const char* what) {
  return fail(BCMT_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

// Weight gradient dW[M,N] = A^T B over K tokens via K-split partials and an
// ordered reduction.
cudaError_t weight_grad(const Launch& lc, Prof& pr, const char* name, int dtype, int dtype_out,
                        int M, int N, long K,
                        const void* A, long lda, const void* B, long ldb, float* part, void* out,
                        Fork* reduce_beside = nullptr, const Launch* lcs = nullptr,
                        Prof* prs = nullptr, int max_pairs = 0) {
  const int splits = dw_splits(dtype, M, N, K, max_pairs);
  EpiArgs ea;
  ea.out = part;
  ea.ldo = N;
  ea.split_stride = (long)M * N;
  pr.begin(name);
  cudaError_t e =
      dw_pair(dtype, M, N)
          ? gemm_tc_pair(lc, 0, M, N, (int)K, A, 1, lda, B, ldb, 1, EPI_PARTIAL, ea, splits)
      : (dtype == 1 && g_use_tc_gemm)
          ? gemm_tc(lc, 0, M, N, (int)K, A, 1, lda, B, ldb, 1, EPI_PARTIAL, ea, splits)
          : gemm_simt(lc, dtype, 0, M, N, (int)K, A, 1, lda, B, ldb, 1, EPI_PARTIAL, ea, splits);
  pr.end(nullptr);
  if (e != cudaSuccess) return e;
  // the ordered sum of the partials, on the side stream when asked
  const Launch& lr = reduce_beside ? *lcs : lc;
  Prof& prr = reduce_beside ? *prs : pr;
  if (reduce_beside) reduce_beside->point();
  prr.begin("reduce_splits");
  e = reduce_splits(lr, part, effective_splits((int)K, splits), (long)M * N, dtype_out, out);
  prr.end(nullptr);
  return e;
}

cudaError_t run_gemm(const Launch& lc, Prof& pr, const char* name, int dtype, int dtype_out, int M,
                     int N, int K, const void* A, long sam, long sak, const void* B, long sbk,
                     long sbn, EpiKind epi, const EpiArgs& ea, int splits = 1) {
  pr.begin(name);
  cudaError_t e =
      (dtype == 1 && g_use_tc_gemm)
          ? gemm_tc(lc, dtype_out, M, N, K, A, sam, sak, B, sbk, sbn, epi, ea, splits)
          : gemm_simt(lc, dtype, dtype_out, M, N, K, A, sam, sak, B, sbk, sbn, epi, ea, splits);
  pr.end(nullptr);
  return e;
}

// Attention kernel for a shape: 1 = single-tile tcgen05 (head width 64,
// L <= 128), 2 = key-tile-walking tcgen05, 0 = SIMT (fp32 and the rest).
int attn_kind(const Geometry& g) {
  if (!g_use_tc_attn) return 0;
  if (attn_tc_supported(g.dtype, g.dh, g.L)) return 1;
  return attn_fl_supported(g.dtype, g.dh, g.L) ? 2 : 0;
}

bcmt_status finish(const bcmt_params* p, cudaStream_t s) {
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "kernel launch");
  if (p->flags & BCMT_FLAG_CHECK) return bcmt_device_status(s);
  return BCMT_OK;
}

// A wait that cannot end, bounded by `cap` SM clock cycles: one thread
// initialises an mbarrier for one arrival and waits for its first phase, which
// nothing completes.  The bounded wait expires, ORs kStatusTimeout into the
// status word and returns; the kernel holds no TMA copy, no tcgen05 operation
// and no TMEM, so it leaves nothing behind.
__global__ void wait_expiry_kernel(unsigned* status, long long cap) {
  __shared__ __align__(8) uint64_t bar;
  tc::mbar_init(&bar, 1);
  tc::fence_mbar_init();
  tc::mbar_wait(&bar, 0, status, cap);
}

}  // namespace
}  // namespace bcmt

using namespace bcmt;

extern "C" {

size_t bcmt_workspace_size(const bcmt_params* p) {
  if (check_params(p) != BCMT_OK) return 0;
  Geometry g(p);
  return fwd_layout(g, nullptr).bytes;
}

size_t bcmt_scratch_size(const bcmt_params* p) {
  if (check_params(p) != BCMT_OK) return 0;
  Geometry g(p);
  return bwd_layout(g, nullptr).bytes;
}

const char* bcmt_last_error(void) { return g_last_error.c_str(); }

bcmt_status bcmt_device_status(void* stream) {
  unsigned* sp = status_ptr();
  if (!sp) return fail(BCMT_ERR_CUDA, "device status word unavailable");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  unsigned v = 0;
  cudaError_t e = cudaMemcpyAsync(&v, sp, sizeof(v), cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e == cudaSuccess) e = cudaMemsetAsync(sp, 0, sizeof(unsigned), s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_fail(e, "reading device status");
  if (v & kStatusTimeout) return fail(BCMT_ERR_TIMEOUT, "a bounded device-side wait expired");
  if (v) return fail(BCMT_ERR_CUDA, "device status 0x%x", v);
  return BCMT_OK;
}

bcmt_status bcmt_forward(const bcmt_params* p, const void* x, const void* q, const void* k,
                         const void* v, const void* w_qkv, const void* w_o, const void* w_p,
                         const void* w_m, const void* w_g, const float* decay, void* y,
                         void* workspace, void* stream) {
  BCMT_TRY(check_params(p));
  Geometry g(p);
  if (g.from_x) {
    BCMT_TRY(check_ptr(x, "x"));
    BCMT_TRY(check_ptr(w_qkv, "w_qkv"));
  } else {
    BCMT_TRY(check_ptr(q, "q"));
    BCMT_TRY(check_ptr(k, "k"));
    BCMT_TRY(check_ptr(v, "v"));
  }
  BCMT_TRY(check_ptr(w_o, "w_o"));
  if (!g.honly) {
    BCMT_TRY(check_ptr(w_p, "w_p"));
    BCMT_TRY(check_ptr(w_m, "w_m"));
    BCMT_TRY(check_ptr(w_g, "w_g"));
    BCMT_TRY(check_ptr(decay, "decay"));
  }
  BCMT_TRY(check_ptr(y, "y"));
  BCMT_TRY(check_ptr(workspace, "workspace"));
  unsigned* sp = status_ptr();
  if (!sp) return fail(BCMT_ERR_CUDA, "no CUDA device / device status word unavailable");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const bool profiling = (p->flags & BCMT_FLAG_PROFILE) != 0;
  // The memory stage runs on the side stream beside the gate GEMM (one
  // stream while profiling).
  std::unique_ptr<Fork> fork_holder(new Fork(profiling ? nullptr : side_stream(), s));
  Fork& fork = *fork_holder;
  Launch lc{fork.main(), sp};
  Prof pr{profiling, fork.main()};
  Launch lcs{fork.side(), sp};
  Prof prs{profiling, fork.side()};
  FwdWs w = fwd_layout(g, workspace);
  const int D = g.D, n = (int)g.n;
  cudaError_t e;
  const bool fuse = fused_gate(g);
  // the weight product W_O W_g of the fused output projection
  const GemmProd wog{D, D, D, w_o, D, 1, w_g, D, 1, w.wog, D};
  bool wog_done = false;

  // Sec. 3.3: Q, K, V projections (with W_O W_g in the same launch when it fits).
  const void *Qp = q, *Kp = k, *Vp = v;
  long ld = D;
  if (g.from_x) {
    e = cudaErrorNotSupported;
    if (fuse) {
      // on CTA pairs (256 x 256 tiles: 2/3 of a single CTA's operand bytes
      // per flop) when both widths allow, else the single-CTA kernel
      pr.begin("gemm_qkv_wog");
      e = gemm_tc_pair_two(lc, n, 3 * D, D, x, D, 1, w_qkv, 3 * D, 1, w.qkv, 3 * D, wog);
      if (e == cudaErrorNotSupported)
        e = gemm_tc_two(lc, n, 3 * D, D, x, D, 1, w_qkv, 3 * D, 1, w.qkv, 3 * D, wog);
      pr.end(nullptr);
      wog_done = e == cudaSuccess;
    }
    if (e == cudaErrorNotSupported) {
      if (fuse) {
        EpiArgs ea;
        ea.out = w.wog;
        ea.ldo = D;
        e = run_gemm(lc, pr, "gemm_wog", g.dtype, g.dtype, D, D, D, w_o, D, 1, w_g, D, 1,
                     EPI_STORE, ea);
        if (e != cudaSuccess) return cuda_fail(e, "W_O W_g");
        wog_done = true;
      }
      EpiArgs ea;
      ea.out = w.qkv;
      ea.ldo = 3 * D;
      e = run_gemm(lc, pr, "gemm_qkv", g.dtype, g.dtype, n, 3 * D, D, x, D, 1, w_qkv, 3 * D, 1,
                   EPI_STORE, ea);
    }
    if (e != cudaSuccess) return cuda_fail(e, "QKV projection");
    Qp = w.qkv;
    Kp = w.qkv + (size_t)D * g.es;
    Vp = w.qkv + (size_t)2 * D * g.es;
    ld = 3 * D;
  }
  // Sec. 3.3: intra-block causal attention -> Concat(heads).
  AttnArgs aa{Qp, Kp, Vp, ld, w.hhat, D, w.lse, g.B, g.T, g.H, g.dh, g.L};
  if (attn_kind(g) == 1) {
    pr.begin("attn_fwd_tc");
    e = attn_fwd_tc(lc, aa);
  } else if (attn_kind(g) == 2) {
    pr.begin("attn_fwd_fl");
    e = attn_fwd_fl(lc, aa);
  } else {
    pr.begin("attn_fwd_simt");
    e = attn_fwd_simt(lc, g.dtype, aa);
  }
  pr.end(nullptr);
  if (e != cudaSuccess) return cuda_fail(e, "block attention");
  // Sec. 3.3: H = Concat(heads) W_O (HOnly: this is the output, Sec. 4.5).  The
  // epilogue also forms partial pooling scores H w_p over each run of columns
  // it stores (32 columns per tcgen05 TMEM load, 4 per SIMT thread).
  const int npart = D / ((g.dtype == BCMT_BF16 && g_use_tc_gemm) ? 32 : 4);
  if (fuse) {
    // H and the gate G = sigmoid(H W_g) (Sec. 3.8) in one product over all
    // SMs, [H | U] = Concat [W_O | W_O W_g]
    if (!wog_done) {
      EpiArgs ea;
      ea.out = w.wog;
      ea.ldo = D;
      e = run_gemm(lc, pr, "gemm_wog", g.dtype, g.dtype, D, D, D, w_o, D, 1, w_g, D, 1,
                   EPI_STORE, ea);
      if (e != cudaSuccess) return cuda_fail(e, "W_O W_g");
    }
    EpiArgs ea;
    ea.out = w.hloc;
    ea.ldo = D;
    ea.w_p = w_p;
    ea.spart = w.spart;
    ea.out2 = w.G;
    ea.ldo2 = D;
    ea.n_split = D;
    ea.b2 = w.wog;
    e = run_gemm(lc, pr, "gemm_wo_gate", g.dtype, g.dtype, n, 2 * D, D, w.hhat, D, 1, w_o, D, 1,
                 EPI_HGATE, ea);
    if (e != cudaSuccess) return cuda_fail(e, "output projection and gate");
  } else {
    EpiArgs ea;
    ea.out = g.honly ? y : w.hloc;
    ea.ldo = D;
    ea.w_p = w_p;
    ea.spart = w.spart;
    e = run_gemm(lc, pr, "gemm_wo", g.dtype, g.dtype, n, D, D, w.hhat, D, 1, w_o, D, 1,
                 g.honly ? EPI_STORE : EPI_STORE_SCORE, ea);
    if (e != cudaSuccess) return cuda_fail(e, "output projection");
  }
  if (!g.honly) {
    // Sec. 3.8 gate G = sigmoid(H W_g) (unless fused above), then the memory
    // chain: one stream of kernels chained by programmatic dependent launch.
    // (Beside the chain on half of the SMs the gate GEMM slowed the chain's
    // kernels about twofold, and each join of two streams left a launch gap.)
    if (!fuse) {
      EpiArgs ea;
      ea.out = w.G;
      ea.ldo = D;
      e = run_gemm(lc, pr, "gemm_gate", g.dtype, g.dtype, n, D, D, w.hloc, D, 1, w_g, D, 1,
                   EPI_GATE, ea);
      if (e != cudaSuccess) return cuda_fail(e, "gate");
    }
    // Sec. 3.4 adaptive block summaries, Sec. 3.5 exponential causal memory
    // (scan), then its projection and one-block shift -> C
    pr.begin("summary_fwd");
    e = summary_fwd(lc, g.dtype, w.hloc, w.spart, npart, w.alpha, w.S, g.B, g.T, D, g.L);
    pr.end(nullptr);
    if (e != cudaSuccess) return cuda_fail(e, "block summaries");
    if (mem_fused(g)) {
      // the scan and P = M W_m in one launch (P whole; the shift is applied
      // by the readers)
      pr.begin("memory_proj_fwd");
      e = memory_proj_fwd(lc, w.S, decay, w_m, w.C, w.M, w.Mb, w.Z, w.Zinv, g.B, g.Nb, D);
      pr.end(nullptr);
      if (e != cudaSuccess) return cuda_fail(e, "causal memory and its projection");
    } else {
      pr.begin("memory_scan_fwd");
      e = memory_scan_fwd(lc, w.S, decay, w.M, g.dtype == BCMT_BF16 ? w.Mb : nullptr, w.Z,
                          w.Zinv, g.B, g.Nb, D);
      pr.end(nullptr);
      if (e != cudaSuccess) return cuda_fail(e, "causal memory");
      // P = M W_m as K-split partials; the shift is applied by the readers
      EpiArgs ea;
      ea.out = w.C;
      ea.ldo = D;
      ea.split_stride = (long)g.B * g.Nb * D;
      e = run_gemm(lc, pr, "gemm_wm", g.dtype, 0, g.B * g.Nb, D, D, w.Mb, D, 1, w_m, D, 1,
                   EPI_PARTIAL, ea, mem_splits(g));
      if (e != cudaSuccess) return cuda_fail(e, "memory projection");
    }
    // Sec. 3.7-3.8: Y = H + G * M_tokens
    pr.begin("inject");
    e = inject(lc, g.dtype, w.hloc, w.G, w.C, mem_splits(g), y, g.B, g.T, D, g.L);
    pr.end(nullptr);
    if (e != cudaSuccess) return cuda_fail(e, "injection");
  }
  fork_holder.reset();  // join the side stream before any status read
  return finish(p, s);
}

bcmt_status bcmt_backward(const bcmt_params* p, const void* dy, const void* x_or_q, const void* k,
                          const void* v, const void* w_qkv,
                          const void* w_o, const void* w_p, const void* w_m, const void* w_g,
                          const float* decay, const void* workspace, void* scratch, void* dx_or_dq,
                          void* dk, void* dv, void* dw_qkv, void* dw_o, void* dw_p, void* dw_m,
                          void* dw_g, float* d_decay, void* stream) {
  BCMT_TRY(check_params(p));
  Geometry g(p);
  BCMT_TRY(check_ptr(dy, "dy"));
  BCMT_TRY(check_ptr(x_or_q, "x_or_q"));
  if (g.from_x) {
    BCMT_TRY(check_ptr(w_qkv, "w_qkv"));
    BCMT_TRY(check_ptr(dw_qkv, "dw_qkv"));
  } else {
    BCMT_TRY(check_ptr(k, "k"));
    BCMT_TRY(check_ptr(v, "v"));
    BCMT_TRY(check_ptr(dk, "dk"));
    BCMT_TRY(check_ptr(dv, "dv"));
  }
  BCMT_TRY(check_ptr(dx_or_dq, "dx_or_dq"));
  BCMT_TRY(check_ptr(w_o, "w_o"));
  BCMT_TRY(check_ptr(dw_o, "dw_o"));
  BCMT_TRY(check_ptr(dw_p, "dw_p"));
  BCMT_TRY(check_ptr(dw_m, "dw_m"));
  BCMT_TRY(check_ptr(dw_g, "dw_g"));
  if (!g.honly) {
    BCMT_TRY(check_ptr(w_p, "w_p"));
    BCMT_TRY(check_ptr(w_m, "w_m"));
    BCMT_TRY(check_ptr(w_g, "w_g"));
    BCMT_TRY(check_ptr(decay, "decay"));
  }
  BCMT_TRY(check_ptr(workspace, "workspace"));
  BCMT_TRY(check_ptr(scratch, "scratch"));
  unsigned* sp = status_ptr();
  if (!sp) return fail(BCMT_ERR_CUDA, "no CUDA device / device status word unavailable");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const bool profiling = (p->flags & BCMT_FLAG_PROFILE) != 0;
  // Weight gradients go to the side stream (kept on one stream while
  // profiling, so every kernel is timed alone).
  std::unique_ptr<Fork> fork_holder(new Fork(profiling ? nullptr : side_stream(), s));
  Fork& fork = *fork_holder;
  Launch lc{fork.main(), sp};
  Prof pr{profiling, fork.main()};
  Launch lcs{fork.side(), sp};
  Prof prs{profiling, fork.side()};
  FwdWs w = fwd_layout(g, const_cast<void*>(workspace));
  BwdWs bw = bwd_layout(g, scratch);
  const int D = g.D, n = (int)g.n;
  cudaError_t e;

  const void* dH = dy;  // HOnly: Y = H
  if (!g.honly) {
    // Sec. 3.8 reversed: dU and the per-block memory gradient (shifted: dP).
    pr.begin("gate_bwd");
    e = gate_bwd(lc, g.dtype, dy, w.G, w.C, mem_splits(g), bw.dU, bw.dP, g.dtype == BCMT_BF16 ? bw.dPb : nullptr,
                 g.B, g.T, D, g.L);
    pr.end(nullptr);
    if (e != cudaSuccess) return cuda_fail(e, "gate backward");
    // side stream: Sec. 3.5 reversed, dM = dP W_m^T and the reverse decayed
    // scan -> dS (and the decay gradient's batch rows).  On the bf16 tensor
    // cores without a decay gradient, when Nb divides 32, one launch computes
    // dM transposed (dM^T = W_m dP^T: a row per channel) and its epilogue runs
    // each channel's scan in registers; otherwise dM as K-split partials and
    // the scan kernel.
    fork.point();
    const bool scan_in_gemm = !d_decay && g.dtype == BCMT_BF16 && g_use_tc_gemm &&
                              gemm_tc_available() && g.Nb <= 32 && 32 % g.Nb == 0;
    if (scan_in_gemm) {
      EpiArgs ea;
      ea.out = bw.dS;
      ea.ldo = D;
      ea.scan_zinv = w.Zinv;
      ea.scan_decay = decay;
      ea.scan_nb = g.Nb;
      e = run_gemm(lcs, prs, "gemm_dm_scan", g.dtype, 0, D, g.B * g.Nb, D, w_m, D, 1, bw.dPb, 1,
                   D, EPI_REVSCAN, ea);
      if (e != cudaSuccess) return cuda_fail(e, "dM and its reverse scan");
    } else {
      {
        EpiArgs ea;
        ea.out = bw.dM;
        ea.ldo = D;
        ea.split_stride = (long)g.B * g.Nb * D;
        e = run_gemm(lcs, prs, "gemm_dm", g.dtype, 0, g.B * g.Nb, D, D, bw.dPb, D, 1, w_m, 1, D,
                     EPI_PARTIAL, ea, dm_splits(g));
        if (e != cudaSuccess) return cuda_fail(e, "dM");
      }
      prs.begin("memory_scan_bwd");
      e = memory_scan_bwd(lcs, bw.dM, dm_splits(g), decay, w.Z, w.M, bw.dS,
                          d_decay ? bw.da_part : nullptr, g.B, g.Nb, D);
      prs.end(nullptr);
      if (e != cudaSuccess) return cuda_fail(e, "memory backward");
    }
    const int scan_done = fork.mark();
    // side stream, then: dW_m = M^T dP and dW_g = H^T dU
    {
      EpiArgs ea;
      ea.out = dw_m;
      ea.ldo = D;
      e = run_gemm(lcs, prs, "gemm_dwm", g.dtype, g.dtype, D, D, g.B * g.Nb, w.Mb, 1, D, bw.dPb, D,
                   1, EPI_STORE, ea);
      if (e != cudaSuccess) return cuda_fail(e, "dW_m");
    }
    // (up to 32 GFLOP on a few SM pairs: it runs beside the pooling backward,
    // which needs the rest, and has until the end of the backward; with the
    // grouped tail it joins dX and dW_QKV there instead)
    if (!tail_grouped(g)) {
      e = weight_grad(lcs, prs, "gemm_dw_g", g.dtype, g.dtype, D, D, g.n, w.hloc, D, bw.dU, D,
                      bw.part, dw_g, nullptr, nullptr, nullptr,
                      2.0 * D * D * (double)g.n <= 32e9 ? device_sms() / 8 : 0);
      if (e != cudaSuccess) return cuda_fail(e, "dW_g");
    }
    // main stream, meanwhile: dH = dU W_g^T (the gate path; the identity
    // path's dY is added by the pooling backward)
    {
      // (the identity path's dY is added by the pooling backward, which
      // reads and writes every row of dH anyway)
      EpiArgs ea;
      ea.out = bw.dH;
      ea.ldo = D;
      e = run_gemm(lc, pr, "gemm_dh", g.dtype, g.dtype, n, D, D, bw.dU, D, 1, w_g, 1, D, EPI_STORE,
                   ea);
      if (e != cudaSuccess) return cuda_fail(e, "dH");
    }
    // Sec. 3.4 reversed once dS is ready: pooling scores, the dW_p partials,
    // and dH += alpha dS + ds w_p
    fork.wait_mark(scan_done);
    pr.begin("summary_bwd");
    e = summary_bwd(lc, g.dtype, w.hloc, w.alpha, w.S, bw.dS, w_p, dy, bw.dH, bw.ds, bw.dwp_part,
                    g.B, g.T, D, g.L);
    pr.end(nullptr);
    if (e != cudaSuccess) return cuda_fail(e, "summary backward");
    fork.point();
    prs.begin("reduce_rows");
    e = reduce_rows(lcs, bw.dwp_part, g.B * g.Nb * summary_bwd_chunks(g.dtype, g.L, g.D), D, g.dtype, dw_p);
    prs.end(nullptr);
    if (e != cudaSuccess) return cuda_fail(e, "dW_p");
    if (d_decay) {  // fp32, summed over the batch rows in order
      prs.begin("reduce_rows");
      e = reduce_rows(lcs, bw.da_part, g.B, D, 0, d_decay);
      prs.end(nullptr);
      if (e != cudaSuccess) return cuda_fail(e, "d_decay");
    }
    dH = bw.dH;
  } else {
    const size_t wb = (size_t)D * D * g.es;
    if ((e = fill_zero(lc, dw_m, wb)) != cudaSuccess || (e = fill_zero(lc, dw_g, wb)) != cudaSuccess ||
        (e = fill_zero(lc, dw_p, (size_t)D * g.es)) != cudaSuccess ||
        (d_decay && (e = fill_zero(lc, d_decay, (size_t)D * 4)) != cudaSuccess))
      return cuda_fail(e, "zeroing HOnly gradients");
  }
  // Sec. 3.3 reversed: dHhat = dH W_O^T, dW_O = Hhat^T dH.
  {
    EpiArgs ea;
    ea.out = bw.dHhat;
    ea.ldo = D;
    e = run_gemm(lc, pr, "gemm_dhhat", g.dtype, g.dtype, n, D, D, dH, D, 1, w_o, 1, D, EPI_STORE,
                 ea);
    if (e != cudaSuccess) return cuda_fail(e, "dHhat");
    // dW_O: a small one (at most 8 GFLOP) goes to the second side stream on a
    // few SM pairs and runs beside the tail of the step (dx, dW_QKV) without
    // holding up dW_QKV; a large one stays on the critical stream with its
    // reduction beside
    if (tail_grouped(g)) {
      // computed with dX at the end of the pass
    } else if (2.0 * D * D * (double)g.n <= 8e9) {
      fork.point2();
      Launch lcs2{fork.side2(), sp};
      Prof prs2{profiling, fork.side2()};
      e = weight_grad(lcs2, prs2, "gemm_dw_o", g.dtype, g.dtype, D, D, g.n, w.hhat, D, dH, D,
                      bw.part_o, dw_o, nullptr, nullptr, nullptr, device_sms() / 12);
    } else {
      e = weight_grad(lc, pr, "gemm_dw_o", g.dtype, g.dtype, D, D, g.n, w.hhat, D, dH, D,
                      bw.part_o, dw_o, &fork, &lcs, &prs);
    }
    if (e != cudaSuccess) return cuda_fail(e, "dW_O");
  }
  // Attention backward -> dQ, dK, dV.
  {
    const void *Qp, *Kp, *Vp;
    long ld;
    void *dQ, *dK, *dV;
    long ldd;
    if (g.from_x) {
      Qp = w.qkv;
      Kp = w.qkv + (size_t)D * g.es;
      Vp = w.qkv + (size_t)2 * D * g.es;
      ld = 3 * D;
      dQ = bw.dqkv;
      dK = bw.dqkv + (size_t)D * g.es;
      dV = bw.dqkv + (size_t)2 * D * g.es;
      ldd = 3 * D;
    } else {
      Qp = x_or_q;
      Kp = k;
      Vp = v;
      ld = D;
      dQ = dx_or_dq;
      dK = dk;
      dV = dv;
      ldd = D;
    }
    AttnBwdArgs ab{{Qp, Kp, Vp, ld, w.hhat, D, w.lse, g.B, g.T, g.H, g.dh, g.L},
                   bw.dHhat, bw.Drow, dQ, dK, dV, ldd};
    if (attn_kind(g) == 1) {
      pr.begin("attn_bwd_tc");
      e = attn_bwd_tc(lc, ab);
    } else if (attn_kind(g) == 2) {
      pr.begin("attn_bwd_fl");
      e = attn_bwd_fl(lc, ab);
    } else {
      pr.begin("attn_bwd_simt");
      e = attn_bwd_simt(lc, g.dtype, ab);
    }
    pr.end(nullptr);
    if (e != cudaSuccess) return cuda_fail(e, "attention backward");
  }
  // Sec. 3.3 reversed: dX = dQKV W_qkv^T, dW_qkv = X^T dQKV.
  if (tail_grouped(g)) {
    // dX and the weight gradients in one launch on the critical stream, then
    // the ordered reductions of the gradients' partials in one more
    const TailPlan tp = tail_plan(g);
    const PairProduct pdx{n, D, 3 * D, bw.dqkv, 3 * D, 1, w_qkv, 1, 3 * D, dx_or_dq, D, 0, 1};
    PairProduct pw[3];
    SplitSum red[3];
    int nw = 0;
    pw[nw] = PairProduct{D, 3 * D, n, x_or_q, 1, D, bw.dqkv, 3 * D, 1, bw.part_qkv, 3 * D,
                         (long)D * 3 * D, tp.s[0]};
    red[nw++] = SplitSum{bw.part_qkv, effective_splits(n, tp.s[0]), (long)D * 3 * D, dw_qkv};
    if (!g.honly) {
      pw[nw] = PairProduct{D, D, n, w.hloc, 1, D, bw.dU, D, 1, bw.part, D, (long)D * D, tp.s[1]};
      red[nw++] = SplitSum{bw.part, effective_splits(n, tp.s[1]), (long)D * D, dw_g};
    }
    pw[nw] = PairProduct{D, D, n, w.hhat, 1, D, dH, D, 1, bw.part_o, D, (long)D * D, tp.s[2]};
    red[nw++] = SplitSum{bw.part_o, effective_splits(n, tp.s[2]), (long)D * D, dw_o};
    pr.begin("gemm_dx_dw");
    e = gemm_tc_pair_group(lc, pdx, pw, nw);
    pr.end(nullptr);
    if (e != cudaSuccess) return cuda_fail(e, "dX and the weight gradients");
    pr.begin("reduce_splits");
    e = reduce_splits_n(lc, red, nw, g.dtype);
    pr.end(nullptr);
    if (e != cudaSuccess) return cuda_fail(e, "weight gradient reduction");
  } else if (g.from_x) {
    EpiArgs ea;
    ea.out = dx_or_dq;
    ea.ldo = D;
    fork.point();  // dQKV is final
    e = weight_grad(lcs, prs, "gemm_dw_qkv", g.dtype, g.dtype, D, 3 * D, g.n, x_or_q, D, bw.dqkv,
                    3 * D, bw.part, dw_qkv);
    if (e != cudaSuccess) return cuda_fail(e, "dW_qkv");
    e = run_gemm(lc, pr, "gemm_dx", g.dtype, g.dtype, n, D, 3 * D, bw.dqkv, 3 * D, 1, w_qkv, 1,
                 3 * D, EPI_STORE, ea);
    if (e != cudaSuccess) return cuda_fail(e, "dX");
  }
  fork_holder.reset();  // join the side stream before any status read
  return finish(p, s);
}

// ------------------------------------------------------------------ decoding
namespace {
DecodeState decode_layout(const Geometry& g, void* base, size_t* bytes) {
  DecodeState st;
  char* p = static_cast<char*>(base);
  size_t off = 0;
  auto take = [&](size_t n) {
    char* r = p ? p + off : nullptr;
    off += al256(n);
    return r;
  };
  auto f32 = [&](size_t n) { return reinterpret_cast<float*>(take(n * 4)); };
  const size_t bd = (size_t)g.B * g.D;
  st.Kc = take((size_t)g.B * g.L * g.D * g.es);
  st.Vc = take((size_t)g.B * g.L * g.D * g.es);
  st.xf = f32(bd);
  st.qkv = f32(3 * bd);
  st.hhat = f32(bd);
  st.H = f32(bd);
  st.U = f32(bd);
  st.pm = f32(g.B);
  st.pden = f32(g.B);
  st.pnum = f32(bd);
  st.N = f32(bd);
  st.Z = f32(bd);
  st.C = f32(bd);
  st.Mr = f32(bd);
  *bytes = off;
  return st;
}
}  // namespace

size_t bcmt_decode_state_size(const bcmt_params* p) {
  if (check_params(p) != BCMT_OK) return 0;
  Geometry g(p);
  size_t bytes = 0;
  decode_layout(g, nullptr, &bytes);
  return bytes;
}

bcmt_status bcmt_decode_reset(const bcmt_params* p, void* state, void* stream) {
  BCMT_TRY(check_params(p));
  BCMT_TRY(check_ptr(state, "state"));
  const size_t bytes = bcmt_decode_state_size(p);
  cudaError_t e = cudaMemsetAsync(state, 0, bytes, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "decode state reset");
  return finish(p, static_cast<cudaStream_t>(stream));
}

bcmt_status bcmt_decode_step(const bcmt_params* p, void* state, long pos, const void* x_t,
                             const void* w_qkv, const void* w_o, const void* w_p,
                             const void* w_m, const void* w_g, const float* decay, void* y_t,
                             void* stream) {
  BCMT_TRY(check_params(p));
  if (!p->input_is_x)
    return fail(BCMT_ERR_ARG, "decoding starts from the token rows x (input_is_x must be 1)");
  if (pos < 0) return fail(BCMT_ERR_ARG, "pos = %ld must be >= 0", pos);
  Geometry g(p);
  BCMT_TRY(check_ptr(state, "state"));
  BCMT_TRY(check_ptr(x_t, "x_t"));
  BCMT_TRY(check_ptr(w_qkv, "w_qkv"));
  BCMT_TRY(check_ptr(w_o, "w_o"));
  BCMT_TRY(check_ptr(y_t, "y_t"));
  if (!g.honly) {
    BCMT_TRY(check_ptr(w_p, "w_p"));
    BCMT_TRY(check_ptr(w_m, "w_m"));
    BCMT_TRY(check_ptr(w_g, "w_g"));
    BCMT_TRY(check_ptr(decay, "decay"));
  }
  unsigned* sp = status_ptr();
  if (!sp) return fail(BCMT_ERR_CUDA, "no CUDA device / device status word unavailable");
  Launch lc{static_cast<cudaStream_t>(stream), sp};
  size_t bytes = 0;
  DecodeArgs a;
  a.s = decode_layout(g, state, &bytes);
  a.B = g.B;
  a.D = g.D;
  a.H = g.H;
  a.dh = g.dh;
  a.L = g.L;
  a.j = (int)(pos % g.L);
  a.honly = g.honly;
  a.x = a.s.xf;
  a.w_qkv = w_qkv;
  a.w_o = w_o;
  a.w_p = w_p;
  a.w_m = w_m;
  a.w_g = w_g;
  a.decay = decay;
  a.y = y_t;
  cudaError_t e = decode_widen(lc, g.dtype, x_t, a.s.xf, (long)g.B * g.D);
  if (e == cudaSuccess) e = decode_step(lc, g.dtype, a);
  if (e != cudaSuccess) return cuda_fail(e, "decode step");
  return finish(p, lc.stream);
}

bcmt_status bcmt_attention_backward_noalloc(const bcmt_params* p, const void* q, const void* k,
                                            const void* v, long ld, const void* o,
                                            const float* lse, const void* dO, void* dq, void* dk,
                                            void* dv, long ld_d, void* stream) {
  BCMT_TRY(check_params(p));
  Geometry g(p);
  BCMT_TRY(check_ptr(q, "q"));
  BCMT_TRY(check_ptr(k, "k"));
  BCMT_TRY(check_ptr(v, "v"));
  BCMT_TRY(check_ptr(o, "o"));
  BCMT_TRY(check_ptr(lse, "lse"));
  BCMT_TRY(check_ptr(dO, "dO"));
  BCMT_TRY(check_ptr(dq, "dq"));
  BCMT_TRY(check_ptr(dk, "dk"));
  BCMT_TRY(check_ptr(dv, "dv"));
  if (ld < g.D || ld_d < g.D)
    return fail(BCMT_ERR_ARG, "row strides ld = %ld and ld_d = %ld must be >= D = %d", ld, ld_d, g.D);
  const long long rows = (long long)g.B * g.H * g.T;
  if (rows > kNoAllocDrowRows)
    return fail(BCMT_ERR_SHAPE,
                "B*H*T = %lld exceeds the %lld rows of the built-in scratch of "
                "bcmt_attention_backward_noalloc",
                rows, kNoAllocDrowRows);
  unsigned* sp = status_ptr();
  if (!sp) return fail(BCMT_ERR_CUDA, "no CUDA device / device status word unavailable");
  Launch lc{static_cast<cudaStream_t>(stream), sp};
  AttnBwdArgs ab{{q, k, v, ld, const_cast<void*>(o), g.D, const_cast<float*>(lse), g.B, g.T, g.H,
                  g.dh, g.L},
                 dO, nullptr, dq, dk, dv, ld_d};
  cudaError_t e = attn_bwd_simt_noalloc(lc, g.dtype, ab);
  if (e != cudaSuccess) return cuda_fail(e, "allocation-free attention backward");
  return finish(p, lc.stream);
}

int bcmt_profile_read(const char** names, int* launches, double* ms, int cap) {
  std::lock_guard<std::mutex> lk(g_prof_mu);
  if (cudaDeviceSynchronize() != cudaSuccess) return -1;
  std::vector<const char*> nm;
  std::vector<int> cnt;
  std::vector<double> tot;
  for (auto& r : g_prof_recs) {
    float t = 0.f;
    if (cudaEventElapsedTime(&t, r.a, r.b) != cudaSuccess) return -1;
    size_t i = 0;
    for (; i < nm.size(); ++i)
      if (strcmp(nm[i], r.name) == 0) break;
    if (i == nm.size()) {
      nm.push_back(r.name);
      cnt.push_back(0);
      tot.push_back(0.0);
    }
    cnt[i] += 1;
    tot[i] += t;
  }
  for (size_t i = 0; i < nm.size() && (int)i < cap; ++i) {
    if (names) names[i] = nm[i];
    if (launches) launches[i] = cnt[i];
    if (ms) ms[i] = tot[i];
  }
  return (int)nm.size();
}

void bcmt_profile_reset(void) {
  std::lock_guard<std::mutex> lk(g_prof_mu);
  g_prof_recs.clear();
  g_prof_pool_used = 0;
}

// ------------------------------------------------------------ test entry points
int bcmt_test_set_tensor_cores(int gemm_on, int attn_on) {
  g_use_tc_gemm = gemm_on != 0;
  g_use_tc_attn = attn_on != 0;
  return (gemm_tc_available() ? 1 : 0) | (attn_tc_supported(1, 64, 64) ? 2 : 0);
}

int bcmt_test_wait_expiry(long long cycles, void* stream) {
  if (cycles < 1 || cycles > tc::kWaitCycles) {
    fail(BCMT_ERR_ARG, "cycles = %lld must be in [1, %lld]", cycles, tc::kWaitCycles);
    return -1;
  }
  unsigned* sp = status_ptr();
  if (!sp) {
    fail(BCMT_ERR_CUDA, "device status word unavailable");
    return -1;
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  wait_expiry_kernel<<<1, 1, 0, s>>>(sp, cycles);
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    fail(BCMT_ERR_CUDA, "wait expiry kernel: %s", cudaGetErrorString(e));
    return -1;
  }
  return 0;
}

int bcmt_test_gemm(int impl, int dtype, int dtype_out, int M, int N, int K, const void* A, long sam,
                   long sak, const void* B, long sbk, long sbn, void* C, long ldc, int splits,
                   void* stream) {
  unsigned* sp = status_ptr();
  if (!sp) return -1;
  Launch lc{static_cast<cudaStream_t>(stream), sp};
  EpiArgs ea;
  ea.out = C;
  ea.ldo = ldc;
  ea.split_stride = (long)M * ldc;
  const EpiKind ek = splits > 1 ? EPI_PARTIAL : EPI_STORE;
  // impl 3, 4, 5: the single-CTA kernel with 128-, 256- or 64-wide tiles
  g_force_bn = impl == 3 ? 128 : impl == 4 ? 256 : impl == 5 ? 64 : 0;
  cudaError_t e =
      (impl == 1 || impl >= 3)
          ? gemm_tc(lc, dtype_out, M, N, K, A, sam, sak, B, sbk, sbn, ek, ea, splits)
      : impl == 2 ? gemm_tc_pair(lc, dtype_out, M, N, K, A, sam, sak, B, sbk, sbn, ek, ea, splits)
                  : gemm_simt(lc, dtype, dtype_out, M, N, K, A, sam, sak, B, sbk, sbn, ek, ea,
                              splits);
  g_force_bn = 0;
  if (e != cudaSuccess) {
    fail(BCMT_ERR_CUDA, "test gemm: %s", cudaGetErrorString(e));
    return -1;
  }
  return splits > 1 ? effective_splits(K, splits) : 1;
}

int bcmt_test_gemm_group(int M0, int N0, int K0, const void* A0, long lda0, const void* B0t,
                         long ldb0t, void* C0, int M1, int N1, int K1, const void* A1t, long lda1t,
                         const void* B1, long ldb1, float* part1, int splits1, int M2, int N2,
                         int K2, const void* A2t, long lda2t, const void* B2, long ldb2,
                         float* part2, int splits2, void* stream) {
  unsigned* sp = status_ptr();
  if (!sp) return -1;
  if (!gemm_tc_available()) {
    fail(BCMT_ERR_CUDA, "test gemm group: tcgen05 GEMM unavailable");
    return -1;
  }
  Launch lc{static_cast<cudaStream_t>(stream), sp};
  const PairProduct p0{M0, N0, K0, A0, lda0, 1, B0t, 1, ldb0t, C0, N0, 0, 1};
  const PairProduct pw[2] = {
      {M1, N1, K1, A1t, 1, lda1t, B1, ldb1, 1, part1, N1, (long)M1 * N1, splits1},
      {M2, N2, K2, A2t, 1, lda2t, B2, ldb2, 1, part2, N2, (long)M2 * N2, splits2}};
  cudaError_t e = gemm_tc_pair_group(lc, p0, pw, M2 > 0 ? 2 : 1);
  if (e != cudaSuccess) {
    fail(BCMT_ERR_CUDA, "test gemm group: %s", cudaGetErrorString(e));
    return -1;
  }
  return effective_splits(K1, splits1);
}

int bcmt_test_attn(int impl, int backward, const bcmt_params* p, const void* q, const void* k,
                   const void* v, long ld, void* o, float* lse, const void* dO, float* drow,
                   void* dq, void* dk, void* dv, long ld_d, void* stream) {
  if (check_params(p) != BCMT_OK) return -1;
  unsigned* sp = status_ptr();
  if (!sp) return -1;
  Launch lc{static_cast<cudaStream_t>(stream), sp};
  Geometry g(p);
  AttnArgs aa{q, k, v, ld, o, g.D, lse, g.B, g.T, g.H, g.dh, g.L};
  cudaError_t e;
  if (!backward) {
    e = impl == 1 ? attn_fwd_tc(lc, aa)
        : impl == 2 ? attn_fwd_fl(lc, aa)
                    : attn_fwd_simt(lc, g.dtype, aa);
  } else {
    AttnBwdArgs ab{aa, dO, drow, dq, dk, dv, ld_d};
    e = impl == 1 ? attn_bwd_tc(lc, ab)
        : impl == 2 ? attn_bwd_fl(lc, ab)
                    : attn_bwd_simt(lc, g.dtype, ab);
  }
  if (e != cudaSuccess) {
    fail(BCMT_ERR_CUDA, "test attention: %s", cudaGetErrorString(e));
    return -1;
  }
  return 0;
}

}  // extern "C"
