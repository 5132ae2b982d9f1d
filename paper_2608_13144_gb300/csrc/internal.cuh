// Internal declarations of the lipcache library (not part of the C ABI).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <cmath>
#include <stdexcept>
#include <string>

#include "lipcache.h"

namespace lc {

// ---------------------------------------------------------------- errors
struct Error : std::runtime_error {
  lipcache_status status;
  Error(lipcache_status s, const std::string& m) : std::runtime_error(m), status(s) {}
};

#define LC_CUDA(call)                                                                          \
  do {                                                                                         \
    cudaError_t e_ = (call);                                                                   \
    if (e_ != cudaSuccess)                                                                     \
      throw ::lc::Error(e_ == cudaErrorMemoryAllocation ? LIPCACHE_E_NOMEM : LIPCACHE_E_CUDA, \
                        std::string(#call) + ": " + cudaGetErrorString(e_));                 \
  } while (0)

#define LC_LAUNCH_CHECK(name)                                                                      \
  do {                                                                                             \
    cudaError_t e_ = cudaGetLastError();                                                           \
    if (e_ != cudaSuccess)                                                                         \
      throw ::lc::Error(LIPCACHE_E_CUDA, std::string("launch of ") + (name) + ": " + cudaGetErrorString(e_)); \
  } while (0)

#define LC_REQUIRE(cond, status, msg) \
  do {                                \
    if (!(cond)) throw ::lc::Error((status), (msg)); \
  } while (0)

// ---------------------------------------------------------------- numerics
// Unit roundoff of FP32 and FP64 (round to nearest).
constexpr double kU32 = 5.9604644775390625e-08;   // 2^-24
constexpr double kU64 = 1.1102230246251565e-16;   // 2^-53

inline double gamma32(int n) { return n * kU32 / (1.0 - n * kU32); }
inline double gamma64(int n) { return n * kU64 / (1.0 - n * kU64); }

// Relative error bound of the canonical FP32 squared distance (see
// dist2_canonical): every term e_j^2 passes one subtraction rounding (which
// at most doubles in the square), at most 32 roundings inside its 32-wide
// chunk and at most d_pad/32 - 1 roundings while the chunk sums are added, so
// |S~ - S| <= gamma_{d_pad/32 + 33} S (all terms are non-negative). A small
// slack covers the FP64 arithmetic that forms the threshold.
inline double eps_recheck(int dpad) { return gamma32(dpad / 32 + 33) * (1.0 + 1.0 / 1024); }

// Relative slack of the tensor-core screen. With TF32 operands (10 explicit
// mantissa bits, error <= 2^-10 relative whether truncated or rounded) a
// product is within (2^-9 + 2^-20)|q_j k_j|; FP32-or-better accumulation of
// d_pad products adds at most d_pad 2^-22 sum|q_j k_j|. The sum |q_j k_j| is
// at most ||q|| ||k|| <= (||q||^2 + ||k||^2)/2. The bound is doubled for
// safety, and the FP32 norms (error gamma_{d_pad}) plus one final rounding
// are added on top.
inline double c_screen(int dpad) {
  return 2.0 * (std::ldexp(1.0, -9) + std::ldexp(1.0, -20) + dpad * std::ldexp(1.0, -22)) + 2.0 * gamma32(dpad) +
         std::ldexp(1.0, -20);
}

// sigma from the power iteration is a Rayleigh-quotient estimate (from
// below); radii used for acceptance divide by sigma * (1 + kSigmaSlack).
constexpr double kSigmaSlack = 1e-9;

// Constants of the probe thresholds of one entry (see thresholds()).
struct ThreshConsts {
  float om_eps_rd;   // 1 - eps_rc, rounded down
  float inv_omg_ru;  // 1 / (1 - gamma_{d_pad/32+33}), rounded up
  float om_c_rd;     // 1 - c_screen, rounded down
};

inline ThreshConsts thresh_consts(int dpad) {
  ThreshConsts t;
  t.om_eps_rd = std::nextafter((float)(1.0 - eps_recheck(dpad)), 0.0f);
  t.inv_omg_ru = std::nextafter((float)(1.0 / (1.0 - gamma32(dpad / 32 + 33))), 2.0f);
  t.om_c_rd = std::nextafter((float)(1.0 - c_screen(dpad)), 0.0f);
  return t;
}

#ifdef __CUDACC__
// Probe thresholds of an entry with radius lower bound r_lo (FP32, already
// rounded down) and FP32 squared norm kn, every step rounded so that it can
// only lower them: the recheck threshold rr <= r_lo^2 (1 - eps_rc) on the
// canonical FP32 squared distance, and the screen term
// tau <= ((1 - c_screen) kn - rr / (1 - gamma)) / 2.
__device__ __forceinline__ void thresholds(float r_lo, float kn, const ThreshConsts& t, float& rr, float& tau) {
  rr = __fmul_rd(__fmul_rd(r_lo, r_lo), t.om_eps_rd);
  const float Rt = __fmul_ru(rr, t.inv_omg_ru);
  tau = __fmul_rd(__fsub_rd(__fmul_rd(t.om_c_rd, kn), Rt), 0.5f);
}
#endif

// ---------------------------------------------------------------- state
struct SpecResult {
  double sigma;
  double theta;
  double residual_rel;
  int iterations;
  int converged;
  int degenerate;
  int pad;
};

struct DevStats {
  unsigned long long candidates;
  unsigned long long errors;
  int abort_flag;  // set by a kernel whose bounded wait expired; cleared per probe
  int fix_count;   // rows of the current certification listed for the FP64 pass (cleared per certification)
  unsigned long long ins_pairs;      // (row, class) pairs refined by the tensor certify kernel
  unsigned long long ins_full_rows;  // row halves it refined over every class
  unsigned long long ins_fp64_rows;  // rows re-certified by the FP64 pass
};

// Scratch of the selection strategy (select.cu), grown on demand.
struct SelectScratch {
  unsigned long long* keys = nullptr;
  int64_t keys_cap = 0;
  float* G = nullptr;  // chunk members' features
  int64_t G_cap = 0;
  int32_t* rows = nullptr;
  int64_t rows_cap = 0;
  int64_t* hit = nullptr;
  int64_t hit_cap = 0;
  uint32_t* cov = nullptr;
  int64_t cov_cap = 0;
  int32_t* list = nullptr;
  int64_t list_cap = 0;
  int32_t* class_cnt = nullptr;
  int64_t class_cap = 0;
  float* kc_mind = nullptr;  // K-center: squared distance to the nearest centre
  int64_t kc_mind_cap = 0;
  int64_t* small = nullptr;       // device: accepted, kept, chunk count
  int64_t* small_host = nullptr;  // pinned
};

// Per-entry table of the cache (structure of arrays, capacity entries).
struct Table {
  float* keys = nullptr;     // capacity x dpad, zero padded
  float* kn = nullptr;       // FP32 ||k||^2
  float* tau = nullptr;      // screen threshold term
  float* rr = nullptr;       // acceptance threshold on the FP32 squared distance
  float* radius = nullptr;   // reported radius r (rounded toward zero)
  int32_t* label = nullptr;  // payload
  int32_t* yG = nullptr;     // GuardNet label of the cached feature
};

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

}  // namespace lc

struct lipcache {
  int device = 0;
  int num_sms = 0;
  int d = 0, C = 0, dpad = 0;
  int64_t capacity = 0, size = 0;
  int64_t table_rows = 0;  // capacity rounded up to 256 (whole key tiles)
  int radius_mode = 0;
  double radius_scale = 1.0;
  int probe_path = LIPCACHE_PROBE_AUTO;
  int last_probe_path = 0;
  int last_grid = 0, last_cluster = 0;
  int squarings = 40, max_iter = 1000;
  bool head_set = false;
  double sigma = 0.0, sigma_residual = 0.0;
  int sigma_iterations = 0;

  // head
  float* W = nullptr;        // C x d
  float* b = nullptr;        // C
  double* Wnorm = nullptr;   // C
  float* Wnorm32 = nullptr;  // C, ||W_c|| rounded up to FP32
  double* pairnorm = nullptr;  // C x C (tight mode)
  double* inv_pairnorm = nullptr;  // C x C: 1 / pairnorm (0 where pairnorm is 0)
  float* ipn_up32 = nullptr;       // C x C: FP32 upper bound of 1 / ||W_y - W_j|| (+inf where it is 0)
  float* ipn_dn32 = nullptr;       // C x C: FP32 lower bound (+inf where ||W_y - W_j|| is 0)
  float* ipn_min32 = nullptr;      // C: min_j of ipn_dn32[y][j] over the rows W_j != W_y (0 if none)
  float* ipn_max32 = nullptr;      // C: max_j of ipn_up32[y][j] over j != y (+inf if some W_j = W_y)
  double* gram[2] = {nullptr, nullptr};  // d x d FP64
  lc::SpecResult* spec = nullptr;        // device
  lc::SpecResult* spec_host = nullptr;   // pinned

  lc::Table table;

  // insert scratch (grows)
  int64_t ins_cap = 0;
  uint8_t* ins_accept = nullptr;
  int32_t* ins_yG = nullptr;
  int32_t* ins_label = nullptr;
  float* ins_radius = nullptr;
  float* ins_rr = nullptr;
  float* ins_kn = nullptr;
  float* ins_tau = nullptr;
  int32_t* ins_rank = nullptr;
  int32_t* ins_fix = nullptr;  // rows listed for the FP64 pass of the current certification
  int32_t* ins_bcount = nullptr;
  int32_t* ins_boffset = nullptr;
  int64_t* ins_total = nullptr;       // device, 4: rows appended; consistency counts
  int64_t* ins_total_host = nullptr;  // pinned, 4
  // The table size also lives on the device: k_scan takes an insert's base
  // index from it and advances it, so inserts chain on their stream without
  // the host. An insert called without a host count does not wait; `size` is
  // then settled (synchronising pending_stream) by the next call that needs it.
  int64_t* size_dev = nullptr;     // device, 1
  int64_t* ins_size0 = nullptr;    // device, 1: base index of the current insert
  int64_t* size_pinned = nullptr;  // pinned, 1
  bool size_pending = false;       // an asynchronous insert is not yet in `size`
  int64_t pending_rows = 0;        // rows passed to those inserts (bounds their growth)
  cudaStream_t pending_stream = nullptr;

  // probe scratch (grows)
  int64_t q_cap = 0;  // rows (multiple of 128)
  float* qpad = nullptr;
  float* kappa = nullptr;
  unsigned long long* best = nullptr;
  // host-buffer probe staging
  int64_t hq_cap = 0;
  float* hq = nullptr;
  int64_t* hidx = nullptr;
  int32_t* hlabel = nullptr;
  float* hdist = nullptr;

  lc::DevStats* stats = nullptr;
  lc::DevStats* stats_host = nullptr;

  // main-kernel timing: a ring of event pairs harvested lazily
  static constexpr int kTimingRing = 64;
  bool timing = false;
  cudaEvent_t tev0[kTimingRing] = {}, tev1[kTimingRing] = {};
  int64_t t_issued = 0, t_harvested = 0;
  double t_ms_total = 0.0;
  int64_t t_count = 0;
  uint8_t t_kind[kTimingRing] = {};  // per slot: 0 probe main kernel, 1 certify kernel
  double ti_ms_total = 0.0;          // certify kernels
  int64_t ti_count = 0;
  float last_ms = 0.f;

  double eps_rc = 0.0, c_scr = 0.0;
  lc::EncodeTiledFn encode = nullptr;
  int pair_clusters = -1;  // resident clusters of the pair probe kernel (-1: not yet queried)
  // Launch state of the tensor probe kernels kept across calls, so that a
  // probe's host side does not repeat the occupancy query, the shared-memory
  // attribute and the tensor-map encoding: [0] k_probe_tc with 256-key
  // tiles, [1] with 128-key tiles, [2] k_probe_pair.
  struct ProbeLaunch {
    int resident = 0;  // clusters that fit (0: not queried yet)
    int smem = 0;      // dynamic shared memory the attribute was set for
    CUtensorMap tmK, tmQ;
    const void* k_base = nullptr;
    uint64_t k_rows = 0;
    const void* q_base = nullptr;
    uint64_t q_rows = 0;
  } probe_launch[3];
  cudaEvent_t launch_event = nullptr;  // recorded right before the main probe kernel when set
  bool probe_carveout_set = false;     // the prologue / finalize kernels' carveout preference
  int debug_flags = 0;     // LIPCACHE_DEBUG_* test hooks
  int last_insert_kernel = 0;  // LIPCACHE_INSERT_*
  float* wt_prep = nullptr;    // the head in the wide-tile certify kernel's shared-memory layout
  size_t wt_prep_cap = 0;      // bytes allocated
  int wt_prep_ncg = 0;         // classes per thread it was laid out for (0: stale)
  lc::SelectScratch sel;

  // radius policy (Sec. 5.4): the probe reads rr_emp / tau_emp instead of
  // the certified thresholds when policy != LIPCACHE_POLICY_CERTIFIED
  int policy = LIPCACHE_POLICY_CERTIFIED;
  double policy_param = 0.0;
  float* rr_emp = nullptr;   // table_rows
  float* tau_emp = nullptr;  // table_rows
  float* rho32 = nullptr;    // C: per-class radius, rounded down
  double* rho = nullptr;     // C: per-class radius (FP64)
  double* cls_sum = nullptr;       // per-block class sums (policy scratch)
  int64_t* cls_cnt = nullptr;      // per-block class counts
  int64_t cls_blocks = 0;

  const float* probe_rr() const { return policy ? rr_emp : table.rr; }
  const float* probe_tau() const { return policy ? tau_emp : table.tau; }
};

namespace lc {

// ---------------------------------------------------------------- launchers
// spectral.cu
void spectral_norm(lipcache* h, cudaStream_t s);
// certify.cu
// Certify H and append the accepted rows; miss_of (nullable, n entries) limits
// acceptance to rows with miss_of[row] < 0 (write-back of probe misses).
void certify_insert(lipcache* h, const float* H, int64_t n, const int32_t* payload, int require_consistency,
                    int64_t* out_index, float* out_radius, cudaStream_t s, const int64_t* miss_of = nullptr);
// policy.cu: switch the probe's thresholds to an empirical radius policy
// (or back to the certified ones); rho_host (nullable) receives C radii.
void set_radius_policy(lipcache* h, int policy, double param, double* rho_host, cudaStream_t s);
// thresholds of entries [first, first + n) under the current policy
void policy_fill(lipcache* h, int64_t first, int64_t n, cudaStream_t s);
// certify.cu: certification of H into the insert scratch only (no append)
// E_DEVICE (after synchronising `s`) if the last certification gave up on a
// bounded wait; nothing was appended then.
constexpr const char* kCertifyAbortMessage =
    "a bounded wait of the tensor certify kernel expired; no row was certified or inserted";
void require_certify_ok(lipcache* h, cudaStream_t s);
// Bring `size` up to date with asynchronous inserts (synchronises their
// stream if one is pending), and write the host size to the device counter
// after a path that grew the table from the host.
void settle_size(lipcache* h);
void store_size_dev(lipcache* h, cudaStream_t s);
void certify_rows(lipcache* h, const float* H, int64_t n, const int32_t* payload, int require_consistency,
                  cudaStream_t s);
// select.cu: radius-prioritised de-duplication of the certified rows of H
// into the cache; returns the number of entries appended.
int64_t select_insert(lipcache* h, const float* H, int64_t n, const int32_t* payload, int require_consistency,
                      int64_t budget_total, int budget_per_class, int64_t* out_index, float* out_radius,
                      cudaStream_t s);
// select.cu: K-center per class (at most budget_per_class centres per class)
int64_t select_kcenter(lipcache* h, const float* H, int64_t n, const int32_t* payload, int require_consistency,
                       int budget_per_class, int64_t* out_index, float* out_radius, cudaStream_t s);
void release_select(lipcache* h);
// Certified-consistency check: argmax of the head on Q against y^G of the hit
// entries; counts (hits, consistent, invalid index) land in ins_total[1..3].
void consistency_check(lipcache* h, const float* Q, int64_t B, const int64_t* hit_index, int8_t* out,
                       cudaStream_t s);
// probe.cu
void probe(lipcache* h, const float* Q, int64_t B, int64_t* out_index, int32_t* out_label, float* out_dist,
           cudaStream_t s);
bool tensor_path_supported(int dpad);
// probe_tc.cu: the tensor probe; `path` is LIPCACHE_PROBE_TENSOR (kernel
// chosen by shape), _TENSOR_SINGLE or _TENSOR_PAIR. Returns the kernel that
// ran (_TENSOR_SINGLE or _TENSOR_PAIR).
int launch_probe_tc(lipcache* h, int64_t B, int path, cudaStream_t s);
// probe_pair.cu
int probe_pair_clusters(lipcache* h);
void launch_probe_pair(lipcache* h, int64_t B, const float* qpad, const float* kappa, unsigned long long* best,
                       cudaStream_t s);
// probe.cu / probe_tc.cu: the probe on caller-provided scratch memory
void probe_external_scratch(lipcache* h, const float* Q, int64_t B, int64_t* out_index, int32_t* out_label,
                            float* out_dist, float* qpad, float* kappa, unsigned long long* best, cudaStream_t s);
int launch_probe_tc_external(lipcache* h, int64_t B, int path, const float* qpad, const float* kappa,
                             unsigned long long* best, cudaStream_t s);
// api.cu: run fn(ctx) with the C ABI's error handling (status + message)
lipcache_status run_guarded(void (*fn)(void*), void* ctx);
// api.cu: harvest completed timing events (blocking on the oldest if `all`
// or if the ring is full).
void harvest_timing(lipcache* h, bool all);

}  // namespace lc
