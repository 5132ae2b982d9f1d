// Device helpers shared by the certify kernels (Sec. 3.3, Algorithm 1; Eqs.
// 20, 21): the kernel arguments, FP32 error-free transformations, the
// compensated dot product, logit error bounds, the running top-two selection
// over refined candidates and the FP64 per-row finals.
#pragma once
#include "internal.cuh"

namespace lc {

struct CertArgs {
  const float* H;
  int64_t n;
  int d, C, hstride, lstride, tight, require_consistency;
  const float* W;
  const float* b;
  const double* Wnorm;
  const double* pairnorm;
  const int32_t* payload;
  double sigma, kappa, eps_rc, gamma_rc, c_scr, g32, g64;
  const float* Wnorm32;  // ||W_c|| rounded up
  float g32f;            // gamma_{d+2} with FP32 rounding slack
  // error factors of the compensated dot products (dot2_factor): the whole
  // feature sequence in one lane, 8-lane groups, and 32-lane warps
  float g2f, g2f8, g2f32;
  double inv_denom;      // kappa / (sigma sqrt 2)
  double inv_denom_safe; // kappa (1 - 8u) / (sigma (1 + slack) sqrt 2)
  ThreshConsts tc;       // constants of the probe thresholds
  const int64_t* miss_of;      // nullable: row accepted only if miss_of[row] < 0 (write-back)
  const double* inv_pairnorm;  // 1 / ||W_y - W_j|| (tight mode)
  const float* ipn_up32;       // FP32 brackets of 1 / ||W_y - W_j|| (tight mode; +inf where the rows coincide)
  const float* ipn_dn32;
  const float* ipn_min32;      // per class: a lower bound of every 1 / ||W_y - W_j|| (tight mode)
  const float* ipn_max32;      // per class: an upper bound of every 1 / ||W_y - W_j|| (tight mode)
  double tight_f;              // 1 - gamma_{d+8} (FP64)
  uint8_t* accept;
  int32_t* yG;
  int32_t* label;
  float* radius;
  float* rr;
  float* kn;
  float* tau;
  int32_t* rank;
  int32_t* bcount;
  // rows whose radius the compensated FP32 refinement cannot pin to kFixRel
  // relative: listed here for the FP64 pass (k_certify_fix); nullable
  int* fix_count;
  int32_t* fix_list;
  float gfix;  // rounding-error factor of the FP64 pass's logits (rounded up)
};

// Relative accuracy the reported radius must reach without the FP64 pass: a
// row whose margin (conservative radius) or minimising term of Eq. 29 (tight
// radius) is not known to within this fraction from the compensated FP32
// refinement's error bounds is re-certified in FP64. Half of the 1e-5 the
// radii are compared at, leaving room for the FP32 rounding of the result.
constexpr double kFixRel = 5e-6;

// The tensor-core certify kernel (certify_tc.cu): whether it takes this
// insert (either radius, d % 16 == 0, 32 <= d <= 256, 2 <= C <= 256, rows
// 16-byte aligned, head resident in shared memory), and its launch; true if
// the kernel runs the FP64 pass over the rows it lists itself.
bool certify_tc_supported(const lipcache* h, const float* H, int64_t n);
bool certify_tc_launch(lipcache* h, const CertArgs& a, cudaStream_t s);

namespace {

constexpr unsigned kFull = 0xffffffffu;

// Start moving `bytes` (a multiple of 16) from global memory at `src` (16-byte
// aligned) into L2, without waiting.
__device__ __forceinline__ void prefetch_l2_bulk(const void* src, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(reinterpret_cast<uint64_t>(src)), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ float warp_sum_f(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
  return v;
}
__device__ __forceinline__ double warp_sum_d(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
  return v;
}
__device__ __forceinline__ double warp_max_d(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmax(v, __shfl_xor_sync(kFull, v, o));
  return v;
}
__device__ __forceinline__ double warp_min_d(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmin(v, __shfl_xor_sync(kFull, v, o));
  return v;
}
// insert v into (t1 >= t2)
__device__ __forceinline__ void top2_push(double& t1, double& t2, double v) {
  if (v > t1) {
    t2 = t1;
    t1 = v;
  } else if (v > t2) {
    t2 = v;
  }
}

// FP32 error-free transformations: a + b = s + e and a * b = p + e exactly
// (Knuth's TwoSum; TwoProduct with a fused multiply-add).
__device__ __forceinline__ void two_sum(float a, float b, float& s, float& e) {
  s = __fadd_rn(a, b);
  const float bb = __fsub_rn(s, a);
  e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
}

// Compensated dot product W_c . h + b_c (Ogita, Rump and Oishi's Dot2, summed
// across the warp with the same transformations), returned as a normalised
// pair hi + lo (|lo| <= ulp(hi)/2) whose exact sum is within
// g2f32 (sum_j |W_cj h_j| + |b_c|) of the exact value (dot2_factor). Every lane
// gets the same bits: each butterfly step combines the two partners' pairs
// symmetrically. wc[j * ws] and hrow[j * hs] address feature j of the
// weights and of the row (global memory, or the transposed shared tiles).
__device__ __forceinline__ void dot2_logit(const float* __restrict__ wc, int ws, const float* __restrict__ hrow, int hs,
                                           float bias, int d, int lane, float& hi, float& lo) {
  float p = 0.f, c = 0.f;
  for (int j = lane; j < d; j += 32) {
    const float w = wc[(size_t)j * ws], x = hrow[(size_t)j * hs];
    const float pr = __fmul_rn(w, x);
    const float er = __fmaf_rn(w, x, -pr);
    float t, q;
    two_sum(p, pr, t, q);
    p = t;
    c = __fadd_rn(c, __fadd_rn(q, er));
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float pb = __shfl_xor_sync(kFull, p, o), cb = __shfl_xor_sync(kFull, c, o);
    float t, q;
    two_sum(p, pb, t, q);
    p = t;
    c = __fadd_rn(__fadd_rn(c, cb), q);
  }
  float t, q;
  two_sum(p, bias, t, q);
  two_sum(t, __fadd_rn(c, q), hi, lo);
}

// Absolute error allowance for subnormal intermediate results: at most
// 2^-150 per rounding, (d + 40) * 2^-150 < 1e-39 in all for d <= 1024.
constexpr float kTinyF = 1e-35f;

// Rounded-up bound E_c of |s~_c - s_c| for an FP32 logit s~_c:
// gamma_{d+2} (||W_c|| ||z|| + |b_c|) (g32f carries the slack for its own
// rounding), 2^-22 |s~_c| for the rounding of the interval ends, and kTinyF.
__device__ __forceinline__ float logit_err(float g32f, float wn, float hn, float b, float sv) {
  return __fmaf_ru(g32f, __fmaf_ru(wn, hn, fabsf(b)), __fmaf_ru(fabsf(sv), 2.3841858e-07f /* 2^-22 */, kTinyF));
}

// (ah, al) > (bh, bl) for pairs normalised by a final TwoSum (hi = RN(hi + lo)):
// round-to-nearest is monotone, so this orders the exact sums.
__device__ __forceinline__ bool pair_gt(float ah, float al, float bh, float bl) {
  return ah > bh || (ah == bh && al > bl);
}

// Per-row result of the candidate refinement: the best and second-best
// refined logits (pairs hi + lo), the error bound of the best, the largest
// upper bound v + e among the other candidates, ||z||^2 (FP32) and y^G.
struct RowVals {
  float h1, l1, e1, h2, l2, up, kn;
  float em;  // the largest error bound among the refined classes
  int y;
};

// Upper bound of ||z|| from the FP32 sum of squares kn (any order: within
// gamma_d < 1e-4 of ||z||^2 for d <= 1024, plus d * 2^-150 for subnormal
// squares).
__device__ __forceinline__ float norm_upper(float kn) {
  return __fmul_ru(__fsqrt_ru(__fmaf_ru(kn, 1.0f + 1e-4f, kTinyF)), 1.0f + 1e-6f);
}

// Bound of |hi + lo - s_c| for a refined logit, rounded up (plus the absolute
// error of subnormal products); g2f: the factor of the refinement's lane
// layout (CertArgs::g2f, g2f8 or g2f32).
__device__ __forceinline__ float refined_err(float g2f, float wn, float hn, float b) {
  return __fmaf_ru(g2f, __fmaf_ru(wn, hn, fabsf(b)), kTinyF);
}

// Running selection over refined candidates, visited in any order: the best
// by (value desc, class asc), the second-best value, and the top two upper
// bounds with the class of the first, so that the largest upper bound among
// the classes other than the best is available at the end.
struct Top2 {
  float b1h = -INFINITY, b1l = 0.f, b2h = -INFINITY, b2l = 0.f, e1 = 0.f;
  float u1 = -INFINITY, u2 = -INFINITY;
  float em = 0.f;  // largest error bound pushed
  int y = -1, cu1 = -1;
  bool nan = false;  // a refined logit is NaN: the row is rejected
  __device__ __forceinline__ void push(int c, float vh, float vl, float e) {
    nan |= !(vh == vh && vl == vl);
    em = fmaxf(em, e);
    const bool eq1 = vh == b1h && vl == b1l;
    if (pair_gt(vh, vl, b1h, b1l) || (eq1 && c < y)) {
      b2h = b1h;
      b2l = b1l;
      b1h = vh;
      b1l = vl;
      e1 = e;
      y = c;
    } else if (pair_gt(vh, vl, b2h, b2l) || (vh == b2h && vl == b2l)) {
      b2h = vh;
      b2l = vl;
    }
    const float up = __fadd_ru(vh, __fadd_ru(vl, e));
    if (up > u1) {
      u2 = u1;
      u1 = up;
      cu1 = c;
    } else if (up > u2) {
      u2 = up;
    }
  }
  __device__ __forceinline__ RowVals result(float kn) const {
    RowVals v;
    v.h1 = nan ? NAN : b1h;
    v.l1 = b1l;
    v.e1 = e1;
    v.h2 = b2h;
    v.l2 = b2l;
    v.up = (cu1 == y) ? u2 : u1;
    v.kn = kn;
    v.em = em;
    v.y = y < 0 ? 0 : y;  // every refined logit NaN: the margin is NaN and the row is rejected
    return v;
  }
};

// FP64 margin, radius, certified lower bound and probe thresholds of one row
// (one thread), and the skip rules of Algorithm 1. Returns whether the row
// was listed for the FP64 pass (after its results are written).
__device__ bool row_finals(const CertArgs& a, int64_t row, const RowVals& v, uint8_t* acc_slot) {
  const double v1 = (double)v.h1 + (double)v.l1, v2 = (double)v.h2 + (double)v.l2;
  const double mval = (v1 == v1 && v2 == v2) ? v1 - v2 : NAN;
  // lower bound of the exact margin with downward rounding
  const double mlo = __dsub_rd(__dsub_rd(v1, (double)v.e1), (double)v.up);
  const double r64 = mval * a.inv_denom;
  const double rs = (mlo > 0.0) ? __dmul_rd(mlo, a.inv_denom_safe) : 0.0;
  const int32_t lab = a.payload ? a.payload[row] : v.y;
  const bool acc = !(a.require_consistency && lab != v.y) && (r64 > 0.0) && !(a.miss_of && a.miss_of[row] >= 0);
  // The margin is known to within e1 + em (the best class's error bound and
  // the largest among the others: whichever class is the true runner-up, the
  // refined runner-up value is within em of it); where that is not below
  // kFixRel m, the row goes to the FP64 pass, which rewrites everything below.
  // (up, an FP32 upper end, cannot serve here: its rounding is an ulp of the
  // logit, far above the refinement's error.)
  const bool fix = a.fix_list && mval == mval && !(mval * kFixRel > (double)v.e1 + (double)v.em);
  if (fix) a.fix_list[atomicAdd(a.fix_count, 1)] = (int32_t)row;
  float rr, tau;
  thresholds(__double2float_rd(rs), v.kn, a.tc, rr, tau);
  a.accept[row] = acc ? 1 : 0;
  a.yG[row] = v.y;
  a.label[row] = lab;
  a.radius[row] = __double2float_rz(r64);
  a.rr[row] = rr;
  a.kn[row] = v.kn;
  a.tau[row] = tau;
  *acc_slot = acc ? 1 : 0;
  return fix;
}

// One term of Eq. 29 for the refined logits vy (error ey) of y^G and vj (ej)
// of a class j: the radius candidate (s_y - s_j) / ||W_y - W_j|| and its
// certified lower bound (rounded downwards, 1 - gamma_{d+8} for the FP64
// reciprocal), folded into running minima. Pairs with W_j = W_y are skipped.
__device__ __forceinline__ void tight_term(const CertArgs& a, int y, int j, double vy, double ey, double vj, double ej,
                                           double& rmin, double& smin) {
  const double pn = a.pairnorm[(size_t)y * a.C + j];
  if (!(pn > 0.0)) return;
  const double ipn = a.inv_pairnorm[(size_t)y * a.C + j];
  rmin = fmin(rmin, (vy - vj) * ipn);
  const double num = __dsub_rd(__dsub_rd(vy, ey), __dadd_ru(vj, ej));
  smin = fmin(smin, __dmul_rd(__dmul_rd(num, ipn), a.tight_f));
}

// The tight radius r* = kappa rmin (Eq. 29), its certified lower bound, the
// probe thresholds and the skip rules of Algorithm 1 for one row (one
// thread). Returns whether the row was listed for the FP64 pass.
__device__ bool tight_write(const CertArgs& a, int64_t row, int y, double rmin, double smin, bool any_nan, float kn,
                            uint8_t* acc_slot) {
  const double r64 = any_nan ? NAN : a.kappa * rmin;
  const double rs = (smin > 0.0 && !any_nan) ? __dmul_rd(a.kappa, smin) : 0.0;
  const int32_t lab = a.payload ? a.payload[row] : y;
  const bool acc = !(a.require_consistency && lab != y) && (r64 > 0.0) && !(a.miss_of && a.miss_of[row] >= 0);
  // rmin - smin bounds the error of rmin (smin is the certified lower bound
  // of the same minimum); rows where it is not below kFixRel rmin (a near
  // tie for y^G or a tiny term of Eq. 29) go to the FP64 pass
  const bool fix = a.fix_list && !any_nan && rmin < INFINITY && !((rmin - smin) < kFixRel * rmin);
  if (fix) a.fix_list[atomicAdd(a.fix_count, 1)] = (int32_t)row;
  float rr, tau;
  thresholds(__double2float_rd(rs), kn, a.tc, rr, tau);
  a.accept[row] = acc ? 1 : 0;
  a.yG[row] = y;
  a.label[row] = lab;
  a.radius[row] = __double2float_rz(r64);
  a.rr[row] = rr;
  a.kn[row] = kn;
  a.tau[row] = tau;
  *acc_slot = acc ? 1 : 0;
  return fix;
}

// ---------------------------------------------------------------- FP64 pass
// Re-certification in FP64 of one row the compensated FP32 refinement could
// not pin down (listed by row_finals / tight_write: a margin, or a minimising
// term of Eq. 29, smaller than 1 / kFixRel times its error bound - rows a hair
// from a decision boundary, a few per 100,000 rows of the scale workload), on
// one warp. FP64 arithmetic on this GPU has a small fraction of the FP32
// throughput, so it is kept to the few operations that need it: FP32 logits
// and error bounds of every class (a lane per class, a fused multiply-add
// chain over the features in order) pick the classes that can matter; those
// are recomputed in FP64 four at a time (products of FP32 values are exact in
// FP64; each lane chains its slice of the features, a five-level tree sums
// the lanes: error below gamma_{d/32+6} of sum |W_cj z_j| + |b_c|);
// comparisons of FP64 values use order-preserving integer keys; y^G, the
// margin or Eq. 29, the certified lower bound, the thresholds and the skip
// rules of Algorithm 1 are then taken from the FP64 values and overwrite the
// row's results. Conservative radius: the candidates are the classes whose
// FP32 interval reaches the second-largest lower end (they include the true
// top two). Tight radius: the possible y^G (intervals reaching the largest
// lower end), then, for the FP64 y^G, the classes whose lower bracket of
// (s_y - s_j) / ||W_y - W_j|| reaches the smallest upper bracket (they
// include the minimiser of Eq. 29). Every value depends only on the row and
// the head, so the stand-alone pass and the tensor kernel's fix warp write
// the same bits.

// Order-preserving integer key of a double: a larger value has a larger key
// (-0 and +0 share the key of 0).
__device__ __forceinline__ long long dkey(double v) {
  long long b = __double_as_longlong(v);
  if (b == (long long)0x8000000000000000ull) b = 0;
  return b >= 0 ? b : (b ^ 0x7fffffffffffffffll);
}
// (key, class) of the larger value, the lower class on equal values
__device__ __forceinline__ void argmax_key(long long& k, int& c, long long k2, int c2) {
  if (c2 >= 0 && (c < 0 || k2 > k || (k2 == k && c2 < c))) {
    k = k2;
    c = c2;
  }
}
__device__ __forceinline__ void warp_argmax_key(long long& k, int& c) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) argmax_key(k, c, __shfl_xor_sync(kFull, k, o), __shfl_xor_sync(kFull, c, o));
}

// Shared-memory scratch of one warp's FP64 pass: the FP64 values of the
// candidates, the row, the FP32 logits and bounds, the bounds of the FP64
// values and the candidate classes. 16-byte aligned base.
struct FixScratch {
  double* cv;
  float* zs;
  float* sv;
  float* ev;
  float* ce;
  int* cls;
};
__host__ __device__ inline size_t fix_scratch_bytes(int d, int C) {
  const size_t C4 = (size_t)(C + 3) / 4 * 4, d4 = (size_t)(d + 3) / 4 * 4;
  return 8 * C4 + 4 * d4 + 16 * C4;
}
__device__ inline FixScratch fix_scratch_at(unsigned char* p, int d, int C) {
  const size_t C4 = (size_t)(C + 3) / 4 * 4, d4 = (size_t)(d + 3) / 4 * 4;
  FixScratch s;
  s.cv = reinterpret_cast<double*>(p);
  s.zs = reinterpret_cast<float*>(p + 8 * C4);
  s.sv = s.zs + d4;
  s.ev = s.sv + C4;
  s.ce = s.ev + C4;
  s.cls = reinterpret_cast<int*>(s.ce + C4);
  return s;
}

// FP64 logits of the N classes cls[0..N) (warp-uniform) of the row zs into
// cv / ce (lane 0 stores), with FP32 bounds of their errors (rounded up).
// W(c, j): feature j of the head's row c. (FP64 instructions occupy the
// sub-partition's FP64 pipe for tens of cycles each on this GPU: no slot is
// computed that is not used.)
template <int N, class WAt>
__device__ __forceinline__ void logits_fp64(const CertArgs& a, const WAt& W, const int* cls,
                                            const float* __restrict__ zs, int lane, double* cv, float* ce) {
  int cc[N];
#pragma unroll
  for (int u = 0; u < N; ++u) cc[u] = cls[u];
  double acc[N];
  float pa[N];
#pragma unroll
  for (int u = 0; u < N; ++u) {
    acc[u] = 0.0;
    pa[u] = 0.f;
  }
  for (int j = lane; j < a.d; j += 32) {
    const float xf = zs[j];
    const double x = (double)xf;
    float w[N];
#pragma unroll
    for (int u = 0; u < N; ++u) w[u] = W(cc[u], j);
#pragma unroll
    for (int u = 0; u < N; ++u) {
      acc[u] = fma((double)w[u], x, acc[u]);
      pa[u] = __fmaf_ru(fabsf(w[u]), fabsf(xf), pa[u]);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1)
#pragma unroll
    for (int u = 0; u < N; ++u) {
      acc[u] += __shfl_xor_sync(kFull, acc[u], o);
      pa[u] = __fadd_ru(pa[u], __shfl_xor_sync(kFull, pa[u], o));
    }
  if (lane == 0)
#pragma unroll
    for (int u = 0; u < N; ++u) {
      const float bc = __ldg(a.b + cc[u]);
      cv[u] = acc[u] + (double)bc;
      ce[u] = __fmaf_ru(a.gfix, __fadd_ru(pa[u], fabsf(bc)), kTinyF);
    }
}

// Refine the n classes cls[0..n) (shared memory) into cv / ce, up to four at
// a time.
template <class WAt>
__device__ __forceinline__ void refine_list_fp64(const CertArgs& a, const WAt& W, const int* cls, int n,
                                                 const float* zs, int lane, double* cv, float* ce) {
  for (int k0 = 0; k0 < n; k0 += 4) {
    const int m = n - k0;
    if (m >= 4)
      logits_fp64<4>(a, W, cls + k0, zs, lane, cv + k0, ce + k0);
    else if (m == 3)
      logits_fp64<3>(a, W, cls + k0, zs, lane, cv + k0, ce + k0);
    else if (m == 2)
      logits_fp64<2>(a, W, cls + k0, zs, lane, cv + k0, ce + k0);
    else
      logits_fp64<1>(a, W, cls + k0, zs, lane, cv + k0, ce + k0);
  }
  __syncwarp();
}

// Append the classes c (c < C) with pred(c) to cls[n...] in ascending order.
template <typename Pred>
__device__ __forceinline__ int collect(int C, int lane, int* cls, int n, Pred pred) {
  for (int cb = 0; cb < C; cb += 32) {
    const int c = cb + lane;
    const bool t = c < C && pred(c);
    const unsigned m = __ballot_sync(kFull, t);
    if (t) cls[n + __popc(m & ((1u << lane) - 1u))] = c;
    n += __popc(m);
  }
  __syncwarp();
  return n;
}

// FP32 logits of NP classes per lane (the lane's classes c0 + 32 t) and the
// top two lower ends of their intervals: the class chains interleaved.
template <int NP, class WAt>
__device__ __forceinline__ void fix_screen(const CertArgs& a, const WAt& W, const FixScratch& s, int c0, float hn,
                                           float& l1, float& l2, bool& nan) {
  const int C = a.C;
  int cc[NP];
  float bc[NP], wn[NP], acc[NP];
#pragma unroll
  for (int t = 0; t < NP; ++t) {
    const int c = c0 + 32 * t;
    cc[t] = c < C ? c : C - 1;  // a valid row; its result is dropped
    bc[t] = __ldg(a.b + cc[t]);
    wn[t] = __ldg(a.Wnorm32 + cc[t]);
  }
  W.template chains<NP>(cc, s.zs, a.d, acc);
#pragma unroll
  for (int t = 0; t < NP; ++t) {
    const int c = c0 + 32 * t;
    if (c < C) {
      const float sc = __fadd_rn(acc[t], bc[t]);
      const float e = logit_err(a.g32f, wn[t], hn, bc[t], sc);
      s.sv[c] = sc;
      s.ev[c] = e;
      nan |= !(sc == sc);
      const float lo = __fsub_rd(sc, e);
      l2 = fmaxf(l2, fminf(l1, lo));
      l1 = fmaxf(l1, lo);
    }
  }
}

// The FP64 pass over one row on one warp (every lane calls it). kn: the
// row's FP32 sum of squares as the certify kernel computed it. W(c, j) reads
// the head; W.chains<NP>(cc, zs, d, acc) forms, for each of NP classes cc[t],
// the FP32 fused multiply-add chain sum_j W_cj zs_j over j = 0, 1, ..., d - 1
// in that order (the chains interleaved).
template <class WAt>
__device__ __forceinline__ void fix_row_warp(const CertArgs& a, int64_t row, float kn, const WAt& W, const FixScratch& s,
                                          int lane) {
  const int d = a.d, C = a.C;
  for (int j = lane; j < d; j += 32) s.zs[j] = __ldg(a.H + (size_t)row * d + j);
  __syncwarp();
  const float hn = norm_upper(kn);
  if (!(hn < INFINITY)) return;  // no finite bounds: keep the FP32 kernel's result
  // FP32 logits (within gamma_{d+2}) and the top two lower ends of their
  // intervals
  float l1 = -INFINITY, l2 = -INFINITY;
  bool nan = false;
  for (int cb = 0; cb < C; cb += 256) {
    const int np = (C - cb + 31) / 32;  // classes per lane in this round (the rest dropped)
    if (np > 4)
      fix_screen<8>(a, W, s, cb + lane, hn, l1, l2, nan);
    else if (np > 2)
      fix_screen<4>(a, W, s, cb + lane, hn, l1, l2, nan);
    else if (np == 2)
      fix_screen<2>(a, W, s, cb + lane, hn, l1, l2, nan);
    else
      fix_screen<1>(a, W, s, cb + lane, hn, l1, l2, nan);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float o1 = __shfl_xor_sync(kFull, l1, o), o2 = __shfl_xor_sync(kFull, l2, o);
    l2 = fmaxf(l2, fminf(l1, o1));
    l1 = fmaxf(l1, o1);
    l2 = fmaxf(l2, fminf(l1, o2));
    l1 = fmaxf(l1, o2);
  }
  if (__any_sync(kFull, nan)) return;  // keep the FP32 kernel's result (a rejected row)
  // the classes that can be y^G (tight) or among the top two (conservative)
  const float Lc = a.tight ? l1 : l2;
  const int nc = collect(C, lane, s.cls, 0, [&](int c) { return __fadd_ru(s.sv[c], s.ev[c]) >= Lc; });
  refine_list_fp64(a, W, s.cls, nc, s.zs, lane, s.cv, s.ce);
  // y^G: the largest refined value, the lower class on ties
  long long ky = 0;
  int y = -1;
  for (int t = lane; t < nc; t += 32) argmax_key(ky, y, dkey(s.cv[t]), s.cls[t]);
  warp_argmax_key(ky, y);
  if (y < 0) return;  // (every lane agrees)
  int ty = 0;  // y's slot
  for (int t = lane; t < nc; t += 32)
    if (s.cls[t] == y) ty = t;
  ty = __reduce_max_sync(kFull, ty);
  const double vy = s.cv[ty];
  const float ey = s.ce[ty];
  if (!a.tight) {
    // the runner-up value and the largest upper end among the other classes
    long long k2 = 0, ku = 0;
    int c2 = -1, cu = -1;
    for (int t = lane; t < nc; t += 32) {
      if (s.cls[t] == y) continue;
      argmax_key(k2, c2, dkey(s.cv[t]), s.cls[t]);
      argmax_key(ku, cu, dkey(__dadd_ru(s.cv[t], (double)s.ce[t])), s.cls[t]);
    }
    warp_argmax_key(k2, c2);
    warp_argmax_key(ku, cu);
    if (lane == 0) {
      double v2 = -INFINITY, up = -INFINITY;
      for (int t = 0; t < nc; ++t) {
        if (s.cls[t] == c2) v2 = s.cv[t];
        if (s.cls[t] == cu) up = __dadd_ru(s.cv[t], (double)s.ce[t]);
      }
      const double mval = vy - v2;
      const double mlo = __dsub_rd(__dsub_rd(vy, (double)ey), up);
      const double r64 = mval * a.inv_denom;
      const double rs = (mlo > 0.0) ? __dmul_rd(mlo, a.inv_denom_safe) : 0.0;
      const int32_t lab = a.payload ? a.payload[row] : y;
      const bool acc = !(a.require_consistency && lab != y) && (r64 > 0.0) && !(a.miss_of && a.miss_of[row] >= 0);
      float rr, tau;
      thresholds(__double2float_rd(rs), kn, a.tc, rr, tau);
      a.accept[row] = acc ? 1 : 0;
      a.yG[row] = y;
      a.label[row] = lab;
      a.radius[row] = __double2float_rz(r64);
      a.rr[row] = rr;
      a.tau[row] = tau;
    }
    __syncwarp();
    return;
  }
  // Eq. 29 for the FP64 y^G: FP32 brackets of every term from the FP32
  // logits and the FP32 brackets of the reciprocal pair norms, then FP64 for
  // the classes whose lower bracket reaches the smallest upper one
  const float vyh = __fadd_ru(__double2float_ru(vy), ey), vyl = __fsub_rd(__double2float_rd(vy), ey);
  const bool brk = a.ipn_up32 != nullptr && a.ipn_dn32 != nullptr;
  __syncwarp();  // every lane has read the candidates' values
  float U = INFINITY;
  if (brk)
    for (int j = lane; j < C; j += 32) {
      const float iu = a.ipn_up32[(size_t)y * C + j];
      if (j == y || !(iu < INFINITY)) continue;  // W_j = W_y: no term
      U = fminf(U, __fmul_ru(__fsub_ru(vyh, __fsub_rd(s.sv[j], s.ev[j])), iu));
    }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) U = fminf(U, __shfl_xor_sync(kFull, U, o));
  const int nj = collect(C, lane, s.cls, 0, [&](int j) {
    if (j == y) return false;
    if (!brk) return true;
    const float iu = a.ipn_up32[(size_t)y * C + j];
    return iu < INFINITY && __fmul_rd(__fsub_rd(vyl, __fadd_ru(s.sv[j], s.ev[j])), a.ipn_dn32[(size_t)y * C + j]) <= U;
  });
  refine_list_fp64(a, W, s.cls, nj, s.zs, lane, s.cv, s.ce);
  // the terms of Eq. 29 and their certified lower bounds (tight_term), one
  // lane per class, minima by key
  long long kr = dkey(INFINITY), ks = dkey(INFINITY);  // no term: r* = +inf
  for (int t = lane; t < nj; t += 32) {
    double rmin = INFINITY, smin = INFINITY;
    tight_term(a, y, s.cls[t], vy, (double)ey, s.cv[t], (double)s.ce[t], rmin, smin);
    kr = min(kr, dkey(rmin));
    ks = min(ks, dkey(smin));
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    kr = min(kr, __shfl_xor_sync(kFull, kr, o));
    ks = min(ks, __shfl_xor_sync(kFull, ks, o));
  }
  if (lane == 0) {
    // back from the keys (dkey is its own inverse on the bits)
    const double rmin = kr < 0 ? __longlong_as_double(kr ^ 0x7fffffffffffffffll) : __longlong_as_double(kr);
    const double smin = ks < 0 ? __longlong_as_double(ks ^ 0x7fffffffffffffffll) : __longlong_as_double(ks);
    const double r64 = a.kappa * rmin;
    const double rs = smin > 0.0 ? __dmul_rd(a.kappa, smin) : 0.0;
    const int32_t lab = a.payload ? a.payload[row] : y;
    const bool acc = !(a.require_consistency && lab != y) && (r64 > 0.0) && !(a.miss_of && a.miss_of[row] >= 0);
    float rr, tau;
    thresholds(__double2float_rd(rs), kn, a.tc, rr, tau);
    a.accept[row] = acc ? 1 : 0;
    a.yG[row] = y;
    a.label[row] = lab;
    a.radius[row] = __double2float_rz(r64);
    a.rr[row] = rr;
    a.tau[row] = tau;
  }
  __syncwarp();
}

}  // namespace
}  // namespace lc
