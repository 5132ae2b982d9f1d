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
// 16-byte aligned, head resident in shared memory), and its launch.
bool certify_tc_supported(const lipcache* h, const float* H, int64_t n);
void certify_tc_launch(lipcache* h, const CertArgs& a, cudaStream_t s);

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
// (one thread), and the skip rules of Algorithm 1.
__device__ void row_finals(const CertArgs& a, int64_t row, const RowVals& v, uint8_t* acc_slot) {
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
  if (a.fix_list && mval == mval && !(mval * kFixRel > (double)v.e1 + (double)v.em))
    a.fix_list[atomicAdd(a.fix_count, 1)] = (int32_t)row;
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
// probe thresholds and the skip rules of Algorithm 1 for one row (one thread).
__device__ void tight_write(const CertArgs& a, int64_t row, int y, double rmin, double smin, bool any_nan, float kn,
                            uint8_t* acc_slot) {
  const double r64 = any_nan ? NAN : a.kappa * rmin;
  const double rs = (smin > 0.0 && !any_nan) ? __dmul_rd(a.kappa, smin) : 0.0;
  const int32_t lab = a.payload ? a.payload[row] : y;
  const bool acc = !(a.require_consistency && lab != y) && (r64 > 0.0) && !(a.miss_of && a.miss_of[row] >= 0);
  // rmin - smin bounds the error of rmin (smin is the certified lower bound
  // of the same minimum); rows where it is not below kFixRel rmin (a near
  // tie for y^G or a tiny term of Eq. 29) go to the FP64 pass
  if (a.fix_list && !any_nan && rmin < INFINITY && !((rmin - smin) < kFixRel * rmin))
    a.fix_list[atomicAdd(a.fix_count, 1)] = (int32_t)row;
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
}

}  // namespace
}  // namespace lc
