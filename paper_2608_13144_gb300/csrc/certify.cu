// Certified insertion (Sec. 3.3, Algorithm 1 loop body; Eqs. 5-6, 20, 21, 29).
//
// For each candidate row z:
//   s = W z + b                          (Eq. 5)
//   y^G = argmax_c s_c                   (Eq. 6; lowest class on ties)
//   m = s_y - max_{j != y} s_j           (Eq. 20)
//   r = kappa m / (sigma sqrt 2)         (Eq. 21)  or
//   r* = kappa min_j (s_y - s_j) / ||W_y - W_j||   (Remark 4.2, Eq. 29)
//   skip if consistency is required and payload != y^G, else if r <= 0.
//
// Accuracy. The radius must be right to ~1e-5 relative even for entries near
// a decision boundary, where m is a small difference of large logits. The
// kernel therefore computes all logits in FP32 with a proven error bound
// E_c = gamma_{d+2} (||W_c|| ||z|| + |b_c|), keeps every class whose FP32
// interval can reach the true top two, and recomputes those classes with a
// compensated FP32 dot product (Dot2, Ogita, Rump and Oishi 2005) kept as an
// unevaluated pair hi + lo, accurate to 2 gamma_{d+40}^2 (||W_c|| ||z|| +
// |b_c|). The true top-1 and runner-up are always among them, so m is the
// margin of the full logit vector to ~1e-10 relative of the logit scale.
// FP64 runs at a small fraction of the FP32 rate on this GPU, so only the
// per-row margin and radius use it. For the tight radius the wide-tile kernel
// refines y^G and the classes whose FP32 bracket of (s_y - s_j) /
// ||W_y - W_j|| can reach the smallest upper bracket (they contain the
// minimiser); the other kernels refine every class in FP64 (products of FP32
// values are exact there).
//
// Besides the reported radius r, the kernel derives a certified lower bound
// r_safe of the exact radius (the refined logits' error bounds, sigma
// inflated by 1e-9, every step rounded downwards) and from it the probe's
// acceptance threshold rr <= r_safe^2 (1 - eps_rc) on the canonical FP32
// squared distance, and the screen term tau.
//
// Three kernels compute the FP32 logits. When d % 4 == 0 and the head fits
// in shared memory, persistent CTAs keep W^T resident and take 128-row chunks
// with 8 x NCG register tiles and the interval pass in registers
// (k_certify_wt, both radii); with d % 4 != 0, 64-row tiles with the logits in
// shared memory (k_certify_wres); for larger heads each CTA streams W from L2
// (k_certify). Insertion order is kept by a block-count scan and a scatter.
#include "certify_common.cuh"
#include "tc_ptx.cuh"

namespace lc {
namespace {

constexpr int kRows = 32;
constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;

// One row with one warp, conservative radius (Eq. 21): the FP32 intervals
// s~_c +- E_c select every class that can be among the true top two; those
// are recomputed with dot2_logit. The true runner-up is among them, so the
// margin is that of the full logit vector. Row: features hrow[j * hs], FP32
// logits lrow[c]; W_cj = wmat[c * wcs + j * wjs]; per-class norms / biases in
// wn32 / bias. Every lane returns the same values.
__device__ RowVals warp_row_refine(const CertArgs& a, const float* __restrict__ hrow, int hs,
                                   const float* __restrict__ lrow, const float* __restrict__ wmat, int wcs, int wjs,
                                   const float* __restrict__ wn32, const float* __restrict__ bias, int lane) {
  const int d = a.d, C = a.C;
  float knp = 0.f;
  for (int j = lane; j < d; j += 32) {
    const float x = hrow[(size_t)j * hs];
    knp = fmaf(x, x, knp);
  }
  const float kn = warp_sum_f(knp);
  const float hn = norm_upper(kn);
  float l1 = -INFINITY, l2 = -INFINITY;
  for (int c = lane; c < C; c += 32) {
    const float sv = lrow[c];
    float lo = __fsub_rd(sv, logit_err(a.g32f, wn32[c], hn, bias[c], sv));
    lo = (lo == lo) ? lo : -INFINITY;  // a NaN logit is no candidate for the top two
    l2 = fmaxf(l2, fminf(l1, lo));
    l1 = fmaxf(l1, lo);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float o1 = __shfl_xor_sync(kFull, l1, o), o2 = __shfl_xor_sync(kFull, l2, o);
    l2 = fmaxf(l2, fminf(l1, o1));
    l1 = fmaxf(l1, o1);
    l2 = fmaxf(l2, fminf(l1, o2));
    l1 = fmaxf(l1, o2);
  }
  const float L2 = l2;
  Top2 t;
  for (int cb = 0; cb < C; cb += 32) {
    const int c = cb + lane;
    bool cand = false;
    if (c < C) {
      const float sv = lrow[c];
      cand = __fadd_ru(sv, logit_err(a.g32f, wn32[c], hn, bias[c], sv)) >= L2;
    }
    unsigned m = __ballot_sync(kFull, cand);
    while (m) {
      const int cc = cb + __ffs(m) - 1;
      m &= m - 1;
      const float bc = bias[cc];
      float vh, vl;
      dot2_logit(wmat + (size_t)cc * wcs, wjs, hrow, hs, bc, d, lane, vh, vl);
      t.push(cc, vh, vl, refined_err(a.g2f32, wn32[cc], hn, bc));
    }
  }
  return t.result(kn);
}

// Rows r = warp, warp + nwarps, ... < nrows of a tile, one warp each; the
// FP64 finals of up to 32 rows run once, one lane per row (FP64 runs at a
// small fraction of the FP32 rate on this GPU).
// Row r: features hb[r * hrs + j * hs], logits lg[r * lstride + c].
__device__ void certify_rows_fast(const CertArgs& a, int64_t row0, int nrows, int warp, int nwarps,
                                  const float* __restrict__ hb, int hrs, int hs, const float* __restrict__ wmat,
                                  int wcs, int wjs, const float* __restrict__ lg, const float* __restrict__ wn32,
                                  const float* __restrict__ bias, int lane, uint8_t* acc_flag) {
  RowVals mine{};
  int k = 0;
  for (int r = warp; r < nrows; r += nwarps, ++k) {
    const RowVals v = warp_row_refine(a, hb + (size_t)r * hrs, hs, lg + (size_t)r * a.lstride, wmat, wcs, wjs,
                                      wn32, bias, lane);
    if (lane == k) mine = v;
  }
  if (lane < k) {
    const int r = warp + lane * nwarps;
    row_finals(a, row0 + r, mine, &acc_flag[r]);
  }
  __syncwarp();
}

// Certify one row with one warp: FP32 interval of every logit, FP64
// refinement of the classes that can be among the true top two (all classes
// for the tight radius), margin, radius, certified lower bound, thresholds
// for the probe, and the skip rules of Algorithm 1. hrow: the row's d
// features in global memory; lrow: its FP32 logits (shared memory); ws / we:
// this warp's C-entry scratch for refined logits and their error bounds.
__device__ void certify_row(const CertArgs& a, int64_t row, const float* __restrict__ hrow,
                            const float* __restrict__ lrow, double* ws, double* we, int lane, uint8_t* acc_slot) {
  const int d = a.d, C = a.C;
    float knp = 0.f;
    double hnp = 0.0;
    for (int j = lane; j < d; j += 32) {
      const float x = __ldg(hrow + j);
      knp = fmaf(x, x, knp);
      hnp = fma((double)x, (double)x, hnp);
    }
    const float kn = warp_sum_f(knp);
    const double hn = sqrt(warp_sum_d(hnp)) * (1.0 + 1e-15);

    // second largest lower bound of the FP32 logit intervals
    double l1 = -INFINITY, l2 = -INFINITY;
    for (int c = lane; c < C; c += 32) {
      const double E = a.g32 * (a.Wnorm[c] * hn + fabs((double)a.b[c]));
      top2_push(l1, l2, (double)lrow[c] - E);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const double o1 = __shfl_xor_sync(kFull, l1, o), o2 = __shfl_xor_sync(kFull, l2, o);
      double t1 = l1, t2 = l2;
      top2_push(t1, t2, o1);
      top2_push(t1, t2, o2);
      l1 = t1;
      l2 = t2;
    }
    const double L2 = l2;

    // FP64 refinement of every class that can be among the true top two
    // (every class for the tight radius). Classes are visited in ascending
    // order, so strict comparisons keep the lowest class on ties.
    double b1 = -INFINITY, b2 = -INFINITY;
    int y = -1;
    for (int cb = 0; cb < C; cb += 32) {
      const int c = cb + lane;
      bool cand = false;
      if (c < C) {
        const double E = a.g32 * (a.Wnorm[c] * hn + fabs((double)a.b[c]));
        cand = a.tight || ((double)lrow[c] + E >= L2) || !(L2 == L2);
        if (!cand) {
          ws[c] = NAN;
          we[c] = NAN;
        }
      }
      unsigned m = __ballot_sync(kFull, cand);
      while (m) {
        const int cc = cb + __ffs(m) - 1;
        m &= m - 1;
        const float* wc = a.W + (size_t)cc * d;
        double p = 0.0, pa = 0.0;
        for (int j = lane; j < d; j += 32) {
          const double t = (double)__ldg(wc + j) * (double)__ldg(hrow + j);
          p += t;
          pa += fabs(t);
        }
        p = warp_sum_d(p);
        pa = warp_sum_d(pa);
        const double bc = (double)__ldg(a.b + cc);
        const double sv = p + bc;
        const double ev = a.g64 * (pa + fabs(bc));
        if (lane == 0) {
          ws[cc] = sv;
          we[cc] = ev;
        }
        if (sv > b1) {
          b2 = b1;
          b1 = sv;
          y = cc;
        } else if (sv > b2) {
          b2 = sv;
        }
      }
    }
    __syncwarp();
    if (y < 0) y = 0;  // every refined logit was NaN: m is NaN and the row is rejected
    const double sy = ws[y], ey = we[y];

    double r64, rs;
    if (!a.tight) {
      double up_other = -INFINITY;
      for (int c = lane; c < C; c += 32)
        if (c != y) up_other = fmax(up_other, __dadd_ru(ws[c], we[c]));
      up_other = warp_max_d(up_other);
      const double mval = (b1 == b1 && b2 == b2) ? b1 - b2 : NAN;
      const double mlo = __dsub_rd(__dsub_rd(sy, ey), up_other);
      r64 = mval * a.inv_denom;
      rs = (mlo > 0.0) ? __dmul_rd(mlo, a.inv_denom_safe) : 0.0;
      if (!(mval == mval)) r64 = NAN;
    } else {
      double rmin = INFINITY, smin = INFINITY;
      bool any_nan = !(sy == sy);
      for (int j = lane; j < C; j += 32) {
        if (j == y) continue;
        const double pn = a.pairnorm[(size_t)y * C + j];
        if (!(ws[j] == ws[j])) any_nan = true;
        if (!(pn > 0.0)) continue;
        const double ipn = a.inv_pairnorm[(size_t)y * C + j];
        rmin = fmin(rmin, (sy - ws[j]) * ipn);
        // ipn is within gamma_{d+4} / 2 of 1 / ||W_y - W_j||; tight_f removes that
        const double num = __dsub_rd(__dsub_rd(sy, ey), __dadd_ru(ws[j], we[j]));
        smin = fmin(smin, __dmul_rd(__dmul_rd(num, ipn), a.tight_f));
      }
      rmin = warp_min_d(rmin);
      smin = warp_min_d(smin);
      any_nan = __any_sync(kFull, any_nan);
      any_nan |= !(hn < INFINITY);  // a NaN or infinite feature: no defined term of Eq. 29
      r64 = any_nan ? NAN : a.kappa * rmin;
      rs = (smin > 0.0 && !any_nan) ? __dmul_rd(a.kappa, smin) : 0.0;
    }

    if (lane == 0) {
      const int32_t lab = a.payload ? a.payload[row] : y;
      const bool acc = !(a.require_consistency && lab != y) && (r64 > 0.0) && !(a.miss_of && a.miss_of[row] >= 0);
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
    __syncwarp();
}

__global__ void __launch_bounds__(kThreads) k_certify(CertArgs a) {
  extern __shared__ __align__(16) unsigned char smem[];
  double* s64 = reinterpret_cast<double*>(smem);        // kWarps x C refined logits
  double* e64 = s64 + (size_t)kWarps * a.C;             // kWarps x C their error bounds
  float* hs = reinterpret_cast<float*>(e64 + (size_t)kWarps * a.C);  // kRows x hstride
  float* lg = hs + (size_t)kRows * a.hstride;           // kRows x lstride FP32 logits
  __shared__ uint8_t acc_flag[kRows];

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t row0 = (int64_t)blockIdx.x * kRows;
  const int nrows = (int)(a.n - row0 < kRows ? a.n - row0 : kRows);
  const int d = a.d, C = a.C;

  for (int idx = threadIdx.x; idx < kRows * d; idx += kThreads) {
    const int r = idx / d, j = idx - r * d;
    hs[r * a.hstride + j] = (r < nrows) ? a.H[(size_t)(row0 + r) * d + j] : 0.f;
  }
  if (threadIdx.x < kRows) acc_flag[threadIdx.x] = 0;
  __syncthreads();

  // FP32 logits: lane = row, warps stride over classes (W loads are warp-uniform).
  {
    const float* hrow = hs + lane * a.hstride;
    for (int c = warp; c < C; c += kWarps) {
      const float* wc = a.W + (size_t)c * d;
      float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
      int j = 0;
      for (; j + 4 <= d; j += 4) {
        s0 = fmaf(__ldg(wc + j), hrow[j], s0);
        s1 = fmaf(__ldg(wc + j + 1), hrow[j + 1], s1);
        s2 = fmaf(__ldg(wc + j + 2), hrow[j + 2], s2);
        s3 = fmaf(__ldg(wc + j + 3), hrow[j + 3], s3);
      }
      for (; j < d; ++j) s0 = fmaf(__ldg(wc + j), hrow[j], s0);
      lg[lane * a.lstride + c] = ((s0 + s1) + (s2 + s3)) + __ldg(a.b + c);
    }
  }
  __syncthreads();

  double* ws = s64 + (size_t)warp * C;
  double* we = e64 + (size_t)warp * C;
  if (a.tight) {
    for (int r = warp; r < nrows; r += kWarps)
      certify_row(a, row0 + r, a.H + (size_t)(row0 + r) * d, lg + r * a.lstride, ws, we, lane, &acc_flag[r]);
  } else {
    certify_rows_fast(a, row0, nrows, warp, kWarps, a.H + (size_t)row0 * d, d, 1, a.W, d, 1, lg, a.Wnorm32, a.b,
                      lane, acc_flag);
  }
  __syncthreads();
  if (warp == 0) {
    const bool f = lane < nrows && acc_flag[lane];
    const unsigned m = __ballot_sync(kFull, f);
    if (lane < nrows) a.rank[row0 + lane] = __popc(m & ((1u << lane) - 1u));
    if (lane == 0) a.bcount[blockIdx.x] = __popc(m);
  }
}

// Certified insertion with the head resident in shared memory (C <= 256 and
// W^T fits): persistent CTAs, tiles of 64 rows.
//  1. The tile's features are transposed into shared memory (h^T).
//  2. FP32 logits by a register-tiled product: each thread accumulates 8 rows
//     x 8 classes, reading 8 features and 8 weights per k with four 128-bit
//     shared loads, one FMA chain per (row, class) in k order (the error
//     bound E_c holds for it).
//  3. Conservative radius: thread (r, q) owns row r and a quarter q of the
//     classes. It forms a quarter of ||z||^2, then the top two interval lower
//     ends of its classes; the row's second-largest lower end L2 decides the
//     candidates (upper end >= L2), which go to a per-row slot list and a
//     compact pair list. Groups of 8 lanes refine one (row, class) pair each
//     with the compensated dot product, and one thread per row selects y^G,
//     the runner-up and the bounds from its slots (in any order, ties to the
//     lowest class) and runs the FP64 finals. A row with more than
//     kMaxCand candidates is redone by one warp with warp_row_refine.
//     The tight radius runs certify_row (FP64) with one warp per row.
constexpr int kWTile = 64;    // rows per tile
constexpr int kHStride = 68;  // h^T row stride (floats): 16-byte aligned, banks spread
constexpr int kMaxCand = 16;  // candidate slots per row
constexpr int kGroup = 8;     // lanes per refined pair

struct TileSmem {
  float knp[4][kWTile];     // quarter sums of ||z||^2
  float2 top[4][kWTile];    // per-quarter top two interval lower ends
  float hn[kWTile];         // upper bound of ||z||
  float kn[kWTile];         // ||z||^2 (FP32)
  int ncand[kWTile];        // candidates per row
  int cls[kWTile][kMaxCand];
  float rh[kWTile][kMaxCand], rl[kWTile][kMaxCand], re[kWTile][kMaxCand];
  int pairs[kWTile * kMaxCand];  // r | slot << 8 | class << 16
  int npairs, novf;
  int ovf[kWTile];
  uint8_t acc_flag[kWTile];
};

// Transposed copy of rows [row0, row0 + nrows) of H (zero past d and nrows)
// into hT[k * kHStride + r]. With 16-byte rows each lane loads float4s of
// its own row and stores four conflict-free scalars (lanes = rows).
__device__ __forceinline__ void load_tile(const CertArgs& a, int64_t row0, int nrows, int dpad, float* hT, int tid,
                                          bool vec) {
  const int d = a.d;
  if (vec) {
    const int warp = tid >> 5, lane = tid & 31;
    const int r = (warp & 1) * 32 + lane;
    const bool live = r < nrows;
    const float4* src = reinterpret_cast<const float4*>(a.H + (size_t)(row0 + (live ? r : 0)) * d);
    constexpr int kB = 8;
    for (int k40 = warp >> 1; k40 < dpad / 4; k40 += 4 * kB) {
      float4 v[kB];
#pragma unroll
      for (int u = 0; u < kB; ++u) {
        const int k4 = k40 + 4 * u;
        v[u] = (live && 4 * k4 < d) ? __ldg(src + k4) : make_float4(0.f, 0.f, 0.f, 0.f);
      }
#pragma unroll
      for (int u = 0; u < kB; ++u) {
        const int k4 = k40 + 4 * u;
        if (k4 < dpad / 4) {
          float* dst = hT + (size_t)(4 * k4) * kHStride + r;
          dst[0] = v[u].x;
          dst[kHStride] = v[u].y;
          dst[2 * kHStride] = v[u].z;
          dst[3 * kHStride] = v[u].w;
        }
      }
    }
  } else {
    for (int idx = tid; idx < kWTile * dpad; idx += kThreads) {
      const int r = idx / dpad, k = idx - r * dpad;
      hT[k * kHStride + r] = (r < nrows && k < d) ? __ldg(a.H + (size_t)(row0 + r) * d + k) : 0.f;
    }
  }
}

__global__ void __launch_bounds__(kThreads, 1) k_certify_wres(CertArgs a, int Cp, int dpad, int n_tiles, int vec) {
  extern __shared__ __align__(16) unsigned char smem[];
  float* wT = reinterpret_cast<float*>(smem);           // dpad x Cp (W transposed, zero padded)
  float* hT = wT + (size_t)dpad * Cp;                   // dpad x kHStride (tile rows transposed)
  float* lg = hT + (size_t)dpad * kHStride;             // kWTile x lstride FP32 logits
  float* wn_s = lg + (size_t)kWTile * a.lstride;        // C norms (rounded up)
  float* b_s = wn_s + a.C;                              // C biases
  float* eA = b_s + a.C;                                // C: g32f ||W_c||, rounded up
  float* eB = eA + a.C;                                 // C: g32f |b_c| + tiny, rounded up
  // FP64 scratch for the tight radius only
  const int sC = a.tight ? a.C : 0;
  double* s64 = reinterpret_cast<double*>(eB + a.C + ((4 * a.C + kWTile * a.lstride) & 1));
  double* e64 = s64 + (size_t)kWarps * sC;
  TileSmem& ts = *reinterpret_cast<TileSmem*>(e64 + (size_t)kWarps * sC);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int d = a.d, C = a.C;
  for (int idx = tid; idx < dpad * Cp; idx += kThreads) {
    const int k = idx / Cp, c = idx - k * Cp;
    wT[idx] = (c < C && k < d) ? __ldg(a.W + (size_t)c * d + k) : 0.f;
  }
  for (int c = tid; c < C; c += kThreads) {
    const float wn = __ldg(a.Wnorm32 + c), bc = __ldg(a.b + c);
    wn_s[c] = wn;
    b_s[c] = bc;
    eA[c] = __fmul_ru(a.g32f, wn);
    eB[c] = __fmaf_ru(a.g32f, fabsf(bc), kTinyF);
  }
  const int rg = tid & 7, cg = tid >> 3;  // rows {4rg..4rg+3, 32+4rg..32+4rg+3}, classes 8cg..8cg+7
  const bool mine = cg * 8 < Cp;
  double* ws = s64 + (size_t)warp * sC;
  double* we = e64 + (size_t)warp * sC;
  const int r3 = tid & (kWTile - 1), q3 = tid >> 6;  // phase 3: row, class quarter
  const int cq = (C + 3) / 4, c_lo = q3 * cq, c_hi = min(C, c_lo + cq);
  const int dq = (d + 3) / 4, k_lo = q3 * dq, k_hi = min(d, k_lo + dq);

  for (int tile = blockIdx.x; tile < n_tiles; tile += gridDim.x) {
    const int64_t row0 = (int64_t)tile * kWTile;
    const int nrows = (int)(a.n - row0 < kWTile ? a.n - row0 : kWTile);
    __syncthreads();  // previous tile done with hT / lg / ts (and wT written on the first pass)
    load_tile(a, row0, nrows, dpad, hT, tid, vec != 0);
    // the next tile's rows (contiguous) start moving into L2 now, so its load
    // phase reads L2 instead of waiting on DRAM
    if (vec && tid == 0 && tile + (int)gridDim.x < n_tiles) {
      const int64_t r1 = (int64_t)(tile + gridDim.x) * kWTile;
      const int64_t n1 = a.n - r1 < kWTile ? a.n - r1 : kWTile;
      prefetch_l2_bulk(a.H + (size_t)r1 * d, (uint32_t)(n1 * d * sizeof(float)));
    }
    if (tid < kWTile) {
      ts.acc_flag[tid] = 0;
      ts.ncand[tid] = 0;
    }
    if (tid == 0) {
      ts.npairs = 0;
      ts.novf = 0;
    }
    __syncthreads();
    if (mine) {
      // accumulators in pairs of classes (2j, 2j+1): one packed FP32x2 FMA
      // (each half an IEEE fma, round to nearest) per row and class pair
      uint64_t acc[8][4];
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = 0ull;
      const float* hp = hT + rg * 4;
      const float* wp = wT + cg * 8;
#pragma unroll 4
      for (int k = 0; k < dpad; ++k) {
        const float4 h0 = *reinterpret_cast<const float4*>(hp + k * kHStride);
        const float4 h1 = *reinterpret_cast<const float4*>(hp + k * kHStride + 32);
        const ulonglong2 w0 = *reinterpret_cast<const ulonglong2*>(wp + (size_t)k * Cp);
        const ulonglong2 w1 = *reinterpret_cast<const ulonglong2*>(wp + (size_t)k * Cp + 4);
        const float hv[8] = {h0.x, h0.y, h0.z, h0.w, h1.x, h1.y, h1.z, h1.w};
        const uint64_t wv[4] = {w0.x, w0.y, w1.x, w1.y};
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const uint32_t hb = __float_as_uint(hv[i]);
          const uint64_t hh = ptx::pack_f32x2(hb, hb);
#pragma unroll
          for (int j = 0; j < 4; ++j) acc[i][j] = ptx::fma_f32x2(wv[j], hh, acc[i][j]);
        }
      }
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int r = (i < 4) ? rg * 4 + i : 32 + rg * 4 + (i - 4);
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const int c = cg * 8 + j;
          const float v = __uint_as_float((uint32_t)(acc[i][j >> 1] >> (32 * (j & 1))));
          if (c < C) lg[r * a.lstride + c] = v + b_s[c];
        }
      }
    }
    if (a.tight) {
      __syncthreads();
      for (int r = warp; r < nrows; r += kWarps)
        certify_row(a, row0 + r, a.H + (size_t)(row0 + r) * d, lg + r * a.lstride, ws, we, lane, &ts.acc_flag[r]);
    } else {
      // quarter of ||z||^2 (independent of the logits)
      {
        float p = 0.f;
        for (int k = k_lo; k < k_hi; ++k) {
          const float x = hT[k * kHStride + r3];
          p = fmaf(x, x, p);
        }
        ts.knp[q3][r3] = p;
      }
      __syncthreads();
      const float kn = (ts.knp[0][r3] + ts.knp[1][r3]) + (ts.knp[2][r3] + ts.knp[3][r3]);
      const float hn = norm_upper(kn);
      if (q3 == 0) {
        ts.kn[r3] = kn;
        ts.hn[r3] = hn;
      }
      const float* lrow = lg + (size_t)r3 * a.lstride;
      float l1 = -INFINITY, l2 = -INFINITY;
      for (int c = c_lo; c < c_hi; ++c) {
        const float sv = lrow[c];
        const float E = __fmaf_ru(eA[c], hn, __fmaf_ru(fabsf(sv), 2.3841858e-07f /* 2^-22 */, eB[c]));
        float lo = __fsub_rd(sv, E);
        lo = (lo == lo) ? lo : -INFINITY;
        l2 = fmaxf(l2, fminf(l1, lo));
        l1 = fmaxf(l1, lo);
      }
      ts.top[q3][r3] = make_float2(l1, l2);
      __syncthreads();
      float L1 = -INFINITY, L2 = -INFINITY;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float2 t = ts.top[q][r3];
        L2 = fmaxf(L2, fminf(L1, t.x));
        L1 = fmaxf(L1, t.x);
        L2 = fmaxf(L2, fminf(L1, t.y));
        L1 = fmaxf(L1, t.y);
      }
      if (r3 < nrows) {
        // candidate mask first (a loop without side effects pipelines its
        // loads), then the slots; a quarter holds at most 64 classes
        unsigned long long cm = 0;
        for (int c = c_lo; c < c_hi; ++c) {
          const float sv = lrow[c];
          const float E = __fmaf_ru(eA[c], hn, __fmaf_ru(fabsf(sv), 2.3841858e-07f, eB[c]));
          cm |= (unsigned long long)(__fadd_ru(sv, E) >= L2) << (c - c_lo);
        }
        while (cm) {
          const int c = c_lo + __ffsll((long long)cm) - 1;
          cm &= cm - 1;
          const int slot = atomicAdd(&ts.ncand[r3], 1);
          if (slot < kMaxCand) {
            ts.cls[r3][slot] = c;
            ts.pairs[atomicAdd(&ts.npairs, 1)] = r3 | (slot << 8) | (c << 16);
          }
        }
      }
      __syncthreads();
      // refine the pairs, kGroup lanes each
      {
        const int g = tid / kGroup, sub = tid % kGroup;
        const int np = ts.npairs;
        for (int base = 0; base < np; base += kThreads / kGroup) {
          const int pi = base + g;
          const int pk = ts.pairs[pi < np ? pi : 0];
          const int r = pk & 0xff, slot = (pk >> 8) & 0xff, c = pk >> 16;
          float p = 0.f, cc = 0.f;
          for (int k = sub; k < d; k += kGroup) {
            const float w = wT[(size_t)k * Cp + c], x = hT[k * kHStride + r];
            const float pr = __fmul_rn(w, x);
            const float er = __fmaf_rn(w, x, -pr);
            float t, q;
            two_sum(p, pr, t, q);
            p = t;
            cc = __fadd_rn(cc, __fadd_rn(q, er));
          }
#pragma unroll
          for (int o = kGroup / 2; o > 0; o >>= 1) {
            const float pb = __shfl_xor_sync(kFull, p, o), cb = __shfl_xor_sync(kFull, cc, o);
            float t, q;
            two_sum(p, pb, t, q);
            p = t;
            cc = __fadd_rn(__fadd_rn(cc, cb), q);
          }
          if (pi < np && sub == 0) {
            float t, q, hi, lo;
            two_sum(p, b_s[c], t, q);
            two_sum(t, __fadd_rn(cc, q), hi, lo);
            ts.rh[r][slot] = hi;
            ts.rl[r][slot] = lo;
            ts.re[r][slot] = refined_err(a.g2f8, wn_s[c], ts.hn[r], b_s[c]);
          }
        }
      }
      __syncthreads();
      if (tid < nrows) {
        const int r = tid, n = ts.ncand[r];
        if (n > kMaxCand) {
          ts.ovf[atomicAdd(&ts.novf, 1)] = r;
        } else {
          Top2 t;
          for (int sl = 0; sl < n; ++sl) t.push(ts.cls[r][sl], ts.rh[r][sl], ts.rl[r][sl], ts.re[r][sl]);
          row_finals(a, row0 + r, t.result(ts.kn[r]), &ts.acc_flag[r]);
        }
      }
      __syncthreads();
      for (int i = warp; i < ts.novf; i += kWarps) {
        const int r = ts.ovf[i];
        const RowVals v = warp_row_refine(a, hT + r, kHStride, lg + (size_t)r * a.lstride, wT, 1, Cp, wn_s, b_s, lane);
        if (lane == 0) row_finals(a, row0 + r, v, &ts.acc_flag[r]);
      }
    }
    __syncthreads();
    if (warp < 2 && row0 + warp * 32 < a.n) {
      const int sub = warp * 32;
      const int nsub = nrows - sub < 32 ? nrows - sub : 32;
      const bool f = lane < nsub && ts.acc_flag[sub + lane];
      const unsigned m = __ballot_sync(kFull, f);
      if (lane < nsub) a.rank[row0 + sub + lane] = __popc(m & ((1u << lane) - 1u));
      if (lane == 0) a.bcount[(row0 + sub) / 32] = __popc(m);
    }
  }
}

// ---------------------------------------------------------------- k_certify_wt
// Certified insertion, conservative radius, head resident in shared memory,
// tiles of 128 rows (persistent CTAs of 8 warps; C <= 256, d % 4 == 0):
//  1. Load: warp w takes feature quarter w % 4 of rows 64 (w / 4) .. + 63,
//     lane = row; the rows are transposed into shared memory (h^T) and the
//     quarter sums of ||z||^2 are formed on the way, in feature order.
//  2. FP32 logits: each thread keeps a register tile of 8 rows x NCG classes
//     (16 row groups x 16 class groups; packed FP32x2 FMAs on class pairs, one
//     FMA chain per (row, class) in k order). Per feature it reads 8 + NCG
//     shared floats for 8 NCG FMAs, so at NCG = 13 the FP32 pipe (every
//     sub-partition equally loaded), not shared memory, bounds the product.
//  3. From the registers: interval lower ends, each row's second-largest
//     lower end L2 (butterfly over the 16 lanes that share the rows), and the
//     candidate classes (upper end >= L2) into per-row slots and a pair list.
//  4. Pair refinement (8 lanes a pair, compensated dot product), per-row
//     selection and FP64 finals, rows with more than kMaxCand candidates by
//     warp_row_refine, 32-row ranks and counts.
// Logits, candidate sets, refined pairs and finals are the values
// k_certify_wres computes, bit for bit. W^T holds class g NCG + j at column
// g GS + j (GS even, GS = 2 mod 4), so the 16 class groups' 64-bit weight
// loads fall on distinct banks.
constexpr int kWtRows = 128;        // rows per tile
constexpr int kWtHst = kWtRows + 4;  // h^T row stride (floats): 16-byte aligned, banks spread

struct WtTile {
  float knp[4][kWtRows];  // quarter sums of ||z||^2
  float hn[kWtRows];      // upper bound of ||z||
  int ncand[kWtRows];
  int yq[kWtRows];        // tight radius: y^G of the row, known from the FP32 intervals
  uint8_t cls[kWtRows][kMaxCand];
  float rh[kWtRows][kMaxCand], rl[kWtRows][kMaxCand], re[kWtRows][kMaxCand];
  int pairs[kWtRows * kMaxCand];  // r | slot << 8 | class << 16; after the refinement, per-warp logit rows
  int ovf[kWtRows];
  int npairs, novf, pad[2];
  uint8_t acc_flag[kWtRows];
};

struct WtLayout {
  int NCG, GS, wst;
  uint32_t off_h, off_e, off_tile, total;
};

// E_c of an FP32 logit s~_c, rounded up, from the per-column terms
// eA = g32f ||W_c|| and eB = g32f |b_c| + tiny (both rounded up) and the
// bound hn of ||z||: gamma_{d+2} (||W_c|| ||z|| + |b_c|) + 2^-22 |s~_c| + tiny.
__device__ __forceinline__ float logit_bound(float eA, float eB, float hn, float sv) {
  return __fmaf_ru(eA, hn, __fmaf_ru(fabsf(sv), 2.3841858e-07f /* 2^-22 */, eB));
}

// Tight radius (Eq. 29) candidates of one row from the FP32 logit intervals
// of this lane's classes (the 16 lanes of a half-warp hold the row). y^G is
// certain when exactly one class's upper end reaches the largest lower end l1
// (then every other interval lies below y's). For each other class j, u_j and
// l_j bracket (s_y - s_j) / ||W_y - W_j|| (outward rounding, FP32 brackets of
// the reciprocal norm); with U = min_j u_j, the minimiser of Eq. 29 is among
// {j : l_j <= U}, since its l_j <= r* <= U. Returns this lane's candidate bits
// (y and those classes) for refinement; `fallback` marks rows the intervals
// cannot settle (several possible y^G, or a NaN logit), `y` the certain y^G.
template <int NCG>
__device__ __forceinline__ unsigned tight_candidates(const CertArgs& a, const float (&sv)[NCG], const float* eA,
                                                     const float* eB, float hn, float l1, int cg, int lane,
                                                     bool live_row, int& y, bool& fallback) {
  const int C = a.C;
  const unsigned half = 0xffffu << (lane & 16);
  unsigned t1 = 0;
  bool nan_l = false;
  int myjc = -1;
  float mlo = 0.f, mhi = 0.f;
#pragma unroll
  for (int jc = 0; jc < NCG; ++jc) {
    const bool live = cg * NCG + jc < C;
    const float E = logit_bound(eA[jc], eB[jc], hn, sv[jc]);
    const float hi = __fadd_ru(sv[jc], E), lo = __fsub_rd(sv[jc], E);
    nan_l |= live && !(sv[jc] == sv[jc]);
    const bool top = live && hi >= l1;
    const bool first = top && myjc < 0;
    myjc = first ? jc : myjc;
    mlo = first ? lo : mlo;
    mhi = first ? hi : mhi;
    t1 |= (unsigned)top << jc;
  }
  int cnt = __popc(t1);
#pragma unroll
  for (int o = 1; o < 16; o <<= 1) cnt += __shfl_xor_sync(kFull, cnt, o);
  const unsigned nanb = __ballot_sync(kFull, nan_l) & half;
  const unsigned hasb = __ballot_sync(kFull, t1 != 0u) & half;
  const int src = hasb ? __ffs((int)hasb) - 1 : lane;
  const int jy = __shfl_sync(kFull, myjc, src);
  const float loy = __shfl_sync(kFull, mlo, src), hiy = __shfl_sync(kFull, mhi, src);
  // (a row whose norm bound is not finite, from an infinite feature or an
  // overflowing |z|^2, goes to the one-warp path, which settles both)
  const bool certain = live_row && cnt == 1 && nanb == 0u && hn < INFINITY;
  const int yc = (src & 15) * NCG + jy;
  float ub = INFINITY;
#pragma unroll
  for (int jc = 0; jc < NCG; ++jc) {
    const int j = cg * NCG + jc;
    const bool live = certain && j < C && j != yc;
    const float iu = live ? __ldg(a.ipn_up32 + (size_t)yc * C + j) : INFINITY;
    const float uj = __fmul_ru(__fsub_ru(hiy, __fsub_rd(sv[jc], logit_bound(eA[jc], eB[jc], hn, sv[jc]))), iu);
    ub = fminf(ub, live ? uj : INFINITY);
  }
#pragma unroll
  for (int o = 1; o < 16; o <<= 1) ub = fminf(ub, __shfl_xor_sync(kFull, ub, o));
  unsigned c = 0;
#pragma unroll
  for (int jc = 0; jc < NCG; ++jc) {
    const int j = cg * NCG + jc;
    const bool live = certain && j < C && j != yc;
    const float il = live ? __ldg(a.ipn_dn32 + (size_t)yc * C + j) : INFINITY;
    const float lj = __fmul_rd(__fsub_rd(loy, __fadd_ru(sv[jc], logit_bound(eA[jc], eB[jc], hn, sv[jc]))), il);
    c |= (unsigned)(certain && j < C && (j == yc || lj <= ub)) << jc;
  }
  y = certain ? yc : -1;
  fallback = live_row && !certain;
  return c;
}

// FP64 tight radius (Eq. 29) of one row from its refined candidates (y^G and
// every class that can be the minimiser), with the certified lower bound and
// the probe thresholds; the skip rules of Algorithm 1.
__device__ void row_finals_tight(const CertArgs& a, int64_t row, int y, int n, const uint8_t* cls, const float* rh,
                                 const float* rl, const float* re, float kn, uint8_t* acc_slot) {
  double vy = NAN, ey = 0.0;
  for (int sl = 0; sl < n; ++sl)
    if (cls[sl] == y) {
      vy = (double)rh[sl] + (double)rl[sl];
      ey = (double)re[sl];
    }
  double rmin = INFINITY, smin = INFINITY;
  bool any_nan = !(vy == vy);
  for (int sl = 0; sl < n; ++sl) {
    const int j = cls[sl];
    if (j == y) continue;
    const double vj = (double)rh[sl] + (double)rl[sl];
    if (!(vj == vj)) any_nan = true;
    tight_term(a, y, j, vy, ey, vj, (double)re[sl], rmin, smin);
  }
  tight_write(a, row, y, rmin, smin, any_nan, kn, acc_slot);
}

// One row of the tight radius on one warp, for rows the FP32 intervals cannot
// settle (several classes may be y^G, a NaN logit, or more candidates than
// slots): every class refined with the compensated dot product (lane = class,
// features in order; the same error bound as the 8-lane refinement), y^G the
// largest refined logit (lowest class on ties), then Eq. 29 over every other
// class in FP64, as row_finals_tight. FP64 stays out of the per-feature work,
// which runs at a small fraction of the FP32 rate on this GPU.
template <int NCG>
__device__ void wt_tight_row_warp(const CertArgs& a, int64_t row, int r, const float* __restrict__ wT, int wst,
                                  int GS, const float* __restrict__ hT, const float* __restrict__ wn_s,
                                  const float* __restrict__ b_s, float kn, int lane, uint8_t* acc_slot) {
  constexpr int kPer = 8;  // classes per lane (C <= 256)
  const int d = a.d, C = a.C;
  const float hn = norm_upper(kn);
  float vh[kPer], vl[kPer], ve[kPer];
  float bh = -INFINITY, bl = 0.f;
  int by = -1;
  bool nan_any = false;
#pragma unroll
  for (int t = 0; t < kPer; ++t) {
    const int c = lane + 32 * t;
    vh[t] = NAN;
    vl[t] = 0.f;
    ve[t] = 0.f;
    if (c < C) {
      const int col = (c / NCG) * GS + (c % NCG);
      float p = 0.f, cc = 0.f;
      for (int k = 0; k < d; ++k) {
        const float w = wT[(size_t)k * wst + col], x = hT[(size_t)k * kWtHst + r];
        const float pr = __fmul_rn(w, x);
        const float er = __fmaf_rn(w, x, -pr);
        float s1, q;
        two_sum(p, pr, s1, q);
        p = s1;
        cc = __fadd_rn(cc, __fadd_rn(q, er));
      }
      float s1, q, hi, lo;
      two_sum(p, b_s[c], s1, q);
      two_sum(s1, __fadd_rn(cc, q), hi, lo);
      vh[t] = hi;
      vl[t] = lo;
      ve[t] = refined_err(a.g2f, wn_s[c], hn, b_s[c]);
      nan_any |= !(hi == hi && lo == lo);
      if (pair_gt(hi, lo, bh, bl)) {  // ascending classes: ties keep the lowest
        bh = hi;
        bl = lo;
        by = c;
      }
    }
  }
  // warp argmax, ties to the lowest class (a total order on non-NaN pairs)
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float oh = __shfl_xor_sync(kFull, bh, o), ol = __shfl_xor_sync(kFull, bl, o);
    const int oy = __shfl_xor_sync(kFull, by, o);
    const bool eq = oh == bh && ol == bl;
    if (oy >= 0 && (by < 0 || pair_gt(oh, ol, bh, bl) || (eq && oy < by))) {
      bh = oh;
      bl = ol;
      by = oy;
    }
  }
  nan_any = __any_sync(kFull, nan_any);
  const int y = by < 0 ? 0 : by;
  float myh = 0.f, myl = 0.f, mye = 0.f;
#pragma unroll
  for (int t = 0; t < kPer; ++t)
    if (lane + 32 * t == y) {
      myh = vh[t];
      myl = vl[t];
      mye = ve[t];
    }
  const int owner = y & 31;
  const double vy = (double)__shfl_sync(kFull, myh, owner) + (double)__shfl_sync(kFull, myl, owner);
  const double ey = (double)__shfl_sync(kFull, mye, owner);
  double rmin = INFINITY, smin = INFINITY;
#pragma unroll
  for (int t = 0; t < kPer; ++t) {
    const int j = lane + 32 * t;
    if (j >= C || j == y) continue;
    tight_term(a, y, j, vy, ey, (double)vh[t] + (double)vl[t], (double)ve[t], rmin, smin);
  }
  rmin = warp_min_d(rmin);
  smin = warp_min_d(smin);
  if (lane == 0) tight_write(a, row, y, rmin, smin, nan_any, kn, acc_slot);
  __syncwarp();
}

// Steps 2-3 of k_certify_wt for one chunk, with ROWS rows per thread (8 for
// chunks of more than 64 rows, 4 otherwise, so that a short chunk still keeps
// two warps on every sub-partition): the FP32 logits, the interval pass, the
// candidate slots and this warp's share of the pair list.
template <int NCG, int ROWS>
__device__ __forceinline__ void wt_chunk_logits(const CertArgs& a, const float* __restrict__ wT,
                                                const float* __restrict__ hT, const float* __restrict__ eA,
                                                const float* __restrict__ eB, const float* __restrict__ bp, WtTile& ts,
                                                int GS, int wst, int nrows, int warp, int lane) {
  constexpr int NPR = NCG / 2;  // class pairs per thread
  constexpr bool kOdd = (NCG & 1) != 0;
  const int d = a.d, C = a.C;
  const int cg = lane & 15, rg = warp * 2 + (lane >> 4);  // rows ROWS rg .. ROWS rg + ROWS - 1, classes cg NCG ..
  const float* wp = wT + cg * GS;
  if (2 * ROWS * warp < nrows) {  // this warp's 2 ROWS rows hold at least one live row
    // 2. FP32 logits of rows ROWS rg .. ROWS rg + ROWS - 1 and classes cg NCG .. cg NCG + NCG - 1
    uint64_t accp[ROWS][NPR > 0 ? NPR : 1];
    float accs[ROWS];
#pragma unroll
    for (int i = 0; i < ROWS; ++i) {
#pragma unroll
      for (int m = 0; m < NPR; ++m) accp[i][m] = 0ull;
      accs[i] = 0.f;
    }
    {
      const float* hb = hT + ROWS * rg;
#pragma unroll 2
      for (int k = 0; k < d; ++k) {
        float hv[ROWS];
#pragma unroll
        for (int v4 = 0; v4 < ROWS / 4; ++v4) {
          const float4 x = *reinterpret_cast<const float4*>(hb + (size_t)k * kWtHst + 4 * v4);
          hv[4 * v4] = x.x;
          hv[4 * v4 + 1] = x.y;
          hv[4 * v4 + 2] = x.z;
          hv[4 * v4 + 3] = x.w;
        }
        const float* wk = wp + (size_t)k * wst;
        uint64_t wv[NPR > 0 ? NPR : 1];
#pragma unroll
        for (int m = 0; m < NPR; ++m) wv[m] = *reinterpret_cast<const uint64_t*>(wk + 2 * m);
        const float w1 = kOdd ? wk[NCG - 1] : 0.f;
#pragma unroll
        for (int i = 0; i < ROWS; ++i) {
          const uint32_t hb32 = __float_as_uint(hv[i]);
          const uint64_t hh = ptx::pack_f32x2(hb32, hb32);
#pragma unroll
          for (int m = 0; m < NPR; ++m) accp[i][m] = ptx::fma_f32x2(wv[m], hh, accp[i][m]);
          if (kOdd) accs[i] = __fmaf_rn(w1, hv[i], accs[i]);
        }
      }
    }
    // 3. interval lower ends, each row's L2, candidates, two rows at a time.
    // The loop stays rolled (its body runs once per chunk and would not stay
    // in the instruction cache unrolled); rows i, i + 1 are always in
    // accp[0..1], the rest shift down. Branch-free over the classes (a
    // divergent branch per class would serialise them): dead classes get
    // -inf lower ends and no candidacy.
#pragma unroll 1
    for (int i = 0; i < ROWS; i += 2) {
      float sv[2][NCG], l1[2], l2[2], hn[2];
      int r[2];
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        r[u] = ROWS * rg + i + u;
        const float kn = (ts.knp[0][r[u]] + ts.knp[1][r[u]]) + (ts.knp[2][r[u]] + ts.knp[3][r[u]]);
        hn[u] = norm_upper(kn);
#pragma unroll
        for (int m = 0; m < NPR; ++m) {
          sv[u][2 * m] = __fadd_rn(__uint_as_float((uint32_t)accp[u][m]), bp[cg * GS + 2 * m]);
          sv[u][2 * m + 1] = __fadd_rn(__uint_as_float((uint32_t)(accp[u][m] >> 32)), bp[cg * GS + 2 * m + 1]);
        }
        if (kOdd) sv[u][NCG - 1] = __fadd_rn(accs[u], bp[cg * GS + NCG - 1]);
      }
#pragma unroll
      for (int ii = 0; ii < ROWS - 2; ++ii) {
#pragma unroll
        for (int m = 0; m < NPR; ++m) accp[ii][m] = accp[ii + 2][m];
        accs[ii] = accs[ii + 2];
      }
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        l1[u] = -INFINITY;
        l2[u] = -INFINITY;
#pragma unroll
        for (int jc = 0; jc < NCG; ++jc) {
          const float E = logit_bound(eA[cg * GS + jc], eB[cg * GS + jc], hn[u], sv[u][jc]);
          float lo = __fsub_rd(sv[u][jc], E);
          lo = (lo == lo && cg * NCG + jc < C) ? lo : -INFINITY;
          l2[u] = fmaxf(l2[u], fminf(l1[u], lo));
          l1[u] = fmaxf(l1[u], lo);
        }
      }
#pragma unroll
      for (int o = 1; o < 16; o <<= 1) {
#pragma unroll
        for (int u = 0; u < 2; ++u) {
          const float o1 = __shfl_xor_sync(kFull, l1[u], o), o2 = __shfl_xor_sync(kFull, l2[u], o);
          l2[u] = fmaxf(l2[u], fminf(l1[u], o1));
          l1[u] = fmaxf(l1[u], o1);
          l2[u] = fmaxf(l2[u], fminf(l1[u], o2));
          l1[u] = fmaxf(l1[u], o2);
        }
      }
      unsigned cm[2];  // candidate bits of this lane's classes
      int incl[2], mine[2], yv[2];
      bool fallback[2];
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        cm[u] = 0;
        yv[u] = -1;
        fallback[u] = false;
        if (!a.tight) {
#pragma unroll
          for (int jc = 0; jc < NCG; ++jc)
            cm[u] |= (unsigned)(cg * NCG + jc < C &&
                                __fadd_ru(sv[u][jc], logit_bound(eA[cg * GS + jc], eB[cg * GS + jc], hn[u], sv[u][jc])) >=
                                    l2[u])
                     << jc;
        } else {
          cm[u] = tight_candidates<NCG>(a, sv[u], eA + cg * GS, eB + cg * GS, hn[u], l1[u], cg, lane, r[u] < nrows,
                                        yv[u], fallback[u]);
        }
        cm[u] = r[u] < nrows ? cm[u] : 0u;
        mine[u] = __popc(cm[u]);
        incl[u] = mine[u];
      }
      // slots of each row: the 16 lanes of this half-warp own it; prefix
      // sum of their candidate counts
#pragma unroll
      for (int o = 1; o < 16; o <<= 1) {
#pragma unroll
        for (int u = 0; u < 2; ++u) {
          const int t = __shfl_up_sync(kFull, incl[u], o, 16);
          if (cg >= o) incl[u] += t;
        }
      }
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        int slot = incl[u] - mine[u];
        unsigned m = cm[u];
        while (m) {
          const int jc = __ffs(m) - 1;
          m &= m - 1;
          if (slot < kMaxCand) ts.cls[r[u]][slot] = (uint8_t)(cg * NCG + jc);
          ++slot;
        }
        if (cg == 15) {
          ts.ncand[r[u]] = fallback[u] ? kMaxCand + 1 : incl[u];
          ts.hn[r[u]] = hn[u];
          ts.yq[r[u]] = yv[u];
        }
      }
    }
  }
  // this warp's 2 ROWS rows into the pair list: one reservation per warp
  __syncwarp();
  {
    const int R = ROWS * (2 * warp + lane / ROWS) + lane % ROWS;
    const int n = lane < 2 * ROWS ? min(ts.ncand[R], kMaxCand) : 0;
    int incl = n;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int t = __shfl_up_sync(kFull, incl, o);
      if (lane >= o) incl += t;
    }
    const int total = __shfl_sync(kFull, incl, 31);
    int base = 0;
    if (lane == 0 && total) base = atomicAdd(&ts.npairs, total);
    base = __shfl_sync(kFull, base, 0) + incl - n;
    for (int sl = 0; sl < n; ++sl) ts.pairs[base + sl] = R | (sl << 8) | ((int)ts.cls[R][sl] << 16);
  }
}

template <int NCG>
__global__ void __launch_bounds__(kThreads, 1) k_certify_wt(CertArgs a, WtLayout L, const float* __restrict__ prep,
                                                             int64_t nb32) {
  extern __shared__ __align__(16) unsigned char smem[];
  const int d = a.d, C = a.C, GS = L.GS, wst = L.wst;
  float* wT = reinterpret_cast<float*>(smem);
  float* hT = reinterpret_cast<float*>(smem + L.off_h);  // d x kWtHst
  float* eA = reinterpret_cast<float*>(smem + L.off_e);  // 16 GS each, grouped columns
  float* eB = eA + 16 * GS;
  float* bp = eB + 16 * GS;
  float* wn_s = bp + 16 * GS;  // C each, by class
  float* b_s = wn_s + C;
  WtTile& ts = *reinterpret_cast<WtTile*>(smem + L.off_tile);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  {
    // the prepared head: L.off_h bytes, 128-bit loads, eight in flight
    const float4* src = reinterpret_cast<const float4*>(prep);
    float4* dst = reinterpret_cast<float4*>(smem);
    const int n4 = (int)(L.off_h / 16);
    constexpr int kB = 8;
    for (int i0 = tid; i0 < n4; i0 += kB * kThreads) {
      float4 v[kB];
#pragma unroll
      for (int u = 0; u < kB; ++u) {
        const int i = i0 + u * kThreads;
        if (i < n4) v[u] = __ldg(src + i);
      }
#pragma unroll
      for (int u = 0; u < kB; ++u) {
        const int i = i0 + u * kThreads;
        if (i < n4) dst[i] = v[u];
      }
    }
  }
  const int g8 = tid / kGroup, sub = tid % kGroup;  // refinement groups
  const int q = warp & 3, dq = (d + 3) / 4, k_lo = q * dq, k_hi = min(d, k_lo + dq);  // load quarter
  // this CTA's rows: a contiguous range of whole 32-row blocks (balanced over
  // the grid), in chunks of up to kWtRows rows
  const int64_t b_lo = (int64_t)blockIdx.x * nb32 / gridDim.x, b_hi = ((int64_t)blockIdx.x + 1) * nb32 / gridDim.x;
  const int64_t row_hi = b_hi * 32 < a.n ? b_hi * 32 : a.n;
  if (tid == 0 && b_lo * 32 < row_hi)
    prefetch_l2_bulk(a.H + (size_t)(b_lo * 32) * d,
                     (uint32_t)((row_hi - b_lo * 32 < kWtRows ? row_hi - b_lo * 32 : kWtRows) * d * sizeof(float)));

  for (int64_t row0 = b_lo * 32; row0 < row_hi; row0 += kWtRows) {
    const int nrows = (int)(row_hi - row0 < kWtRows ? row_hi - row0 : kWtRows);
    __syncthreads();  // the previous chunk is done with h^T and the lists (W^T written on the first pass)
    // the next chunk's rows start moving into L2
    if (tid == 0 && row0 + kWtRows < row_hi) {
      const int64_t r1 = row0 + kWtRows;
      const int64_t n1 = row_hi - r1 < kWtRows ? row_hi - r1 : kWtRows;
      prefetch_l2_bulk(a.H + (size_t)r1 * d, (uint32_t)(n1 * d * sizeof(float)));
    }
    // 1. load, transpose, quarter sums (32-row blocks past nrows are skipped;
    //    rows past nrows are never selected)
    for (int half = 0; half < 2; ++half) {
      const int rb = (warp >> 2) * 64 + half * 32;
      if (rb >= nrows) continue;
      const int r = rb + lane;
      const bool live = r < nrows;
      const float* src = a.H + (size_t)(row0 + (live ? r : 0)) * d;
      float p = 0.f;
      if ((dq & 3) == 0) {
        constexpr int kB = 8;
        for (int k0 = k_lo; k0 < k_hi; k0 += 4 * kB) {
          float4 v[kB];
#pragma unroll
          for (int u = 0; u < kB; ++u) {
            const int k = k0 + 4 * u;
            v[u] = (live && k < k_hi) ? __ldg(reinterpret_cast<const float4*>(src + k))
                                      : make_float4(0.f, 0.f, 0.f, 0.f);
          }
#pragma unroll
          for (int u = 0; u < kB; ++u) {
            const int k = k0 + 4 * u;
            if (k < k_hi) {
              p = fmaf(v[u].x, v[u].x, p);
              p = fmaf(v[u].y, v[u].y, p);
              p = fmaf(v[u].z, v[u].z, p);
              p = fmaf(v[u].w, v[u].w, p);
              float* dst = hT + (size_t)k * kWtHst + r;
              dst[0] = v[u].x;
              dst[kWtHst] = v[u].y;
              dst[2 * kWtHst] = v[u].z;
              dst[3 * kWtHst] = v[u].w;
            }
          }
        }
      } else {
        for (int k = k_lo; k < k_hi; ++k) {
          const float x = live ? __ldg(src + k) : 0.f;
          p = fmaf(x, x, p);
          hT[(size_t)k * kWtHst + r] = x;
        }
      }
      ts.knp[q][r] = p;
    }
    if (tid < kWtRows) {
      ts.ncand[tid] = 0;
      ts.acc_flag[tid] = 0;
    }
    if (tid == 0) {
      ts.npairs = 0;
      ts.novf = 0;
    }
    __syncthreads();
    if (nrows > 64)
      wt_chunk_logits<NCG, 8>(a, wT, hT, eA, eB, bp, ts, GS, wst, nrows, warp, lane);
    else
      wt_chunk_logits<NCG, 4>(a, wT, hT, eA, eB, bp, ts, GS, wst, nrows, warp, lane);
    __syncthreads();
    // 4. refine the pairs, kGroup lanes a pair, two pairs a group at a time
    constexpr int kGroups = kThreads / kGroup;
    const int np = ts.npairs;
    for (int base = 0; base < np; base += 2 * kGroups) {
      int pi[2], r[2], slot[2], c[2], col[2];
      float p[2] = {0.f, 0.f}, cc[2] = {0.f, 0.f};
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        pi[u] = base + u * kGroups + g8;
        const int pk = ts.pairs[pi[u] < np ? pi[u] : 0];
        r[u] = pk & 0xff;
        slot[u] = (pk >> 8) & 0xff;
        c[u] = pk >> 16;
        col[u] = (c[u] / NCG) * GS + (c[u] % NCG);
      }
      for (int k = sub; k < d; k += kGroup) {
#pragma unroll
        for (int u = 0; u < 2; ++u) {
          const float w = wT[(size_t)k * wst + col[u]], x = hT[(size_t)k * kWtHst + r[u]];
          const float pr = __fmul_rn(w, x);
          const float er = __fmaf_rn(w, x, -pr);
          float t, qq;
          two_sum(p[u], pr, t, qq);
          p[u] = t;
          cc[u] = __fadd_rn(cc[u], __fadd_rn(qq, er));
        }
      }
#pragma unroll
      for (int o = kGroup / 2; o > 0; o >>= 1) {
#pragma unroll
        for (int u = 0; u < 2; ++u) {
          const float pb = __shfl_xor_sync(kFull, p[u], o), cb = __shfl_xor_sync(kFull, cc[u], o);
          float t, qq;
          two_sum(p[u], pb, t, qq);
          p[u] = t;
          cc[u] = __fadd_rn(__fadd_rn(cc[u], cb), qq);
        }
      }
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        if (pi[u] < np && sub == 0) {
          float t, qq, hi, lo;
          two_sum(p[u], b_s[c[u]], t, qq);
          two_sum(t, __fadd_rn(cc[u], qq), hi, lo);
          ts.rh[r[u]][slot[u]] = hi;
          ts.rl[r[u]][slot[u]] = lo;
          ts.re[r[u]][slot[u]] = refined_err(a.g2f8, wn_s[c[u]], ts.hn[r[u]], b_s[c[u]]);
        }
      }
    }
    __syncthreads();
    if (tid < nrows) {
      const int r = tid, n = ts.ncand[r];
      if (n > kMaxCand) {
        ts.ovf[atomicAdd(&ts.novf, 1)] = r;
      } else {
        const float kn = (ts.knp[0][r] + ts.knp[1][r]) + (ts.knp[2][r] + ts.knp[3][r]);
        if (a.tight) {
          row_finals_tight(a, row0 + r, ts.yq[r], n, ts.cls[r], ts.rh[r], ts.rl[r], ts.re[r], kn, &ts.acc_flag[r]);
        } else {
          Top2 t;
          for (int sl = 0; sl < n; ++sl) t.push(ts.cls[r][sl], ts.rh[r][sl], ts.rl[r][sl], ts.re[r][sl]);
          row_finals(a, row0 + r, t.result(kn), &ts.acc_flag[r]);
        }
      }
    }
    __syncthreads();
    // rows with more than kMaxCand candidates: FP32 logits again (the same
    // FMA chains, into this warp's share of the dead pair list), then the
    // one-warp refinement
    // (tight radius: the rows the intervals could not settle, all classes
    // refined on one warp by wt_tight_row_warp)
    for (int i = warp; i < ts.novf; i += kWarps) {
      const int r = ts.ovf[i];
      if (a.tight) {
        const float kn = (ts.knp[0][r] + ts.knp[1][r]) + (ts.knp[2][r] + ts.knp[3][r]);
        wt_tight_row_warp<NCG>(a, row0 + r, r, wT, wst, GS, hT, wn_s, b_s, kn, lane, &ts.acc_flag[r]);
        continue;
      }
      float* lrow = reinterpret_cast<float*>(ts.pairs) + (size_t)warp * C;
      for (int c = lane; c < C; c += 32) {
        const int col = (c / NCG) * GS + (c % NCG);
        float v = 0.f;
        for (int k = 0; k < d; ++k) v = __fmaf_rn(wT[(size_t)k * wst + col], hT[(size_t)k * kWtHst + r], v);
        lrow[c] = __fadd_rn(v, b_s[c]);
      }
      __syncwarp();
      const RowVals v = warp_row_refine(a, hT + r, kWtHst, lrow, a.W, d, 1, a.Wnorm32, a.b, lane);
      if (lane == 0) row_finals(a, row0 + r, v, &ts.acc_flag[r]);
      __syncwarp();
    }
    __syncthreads();
    if (warp < kWtRows / 32 && warp * 32 < nrows) {
      const int s0 = warp * 32;
      const int nsub = nrows - s0 < 32 ? nrows - s0 : 32;
      const bool f = lane < nsub && ts.acc_flag[s0 + lane];
      const unsigned m = __ballot_sync(kFull, f);
      if (lane < nsub) a.rank[row0 + s0 + lane] = __popc(m & ((1u << lane) - 1u));
      if (lane == 0) a.bcount[(row0 + s0) / 32] = __popc(m);
    }
  }
}

WtLayout wt_layout(int d, int C, int NCG) {
  WtLayout L;
  L.NCG = NCG;
  L.GS = NCG + (NCG & 1);
  if (L.GS % 4 == 0) L.GS += 2;
  L.wst = ((16 * L.GS - 4 + 31) / 32) * 32 + 4;
  auto al = [](size_t x) { return (uint32_t)((x + 15) / 16 * 16); };
  L.off_e = al(sizeof(float) * (size_t)d * L.wst);
  L.off_h = al(L.off_e + sizeof(float) * (3 * 16 * (size_t)L.GS + 2 * (size_t)C));
  L.off_tile = al(L.off_h + sizeof(float) * (size_t)d * kWtHst);
  L.total = L.off_tile + (uint32_t)sizeof(WtTile);
  return L;
}

// The head in k_certify_wt's shared-memory layout (its first L.off_h bytes):
// W^T in grouped columns (class g NCG + j at column g GS + j, zero padded),
// then the per-column error terms eA = g32f ||W_c|| and eB = g32f |b_c| +
// tiny (rounded up) and biases, then ||W_c|| and b_c by class.
__global__ void k_wt_prepare(CertArgs a, WtLayout L, float* __restrict__ out) {
  const int d = a.d, C = a.C, NCG = L.NCG, GS = L.GS, wst = L.wst;
  float* eA = out + L.off_e / sizeof(float);
  float* eB = eA + 16 * GS;
  float* bp = eB + 16 * GS;
  float* wn_s = bp + 16 * GS;
  float* b_s = wn_s + C;
  const int stride = gridDim.x * blockDim.x;
  for (int idx = blockIdx.x * blockDim.x + threadIdx.x; idx < d * wst; idx += stride) {
    const int k = idx / wst, col = idx - k * wst;
    const int g = col / GS, j = col - g * GS, c = g * NCG + j;
    out[idx] = (col < 16 * GS && j < NCG && c < C) ? a.W[(size_t)c * d + k] : 0.f;
  }
  for (int col = blockIdx.x * blockDim.x + threadIdx.x; col < 16 * GS; col += stride) {
    const int g = col / GS, j = col - g * GS, c = g * NCG + j;
    const bool live = j < NCG && c < C;
    const float wn = live ? a.Wnorm32[c] : 0.f, bc = live ? a.b[c] : 0.f;
    eA[col] = __fmul_ru(a.g32f, wn);
    eB[col] = __fmaf_ru(a.g32f, fabsf(bc), kTinyF);
    bp[col] = bc;
  }
  for (int c = blockIdx.x * blockDim.x + threadIdx.x; c < C; c += stride) {
    wn_s[c] = a.Wnorm32[c];
    b_s[c] = a.b[c];
  }
}

// Smallest compiled per-thread class count covering C classes in 16 groups.
int wt_ncg(int C) {
  const int need = (C + 15) / 16;
  return need <= 1 ? 1 : need <= 4 ? 4 : need <= 7 ? 7 : need <= 13 ? 13 : need <= 16 ? 16 : 0;
}

// ---------------------------------------------------------------- FP64 pass
// The stand-alone FP64 pass (fix_row_warp) over the rows a certify kernel
// listed, for the kernels that do not run it themselves: a warp per listed
// row, kFixWarps rows per block; the head is staged once per block into
// shared memory (rows padded to d + 1 floats, so that a lane per class reads
// without bank conflicts) when it fits, else read from global memory.
constexpr int kFixWarps = 8;

// The head's rows in memory, row c at w + c ws.
struct WRows {
  const float* w;
  int ws;
  __device__ __forceinline__ float operator()(int c, int j) const { return w[(size_t)c * ws + j]; }
  template <int NP>
  __device__ __forceinline__ void chains(const int (&cc)[NP], const float* __restrict__ zs, int d,
                                         float (&acc)[NP]) const {
    const float* wc[NP];
#pragma unroll
    for (int t = 0; t < NP; ++t) {
      wc[t] = w + (size_t)cc[t] * ws;
      acc[t] = 0.f;
    }
#pragma unroll 4
    for (int j = 0; j < d; ++j) {
      const float z = zs[j];
#pragma unroll
      for (int t = 0; t < NP; ++t) acc[t] = fmaf(wc[t][j], z, acc[t]);
    }
  }
};

__global__ void __launch_bounds__(kFixWarps * 32) k_certify_fix(const CertArgs a, DevStats* stats, int w_smem) {
  extern __shared__ __align__(16) unsigned char fix_smem[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int d = a.d, C = a.C;
  const int nfix = *a.fix_count;
  if (blockIdx.x == 0 && threadIdx.x == 0 && nfix > 0) atomicAdd(&stats->ins_fp64_rows, (unsigned long long)nfix);
  if ((int)blockIdx.x * kFixWarps >= nfix) return;  // no row for this block
  unsigned char* p = fix_smem;
  WRows W{a.W, d};
  if (w_smem) {
    // asynchronous 4-byte copies, all in flight at once
    float* wsm = reinterpret_cast<float*>(p);
    p += ((size_t)C * (d + 1) + 3) / 4 * 16;
    for (int c = warp; c < C; c += kFixWarps)
      for (int j = lane; j < d; j += 32) {
        const uint32_t dst = (uint32_t)__cvta_generic_to_shared(wsm + (size_t)c * (d + 1) + j);
        asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(dst), "l"(a.W + (size_t)c * d + j) : "memory");
      }
    asm volatile("cp.async.wait_all;" ::: "memory");
    W = WRows{wsm, d + 1};
  }
  __syncthreads();
  const FixScratch sc = fix_scratch_at(p + (size_t)warp * fix_scratch_bytes(d, C), d, C);
  for (int k = (int)blockIdx.x * kFixWarps + warp; k < nfix; k += (int)gridDim.x * kFixWarps) {
    const int64_t row = a.fix_list[k];
    fix_row_warp(a, row, a.kn[row], W, sc, lane);
  }
}

size_t fix_smem_bytes(int d, int C, bool w_smem) {
  const size_t w = w_smem ? ((size_t)C * (d + 1) + 3) / 4 * 16 : 0;
  return w + (size_t)kFixWarps * fix_scratch_bytes(d, C);
}

// Exclusive scan of the per-block accepted counts (one block).
// (after an aborted certify kernel every count reads as 0: nothing is
// appended). The table's device size gives the insert's base index (size0)
// and advances by the total.
__global__ void __launch_bounds__(1024) k_scan(int32_t* __restrict__ cnt, int32_t* __restrict__ off, int nb,
                                               int64_t* __restrict__ total, const DevStats* __restrict__ st,
                                               int64_t* __restrict__ size_dev, int64_t* __restrict__ size0,
                                               const int32_t* __restrict__ fix_list, const uint8_t* __restrict__ accept,
                                               int32_t* __restrict__ rank, int64_t n) {
  __shared__ int64_t carry;
  const int tid = threadIdx.x;
  if (tid == 0) carry = 0;
  // the FP64 pass may have changed a listed row's acceptance: recount its
  // 32-row block (rows listed twice in a block write the same values)
  const int nfix = st->fix_count;
  for (int k = tid; k < nfix; k += 1024) {
    const int64_t r0 = (int64_t)(fix_list[k] / kRows) * kRows;
    const int64_t r1 = r0 + kRows < n ? r0 + kRows : n;
    int c = 0;
    for (int64_t r = r0; r < r1; ++r) {
      rank[r] = c;
      c += accept[r] ? 1 : 0;
    }
    cnt[r0 / kRows] = c;
  }
  __syncthreads();
  // exclusive scan, 2,048 counts a pass: two per thread, warp shuffles, then
  // the 32 warp totals on one warp
  __shared__ int32_t wsum[32];
  const int lane = tid & 31, warp = tid >> 5;
  const bool live = st->abort_flag == 0;
  for (int base = 0; base < nb; base += 2048) {
    const int i0 = base + 2 * tid;
    const int v0 = (i0 < nb && live) ? cnt[i0] : 0;
    const int v1 = (i0 + 1 < nb && live) ? cnt[i0 + 1] : 0;
    int x = v0 + v1;  // inclusive scan of the thread pairs within the warp
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) wsum[warp] = x;
    __syncthreads();
    if (warp == 0) {
      int w = wsum[lane];
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, w, o);
        if (lane >= o) w += y;
      }
      wsum[lane] = w;  // inclusive over the warps
    }
    __syncthreads();
    const int64_t before = carry + (warp > 0 ? wsum[warp - 1] : 0) + (x - v0 - v1);
    if (i0 < nb) off[i0] = (int32_t)before;
    if (i0 + 1 < nb) off[i0 + 1] = (int32_t)(before + v0);
    __syncthreads();
    if (tid == 0) carry += wsum[31];
    __syncthreads();
  }
  if (tid == 0) {
    *total = carry;
    const int64_t s0 = *size_dev;
    *size0 = s0;
    *size_dev = s0 + carry;
  }
}

__global__ void k_set_i64(int64_t* __restrict__ p, int64_t v) { *p = v; }

struct ScatterArgs {
  const float* H;
  int64_t n;
  const int64_t* size0;  // device: the insert's base index
  int d, dpad;
  const uint8_t* accept;
  const int32_t* yG;
  const int32_t* label;
  const float* radius;
  const float* rr;
  const float* kn;
  const float* tau;
  const int32_t* rank;
  const int32_t* boff;
  Table t;
  int64_t* out_index;
  float* out_radius;
  const DevStats* st;  // abort_flag set: the certify kernel gave up, nothing is appended
};

// Append accepted rows in input order. Each warp moves kScatterRows rows:
// lane u < kScatterRows resolves row u's destination and copies its
// per-entry fields, then the warp copies the keys of all its rows with every
// load issued before the stores (float4s for 16-byte rows). The first 128
// floats of every row are loaded before the destinations are known: those
// loads depend on nothing (the rows were just read by the certify kernel and
// mostly sit in L2), so they overlap the chain of dependent loads that
// resolves the destinations; a rejected row is read for nothing.
constexpr int kScatterRows = 8;

__global__ void __launch_bounds__(256) k_scatter(ScatterArgs a, int vec) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t row0 = ((int64_t)blockIdx.x * 8 + warp) * kScatterRows;
  if (row0 >= a.n) return;
  const int n4 = a.dpad / 4, d4 = a.d / 4;
  float4 v0[kScatterRows];
  if (vec) {
#pragma unroll
    for (int u = 0; u < kScatterRows; ++u)
      v0[u] = (row0 + u < a.n && lane < d4) ? __ldg(reinterpret_cast<const float4*>(a.H + (size_t)(row0 + u) * a.d) + lane)
                                            : make_float4(0.f, 0.f, 0.f, 0.f);
  }
  int64_t mydst = -2;  // past the end
  if (lane < kScatterRows && row0 + lane < a.n) {
    const int64_t row = row0 + lane;
    const bool dead = a.st->abort_flag != 0;
    mydst = (!dead && a.accept[row]) ? *a.size0 + a.boff[row / kRows] + a.rank[row] : -1;
    if (mydst >= 0) {
      a.t.kn[mydst] = a.kn[row];
      a.t.tau[mydst] = a.tau[row];
      a.t.rr[mydst] = a.rr[row];
      a.t.radius[mydst] = a.radius[row];
      a.t.label[mydst] = a.label[row];
      a.t.yG[mydst] = a.yG[row];
    }
    if (a.out_index) a.out_index[row] = mydst;
    if (a.out_radius) a.out_radius[row] = dead ? NAN : a.radius[row];
  }
  int64_t dst[kScatterRows];
#pragma unroll
  for (int u = 0; u < kScatterRows; ++u) dst[u] = __shfl_sync(0xffffffffu, mydst, u);
  if (vec) {
    if (lane < n4) {
#pragma unroll
      for (int u = 0; u < kScatterRows; ++u)
        if (dst[u] >= 0) reinterpret_cast<float4*>(a.t.keys + (size_t)dst[u] * a.dpad)[lane] = v0[u];
    }
    for (int j4 = lane + 32; j4 < n4; j4 += 32) {
      float4 v[kScatterRows];
#pragma unroll
      for (int u = 0; u < kScatterRows; ++u)
        v[u] = (dst[u] >= 0 && j4 < d4) ? __ldg(reinterpret_cast<const float4*>(a.H + (size_t)(row0 + u) * a.d) + j4)
                                        : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
      for (int u = 0; u < kScatterRows; ++u)
        if (dst[u] >= 0) reinterpret_cast<float4*>(a.t.keys + (size_t)dst[u] * a.dpad)[j4] = v[u];
    }
  } else {
    for (int j = lane; j < a.dpad; j += 32) {
      float v[kScatterRows];
#pragma unroll
      for (int u = 0; u < kScatterRows; ++u)
        v[u] = (dst[u] >= 0 && j < a.d) ? __ldg(a.H + (size_t)(row0 + u) * a.d + j) : 0.f;
#pragma unroll
      for (int u = 0; u < kScatterRows; ++u)
        if (dst[u] >= 0) a.t.keys[(size_t)dst[u] * a.dpad + j] = v[u];
    }
  }
}

// Certified-consistency check of probe hits: the insert path's argmax y^G of
// each query (already in yq) against y^G of the hit entry. counts[0..2]:
// hits, consistent hits, indices outside [-1, size).
__global__ void __launch_bounds__(256) k_consistency(const int64_t* __restrict__ hit, const int32_t* __restrict__ yq,
                                                     const int32_t* __restrict__ yG_table, int64_t size, int64_t B,
                                                     int8_t* __restrict__ out, int64_t* __restrict__ counts) {
  const int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  int h = 0, c = 0, bad = 0;
  if (k < B) {
    const int64_t i = hit[k];
    int8_t v = -1;
    if (i >= 0 && i < size) {
      h = 1;
      c = yq[k] == yG_table[i];
      v = (int8_t)c;
    } else if (i != -1) {
      bad = 1;
    }
    if (out) out[k] = v;
  }
  const unsigned full = 0xffffffffu;
  h = __popc(__ballot_sync(full, h));
  c = __popc(__ballot_sync(full, c));
  bad = __popc(__ballot_sync(full, bad));
  if ((threadIdx.x & 31) == 0) {
    if (h) atomicAdd(reinterpret_cast<unsigned long long*>(counts), (unsigned long long)h);
    if (c) atomicAdd(reinterpret_cast<unsigned long long*>(counts + 1), (unsigned long long)c);
    if (bad) atomicAdd(reinterpret_cast<unsigned long long*>(counts + 2), (unsigned long long)bad);
  }
}

template <typename T>
void grow(T*& p, int64_t n) {
  if (p) cudaFree(p);
  p = nullptr;
  LC_CUDA(cudaMalloc(&p, sizeof(T) * (size_t)(n > 0 ? n : 1)));
}

void ensure_insert_scratch(lipcache* h, int64_t n) {
  if (n <= h->ins_cap) return;
  int64_t cap = h->ins_cap ? h->ins_cap : 1024;
  while (cap < n) cap *= 2;
  const int64_t nb = (cap + kRows - 1) / kRows;
  grow(h->ins_accept, cap);
  grow(h->ins_yG, cap);
  grow(h->ins_label, cap);
  grow(h->ins_radius, cap);
  grow(h->ins_rr, cap);
  grow(h->ins_kn, cap);
  grow(h->ins_tau, cap);
  grow(h->ins_rank, cap);
  grow(h->ins_fix, cap);
  grow(h->ins_bcount, nb);
  grow(h->ins_boffset, nb);
  h->ins_cap = cap;
}

}  // namespace

size_t certify_smem_bytes(int d, int C) {
  const int hstride = d + 1 + (d & 1);
  const int lstride = C | 1;
  return sizeof(double) * 2 * kWarps * (size_t)C + sizeof(float) * (size_t)kRows * (hstride + lstride);
}

namespace {

// Error factor G of a compensated dot product (Dot2) evaluated as L lane
// chains of n terms each, combined by a butterfly of log2 L levels, then the
// bias: |hi + lo - exact| <= G (sum |W_cj z_j| + |b_c|). The pair hi + lo is
// error-free except for the plain FP32 sum c of the TwoProduct and TwoSum
// error terms: each term passes at most D = n + 2 log2 L + 2 roundings (the
// chain, two per butterfly level, one before the final TwoSum), and the terms
// sum to at most u (n + log2 L + 2) (sum |W_cj z_j| + |b_c|) (the products'
// errors, then one TwoSum error per chain step, per level and for the bias,
// each bounded by u times a partial sum). Hence G = gamma_D u (n + log2 L + 2),
// with a margin for the second-order factors and the float conversion.
double dot2_factor(int n, int L) {
  int lg = 0;
  while ((1 << lg) < L) ++lg;
  return gamma32(n + 2 * lg + 2) * kU32 * (double)(n + lg + 2) * (1.0 + 1e-3);
}

// With timing enabled: a slot of the event ring for a certify kernel, its
// start recorded on `s` (-1 when timing is off).
int timing_begin(lipcache* h, cudaStream_t s) {
  if (!h->timing) return -1;
  if (h->t_issued - h->t_harvested >= lipcache::kTimingRing) harvest_timing(h, false);
  const int slot = (int)(h->t_issued % lipcache::kTimingRing);
  h->t_kind[slot] = 1;
  LC_CUDA(cudaEventRecord(h->tev0[slot], s));
  return slot;
}

// Per-row certification of H (n rows) into the insert scratch: accept, y^G,
// label, radius, probe thresholds, per-32-row ranks and counts.
void launch_certify(lipcache* h, const float* H, int64_t n, const int32_t* payload, int require_consistency,
                    const int64_t* miss_of, cudaStream_t s) {
  ensure_insert_scratch(h, n);
  // the abort flag (raised by the tensor kernel if one of its bounded waits
  // expires) and the FP64 pass's row count
  LC_CUDA(cudaMemsetAsync(&h->stats->abort_flag, 0, 2 * sizeof(int), s));
  CertArgs a;
  a.H = H;
  a.n = n;
  a.d = h->d;
  a.C = h->C;
  a.hstride = h->d + 1 + (h->d & 1);
  a.lstride = h->C | 1;
  a.tight = h->radius_mode == LIPCACHE_RADIUS_TIGHT;
  a.require_consistency = require_consistency ? 1 : 0;
  a.W = h->W;
  a.b = h->b;
  a.Wnorm = h->Wnorm;
  a.pairnorm = h->pairnorm;
  a.payload = payload;
  a.sigma = h->sigma;
  a.kappa = h->radius_scale;
  a.eps_rc = h->eps_rc;
  a.gamma_rc = gamma32(h->dpad / 32 + 33);
  a.c_scr = h->c_scr;
  a.g32 = gamma32(h->d + 2) * (1.0 + 1e-6);
  a.g64 = gamma64(h->d + 8) * (1.0 + 1e-6);
  a.Wnorm32 = h->Wnorm32;
  a.g32f = (float)(gamma32(h->d + 2) * (1.0 + 1e-4));
  a.g2f = (float)dot2_factor(h->d, 1);             // a lane per class over every feature
  a.g2f8 = (float)dot2_factor((h->d + 7) / 8, 8);    // 8-lane groups
  a.g2f32 = (float)dot2_factor((h->d + 31) / 32, 32);  // whole warps
  a.tc = thresh_consts(h->dpad);
  a.miss_of = miss_of;
  a.inv_pairnorm = h->inv_pairnorm;
  a.ipn_up32 = h->ipn_up32;
  a.ipn_dn32 = h->ipn_dn32;
  a.ipn_min32 = h->ipn_min32;
  a.ipn_max32 = h->ipn_max32;
  a.tight_f = 1.0 - gamma64(h->d + 8);
  a.inv_denom = h->radius_scale / (h->sigma * 1.4142135623730951);
  a.inv_denom_safe = h->radius_scale * (1.0 - 8 * kU64) / (h->sigma * (1.0 + kSigmaSlack) * 1.4142135623730951);
  a.accept = h->ins_accept;
  a.yG = h->ins_yG;
  a.label = h->ins_label;
  a.radius = h->ins_radius;
  a.rr = h->ins_rr;
  a.kn = h->ins_kn;
  a.tau = h->ins_tau;
  a.rank = h->ins_rank;
  a.bcount = h->ins_bcount;
  a.fix_count = &h->stats->fix_count;
  a.fix_list = h->ins_fix;
  // rounding bound of the FP64 pass's logits: a chain of ceil(d/32) products
  // per lane, a five-level tree and the bias
  a.gfix = (float)(gamma64((h->d + 31) / 32 + 6) * 1.001);
  const int nb = (int)((n + kRows - 1) / kRows);
  const int Cp = (h->C + 7) / 8 * 8;
  const size_t smem_wres = sizeof(float) * ((size_t)h->dpad * Cp + (size_t)h->dpad * kHStride +
                                            (size_t)kWTile * a.lstride + 1 + 4 * (size_t)h->C) +
                           sizeof(double) * 2 * kWarps * (size_t)(a.tight ? h->C : 0) + sizeof(TileSmem);
  int slot = -1;
  const int ncg = wt_ncg(h->C);
  const bool vec16 = h->d % 4 == 0 && ((uintptr_t)H & 15) == 0;
  const WtLayout L = wt_layout(h->d, h->C, ncg > 0 ? ncg : 1);
  bool fixed_in_kernel = false;
  if (certify_tc_supported(h, H, n)) {
    slot = timing_begin(h, s);
    fixed_in_kernel = certify_tc_launch(h, a, s);
    h->last_insert_kernel = LIPCACHE_INSERT_TENSOR;
  } else if ((!a.tight || h->ipn_up32) && vec16 && ncg > 0 && L.total <= 227 * 1024 &&
             !(h->debug_flags & LIPCACHE_DEBUG_INSERT_TILE64)) {
    const int64_t nb32 = (n + 31) / 32;
    const int grid = nb32 < h->num_sms ? (int)nb32 : h->num_sms;
    if (h->wt_prep_ncg != ncg) {
      if (h->wt_prep_cap < L.off_h) {
        if (h->wt_prep) cudaFree(h->wt_prep);
        h->wt_prep = nullptr;
        h->wt_prep_cap = 0;
        LC_CUDA(cudaMalloc(&h->wt_prep, L.off_h));
        h->wt_prep_cap = L.off_h;
      }
      k_wt_prepare<<<64, 256, 0, s>>>(a, L, h->wt_prep);
      LC_LAUNCH_CHECK("k_wt_prepare");
      h->wt_prep_ncg = ncg;
    }
    void (*kern)(CertArgs, WtLayout, const float*, int64_t) = ncg == 1    ? k_certify_wt<1>
                                            : ncg == 4  ? k_certify_wt<4>
                                            : ncg == 7  ? k_certify_wt<7>
                                            : ncg == 13 ? k_certify_wt<13>
                                                        : k_certify_wt<16>;
    LC_CUDA(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)L.total));
    slot = timing_begin(h, s);
    kern<<<grid, kThreads, L.total, s>>>(a, L, h->wt_prep, nb32);
    LC_LAUNCH_CHECK("k_certify_wt");
    h->last_insert_kernel = LIPCACHE_INSERT_WIDE_TILE;
  } else if (h->C <= 256 && smem_wres <= 220 * 1024) {
    const int n_tiles = (int)((n + kWTile - 1) / kWTile);
    const int grid = n_tiles < h->num_sms ? n_tiles : h->num_sms;
    LC_CUDA(cudaFuncSetAttribute(k_certify_wres, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_wres));
    const int vec = (h->d % 4 == 0 && ((uintptr_t)H & 15) == 0) ? 1 : 0;
    slot = timing_begin(h, s);
    k_certify_wres<<<grid, kThreads, smem_wres, s>>>(a, Cp, h->dpad, n_tiles, vec);
    LC_LAUNCH_CHECK("k_certify_wres");
    h->last_insert_kernel = LIPCACHE_INSERT_TILE64;
  } else {
    const size_t smem = certify_smem_bytes(h->d, h->C);
    LC_CUDA(cudaFuncSetAttribute(k_certify, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
    slot = timing_begin(h, s);
    k_certify<<<nb, kThreads, smem, s>>>(a);
    LC_LAUNCH_CHECK("k_certify");
    h->last_insert_kernel = LIPCACHE_INSERT_STREAMED;
  }
  // the FP64 pass over the rows the kernel listed (a few per 100,000; none
  // from the kernels that refine in FP64 already), unless the kernel ran it
  if (!fixed_in_kernel) {
    const bool w_smem = fix_smem_bytes(h->d, h->C, true) <= 200 * 1024;
    const size_t fsm = fix_smem_bytes(h->d, h->C, w_smem);
    if (fsm > 48 * 1024) LC_CUDA(cudaFuncSetAttribute(k_certify_fix, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)fsm));
    k_certify_fix<<<h->num_sms, kFixWarps * 32, fsm, s>>>(a, h->stats, w_smem ? 1 : 0);
    LC_LAUNCH_CHECK("k_certify_fix");
  }
  if (slot >= 0) {
    LC_CUDA(cudaEventRecord(h->tev1[slot], s));
    ++h->t_issued;
  }
}

}  // namespace

void certify_insert(lipcache* h, const float* H, int64_t n, const int32_t* payload, int require_consistency,
                    int64_t* out_index, float* out_radius, cudaStream_t s, const int64_t* miss_of) {
  launch_certify(h, H, n, payload, require_consistency, miss_of, s);
  const int nb = (int)((n + kRows - 1) / kRows);
  k_scan<<<1, 1024, 0, s>>>(h->ins_bcount, h->ins_boffset, nb, h->ins_total, h->stats, h->size_dev, h->ins_size0,
                            h->ins_fix, h->ins_accept, h->ins_rank, n);
  LC_LAUNCH_CHECK("k_scan");
  ScatterArgs sa;
  sa.H = H;
  sa.n = n;
  sa.size0 = h->ins_size0;
  sa.d = h->d;
  sa.dpad = h->dpad;
  sa.accept = h->ins_accept;
  sa.yG = h->ins_yG;
  sa.label = h->ins_label;
  sa.radius = h->ins_radius;
  sa.rr = h->ins_rr;
  sa.kn = h->ins_kn;
  sa.tau = h->ins_tau;
  sa.rank = h->ins_rank;
  sa.boff = h->ins_boffset;
  sa.t = h->table;
  sa.out_index = out_index;
  sa.out_radius = out_radius;
  sa.st = h->stats;
  const int vec = (h->d % 4 == 0 && ((uintptr_t)H & 15) == 0) ? 1 : 0;
  const int64_t rows_per_block = 8 * kScatterRows;
  k_scatter<<<(unsigned)((n + rows_per_block - 1) / rows_per_block), 256, 0, s>>>(sa, vec);
  LC_LAUNCH_CHECK("k_scatter");
}

void store_size_dev(lipcache* h, cudaStream_t s) {
  k_set_i64<<<1, 1, 0, s>>>(h->size_dev, h->size);
  LC_LAUNCH_CHECK("k_set_i64");
}

void settle_size(lipcache* h) {
  if (!h->size_pending) return;
  LC_CUDA(cudaMemcpyAsync(h->size_pinned, h->size_dev, sizeof(int64_t), cudaMemcpyDeviceToHost, h->pending_stream));
  LC_CUDA(cudaStreamSynchronize(h->pending_stream));
  h->size = *h->size_pinned;
  h->size_pending = false;
  h->pending_rows = 0;
}

void require_certify_ok(lipcache* h, cudaStream_t s) {
  LC_CUDA(cudaMemcpyAsync(h->stats_host, h->stats, sizeof(DevStats), cudaMemcpyDeviceToHost, s));
  LC_CUDA(cudaStreamSynchronize(s));
  LC_REQUIRE(h->stats_host->abort_flag == 0, LIPCACHE_E_DEVICE, kCertifyAbortMessage);
}

void certify_rows(lipcache* h, const float* H, int64_t n, const int32_t* payload, int require_consistency,
                  cudaStream_t s) {
  launch_certify(h, H, n, payload, require_consistency, nullptr, s);
}

void consistency_check(lipcache* h, const float* Q, int64_t B, const int64_t* hit_index, int8_t* out,
                       cudaStream_t s) {
  launch_certify(h, Q, B, nullptr, 0, nullptr, s);
  LC_CUDA(cudaMemsetAsync(h->ins_total + 1, 0, 3 * sizeof(int64_t), s));
  k_consistency<<<(unsigned)((B + 255) / 256), 256, 0, s>>>(hit_index, h->ins_yG, h->table.yG, h->size, B, out,
                                                           h->ins_total + 1);
  LC_LAUNCH_CHECK("k_consistency");
}

}  // namespace lc
