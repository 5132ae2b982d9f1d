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
// interval can reach the true top two, and recomputes those classes in FP64
// (products of FP32 values are exact in FP64). The true top-1 and runner-up
// are always among them, so m equals the FP64 margin of the full logit
// vector. The tight radius needs every class and refines all of them.
//
// Besides the reported radius r, the kernel derives a certified lower bound
// r_safe (FP64 error bounds of the two logits, sigma inflated by 1e-9) and
// from it the probe's acceptance threshold rr = RZ(r_safe^2 (1 - eps_rc)) on
// the canonical FP32 squared distance, and the screen term tau.
//
// Insertion order is kept by a block-count scan and a scatter.
#include "internal.cuh"

namespace lc {
namespace {

constexpr int kRows = 32;
constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr unsigned kFull = 0xffffffffu;

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
  uint8_t* accept;
  int32_t* yG;
  int32_t* label;
  float* radius;
  float* rr;
  float* kn;
  float* tau;
  int32_t* rank;
  int32_t* bcount;
};

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
  for (int r = warp; r < nrows; r += kWarps) {
    const int64_t row = row0 + r;
    const float* hrow = hs + r * a.hstride;
    const float* lrow = lg + r * a.lstride;
    float knp = 0.f;
    double hnp = 0.0;
    for (int j = lane; j < d; j += 32) {
      const float x = hrow[j];
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
          const double t = (double)__ldg(wc + j) * (double)hrow[j];
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
    const double sqrt2 = 1.4142135623730951;
    if (!a.tight) {
      double up_other = -INFINITY;
      for (int c = lane; c < C; c += 32)
        if (c != y) up_other = fmax(up_other, ws[c] + we[c]);
      up_other = warp_max_d(up_other);
      const double mval = (b1 == b1 && b2 == b2) ? b1 - b2 : NAN;
      const double mlo = (sy - ey) - up_other;
      r64 = a.kappa * mval / (a.sigma * sqrt2);
      rs = (mlo > 0.0) ? a.kappa * mlo * (1.0 - 8 * kU64) / (a.sigma * (1.0 + kSigmaSlack) * sqrt2) : 0.0;
      if (!(mval == mval)) r64 = NAN;
    } else {
      double rmin = INFINITY, smin = INFINITY;
      bool any_nan = !(sy == sy);
      for (int j = lane; j < C; j += 32) {
        if (j == y) continue;
        const double pn = a.pairnorm[(size_t)y * C + j];
        if (!(ws[j] == ws[j])) any_nan = true;
        if (!(pn > 0.0)) continue;
        rmin = fmin(rmin, (sy - ws[j]) / pn);
        smin = fmin(smin, ((sy - ey) - (ws[j] + we[j])) / (pn * (1.0 + 1e-14)));
      }
      rmin = warp_min_d(rmin);
      smin = warp_min_d(smin);
      any_nan = __any_sync(kFull, any_nan);
      r64 = any_nan ? NAN : a.kappa * rmin;
      rs = (smin > 0.0 && !any_nan) ? a.kappa * smin * (1.0 - 8 * kU64) : 0.0;
    }

    if (lane == 0) {
      const int32_t lab = a.payload ? a.payload[row] : y;
      const bool acc = !(a.require_consistency && lab != y) && (r64 > 0.0);
      const double rr64 = rs * rs * (1.0 - a.eps_rc);
      const float rr = __double2float_rz(rr64);
      const double Rt = (double)rr / (1.0 - a.gamma_rc) * (1.0 + 1e-15);
      const float tau = __double2float_rd(((1.0 - a.c_scr) * (double)kn - Rt) * 0.5);
      a.accept[row] = acc ? 1 : 0;
      a.yG[row] = y;
      a.label[row] = lab;
      a.radius[row] = __double2float_rz(r64);
      a.rr[row] = rr;
      a.kn[row] = kn;
      a.tau[row] = tau;
      acc_flag[r] = acc ? 1 : 0;
    }
    __syncwarp();
  }
  __syncthreads();
  if (warp == 0) {
    const bool f = lane < nrows && acc_flag[lane];
    const unsigned m = __ballot_sync(kFull, f);
    if (lane < nrows) a.rank[row0 + lane] = __popc(m & ((1u << lane) - 1u));
    if (lane == 0) a.bcount[blockIdx.x] = __popc(m);
  }
}

// Exclusive scan of the per-block accepted counts (one block).
__global__ void __launch_bounds__(1024) k_scan(const int32_t* __restrict__ cnt, int32_t* __restrict__ off, int nb,
                                               int64_t* __restrict__ total) {
  __shared__ int32_t buf[1024];
  __shared__ int64_t carry;
  const int tid = threadIdx.x;
  if (tid == 0) carry = 0;
  __syncthreads();
  for (int base = 0; base < nb; base += 1024) {
    const int i = base + tid;
    const int v = i < nb ? cnt[i] : 0;
    buf[tid] = v;
    __syncthreads();
    for (int s = 1; s < 1024; s <<= 1) {
      const int t = tid >= s ? buf[tid - s] : 0;
      __syncthreads();
      buf[tid] += t;
      __syncthreads();
    }
    if (i < nb) off[i] = (int32_t)(carry + buf[tid] - v);
    __syncthreads();
    if (tid == 1023) carry += buf[1023];
    __syncthreads();
  }
  if (tid == 0) *total = carry;
}

struct ScatterArgs {
  const float* H;
  int64_t n, size0;
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
};

// Append accepted rows in input order; one warp per row.
__global__ void __launch_bounds__(256) k_scatter(ScatterArgs a) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t row = (int64_t)blockIdx.x * 8 + warp;
  if (row >= a.n) return;
  const bool acc = a.accept[row] != 0;
  const int64_t dst = acc ? a.size0 + a.boff[row / kRows] + a.rank[row] : -1;
  if (acc) {
    float* kd = a.t.keys + (size_t)dst * a.dpad;
    const float* hs = a.H + (size_t)row * a.d;
    for (int j = lane; j < a.dpad; j += 32) kd[j] = j < a.d ? hs[j] : 0.f;
    if (lane == 0) {
      a.t.kn[dst] = a.kn[row];
      a.t.tau[dst] = a.tau[row];
      a.t.rr[dst] = a.rr[row];
      a.t.radius[dst] = a.radius[row];
      a.t.label[dst] = a.label[row];
      a.t.yG[dst] = a.yG[row];
    }
  }
  if (lane == 0) {
    if (a.out_index) a.out_index[row] = dst;
    if (a.out_radius) a.out_radius[row] = a.radius[row];
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

void certify_insert(lipcache* h, const float* H, int64_t n, const int32_t* payload, int require_consistency,
                    int64_t* out_index, float* out_radius, cudaStream_t s) {
  ensure_insert_scratch(h, n);
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
  a.accept = h->ins_accept;
  a.yG = h->ins_yG;
  a.label = h->ins_label;
  a.radius = h->ins_radius;
  a.rr = h->ins_rr;
  a.kn = h->ins_kn;
  a.tau = h->ins_tau;
  a.rank = h->ins_rank;
  a.bcount = h->ins_bcount;
  const int nb = (int)((n + kRows - 1) / kRows);
  const size_t smem = certify_smem_bytes(h->d, h->C);
  LC_CUDA(cudaFuncSetAttribute(k_certify, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  k_certify<<<nb, kThreads, smem, s>>>(a);
  LC_LAUNCH_CHECK("k_certify");
  k_scan<<<1, 1024, 0, s>>>(h->ins_bcount, h->ins_boffset, nb, h->ins_total);
  LC_LAUNCH_CHECK("k_scan");
  ScatterArgs sa;
  sa.H = H;
  sa.n = n;
  sa.size0 = h->size;
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
  k_scatter<<<(unsigned)((n + 7) / 8), 256, 0, s>>>(sa);
  LC_LAUNCH_CHECK("k_scatter");
}

}  // namespace lc
