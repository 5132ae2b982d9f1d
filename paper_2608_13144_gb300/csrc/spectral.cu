// Spectral norm of the GuardNet head: sigma_max(W), the Lipschitz constant of
// f(z) = W z + b (Sec. 4.1, Eqs. 17-19; the bias cancels in logit
// differences). Algorithm 1 computes it once per cache, before any radius.
//
// Method: power iteration on A = W^T W in FP64. Power iteration alone needs
// about log(tol) / log(lambda_2/lambda_1) steps, which is thousands for the
// small spectral gaps of Gaussian heads, so the start vector is produced by
// `squarings` normalised squarings A_{k+1} = (A_k / tr A_k)^2, i.e. by the
// power iteration with A^(2^k) (2^40 steps for the default 40). The final
// iteration then runs on W itself (w = W v, theta = ||w||^2 = v^T A v,
// u = W^T w) until successive Rayleigh quotients agree to 1e-13 relative and
// ||A v - theta v|| <= 1e-10 theta.
#include "internal.cuh"

namespace lc {
namespace {

constexpr int kTile = 16;

// A = W^T W (d x d, FP64). Products of FP32 values are exact in FP64; the
// accumulation order is the same for (i, j) and (j, i), so A is bitwise
// symmetric.
__global__ void k_gram(const float* __restrict__ W, int C, int d, double* __restrict__ A) {
  const int j = blockIdx.x * kTile + threadIdx.x;
  const int i = blockIdx.y * kTile + threadIdx.y;
  if (i >= d || j >= d) return;
  double acc = 0.0;
  for (int c = 0; c < C; ++c) acc = fma((double)W[(size_t)c * d + i], (double)W[(size_t)c * d + j], acc);
  A[(size_t)i * d + j] = acc;
}

// B = (A / tr A)^2 with a tiled FP64 product; every block recomputes the
// trace (d loads). A zero trace (W = 0) yields B = 0.
__global__ void k_square(const double* __restrict__ A, double* __restrict__ B, int d) {
  __shared__ double As[kTile][kTile + 1];
  __shared__ double Bs[kTile][kTile + 1];
  __shared__ double red[kTile * kTile];
  const int tx = threadIdx.x, ty = threadIdx.y, tid = ty * kTile + tx;
  double t = 0.0;
  for (int k = tid; k < d; k += kTile * kTile) t += A[(size_t)k * d + k];
  red[tid] = t;
  __syncthreads();
  for (int s = kTile * kTile / 2; s > 0; s >>= 1) {
    if (tid < s) red[tid] += red[tid + s];
    __syncthreads();
  }
  const double tr = red[0];
  const double inv = tr > 0.0 ? 1.0 / tr : 0.0;
  const int i = blockIdx.y * kTile + ty;
  const int j = blockIdx.x * kTile + tx;
  double acc = 0.0;
  for (int k0 = 0; k0 < d; k0 += kTile) {
    As[ty][tx] = (i < d && k0 + tx < d) ? A[(size_t)i * d + k0 + tx] * inv : 0.0;
    Bs[ty][tx] = (k0 + ty < d && j < d) ? A[(size_t)(k0 + ty) * d + j] * inv : 0.0;
    __syncthreads();
#pragma unroll
    for (int k = 0; k < kTile; ++k) acc = fma(As[ty][k], Bs[k][tx], acc);
    __syncthreads();
  }
  if (i < d && j < d) B[(size_t)i * d + j] = acc;
}

constexpr int kPowerThreads = 256;

__device__ double block_sum(double v, double* red) {
  const int tid = threadIdx.x;
  red[tid] = v;
  __syncthreads();
  for (int s = kPowerThreads / 2; s > 0; s >>= 1) {
    if (tid < s) red[tid] += red[tid + s];
    __syncthreads();
  }
  const double r = red[0];
  __syncthreads();
  return r;
}

// Final power iteration on W (one block). `As` is the last squared matrix
// (or nullptr to start from a fixed, slightly perturbed all-ones vector).
__global__ void __launch_bounds__(kPowerThreads) k_power(const float* __restrict__ W, int C, int d,
                                                         const double* __restrict__ As, int max_iter,
                                                         SpecResult* __restrict__ res) {
  extern __shared__ double sm[];
  double* v = sm;          // d
  double* w = v + d;       // C
  double* u = w + C;       // d
  __shared__ double red[kPowerThreads];
  __shared__ int jstar;
  const int tid = threadIdx.x;

  if (As) {
    if (tid == 0) {
      int best = 0;
      for (int k = 1; k < d; ++k)
        if (As[(size_t)k * d + k] > As[(size_t)best * d + best]) best = k;
      jstar = best;
    }
    __syncthreads();
    for (int k = tid; k < d; k += kPowerThreads) v[k] = As[(size_t)k * d + jstar];
  } else {
    for (int k = tid; k < d; k += kPowerThreads) {
      unsigned x = (unsigned)k * 2654435761u;
      x ^= x >> 15;
      v[k] = 1.0 + 0.01 * (double)(x & 0xffff) / 65536.0;
    }
  }
  __syncthreads();
  double nv = 0.0;
  for (int k = tid; k < d; k += kPowerThreads) nv += v[k] * v[k];
  nv = sqrt(block_sum(nv, red));

  double theta = 0.0, theta_prev = -1.0, resid = INFINITY;
  int it = 0, converged = 0;
  if (!(nv > 0.0)) {
    if (tid == 0) {
      res->sigma = 0.0;
      res->theta = 0.0;
      res->residual_rel = 0.0;
      res->iterations = 0;
      res->converged = 1;
      res->degenerate = 1;
    }
    return;
  }
  for (int k = tid; k < d; k += kPowerThreads) v[k] /= nv;
  __syncthreads();

  for (it = 1; it <= max_iter; ++it) {
    for (int c = tid; c < C; c += kPowerThreads) {
      double acc = 0.0;
      for (int k = 0; k < d; ++k) acc = fma((double)W[(size_t)c * d + k], v[k], acc);
      w[c] = acc;
    }
    __syncthreads();
    double p = 0.0;
    for (int c = tid; c < C; c += kPowerThreads) p += w[c] * w[c];
    theta = block_sum(p, red);
    for (int k = tid; k < d; k += kPowerThreads) {
      double acc = 0.0;
      for (int c = 0; c < C; ++c) acc = fma((double)W[(size_t)c * d + k], w[c], acc);
      u[k] = acc;
    }
    __syncthreads();
    double pr = 0.0, pu = 0.0;
    for (int k = tid; k < d; k += kPowerThreads) {
      const double e = u[k] - theta * v[k];
      pr += e * e;
      pu += u[k] * u[k];
    }
    resid = sqrt(block_sum(pr, red));
    const double nu = sqrt(block_sum(pu, red));
    if (!(nu > 0.0)) {  // v is in the null space of W: only possible for W = 0
      theta = 0.0;
      resid = 0.0;
      converged = 1;
      break;
    }
    for (int k = tid; k < d; k += kPowerThreads) v[k] = u[k] / nu;
    __syncthreads();
    if (it >= 2 && fabs(theta - theta_prev) <= 1e-13 * theta && resid <= 1e-10 * theta) {
      converged = 1;
      break;
    }
    theta_prev = theta;
  }
  if (tid == 0) {
    res->theta = theta;
    res->sigma = sqrt(theta);
    res->residual_rel = theta > 0.0 ? resid / theta : 0.0;
    res->iterations = it > max_iter ? max_iter : it;
    res->converged = converged;
    res->degenerate = !(theta > 0.0);
  }
}

// ||W_c|| for every class and, for the tight radius, ||W_y - W_j|| for every
// pair (FP64; the differences of FP32 weights are exact, the sum of d squares
// is within gamma_d of the exact one) with its reciprocal, and FP32 brackets
// of the reciprocal (the FP64 value widened by 1e-12, far above its error,
// then rounded outward; +inf for coinciding rows, which the tight radius skips).
__global__ void k_row_norms(const float* __restrict__ W, int C, int d, double* __restrict__ Wnorm,
                            float* __restrict__ Wnorm32, double* __restrict__ pairnorm,
                            double* __restrict__ inv_pairnorm, float* __restrict__ ipn_up32,
                            float* __restrict__ ipn_dn32) {
  const int y = blockIdx.y;
  const int j = blockIdx.x * blockDim.x + threadIdx.x;
  if (j >= C) return;
  double acc = 0.0;
  if (pairnorm) {
    for (int k = 0; k < d; ++k) {
      const double e = (double)W[(size_t)y * d + k] - (double)W[(size_t)j * d + k];
      acc = fma(e, e, acc);
    }
    pairnorm[(size_t)y * C + j] = sqrt(acc);
    const double ipn = acc > 0.0 ? 1.0 / sqrt(acc) : 0.0;
    inv_pairnorm[(size_t)y * C + j] = ipn;
    ipn_up32[(size_t)y * C + j] = acc > 0.0 ? __double2float_ru(ipn * (1.0 + 1e-12)) : INFINITY;
    ipn_dn32[(size_t)y * C + j] = acc > 0.0 ? __double2float_rd(ipn * (1.0 - 1e-12)) : INFINITY;
  }
  if (j == y) {
    double n2 = 0.0;
    for (int k = 0; k < d; ++k) n2 = fma((double)W[(size_t)y * d + k], (double)W[(size_t)y * d + k], n2);
    Wnorm[y] = sqrt(n2);
    Wnorm32[y] = __double2float_ru(sqrt(n2) * (1.0 + 1e-15));
  }
}

// Bounds of a whole row of the bracket tables, which the tensor certify
// kernel's tight-radius screen uses in place of the tables:
// ipn_min32[y] <= 1 / ||W_y - W_j|| for every j with W_j != W_y (the minimum of
// the FP32 lower brackets; 0 when every other row equals W_y) and
// ipn_max32[y] >= 1 / ||W_y - W_j|| for every j != y (+inf when some W_j = W_y).
__global__ void k_ipn_min(const double* __restrict__ pairnorm, const float* __restrict__ ipn_dn32,
                          const float* __restrict__ ipn_up32, int C, float* __restrict__ ipn_min32,
                          float* __restrict__ ipn_max32) {
  const int y = blockIdx.x * blockDim.x + threadIdx.x;
  if (y >= C) return;
  float m = INFINITY, mx = 0.f;
  for (int j = 0; j < C; ++j) {
    if (j == y) continue;
    if (pairnorm[(size_t)y * C + j] > 0.0) m = fminf(m, ipn_dn32[(size_t)y * C + j]);
    mx = fmaxf(mx, ipn_up32[(size_t)y * C + j]);
  }
  ipn_min32[y] = m < INFINITY ? m : 0.f;
  ipn_max32[y] = mx;
}

}  // namespace

void spectral_norm(lipcache* h, cudaStream_t s) {
  const int d = h->d, C = h->C;
  dim3 blk(kTile, kTile), grd((d + kTile - 1) / kTile, (d + kTile - 1) / kTile);
  const double* As = nullptr;
  if (h->squarings > 0) {
    k_gram<<<grd, blk, 0, s>>>(h->W, C, d, h->gram[0]);
    LC_LAUNCH_CHECK("k_gram");
    int cur = 0;
    for (int k = 0; k < h->squarings; ++k) {
      k_square<<<grd, blk, 0, s>>>(h->gram[cur], h->gram[cur ^ 1], d);
      LC_LAUNCH_CHECK("k_square");
      cur ^= 1;
    }
    As = h->gram[cur];
  }
  const size_t smem = sizeof(double) * (size_t)(2 * d + C);
  k_power<<<1, kPowerThreads, smem, s>>>(h->W, C, d, As, h->max_iter, h->spec);
  LC_LAUNCH_CHECK("k_power");
  dim3 rb(128), rg((C + 127) / 128, C);
  const bool tight = h->radius_mode == LIPCACHE_RADIUS_TIGHT;
  k_row_norms<<<rg, rb, 0, s>>>(h->W, C, d, h->Wnorm, h->Wnorm32, tight ? h->pairnorm : nullptr,
                                tight ? h->inv_pairnorm : nullptr, tight ? h->ipn_up32 : nullptr,
                                tight ? h->ipn_dn32 : nullptr);
  LC_LAUNCH_CHECK("k_row_norms");
  if (tight) {
    k_ipn_min<<<(C + 127) / 128, 128, 0, s>>>(h->pairnorm, h->ipn_dn32, h->ipn_up32, C, h->ipn_min32, h->ipn_max32);
    LC_LAUNCH_CHECK("k_ipn_min");
  }
}

}  // namespace lc
