// Empirical reuse boundaries as radius policies of the probe (Sec. 5.4).
//
// The paper compares the certified radius with two empirical boundaries: one
// global nearest-neighbour threshold, and a radius from inter-class distance
// statistics. Both run through the unchanged probe kernels: a policy only
// replaces the per-entry thresholds (rr, tau) that the probe reads.
//
//   GLOBAL      r_i = tau for every entry.
//   INTERCLASS  mu_c = mean of the cached keys with label c; r_i = rho_{label_i}
//               with rho_c = beta / 2 * min_{c' != c present} ||mu_c - mu_c'||.
//               Labels outside [0, C), classes without entries and a class
//               with no other class present get radius 0. The statistics are
//               those of the cache when the policy is set; entries inserted
//               later take rho of their label from that snapshot.
//
// The thresholds are derived from r exactly as the certified ones are from
// r_safe (rounded down, deflated by the recheck error bound), so a GPU hit
// still lies strictly inside the policy's radius.
#include "internal.cuh"

namespace lc {
namespace {

constexpr int kBatch = 8;

// Class sums of one chunk of entries over a slice of columns: thread j owns
// column blockIdx.y * wcol + j, so every shared accumulator has a single
// writer (no atomics) and the sums are deterministic. The chunk's partial
// sums go to part_sum[blockIdx.x][c][col], counts to part_cnt[blockIdx.x][c].
__global__ void k_class_partial(const float* __restrict__ keys, const int32_t* __restrict__ label, int64_t size,
                                int dpad, int C, int wcol, int64_t chunk, double* __restrict__ part_sum,
                                int64_t* __restrict__ part_cnt) {
  extern __shared__ double acc[];  // C x wcol, then C counts (int64)
  long long* cnt = reinterpret_cast<long long*>(acc + (size_t)C * wcol);
  const int j = threadIdx.x;
  const int col = blockIdx.y * wcol + j;
  for (int i = j; i < C * wcol; i += blockDim.x) acc[i] = 0.0;
  for (int i = j; i < C; i += blockDim.x) cnt[i] = 0;
  __syncthreads();
  const int64_t e0 = (int64_t)blockIdx.x * chunk;
  const int64_t e1 = e0 + chunk < size ? e0 + chunk : size;
  const bool active = j < wcol && col < dpad;
  const bool counter = j == 0 && blockIdx.y == 0;
  if (active) {
    for (int64_t e = e0; e < e1; e += kBatch) {
      int c[kBatch];
      float v[kBatch];
#pragma unroll
      for (int u = 0; u < kBatch; ++u) {
        const bool in = e + u < e1;
        c[u] = in ? __ldg(label + e + u) : -1;
        v[u] = in ? __ldg(keys + (size_t)(e + u) * dpad + col) : 0.f;
      }
#pragma unroll
      for (int u = 0; u < kBatch; ++u) {
        if (c[u] >= 0 && c[u] < C) {
          acc[c[u] * wcol + j] += (double)v[u];
          if (counter) cnt[c[u]] += 1;
        }
      }
    }
  }
  __syncthreads();
  if (active)
    for (int cc = 0; cc < C; ++cc) part_sum[((size_t)blockIdx.x * C + cc) * dpad + col] = acc[cc * wcol + j];
  if (blockIdx.y == 0)
    for (int cc = j; cc < C; cc += blockDim.x) part_cnt[(size_t)blockIdx.x * C + cc] = cnt[cc];
}

// Centroids: mu[c][col] = (sum over chunks, in chunk order) / count. One
// block per class; mu and the total count go to slot nb of the scratch.
__global__ void k_class_centroid(double* __restrict__ part_sum, int64_t* __restrict__ part_cnt, int nb, int C,
                                 int dpad) {
  const int c = blockIdx.x;
  int64_t n = 0;
  for (int b = 0; b < nb; ++b) n += part_cnt[(size_t)b * C + c];
  for (int col = threadIdx.x; col < dpad; col += blockDim.x) {
    double s = 0.0;
    for (int b = 0; b < nb; ++b) s += part_sum[((size_t)b * C + c) * dpad + col];
    part_sum[((size_t)nb * C + c) * dpad + col] = n > 0 ? s / (double)n : 0.0;
  }
  if (threadIdx.x == 0) part_cnt[(size_t)nb * C + c] = n;
}

constexpr int kRhoThreads = 128;

// rho_c = beta / 2 * distance to the nearest other present class centroid.
__global__ void __launch_bounds__(kRhoThreads) k_class_rho(const double* __restrict__ mu,
                                                           const int64_t* __restrict__ cnt, int C, int dpad,
                                                           double beta, double* __restrict__ rho,
                                                           float* __restrict__ rho32) {
  __shared__ double red[kRhoThreads];
  const int c = blockIdx.x, t = threadIdx.x;
  double best = INFINITY;
  if (cnt[c] > 0) {
    for (int c2 = 0; c2 < C; ++c2) {
      if (c2 == c || cnt[c2] == 0) continue;
      double p = 0.0;
      for (int col = t; col < dpad; col += kRhoThreads) {
        const double e = mu[(size_t)c * dpad + col] - mu[(size_t)c2 * dpad + col];
        p = fma(e, e, p);
      }
      red[t] = p;
      __syncthreads();
      for (int s = kRhoThreads / 2; s > 0; s >>= 1) {
        if (t < s) red[t] += red[t + s];
        __syncthreads();
      }
      best = fmin(best, red[0]);
      __syncthreads();
    }
  }
  if (t == 0) {
    const double r = (best < INFINITY) ? beta * 0.5 * sqrt(best) : 0.0;
    rho[c] = r;
    rho32[c] = __double2float_rd(r);
  }
}

// Empirical thresholds of entries [0, n).
__global__ void k_policy_fill(const float* __restrict__ kn, const int32_t* __restrict__ label, int64_t n, int C,
                              int policy, float param32, const float* __restrict__ rho32, ThreshConsts tc,
                              float* __restrict__ rr_emp, float* __restrict__ tau_emp) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  float r = param32;
  if (policy == LIPCACHE_POLICY_INTERCLASS) {
    const int32_t c = label[i];
    r = (c >= 0 && c < C) ? rho32[c] : 0.f;
  }
  float rr, tau;
  thresholds(r, kn[i], tc, rr, tau);
  rr_emp[i] = rr;
  tau_emp[i] = tau;
}

template <typename T>
void alloc(T*& p, size_t n) {
  if (!p) LC_CUDA(cudaMalloc(&p, sizeof(T) * (n > 0 ? n : 1)));
}

}  // namespace

void set_radius_policy(lipcache* h, int policy, double param, double* rho_host, cudaStream_t s) {
  const int C = h->C, dpad = h->dpad;
  if (policy == LIPCACHE_POLICY_CERTIFIED) {
    h->policy = policy;
    h->policy_param = 0.0;
    return;
  }
  if (!h->rr_emp) {
    alloc(h->rr_emp, (size_t)h->table_rows);
    alloc(h->tau_emp, (size_t)h->table_rows);
    // rows past the last entry: never accepted, always screened out
    LC_CUDA(cudaMemsetAsync(h->rr_emp, 0, sizeof(float) * (size_t)h->table_rows, s));
    LC_CUDA(cudaMemsetAsync(h->tau_emp, 0x7f, sizeof(float) * (size_t)h->table_rows, s));
  }
  alloc(h->rho, (size_t)C);
  alloc(h->rho32, (size_t)C);
  if (policy == LIPCACHE_POLICY_INTERCLASS && h->size > 0) {
    // column slice: C x wcol FP64 accumulators (plus C counts) within 220 KB
    int wcol = (int)((220 * 1024 - 8 * (size_t)C) / (8 * (size_t)C));
    wcol = wcol >= dpad ? dpad : (wcol / 8) * 8;
    LC_REQUIRE(wcol >= 8, LIPCACHE_E_INVALID, "too many classes for the class-centroid kernel");
    const int slices = (dpad + wcol - 1) / wcol;
    const int nb = h->num_sms;
    const int64_t chunk = (h->size + nb - 1) / nb;
    if (h->cls_blocks < nb) {
      if (h->cls_sum) cudaFree(h->cls_sum);
      if (h->cls_cnt) cudaFree(h->cls_cnt);
      h->cls_sum = nullptr;
      h->cls_cnt = nullptr;
      h->cls_blocks = 0;
      alloc(h->cls_sum, (size_t)(nb + 1) * C * dpad);
      alloc(h->cls_cnt, (size_t)(nb + 1) * C);
      h->cls_blocks = nb;
    }
    const size_t smem = sizeof(double) * ((size_t)C * wcol + C);
    LC_CUDA(cudaFuncSetAttribute(k_class_partial, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
    const int threads = (wcol + 31) / 32 * 32;
    k_class_partial<<<dim3(nb, slices), threads, smem, s>>>(h->table.keys, h->table.label, h->size, dpad, C, wcol,
                                                            chunk, h->cls_sum, h->cls_cnt);
    LC_LAUNCH_CHECK("k_class_partial");
    k_class_centroid<<<C, 128, 0, s>>>(h->cls_sum, h->cls_cnt, nb, C, dpad);
    LC_LAUNCH_CHECK("k_class_centroid");
    k_class_rho<<<C, kRhoThreads, 0, s>>>(h->cls_sum + (size_t)nb * C * dpad, h->cls_cnt + (size_t)nb * C, C, dpad,
                                          param, h->rho, h->rho32);
    LC_LAUNCH_CHECK("k_class_rho");
  } else {
    // GLOBAL: every class gets tau; INTERCLASS on an empty cache: 0
    const double v = policy == LIPCACHE_POLICY_GLOBAL ? param : 0.0;
    double* tmp = nullptr;
    LC_CUDA(cudaMallocHost(&tmp, sizeof(double) * C));
    for (int c = 0; c < C; ++c) tmp[c] = v;
    cudaError_t e = cudaMemcpyAsync(h->rho, tmp, sizeof(double) * C, cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    cudaFreeHost(tmp);
    LC_CUDA(e);
    float* t32 = nullptr;
    LC_CUDA(cudaMallocHost(&t32, sizeof(float) * C));
    float v32 = (float)v;
    if ((double)v32 > v) v32 = std::nextafter(v32, 0.0f);  // round down
    for (int c = 0; c < C; ++c) t32[c] = v32;
    e = cudaMemcpyAsync(h->rho32, t32, sizeof(float) * C, cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    cudaFreeHost(t32);
    LC_CUDA(e);
  }
  h->policy = policy;
  h->policy_param = param;
  policy_fill(h, 0, h->size, s);
  if (rho_host) {
    LC_CUDA(cudaMemcpyAsync(rho_host, h->rho, sizeof(double) * C, cudaMemcpyDeviceToHost, s));
  }
  LC_CUDA(cudaStreamSynchronize(s));
}

void policy_fill(lipcache* h, int64_t first, int64_t n, cudaStream_t s) {
  if (h->policy == LIPCACHE_POLICY_CERTIFIED || n <= 0) return;
  float p32 = (float)h->policy_param;
  if ((double)p32 > h->policy_param) p32 = std::nextafter(p32, 0.0f);
  k_policy_fill<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(h->table.kn + first, h->table.label + first, n, h->C,
                                                            h->policy, p32, h->rho32, thresh_consts(h->dpad),
                                                            h->rr_emp + first, h->tau_emp + first);
  LC_LAUNCH_CHECK("k_policy_fill");
}

}  // namespace lc
