// Selection strategies S of Algorithm 1 (Sec. 5.5): radius-prioritised
// de-duplication (the paper's default) and K-center per class (at the end
// of the file).
//
// The candidates that Algorithm 1 accepts are visited in order of decreasing
// certified radius (the FP32 radius, ties to the lower row). A candidate is
// kept unless the lookup of Eq. 13 would already hit it -- it lies strictly
// inside the ball of an entry in the cache, whether there before the call or
// kept earlier in it -- or its class (payload label in [0, C)) or the call
// has used its budget. Kept entries are appended in visiting order.
//
// GPU schedule. The order is a bitonic sort of 64-bit keys (radius bits
// descending, row ascending). Candidates are then processed in chunks of
// kSelChunk in that order: the chunk is probed against the cache as it stands
// (a hit = covered by an earlier entry), its pairwise coverage by earlier
// members of the same chunk is computed as a bit matrix (canonical FP32
// distance against the member's acceptance threshold rr, the probe's test),
// one warp resolves the chunk sequentially, and the kept members are
// appended. Coverage uses the probe's conservative thresholds, so a skipped
// candidate is always exactly covered; pairs within ~2e-6 relative of a
// radius may be judged "not covered" where exact arithmetic says "covered".
#include "internal.cuh"
#include "probe_common.cuh"

namespace lc {
namespace {

constexpr int kSelChunk = 4096;
constexpr int kSelWords = kSelChunk / 32;

// Sort key: radius descending, row ascending; rejected rows last.
__global__ void k_sel_keys(const uint8_t* __restrict__ accept, const float* __restrict__ radius, int64_t n,
                           int64_t npow, unsigned long long* __restrict__ keys, int64_t* __restrict__ n_acc) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= npow) return;
  unsigned long long k = ~0ull;
  bool acc = false;
  if (i < n && accept[i]) {
    acc = true;
    k = ((unsigned long long)(0xFFFFFFFFu - __float_as_uint(radius[i])) << 32) | (unsigned long long)(uint32_t)i;
  }
  keys[i] = k;
  const unsigned m = __ballot_sync(0xffffffffu, acc);
  if ((threadIdx.x & 31) == 0 && m) atomicAdd(reinterpret_cast<unsigned long long*>(n_acc), (unsigned long long)__popc(m));
}

// One compare-exchange pass of a bitonic sort (ascending) of npow keys.
__global__ void k_bitonic(unsigned long long* __restrict__ a, int64_t npow, int64_t j, int64_t k) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= npow) return;
  const int64_t x = i ^ j;
  if (x > i) {
    const unsigned long long ai = a[i], ax = a[x];
    const bool up = (i & k) == 0;
    if ((ai > ax) == up) {
      a[i] = ax;
      a[x] = ai;
    }
  }
}

// Chunk members: rows in visiting order and their features (kc x d).
__global__ void k_sel_gather(const unsigned long long* __restrict__ keys, int64_t c0, int kc, const float* __restrict__ H,
                             int d, int32_t* __restrict__ rows, float* __restrict__ G) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int p = blockIdx.x * 8 + warp;
  if (p >= kc) return;
  const int64_t row = (int64_t)(keys[c0 + p] & 0xFFFFFFFFull);
  if (lane == 0) rows[p] = (int32_t)row;
  for (int j = lane; j < d; j += 32) G[(size_t)p * d + j] = H[(size_t)row * d + j];
}

// Coverage inside the chunk: bit i of cov[j * kSelWords + i / 32] is set iff
// i < j and member j lies inside member i's ball (canonical FP32 squared
// distance below rr of member i). Block (ti, tj) computes the 32 x 32 tile of
// members i in tile ti, j in tile tj (ti <= tj); warp w handles j = 4w..4w+3
// of the tile, lane = i; the d features stream through shared memory in
// 32-float chunks, which is the canonical summation order.
__global__ void __launch_bounds__(256) k_sel_cover(const float* __restrict__ G, int d, int kc,
                                                   const int32_t* __restrict__ rows, const float* __restrict__ rr,
                                                   uint32_t* __restrict__ cov) {
  const int ti = blockIdx.x, tj = blockIdx.y;
  if (ti > tj) return;
  __shared__ float zi[32][33], zj[32][33];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int i = ti * 32 + lane;
  float total[4] = {0.f, 0.f, 0.f, 0.f};
  for (int c = 0; c < d; c += 32) {
    for (int e = threadIdx.x; e < 32 * 32; e += 256) {
      const int r = e >> 5, f = e & 31;
      const int gi = ti * 32 + r, gj = tj * 32 + r;
      zi[r][f] = (gi < kc && c + f < d) ? G[(size_t)gi * d + c + f] : 0.f;
      zj[r][f] = (gj < kc && c + f < d) ? G[(size_t)gj * d + c + f] : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int jl = warp * 4 + q;
      float p = 0.f;
#pragma unroll
      for (int f = 0; f < 32; ++f) {
        const float e = __fsub_rn(zj[jl][f], zi[lane][f]);
        p = __fmaf_rn(e, e, p);
      }
      total[q] = __fadd_rn(total[q], p);
    }
    __syncthreads();
  }
  const float thr = i < kc ? rr[rows[i]] : 0.f;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int j = tj * 32 + warp * 4 + q;
    const bool bit = i < kc && j < kc && i < j && total[q] < thr;
    const unsigned m = __ballot_sync(0xffffffffu, bit);
    if (lane == 0 && j < kc) cov[(size_t)j * kSelWords + ti] = m;
  }
}

struct ResolveArgs {
  const uint32_t* cov;
  const int32_t* rows;
  const int64_t* hit;      // per member: cache index it hits, -1 if none
  const int32_t* label;    // per row (certify scratch)
  int32_t* class_cnt;      // per class, kept in this call
  int64_t* kept_total;     // kept in this call
  int32_t* list;           // kept members in order
  int32_t* n_list;
  int kc, C, budget_pc;
  int64_t budget_total;
};

// One warp walks the chunk in order; member j is kept iff it hits nothing in
// the cache, no kept member i < j of the chunk covers it and its budgets
// allow. Lane l holds the kept-set words l, l + 32, l + 64, l + 96. The
// members' hit flags and labels are staged in shared memory first, and the
// coverage rows are read kAhead members ahead of the decision.
constexpr int kAhead = 8;

__device__ __forceinline__ void load_cov_row(const uint32_t* __restrict__ cov, int j, int kc, int lane,
                                             uint32_t (&w)[kSelWords / 32]) {
#pragma unroll
  for (int t = 0; t < kSelWords / 32; ++t) {
    const int wi = lane + 32 * t;
    w[t] = (j < kc && wi <= (j >> 5)) ? __ldcg(cov + (size_t)j * kSelWords + wi) : 0u;
  }
}

__global__ void __launch_bounds__(32) k_sel_resolve(ResolveArgs a) {
  __shared__ int32_t lab_s[kSelChunk];
  __shared__ uint8_t free_s[kSelChunk];
  const int lane = threadIdx.x;
  for (int j = lane; j < a.kc; j += 32) {
    lab_s[j] = a.label[a.rows[j]];
    free_s[j] = a.hit[j] < 0 ? 1 : 0;
  }
  __syncwarp();
  uint32_t sel[kSelWords / 32] = {0u, 0u, 0u, 0u};
  uint32_t ring[kAhead][kSelWords / 32];
#pragma unroll
  for (int q = 0; q < kAhead; ++q) load_cov_row(a.cov, q, a.kc, lane, ring[q]);
  int nk = 0;
  int64_t tot = *a.kept_total;
  for (int j0 = 0; j0 < a.kc; j0 += kAhead) {
#pragma unroll
    for (int q = 0; q < kAhead; ++q) {
      const int j = j0 + q;
      const bool open = j < a.kc && !(a.budget_total > 0 && tot >= a.budget_total);
      bool take = open && free_s[j < a.kc ? j : 0] != 0;
      if (take) {
        uint32_t any = 0u;
#pragma unroll
        for (int t = 0; t < kSelWords / 32; ++t) any |= ring[q][t] & sel[t];
        take = !__any_sync(0xffffffffu, any != 0u);
      }
      const int32_t lab = lab_s[j < a.kc ? j : 0];
      const bool in_cls = a.budget_pc > 0 && lab >= 0 && lab < a.C;
      if (take && in_cls) take = a.class_cnt[lab] < a.budget_pc;
      if (take) {
        const int w = j >> 5;
        if (lane == (w & 31)) {
#pragma unroll
          for (int t = 0; t < kSelWords / 32; ++t)
            if (t == (w >> 5)) sel[t] |= 1u << (j & 31);
        }
        if (lane == 0) {
          a.list[nk] = j;
          if (in_cls) a.class_cnt[lab] += 1;
        }
        ++nk;
        ++tot;
      }
      __syncwarp();
      load_cov_row(a.cov, j + kAhead, a.kc, lane, ring[q]);  // the slot of j now holds j + kAhead
    }
  }
  if (lane == 0) {
    *a.n_list = nk;
    *a.kept_total = tot;
  }
}

struct SelScatterArgs {
  const int32_t* list;
  const int32_t* n_list;
  const int32_t* rows;
  const float* G;
  int d, dpad;
  int64_t size0;
  const float* rr;
  const float* tau;
  const float* kn;
  const float* radius;
  const int32_t* label;
  const int32_t* yG;
  Table t;
  int64_t* out_index;
};

// Append the kept members in order; one warp per member.
__global__ void k_sel_scatter(SelScatterArgs a) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int q = blockIdx.x * 8 + warp;
  if (q >= *a.n_list) return;
  const int p = a.list[q];
  const int32_t row = a.rows[p];
  const int64_t dst = a.size0 + q;
  float* kd = a.t.keys + (size_t)dst * a.dpad;
  for (int j = lane; j < a.dpad; j += 32) kd[j] = j < a.d ? a.G[(size_t)p * a.d + j] : 0.f;
  if (lane == 0) {
    a.t.rr[dst] = a.rr[row];
    a.t.tau[dst] = a.tau[row];
    a.t.kn[dst] = a.kn[row];
    a.t.radius[dst] = a.radius[row];
    a.t.label[dst] = a.label[row];
    a.t.yG[dst] = a.yG[row];
    if (a.out_index) a.out_index[row] = dst;
  }
}

__global__ void k_fill_i64(int64_t* __restrict__ p, int64_t n, int64_t v) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) p[i] = v;
}
__global__ void k_copy_f32(const float* __restrict__ s, float* __restrict__ d, int64_t n) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) d[i] = s[i];
}

// ---------------------------------------------------------------- K-center
// Per class (payload label in [0, C)) among the certified candidates:
// Gonzalez's farthest-point greedy, first centre the largest radius, ties to
// the lower row, at most budget_per_class centres. The candidates are sorted
// by (label, row); one block per class walks its segment once per centre
// (cost: centres x class size x d). Distances are the canonical FP32 squared
// distance, so near-ties (~1e-6 relative) may resolve differently from an
// FP64 evaluation.
// Sort key of the per-class K-center: label, then row; others last.
__global__ void k_kc_keys(const uint8_t* __restrict__ accept, const int32_t* __restrict__ label, int64_t n,
                          int64_t npow, int C, unsigned long long* __restrict__ keys, int64_t* __restrict__ n_acc) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= npow) return;
  unsigned long long k = ~0ull;
  bool in = false;
  if (i < n && accept[i] && label[i] >= 0 && label[i] < C) {
    in = true;
    k = ((unsigned long long)(uint32_t)label[i] << 32) | (unsigned long long)(uint32_t)i;
  }
  keys[i] = k;
  const unsigned m = __ballot_sync(0xffffffffu, in);
  if ((threadIdx.x & 31) == 0 && m) atomicAdd(reinterpret_cast<unsigned long long*>(n_acc), (unsigned long long)__popc(m));
}

// Class segments [seg[2c], seg[2c+1]) of the sorted keys (zero-initialised).
__global__ void k_kc_segments(const unsigned long long* __restrict__ keys, int64_t n_acc, int32_t* __restrict__ seg) {
  const int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (p >= n_acc) return;
  const uint32_t c = (uint32_t)(keys[p] >> 32);
  if (p == 0 || (uint32_t)(keys[p - 1] >> 32) != c) seg[2 * c] = (int32_t)p;
  if (p == n_acc - 1 || (uint32_t)(keys[p + 1] >> 32) != c) seg[2 * c + 1] = (int32_t)(p + 1);
}

constexpr int kKcThreads = 256;

__device__ __forceinline__ unsigned long long block_max_u64(unsigned long long v, unsigned long long* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const unsigned long long w = __shfl_xor_sync(0xffffffffu, v, o);
    v = w > v ? w : v;
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  unsigned long long m = red[0];
  for (int w = 1; w < kKcThreads / 32; ++w) m = red[w] > m ? red[w] : m;
  return m;
}

// Gonzalez's farthest-point greedy for one class per block: first the
// candidate of largest radius, then repeatedly the one farthest (canonical
// FP32 squared distance) from the centres so far; ties to the lower row.
// mind[p] holds each segment member's squared distance to the nearest centre
// (negative once chosen); the chosen rows go to out[s0 ..] in order.
__global__ void __launch_bounds__(kKcThreads) k_kcenter(const unsigned long long* __restrict__ keys,
                                                        const int32_t* __restrict__ seg, const float* __restrict__ H,
                                                        int d, const float* __restrict__ radius, int budget,
                                                        float* __restrict__ mind, int32_t* __restrict__ out,
                                                        int32_t* __restrict__ cnt) {
  extern __shared__ float zc[];  // the newest centre's features (d)
  __shared__ unsigned long long red[kKcThreads / 32];
  const int c = blockIdx.x, tid = threadIdx.x;
  const int s0 = seg[2 * c], s1 = seg[2 * c + 1];
  const int nc = s1 - s0;
  if (nc <= 0) {
    if (tid == 0) cnt[c] = 0;
    return;
  }
  unsigned long long best = 0ull;
  for (int p = s0 + tid; p < s1; p += kKcThreads) {
    const uint32_t row = (uint32_t)(keys[p] & 0xFFFFFFFFull);
    const unsigned long long k = ((unsigned long long)__float_as_uint(radius[row]) << 32) | (0xFFFFFFFFu - row);
    best = k > best ? k : best;
    mind[p] = INFINITY;
  }
  best = block_max_u64(best, red);
  const int want = budget < nc ? budget : nc;
  for (int t = 0; t < want; ++t) {
    const uint32_t row = 0xFFFFFFFFu - (uint32_t)(best & 0xFFFFFFFFull);
    if (tid == 0) out[s0 + t] = (int32_t)row;
    for (int j = tid; j < d; j += kKcThreads) zc[j] = H[(size_t)row * d + j];
    __syncthreads();
    if (t + 1 == want) break;
    best = 0ull;
    for (int p = s0 + tid; p < s1; p += kKcThreads) {
      const uint32_t r = (uint32_t)(keys[p] & 0xFFFFFFFFull);
      float m = mind[p];
      if (r == row) m = -1.f;  // chosen
      if (m >= 0.f) {
        const float* z = H + (size_t)r * d;
        float total = 0.f;
        for (int c0 = 0; c0 < d; c0 += 32) {
          float q = 0.f;
          const int ce = c0 + 32 < d ? c0 + 32 : d;
          for (int j = c0; j < ce; ++j) {
            const float e = __fsub_rn(z[j], zc[j]);
            q = __fmaf_rn(e, e, q);
          }
          total = __fadd_rn(total, q);
        }
        m = fminf(m, total);
        const unsigned long long k = ((unsigned long long)__float_as_uint(m) << 32) | (0xFFFFFFFFu - r);
        best = k > best ? k : best;
      }
      mind[p] = m;
    }
    best = block_max_u64(best, red);
  }
  if (tid == 0) cnt[c] = want;
}

// Append the centres class by class (offsets = exclusive scan of cnt).
__global__ void k_kc_scatter(const int32_t* __restrict__ seg, const int32_t* __restrict__ cnt,
                             const int32_t* __restrict__ off, const int32_t* __restrict__ out, const float* __restrict__ H,
                             int d, int dpad, int64_t size0, const float* __restrict__ rr, const float* __restrict__ tau,
                             const float* __restrict__ kn, const float* __restrict__ radius,
                             const int32_t* __restrict__ label, const int32_t* __restrict__ yG, Table t,
                             int64_t* __restrict__ out_index) {
  const int c = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int q = blockIdx.x * 8 + warp; q < cnt[c]; q += gridDim.x * 8) {
    const int32_t row = out[seg[2 * c] + q];
    const int64_t dst = size0 + off[c] + q;
    float* kd = t.keys + (size_t)dst * dpad;
    for (int j = lane; j < dpad; j += 32) kd[j] = j < d ? H[(size_t)row * d + j] : 0.f;
    if (lane == 0) {
      t.rr[dst] = rr[row];
      t.tau[dst] = tau[row];
      t.kn[dst] = kn[row];
      t.radius[dst] = radius[row];
      t.label[dst] = label[row];
      t.yG[dst] = yG[row];
      if (out_index) out_index[row] = dst;
    }
  }
}

// Exclusive scan of C counts (C <= 1024), total in *total.
__global__ void __launch_bounds__(1024) k_kc_scan(const int32_t* __restrict__ cnt, int C, int32_t* __restrict__ off,
                                                  int64_t* __restrict__ total) {
  __shared__ int32_t buf[1024];
  const int t = threadIdx.x;
  const int v = t < C ? cnt[t] : 0;
  buf[t] = v;
  __syncthreads();
  for (int s = 1; s < 1024; s <<= 1) {
    const int x = t >= s ? buf[t - s] : 0;
    __syncthreads();
    buf[t] += x;
    __syncthreads();
  }
  if (t < C) off[t] = buf[t] - v;
  if (t == 1023) *total = buf[1023];
}

template <typename T>
void grow_to(T*& p, int64_t& cap, int64_t n) {
  if (n <= cap) return;
  if (p) cudaFree(p);
  p = nullptr;
  cap = 0;
  LC_CUDA(cudaMalloc(&p, sizeof(T) * (size_t)n));
  cap = n;
}

}  // namespace

int64_t select_insert(lipcache* h, const float* H, int64_t n, const int32_t* payload, int require_consistency,
                      int64_t budget_total, int budget_per_class, int64_t* out_index, float* out_radius,
                      cudaStream_t s) {
  SelectScratch& x = h->sel;
  certify_rows(h, H, n, payload, require_consistency, s);
  require_certify_ok(h, s);
  const unsigned nb = (unsigned)((n + 255) / 256);
  if (out_index) {
    k_fill_i64<<<nb, 256, 0, s>>>(out_index, n, -1);
    LC_LAUNCH_CHECK("k_fill_i64");
  }
  if (out_radius) {
    k_copy_f32<<<nb, 256, 0, s>>>(h->ins_radius, out_radius, n);
    LC_LAUNCH_CHECK("k_copy_f32");
  }
  // visiting order
  int64_t npow = 1;
  while (npow < n) npow <<= 1;
  grow_to(x.keys, x.keys_cap, npow);
  if (!x.small) {
    LC_CUDA(cudaMalloc(&x.small, sizeof(int64_t) * 4));
    LC_CUDA(cudaMallocHost(&x.small_host, sizeof(int64_t) * 4));
  }
  LC_CUDA(cudaMemsetAsync(x.small, 0, sizeof(int64_t) * 4, s));  // [0] accepted, [1] kept, [2] chunk count
  const unsigned npb = (unsigned)((npow + 255) / 256);
  k_sel_keys<<<npb, 256, 0, s>>>(h->ins_accept, h->ins_radius, n, npow, x.keys, x.small);
  LC_LAUNCH_CHECK("k_sel_keys");
  for (int64_t k = 2; k <= npow; k <<= 1)
    for (int64_t j = k >> 1; j > 0; j >>= 1) {
      k_bitonic<<<npb, 256, 0, s>>>(x.keys, npow, j, k);
      LC_LAUNCH_CHECK("k_bitonic");
    }
  LC_CUDA(cudaMemcpyAsync(x.small_host, x.small, sizeof(int64_t), cudaMemcpyDeviceToHost, s));
  LC_CUDA(cudaStreamSynchronize(s));
  const int64_t n_acc = x.small_host[0];

  // chunk scratch
  grow_to(x.G, x.G_cap, (int64_t)kSelChunk * h->d);
  grow_to(x.rows, x.rows_cap, kSelChunk);
  grow_to(x.hit, x.hit_cap, kSelChunk);
  grow_to(x.cov, x.cov_cap, (int64_t)kSelChunk * kSelWords);
  grow_to(x.list, x.list_cap, kSelChunk + 1);
  grow_to(x.class_cnt, x.class_cap, h->C);
  LC_CUDA(cudaMemsetAsync(x.class_cnt, 0, sizeof(int32_t) * h->C, s));

  int64_t kept = 0;
  for (int64_t c0 = 0; c0 < n_acc; c0 += kSelChunk) {
    if (budget_total > 0 && kept >= budget_total) break;
    const int kc = (int)(n_acc - c0 < kSelChunk ? n_acc - c0 : kSelChunk);
    k_sel_gather<<<(unsigned)((kc + 7) / 8), 256, 0, s>>>(x.keys, c0, kc, H, h->d, x.rows, x.G);
    LC_LAUNCH_CHECK("k_sel_gather");
    probe(h, x.G, kc, x.hit, nullptr, nullptr, s);
    const int tiles = (kc + 31) / 32;
    k_sel_cover<<<dim3((unsigned)tiles, (unsigned)tiles), 256, 0, s>>>(x.G, h->d, kc, x.rows, h->ins_rr, x.cov);
    LC_LAUNCH_CHECK("k_sel_cover");
    ResolveArgs ra;
    ra.cov = x.cov;
    ra.rows = x.rows;
    ra.hit = x.hit;
    ra.label = h->ins_label;
    ra.class_cnt = x.class_cnt;
    ra.kept_total = x.small + 1;
    ra.list = x.list;
    ra.n_list = reinterpret_cast<int32_t*>(x.small + 2);
    ra.kc = kc;
    ra.C = h->C;
    ra.budget_pc = budget_per_class;
    ra.budget_total = budget_total;
    k_sel_resolve<<<1, 32, 0, s>>>(ra);
    LC_LAUNCH_CHECK("k_sel_resolve");
    SelScatterArgs sa;
    sa.list = x.list;
    sa.n_list = ra.n_list;
    sa.rows = x.rows;
    sa.G = x.G;
    sa.d = h->d;
    sa.dpad = h->dpad;
    sa.size0 = h->size;
    sa.rr = h->ins_rr;
    sa.tau = h->ins_tau;
    sa.kn = h->ins_kn;
    sa.radius = h->ins_radius;
    sa.label = h->ins_label;
    sa.yG = h->ins_yG;
    sa.t = h->table;
    sa.out_index = out_index;
    k_sel_scatter<<<(unsigned)((kc + 7) / 8), 256, 0, s>>>(sa);
    LC_LAUNCH_CHECK("k_sel_scatter");
    LC_CUDA(cudaMemcpyAsync(x.small_host + 2, x.small + 2, sizeof(int64_t), cudaMemcpyDeviceToHost, s));
    LC_CUDA(cudaStreamSynchronize(s));
    const int64_t got = (int64_t)(int32_t)(x.small_host[2] & 0xFFFFFFFFll);
    h->size += got;
    kept += got;
  }
  store_size_dev(h, s);  // the table grew from the host
  return kept;
}

int64_t select_kcenter(lipcache* h, const float* H, int64_t n, const int32_t* payload, int require_consistency,
                       int budget_per_class, int64_t* out_index, float* out_radius, cudaStream_t s) {
  SelectScratch& x = h->sel;
  const int C = h->C;
  certify_rows(h, H, n, payload, require_consistency, s);
  require_certify_ok(h, s);
  const unsigned nb = (unsigned)((n + 255) / 256);
  if (out_index) {
    k_fill_i64<<<nb, 256, 0, s>>>(out_index, n, -1);
    LC_LAUNCH_CHECK("k_fill_i64");
  }
  if (out_radius) {
    k_copy_f32<<<nb, 256, 0, s>>>(h->ins_radius, out_radius, n);
    LC_LAUNCH_CHECK("k_copy_f32");
  }
  int64_t npow = 1;
  while (npow < n) npow <<= 1;
  grow_to(x.keys, x.keys_cap, npow);
  if (!x.small) {
    LC_CUDA(cudaMalloc(&x.small, sizeof(int64_t) * 4));
    LC_CUDA(cudaMallocHost(&x.small_host, sizeof(int64_t) * 4));
  }
  LC_CUDA(cudaMemsetAsync(x.small, 0, sizeof(int64_t) * 4, s));
  const unsigned npb = (unsigned)((npow + 255) / 256);
  k_kc_keys<<<npb, 256, 0, s>>>(h->ins_accept, h->ins_label, n, npow, C, x.keys, x.small);
  LC_LAUNCH_CHECK("k_kc_keys");
  for (int64_t k = 2; k <= npow; k <<= 1)
    for (int64_t j = k >> 1; j > 0; j >>= 1) {
      k_bitonic<<<npb, 256, 0, s>>>(x.keys, npow, j, k);
      LC_LAUNCH_CHECK("k_bitonic");
    }
  LC_CUDA(cudaMemcpyAsync(x.small_host, x.small, sizeof(int64_t), cudaMemcpyDeviceToHost, s));
  LC_CUDA(cudaStreamSynchronize(s));
  const int64_t n_in = x.small_host[0];
  if (n_in == 0) return 0;
  // per-class segments, counts and offsets share one int32 scratch: seg[2C], cnt[C], off[C]
  grow_to(x.list, x.list_cap, 4 * (int64_t)C + 1);
  int32_t* seg = x.list;
  int32_t* cnt = seg + 2 * C;
  int32_t* off = cnt + C;
  LC_CUDA(cudaMemsetAsync(seg, 0, sizeof(int32_t) * 2 * C, s));
  k_kc_segments<<<(unsigned)((n_in + 255) / 256), 256, 0, s>>>(x.keys, n_in, seg);
  LC_LAUNCH_CHECK("k_kc_segments");
  grow_to(x.kc_mind, x.kc_mind_cap, n_in);
  grow_to(x.rows, x.rows_cap, n_in);
  k_kcenter<<<C, kKcThreads, sizeof(float) * (size_t)h->d, s>>>(x.keys, seg, H, h->d, h->ins_radius, budget_per_class,
                                                                x.kc_mind, x.rows, cnt);
  LC_LAUNCH_CHECK("k_kcenter");
  k_kc_scan<<<1, 1024, 0, s>>>(cnt, C, off, x.small + 1);
  LC_LAUNCH_CHECK("k_kc_scan");
  const int per = budget_per_class;
  k_kc_scatter<<<dim3((unsigned)((per + 7) / 8 < 64 ? (per + 7) / 8 : 64), (unsigned)C), 256, 0, s>>>(
      seg, cnt, off, x.rows, H, h->d, h->dpad, h->size, h->ins_rr, h->ins_tau, h->ins_kn, h->ins_radius,
      h->ins_label, h->ins_yG, h->table, out_index);
  LC_LAUNCH_CHECK("k_kc_scatter");
  LC_CUDA(cudaMemcpyAsync(x.small_host + 1, x.small + 1, sizeof(int64_t), cudaMemcpyDeviceToHost, s));
  LC_CUDA(cudaStreamSynchronize(s));
  const int64_t kept = x.small_host[1];
  h->size += kept;
  store_size_dev(h, s);  // the table grew from the host
  return kept;
}

void release_select(lipcache* h) {
  SelectScratch& x = h->sel;
  cudaFree(x.keys);
  cudaFree(x.G);
  cudaFree(x.rows);
  cudaFree(x.hit);
  cudaFree(x.cov);
  cudaFree(x.list);
  cudaFree(x.class_cnt);
  cudaFree(x.kc_mind);
  cudaFree(x.small);
  if (x.small_host) cudaFreeHost(x.small_host);
  x = SelectScratch{};
}

}  // namespace lc
