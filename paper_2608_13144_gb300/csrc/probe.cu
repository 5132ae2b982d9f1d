// Online certified lookup (Sec. 3.4, Algorithm 2; Eqs. 13-15).
//
//   H(q) = { i : ||q - z_i|| < r_i }          hit set, strict (Eq. 13)
//   i*   = argmin_{i in H(q)} ||q - z_i||     nearest hit, lowest index on ties (Eq. 14)
//   hit -> payload of i*, miss -> fall back to MainNet (Eq. 15)
//
// Acceptance. A pair (q, i) is accepted iff the canonical FP32 squared
// distance S~ (dist2_canonical: direct differences, 32-wide FMA chunks added
// in order) is below rr_i = RZ(r_safe,i^2 (1 - eps_rc)). Since
// |S~ - S| <= gamma_{d_pad/32+33} S < eps_rc S, every accepted pair has an
// exact distance below r_safe,i <= r_i: the GPU never accepts a pair the
// exact rule rejects.
//
// Selection. Each accepted pair is reduced into a per-query 64-bit word
// (bits(S~) << 32 | i) with atomicMin. S~ >= 0, so its IEEE bits order like
// its value, and equal distances resolve to the lowest index.
//
// Kernels: k_prologue (pads the queries, per-query screen constant, clears
// the reduction words), the main kernel (exact: every pair on CUDA cores;
// tensor: tcgen05 screen + recheck, probe_tc.cu), k_finalize (unpacks).
#include "internal.cuh"
#include "probe_common.cuh"

namespace lc {
namespace {
// The kernel LIPCACHE_PROBE_AUTO picks: the tensor path where supported,
// except for batches so small (B N d_pad below 2^24 multiply-adds) that the
// exact kernel's smaller fixed cost wins (measured on GB300: 256 queries x
// 1,024 keys at d = 16 take 8.1 us exact against 11.7 us on tensor cores;
// 256 x 50,000 at d = 64 take 80 against 14 us). Both return the same bits.
int auto_path(const lipcache* h, int64_t B) {
  if (!tensor_path_supported(h->dpad)) return LIPCACHE_PROBE_EXACT;
  const double macs = (double)B * (double)h->size * (double)h->dpad;
  return macs < 16777216.0 ? LIPCACHE_PROBE_EXACT : LIPCACHE_PROBE_TENSOR;
}

constexpr unsigned kFull = 0xffffffffu;

__global__ void __launch_bounds__(256) k_prologue(const float* __restrict__ Q, int64_t B, int d, int dpad,
                                                  int64_t Bpad, float* __restrict__ qpad, float* __restrict__ kappa,
                                                  unsigned long long* __restrict__ best, double one_minus_c,
                                                  DevStats* __restrict__ st) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (blockIdx.x == 0 && threadIdx.x == 0) st->abort_flag = 0;
  const int64_t row = (int64_t)blockIdx.x * 8 + warp;
  if (row >= Bpad) return;
  float part = 0.f;
  float* dst = qpad + (size_t)row * dpad;
  const float* src = Q + (size_t)row * d;
  for (int j = lane; j < dpad; j += 32) {
    const float x = (row < B && j < d) ? src[j] : 0.f;
    dst[j] = x;
    part = fmaf(x, x, part);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(kFull, part, o);
  if (lane == 0) {
    kappa[row] = row < B ? __double2float_rd(one_minus_c * (double)part * 0.5) : INFINITY;
    best[row] = ~0ull;
  }
}

// Exact probe: the canonical FP32 squared distance of every pair.
// CTA tile: 64 queries x 64 keys, 256 threads, 4 x 4 pairs per thread.
constexpr int kEQ = 64, kEK = 64, kES = kEQ + 4;

__global__ void __launch_bounds__(256) k_probe_exact(const float* __restrict__ qpad, int64_t B,
                                                     const float* __restrict__ keys, const float* __restrict__ rr,
                                                     int64_t N, int dpad, unsigned long long* __restrict__ best) {
  __shared__ __align__(16) float qs[32][kES];
  __shared__ __align__(16) float ks[32][kES];
  const int tid = threadIdx.x;
  const int tq = tid >> 4, tk = tid & 15;
  const int64_t q0 = (int64_t)blockIdx.y * kEQ, k0 = (int64_t)blockIdx.x * kEK;
  const int lr = tid & 63, lp = tid >> 6;  // loader: row, 8-float part
  float tot[4][4], p[4][4];
#pragma unroll
  for (int a = 0; a < 4; ++a)
#pragma unroll
    for (int b = 0; b < 4; ++b) tot[a][b] = 0.f;

  for (int c0 = 0; c0 < dpad; c0 += 32) {
    {
      const int64_t qr = q0 + lr, kr = k0 + lr;
      float4 x0 = make_float4(0.f, 0.f, 0.f, 0.f), x1 = x0, y0 = x0, y1 = x0;
      if (qr < B) {
        const float4* src = reinterpret_cast<const float4*>(qpad + (size_t)qr * dpad + c0 + lp * 8);
        x0 = src[0];
        x1 = src[1];
      }
      if (kr < N) {
        const float4* src = reinterpret_cast<const float4*>(keys + (size_t)kr * dpad + c0 + lp * 8);
        y0 = src[0];
        y1 = src[1];
      }
      const int j = lp * 8;
      qs[j + 0][lr] = x0.x; qs[j + 1][lr] = x0.y; qs[j + 2][lr] = x0.z; qs[j + 3][lr] = x0.w;
      qs[j + 4][lr] = x1.x; qs[j + 5][lr] = x1.y; qs[j + 6][lr] = x1.z; qs[j + 7][lr] = x1.w;
      ks[j + 0][lr] = y0.x; ks[j + 1][lr] = y0.y; ks[j + 2][lr] = y0.z; ks[j + 3][lr] = y0.w;
      ks[j + 4][lr] = y1.x; ks[j + 5][lr] = y1.y; ks[j + 6][lr] = y1.z; ks[j + 7][lr] = y1.w;
    }
    __syncthreads();
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
      for (int b = 0; b < 4; ++b) p[a][b] = 0.f;
#pragma unroll 8
    for (int j = 0; j < 32; ++j) {
      const float4 qv = *reinterpret_cast<const float4*>(&qs[j][tq * 4]);
      const float4 kv = *reinterpret_cast<const float4*>(&ks[j][tk * 4]);
      const float qa[4] = {qv.x, qv.y, qv.z, qv.w};
      const float kb[4] = {kv.x, kv.y, kv.z, kv.w};
#pragma unroll
      for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int b = 0; b < 4; ++b) {
          const float e = __fsub_rn(qa[a], kb[b]);
          p[a][b] = __fmaf_rn(e, e, p[a][b]);
        }
    }
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
      for (int b = 0; b < 4; ++b) tot[a][b] = __fadd_rn(tot[a][b], p[a][b]);
    __syncthreads();
  }
#pragma unroll
  for (int b = 0; b < 4; ++b) {
    const int64_t kr = k0 + tk * 4 + b;
    if (kr >= N) continue;
    const float thr = rr[kr];
#pragma unroll
    for (int a = 0; a < 4; ++a) {
      const int64_t qr = q0 + tq * 4 + a;
      if (qr < B && tot[a][b] < thr) atomicMin(best + qr, pack_hit(tot[a][b], kr));
    }
  }
}

__global__ void k_finalize(const unsigned long long* __restrict__ best, int64_t B, const int32_t* __restrict__ label,
                           int64_t* __restrict__ out_index, int32_t* __restrict__ out_label,
                           float* __restrict__ out_dist, const DevStats* __restrict__ st) {
  const int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (q >= B) return;
  unsigned long long v = best[q];
  if (st->abort_flag) v = ~0ull;
  if (v == ~0ull) {
    out_index[q] = -1;
    if (out_label) out_label[q] = -1;
    if (out_dist) out_dist[q] = INFINITY;
  } else {
    const int64_t i = (int64_t)(v & 0xffffffffull);
    out_index[q] = i;
    if (out_label) out_label[q] = label[i];
    if (out_dist) out_dist[q] = sqrtf(__uint_as_float((unsigned)(v >> 32)));
  }
}

void ensure_probe_scratch(lipcache* h, int64_t Bpad) {
  if (Bpad <= h->q_cap) return;
  int64_t cap = h->q_cap ? h->q_cap : 1024;
  while (cap < Bpad) cap *= 2;
  if (h->qpad) cudaFree(h->qpad);
  if (h->kappa) cudaFree(h->kappa);
  if (h->best) cudaFree(h->best);
  h->qpad = nullptr;
  h->kappa = nullptr;
  h->best = nullptr;
  h->q_cap = 0;
  LC_CUDA(cudaMalloc(&h->qpad, sizeof(float) * (size_t)cap * h->dpad));
  LC_CUDA(cudaMalloc(&h->kappa, sizeof(float) * (size_t)cap));
  LC_CUDA(cudaMalloc(&h->best, sizeof(unsigned long long) * (size_t)cap));
  h->q_cap = cap;
}

}  // namespace

bool tensor_path_supported(int dpad) { return dpad <= 256; }

void reserve_probe(lipcache* h, int64_t max_batch) {
  ensure_probe_scratch(h, (max_batch + 127) / 128 * 128);
}

// The small kernels around the tensor probe prefer the same shared-memory
// carveout as the probe itself, so that the SM does not switch its L1 /
// shared-memory split between the three launches of a probe.
void set_probe_carveout(lipcache* h) {
  if (h->probe_carveout_set) return;
  LC_CUDA(cudaFuncSetAttribute(k_prologue, cudaFuncAttributePreferredSharedMemoryCarveout,
                               (int)cudaSharedmemCarveoutMaxShared));
  LC_CUDA(cudaFuncSetAttribute(k_finalize, cudaFuncAttributePreferredSharedMemoryCarveout,
                               (int)cudaSharedmemCarveoutMaxShared));
  h->probe_carveout_set = true;
}

void probe(lipcache* h, const float* Q, int64_t B, int64_t* out_index, int32_t* out_label, float* out_dist,
           cudaStream_t s) {
  const int64_t Bpad = (B + 127) / 128 * 128;
  ensure_probe_scratch(h, Bpad);
  set_probe_carveout(h);
  k_prologue<<<(unsigned)((Bpad + 7) / 8), 256, 0, s>>>(Q, B, h->d, h->dpad, Bpad, h->qpad, h->kappa, h->best,
                                                      1.0 - h->c_scr, h->stats);
  LC_LAUNCH_CHECK("k_prologue");
  int path = h->probe_path;
  if (path == LIPCACHE_PROBE_AUTO) path = auto_path(h, B);
  h->last_probe_path = path;
  if (h->size > 0) {
    int slot = -1;
    if (h->timing) {
      if (h->t_issued - h->t_harvested >= lipcache::kTimingRing) harvest_timing(h, false);
      slot = (int)(h->t_issued % lipcache::kTimingRing);
      h->t_kind[slot] = 0;
    }
    if (path != LIPCACHE_PROBE_EXACT) {
      // the start event is recorded by the launcher, after its host-side
      // preparation, right before the kernel
      h->launch_event = slot >= 0 ? h->tev0[slot] : nullptr;
      h->last_probe_path = launch_probe_tc(h, B, path, s);
      h->launch_event = nullptr;
    } else {
      if (slot >= 0) LC_CUDA(cudaEventRecord(h->tev0[slot], s));
      dim3 grid((unsigned)((h->size + kEK - 1) / kEK), (unsigned)((B + kEQ - 1) / kEQ));
      h->last_grid = (int)(grid.x * grid.y);
      h->last_cluster = 1;
      k_probe_exact<<<grid, 256, 0, s>>>(h->qpad, B, h->table.keys, h->probe_rr(), h->size, h->dpad, h->best);
      LC_LAUNCH_CHECK("k_probe_exact");
    }
    if (slot >= 0) {
      LC_CUDA(cudaEventRecord(h->tev1[slot], s));
      ++h->t_issued;
    }
  }
  k_finalize<<<(unsigned)((B + 255) / 256), 256, 0, s>>>(h->best, B, h->table.label, out_index, out_label, out_dist,
                                                       h->stats);
  LC_LAUNCH_CHECK("k_finalize");
}

// The same launch sequence as probe(), on scratch memory the caller
// provides (qpad: Bpad x d_pad floats, kappa: Bpad floats, best: Bpad words,
// Bpad = B rounded up to 128). Allocates nothing.
void probe_external_scratch(lipcache* h, const float* Q, int64_t B, int64_t* out_index, int32_t* out_label,
                            float* out_dist, float* qpad, float* kappa, unsigned long long* best, cudaStream_t s) {
  const int64_t Bpad = (B + 127) / 128 * 128;
  set_probe_carveout(h);
  k_prologue<<<(unsigned)((Bpad + 7) / 8), 256, 0, s>>>(Q, B, h->d, h->dpad, Bpad, qpad, kappa, best,
                                                      1.0 - h->c_scr, h->stats);
  LC_LAUNCH_CHECK("k_prologue");
  int path = h->probe_path;
  if (path == LIPCACHE_PROBE_AUTO) path = auto_path(h, B);
  h->last_probe_path = path;
  if (h->size > 0) {
    if (path != LIPCACHE_PROBE_EXACT) {
      h->last_probe_path = launch_probe_tc_external(h, B, path, qpad, kappa, best, s);
    } else {
      dim3 grid((unsigned)((h->size + kEK - 1) / kEK), (unsigned)((B + kEQ - 1) / kEQ));
      k_probe_exact<<<grid, 256, 0, s>>>(qpad, B, h->table.keys, h->probe_rr(), h->size, h->dpad, best);
      LC_LAUNCH_CHECK("k_probe_exact");
    }
  }
  k_finalize<<<(unsigned)((B + 255) / 256), 256, 0, s>>>(best, B, h->table.label, out_index, out_label, out_dist,
                                                       h->stats);
  LC_LAUNCH_CHECK("k_finalize");
}

}  // namespace lc
