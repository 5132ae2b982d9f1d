// Tensor-core probe: screen every (query, key) pair with a TF32 tcgen05
// contraction, recheck the few candidates with the exact canonical FP32
// distance (Sec. 3.4, Algorithm 2, Eqs. 13-15; cost model Eq. 16).
//
// Screen. For a pair with exact squared distance S = |q|^2 + |k|^2 - 2 q.k,
// the tensor cores return a = q.k up to |a - q.k| <= c |q| |k| <= c (|q|^2 +
// |k|^2) / 2 (TF32 operands, FP32 accumulation; c = c_screen). Every pair the
// recheck can accept has S < R_k = rr_k / (1 - gamma_rc), hence
//     a > (1 - c) |q|^2 / 2 + ((1 - c) |k|^2 - R_k) / 2 = kappa_q + tau_k,
// with kappa_q (per query, k_prologue) rounded down and tau_k (per key,
// stored at insertion) rounded down. The epilogue keeps a pair iff
// fl(a - tau_k) >= kappa_q, which therefore never drops an acceptable pair;
// the separable form costs one subtraction and one max per pair.
//
// Schedule (one persistent CTA per SM, 320 threads):
//   warp 0     TMA producer: the CTA's key tile (BN keys x d_pad, resident,
//              one barrier pair per 32-float chunk so the next tile streams in
//              while the last query tile still runs) and the query tiles
//              (128 queries x 32 floats per stage, 4-stage ring);
//   warp 1     allocates TMEM, issues tcgen05.mma kind::tf32 (M=128 queries,
//              N=BN keys, K=8) from one thread into one of two TMEM
//              accumulators;
//   warps 2-9  epilogue: tcgen05.ld of the accumulator (warp w reads TMEM
//              lane quarter w % 4, column half (w - 2) / 4), screen, recheck,
//              atomicMin of the packed (distance, index) word.
// A work unit is one key tile against a group of query tiles; units are
// dealt round-robin over the persistent CTAs.
#include "internal.cuh"
#include "probe_common.cuh"
#include "tc_ptx.cuh"

namespace lc {
int tc_key_tile(int dpad);
namespace {

constexpr int kBM = 128;              // queries per tile (MMA M)
constexpr int kChunkF = 32;           // floats per K chunk (one 128-byte swizzle row)
constexpr int kStages = 4;            // query ring depth
constexpr int kQStageBytes = kBM * 128;
constexpr int kThreads = 320;
constexpr int kEpiWarps = 8;
constexpr long long kWaitLimit = 1LL << 31;  // ~1 s at GB300 clocks

struct TcArgs {
  int nch;       // d_pad / 32
  int dpad;
  int nq;        // query tiles
  int qpg;       // query tiles per unit
  int n_qg;      // query groups
  int n_units;   // key tiles x query groups
  const float* kappa;
  const float* qpad;
  const float* keys;
  const float* tau;
  const float* rr;
  unsigned long long* best;
  DevStats* stats;
};

template <int BN>
struct Layout {
  static constexpr int kKChunkBytes = BN * 128;
  static constexpr int kTmemCols = 2 * BN;
  int nch;
  __device__ __host__ int kbytes() const { return nch * kKChunkBytes; }
  __device__ __host__ int qoff() const { return kbytes(); }
  __device__ __host__ int baroff() const { return qoff() + kStages * kQStageBytes; }
  // barriers: full_k[nch], empty_k[nch], full_q[S], empty_q[S], acc_full[2], acc_empty[2], drain
  __device__ __host__ int nbar() const { return 2 * nch + 2 * kStages + 5; }
  __device__ __host__ int miscoff() const { return baroff() + 8 * nbar(); }
  __device__ __host__ int total() const { return miscoff() + 16; }
};

__device__ __forceinline__ void unit_range(const TcArgs& a, int u, int BN, int& kt, int& qt0, int& qt1) {
  kt = u / a.n_qg;
  const int g = u - kt * a.n_qg;
  qt0 = g * a.qpg;
  qt1 = min(a.nq, qt0 + a.qpg);
  (void)BN;
}

template <int BN>
__global__ void __launch_bounds__(kThreads, 1)
    k_probe_tc(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK, const TcArgs a) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  // 1024-byte alignment of the swizzled tiles
  unsigned char* smem = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  const Layout<BN> L{a.nch};
  const uint32_t s_base = ptx::smem_u32(smem);
  const uint32_t s_k = s_base;
  const uint32_t s_q = s_base + L.qoff();
  const uint32_t s_bar = s_base + L.baroff();
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L.baroff());
  (void)bars;
  const uint32_t full_k = s_bar, empty_k = s_bar + 8 * a.nch;
  const uint32_t full_q = s_bar + 16 * a.nch, empty_q = full_q + 8 * kStages;
  const uint32_t acc_full = empty_q + 8 * kStages, acc_empty = acc_full + 16, drain = acc_empty + 16;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L.miscoff());
  volatile int* abort_s = reinterpret_cast<volatile int*>(smem + L.miscoff() + 4);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int c = 0; c < a.nch; ++c) {
      ptx::mbar_init(full_k + 8 * c, 1);
      ptx::mbar_init(empty_k + 8 * c, 1);
    }
    for (int s = 0; s < kStages; ++s) {
      ptx::mbar_init(full_q + 8 * s, 1);
      ptx::mbar_init(empty_q + 8 * s, 1);
    }
    for (int b = 0; b < 2; ++b) {
      ptx::mbar_init(acc_full + 8 * b, 1);
      ptx::mbar_init(acc_empty + 8 * b, kEpiWarps);
    }
    ptx::mbar_init(drain, 1);
    *abort_s = 0;
    ptx::fence_mbar_init();
    ptx::tma_prefetch_desc(&tmQ);
    ptx::tma_prefetch_desc(&tmK);
  }
  if (warp == 1) {
    ptx::tmem_alloc(ptx::smem_u32(tmem_slot), (uint32_t)Layout<BN>::kTmemCols);
    ptx::tmem_relinquish();
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      int qs = 0;
      uint32_t qph = 0;
      int i = 0;
      int last_unit_par = -1;
      uint32_t last_q_par[kStages];
      bool q_used[kStages];
      for (int s = 0; s < kStages; ++s) {
        q_used[s] = false;
        last_q_par[s] = 0;
      }
      bool ok = true;
      for (int u = blockIdx.x; u < a.n_units && ok; u += gridDim.x, ++i) {
        int kt, qt0, qt1;
        unit_range(a, u, BN, kt, qt0, qt1);
        for (int c = 0; c < a.nch && ok; ++c) {
          ok = ptx::mbar_wait(empty_k + 8 * c, (uint32_t)(i & 1) ^ 1u, abort_s, kWaitLimit);
          if (!ok) break;
          ptx::mbar_expect_tx(full_k + 8 * c, (uint32_t)Layout<BN>::kKChunkBytes);
          ptx::tma_load_2d(s_k + c * Layout<BN>::kKChunkBytes, &tmK, c * kChunkF, kt * BN, full_k + 8 * c);
        }
        if (ok) last_unit_par = i & 1;
        for (int qt = qt0; qt < qt1 && ok; ++qt) {
          for (int c = 0; c < a.nch && ok; ++c) {
            ok = ptx::mbar_wait(empty_q + 8 * qs, qph ^ 1u, abort_s, kWaitLimit);
            if (!ok) break;
            ptx::mbar_expect_tx(full_q + 8 * qs, (uint32_t)kQStageBytes);
            ptx::tma_load_2d(s_q + qs * kQStageBytes, &tmQ, c * kChunkF, qt * kBM, full_q + 8 * qs);
            q_used[qs] = true;
            last_q_par[qs] = qph;
            if (++qs == kStages) {
              qs = 0;
              qph ^= 1u;
            }
          }
        }
      }
      // Let every copy this thread issued land before the CTA can exit.
      // (Bounded; a phase that already completed returns at once.)
      volatile int never = 0;
      for (int s = 0; s < kStages; ++s)
        if (q_used[s]) ptx::mbar_wait(full_q + 8 * s, last_q_par[s], &never, kWaitLimit);
      if (last_unit_par >= 0)
        for (int c = 0; c < a.nch; ++c) ptx::mbar_wait(full_k + 8 * c, (uint32_t)last_unit_par, &never, kWaitLimit);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = ptx::idesc_tf32(kBM, BN);
      int qs = 0;
      uint32_t qph = 0;
      int t = 0, i = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < a.n_units && ok; u += gridDim.x, ++i) {
        int kt, qt0, qt1;
        unit_range(a, u, BN, kt, qt0, qt1);
        for (int qt = qt0; qt < qt1 && ok; ++qt, ++t) {
          const int buf = t & 1;
          ok = ptx::mbar_wait(acc_empty + 8 * buf, (uint32_t)((t >> 1) & 1) ^ 1u, abort_s, kWaitLimit);
          if (!ok) break;
          ptx::tc_fence_after();
          const uint32_t d_tmem = tmem + (uint32_t)(buf * BN);
          for (int c = 0; c < a.nch && ok; ++c) {
            ok = ptx::mbar_wait(full_k + 8 * c, (uint32_t)(i & 1), abort_s, kWaitLimit);
            if (ok) ok = ptx::mbar_wait(full_q + 8 * qs, qph, abort_s, kWaitLimit);
            if (!ok) break;
            ptx::tc_fence_after();
            const uint32_t qa = s_q + qs * kQStageBytes;
            const uint32_t kb = s_k + c * Layout<BN>::kKChunkBytes;
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              ptx::mma_tf32(d_tmem, ptx::sw128_kmajor_desc(qa + kk * 32), ptx::sw128_kmajor_desc(kb + kk * 32), idesc,
                            (c | kk) != 0);
            ptx::mma_commit(empty_q + 8 * qs);
            if (qt == qt1 - 1) ptx::mma_commit(empty_k + 8 * c);
            if (++qs == kStages) {
              qs = 0;
              qph ^= 1u;
            }
          }
          if (ok) ptx::mma_commit(acc_full + 8 * buf);
        }
      }
      // all issued MMAs complete before TMEM can be released
      volatile int never = 0;
      ptx::mma_commit(drain);
      ptx::mbar_wait(drain, 0, &never, kWaitLimit);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ epilogue
    const int ew = warp - 2;
    const int quarter = warp & 3;         // TMEM lane quarter this warp may access
    const int half = ew >> 2;             // column half
    constexpr int kColsPerWarp = BN / 2;
    constexpr int kChunks = kColsPerWarp / 32;
    const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
    int t = 0;
    bool ok = true;
    unsigned long long ncand = 0;
    for (int u = blockIdx.x; u < a.n_units && ok; u += gridDim.x) {
      int kt, qt0, qt1;
      unit_range(a, u, BN, kt, qt0, qt1);
      const int key0 = kt * BN + half * kColsPerWarp;
      const float4* tau4 = reinterpret_cast<const float4*>(a.tau + key0);
      for (int qt = qt0; qt < qt1; ++qt, ++t) {
        const int buf = t & 1;
        ok = ptx::mbar_wait(acc_full + 8 * buf, (uint32_t)((t >> 1) & 1), abort_s, kWaitLimit);
        ok = __all_sync(0xffffffffu, ok);  // warp-uniform before the aligned TMEM loads
        if (!ok) break;
        ptx::tc_fence_after();
        const int row = qt * kBM + quarter * 32 + lane;
        const float kap = __ldg(a.kappa + row);
        const uint32_t tbase = tmem + lane_base + (uint32_t)(buf * BN + half * kColsPerWarp);
        uint32_t r[2][32];
        ptx::tmem_ld32(tbase, r[0]);
        ptx::tmem_wait_ld();
#pragma unroll
        for (int ch = 0; ch < kChunks; ++ch) {
          if (ch + 1 < kChunks) ptx::tmem_ld32(tbase + (uint32_t)((ch + 1) * 32), r[(ch + 1) & 1]);
          const uint32_t* v = r[ch & 1];
          float m = -INFINITY;
          float tv[32];
#pragma unroll
          for (int j4 = 0; j4 < 8; ++j4) {
            const float4 t4 = __ldg(tau4 + ch * 8 + j4);
            tv[4 * j4 + 0] = t4.x;
            tv[4 * j4 + 1] = t4.y;
            tv[4 * j4 + 2] = t4.z;
            tv[4 * j4 + 3] = t4.w;
          }
#pragma unroll
          for (int j = 0; j < 32; ++j) m = fmaxf(m, __uint_as_float(v[j]) - tv[j]);
          if (m >= kap) {
            uint32_t mask = 0;
#pragma unroll
            for (int j = 0; j < 32; ++j) mask |= (uint32_t)(__uint_as_float(v[j]) - tv[j] >= kap) << j;
            const float* qrow = a.qpad + (size_t)row * a.dpad;
            while (mask) {
              const int j = __ffs(mask) - 1;
              mask &= mask - 1;
              const int key = key0 + ch * 32 + j;
              const float d2 = dist2_canonical(qrow, a.keys + (size_t)key * a.dpad, a.dpad);
              ++ncand;
              if (d2 < __ldg(a.rr + key)) atomicMin(a.best + row, pack_hit(d2, key));
            }
          }
          __syncwarp();
          if (ch + 1 < kChunks) ptx::tmem_wait_ld();
        }
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(acc_empty + 8 * buf);
      }
    }
    // candidate count: one atomic per warp
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) ncand += __shfl_xor_sync(0xffffffffu, ncand, o);
    if (lane == 0 && ncand) atomicAdd(&a.stats->candidates, ncand);
  }

  ptx::tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0 && *abort_s) {
    atomicAdd(&a.stats->errors, 1ull);
    atomicExch(&a.stats->abort_flag, 1);
  }
  if (warp == 1) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, (uint32_t)Layout<BN>::kTmemCols);
  }
}

void encode_2d(lipcache* h, CUtensorMap* map, const float* base, uint64_t rows, uint32_t box_rows) {
  LC_REQUIRE(h->encode != nullptr, LIPCACHE_E_CUDA, "cuTensorMapEncodeTiled is unavailable from the driver");
  const cuuint64_t dims[2] = {(cuuint64_t)h->dpad, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)h->dpad * sizeof(float)};
  const cuuint32_t box[2] = {(cuuint32_t)kChunkF, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  const CUresult r = h->encode(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float*>(base), dims, strides, box,
                               estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  LC_REQUIRE(r == CUDA_SUCCESS, LIPCACHE_E_CUDA, "cuTensorMapEncodeTiled failed: " + std::to_string((int)r));
}

template <int BN>
void launch(lipcache* h, int64_t B, cudaStream_t s) {
  const int64_t Bpad = (B + kBM - 1) / kBM * kBM;
  CUtensorMap tmQ, tmK;
  encode_2d(h, &tmQ, h->qpad, (uint64_t)Bpad, kBM);
  encode_2d(h, &tmK, h->table.keys, (uint64_t)h->table_rows, BN);
  TcArgs a;
  a.nch = h->dpad / kChunkF;
  a.dpad = h->dpad;
  a.nq = (int)(Bpad / kBM);
  const int64_t n_kt = (h->size + BN - 1) / BN;
  const int64_t target = 2LL * h->num_sms;
  int n_qg = (int)((target + n_kt - 1) / n_kt);
  if (n_qg < 1) n_qg = 1;
  if (n_qg > a.nq) n_qg = a.nq;
  a.qpg = (a.nq + n_qg - 1) / n_qg;
  a.n_qg = (a.nq + a.qpg - 1) / a.qpg;
  const int64_t n_units = n_kt * a.n_qg;
  LC_REQUIRE(n_units < (1LL << 31), LIPCACHE_E_INVALID, "too many work units");
  a.n_units = (int)n_units;
  a.kappa = h->kappa;
  a.qpad = h->qpad;
  a.keys = h->table.keys;
  a.tau = h->table.tau;
  a.rr = h->table.rr;
  a.best = h->best;
  a.stats = h->stats;
  const Layout<BN> L{a.nch};
  const int smem = L.total() + 1024;
  LC_CUDA(cudaFuncSetAttribute(k_probe_tc<BN>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
  const int grid = (int)(n_units < h->num_sms ? n_units : h->num_sms);
  k_probe_tc<BN><<<grid, kThreads, smem, s>>>(tmQ, tmK, a);
  LC_LAUNCH_CHECK("k_probe_tc");
}

template <int BN>
void launch_external(lipcache* h, int64_t B, const float* qpad, const float* kappa, unsigned long long* best,
                     cudaStream_t s) {
  const int64_t Bpad = (B + kBM - 1) / kBM * kBM;
  CUtensorMap tmQ, tmK;
  encode_2d(h, &tmQ, qpad, (uint64_t)Bpad, kBM);
  encode_2d(h, &tmK, h->table.keys, (uint64_t)h->table_rows, BN);
  TcArgs a;
  a.nch = h->dpad / kChunkF;
  a.dpad = h->dpad;
  a.nq = (int)(Bpad / kBM);
  const int64_t n_kt = (h->size + BN - 1) / BN;
  const int64_t target = 2LL * h->num_sms;
  int n_qg = (int)((target + n_kt - 1) / n_kt);
  if (n_qg < 1) n_qg = 1;
  if (n_qg > a.nq) n_qg = a.nq;
  a.qpg = (a.nq + n_qg - 1) / n_qg;
  a.n_qg = (a.nq + a.qpg - 1) / a.qpg;
  const int64_t n_units = n_kt * a.n_qg;
  LC_REQUIRE(n_units < (1LL << 31), LIPCACHE_E_INVALID, "too many work units");
  a.n_units = (int)n_units;
  a.kappa = kappa;
  a.qpad = qpad;
  a.keys = h->table.keys;
  a.tau = h->table.tau;
  a.rr = h->table.rr;
  a.best = best;
  a.stats = h->stats;
  const Layout<BN> L{a.nch};
  const int smem = L.total() + 1024;
  LC_CUDA(cudaFuncSetAttribute(k_probe_tc<BN>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
  const int grid = (int)(n_units < h->num_sms ? n_units : h->num_sms);
  k_probe_tc<BN><<<grid, kThreads, smem, s>>>(tmQ, tmK, a);
  LC_LAUNCH_CHECK("k_probe_tc");
}

}  // namespace

void launch_probe_tc_external(lipcache* h, int64_t B, const float* qpad, const float* kappa, unsigned long long* best,
                              cudaStream_t s) {
  LC_REQUIRE(tensor_path_supported(h->dpad), LIPCACHE_E_INVALID, "the tensor probe supports d <= 256");
  if (tc_key_tile(h->dpad) == 256)
    launch_external<256>(h, B, qpad, kappa, best, s);
  else
    launch_external<128>(h, B, qpad, kappa, best, s);
}

int tc_key_tile(int dpad) { return dpad <= 128 ? 256 : 128; }

void launch_probe_tc(lipcache* h, int64_t B, cudaStream_t s) {
  LC_REQUIRE(tensor_path_supported(h->dpad), LIPCACHE_E_INVALID, "the tensor probe supports d <= 256");
  if (tc_key_tile(h->dpad) == 256)
    launch<256>(h, B, s);
  else
    launch<128>(h, B, s);
}

}  // namespace lc
