// Tensor-core probe on CTA pairs: the screen + recheck of probe_tc.cu with
// 2-SM tcgen05 MMAs (Sec. 3.4, Algorithm 2, Eqs. 13-15; cost model Eq. 16).
//
// The screen, its bound and the recheck are those of probe_tc.cu; what
// changes is the schedule. At the single-CTA MMA shape (M = 128 queries,
// N = 256 keys) the operand reads plus the query-stage writes fill the SM's
// shared-memory bandwidth, so the epilogue's reads come out of MMA
// throughput. A pair MMA (tcgen05.mma.cta_group::2, M = 256, N = 256) reads
// per CTA only its own 128 queries and its own 128 keys for the same work,
// a third less shared-memory traffic.
//
// Clusters of four CTAs = two pairs. A pair owns one key tile of 256 keys
// (128 resident in each CTA, the B operand halves) and multiplies it by query
// tiles of 256 (128 per CTA, the A operand halves). Both pairs of a cluster
// stream the same query tiles: every CTA TMA-loads one 64-row quarter of its
// half of each query stage and multicasts it to itself and to the CTA at the
// same position of the other pair, so each query byte leaves L2 once per 512
// keys (as in probe_tc.cu). TMA completion bytes of both CTAs of a pair are
// counted on the pair leader's barriers (.cta_group::2).
// Per CTA (320 threads):
//   warp 0     TMA producer (both CTAs): the CTA's key half (one barrier pair
//              per 32-float chunk) and its query quarter of every stage;
//   warp 1     allocates the pair's TMEM (both CTAs); in the leader, one
//              thread issues the pair MMAs into one of two accumulators and
//              releases query stages (all four CTAs), key chunks and
//              accumulators (both CTAs of the pair) with multicast commits;
//   warps 2-9  epilogue (both CTAs): tcgen05.ld of the CTA's 128 accumulator
//              rows, screen, recheck, atomicMin; they hand the accumulator
//              back with an arrival on the leader's barrier.
// Every wait is bounded; a role that gives up raises the CTA's abort flag and
// the batch's queries become misses (counted in device_errors).
#include "internal.cuh"
#include "probe_common.cuh"
#include "tc_ptx.cuh"

namespace lc {
namespace {

constexpr int kBM = 256;              // queries per pair tile (MMA M)
constexpr int kHM = kBM / 2;          // queries per CTA
constexpr int kBN = 256;              // keys per pair tile (MMA N)
constexpr int kHN = kBN / 2;          // keys per CTA
constexpr int kChunkF = 32;           // floats per K chunk (one 128-byte swizzle row)
constexpr int kMaxStages = 8;
constexpr int kMaxChunks = 8;         // d_pad <= 256
constexpr int kQStageBytes = kHM * 128;   // this CTA's 128 query rows of one chunk
constexpr int kQQuarterBytes = kQStageBytes / 2;
constexpr int kKChunkBytes = kHN * 128;   // this CTA's 128 keys of one chunk
constexpr int kEpiWarps = 8;
constexpr int kThreads = 32 * (2 + kEpiWarps);
constexpr int kCluster = 4;
constexpr int kTmemCols = 2 * kBN;
constexpr int kTauBytes = 4 * kBN * 4;    // one private tau slice per epilogue warp
constexpr int kSmemBudget = 227 * 1024 - 1024;
constexpr long long kWaitLimit = 1LL << 31;  // ~1 s at GB300 clocks

struct PairArgs {
  int nst;       // query ring stages
  int nch;       // d_pad / 32
  int dpad;
  int nq;        // query tiles of 256
  int64_t bpad;  // padded query rows (multiple of 128; rows past it are zero-filled by the TMA)
  int qpg;       // query tiles per unit
  int n_qg;      // query groups
  int n_units;   // key-tile quads x query groups
  int n_kt;      // key tiles of 256 holding cache entries
  const float* kappa;
  const float* qpad;
  const float* keys;
  const float* tau;
  const float* rr;
  unsigned long long* best;
  DevStats* stats;
  int debug_stall;  // test hook: the MMA issuer first waits on a barrier nothing arrives on
};

struct PairLayout {
  int nch, nst;
  __device__ __host__ int kbytes() const { return nch * kKChunkBytes; }
  __device__ __host__ int qoff() const { return kbytes(); }
  __device__ __host__ int tauoff() const { return qoff() + nst * kQStageBytes; }
  __device__ __host__ int baroff() const { return tauoff() + kTauBytes; }
  // full_k[nch], empty_k[nch], full_q[nst], empty_q[nst], acc_full[2], acc_empty[2], drain
  __device__ __host__ int nbar() const { return 2 * nch + 2 * nst + 5; }
  __device__ __host__ int miscoff() const { return baroff() + 8 * nbar(); }
  __device__ __host__ int total() const { return miscoff() + 16; }
  static __host__ int stages_for(int nch) {
    for (int n = kMaxStages; n >= 2; --n)
      if (PairLayout{nch, n}.total() <= kSmemBudget) return n;
    return 0;
  }
};

// Unit u -> this pair's key tile and the unit's query-tile range.
__device__ __forceinline__ void unit_range(const PairArgs& a, int u, uint32_t pair, int& kt, int& qt0, int& qt1) {
  const int quad = u / a.n_qg;
  const int g = u - quad * a.n_qg;
  kt = quad * 2 + (int)pair;
  qt0 = g * a.qpg;
  qt1 = min(a.nq, qt0 + a.qpg);
}

__global__ void __launch_bounds__(kThreads, 1)
    k_probe_pair(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK, const PairArgs a) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* smem =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  const PairLayout L{a.nch, a.nst};
  const uint32_t s_base = ptx::smem_u32(smem);
  const uint32_t s_k = s_base;
  const uint32_t s_q = s_base + L.qoff();
  const uint32_t s_bar = s_base + L.baroff();
  const uint32_t full_k = s_bar, empty_k = s_bar + 8 * a.nch;
  const uint32_t full_q = s_bar + 16 * a.nch, empty_q = full_q + 8 * a.nst;
  const uint32_t acc_full = empty_q + 8 * a.nst, acc_empty = acc_full + 16, drain = acc_empty + 16;
  float* tau_s = reinterpret_cast<float*>(smem + L.tauoff());
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L.miscoff());
  volatile int* abort_s = reinterpret_cast<volatile int*>(smem + L.miscoff() + 4);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = ptx::cluster_ctarank();
  const uint32_t pair = rank >> 1, pos = rank & 1, leader = rank & ~1u;
  const uint16_t pair_mask = (uint16_t)(0x3u << (2 * pair));
  const int cluster_id = blockIdx.x / kCluster, n_clusters = gridDim.x / kCluster;

  if (threadIdx.x == 0) {
    for (int c = 0; c < a.nch; ++c) {
      ptx::mbar_init(full_k + 8 * c, 1);   // leader: its own arrival, bytes of both CTAs
      ptx::mbar_init(empty_k + 8 * c, 1);  // one pair commit
    }
    for (int s = 0; s < a.nst; ++s) {
      ptx::mbar_init(full_q + 8 * s, 1);   // leader: its own arrival, bytes of both CTAs
      ptx::mbar_init(empty_q + 8 * s, 2);  // commits of both pairs (the stage feeds both)
    }
    for (int b = 0; b < 2; ++b) {
      ptx::mbar_init(acc_full + 8 * b, 1);              // one pair commit
      ptx::mbar_init(acc_empty + 8 * b, 2 * kEpiWarps); // leader: both CTAs' epilogue warps
    }
    ptx::mbar_init(drain, 1);
    *abort_s = 0;
    ptx::fence_mbar_init();
    ptx::tma_prefetch_desc(&tmQ);
    ptx::tma_prefetch_desc(&tmK);
  }
  if (warp == 1) {
    ptx::tmem_alloc_pair(ptx::smem_u32(tmem_slot), (uint32_t)kTmemCols);
    ptx::tmem_relinquish_pair();
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  ptx::cluster_sync();  // every barrier of the cluster exists before any copy or arrival targets it
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const uint32_t lead_full_k = ptx::mapa(full_k, leader), lead_full_q = ptx::mapa(full_q, leader);
      const uint16_t q_mask = (uint16_t)((1u << rank) | (1u << (rank ^ 2u)));
      int qs = 0;
      uint32_t qph = 0;
      int i = 0;
      bool ok = true;
      for (int u = cluster_id; u < a.n_units && ok; u += n_clusters, ++i) {
        int kt, qt0, qt1;
        unit_range(a, u, pair, kt, qt0, qt1);
        for (int qt = qt0; qt < qt1 && ok; ++qt) {
          for (int c = 0; c < a.nch && ok; ++c) {
            if (qt == qt0) {
              // this CTA's half of key chunk c, once the previous unit's last
              // query tile is done with it (past the table: zero fill)
              ok = ptx::mbar_wait(empty_k + 8 * c, (uint32_t)(i & 1) ^ 1u, abort_s, kWaitLimit);
              if (!ok) break;
              if (pos == 0) ptx::mbar_expect_tx(full_k + 8 * c, (uint32_t)(2 * kKChunkBytes));
              ptx::tma_load_2d_pair(s_k + c * kKChunkBytes, &tmK, c * kChunkF, kt * kBN + (int)pos * kHN,
                                    lead_full_k + 8 * c);
            }
            // stage qs is free in this CTA and in its counterpart of the other pair
            ok = ptx::mbar_wait(empty_q + 8 * qs, qph ^ 1u, abort_s, kWaitLimit);
            if (!ok) break;
            if (pos == 0) ptx::mbar_expect_tx(full_q + 8 * qs, (uint32_t)(2 * kQStageBytes));
            ptx::tma_load_2d_pair_multicast(s_q + qs * kQStageBytes + pair * kQQuarterBytes, &tmQ, c * kChunkF,
                                            qt * kBM + (int)pos * kHM + (int)pair * (kHM / 2),
                                            lead_full_q + 8 * qs, q_mask);
            if (++qs == a.nst) {
              qs = 0;
              qph ^= 1u;
            }
          }
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer (pair leader)
    if (pos == 0 && lane == 0) {
      constexpr uint32_t idesc = ptx::idesc_tf32(kBM, kBN);
      const uint64_t qdesc0 = ptx::sw128_kmajor_desc(s_q);
      const uint64_t kdesc0 = ptx::sw128_kmajor_desc(s_k);
      constexpr uint64_t kQStride = kQStageBytes >> 4;
      constexpr uint64_t kKStride = kKChunkBytes >> 4;
      const int nst = a.nst, nch = a.nch;
      int qs = 0;
      uint32_t qph = 0;
      int t = 0, i = 0;
      // failure-detection test: no arrival ever completes this phase, so the
      // bounded wait expires and the kernel takes its abort path
      bool ok = !a.debug_stall || ptx::mbar_wait(drain, 0, abort_s, kWaitLimit);
      for (int u = cluster_id; u < a.n_units && ok; u += n_clusters, ++i) {
        int kt, qt0, qt1;
        unit_range(a, u, pair, kt, qt0, qt1);
        for (int qt = qt0; qt < qt1 && ok; ++qt, ++t) {
          const int buf = t & 1;
          // both CTAs' epilogues are done with this accumulator
          ok = ptx::mbar_wait_cluster(acc_empty + 8 * buf, (uint32_t)((t >> 1) & 1) ^ 1u, abort_s, kWaitLimit);
          if (!ok) break;
          ptx::tc_fence_after();
          const uint32_t d_tmem = tmem + (uint32_t)(buf * kBN);
          const bool first = qt == qt0, last = qt == qt1 - 1;
          uint64_t kd = kdesc0;
          if (first || last) {
            for (int c = 0; c < nch; ++c, kd += kKStride) {
              if (first && !ptx::mbar_wait(full_k + 8 * c, (uint32_t)(i & 1), abort_s, kWaitLimit)) {
                ok = false;
                break;
              }
              if (!ptx::mbar_wait(full_q + 8 * qs, qph, abort_s, kWaitLimit)) {
                ok = false;
                break;
              }
              const uint64_t qd = qdesc0 + (uint64_t)qs * kQStride;
              ptx::mma_tf32_pair(d_tmem, qd, kd, idesc, c != 0);
              ptx::mma_tf32_pair(d_tmem, qd + 2, kd + 2, idesc, 1u);
              ptx::mma_tf32_pair(d_tmem, qd + 4, kd + 4, idesc, 1u);
              ptx::mma_tf32_pair(d_tmem, qd + 6, kd + 6, idesc, 1u);
              ptx::mma_commit_pair_multicast(empty_q + 8 * qs, (uint16_t)0xF);
              if (last) ptx::mma_commit_pair_multicast(empty_k + 8 * c, pair_mask);
              if (++qs == nst) {
                qs = 0;
                qph ^= 1u;
              }
            }
          } else {
            for (int c = 0; c < nch; ++c, kd += kKStride) {
              if (!ptx::mbar_wait(full_q + 8 * qs, qph, abort_s, kWaitLimit)) {
                ok = false;
                break;
              }
              const uint64_t qd = qdesc0 + (uint64_t)qs * kQStride;
              ptx::mma_tf32_pair(d_tmem, qd, kd, idesc, c != 0);
              ptx::mma_tf32_pair(d_tmem, qd + 2, kd + 2, idesc, 1u);
              ptx::mma_tf32_pair(d_tmem, qd + 4, kd + 4, idesc, 1u);
              ptx::mma_tf32_pair(d_tmem, qd + 6, kd + 6, idesc, 1u);
              ptx::mma_commit_pair_multicast(empty_q + 8 * qs, (uint16_t)0xF);
              if (++qs == nst) {
                qs = 0;
                qph ^= 1u;
              }
            }
          }
          if (ok) ptx::mma_commit_pair_multicast(acc_full + 8 * buf, pair_mask);
        }
      }
      // all issued MMAs complete before the pair's TMEM can be released
      volatile int never = 0;
      ptx::mma_commit_pair_multicast(drain, (uint16_t)(1u << rank));
      ptx::mbar_wait(drain, 0, &never, kWaitLimit);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ epilogue (both CTAs)
    const int ew = warp - 2;
    const int quarter = warp & 3;  // TMEM lane quarter this warp may access
    const int half = ew >> 2;      // column slice
    constexpr int kColsPerWarp = kBN * 4 / kEpiWarps;
    constexpr int kChunks = kColsPerWarp / 32;
    const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
    const uint32_t lead_acc_empty = ptx::mapa(acc_empty, leader);
    float* my_tau = tau_s + ew * kColsPerWarp;
    int t = 0;
    bool ok = true;
    unsigned long long ncand = 0;
    for (int u = cluster_id; u < a.n_units && ok; u += n_clusters) {
      int kt, qt0, qt1;
      unit_range(a, u, pair, kt, qt0, qt1);
      const bool live = kt < a.n_kt;
      const int key0 = kt * kBN + half * kColsPerWarp;
      __syncwarp();
      if (live)
        for (int v4 = lane; v4 < kColsPerWarp / 4; v4 += 32)
          reinterpret_cast<float4*>(my_tau)[v4] = __ldg(reinterpret_cast<const float4*>(a.tau + key0) + v4);
      __syncwarp();
      float tmin[kChunks];
#pragma unroll
      for (int ch = 0; ch < kChunks; ++ch) {
        float m = live ? my_tau[ch * 32 + lane] : INFINITY;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) m = fminf(m, __shfl_xor_sync(0xffffffffu, m, o));
        tmin[ch] = m;
      }
      const int row_off = (int)pos * kHM + quarter * 32 + lane;
      int64_t row = (int64_t)qt0 * kBM + row_off;
      float kap = row < a.bpad ? __ldg(a.kappa + row) : INFINITY;
      for (int qt = qt0; qt < qt1; ++qt, ++t) {
        const int buf = t & 1;
        row = (int64_t)qt * kBM + row_off;
        const int64_t row_next = row + kBM;
        const float kap_next = (qt + 1 < qt1 && row_next < a.bpad) ? __ldg(a.kappa + row_next) : INFINITY;
        ok = ptx::mbar_wait(acc_full + 8 * buf, (uint32_t)((t >> 1) & 1), abort_s, kWaitLimit);
        ok = __all_sync(0xffffffffu, ok);  // warp-uniform before the aligned TMEM loads
        if (!ok) break;
        ptx::tc_fence_after();
        if (live) {
          const uint32_t tbase = tmem + lane_base + (uint32_t)(buf * kBN + half * kColsPerWarp);
          uint32_t r[2][32];
          ptx::tmem_ld32(tbase, r[0]);
          ptx::tmem_wait_ld();
#pragma unroll
          for (int ch = 0; ch < kChunks; ++ch) {
            if (ch + 1 < kChunks) ptx::tmem_ld32(tbase + (uint32_t)((ch + 1) * 32), r[(ch + 1) & 1]);
            const uint32_t* v = r[ch & 1];
            // coarse test of the chunk (probe_tc.cu): fl(max a - min tau)
            float m0 = -INFINITY, m1 = -INFINITY;
#pragma unroll
            for (int j = 0; j < 16; j += 2) {
              m0 = ptx::max3_f32(m0, __uint_as_float(v[j]), __uint_as_float(v[j + 1]));
              m1 = ptx::max3_f32(m1, __uint_as_float(v[16 + j]), __uint_as_float(v[16 + j + 1]));
            }
            if (__fsub_rn(fmaxf(m0, m1), tmin[ch]) >= kap) {
              uint32_t mask = 0;
#pragma unroll
              for (int j = 0; j < 32; ++j)
                mask |= (uint32_t)(__uint_as_float(v[j]) - my_tau[ch * 32 + j] >= kap) << j;
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
        }
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive_cluster(lead_acc_empty + 8 * buf);
        kap = kap_next;
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) ncand += __shfl_xor_sync(0xffffffffu, ncand, o);
    if (lane == 0 && ncand) atomicAdd(&a.stats->candidates, ncand);
  }

  ptx::tc_fence_before();
  __syncthreads();
  if (*abort_s) {
    // A role gave up: leave time for copies and arrivals other CTAs may still
    // direct at this one before the cluster retires.
    if (threadIdx.x == 0) {
      atomicAdd(&a.stats->errors, 1ull);
      atomicExch(&a.stats->abort_flag, 1);
    }
    __nanosleep(50000);
  }
  ptx::cluster_sync();  // no copy, commit or arrival can target an exited CTA
  if (warp == 1) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc_pair(tmem, (uint32_t)kTmemCols);
  }
}

void encode_rows(lipcache* h, CUtensorMap* map, const float* base, uint64_t rows, uint32_t box_rows) {
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

cudaLaunchConfig_t pair_config(int smem, cudaStream_t s, cudaLaunchAttribute* attr) {
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = (size_t)smem;
  cfg.stream = s;
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = kCluster;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cfg;
}

}  // namespace

// Clusters of four that can be resident at once (0: use probe_tc.cu).
int probe_pair_clusters(lipcache* h) {
  if (h->pair_clusters >= 0) return h->pair_clusters;
  h->pair_clusters = 0;
  if (h->dpad > kMaxChunks * kChunkF) return 0;
  const int nch = h->dpad / kChunkF;
  const int nst = PairLayout::stages_for(nch);
  if (nst < 2) return 0;
  const int smem = PairLayout{nch, nst}.total() + 1024;
  if (cudaFuncSetAttribute(k_probe_pair, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBudget + 1024) !=
      cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = pair_config(smem, nullptr, attr);
  cfg.gridDim = dim3((unsigned)(h->num_sms / kCluster * kCluster));
  int resident = 0;
  if (cudaOccupancyMaxActiveClusters(&resident, k_probe_pair, &cfg) != cudaSuccess) {
    cudaGetLastError();
    resident = 0;
  }
  h->pair_clusters = resident;
  return resident;
}

void launch_probe_pair(lipcache* h, int64_t B, const float* qpad, const float* kappa, unsigned long long* best,
                       cudaStream_t s) {
  const int clusters_max = probe_pair_clusters(h);
  LC_REQUIRE(clusters_max >= 1, LIPCACHE_E_CUDA, "no cluster of the pair probe kernel fits on this device");
  const int64_t Bpad = (B + 127) / 128 * 128;  // rows of the padded query buffer
  lipcache::ProbeLaunch& pl = h->probe_launch[2];
  if (pl.q_base != qpad || pl.q_rows != (uint64_t)Bpad) {
    encode_rows(h, &pl.tmQ, qpad, (uint64_t)Bpad, kHM / 2);  // a quarter of the pair's query tile per CTA
    pl.q_base = qpad;
    pl.q_rows = (uint64_t)Bpad;
  }
  if (pl.k_base != h->table.keys || pl.k_rows != (uint64_t)h->table_rows) {
    encode_rows(h, &pl.tmK, h->table.keys, (uint64_t)h->table_rows, kHN);
    pl.k_base = h->table.keys;
    pl.k_rows = (uint64_t)h->table_rows;
  }
  PairArgs a;
  a.nch = h->dpad / kChunkF;
  a.nst = PairLayout::stages_for(a.nch);
  a.dpad = h->dpad;
  a.bpad = Bpad;
  a.nq = (int)((Bpad + kBM - 1) / kBM);
  const int64_t n_kt = (h->size + kBN - 1) / kBN;
  const int64_t n_quads = (n_kt + 1) / 2;
  // query groups per key-tile quad: the fewest that minimise the busiest
  // cluster's share, (units per cluster, rounded up) x (query tiles per unit)
  // (each extra group reloads the quad's key tiles from L2; 100,000 keys at
  // d = 256: 2 groups, 287 -> 270 us)
  int n_qg = 1;
  {
    int64_t best = -1;
    for (int g = 1; g <= a.nq; ++g) {
      const int qpg = (a.nq + g - 1) / g;
      const int ng = (a.nq + qpg - 1) / qpg;
      const int64_t cost = (n_quads * ng + clusters_max - 1) / clusters_max * qpg;
      if (best < 0 || cost < best) {
        best = cost;
        n_qg = ng;
      }
    }
  }
  a.qpg = (a.nq + n_qg - 1) / n_qg;
  a.n_qg = (a.nq + a.qpg - 1) / a.qpg;
  const int64_t n_units = n_quads * a.n_qg;
  LC_REQUIRE(n_units < (1LL << 31), LIPCACHE_E_INVALID, "too many work units");
  a.n_units = (int)n_units;
  a.n_kt = (int)n_kt;
  a.kappa = kappa;
  a.qpad = qpad;
  a.keys = h->table.keys;
  a.tau = h->probe_tau();
  a.rr = h->probe_rr();
  a.best = best;
  a.stats = h->stats;
  a.debug_stall = (h->debug_flags & LIPCACHE_DEBUG_STALL_PROBE) ? 1 : 0;
  const int smem = PairLayout{a.nch, a.nst}.total() + 1024;
  if (pl.smem == 0) {
    // the attribute belongs to the kernel: the largest size any shape uses
    LC_CUDA(cudaFuncSetAttribute(k_probe_pair, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBudget + 1024));
    pl.smem = kSmemBudget + 1024;
  }
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = pair_config(smem, s, attr);
  int clusters = clusters_max;
  if (n_units < clusters) clusters = (int)n_units;
  cfg.gridDim = dim3((unsigned)(clusters * kCluster));
  h->last_grid = clusters * kCluster;
  h->last_cluster = kCluster;
  if (h->launch_event) LC_CUDA(cudaEventRecord(h->launch_event, s));
  LC_CUDA(cudaLaunchKernelEx(&cfg, k_probe_pair, pl.tmQ, pl.tmK, a));
  LC_LAUNCH_CHECK("k_probe_pair");
}

}  // namespace lc
