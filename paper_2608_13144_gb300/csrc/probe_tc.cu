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
// fl(a - tau_k) >= kappa_q, which therefore never drops an acceptable pair.
// It first tests each 32-key chunk with fl(max a - min tau) >= kappa_q (one
// three-input max per two pairs), which no chunk holding a kept pair fails.
//
// Schedule. Persistent CTAs, one per SM, launched as clusters of two. The two
// CTAs of a cluster own two adjacent key tiles and stream the SAME sequence of
// query tiles: each CTA TMA-loads one half of every query stage with
// .multicast::cluster into both CTAs' shared memory, so the L2 delivers each
// query byte once per pair of SMs (the query stream from L2 is what limits a
// single CTA). Per CTA (320 threads):
//   warp 0     TMA producer: the CTA's key tile (BN keys x d_pad, resident,
//              one barrier pair per 32-float chunk so the next tile streams in
//              while the last query tile still runs) and its half of each
//              query stage (128 queries x 32 floats per stage, multi-stage ring);
//   warp 1     allocates TMEM, issues tcgen05.mma kind::tf32 (M=128 queries,
//              N=BN keys, K=8) from one thread into one of two TMEM
//              accumulators; releases each query stage in BOTH CTAs;
//   warps 2-9  epilogue: tcgen05.ld of the accumulator (warp w reads TMEM
//              lane quarter w % 4, column half (w - 2) / 4), screen, recheck,
//              atomicMin of the packed (distance, index) word.
// Work: the items (key-tile pair, query tile), pair-major, are split into
// equal contiguous ranges, one per cluster; a run is the part of a range on
// one pair, and its key tile stays resident through the run (a pair split
// between two clusters is loaded by both). When the number of key tiles is odd
// the last pair's second tile lies past the table: that CTA multiplies the
// TMA's zero fill and its epilogue skips the run, so both CTAs still consume
// every query stage.
#include "internal.cuh"
#include "probe_common.cuh"
#include "tc_ptx.cuh"

namespace lc {
int tc_key_tile(int dpad);
namespace {

constexpr int kBM = 128;              // queries per tile (MMA M)
constexpr int kChunkF = 32;           // floats per K chunk (one 128-byte swizzle row)
constexpr int kMaxStages = 8;         // query ring depth limit (runtime count fills shared memory)
constexpr int kMaxChunks = 8;         // d_pad <= 256
constexpr int kQStageBytes = kBM * 128;
constexpr int kQHalfBytes = kQStageBytes / 2;
#ifndef LC_EPI_WARPS
#define LC_EPI_WARPS 8
#endif
constexpr int kEpiWarps = LC_EPI_WARPS;  // 4 or 8: one or two per SM sub-partition
constexpr int kThreads = 32 * (2 + kEpiWarps);
constexpr int kCluster = 2;
constexpr uint16_t kClusterMask = 0x3;
constexpr int kSmemBudget = 227 * 1024 - 1024;  // opt-in limit minus the alignment slack
constexpr long long kWaitLimit = 1LL << 31;     // ~1 s at GB300 clocks
constexpr int64_t kPairedReleaseItems = 64;     // items per cluster from which stages are released in pairs

struct TcArgs {
  int nst;       // query ring stages
  int qgroup;    // stages released together, 1 or 2 (the kernel instantiation; divides nst)
  int tau_staged;  // screen terms copied to shared memory per run (short runs), else read through L1
  int nch;       // d_pad / 32
  int dpad;
  int nq;        // query tiles
  int n_pairs;   // key-tile pairs
  int n_kt;      // key tiles holding cache entries
  const float* kappa;
  const float* qpad;
  const float* keys;
  const float* tau;
  const float* rr;
  unsigned long long* best;
  DevStats* stats;
  int debug_stall;  // test hook: the MMA issuer first waits on a barrier nothing arrives on
};

template <int BN>
struct Layout {
  static constexpr int kKChunkBytes = BN * 128;
  static constexpr int kTmemCols = 2 * BN;
  static constexpr int kTauStaged = 4 * BN * 4;  // one private slice of screen terms per epilogue warp
  int nch, nst, tau_staged;  // tau_staged: the screen terms copied per run (else read through L1)
  __device__ __host__ int kbytes() const { return nch * kKChunkBytes; }
  __device__ __host__ int qoff() const { return kbytes(); }
  __device__ __host__ int tauoff() const { return qoff() + nst * kQStageBytes; }
  __device__ __host__ int baroff() const { return tauoff() + (tau_staged ? kTauStaged : 0); }
  // barriers: full_k[nch], empty_k[nch], full_q[nst], empty_q[nst], acc_full[2], acc_empty[2], drain
  __device__ __host__ int nbar() const { return 2 * nch + 2 * nst + 5; }
  __device__ __host__ int miscoff() const { return baroff() + 8 * nbar(); }
  __device__ __host__ int total() const { return miscoff() + 16; }
  // deepest ring that fits the shared-memory budget
  static __host__ int stages_for(int nch, int tau_staged) {
    for (int n = kMaxStages; n >= 2; --n) {
      Layout<BN> L{nch, n, tau_staged};
      if (L.total() <= kSmemBudget) return n;
    }
    return 0;
  }
};

// The runs of one cluster: its range [it, end) of items (pair, query tile),
// pair-major; next() gives this CTA's key tile and the run's query tiles.
struct RunCursor {
  long long it, end;
  __device__ RunCursor(const TcArgs& a, int cluster_id, int n_clusters) {
    const long long T = (long long)a.n_pairs * a.nq;
    it = T * cluster_id / n_clusters;
    end = T * (cluster_id + 1) / n_clusters;
  }
  __device__ bool next(const TcArgs& a, uint32_t rank, int& kt, int& qt0, int& qt1) {
    if (it >= end) return false;
    const int pair = (int)(it / a.nq);
    qt0 = (int)(it - (long long)pair * a.nq);
    const long long run_end = min(end, (long long)(pair + 1) * a.nq);
    qt1 = qt0 + (int)(run_end - it);
    kt = pair * kCluster + (int)rank;
    it = run_end;
    return true;
  }
};

// MODE 0: short ranges (screen terms staged in shared memory, stages released
// one at a time); 1: long ranges (screen terms through L1), single releases;
// 2: long ranges, stages released in pairs.
template <int BN, int MODE>
__global__ void __launch_bounds__(kThreads, 1)
    k_probe_tc(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK, const TcArgs a) {
  constexpr int QG = MODE == 2 ? 2 : 1;  // query stages released together
  constexpr bool kTauStaged = MODE == 0;
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  // 1024-byte alignment of the swizzled tiles
  unsigned char* smem =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  const Layout<BN> L{a.nch, a.nst, a.tau_staged};
  const uint32_t s_base = ptx::smem_u32(smem);
  const uint32_t s_k = s_base;
  const uint32_t s_q = s_base + L.qoff();
  const uint32_t s_bar = s_base + L.baroff();
  const uint32_t full_k = s_bar, empty_k = s_bar + 8 * a.nch;
  const uint32_t full_q = s_bar + 16 * a.nch, empty_q = full_q + 8 * a.nst;
  const uint32_t acc_full = empty_q + 8 * a.nst, acc_empty = acc_full + 16, drain = acc_empty + 16;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L.miscoff());
  volatile int* abort_s = reinterpret_cast<volatile int*>(smem + L.miscoff() + 4);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = ptx::cluster_ctarank();
  const int cluster_id = blockIdx.x / kCluster, n_clusters = gridDim.x / kCluster;

  if (threadIdx.x == 0) {
    for (int c = 0; c < a.nch; ++c) {
      ptx::mbar_init(full_k + 8 * c, 1);
      ptx::mbar_init(empty_k + 8 * c, 1);
    }
    for (int s = 0; s < a.nst; ++s) {
      ptx::mbar_init(full_q + 8 * s, 1);         // own arrival; bytes from both CTAs
      ptx::mbar_init(empty_q + 8 * s, kCluster); // released by the MMA of both CTAs
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
  ptx::cluster_sync();  // the peer's barriers exist before any multicast reaches them
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      int qs = 0;
      uint32_t qph = 0;
      int i = 0;
      int last_k_par[kMaxChunks];
      uint32_t last_q_par[kMaxStages];
      bool q_used[kMaxStages];
      for (int c = 0; c < kMaxChunks; ++c) last_k_par[c] = -1;
      for (int s = 0; s < kMaxStages; ++s) {
        q_used[s] = false;
        last_q_par[s] = 0;
      }
      bool ok = true;
      RunCursor rc(a, cluster_id, n_clusters);
      int kt, qt0, qt1;
      for (; ok && rc.next(a, rank, kt, qt0, qt1); ++i) {
        for (int qt = qt0; qt < qt1 && ok; ++qt) {
          for (int c = 0; c < a.nch && ok; ++c) {
            if (qt == qt0) {
              // key chunk c of this run, as soon as the previous run's last
              // query tile has finished with it (past the table: zero fill)
              ok = ptx::mbar_wait(empty_k + 8 * c, (uint32_t)(i & 1) ^ 1u, abort_s, kWaitLimit);
              if (!ok) break;
              ptx::mbar_expect_tx(full_k + 8 * c, (uint32_t)Layout<BN>::kKChunkBytes);
              ptx::tma_load_2d(s_k + c * Layout<BN>::kKChunkBytes, &tmK, c * kChunkF, kt * BN, full_k + 8 * c);
              last_k_par[c] = i & 1;
            }
            // stage qs is free in both CTAs (its group was released); fetch
            // this CTA's half for both
            if (QG == 1 || (qs & 1) == 0) {
              ok = ptx::mbar_wait(empty_q + 8 * (qs >> (QG - 1)), qph ^ 1u, abort_s, kWaitLimit);
              if (!ok) break;
            }
            ptx::mbar_expect_tx(full_q + 8 * qs, (uint32_t)kQStageBytes);
            ptx::tma_load_2d_multicast(s_q + qs * kQStageBytes + rank * kQHalfBytes, &tmQ, c * kChunkF,
                                       qt * kBM + (int)rank * (kBM / 2), full_q + 8 * qs, kClusterMask);
            q_used[qs] = true;
            last_q_par[qs] = qph;
            if (++qs == a.nst) {
              qs = 0;
              qph ^= 1u;
            }
          }
        }
      }
      // Let every copy into this CTA land before it can exit. (Bounded; a
      // phase that already completed returns at once.)
      volatile int never = 0;
      for (int s = 0; s < a.nst; ++s)
        if (q_used[s]) ptx::mbar_wait(full_q + 8 * s, last_q_par[s], &never, kWaitLimit);
      for (int c = 0; c < a.nch; ++c)
        if (last_k_par[c] >= 0) ptx::mbar_wait(full_k + 8 * c, (uint32_t)last_k_par[c], &never, kWaitLimit);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    // The tensor pipe queues about one MMA ahead, so this loop keeps the work
    // between MMA issues minimal: shared-memory descriptors are built once and
    // advanced by adding encoded offsets (the start-address field holds
    // address >> 4, so +32 bytes is +2 and never carries out of the field).
    if (lane == 0) {
      constexpr uint32_t idesc = ptx::idesc_tf32(kBM, BN);
      const uint64_t qdesc0 = ptx::sw128_kmajor_desc(s_q);
      const uint64_t kdesc0 = ptx::sw128_kmajor_desc(s_k);
      constexpr uint64_t kQStride = kQStageBytes >> 4;
      constexpr uint64_t kKStride = Layout<BN>::kKChunkBytes >> 4;
      const int nst = a.nst, nch = a.nch;
      int qs = 0;
      uint32_t qph = 0;
      int t = 0, i = 0;
      // failure-detection test: no arrival ever completes this phase, so the
      // bounded wait expires and the kernel takes its abort path
      bool ok = !a.debug_stall || ptx::mbar_wait(drain, 0, abort_s, kWaitLimit);
      RunCursor rc(a, cluster_id, n_clusters);
      int kt, qt0, qt1;
      for (; ok && rc.next(a, rank, kt, qt0, qt1); ++i) {
        for (int qt = qt0; qt < qt1 && ok; ++qt, ++t) {
          const int buf = t & 1;
          ok = ptx::mbar_wait(acc_empty + 8 * buf, (uint32_t)((t >> 1) & 1) ^ 1u, abort_s, kWaitLimit);
          if (!ok) break;
          ptx::tc_fence_after();
          const uint32_t d_tmem = tmem + (uint32_t)(buf * BN);
          const bool first = qt == qt0, last = qt == qt1 - 1;
          uint64_t kd = kdesc0;
          if (first || last) {
            // Run edges: the key chunk arrives once per run (TMA completion on
            // the mbarrier already orders the copies before the MMA's reads),
            // and the last query tile hands each chunk back to the producer.
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
              ptx::mma_tf32(d_tmem, qd, kd, idesc, c != 0);
              ptx::mma_tf32(d_tmem, qd + 2, kd + 2, idesc, 1u);
              ptx::mma_tf32(d_tmem, qd + 4, kd + 4, idesc, 1u);
              ptx::mma_tf32(d_tmem, qd + 6, kd + 6, idesc, 1u);
              if (QG == 1 || (qs & 1)) ptx::mma_commit_multicast(empty_q + 8 * (qs >> (QG - 1)), kClusterMask);
              if (last) ptx::mma_commit(empty_k + 8 * c);
              if (++qs == nst) {
                qs = 0;
                qph ^= 1u;
              }
            }
          } else if (QG == 2) {
            // Steady state, stages released in pairs (nch and nst even, so
            // a tile starts on the first stage of a pair): the stage waits,
            // eight MMAs and one release per two stages, no predicated
            // tensor-pipe instructions.
            for (int c = 0; c < nch && ok; c += 2, kd += 2 * kKStride) {
              if (!ptx::mbar_wait(full_q + 8 * qs, qph, abort_s, kWaitLimit)) {
                ok = false;
                break;
              }
              uint64_t qd = qdesc0 + (uint64_t)qs * kQStride;
              ptx::mma_tf32(d_tmem, qd, kd, idesc, c != 0);
              ptx::mma_tf32(d_tmem, qd + 2, kd + 2, idesc, 1u);
              ptx::mma_tf32(d_tmem, qd + 4, kd + 4, idesc, 1u);
              ptx::mma_tf32(d_tmem, qd + 6, kd + 6, idesc, 1u);
              ++qs;  // (even, below nst - 1: no wrap)
              if (!ptx::mbar_wait(full_q + 8 * qs, qph, abort_s, kWaitLimit)) {
                ok = false;
                break;
              }
              qd = qdesc0 + (uint64_t)qs * kQStride;
              const uint64_t kd1 = kd + kKStride;
              ptx::mma_tf32(d_tmem, qd, kd1, idesc, 1u);
              ptx::mma_tf32(d_tmem, qd + 2, kd1 + 2, idesc, 1u);
              ptx::mma_tf32(d_tmem, qd + 4, kd1 + 4, idesc, 1u);
              ptx::mma_tf32(d_tmem, qd + 6, kd1 + 6, idesc, 1u);
              ptx::mma_commit_multicast(empty_q + 8 * (qs >> 1), kClusterMask);
              if (++qs == nst) {
                qs = 0;
                qph ^= 1u;
              }
            }
          } else {
            // Steady state: nothing but the stage wait, four MMAs and the
            // stage release (no predicated tensor-pipe instructions).
            for (int c = 0; c < nch; ++c, kd += kKStride) {
              if (!ptx::mbar_wait(full_q + 8 * qs, qph, abort_s, kWaitLimit)) {
                ok = false;
                break;
              }
              const uint64_t qd = qdesc0 + (uint64_t)qs * kQStride;
              ptx::mma_tf32(d_tmem, qd, kd, idesc, c != 0);
              ptx::mma_tf32(d_tmem, qd + 2, kd + 2, idesc, 1u);
              ptx::mma_tf32(d_tmem, qd + 4, kd + 4, idesc, 1u);
              ptx::mma_tf32(d_tmem, qd + 6, kd + 6, idesc, 1u);
              ptx::mma_commit_multicast(empty_q + 8 * qs, kClusterMask);
              if (++qs == nst) {
                qs = 0;
                qph ^= 1u;
              }
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
    const int half = ew >> 2;             // column slice
    constexpr int kColsPerWarp = BN * 4 / kEpiWarps;
    constexpr int kChunks = kColsPerWarp / 32;
    // this warp's private slice of the screen terms when they are staged
    float* my_tau = reinterpret_cast<float*>(smem + L.tauoff()) + ew * kColsPerWarp;
    const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
    int t = 0;
    bool ok = true;
    unsigned long long ncand = 0;
    RunCursor rc(a, cluster_id, n_clusters);
    int kt, qt0, qt1;
    while (ok && rc.next(a, rank, kt, qt0, qt1)) {
      const bool live = kt < a.n_kt;
      const int key0 = kt * BN + half * kColsPerWarp;
      // the minimum of this warp's screen terms over each 32-key chunk of
      // the run's key tile. The per-pair test, which few chunks reach, reads
      // the terms themselves from a copy in shared memory made here when the
      // runs are short, else through L1 (the space goes to a deeper query
      // ring).
      if (kTauStaged) {
        __syncwarp();
        if (live)
          for (int v4 = lane; v4 < kColsPerWarp / 4; v4 += 32)
            reinterpret_cast<float4*>(my_tau)[v4] = __ldg(reinterpret_cast<const float4*>(a.tau + key0) + v4);
        __syncwarp();
      }
      const float* __restrict__ tau_g = a.tau + key0;
      float tmin[kChunks];
#pragma unroll
      for (int ch = 0; ch < kChunks; ++ch) {
        float m = !live ? INFINITY : kTauStaged ? my_tau[ch * 32 + lane] : __ldg(tau_g + ch * 32 + lane);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) m = fminf(m, __shfl_xor_sync(0xffffffffu, m, o));
        tmin[ch] = m;
      }
      float kap = __ldg(a.kappa + qt0 * kBM + quarter * 32 + lane);
      for (int qt = qt0; qt < qt1; ++qt, ++t) {
        const int buf = t & 1;
        const int row = qt * kBM + quarter * 32 + lane;
        // next tile's screen constant, fetched while this accumulator is produced
        const float kap_next = (qt + 1 < qt1) ? __ldg(a.kappa + row + kBM) : 0.f;
        ok = ptx::mbar_wait(acc_full + 8 * buf, (uint32_t)((t >> 1) & 1), abort_s, kWaitLimit);
        ok = __all_sync(0xffffffffu, ok);  // warp-uniform before the aligned TMEM loads
        if (!ok) break;
        ptx::tc_fence_after();
        if (live) {
          const uint32_t tbase = tmem + lane_base + (uint32_t)(buf * BN + half * kColsPerWarp);
          uint32_t r[2][32];
          ptx::tmem_ld32(tbase, r[0]);
          ptx::tmem_wait_ld();
#pragma unroll
          for (int ch = 0; ch < kChunks; ++ch) {
            if (ch + 1 < kChunks) ptx::tmem_ld32(tbase + (uint32_t)((ch + 1) * 32), r[(ch + 1) & 1]);
            const uint32_t* v = r[ch & 1];
            // Coarse test of the chunk: a_j - tau_j <= max_j a_j - min_j tau_j
            // exactly, and rounding is monotone, so a chunk whose
            // fl(max a - min tau) is below kappa holds no pair that passes
            // fl(a_j - tau_j) >= kappa. Two independent three-input max chains.
            float m0 = -INFINITY, m1 = -INFINITY;
#pragma unroll
            for (int j = 0; j < 16; j += 2) {
              m0 = ptx::max3_f32(m0, __uint_as_float(v[j]), __uint_as_float(v[j + 1]));
              m1 = ptx::max3_f32(m1, __uint_as_float(v[16 + j]), __uint_as_float(v[16 + j + 1]));
            }
            if (__fsub_rn(fmaxf(m0, m1), tmin[ch]) >= kap) {
              uint32_t mask = 0;
              if (kTauStaged) {
#pragma unroll
                for (int j = 0; j < 32; ++j) mask |= (uint32_t)(__uint_as_float(v[j]) - my_tau[ch * 32 + j] >= kap) << j;
              } else {
#pragma unroll
                for (int j = 0; j < 32; ++j)
                  mask |= (uint32_t)(__uint_as_float(v[j]) - __ldg(tau_g + ch * 32 + j) >= kap) << j;
              }
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
        if (lane == 0) ptx::mbar_arrive(acc_empty + 8 * buf);
        kap = kap_next;
      }
    }
    // candidate count: one atomic per warp
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) ncand += __shfl_xor_sync(0xffffffffu, ncand, o);
    if (lane == 0 && ncand) atomicAdd(&a.stats->candidates, ncand);
  }

  ptx::tc_fence_before();
  __syncthreads();
  if (*abort_s) {
    // A role gave up: leave time for copies the peer may still be
    // multicasting into this CTA before the cluster retires.
    if (threadIdx.x == 0) {
      atomicAdd(&a.stats->errors, 1ull);
      atomicExch(&a.stats->abort_flag, 1);
    }
    __nanosleep(50000);
  }
  ptx::cluster_sync();  // no remote arrival or copy can target an exited CTA
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
void launch(lipcache* h, int64_t B, const float* qpad, const float* kappa, unsigned long long* best, cudaStream_t s) {
  const int64_t Bpad = (B + kBM - 1) / kBM * kBM;
  lipcache::ProbeLaunch& pl = h->probe_launch[BN == 256 ? 0 : 1];
  if (pl.q_base != qpad || pl.q_rows != (uint64_t)Bpad) {
    encode_2d(h, &pl.tmQ, qpad, (uint64_t)Bpad, kBM / 2);  // half a query tile per CTA of the pair
    pl.q_base = qpad;
    pl.q_rows = (uint64_t)Bpad;
  }
  if (pl.k_base != h->table.keys || pl.k_rows != (uint64_t)h->table_rows) {
    encode_2d(h, &pl.tmK, h->table.keys, (uint64_t)h->table_rows, BN);
    pl.k_base = h->table.keys;
    pl.k_rows = (uint64_t)h->table_rows;
  }
  TcArgs a;
  a.nch = h->dpad / kChunkF;
  // (the ring depth depends on whether the screen terms are staged: below)
  a.dpad = h->dpad;
  a.nq = (int)(Bpad / kBM);
  const int64_t n_kt = (h->size + BN - 1) / BN;
  const int64_t n_pairs = (n_kt + kCluster - 1) / kCluster;
  const int max_clusters = h->num_sms / kCluster;
  LC_REQUIRE(max_clusters >= 1, LIPCACHE_E_CUDA, "device has fewer than two SMs");
  // Long ranges (many items per cluster, the large caches): the screen terms
  // are read through L1, the shared memory goes to the query ring, and the
  // stages are released two at a time (one commit per pair) when a tile's
  // stages pair up and the ring holds whole pairs. Short ranges keep the
  // staged screen terms and single releases, which measure faster there.
  const bool long_ranges = n_pairs * a.nq / max_clusters >= kPairedReleaseItems;
  a.tau_staged = long_ranges ? 0 : 1;
  a.nst = Layout<BN>::stages_for(a.nch, a.tau_staged);
  LC_REQUIRE(a.nst >= 2, LIPCACHE_E_INVALID, "key tile does not fit shared memory");
  a.qgroup = (long_ranges && a.nst % 2 == 0 && a.nch % 2 == 0) ? 2 : 1;
  LC_REQUIRE(n_pairs * a.nq < (1LL << 40), LIPCACHE_E_INVALID, "too many work items");
  a.n_pairs = (int)n_pairs;
  a.n_kt = (int)n_kt;
  a.kappa = kappa;
  a.qpad = qpad;
  a.keys = h->table.keys;
  a.tau = h->probe_tau();
  a.rr = h->probe_rr();
  a.best = best;
  a.stats = h->stats;
  a.debug_stall = (h->debug_flags & LIPCACHE_DEBUG_STALL_PROBE) ? 1 : 0;
  const Layout<BN> L{a.nch, a.nst, a.tau_staged};
  const int smem = L.total() + 1024;
  if (pl.smem == 0) {
    // the attribute belongs to the kernel, not to this cache: set it to the
    // largest size any shape uses, so other caches' launches stay valid
    LC_CUDA(cudaFuncSetAttribute(k_probe_tc<BN, 0>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBudget + 1024));
    LC_CUDA(cudaFuncSetAttribute(k_probe_tc<BN, 1>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBudget + 1024));
    LC_CUDA(cudaFuncSetAttribute(k_probe_tc<BN, 2>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBudget + 1024));
    pl.smem = kSmemBudget + 1024;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(max_clusters * kCluster));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = (size_t)smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = kCluster;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  // persistent grid: no more clusters than can be resident at once
  if (pl.resident == 0) LC_CUDA(cudaOccupancyMaxActiveClusters(&pl.resident, k_probe_tc<BN, 0>, &cfg));
  const int resident = pl.resident;
  LC_REQUIRE(resident >= 1, LIPCACHE_E_CUDA, "no CTA pair of the probe kernel fits on this device");
  int clusters = max_clusters < resident ? max_clusters : resident;
  if (n_pairs * a.nq < clusters) clusters = (int)(n_pairs * a.nq);  // one item per cluster at least
  cfg.gridDim = dim3((unsigned)(clusters * kCluster));
  h->last_grid = clusters * kCluster;
  h->last_cluster = kCluster;
  if (h->launch_event) LC_CUDA(cudaEventRecord(h->launch_event, s));
  void (*kern)(CUtensorMap, CUtensorMap, TcArgs) =
      a.tau_staged ? k_probe_tc<BN, 0> : a.qgroup == 2 ? k_probe_tc<BN, 2> : k_probe_tc<BN, 1>;
  LC_CUDA(cudaLaunchKernelEx(&cfg, kern, pl.tmQ, pl.tmK, a));
  LC_LAUNCH_CHECK("k_probe_tc");
}

}  // namespace

int tc_key_tile(int dpad) { return dpad <= 128 ? 256 : 128; }

int launch_probe_tc_external(lipcache* h, int64_t B, int path, const float* qpad, const float* kappa,
                             unsigned long long* best, cudaStream_t s) {
  LC_REQUIRE(tensor_path_supported(h->dpad), LIPCACHE_E_INVALID, "the tensor probe supports d <= 256");
  // Pair MMAs read a third less shared memory per flop; that decides for
  // d_pad > 128, where the single-CTA kernel has to use 128-key tiles. At
  // d_pad <= 128 its 256-key tiles on all SMs (clusters of four leave some
  // idle) are faster.
  const bool pair = path == LIPCACHE_PROBE_TENSOR_PAIR || (path == LIPCACHE_PROBE_TENSOR && h->dpad > 128);
  if (pair && probe_pair_clusters(h) >= 1) {
    launch_probe_pair(h, B, qpad, kappa, best, s);
    return LIPCACHE_PROBE_TENSOR_PAIR;
  }
  if (tc_key_tile(h->dpad) == 256)
    launch<256>(h, B, qpad, kappa, best, s);
  else
    launch<128>(h, B, qpad, kappa, best, s);
  return LIPCACHE_PROBE_TENSOR_SINGLE;
}

int launch_probe_tc(lipcache* h, int64_t B, int path, cudaStream_t s) {
  return launch_probe_tc_external(h, B, path, h->qpad, h->kappa, h->best, s);
}

}  // namespace lc
