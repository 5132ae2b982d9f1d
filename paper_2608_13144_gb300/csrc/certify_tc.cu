// Certified insertion on the tensor cores (Sec. 3.3, Algorithm 1 loop body;
// Eqs. 5, 6, 20, 21; the tight radius of Remark 4.2, Eq. 29).
//
// The head logits of a batch, s = W z + b for every row z, form one dense
// contraction (rows x d) . (d x C). This kernel runs it as TF32 tcgen05 MMAs
// (M = 128 rows, N = C padded to a multiple of 16, K = 8 per instruction) into
// tensor memory, and uses the result only as a screen that picks the classes
// that can be among the true top two; those are recomputed with the same
// compensated FP32 dot product, in the same order, as the wide-tile kernel, and
// the FP64 finals are shared. The conservative radii, labels and thresholds
// therefore come out bit for bit as from the FP32 kernels; tight radii agree
// with theirs within the refinement bound (bit for bit wherever both refine
// y^G and the minimiser in the same order).
//
// Screen bound. The MMA returns a_c with |a_c - W_c . z| <= c ||W_c|| ||z||
// (c = c_screen: TF32 operands within 2^-10 relative, FP32-accurate
// accumulation, doubled for safety; the probe's screen uses the same bound),
// and s~_c = fl(a_c + b_c) adds at most 2^-24 |a_c + b_c| <= 2^-24 Mb, with
// hn >= ||z||, wmax >= max_c ||W_c|| and Mb = (1 + c) wmax hn + max_c |b_c|:
//     |s~_c - s_c| <= E = c wmax hn + 2^-22 Mb + tiny      (rounded up).
// Mb also bounds every partial sum of the MMA, so when Mb < 1e38 no screen
// value overflows or is NaN; a row with a larger (or NaN) Mb - NaN or infinite
// features, or values near the FP32 range - has every class refined.
// Conservative radius: if l2 is the second-largest s~_c, every class of the
// true top two has s_c >= (true runner-up) >= l2 - E, hence s~_c >= l2 - 2E >=
// T = RD(l2 - 2E): the classes with s~_c >= T are the candidates.
// Tight radius: with y1 / y2 the screen's top two, y1 is certainly y^G when
// y2's upper end is below y1's lower end; then the candidates are y1 and the
// classes whose lower bracket of (s_y - s_j) / ||W_y - W_j|| reaches u_{y2},
// first with the head row's smallest reciprocal pair norm, then with the
// class's own (the minimiser of Eq. 29 always passes). Otherwise one test
// valid for every possible y^G (its logit above lo_1, since it is at least
// s_y1; r* below a bound from y1's row) picks the candidates, and y^G is the
// largest refined one.
// Each half reduces Eq. 29 over its own candidates in FP64; rows with more
// candidates than slots take a one-warp path over every class.
//
// Schedule. Persistent CTAs, one per SM, 384 threads:
//   warp 0     TMA producer: W (resident, 128-byte swizzle, rows past C zero
//              filled), then each tile's 128 rows (one 16 KB box per 32-feature
//              chunk, features past d zero filled) into one of nzb buffers,
//              and the CTA's next tile into L2;
//   warp 1     TMEM allocation; one thread issues the MMAs of a tile into one
//              of two accumulators (columns 0 / 256);
//   warps 2-9  epilogue, two warps per TMEM lane quarter (32 rows), each
//              taking every other 32-column chunk of the classes: ||z||^2
//              (two of its four k-ordered partial chains each) from the tile
//              in shared memory and the top two s~ of its columns (with their
//              classes for the tight radius), exchanged with the partner warp
//              through a named barrier; then the candidates of its columns
//              into the warp's pair list. The four groups of 8 lanes refine
//              the list eight pairs at a time (two per group) into cells by
//              (row, slot), from which each row's lane takes its own results.
//              Conservative radius: a row with more than kMaxCandTc candidates
//              in a half, or whose Mb is not below 1e38, has every class of
//              that half refined; the partners' running selections are merged
//              and one thread per row runs the FP64 finals. Tight radius: see
//              above; such rows take the one-warp path. Rows the finals list
//              for the FP64 pass go into a queue in shared memory;
//   warp 10    the FP64 pass (fix_row_warp) over the queued rows, with the
//              head read in place, while the epilogue goes on with later
//              tiles (when its queue and scratch fit in shared memory; else
//              the rows stay listed for the stand-alone pass);
//   warp 11    idle.
// Every mbarrier wait is bounded; a role that gives up raises the CTA's abort
// flag, the others drain, and the launch counts a device error.
#include "certify_common.cuh"
#include "tc_ptx.cuh"

namespace lc {
namespace {

constexpr int kBM = 128;                      // rows per tile (MMA M, TMEM lanes)
constexpr int kChunkF = 32;                   // features per 128-byte swizzle row
constexpr int kMaxChunks = 8;                 // d <= 256
constexpr uint32_t kZChunkBytes = kBM * 128;  // one 32-feature chunk of a tile
constexpr int kEpiWarps = 8;
constexpr int kFixWarp = 2 + kEpiWarps;       // the in-kernel FP64 pass
// twelve warps (the last one idle): three per SM sub-partition give each
// thread the same 168 registers as ten, without spills
constexpr int kThreads = 32 * (4 + kEpiWarps);
constexpr int kFixQ = 32;                     // slots of the FP64 pass's row queue
constexpr int kMaxCandTc = 8;                 // candidate slots per row and column half
constexpr int kListCap = 32 * kMaxCandTc;     // pair list of one epilogue warp
// per epilogue warp: the pair list, then the refined pairs hi / lo by (row lane, slot)
constexpr uint32_t kWarpScratch = kListCap * 4 + 32 * kMaxCandTc * 8;
constexpr int kGroupTc = 8;                   // lanes per refined pair
constexpr int kNoClass = 0xffff;              // "no class yet" in the indexed top-two trackers
constexpr uint32_t kTmemCols = 512;           // two accumulators of up to 256 columns
constexpr uint32_t kAccStride = 256;
constexpr long long kWaitLimit = 1LL << 31;   // ~1 s at GB300 clocks
constexpr int kSmemBudget = 227 * 1024 - 1024;

// Per-row state a half hands to its partner after the first pass: the top
// two s~ of its columns, its half of ||z||^2 and (tight radius) the classes of
// the top two (low / high 16 bits).
struct Pass1 {
  float l1, l2, psum;
  int idx;
};

// Exchange area of the tight radius (in the space of the conservative
// radius's Top2 exchange): each half's best refined candidate (value and
// class) and overflow flag, and half 1's partial minima of Eq. 29.
struct TightX {
  float2 bv[2][128];
  int16_t bc[2][128];  // -1: no candidate
  uint8_t ovf[2][128];
  double rmin[128], smin[128];
  uint8_t nan[128];
};

static_assert(sizeof(TightX) <= kBM * sizeof(Top2), "the tight exchange shares the Top2 exchange area");

// (a1, j1) >= (a2, j2) are the top two (value, class) of one set; merge in
// the top two (b1, k1) >= (b2, k2) of a disjoint set. Larger value first,
// lower class on equal values.
__device__ __forceinline__ void top2i_merge(float& a1, int& j1, float& a2, int& j2, float b1, int k1, float b2,
                                            int k2) {
  auto better = [](float x, int i, float y, int k) { return x > y || (x == y && i < k); };
  if (better(b1, k1, a1, j1)) {
    if (!better(a1, j1, b2, k2)) {
      a1 = b2;
      j1 = k2;
    }
    a2 = a1;
    j2 = j1;
    a1 = b1;
    j1 = k1;
  } else if (better(b1, k1, a2, j2)) {
    a2 = b1;
    j2 = k1;
  }
}

// Shared-memory layout (offsets from a 1024-byte aligned base).
// Queue of the rows listed for the FP64 pass, from the epilogue warps to the
// fix warp (shared memory): entry k sits in slot k % kFixQ once seq[slot] = k.
struct FixQueue {
  int n;      // entries pushed
  int taken;  // entries the fix warp has finished (their slots are free)
  int done;   // epilogue warps past their last tile
  int beat;   // advanced by the epilogue every tile (the fix warp's wait bound)
  int seq[kFixQ];
  int row[kFixQ];
  float kn[kFixQ];
};

struct TcLayout {
  int nch, Cpad, nzb, infix;
  uint32_t wbytes, zbytes;
  uint32_t off_z, off_bias, off_wn, off_list, off_x1, off_x2, off_acc, off_bar, off_misc, off_fixq, off_fixs, total;
};

// infix: the fix warp runs the FP64 pass in the kernel (its queue and scratch
// in shared memory); else the rows stay listed for the stand-alone pass.
TcLayout tc_layout(int d, int C, int nzb, int infix) {
  TcLayout L;
  L.nch = (d + kChunkF - 1) / kChunkF;
  L.Cpad = (C + 15) / 16 * 16;
  L.nzb = nzb;
  L.infix = infix;
  L.wbytes = (uint32_t)L.nch * (uint32_t)L.Cpad * 128u;  // a multiple of 2048
  L.zbytes = (uint32_t)L.nch * kZChunkBytes;
  L.off_z = L.wbytes;
  L.off_bias = L.off_z + (uint32_t)nzb * L.zbytes;
  L.off_wn = L.off_bias + 256 * 4;
  L.off_list = L.off_wn + 256 * 4;
  L.off_x1 = L.off_list + kEpiWarps * kWarpScratch;
  L.off_x2 = L.off_x1 + 2 * kBM * (uint32_t)sizeof(Pass1);
  L.off_acc = L.off_x2 + kBM * (uint32_t)sizeof(Top2);
  L.off_bar = (L.off_acc + kBM + 32 + 7) / 8 * 8;  // + ok flags of the halves (2 x 4 ints)
  L.off_misc = L.off_bar + (8 + 2 * kMaxChunks) * 8;  // the barrier map is in the kernel
  L.off_fixq = L.off_misc + 16;
  L.off_fixs = (L.off_fixq + (infix ? (uint32_t)sizeof(FixQueue) : 0u) + 15) / 16 * 16;
  L.total = L.off_fixs + (infix ? (uint32_t)fix_scratch_bytes(d, C) : 0u);
  return L;
}

// Packed FP32 pairs: two additions / multiplications in one instruction (each
// lane rounded to nearest, as the scalar operation), and packing.
__device__ __forceinline__ uint64_t add_f32x2(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__device__ __forceinline__ uint64_t mul_f32x2(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__device__ __forceinline__ uint64_t pack2_f32(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void unpack2_f32(uint64_t v, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
// Byte offset of feature k of row r in a 128-byte-swizzled K-major tile whose
// 32-feature chunks are `chunk_bytes` apart (TMA SWIZZLE_128B: the 16-byte
// unit index is XORed with the row index mod 8).
__device__ __forceinline__ uint32_t sw_off(int r, int k, uint32_t chunk_bytes) {
  return (uint32_t)(k >> 5) * chunk_bytes + (uint32_t)r * 128u + ((((uint32_t)(k >> 2) & 7u) ^ ((uint32_t)r & 7u)) << 4) +
         (((uint32_t)k & 3u) << 2);
}

// 16 bytes of shared memory at byte address `addr` (16-byte aligned).
__device__ __forceinline__ float4 lds_f4(uint32_t addr) {
  float4 v;
  asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];" : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w) : "r"(addr));
  return v;
}

// Named barrier of the two epilogue warps of one lane quarter.
__device__ __forceinline__ void pair_barrier(int id) { asm volatile("bar.sync %0, 64;" ::"r"(id) : "memory"); }

// The resident head in shared memory (TMA 128-byte swizzle, 32-feature chunks
// wchunk bytes apart) as the FP64 pass reads it.
struct WSwz {
  uint32_t s_w, wchunk;
  __device__ __forceinline__ float operator()(int c, int j) const {
    float v;
    asm volatile("ld.shared.f32 %0, [%1];" : "=f"(v) : "r"(s_w + sw_off(c, j, wchunk)));
    return v;
  }
  // sum_j W_cj zs_j for NP classes, fused multiply-adds in feature order
  // (d % 16 == 0), four features per 16-byte load
  template <int NP>
  __device__ __forceinline__ void chains(const int (&cc)[NP], const float* __restrict__ zs, int d,
                                         float (&acc)[NP]) const {
    uint32_t rb[NP], x[NP];
#pragma unroll
    for (int t = 0; t < NP; ++t) {
      rb[t] = s_w + (uint32_t)cc[t] * 128u;
      x[t] = (uint32_t)cc[t] & 7u;
      acc[t] = 0.f;
    }
    for (int k = 0; k < d; k += kChunkF) {
      const uint32_t co = (uint32_t)(k / kChunkF) * wchunk;
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        if (k + 4 * u < d) {
          const float4 z = *reinterpret_cast<const float4*>(zs + k + 4 * u);
#pragma unroll
          for (int t = 0; t < NP; ++t) {
            const float4 w = lds_f4(rb[t] + co + ((((uint32_t)u) ^ x[t]) << 4));
            acc[t] = fmaf(w.x, z.x, acc[t]);
            acc[t] = fmaf(w.y, z.y, acc[t]);
            acc[t] = fmaf(w.z, z.z, acc[t]);
            acc[t] = fmaf(w.w, z.w, acc[t]);
          }
        }
      }
    }
  }
};

// Hand a listed row to the fix warp (one lane; after the row's results are
// written). Waits, bounded, for a free slot; false if the kernel aborted.
__device__ __noinline__ bool fixq_push(FixQueue* q, int row, float kn, volatile int* abort_s, long long limit) {
  __threadfence_block();  // the row's results before the entry
  const int k = atomicAdd(&q->n, 1);
  volatile int* taken = &q->taken;
  if (*taken <= k - kFixQ) {
    const long long t0 = clock64();
    while (*taken <= k - kFixQ) {
      if (*abort_s) return false;
      if (clock64() - t0 > limit) {
        *abort_s = 1;
        return false;
      }
      __nanosleep(128);
    }
  }
  const int sl = k % kFixQ;
  q->row[sl] = row;
  q->kn[sl] = kn;
  __threadfence_block();
  *(volatile int*)&q->seq[sl] = k;
  return true;
}

// Top2 over the union of two disjoint class sets from the two sets' states:
// the same y^G, runner-up value and bounds as pushing every class into one.
__device__ __forceinline__ void top2_merge(Top2& A, const Top2& B) {
  const bool b_best = B.y >= 0 && (A.y < 0 || pair_gt(B.b1h, B.b1l, A.b1h, A.b1l) ||
                                   (B.b1h == A.b1h && B.b1l == A.b1l && B.y < A.y));
  const Top2& Wn = b_best ? B : A;
  const Top2& Ls = b_best ? A : B;
  float sh = Wn.b2h, sl = Wn.b2l;
  if (pair_gt(Ls.b1h, Ls.b1l, sh, sl) || (Ls.b1h == sh && Ls.b1l == sl)) {
    sh = Ls.b1h;
    sl = Ls.b1l;
  }
  // largest upper bound among the classes other than the winner
  const float up = fmaxf((Wn.cu1 == Wn.y) ? Wn.u2 : Wn.u1, Ls.u1);
  Top2 R;
  R.b1h = Wn.b1h;
  R.b1l = Wn.b1l;
  R.e1 = Wn.e1;
  R.y = Wn.y;
  R.b2h = sh;
  R.b2l = sl;
  R.u1 = up;
  R.u2 = up;
  R.cu1 = -2;
  R.em = fmaxf(A.em, B.em);
  R.nan = A.nan || B.nan;
  A = R;
}

// Compensated dot products W_c . z_r + b_c of two (row, class) pairs by the 8
// lanes of a group (lane sub takes features sub, sub + 8, ...; the two chains
// interleaved for instruction-level parallelism), each in exactly the order of
// the wide-tile kernel's refinement: TwoProduct and TwoSum per feature, a
// butterfly over the group, then the bias. Every lane of the group returns the
// same pairs hi + lo. ws / zs: shared-memory byte addresses of the head and of
// the tile's features (128-byte swizzle, chunks wchunk / kZChunkBytes apart).
__device__ __forceinline__ void refine2(uint32_t ws, uint32_t wchunk, uint32_t zs, const int (&c)[2],
                                        const int (&r)[2], const float (&bias)[2], int d, int sub, float (&hi)[2],
                                        float (&lo)[2]) {
  // lane sub reads the 16-byte unit 2 jj + sub / 4 of each 32-feature chunk
  // (jj = 0..3), word sub % 4; the swizzle XORs the unit with the row mod 8
  const uint32_t s2 = (uint32_t)sub >> 2, s3 = ((uint32_t)sub & 3u) << 2;
  uint32_t wb[2], zb[2], ow[2][4], oz[2][4];
#pragma unroll
  for (int u = 0; u < 2; ++u) {
    wb[u] = ws + (uint32_t)c[u] * 128u + s3;
    zb[u] = zs + (uint32_t)r[u] * 128u + s3;
#pragma unroll
    for (int jj = 0; jj < 4; ++jj) {
      ow[u][jj] = ((2u * jj + s2) ^ ((uint32_t)c[u] & 7u)) << 4;
      oz[u][jj] = ((2u * jj + s2) ^ ((uint32_t)r[u] & 7u)) << 4;
    }
  }
  // both chains in packed FP32 pairs: (pair 0, pair 1) in (low, high) halves;
  // every operation rounds each half exactly as the scalar one would
  uint64_t P = 0ull, CC = 0ull;
  constexpr uint64_t kSign2 = 0x8000000080000000ull;
  auto step = [&](uint32_t wa0, uint32_t za0, uint32_t wa1, uint32_t za1) {
    float w0, x0, w1, x1;
    asm volatile("ld.shared.f32 %0, [%1];" : "=f"(w0) : "r"(wa0));
    asm volatile("ld.shared.f32 %0, [%1];" : "=f"(x0) : "r"(za0));
    asm volatile("ld.shared.f32 %0, [%1];" : "=f"(w1) : "r"(wa1));
    asm volatile("ld.shared.f32 %0, [%1];" : "=f"(x1) : "r"(za1));
    const uint64_t w = pack2_f32(w0, w1), x = pack2_f32(x0, x1);
    const uint64_t pr = mul_f32x2(w, x);                // TwoProduct: pr + er = w x
    const uint64_t er = ptx::fma_f32x2(w, x, pr ^ kSign2);
    const uint64_t sm = add_f32x2(P, pr);               // TwoSum(P, pr) = sm + q
    const uint64_t bb = ptx::sub_f32x2(sm, P);
    const uint64_t q = add_f32x2(ptx::sub_f32x2(P, ptx::sub_f32x2(sm, bb)), ptx::sub_f32x2(pr, bb));
    P = sm;
    CC = add_f32x2(CC, add_f32x2(q, er));
  };
  // a chunk's sixteen loads are issued together, then its four steps (the
  // loads are volatile, so their order is the program's)
  auto ld = [](uint32_t addr) {
    float v;
    asm volatile("ld.shared.f32 %0, [%1];" : "=f"(v) : "r"(addr));
    return v;
  };
  auto step_v = [&](float w0, float x0, float w1, float x1) {
    const uint64_t w = pack2_f32(w0, w1), x = pack2_f32(x0, x1);
    const uint64_t pr = mul_f32x2(w, x);                // TwoProduct: pr + er = w x
    const uint64_t er = ptx::fma_f32x2(w, x, pr ^ kSign2);
    const uint64_t sm = add_f32x2(P, pr);               // TwoSum(P, pr) = sm + q
    const uint64_t bb = ptx::sub_f32x2(sm, P);
    const uint64_t q = add_f32x2(ptx::sub_f32x2(P, ptx::sub_f32x2(sm, bb)), ptx::sub_f32x2(pr, bb));
    P = sm;
    CC = add_f32x2(CC, add_f32x2(q, er));
  };
  const int nfull = d >> 5;
  for (int kc = 0; kc < nfull; ++kc) {
    float w0[4], x0[4], w1[4], x1[4];
#pragma unroll
    for (int jj = 0; jj < 4; ++jj) {
      w0[jj] = ld(wb[0] + ow[0][jj]);
      x0[jj] = ld(zb[0] + oz[0][jj]);
      w1[jj] = ld(wb[1] + ow[1][jj]);
      x1[jj] = ld(zb[1] + oz[1][jj]);
    }
#pragma unroll
    for (int jj = 0; jj < 4; ++jj) step_v(w0[jj], x0[jj], w1[jj], x1[jj]);
#pragma unroll
    for (int u = 0; u < 2; ++u) {
      wb[u] += wchunk;
      zb[u] += kZChunkBytes;
    }
  }
  if (d & 16) {  // a last half chunk (d % 32 == 16): units 0-3
#pragma unroll
    for (int jj = 0; jj < 2; ++jj) step(wb[0] + ow[0][jj], zb[0] + oz[0][jj], wb[1] + ow[1][jj], zb[1] + oz[1][jj]);
  }
  float p[2], cc[2];
  unpack2_f32(P, p[0], p[1]);
  unpack2_f32(CC, cc[0], cc[1]);
#pragma unroll
  for (int o = kGroupTc / 2; o > 0; o >>= 1) {
#pragma unroll
    for (int u = 0; u < 2; ++u) {
      const float pb = __shfl_xor_sync(kFull, p[u], o), cb = __shfl_xor_sync(kFull, cc[u], o);
      float t, q;
      two_sum(p[u], pb, t, q);
      p[u] = t;
      cc[u] = __fadd_rn(__fadd_rn(cc[u], cb), q);
    }
  }
#pragma unroll
  for (int u = 0; u < 2; ++u) {
    float t, q;
    two_sum(p[u], bias[u], t, q);
    two_sum(t, __fadd_rn(cc[u], q), hi[u], lo[u]);
  }
}

// The same compensated dot product W_c . z_r + b_c as refine2, for one
// (row, class) pair on one lane, with the same bits: the eight chains of
// refine2's group (lane s: features s, s + 8, s + 16, ... in ascending order)
// run side by side in this lane, then the group's butterfly (xor 4, 2, 1) is
// taken in the same tree inside the lane, then the bias. TwoSum's error term
// is the exact rounding error whichever operand comes first and FP32 addition
// commutes, so after each level every lane of refine2's group holds the pair
// this lane holds (checked by an FP32 emulation of both layouts on the CPU).
// Eight independent chains per lane instead of one, and no shuffles. The
// chains are scalar: packing them two to an FP32x2 register costs a move per
// operand and a sign flip per product on the integer pipe, which measured
// slower. The next span's four 16-byte loads are issued before this span's
// arithmetic.
__device__ __forceinline__ void refine_lane(uint32_t ws, uint32_t wchunk, uint32_t zs, int c, int r, float bias, int d,
                                            float& hi, float& lo) {
  const uint32_t xw = (uint32_t)c & 7u, xz = (uint32_t)r & 7u;
  const uint32_t wrow = ws + (uint32_t)c * 128u, zrow = zs + (uint32_t)r * 128u;
  // span i: features 8 i .. 8 i + 7 = units 2 (i % 4) (chains 0-3) and
  // 2 (i % 4) + 1 (chains 4-7) of chunk i / 4, swizzled with the row mod 8;
  // the second unit's address is the first's with bit 4 flipped
  auto aw = [&](int i) { return wrow + (uint32_t)(i >> 2) * wchunk + (((2u * (uint32_t)(i & 3)) ^ xw) << 4); };
  auto az = [&](int i) { return zrow + (uint32_t)(i >> 2) * kZChunkBytes + (((2u * (uint32_t)(i & 3)) ^ xz) << 4); };
  float p[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f}, cc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  auto span = [&](const float4& w0, const float4& w1, const float4& z0, const float4& z1) {
    const float w[8] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
    const float x[8] = {z0.x, z0.y, z0.z, z0.w, z1.x, z1.y, z1.z, z1.w};
#pragma unroll
    for (int s = 0; s < 8; ++s) {
      const float pr = __fmul_rn(w[s], x[s]);  // TwoProduct: pr + er = w x
      const float er = __fmaf_rn(w[s], x[s], -pr);
      const float sm = __fadd_rn(p[s], pr);    // TwoSum(p, pr) = sm + q
      const float bb = __fsub_rn(sm, p[s]);
      const float q = __fadd_rn(__fsub_rn(p[s], __fsub_rn(sm, bb)), __fsub_rn(pr, bb));
      p[s] = sm;
      cc[s] = __fadd_rn(cc[s], __fadd_rn(q, er));
    }
  };
  const int nsp = d >> 3;  // (d % 16 == 0)
  float4 w0 = lds_f4(aw(0)), w1 = lds_f4(aw(0) ^ 16u), z0 = lds_f4(az(0)), z1 = lds_f4(az(0) ^ 16u);
#pragma unroll 2
  for (int i = 0; i < nsp; ++i) {
    const int n = i + 1 < nsp ? i + 1 : i;  // (the last span loads itself again)
    const uint32_t anw = aw(n), anz = az(n);
    const float4 nw0 = lds_f4(anw), nw1 = lds_f4(anw ^ 16u), nz0 = lds_f4(anz), nz1 = lds_f4(anz ^ 16u);
    span(w0, w1, z0, z1);
    w0 = nw0;
    w1 = nw1;
    z0 = nz0;
    z1 = nz1;
  }
#pragma unroll
  for (int o = kGroupTc / 2; o > 0; o >>= 1) {
#pragma unroll
    for (int s = 0; s < o; ++s) {
      float t, q;
      two_sum(p[s], p[s + o], t, q);
      p[s] = t;
      cc[s] = __fadd_rn(__fadd_rn(cc[s], cc[s + o]), q);
    }
  }
  float t, q;
  two_sum(p[0], bias, t, q);
  two_sum(t, __fadd_rn(cc[0], q), hi, lo);
}

// refine_lane with the pair shared by K = 2 or 4 lanes (t = lane % K), for
// the last pairs of a list, which would leave most lanes of a whole round
// idle. K = 2: lane t runs chains 4 t .. 4 t + 3 (the 16-byte unit 2 jj + t
// of each span); the butterfly's first level (chain s with s + 4) is a
// shuffle with lane t ^ 1, the others stay in the lane. K = 4: lane t runs
// chains t and t + 4 (word t of both units); the first level is in the lane,
// the second (s with s + 2) a shuffle with lane t ^ 2, the third with t ^ 1.
// Every lane of the K returns the same bits as refine_lane. All 32 lanes call
// it together (the shuffles take the whole warp).
template <int K>
__device__ __forceinline__ void refine_lanes(uint32_t ws, uint32_t wchunk, uint32_t zs, int c, int r, float bias, int d,
                                             int t, float& hi, float& lo) {
  static_assert(K == 2 || K == 4, "two or four lanes per pair");
  constexpr int NC = 8 / K;  // chains per lane
  const uint32_t xw = (uint32_t)c & 7u, xz = (uint32_t)r & 7u;
  const uint32_t wrow = ws + (uint32_t)c * 128u, zrow = zs + (uint32_t)r * 128u;
  float p[NC], cc[NC];
#pragma unroll
  for (int j = 0; j < NC; ++j) p[j] = cc[j] = 0.f;
  auto step = [&](int j, float w, float x) {
    const float pr = __fmul_rn(w, x);
    const float er = __fmaf_rn(w, x, -pr);
    const float sm = __fadd_rn(p[j], pr);
    const float bb = __fsub_rn(sm, p[j]);
    const float q = __fadd_rn(__fsub_rn(p[j], __fsub_rn(sm, bb)), __fsub_rn(pr, bb));
    p[j] = sm;
    cc[j] = __fadd_rn(cc[j], __fadd_rn(q, er));
  };
  const int nsp = d >> 3;
  for (int i = 0; i < nsp; ++i) {
    const uint32_t u = 2u * (uint32_t)(i & 3);  // first unit of the span
    const uint32_t ow = (uint32_t)(i >> 2) * wchunk, oz = (uint32_t)(i >> 2) * kZChunkBytes;
    if constexpr (K == 2) {
      const float4 w = lds_f4(wrow + ow + (((u + (uint32_t)t) ^ xw) << 4));
      const float4 z = lds_f4(zrow + oz + (((u + (uint32_t)t) ^ xz) << 4));
      step(0, w.x, z.x);
      step(1, w.y, z.y);
      step(2, w.z, z.z);
      step(3, w.w, z.w);
    } else {
      float w0, w1, z0, z1;
      asm volatile("ld.shared.f32 %0, [%1];" : "=f"(w0) : "r"(wrow + ow + ((u ^ xw) << 4) + 4u * (uint32_t)t));
      asm volatile("ld.shared.f32 %0, [%1];" : "=f"(w1) : "r"(wrow + ow + (((u + 1u) ^ xw) << 4) + 4u * (uint32_t)t));
      asm volatile("ld.shared.f32 %0, [%1];" : "=f"(z0) : "r"(zrow + oz + ((u ^ xz) << 4) + 4u * (uint32_t)t));
      asm volatile("ld.shared.f32 %0, [%1];" : "=f"(z1) : "r"(zrow + oz + (((u + 1u) ^ xz) << 4) + 4u * (uint32_t)t));
      step(0, w0, z0);  // chain t
      step(1, w1, z1);  // chain t + 4
    }
  }
  auto comb = [](float& pa, float& ca, float pb, float cb) {
    float s, q;
    two_sum(pa, pb, s, q);
    pa = s;
    ca = __fadd_rn(__fadd_rn(ca, cb), q);
  };
  if constexpr (K == 2) {
#pragma unroll
    for (int j = 0; j < 4; ++j) comb(p[j], cc[j], __shfl_xor_sync(kFull, p[j], 1), __shfl_xor_sync(kFull, cc[j], 1));
    comb(p[0], cc[0], p[2], cc[2]);
    comb(p[1], cc[1], p[3], cc[3]);
    comb(p[0], cc[0], p[1], cc[1]);
  } else {
    comb(p[0], cc[0], p[1], cc[1]);
    comb(p[0], cc[0], __shfl_xor_sync(kFull, p[0], 2), __shfl_xor_sync(kFull, cc[0], 2));
    comb(p[0], cc[0], __shfl_xor_sync(kFull, p[0], 1), __shfl_xor_sync(kFull, cc[0], 1));
  }
  float tt, q;
  two_sum(p[0], bias, tt, q);
  two_sum(tt, __fadd_rn(cc[0], q), hi, lo);
}

// The tight radius (Eq. 29) of one row on one warp, for rows the screen
// cannot settle (several possible y^G, Mb not below 1e38, more candidates than
// slots): every class refined with the compensated dot product by the four
// 8-lane groups, two classes per group at a time (refine2, the error factor of
// 8-lane groups), into the warp's result cells by class; then, lane = class,
// y^G the largest refined logit (lowest class on ties) and Eq. 29 over every
// other class in FP64. The row's features come from the tile in shared memory
// (row rz). res_hi / res_lo: the warp's cells (at least 256 each), free here.
// Returns (on every lane) whether the row was listed for the FP64 pass.
__device__ bool tc_tight_row_warp(const CertArgs& a, int64_t row, int rz, uint32_t s_w, uint32_t wchunk, uint32_t zs,
                                  const float* __restrict__ wn_s, const float* __restrict__ b_s, float kn, int lane,
                                  float* res_hi, float* res_lo, uint8_t* acc_slot) {
  constexpr int kPer = 8;  // classes per lane (C <= 256)
  const int d = a.d, C = a.C;
  const int g8 = lane / kGroupTc, sub = lane % kGroupTc;
  const float hn = norm_upper(kn);
  for (int c0 = 0; c0 < C; c0 += 2 * (32 / kGroupTc)) {
    int cp[2];
#pragma unroll
    for (int u = 0; u < 2; ++u) {
      const int c = c0 + 2 * g8 + u;
      cp[u] = c < C ? c : C - 1;  // a valid class; the result is not stored
    }
    const int rp[2] = {rz, rz};
    const float bp[2] = {b_s[cp[0]], b_s[cp[1]]};
    float hi[2], lo[2];
    refine2(s_w, wchunk, zs, cp, rp, bp, d, sub, hi, lo);
    if (sub == 0)
#pragma unroll
      for (int u = 0; u < 2; ++u)
        if (c0 + 2 * g8 + u < C) {
          res_hi[c0 + 2 * g8 + u] = hi[u];
          res_lo[c0 + 2 * g8 + u] = lo[u];
        }
  }
  __syncwarp();
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
      const float hi = res_hi[c], lo = res_lo[c];
      vh[t] = hi;
      vl[t] = lo;
      ve[t] = refined_err(a.g2f8, wn_s[c], hn, b_s[c]);
      nan_any |= !(hi == hi && lo == lo);
      if (pair_gt(hi, lo, bh, bl)) {  // ascending classes: ties keep the lowest
        bh = hi;
        bl = lo;
        by = c;
      }
    }
  }
  __syncwarp();  // the cells are read before the next row's refinement
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
  bool fix = false;
  if (lane == 0) fix = tight_write(a, row, y, rmin, smin, nan_any, kn, acc_slot);
  return __shfl_sync(kFull, fix ? 1 : 0, 0) != 0;
}

template <bool TIGHT>
__global__ void __launch_bounds__(kThreads, 1)
    k_certify_tc(const __grid_constant__ CUtensorMap tmH, const __grid_constant__ CUtensorMap tmW, const CertArgs a,
                 const TcLayout L, int n_tiles, DevStats* stats, int debug_stall) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* smem =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  const uint32_t s_base = ptx::smem_u32(smem);
  const uint32_t s_w = s_base, s_z = s_base + L.off_z;
  const uint32_t bar = s_base + L.off_bar;
  // barriers: wfull, zempty[2], accfull[2], accempty[2], drain, zfull[2][kMaxChunks]
  // (one per 32-feature chunk of each feature buffer, so the MMAs start on
  // the first chunk while the others land)
  const uint32_t wfull = bar, zempty = bar + 8, accfull = bar + 24, accempty = bar + 40, drain = bar + 56,
                 zfull = bar + 64;
  auto zfull_of = [&](int zb, int c) { return zfull + 8u * (uint32_t)(zb * kMaxChunks + c); };
  float* bias_s = reinterpret_cast<float*>(smem + L.off_bias);
  float* wn_s = reinterpret_cast<float*>(smem + L.off_wn);
  unsigned char* scratch = smem + L.off_list;
  Pass1* x1 = reinterpret_cast<Pass1*>(smem + L.off_x1);
  Top2* x2 = reinterpret_cast<Top2*>(smem + L.off_x2);
  uint8_t* acc_s = smem + L.off_acc;
  volatile int* okf = reinterpret_cast<volatile int*>(smem + L.off_acc + kBM);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L.off_misc);
  volatile int* abort_s = reinterpret_cast<volatile int*>(smem + L.off_misc + 4);
  FixQueue* fixq = L.infix ? reinterpret_cast<FixQueue*>(smem + L.off_fixq) : nullptr;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int d = a.d, C = a.C;
  if (threadIdx.x == 0) {
    ptx::mbar_init(wfull, 1);
    for (int b = 0; b < 2; ++b) {
      for (int c = 0; c < kMaxChunks; ++c) ptx::mbar_init(zfull_of(b, c), 1);
      ptx::mbar_init(zempty + 8 * b, kEpiWarps);
      ptx::mbar_init(accfull + 8 * b, 1);
      ptx::mbar_init(accempty + 8 * b, kEpiWarps);
    }
    ptx::mbar_init(drain, 1);
    *abort_s = 0;
    if (fixq) {
      fixq->n = fixq->taken = fixq->done = fixq->beat = 0;
      for (int i = 0; i < kFixQ; ++i) fixq->seq[i] = -1;
    }
    ptx::fence_mbar_init();
    ptx::tma_prefetch_desc(&tmH);
    ptx::tma_prefetch_desc(&tmW);
  }
  for (int i = threadIdx.x; i < 256; i += kThreads) {
    bias_s[i] = i < C ? __ldg(a.b + i) : 0.f;
    wn_s[i] = i < C ? __ldg(a.Wnorm32 + i) : 0.f;
  }
  if (warp == 1) {
    ptx::tmem_alloc(ptx::smem_u32(tmem_slot), kTmemCols);
    ptx::tmem_relinquish();
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      ptx::mbar_expect_tx(wfull, L.wbytes);
      for (int c = 0; c < L.nch; ++c)
        ptx::tma_load_2d(s_w + (uint32_t)c * (uint32_t)L.Cpad * 128u, &tmW, c * kChunkF, 0, wfull);
      bool used[2] = {false, false};
      uint32_t lastp[2] = {0u, 0u};
      int t = 0;
      for (int tile = blockIdx.x; tile < n_tiles; tile += gridDim.x, ++t) {
        const int zb = t % L.nzb;
        const uint32_t par = (uint32_t)(t / L.nzb) & 1u;
        if (!ptx::mbar_wait(zempty + 8 * zb, par ^ 1u, abort_s, kWaitLimit)) break;
        for (int c = 0; c < L.nch; ++c) {
          ptx::mbar_expect_tx(zfull_of(zb, c), kZChunkBytes);
          ptx::tma_load_2d(s_z + (uint32_t)zb * L.zbytes + (uint32_t)c * kZChunkBytes, &tmH, c * kChunkF, tile * kBM,
                           zfull_of(zb, c));
        }
        used[zb] = true;
        lastp[zb] = par;
        // the CTA's next tile starts moving into L2 while this one is worked on
        const int nxt = tile + (int)gridDim.x;
        if (nxt < n_tiles) {
          const int64_t r0 = (int64_t)nxt * kBM;
          const int64_t nr = a.n - r0 < kBM ? a.n - r0 : kBM;
          prefetch_l2_bulk(a.H + (size_t)r0 * d, (uint32_t)(nr * d * sizeof(float)));
        }
      }
      // every copy into this CTA lands before it can exit (bounded; a phase
      // that already completed returns at once)
      volatile int never = 0;
      for (int b = 0; b < 2; ++b)
        for (int c = 0; c < L.nch && used[b]; ++c) ptx::mbar_wait(zfull_of(b, c), lastp[b], &never, kWaitLimit);
      ptx::mbar_wait(wfull, 0, &never, kWaitLimit);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t idesc = ptx::idesc_tf32(kBM, L.Cpad);
      const uint64_t zdesc0 = ptx::sw128_kmajor_desc(s_z), wdesc0 = ptx::sw128_kmajor_desc(s_w);
      const uint64_t zstep = kZChunkBytes >> 4, wstep = ((uint32_t)L.Cpad * 128u) >> 4, zbstep = L.zbytes >> 4;
      // failure-detection test: no arrival completes this phase before the
      // final drain, so the bounded wait expires and the kernel aborts
      bool ok = !debug_stall || ptx::mbar_wait(drain, 0, abort_s, kWaitLimit);
      ok = ok && ptx::mbar_wait(wfull, 0, abort_s, kWaitLimit);
      int t = 0;
      for (int tile = blockIdx.x; tile < n_tiles && ok; tile += gridDim.x, ++t) {
        const int buf = t & 1, zb = t % L.nzb;
        ok = ptx::mbar_wait(accempty + 8 * buf, ((uint32_t)(t >> 1) & 1u) ^ 1u, abort_s, kWaitLimit);
        if (!ok) break;
        ptx::tc_fence_after();
        const uint32_t d_tmem = tmem + (uint32_t)buf * kAccStride;
        uint64_t zd = zdesc0 + (uint64_t)zb * zbstep, wd = wdesc0;
        for (int c = 0; c < L.nch; ++c, zd += zstep, wd += wstep) {
          if (!ptx::mbar_wait(zfull_of(zb, c), (uint32_t)(t / L.nzb) & 1u, abort_s, kWaitLimit)) {
            ok = false;
            break;
          }
          ptx::tc_fence_after();
          ptx::mma_tf32(d_tmem, zd, wd, idesc, c != 0);
          ptx::mma_tf32(d_tmem, zd + 2, wd + 2, idesc, 1u);
          ptx::mma_tf32(d_tmem, zd + 4, wd + 4, idesc, 1u);
          ptx::mma_tf32(d_tmem, zd + 6, wd + 6, idesc, 1u);
        }
        if (!ok) break;
        ptx::mma_commit(accfull + 8 * buf);
      }
      // every issued MMA completes before TMEM can be released
      volatile int never = 0;
      ptx::mma_commit(drain);
      ptx::mbar_wait(drain, 0, &never, kWaitLimit);
    }
    __syncwarp();
  } else if (warp == kFixWarp) {
    // ------------------------------------------------------------ FP64 pass
    // the rows the epilogue lists, one at a time, while the epilogue goes on
    // with later tiles (fix_row_warp); the head is read in place
    if (fixq) {
      const WSwz W{s_w, (uint32_t)L.Cpad * 128u};
      const FixScratch sc = fix_scratch_at(smem + L.off_fixs, d, C);
      volatile FixQueue* vq = fixq;
      bool head_ok = false;
      unsigned long long nfixed = 0;
      for (int k = 0;; ++k) {
        // 1: entry k is in its slot; 0: every epilogue warp is done and no
        // entry k will come, or the kernel aborted. The wait is bounded by
        // the epilogue's progress (a tile every few microseconds).
        int st = 0;
        if (lane == 0) {
          int beat = vq->beat;
          long long t0 = clock64();
          for (;;) {
            if (vq->seq[k % kFixQ] == k) {
              st = 1;
              break;
            }
            if (*abort_s) break;
            if (vq->done == kEpiWarps) {
              __threadfence_block();
              if (vq->n <= k) break;  // (else the entry is being written)
            }
            const int b = vq->beat;
            if (b != beat) {
              beat = b;
              t0 = clock64();
            } else if (clock64() - t0 > kWaitLimit) {
              *abort_s = 1;
              break;
            }
            __nanosleep(256);
          }
        }
        if (__shfl_sync(kFull, st, 0) == 0) break;
        __threadfence_block();
        const int row = vq->row[k % kFixQ];
        const float kn = vq->kn[k % kFixQ];
        if (!head_ok) head_ok = __all_sync(kFull, ptx::mbar_wait(wfull, 0, abort_s, kWaitLimit));
        if (!head_ok) break;
        fix_row_warp(a, (int64_t)row, kn, W, sc, lane);
        ++nfixed;
        __syncwarp();
        if (lane == 0) {
          __threadfence_block();
          vq->taken = k + 1;
        }
      }
      if (lane == 0 && nfixed) atomicAdd(&stats->ins_fp64_rows, nfixed);
    }
  } else if (warp < 2 + kEpiWarps) {
    // ------------------------------------------------------------ epilogue
    const int ew = warp - 2, quarter = warp & 3, half = ew >> 2;
    const int r = quarter * 32 + lane;  // row of the tile = TMEM lane
    const int nck = (C + 31) / 32;
    // this half's classes: the 32-column chunks half, half + 2, ... (t-th
    // class of the half: chunk 2 (t / 32) + half, column t % 32)
    int ncls = 0;
    for (int ch = half; ch < nck; ch += 2) ncls += min(32, C - ch * 32);
    const int g8 = lane / kGroupTc, sub = lane % kGroupTc;
    // the warp's pair list (row lane | slot << 5 | class << 8) and the refined
    // values by (row lane, slot)
    int* list = reinterpret_cast<int*>(scratch + (size_t)ew * kWarpScratch);
    float* res_hi = reinterpret_cast<float*>(scratch + (size_t)ew * kWarpScratch + kListCap * 4);
    float* res_lo = res_hi + 32 * kMaxCandTc;
    const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
    const int dq = d / 4;
    const int bar_id = 1 + quarter;
    const uint32_t wchunk = (uint32_t)L.Cpad * 128u;
    // screen bound terms: c ||W_c|| <= cw and (1 + c) ||W_c|| <= cw1 for every
    // class, |b_c| <= bmax (rounded up; a NaN bias propagates into bmax)
    float wmax = 0.f, bmax = 0.f;
    for (int c = lane; c < C; c += 32) {
      wmax = fmaxf(wmax, __ldg(a.Wnorm32 + c));
      const float ab = fabsf(__ldg(a.b + c));
      bmax = (ab > bmax || ab != ab) ? ab : bmax;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      wmax = fmaxf(wmax, __shfl_xor_sync(kFull, wmax, o));
      const float ob = __shfl_xor_sync(kFull, bmax, o);
      bmax = (ob > bmax || ob != ob) ? ob : bmax;
    }
    // tight radius: the smallest lower bound of 1 / ||W_y - W_j|| over the
    // head
    float imA = INFINITY;
    if constexpr (TIGHT) {
      for (int c = lane; c < C; c += 32) imA = fminf(imA, __ldg(a.ipn_min32 + c));
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) imA = fminf(imA, __shfl_xor_sync(kFull, imA, o));
    }
    const float c32 = __double2float_ru(a.c_scr);
    const float cw = __fmul_ru(c32, wmax), cw1 = __fmul_ru(__fadd_ru(1.f, c32), wmax);
    // top two of the s~ in a 32-column chunk, four independent trackers
    // (columns j % 4); columns past C are masked when the chunk is partial
    auto pass1_chunk = [&](const uint32_t (&v)[32], int ch, float (&t1)[4], float (&t2)[4]) {
      const int lim = min(32, C - ch * 32);
      const float4* b4 = reinterpret_cast<const float4*>(bias_s + ch * 32);
      if (lim == 32) {
        // a full chunk, two values at a time: with hi / lo the larger /
        // smaller of the two, the new second largest is the largest of t2,
        // min(t1, hi) and lo (five min / max for two values instead of six,
        // and no mask)
#pragma unroll
        for (int j4 = 0; j4 < 8; ++j4) {
          const float4 bb = b4[j4];
          const float bv[4] = {bb.x, bb.y, bb.z, bb.w};
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const int k = 2 * (j4 & 1) + h;  // tracker
            const float sa = __fadd_rn(__uint_as_float(v[4 * j4 + 2 * h]), bv[2 * h]);
            const float sb = __fadd_rn(__uint_as_float(v[4 * j4 + 2 * h + 1]), bv[2 * h + 1]);
            const float hi2 = fmaxf(sa, sb), lo2 = fminf(sa, sb);
            t2[k] = ptx::max3_f32(t2[k], fminf(t1[k], hi2), lo2);
            t1[k] = fmaxf(t1[k], hi2);
          }
        }
        return;
      }
#pragma unroll
      for (int j4 = 0; j4 < 8; ++j4) {
        const float4 bb = b4[j4];
        const float bv[4] = {bb.x, bb.y, bb.z, bb.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int j = 4 * j4 + e;
          float sv = __fadd_rn(__uint_as_float(v[j]), bv[e]);
          sv = (lim == 32 || j < lim) ? sv : -INFINITY;
          t2[e] = fmaxf(t2[e], fminf(t1[e], sv));
          t1[e] = fmaxf(t1[e], sv);
        }
      }
    };
    // the candidates of a chunk: bit j set iff s~ >= T
    auto pass2_chunk = [&](const uint32_t (&v)[32], int ch, float T) -> uint32_t {
      const int lim = min(32, C - ch * 32);
      const float4* b4 = reinterpret_cast<const float4*>(bias_s + ch * 32);
      uint32_t mask = 0;
#pragma unroll
      for (int j4 = 0; j4 < 8; ++j4) {
        const float4 bb = b4[j4];
        const float bv[4] = {bb.x, bb.y, bb.z, bb.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int j = 4 * j4 + e;
          const float sv = __fadd_rn(__uint_as_float(v[j]), bv[e]);
          mask |= (uint32_t)(sv >= T) << j;
        }
      }
      return lim == 32 ? mask : mask & ((1u << lim) - 1u);
    };
    // tight radius: the top two with their classes (four trackers), and the
    // candidates of Eq. 29: bit j set unless (lo_y - hi_j) ipn_min(y) > U
    auto pass1_chunk_idx = [&](const uint32_t (&v)[32], int ch, float (&t1)[4], int (&i1)[4], float (&t2)[4],
                               int (&i2)[4]) {
      const int lim = min(32, C - ch * 32);
      const float4* b4 = reinterpret_cast<const float4*>(bias_s + ch * 32);
#pragma unroll
      for (int j4 = 0; j4 < 8; ++j4) {
        const float4 bb = b4[j4];
        const float bv[4] = {bb.x, bb.y, bb.z, bb.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int j = 4 * j4 + e, c = ch * 32 + j;
          float sv = __fadd_rn(__uint_as_float(v[j]), bv[e]);
          sv = (lim == 32 || j < lim) ? sv : -INFINITY;
          const bool g1 = sv > t1[e], g2 = sv > t2[e];
          t2[e] = g1 ? t1[e] : (g2 ? sv : t2[e]);
          i2[e] = g1 ? i1[e] : (g2 ? c : i2[e]);
          t1[e] = g1 ? sv : t1[e];
          i1[e] = g1 ? c : i1[e];
        }
      }
    };
    // A class passes the bound test (lo - hi_j) im <= U, then - when y^G is
    // certain - the exact one with its own FP32 bracket of 1 / ||W_y - W_j||
    // (irow: the bracket-table row of y). The brackets are loaded only where
    // the bound test passed, sixteen predicated loads in flight at a time.
    auto pass2_chunk_tight = [&](const uint32_t (&v)[32], int ch, float E, float lo, float im, float U,
                                 const float* __restrict__ irow, bool exact) -> uint32_t {
      const int lim = min(32, C - ch * 32);
      const float* bc = bias_s + ch * 32;
      uint32_t crude = 0;
#pragma unroll
      for (int j = 0; j < 32; ++j) {
        const float hj = __fadd_ru(__fadd_rn(__uint_as_float(v[j]), bc[j]), E);
        crude |= (uint32_t)(__fmul_rd(__fsub_rd(lo, hj), im) <= U) << j;
      }
      crude &= lim == 32 ? 0xffffffffu : (1u << lim) - 1u;
      uint32_t mask = exact ? 0u : crude;
      // a full chunk with 16-byte aligned bracket rows: each half's 16
      // brackets in four 16-byte loads, by the lanes with a class there
      const bool vec4 = lim == 32 && (C & 3) == 0;
#pragma unroll
      for (int h16 = 0; h16 < 2; ++h16) {
        float p[16];
        if (vec4) {
          const uint32_t hb = (crude >> (16 * h16)) & 0xffffu;
          if (exact && hb) {
            const float4* src = reinterpret_cast<const float4*>(irow + ch * 32 + 16 * h16);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              const float4 q = __ldg(src + i);
              p[4 * i] = q.x;
              p[4 * i + 1] = q.y;
              p[4 * i + 2] = q.z;
              p[4 * i + 3] = q.w;
            }
          } else {
#pragma unroll
            for (int k = 0; k < 16; ++k) p[k] = 0.f;
          }
        } else {
#pragma unroll
          for (int k = 0; k < 16; ++k) {
            const int j = 16 * h16 + k;
            p[k] = (exact && ((crude >> j) & 1u)) ? __ldg(irow + ch * 32 + j) : 0.f;
          }
        }
#pragma unroll
        for (int k = 0; k < 16; ++k) {
          const int j = 16 * h16 + k;
          const float hj = __fadd_ru(__fadd_rn(__uint_as_float(v[j]), bc[j]), E);
          mask |= (uint32_t)(exact && ((crude >> j) & 1u) && __fmul_rd(__fsub_rd(lo, hj), p[k]) <= U) << j;
        }
      }
      return mask;
    };

    unsigned long long n_pairs = 0, n_full = 0;  // this warp's refinement counts
    int t = 0;
    for (int tile = blockIdx.x; tile < n_tiles; tile += gridDim.x, ++t) {
      const int buf = t & 1, zb = t % L.nzb;
      if (fixq && ew == 0 && lane == 0) *(volatile int*)&fixq->beat = t + 1;
      bool ok = ptx::mbar_wait(accfull + 8 * buf, (uint32_t)(t >> 1) & 1u, abort_s, kWaitLimit);
      for (int c = 0; c < L.nch && ok; ++c)  // the features are visible to these threads too
        ok = ptx::mbar_wait(zfull_of(zb, c), (uint32_t)(t / L.nzb) & 1u, abort_s, kWaitLimit);
      ok = __all_sync(kFull, ok);  // warp-uniform before the aligned TMEM loads
      ptx::tc_fence_after();
      const uint32_t zs = s_z + (uint32_t)zb * L.zbytes;
      const int64_t grow = (int64_t)tile * kBM + r;
      const bool live = grow < a.n;
      const uint32_t tacc = tmem + lane_base + (uint32_t)buf * kAccStride;
      Pass1 mine{-INFINITY, -INFINITY, 0.f, kNoClass | (kNoClass << 16)};
      if (ok) {
        // two of the four k-ordered partial sums of ||z||^2 (quarters 2 half,
        // 2 half + 1 of the features; the FP32 kernels form the same chains)
        float pc[2];
#pragma unroll
        for (int j = 0; j < 2; ++j) {
          const int q = 2 * half + j;
          float p = 0.f;
          for (int k = q * dq; k < (q + 1) * dq; k += 4) {
            const float4 v = lds_f4(zs + sw_off(r, k, kZChunkBytes));
            p = fmaf(v.x, v.x, p);
            p = fmaf(v.y, v.y, p);
            p = fmaf(v.z, v.z, p);
            p = fmaf(v.w, v.w, p);
          }
          pc[j] = p;
        }
        mine.psum = pc[0] + pc[1];
        // pass 1: top two s~ of this half's columns (two chunks per TMEM wait)
        float t1[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY}, t2[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
        if constexpr (TIGHT) {
          int i1[4] = {kNoClass, kNoClass, kNoClass, kNoClass}, i2[4] = {kNoClass, kNoClass, kNoClass, kNoClass};
          for (int ch = half; ch < nck; ch += 4) {
            uint32_t va[32], vb[32];
            const bool two = ch + 2 < nck;
            ptx::tmem_ld32(tacc + (uint32_t)(ch * 32), va);
            if (two) ptx::tmem_ld32(tacc + (uint32_t)((ch + 2) * 32), vb);
            ptx::tmem_wait_ld();
            pass1_chunk_idx(va, ch, t1, i1, t2, i2);
            if (two) pass1_chunk_idx(vb, ch + 2, t1, i1, t2, i2);
          }
#pragma unroll
          for (int e = 1; e < 4; ++e) top2i_merge(t1[0], i1[0], t2[0], i2[0], t1[e], i1[e], t2[e], i2[e]);
          mine.idx = (i1[0] & 0xffff) | (i2[0] << 16);
        } else {
          for (int ch = half; ch < nck; ch += 4) {
            uint32_t va[32], vb[32];
            const bool two = ch + 2 < nck;
            ptx::tmem_ld32(tacc + (uint32_t)(ch * 32), va);
            if (two) ptx::tmem_ld32(tacc + (uint32_t)((ch + 2) * 32), vb);
            ptx::tmem_wait_ld();
            pass1_chunk(va, ch, t1, t2);
            if (two) pass1_chunk(vb, ch + 2, t1, t2);
          }
#pragma unroll
          for (int e = 1; e < 4; ++e) {
            t2[0] = fmaxf(fmaxf(t2[0], t2[e]), fminf(t1[0], t1[e]));
            t1[0] = fmaxf(t1[0], t1[e]);
          }
        }
        mine.l1 = t1[0];
        mine.l2 = t2[0];
      }
      x1[half * kBM + r] = mine;
      if (lane == 0) okf[half * 4 + quarter] = ok ? 1 : 0;
      pair_barrier(bar_id);
      const Pass1 o = x1[(half ^ 1) * kBM + r];
      if (!ok || okf[(half ^ 1) * 4 + quarter] == 0) break;  // both warps of the pair leave together
      float L1 = fmaxf(mine.l1, o.l1), L2 = fmaxf(fmaxf(mine.l2, o.l2), fminf(mine.l1, o.l1));
      int y = kNoClass, j2 = kNoClass;
      if constexpr (TIGHT) {
        // both warps merge in the same order (half 0's list first), so they
        // agree on the classes
        const Pass1& p0 = half == 0 ? mine : o;
        const Pass1& p1 = half == 0 ? o : mine;
        L1 = p0.l1;
        L2 = p0.l2;
        y = p0.idx & 0xffff;
        j2 = p0.idx >> 16;
        top2i_merge(L1, y, L2, j2, p1.l1, p1.idx & 0xffff, p1.l2, p1.idx >> 16);
      }
      const float kn = __fadd_rn(mine.psum, o.psum);  // (q0 + q1) + (q2 + q3)
      const float hn = norm_upper(kn);
      // |s~_c| <= Mb, so every screen value and partial sum is finite when
      // Mb is; E covers the MMA error and the rounding of the bias addition
      const float Mb = __fmaf_ru(cw1, hn, bmax);
      const float E = __fmaf_ru(cw, hn, __fmaf_ru(Mb, 2.3841858e-07f /* 2^-22 */, kTinyF));
      const float T = __fsub_rd(L2, __fmul_ru(2.f, E));
      bool fb = live && !(Mb < 1e38f);  // NaN / infinite features, or a bound near FP32 overflow
      // tight radius. If y1 (the screen's top class) is certainly y^G (the
      // runner-up's upper end below lo_1), U1 = u_{y2}(y1) bounds r*/kappa
      // from above and (lo_1 - hi_j) ipn_min(y1) <= l_j bounds every class's
      // bracket from below, so the minimiser of Eq. 29 passes (lo_1 - hi_j)
      // ipn_min(y1) <= U1 (then also with its own bracket l_j). Otherwise every
      // possible y^G has s_{y^G} >= s_y1 >= lo_1 and r*/kappa below U* (below),
      // so one test with lo_1, U* and the head's smallest ipn keeps the
      // minimiser for whichever class is y^G; y^G is then the largest refined
      // candidate.
      float lo1 = 0.f, U1 = 0.f, im1 = 0.f;
      bool unc = false;
      if constexpr (TIGHT) {
        lo1 = __fsub_rd(L1, E);
        const float hi1 = __fadd_ru(L1, E), lo2 = __fsub_rd(L2, E), hi2 = __fadd_ru(L2, E);
        const bool settled = live && !fb && y < C && j2 < C;
        if (settled) {
          unc = !(hi2 < lo1);
          if (!unc) {
            U1 = __fmul_ru(__fsub_ru(hi1, lo2), __ldg(a.ipn_up32 + (size_t)y * C + j2));
            im1 = __ldg(a.ipn_min32 + y);
          } else {
            // r* <= u_{y2}(y1) if y1 is y^G; for any other possible y^G (its
            // s~ <= l2) r* <= (hi_2 - lo_1) / ||W_y - W_y1|| <= (hi_2 - lo_1)
            // ipn_max(y1), the pair norms being symmetric. When hi_2 = lo_1 and
            // some W_g = W_y1 that term is 0 x inf = NaN, which fmaxf drops:
            // such a g is y^G only by tying y1, and its term against y2 has
            // the pair norm ||W_y1 - W_y2||, so the first term bounds it.
            U1 = fmaxf(__fmul_ru(__fsub_ru(hi1, lo2), __ldg(a.ipn_up32 + (size_t)y * C + j2)),
                       __fmul_ru(__fsub_ru(hi2, lo1), __ldg(a.ipn_max32 + y)));
            // lo_1 itself bounds s_{y^G} from below (s_{y^G} >= s_y1 >= lo_1)
            im1 = imA;
          }
        }
        fb = live && !settled;  // the whole row goes to the one-warp path (both halves agree)
      }
      // row of the lower-bracket table for y1 (a valid address also when unused)
      const float* irow1 = a.ipn_dn32 ? a.ipn_dn32 + (size_t)(y < C ? y : 0) * C : nullptr;

      // pass 2: the candidates of this half's columns into the warp's list;
      // the row's lane keeps its slots' classes (one byte each)
      int P = 0, cnt = 0;
      uint32_t cls_lo = 0, cls_hi = 0;
      auto append = [&](uint32_t mask, int ch) {
        if (!live || fb) mask = 0;
        while (__any_sync(kFull, mask != 0)) {
          const bool has = mask != 0;
          const int jb = __ffs((int)mask) - 1;
          mask &= mask - 1;
          const bool take = has && cnt < kMaxCandTc;
          const unsigned mb = __ballot_sync(kFull, take);
          if (take) {
            const int c = ch * 32 + jb;
            list[P + __popc(mb & ((1u << lane) - 1u))] = lane | (cnt << 5) | (c << 8);
            if (cnt < 4)
              cls_lo |= (uint32_t)c << (8 * cnt);
            else
              cls_hi |= (uint32_t)c << (8 * (cnt - 4));
          }
          cnt += has ? 1 : 0;
          P += __popc(mb);
        }
      };
      for (int ch = half; ch < nck; ch += 4) {
        uint32_t va[32], vb[32];
        const bool two = ch + 2 < nck;
        ptx::tmem_ld32(tacc + (uint32_t)(ch * 32), va);
        if (two) ptx::tmem_ld32(tacc + (uint32_t)((ch + 2) * 32), vb);
        ptx::tmem_wait_ld();
        uint32_t ma, mbk = 0u;
        if constexpr (TIGHT) {
          ma = pass2_chunk_tight(va, ch, E, lo1, im1, U1, irow1, !unc);
          if (two) mbk = pass2_chunk_tight(vb, ch + 2, E, lo1, im1, U1, irow1, !unc);
        } else {
          ma = pass2_chunk(va, ch, T);
          if (two) mbk = pass2_chunk(vb, ch + 2, T);
        }
        append(ma, ch);
        if (two) append(mbk, ch + 2);
      }
      const bool ovf = cnt > kMaxCandTc;  // (tight: the row goes to the one-warp path, below)
      if constexpr (!TIGHT) fb = fb || ovf;
      ptx::tc_fence_before();
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(accempty + 8 * buf);  // the accumulator is free for tile t + 2

      // refinement: each lane takes one pair of the list at a time
      // (refine_lane, the bits of refine2) and stores hi / lo at the pair's
      // (row lane, slot) = e & 0xff: lane + 32 slot. A last round of at most
      // 16 (8) pairs shares each pair between two (four) lanes
      // (refine_lanes), so that it takes about half (a quarter) of a whole
      // round.
      const int rq = quarter * 32;  // first row of the warp
      const int pfull = (P & 31) > 16 ? P : P & ~31;
      for (int i = lane; i < pfull; i += 32) {
        const int e = list[i];
        const int c = e >> 8;
        float hi, lo;
        refine_lane(s_w, wchunk, zs, c, rq + (e & 31), bias_s[c], d, hi, lo);
        res_hi[e & 0xff] = hi;
        res_lo[e & 0xff] = lo;
      }
      if (pfull < P) {  // (warp-uniform)
        const int kk = P - pfull > 8 ? 2 : 4;
        const int i = pfull + lane / kk;
        const int e = list[i < P ? i : pfull];
        const int c = e >> 8;
        float hi, lo;
        if (kk == 2)
          refine_lanes<2>(s_w, wchunk, zs, c, rq + (e & 31), bias_s[c], d, lane & 1, hi, lo);
        else
          refine_lanes<4>(s_w, wchunk, zs, c, rq + (e & 31), bias_s[c], d, lane & 3, hi, lo);
        if (i < P && lane % kk == 0) {
          res_hi[e & 0xff] = hi;
          res_lo[e & 0xff] = lo;
        }
      }
      __syncwarp();  // every refined pair is visible to its row's lane
      if constexpr (!TIGHT) {
        __syncwarp();
        // each row's lane pushes its own candidates into its running selection
        Top2 tp;
        if (!fb) {
          const int ns = cnt < kMaxCandTc ? cnt : kMaxCandTc;
          for (int sl = 0; sl < ns; ++sl) {
            const int c = (int)(((sl < 4 ? cls_lo >> (8 * sl) : cls_hi >> (8 * (sl - 4)))) & 0xffu);
            tp.push(c, res_hi[lane + 32 * sl], res_lo[lane + 32 * sl], refined_err(a.g2f8, wn_s[c], hn, bias_s[c]));
          }
        }
        // rows that need every class of this half refined, one row at a time,
        // eight classes a round through the row's result cells
        const unsigned fbm = __ballot_sync(kFull, fb);
        if (lane == 0) {
          n_full += (unsigned long long)__popc(fbm);
          n_pairs += (unsigned long long)P + (unsigned long long)__popc(fbm) * (unsigned long long)ncls;
        }
        for (unsigned fr = fbm; fr != 0; fr &= fr - 1) {
          const int ow = __ffs((int)fr) - 1;
          if (lane == ow) tp = Top2();
          for (int t2 = 0; t2 < ncls; t2 += 2 * (32 / kGroupTc)) {
            int tq[2] = {t2 + 2 * g8, t2 + 2 * g8 + 1};
            int cp[2];
#pragma unroll
            for (int u = 0; u < 2; ++u) {
              const int tt = tq[u] < ncls ? tq[u] : t2;
              cp[u] = (2 * (tt >> 5) + half) * 32 + (tt & 31);
            }
            const int rp[2] = {rq + ow, rq + ow};
            const float bp[2] = {bias_s[cp[0]], bias_s[cp[1]]};
            float hi[2], lo[2];
            refine2(s_w, wchunk, zs, cp, rp, bp, d, sub, hi, lo);
            if (sub == 0) {
#pragma unroll
              for (int u = 0; u < 2; ++u) {
                res_hi[ow + 32 * (2 * g8 + u)] = hi[u];
                res_lo[ow + 32 * (2 * g8 + u)] = lo[u];
              }
            }
            __syncwarp();
            if (lane == ow)
              for (int u = 0; u < 2 * (32 / kGroupTc) && t2 + u < ncls; ++u) {
                const int tt = t2 + u;
                const int c = (2 * (tt >> 5) + half) * 32 + (tt & 31);
                tp.push(c, res_hi[ow + 32 * u], res_lo[ow + 32 * u], refined_err(a.g2f8, wn_s[c], hn, bias_s[c]));
              }
            __syncwarp();
          }
        }
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(zempty + 8 * zb);  // this warp is done with the tile's features

        // merge the halves; FP64 finals and the row's rank in its 32-row block
        if (half == 1) x2[r] = tp;
        pair_barrier(bar_id);
        if (half == 0) {
          top2_merge(tp, x2[r]);
          if (live) {
            if (row_finals(a, grow, tp.result(kn), &acc_s[r]) && fixq) fixq_push(fixq, (int)grow, kn, abort_s, kWaitLimit);
          } else {
            acc_s[r] = 0;
          }
          const unsigned mb = __ballot_sync(kFull, live && acc_s[r] != 0);
          if (live) a.rank[grow] = __popc(mb & ((1u << lane) - 1u));
          const int64_t blk0 = (int64_t)tile * kBM + quarter * 32;
          if (lane == 0 && blk0 < a.n) a.bcount[blk0 / 32] = __popc(mb);
        }
      } else {
        // tight radius (Eq. 29): y^G is the largest refined candidate (each
        // half's best, merged in the same order by both); each half's minima
        // over its own candidates; half 0 combines them and takes the rows the
        // screen could not settle
        TightX& tx = *reinterpret_cast<TightX*>(smem + L.off_x2);
        const int ns = cnt < kMaxCandTc ? cnt : kMaxCandTc;
        auto slot_class = [&](int sl) {
          return (int)((sl < 4 ? cls_lo >> (8 * sl) : cls_hi >> (8 * (sl - 4))) & 0xffu);
        };
        float bh = -INFINITY, bl = 0.f;
        int bc = -1;
        if (live && !fb && !ovf)
          for (int sl = 0; sl < ns; ++sl) {
            const int c = slot_class(sl);
            const float h = res_hi[lane + 32 * sl], l = res_lo[lane + 32 * sl];
            if (bc < 0 || pair_gt(h, l, bh, bl) || (h == bh && l == bl && c < bc)) {
              bh = h;
              bl = l;
              bc = c;
            }
          }
        tx.bv[half][r] = make_float2(bh, bl);
        tx.bc[half][r] = (int16_t)bc;
        tx.ovf[half][r] = ovf ? 1 : 0;
        pair_barrier(bar_id);
        const bool rowfb = fb || (live && (tx.ovf[0][r] != 0 || tx.ovf[1][r] != 0));
        double rmin = INFINITY, smin = INFINITY;
        bool any_nan = false;
        int yg = y;
        if (live && !rowfb) {
          float2 v2 = tx.bv[0][r];
          yg = tx.bc[0][r];
          const float2 w2 = tx.bv[1][r];
          const int c1 = tx.bc[1][r];
          if (c1 >= 0 && (yg < 0 || pair_gt(w2.x, w2.y, v2.x, v2.y) || (w2.x == v2.x && w2.y == v2.y && c1 < yg))) {
            v2 = w2;
            yg = c1;
          }
          any_nan = yg < 0;  // no candidate (cannot happen: y1 always passes)
          if (any_nan) yg = y;
          const double vy = (double)v2.x + (double)v2.y;
          const double ey = (double)refined_err(a.g2f8, wn_s[yg], hn, bias_s[yg]);
          any_nan = any_nan || !(vy == vy);
          // unrolled over the slots so that the pair-table loads of all
          // candidates are in flight together
#pragma unroll
          for (int sl = 0; sl < kMaxCandTc; ++sl) {
            const int j = slot_class(sl);
            if (sl < ns && j != yg) {
              const double vj = (double)res_hi[lane + 32 * sl] + (double)res_lo[lane + 32 * sl];
              any_nan |= !(vj == vj);
              tight_term(a, yg, j, vy, ey, vj, (double)refined_err(a.g2f8, wn_s[j], hn, bias_s[j]), rmin, smin);
            }
          }
        }
        const unsigned fbm = __ballot_sync(kFull, rowfb);
        if (lane == 0) {
          n_pairs += (unsigned long long)P;
          if (half == 0) {
            n_full += (unsigned long long)__popc(fbm);
            n_pairs += (unsigned long long)__popc(fbm) * (unsigned long long)C;
          }
        }
        if (half == 1) {
          tx.rmin[r] = rmin;
          tx.smin[r] = smin;
          tx.nan[r] = any_nan ? 1 : 0;
        }
        pair_barrier(bar_id);
        if (half == 0) {
          if (!rowfb) acc_s[r] = 0;
          if (live && !rowfb &&
              tight_write(a, grow, yg, fmin(rmin, tx.rmin[r]), fmin(smin, tx.smin[r]), any_nan || tx.nan[r] != 0, kn,
                          &acc_s[r]) &&
              fixq)
            fixq_push(fixq, (int)grow, kn, abort_s, kWaitLimit);
        }
        // the rows the screen could not settle, alternately on the two warps
        int k = 0;
        for (unsigned fr = fbm; fr != 0; fr &= fr - 1, ++k) {
          const int ow = __ffs((int)fr) - 1;
          if ((k & 1) == half) {
            const float knw = __shfl_sync(kFull, kn, ow);
            const int64_t frow = (int64_t)tile * kBM + rq + ow;
            if (tc_tight_row_warp(a, frow, rq + ow, s_w, wchunk, zs, wn_s, bias_s, knw, lane, res_hi, res_lo,
                                  &acc_s[rq + ow]) &&
                fixq && lane == 0)
              fixq_push(fixq, (int)frow, knw, abort_s, kWaitLimit);
            __syncwarp();
          }
        }
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(zempty + 8 * zb);  // this warp is done with the tile's features
        pair_barrier(bar_id);  // every acceptance flag of the 32 rows is written
        if (half == 0) {
          const unsigned mb = __ballot_sync(kFull, live && acc_s[r] != 0);
          if (live) a.rank[grow] = __popc(mb & ((1u << lane) - 1u));
          const int64_t blk0 = (int64_t)tile * kBM + quarter * 32;
          if (lane == 0 && blk0 < a.n) a.bcount[blk0 / 32] = __popc(mb);
        }
      }
    }
    if (lane == 0 && (n_pairs | n_full)) {
      atomicAdd(&stats->ins_pairs, n_pairs);
      atomicAdd(&stats->ins_full_rows, n_full);
    }
    // every row this warp lists is in the queue: the fix warp may finish
    __syncwarp();
    if (fixq && lane == 0) {
      __threadfence_block();
      atomicAdd(&fixq->done, 1);
    }
  }
  ptx::tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0 && *abort_s) {
    atomicAdd(&stats->errors, 1ull);
    atomicExch(&stats->abort_flag, 1);
  }
  if (warp == 1) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, kTmemCols);
  }
}

void encode_rows(lipcache* h, CUtensorMap* map, const float* base, uint64_t rows, uint32_t box_rows) {
  LC_REQUIRE(h->encode != nullptr, LIPCACHE_E_CUDA, "cuTensorMapEncodeTiled is unavailable from the driver");
  const cuuint64_t dims[2] = {(cuuint64_t)h->d, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)h->d * sizeof(float)};
  const cuuint32_t box[2] = {(cuuint32_t)kChunkF, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  const CUresult r = h->encode(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float*>(base), dims, strides, box,
                               estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  LC_REQUIRE(r == CUDA_SUCCESS, LIPCACHE_E_CUDA, "cuTensorMapEncodeTiled failed: " + std::to_string((int)r));
}

// Two feature buffers when they fit next to the resident head, else one.
// The FP64 pass in the kernel when its queue and scratch fit as well (and
// `fix_in_kernel` allows it).
bool tc_plan(int d, int C, TcLayout& L, bool fix_in_kernel = true) {
  for (int nzb = 2; nzb >= 1; --nzb)
    for (int infix = fix_in_kernel ? 1 : 0; infix >= 0; --infix) {
      L = tc_layout(d, C, nzb, infix);
      if (L.total <= (uint32_t)kSmemBudget) return true;
    }
  return false;
}

}  // namespace

bool certify_tc_supported(const lipcache* h, const float* H, int64_t n) {
  if (h->encode == nullptr) return false;
  // the tight radius needs the bracket tables of the head's pair norms
  if (h->radius_mode == LIPCACHE_RADIUS_TIGHT &&
      (h->ipn_up32 == nullptr || h->ipn_min32 == nullptr || h->ipn_max32 == nullptr))
    return false;
  if (h->debug_flags & (LIPCACHE_DEBUG_INSERT_TILE64 | LIPCACHE_DEBUG_INSERT_WIDE_TILE)) return false;
  // TMA: 16-byte aligned rows of d floats, 32-feature boxes (at most
  // kMaxChunks of them); MMA: N <= 256
  if (h->d < kChunkF || h->d > kChunkF * kMaxChunks || h->d % 16 != 0 || ((uintptr_t)H & 15) != 0) return false;
  if (h->C < 2 || h->C > 256 || n <= 0 || n > ((int64_t)1 << 30)) return false;
  TcLayout L;
  return tc_plan(h->d, h->C, L);
}

bool certify_tc_launch(lipcache* h, const CertArgs& a, cudaStream_t s) {
  TcLayout L;
  LC_REQUIRE(tc_plan(h->d, h->C, L, !(h->debug_flags & LIPCACHE_DEBUG_INSERT_FIX_STANDALONE)), LIPCACHE_E_INVALID,
             "head does not fit the tensor certify kernel");
  CUtensorMap tmH, tmW;
  encode_rows(h, &tmH, a.H, (uint64_t)a.n, kBM);
  encode_rows(h, &tmW, h->W, (uint64_t)h->C, (uint32_t)L.Cpad);
  const int n_tiles = (int)((a.n + kBM - 1) / kBM);
  const int grid = n_tiles < h->num_sms ? n_tiles : h->num_sms;
  // at least half of the SM's shared memory, so one CTA (and one 512-column
  // TMEM allocation) per SM
  const int smem = (int)L.total + 1024 > 120 * 1024 ? (int)L.total + 1024 : 120 * 1024;
  auto kern = a.tight ? k_certify_tc<true> : k_certify_tc<false>;
  LC_CUDA(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
  kern<<<grid, kThreads, smem, s>>>(tmH, tmW, a, L, n_tiles, h->stats,
                                    (h->debug_flags & LIPCACHE_DEBUG_STALL_INSERT) ? 1 : 0);
  LC_LAUNCH_CHECK("k_certify_tc");
  return L.infix != 0;
}

}  // namespace lc
