/*
 * lipcache.h — C ABI of the GB300-native certified cache lookup.
 *
 * The library implements the data-parallel hot path of LipCache
 * (arxiv 2608.13144): certified insertion of GuardNet features into a
 * feature cache (Sec. 3.3, Algorithm 1; Eqs. 17-21, 29) and batched online
 * lookup with MainNet fallback (Sec. 3.4, Algorithm 2; Eqs. 13-15).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - Every function returns a lipcache_status. On failure nothing the caller
 *    owns has been written unless stated, and lipcache_last_error() returns
 *    a thread-local, human-readable message. No C++ exception crosses the ABI.
 *  - Pointers are DEVICE pointers (CUDA global memory of the device the cache
 *    was created on) unless marked "host". The caller owns every input and
 *    output buffer; the library owns the cache table, its copies of W and b,
 *    sigma_max(W) and all scratch memory.
 *  - Work is enqueued on the caller's stream (a cudaStream_t; NULL = legacy
 *    default stream). Functions that return a host scalar synchronise that
 *    stream before returning; lipcache_probe does not and returns as soon as
 *    its kernels are enqueued.
 *  - Feature vectors are FP32, row-major, d contiguous floats per row, any
 *    4-byte alignment. Indices are int64 in cache insertion order.
 *  - A cache handle is not thread-safe: calls on one handle must be
 *    serialised by the caller. Distinct handles are independent.
 *  - Inputs are not validated element by element: a NaN logit margin fails
 *    r > 0 (the row is rejected); a NaN query fails the strict hit test
 *    (it misses and falls back to MainNet).
 */
#ifndef LIPCACHE_H
#define LIPCACHE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Opaque cache handle. */
typedef struct lipcache lipcache_t;

/* Binary-compatible with cudaStream_t / CUstream. */
typedef struct CUstream_st* lipcache_stream_t;

typedef enum lipcache_status {
  LIPCACHE_OK = 0,
  LIPCACHE_E_INVALID = 1,         /* bad argument (size, pointer, mode) */
  LIPCACHE_E_STATE = 2,           /* call not allowed now (e.g. probe before set_head) */
  LIPCACHE_E_DEGENERATE_HEAD = 3, /* sigma_max(W) <= 0: Algorithm 1 stops construction */
  LIPCACHE_E_FULL = 4,            /* insert would exceed the capacity; nothing inserted */
  LIPCACHE_E_NOT_CONVERGED = 5,   /* spectral power iteration hit its iteration limit */
  LIPCACHE_E_CUDA = 6,            /* a CUDA runtime call failed (message has the detail) */
  LIPCACHE_E_NOMEM = 7,           /* device or host allocation failed */
  LIPCACHE_E_DEVICE = 8           /* a kernel reported an error (a bounded wait expired) */
} lipcache_status;

/* Radius modes rho (policy tuple, Sec. 3.4). */
#define LIPCACHE_RADIUS_CONSERVATIVE 0 /* r  = m / (sigma_max(W) sqrt 2), Eq. 21 */
#define LIPCACHE_RADIUS_TIGHT 1        /* r* = min_j (s_y - s_j) / ||W_y - W_j||, Eq. 29 */

/* Certify kernels (lipcache_info.last_insert_kernel).
 * TENSOR: TF32 tcgen05 screen of the logits into tensor memory, both radii
 *   (d % 16 == 0, 32 <= d <= 256, 2 <= C <= 256, head resident in shared
 *   memory); it refines and finishes rows as WIDE_TILE does (conservative
 *   radius: the same bits; tight radius: within the refinement bound).
 * WIDE_TILE: head resident in shared memory, 128-row tiles, logits in
 *   registers (d % 4 == 0, head small enough; both radii, the tight one
 *   refining only the classes that can be its minimiser).
 * TILE64: head resident, 64-row tiles, logits in shared memory.
 * STREAMED: head read from L2 (large heads).
 * For the conservative radius TENSOR, WIDE_TILE and TILE64 give the same bits;
 * STREAMED refines with a 32-lane compensated sum, so its radii agree with
 * theirs within the refinement bound. For the tight radius TILE64 and
 * STREAMED refine every class in FP64, and all kernels agree within the
 * refinement bound. */
#define LIPCACHE_INSERT_WIDE_TILE 1
#define LIPCACHE_INSERT_TILE64 2
#define LIPCACHE_INSERT_STREAMED 3
#define LIPCACHE_INSERT_TENSOR 4

/* Radius policies of the probe (lipcache_set_radius_policy). */
#define LIPCACHE_POLICY_CERTIFIED 0  /* per-entry certified radius (Eq. 21 or Eq. 29) */
#define LIPCACHE_POLICY_GLOBAL 1     /* one global nearest-neighbour threshold (Sec. 5.4) */
#define LIPCACHE_POLICY_INTERCLASS 2 /* radius from inter-class centroid distances (Sec. 5.4) */

/* Probe kernels. All return identical results; they differ in speed. */
#define LIPCACHE_PROBE_AUTO 0          /* tensor path when supported (d <= 256) and B N d_pad >= 2^24, else exact */
#define LIPCACHE_PROBE_TENSOR 1        /* tcgen05 TF32 screen, then exact FP32 recheck of candidates;
                                          the kernel is chosen by shape: TENSOR_SINGLE for
                                          d_pad <= 128, TENSOR_PAIR above (when clusters of four fit) */
#define LIPCACHE_PROBE_EXACT 2         /* exact FP32 distance of every pair on CUDA cores */
#define LIPCACHE_PROBE_TENSOR_SINGLE 3 /* the tensor screen with single-CTA MMAs (clusters of two) */
#define LIPCACHE_PROBE_TENSOR_PAIR 4   /* the tensor screen with CTA-pair MMAs (clusters of four) */

/* Limits checked by lipcache_create. */
#define LIPCACHE_MAX_DIM 1024
#define LIPCACHE_MAX_CLASSES 1024
#define LIPCACHE_MAX_CAPACITY 2147483647LL /* indices are packed in 31 bits */

typedef struct lipcache_info {
  int32_t d;                /* feature dimension */
  int32_t C;                /* classes */
  int32_t d_pad;            /* row stride of the key table: d rounded up to 32 */
  int32_t radius_mode;      /* LIPCACHE_RADIUS_* */
  int64_t capacity;         /* maximum number of cache entries */
  int64_t size;             /* current number of cache entries */
  int32_t head_set;         /* 1 after a successful lipcache_set_head */
  int32_t sigma_iterations; /* power iterations used by the last set_head */
  double sigma;             /* sigma_max(W) of the current head (0 before set_head) */
  double sigma_residual;    /* ||W^T W v - theta v|| / theta at exit */
  double radius_scale;      /* kappa in (0, 1]: radius tightening factor (Sec. 5.6) */
  double eps_recheck;       /* relative deflation of r^2 covering the FP32 recheck error */
  double c_screen;          /* relative slack of the tensor-core screen */
  int64_t candidates;       /* screen candidates rechecked since the last reset */
  int64_t device_errors;    /* kernel-reported errors since the last reset */
  int32_t probe_path;       /* LIPCACHE_PROBE_* configured for lipcache_probe */
  int32_t last_probe_path;  /* kernel that served the last probe: _EXACT, _TENSOR_SINGLE or _TENSOR_PAIR */
  float last_probe_ms;      /* main-kernel time of the last probe (timing enabled) */
  int32_t num_sms;          /* SMs of the device */
  double kernel_ms_total;   /* summed main-kernel time of timed probes since the last reset */
  int64_t kernel_launches;  /* number of timed probes in kernel_ms_total */
  int32_t last_grid;        /* CTAs launched by the last probe's main kernel */
  int32_t last_cluster;     /* CTAs per cluster of that launch (1 = no cluster) */
  int32_t radius_policy;    /* LIPCACHE_POLICY_* the probe uses */
  int32_t last_insert_kernel; /* kernel that certified the last insert: LIPCACHE_INSERT_* (0 before any) */
  double policy_param;      /* tau (GLOBAL) or beta (INTERCLASS); 0 for CERTIFIED */
  double insert_kernel_ms_total; /* summed certify-kernel time of timed inserts since the last reset */
  int64_t insert_kernel_launches; /* number of timed certify kernels in insert_kernel_ms_total */
  int64_t insert_refined_pairs; /* (row, class) pairs the tensor certify kernel refined (compensated dot
                                   product) since the last reset */
  int64_t insert_full_rows;     /* row halves it refined over every class of the half (more candidates
                                   than slots, a NaN logit or an unbounded screen error) */
  int64_t insert_fp64_rows;     /* rows re-certified in FP64 since the last reset: rows whose margin (or
                                   minimising term of Eq. 29) the compensated FP32 refinement could not
                                   pin to 5e-6 relative */
} lipcache_info;

/*
 * Create an empty cache for d-dimensional GuardNet features and a C-class
 * head (Sec. 3.1 notation: z in R^d, W in R^{C x d}). Allocates the key table
 * for `capacity` entries on the current CUDA device.
 *   d           1 .. LIPCACHE_MAX_DIM
 *   C           2 .. LIPCACHE_MAX_CLASSES
 *   capacity    1 .. LIPCACHE_MAX_CAPACITY
 *   radius_mode LIPCACHE_RADIUS_CONSERVATIVE or LIPCACHE_RADIUS_TIGHT
 *   out         host; receives the handle (NULL on failure)
 * Errors: E_INVALID, E_NOMEM, E_CUDA (e.g. no device).
 */
lipcache_status lipcache_create(int32_t d, int32_t C, int64_t capacity, int32_t radius_mode, lipcache_t** out);

/*
 * Install the GuardNet affine head f(z) = W z + b (Eq. 5) and compute its
 * Lipschitz constant sigma_max(W) (Eqs. 17-19; Algorithm 1, first step) by
 * power iteration on W^T W in FP64, accelerated by repeated squaring, until
 * successive Rayleigh quotients agree to 1e-13 and the eigen-residual is
 * below 1e-10 theta.
 *   W         C x d row-major FP32 (device); copied, the caller may free it after return
 *   b         C FP32 (device); copied
 *   sigma_out host, nullable; receives sigma_max(W)
 * Synchronises `stream`. Allowed only while the cache is empty (radii depend
 * on W). Errors: E_STATE (cache not empty), E_DEGENERATE_HEAD (sigma <= 0;
 * Algorithm 1 stops construction), E_NOT_CONVERGED, E_INVALID (NULL W or b),
 * E_CUDA.
 */
lipcache_status lipcache_set_head(lipcache_t* h, const float* W, const float* b, double* sigma_out,
                                  lipcache_stream_t stream);

/*
 * Certify n candidate rows and append the accepted ones (Algorithm 1 with
 * every accepted candidate selected). For each row z: logits s = W z + b,
 * y^G = argmax s (lowest class on ties), margin m = s_y - max_{j!=y} s_j
 * (Eq. 20), radius r = kappa * m / (sigma sqrt 2) (Eq. 21) or the tight r*
 * (Eq. 29); payload = payload[i] if given else y^G (proxy label). A row is
 * skipped if require_consistency != 0 and payload != y^G, else if r <= 0.
 * Accepted rows get consecutive indices in input order.
 *   H           n x d FP32 (device)
 *   n           >= 0; n == 0 is a no-op
 *   payload     n int32 (device), nullable -> proxy labels y^G
 *   out_index   n int64 (device), nullable; cache index or -1 if skipped
 *   out_radius  n FP32 (device), nullable; r of every row rounded toward zero
 *               (also for skipped rows)
 *   n_accepted  host, nullable; number of rows appended
 * With n_accepted given (or a radius policy other than CERTIFIED), synchronises
 * `stream`. With n_accepted NULL the call is asynchronous on `stream`: the
 * table's size is kept on the device (each insert takes its first index from
 * it), out_index / out_radius are valid once the stream reaches them, and the
 * host learns the size from the next call that needs it (lipcache_size,
 * get_info, probe, ... synchronise that stream first; an insert on another
 * stream does too). A device error of an asynchronous insert leaves its rows
 * out (out_index -1) and shows in lipcache_info.device_errors.
 * All or nothing: if size + n > capacity nothing is written and E_FULL is
 * returned (checked against size plus the rows of unsettled asynchronous
 * inserts, settling them when that bound exceeds the capacity).
 * Errors: E_STATE (no head), E_FULL, E_INVALID, E_CUDA, E_DEVICE.
 */
lipcache_status lipcache_insert(lipcache_t* h, const float* H, int64_t n, const int32_t* payload,
                                int32_t require_consistency, int64_t* out_index, float* out_radius,
                                int64_t* n_accepted, lipcache_stream_t stream);

/*
 * Batched certified lookup (Algorithm 2, Eqs. 13-15): for every query q the
 * hit set H(q) = { i : ||q - z_i|| < r_i } (strict) and the nearest hit
 * i* = argmin_{i in H(q)} ||q - z_i||, ties to the lowest index. A miss
 * means "fall back to MainNet".
 * The GPU accepts an entry only if its FP32 distance is below r_i deflated by
 * a proven error bound, so it never accepts a pair whose exact distance is
 * not below r_i; pairs within ~2e-6 relative of the boundary may be missed.
 *   Q          B x d FP32 (device)
 *   B          >= 0; B == 0 is a no-op
 *   out_index  B int64 (device): i*, or -1 on a miss
 *   out_label  B int32 (device), nullable: payload of i*, or -1
 *   out_dist   B FP32 (device), nullable: ||q - z_i*|| (FP32), or +inf
 * Asynchronous on `stream`. Errors: E_STATE (no head), E_INVALID, E_NOMEM
 * (scratch growth), E_CUDA. A device-side failure (bounded wait expired)
 * turns the affected queries into misses and is counted in
 * lipcache_info.device_errors.
 */
lipcache_status lipcache_probe(lipcache_t* h, const float* Q, int64_t B, int64_t* out_index, int32_t* out_label,
                               float* out_dist, lipcache_stream_t stream);

/* Selection strategies S (Algorithm 1, last steps; lipcache_insert_select). */
#define LIPCACHE_SELECT_ALL 0          /* every certified candidate, in input order (= lipcache_insert) */
#define LIPCACHE_SELECT_RADIUS_DEDUP 1 /* radius-prioritised de-duplication (Sec. 5.5) */
#define LIPCACHE_SELECT_KCENTER 2      /* K-center per class (Sec. 5.5) */

/*
 * Algorithm 1 with a selection strategy S: certify the n candidate rows as
 * lipcache_insert does, then append the ones S selects.
 *   LIPCACHE_SELECT_RADIUS_DEDUP (the default strategy of Sec. 5.5; the paper
 *   names it without a formula): the certified candidates are visited in
 *   order of decreasing radius (the FP32 radius, ties to the lower row); a
 *   candidate is skipped if lipcache_probe would already hit it -- it lies
 *   strictly inside the ball of an entry of the cache, present before the
 *   call or kept earlier in it -- or if its class (payload label in [0, C))
 *   has budget_per_class entries kept by this call, or the call has kept
 *   budget_total. Kept rows are appended in visiting order. The coverage test
 *   is the probe's conservative one, so a skipped row is always exactly
 *   covered; a row within ~2e-6 relative of a ball's boundary may be kept
 *   where exact arithmetic would skip it.
 *   LIPCACHE_SELECT_KCENTER (the alternative Sec. 5.5 names): per class
 *   (payload label in [0, C); other labels are not selected), Gonzalez's
 *   farthest-point greedy over the class's certified candidates: first the
 *   largest radius, then repeatedly the candidate farthest from the centres
 *   so far (canonical FP32 squared distance; ties to the lower row), up to
 *   budget_per_class (required > 0; budget_total must be 0). Appended class
 *   by class in selection order. Cost: centres x class size x d per class.
 *   LIPCACHE_SELECT_ALL: lipcache_insert (budgets must be 0).
 *   budget_total, budget_per_class   <= 0: unlimited
 *   out_index    n int64 (device), nullable: cache index of a kept row, else -1
 *   out_radius   n FP32 (device), nullable: as for lipcache_insert
 *   n_selected   host, nullable: rows appended
 * Requires the certified radius policy (the coverage test uses the certified
 * balls). Synchronises `stream` (once per 4,096 candidates). All or nothing
 * on capacity: E_FULL, before any work, if size + min(n, budget_total)
 * exceeds it (K-center: min(n, C x budget_per_class)). Errors: those of
 * lipcache_insert and lipcache_probe; E_STATE under an empirical radius
 * policy; E_INVALID for an unknown strategy or budgets it does not take.
 */
lipcache_status lipcache_insert_select(lipcache_t* h, const float* H, int64_t n, const int32_t* payload,
                                       int32_t require_consistency, int32_t strategy, int64_t budget_total,
                                       int32_t budget_per_class, int64_t* out_index, float* out_radius,
                                       int64_t* n_selected, lipcache_stream_t stream);

/*
 * Lookup with write-back (Algorithm 2 with its write-back flag set): probe
 * the batch as lipcache_probe does, then certify every missed query as
 * lipcache_insert does and append the accepted ones, in query order, all on
 * `stream` with no host round trip in between. The whole batch is probed
 * against the cache as it stood when the call began (Algorithm 2 forms the
 * distances D_{k,i} once, before its per-query loop), so a query never hits
 * an entry written back by the same batch. Hits are never inserted.
 *   Q, B, out_label, out_dist   as for lipcache_probe
 *   out_index     B int64 (device), required: i*, or -1 on a miss
 *   payload       B int32 (device), nullable -> proxy labels y^G (the label
 *                 Algorithm 2 derives from the GuardNet logits)
 *   require_consistency  as for lipcache_insert
 *   out_inserted  B int64 (device), nullable: new cache index of a written-
 *                 back query, else -1 (hit, or skipped by Algorithm 1's rules)
 *   n_inserted    host, nullable: number of entries appended
 * Synchronises `stream`. All or nothing: if size + B > capacity nothing is
 * probed or written and E_FULL is returned (the number of misses is not known
 * in advance). Errors: those of lipcache_probe and lipcache_insert;
 * E_DEVICE if a bounded wait of the probe kernel expired (the probe outputs
 * then report misses and nothing is written back).
 */
lipcache_status lipcache_probe_writeback(lipcache_t* h, const float* Q, int64_t B, const int32_t* payload,
                                         int32_t require_consistency, int64_t* out_index, int32_t* out_label,
                                         float* out_dist, int64_t* out_inserted, int64_t* n_inserted,
                                         lipcache_stream_t stream);

/*
 * Certified-consistency check (the rate reported with every experiment of
 * Sec. 5; by the Lemma of Sec. 4.2 it is 1 for certified radii): for every
 * query k with hit_index[k] >= 0, whether the head's argmax on q_k (Eq. 5,
 * lowest class on ties) equals y^G of entry hit_index[k]. The argmax is that
 * of the insert path (FP32 logits with proven error bounds, candidates
 * recomputed with a compensated dot product), so it can differ from the
 * exact one only when the two largest logits are within ~1e-9 relative.
 *   Q               B x d FP32 (device)
 *   hit_index       B int64 (device), e.g. lipcache_probe's out_index;
 *                   values must be -1 or in [0, size)
 *   out_consistent  B int8 (device), nullable: 1 consistent, 0 not, -1 miss
 *   n_hits          host, nullable: queries with hit_index >= 0
 *   n_consistent    host, nullable: of those, the consistent ones
 * Synchronises `stream`. Errors: E_STATE (no head), E_INVALID (NULL Q or
 * hit_index, or an index outside [-1, size): reported after the kernel ran;
 * out_consistent is then -1 for such queries and they are not counted),
 * E_NOMEM, E_CUDA.
 */
lipcache_status lipcache_consistency(lipcache_t* h, const float* Q, int64_t B, const int64_t* hit_index,
                                     int8_t* out_consistent, int64_t* n_hits, int64_t* n_consistent,
                                     lipcache_stream_t stream);

/*
 * Radius policy of the probe: the certified per-entry radius (the default),
 * or one of the two empirical reuse boundaries Sec. 5.4 compares it with.
 * The probe kernels are unchanged; only the per-entry thresholds they read
 * are replaced (the certified ones are kept and come back with
 * LIPCACHE_POLICY_CERTIFIED).
 *   LIPCACHE_POLICY_CERTIFIED   param ignored
 *   LIPCACHE_POLICY_GLOBAL      param = tau > 0: r_i = tau for every entry
 *   LIPCACHE_POLICY_INTERCLASS  param = beta > 0: mu_c = mean key of the
 *       entries with payload label c; r_i = rho_{label_i} with rho_c =
 *       beta / 2 * min over present classes c' != c of ||mu_c - mu_c'||.
 *       Labels outside [0, C), empty classes and a class with no other class
 *       present get 0. The statistics are those of the cache at this call;
 *       entries inserted later take rho of their label from this snapshot.
 * Thresholds derive from r as the certified ones do from r_safe, so a hit
 * always lies strictly inside the policy's radius. Empirical boundaries
 * carry no certificate: lipcache_consistency measures what they give up.
 *   rho_out  host, nullable: C per-class radii (tau for every class under
 *            GLOBAL, 0 under CERTIFIED)
 * Synchronises `stream`. Errors: E_STATE (no head), E_INVALID (policy, or
 * param not finite and > 0), E_NOMEM, E_CUDA.
 */
lipcache_status lipcache_set_radius_policy(lipcache_t* h, int32_t policy, double param, double* rho_out,
                                           lipcache_stream_t stream);

/*
 * Read back cache entries [first, first + n) (insertion order): the triples
 * (z_i, y~_i, r_i) of the cache (Sec. 3.1), with y^G of each key, e.g. to
 * inspect a cache or to persist it: re-inserting the returned keys with their
 * labels as payload into a cache with the same head rebuilds the same entries.
 *   keys_host    n x d FP32 (host), nullable
 *   radius_host  n FP32 (host), nullable: the reported radius r of each entry
 *   label_host   n int32 (host), nullable: payload
 *   yG_host      n int32 (host), nullable: GuardNet label of the key
 * Synchronises `stream`. Errors: E_INVALID (range outside [0, size)), E_CUDA.
 */
lipcache_status lipcache_read_entries(lipcache_t* h, int64_t first, int64_t n, float* keys_host, float* radius_host,
                                      int32_t* label_host, int32_t* yG_host, lipcache_stream_t stream);

/*
 * Copy the head set by lipcache_set_head, W and b of the affine
 * classification head (Eq. 5), back to the host (with
 * lipcache_read_entries, what a checkpoint needs: a cache is restored by
 * set_head and re-inserting the entries' keys with their labels as payload,
 * which re-certifies them to the same radii).
 *   W_host  C x d FP32 row-major (host), nullable
 *   b_host  C FP32 (host), nullable
 * Synchronises `stream`. Errors: E_STATE (no head), E_CUDA.
 */
lipcache_status lipcache_read_head(lipcache_t* h, float* W_host, float* b_host, lipcache_stream_t stream);

/*
 * Test hooks for failure detection. LIPCACHE_DEBUG_STALL_PROBE makes the MMA
 * issuer of the tensor probe kernels first wait on an mbarrier that nothing
 * arrives on: the bounded wait (~2^31 cycles, about a second) expires, the
 * kernel takes its abort path (no trap, no hang), the batch's queries come
 * back as misses, lipcache_info.device_errors counts the aborted CTAs, and
 * the synchronous entry points (lipcache_probe_host, _probe_writeback)
 * return LIPCACHE_E_DEVICE. The exact kernel has no waits and is unaffected.
 * flags = 0 restores normal operation. Errors: E_INVALID (unknown bits).
 */
#define LIPCACHE_DEBUG_STALL_PROBE 1
/* Certify inserted rows with the 64-row-tile kernel where the wide-tile one
 * would run; both compute the same values, so tests compare them bit for bit. */
#define LIPCACHE_DEBUG_INSERT_TILE64 2
/* Certify with the wide-tile kernel where the tensor one would run (tests
 * compare the two). */
#define LIPCACHE_DEBUG_INSERT_WIDE_TILE 4
/* The MMA issuer of the tensor certify kernel first waits on an mbarrier that
 * nothing arrives on: the bounded wait expires, the kernel aborts, no row is
 * appended and lipcache_insert (and the other certifying entry points)
 * return LIPCACHE_E_DEVICE with the cache unchanged. */
#define LIPCACHE_DEBUG_STALL_INSERT 8
/* The tensor certify kernel leaves the rows it lists for the FP64 pass to
 * the stand-alone pass launched after it, instead of re-certifying them on
 * its own spare warp; both compute the same values (tests compare them bit
 * for bit; the bench times both). */
#define LIPCACHE_DEBUG_INSERT_FIX_STANDALONE 16
lipcache_status lipcache_set_debug(lipcache_t* h, int32_t flags);

/*
 * lipcache_probe (Algorithm 2, Eqs. 13-15) for callers holding HOST buffers:
 * copies Q to the device, probes, copies the results back and synchronises
 * `stream`.
 *   Q_host     B x d FP32 (host; pinned memory gives asynchronous copies)
 *   out_*_host host, same meaning as lipcache_probe (out_label/out_dist nullable)
 * Returns LIPCACHE_E_DEVICE (outputs written: all misses) if a bounded wait
 * of the probe kernel expired during the call.
 */
lipcache_status lipcache_probe_host(lipcache_t* h, const float* Q_host, int64_t B, int64_t* out_index_host,
                                    int32_t* out_label_host, float* out_dist_host, lipcache_stream_t stream);

/*
 * lipcache_probe for callers that cannot allocate device memory while they
 * run — e.g. a serving loop whose device memory belongs entirely to another
 * allocator, or whose latency budget cannot absorb cudaMalloc/cudaFree, which
 * may block and synchronise the device. The paper has no counterpart: this is
 * an interface choice of this library, not part of the method.
 * Same arguments, results and errors as lipcache_probe, but the probe's
 * scratch lives in one fixed array compiled into the library
 * (LIPCACHE_NOALLOC_SCRATCH_BYTES per device, held by every GPU that loads
 * the library until the process exits) and nothing is allocated.
 * Limit: ceil(B/128)*128 * (4*d_pad + 12) bytes, plus alignment, must fit the
 * array (e.g. 4,096 queries at d <= 256); larger batches get E_INVALID with
 * the sizes in the message. The first call on a device resolves the array's
 * device address (cudaGetSymbolAddress); make that first call before any
 * stream capture. All calls on a device share the array: calls whose GPU work
 * overlaps (other streams, handles or threads on the same device) race on it
 * and must be serialised by the caller. The resolved address is cached for the
 * life of the process: like every handle, it does not survive a reset of the
 * device's primary context (cudaDeviceReset); do not call this entry point
 * after one.
 */
#define LIPCACHE_NOALLOC_SCRATCH_BYTES 4259840
lipcache_status lipcache_probe_noalloc(lipcache_t* h, const float* Q, int64_t B, int64_t* out_index,
                                       int32_t* out_label, float* out_dist, lipcache_stream_t stream);

/* Select the probe kernel (LIPCACHE_PROBE_*) that evaluates the lookup of
 * Algorithm 2 (Eqs. 13-15, the O(Nd) scan of Sec. 3.4 / Eq. 16); every path
 * returns the same results. E_INVALID for an unknown path or TENSOR when
 * d > 256. */
lipcache_status lipcache_set_probe_path(lipcache_t* h, int32_t path);

/* Radius tightening kappa in (0, 1] (Sec. 5.6): radii of rows inserted
 * afterwards are multiplied by kappa. Only while the cache is empty. */
lipcache_status lipcache_set_radius_scale(lipcache_t* h, double kappa);

/* Options of the spectral norm sigma_max(W) (Sec. 4.1, Eqs. 17-19):
 * `squarings` (0..60) normalised squarings of W^T W before the power
 * iteration and `max_iter` (>= 1) power iterations. */
lipcache_status lipcache_set_spectral_options(lipcache_t* h, int32_t squarings, int32_t max_iter);

/* Pre-size the probe scratch for batches of up to max_batch queries so that
 * later probes allocate nothing (memory management of this library; no
 * counterpart in the paper). */
lipcache_status lipcache_reserve(lipcache_t* h, int64_t max_batch);

/* Instrumentation (no counterpart in the paper). When on, each probe times
 * its main kernel (the screen/recheck kernel, not the prologue and
 * finalize), and each certifying call its certify kernel, with a pair of
 * CUDA events recorded on the call's stream. lipcache_get_info returns the
 * last probe duration and, for probes and certify kernels, the sum and count
 * since the last lipcache_reset_stats. */
lipcache_status lipcache_enable_timing(lipcache_t* h, int32_t on);

/* Fill *info (host): sizes, sigma_max (Sec. 4.1), kernels used, counters and
 * timings (introspection; no counterpart in the paper). Synchronises the
 * device work of this handle. */
lipcache_status lipcache_get_info(lipcache_t* h, lipcache_info* info);

/* Zero the candidate / device-error counters and the kernel-time sum
 * (instrumentation; no counterpart in the paper). */
lipcache_status lipcache_reset_stats(lipcache_t* h);

/* Number of cache entries |C| (Sec. 3.1; 0 for NULL). Settles asynchronous
 * inserts first (synchronises their stream). */
int64_t lipcache_size(const lipcache_t* h);

/* Free the cache C (Sec. 3.1), its head and its device memory, after waiting
 * for asynchronous inserts still running. NULL-safe. */
void lipcache_destroy(lipcache_t* h);

/* Message of the last failed call on this thread ("" if none; error
 * reporting of this library, no counterpart in the paper). */
const char* lipcache_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* LIPCACHE_H */
