// C ABI of the certified cache lookup: argument checks, ownership of the
// cache table and scratch memory, and kernel launches on the caller's stream.
// Declarations and contracts: include/lipcache.h.
#include <nvtx3/nvToolsExt.h>

#include <cstdio>
#include <cstring>
#include <string>

#include "internal.cuh"

#define LC_API extern "C" __attribute__((visibility("default")))

namespace lc {
size_t certify_smem_bytes(int d, int C);
void reserve_probe(lipcache* h, int64_t max_batch);
}  // namespace lc

namespace {

thread_local std::string g_err;

// An NVTX range around an entry point (a no-op unless a profiler is attached),
// so that `ncu --nvtx` can select a call's kernels.
struct Range {
  explicit Range(const char* name) { nvtxRangePushA(name); }
  ~Range() { nvtxRangePop(); }
};

template <typename F>
lipcache_status guarded(F&& f) {
  try {
    f();
    g_err.clear();
    return LIPCACHE_OK;
  } catch (const lc::Error& e) {
    g_err = e.what();
    return e.status;
  } catch (const std::bad_alloc&) {
    g_err = "host allocation failed";
    return LIPCACHE_E_NOMEM;
  } catch (const std::exception& e) {
    g_err = e.what();
    return LIPCACHE_E_CUDA;
  } catch (...) {
    g_err = "unknown error";
    return LIPCACHE_E_CUDA;
  }
}

void use_device(const lipcache* h) { LC_CUDA(cudaSetDevice(h->device)); }

// The exact table size (after asynchronous inserts), on the cache's device.
void sync_size(lipcache* h) {
  use_device(h);
  lc::settle_size(h);
}

template <typename T>
void dev_alloc(T*& p, size_t n) {
  LC_CUDA(cudaMalloc(&p, sizeof(T) * (n ? n : 1)));
}

template <typename T>
void dev_free(T*& p) {
  if (p) cudaFree(p);
  p = nullptr;
}

void release(lipcache* h) {
  if (!h) return;
  cudaSetDevice(h->device);
  // asynchronous inserts may still be writing the table
  if (h->size_pending) cudaStreamSynchronize(h->pending_stream);
  dev_free(h->W);
  dev_free(h->wt_prep);
  dev_free(h->b);
  dev_free(h->Wnorm);
  dev_free(h->Wnorm32);
  dev_free(h->pairnorm);
  dev_free(h->inv_pairnorm);
  dev_free(h->ipn_up32);
  dev_free(h->ipn_dn32);
  dev_free(h->ipn_min32);
  dev_free(h->ipn_max32);
  dev_free(h->gram[0]);
  dev_free(h->gram[1]);
  dev_free(h->spec);
  if (h->spec_host) cudaFreeHost(h->spec_host);
  lc::release_select(h);
  dev_free(h->rr_emp);
  dev_free(h->tau_emp);
  dev_free(h->rho);
  dev_free(h->rho32);
  dev_free(h->cls_sum);
  dev_free(h->cls_cnt);
  dev_free(h->table.keys);
  dev_free(h->table.kn);
  dev_free(h->table.tau);
  dev_free(h->table.rr);
  dev_free(h->table.radius);
  dev_free(h->table.label);
  dev_free(h->table.yG);
  dev_free(h->ins_accept);
  dev_free(h->ins_yG);
  dev_free(h->ins_label);
  dev_free(h->ins_radius);
  dev_free(h->ins_rr);
  dev_free(h->ins_kn);
  dev_free(h->ins_tau);
  dev_free(h->ins_rank);
  dev_free(h->ins_fix);
  dev_free(h->ins_bcount);
  dev_free(h->ins_boffset);
  dev_free(h->ins_total);
  dev_free(h->size_dev);
  dev_free(h->ins_size0);
  if (h->size_pinned) cudaFreeHost(h->size_pinned);
  if (h->ins_total_host) cudaFreeHost(h->ins_total_host);
  dev_free(h->qpad);
  dev_free(h->kappa);
  dev_free(h->best);
  dev_free(h->hq);
  dev_free(h->hidx);
  dev_free(h->hlabel);
  dev_free(h->hdist);
  dev_free(h->stats);
  if (h->stats_host) cudaFreeHost(h->stats_host);
  for (int i = 0; i < lipcache::kTimingRing; ++i) {
    if (h->tev0[i]) cudaEventDestroy(h->tev0[i]);
    if (h->tev1[i]) cudaEventDestroy(h->tev1[i]);
  }
  delete h;
}

void check_handle(const lipcache* h) { LC_REQUIRE(h != nullptr, LIPCACHE_E_INVALID, "NULL cache handle"); }

void resolve_encoder(lipcache* h) {
  void* fn = nullptr;
  cudaDriverEntryPointQueryResult q;
  cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
  if (e == cudaSuccess && q == cudaDriverEntryPointSuccess) h->encode = reinterpret_cast<lc::EncodeTiledFn>(fn);
}

}  // namespace

// Runs fn(ctx) under the same error handling as every other entry point.
lipcache_status lc::run_guarded(void (*fn)(void*), void* ctx) {
  return guarded([&] { fn(ctx); });
}

void lc::harvest_timing(lipcache* h, bool all) {
  while (h->t_harvested < h->t_issued) {
    const int slot = (int)(h->t_harvested % lipcache::kTimingRing);
    const bool full = h->t_issued - h->t_harvested >= lipcache::kTimingRing;
    if (!all && !full) break;
    LC_CUDA(cudaEventSynchronize(h->tev1[slot]));
    float ms = 0.f;
    LC_CUDA(cudaEventElapsedTime(&ms, h->tev0[slot], h->tev1[slot]));
    if (h->t_kind[slot]) {
      h->ti_ms_total += ms;
      ++h->ti_count;
    } else {
      h->last_ms = ms;
      h->t_ms_total += ms;
      ++h->t_count;
    }
    ++h->t_harvested;
  }
}

// After a synchronised probe: E_DEVICE if a bounded wait of the kernel expired.
static void require_no_abort(lipcache* h, cudaStream_t s) {
  LC_CUDA(cudaMemcpyAsync(h->stats_host, h->stats, sizeof(lc::DevStats), cudaMemcpyDeviceToHost, s));
  LC_CUDA(cudaStreamSynchronize(s));
  LC_REQUIRE(h->stats_host->abort_flag == 0, LIPCACHE_E_DEVICE,
             "a bounded wait of the probe kernel expired; the batch's queries were reported as misses");
}

LC_API const char* lipcache_last_error(void) { return g_err.c_str(); }

LC_API lipcache_status lipcache_create(int32_t d, int32_t C, int64_t capacity, int32_t radius_mode,
                                       lipcache_t** out) {
  if (out) *out = nullptr;
  lipcache* h = nullptr;
  lipcache_status st = guarded([&] {
    LC_REQUIRE(out != nullptr, LIPCACHE_E_INVALID, "out is NULL");
    LC_REQUIRE(d >= 1 && d <= LIPCACHE_MAX_DIM, LIPCACHE_E_INVALID, "d must be in [1, LIPCACHE_MAX_DIM]");
    LC_REQUIRE(C >= 2 && C <= LIPCACHE_MAX_CLASSES, LIPCACHE_E_INVALID, "C must be in [2, LIPCACHE_MAX_CLASSES]");
    LC_REQUIRE(capacity >= 1 && capacity <= LIPCACHE_MAX_CAPACITY, LIPCACHE_E_INVALID,
               "capacity must be in [1, 2^31 - 1]");
    LC_REQUIRE(radius_mode == LIPCACHE_RADIUS_CONSERVATIVE || radius_mode == LIPCACHE_RADIUS_TIGHT,
               LIPCACHE_E_INVALID, "unknown radius mode");
    LC_REQUIRE(lc::certify_smem_bytes(d, C) <= 200 * 1024, LIPCACHE_E_INVALID,
               "d and C too large together for the insert kernel's shared memory");
    h = new lipcache();
    LC_CUDA(cudaGetDevice(&h->device));
    LC_CUDA(cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, h->device));
    h->d = d;
    h->C = C;
    h->dpad = (d + 31) / 32 * 32;
    h->capacity = capacity;
    h->radius_mode = radius_mode;
    h->eps_rc = lc::eps_recheck(h->dpad);
    h->c_scr = lc::c_screen(h->dpad);
    dev_alloc(h->W, (size_t)C * d);
    dev_alloc(h->b, (size_t)C);
    dev_alloc(h->Wnorm, (size_t)C);
    dev_alloc(h->Wnorm32, (size_t)C);
    if (radius_mode == LIPCACHE_RADIUS_TIGHT) {
      dev_alloc(h->pairnorm, (size_t)C * C);
      dev_alloc(h->inv_pairnorm, (size_t)C * C);
      dev_alloc(h->ipn_up32, (size_t)C * C);
      dev_alloc(h->ipn_dn32, (size_t)C * C);
      dev_alloc(h->ipn_min32, (size_t)C);
      dev_alloc(h->ipn_max32, (size_t)C);
    }
    dev_alloc(h->gram[0], (size_t)d * d);
    dev_alloc(h->gram[1], (size_t)d * d);
    dev_alloc(h->spec, 1);
    LC_CUDA(cudaMallocHost(&h->spec_host, sizeof(lc::SpecResult)));
    // Whole key tiles: rows past the current size are zero keys whose screen
    // term tau is 0x7f7f7f7f (3.4e38), so no probe ever selects them.
    h->table_rows = (capacity + 255) / 256 * 256;
    const size_t rows = (size_t)h->table_rows;
    dev_alloc(h->table.keys, rows * h->dpad);
    LC_CUDA(cudaMemset(h->table.keys, 0, sizeof(float) * rows * h->dpad));
    dev_alloc(h->table.kn, rows);
    dev_alloc(h->table.tau, rows);
    LC_CUDA(cudaMemset(h->table.tau, 0x7f, sizeof(float) * rows));
    dev_alloc(h->table.rr, rows);
    LC_CUDA(cudaMemset(h->table.rr, 0, sizeof(float) * rows));
    dev_alloc(h->table.radius, rows);
    dev_alloc(h->table.label, rows);
    dev_alloc(h->table.yG, rows);
    dev_alloc(h->ins_total, 4);
    LC_CUDA(cudaMallocHost(&h->ins_total_host, 4 * sizeof(int64_t)));
    dev_alloc(h->size_dev, 1);
    LC_CUDA(cudaMemset(h->size_dev, 0, sizeof(int64_t)));
    dev_alloc(h->ins_size0, 1);
    LC_CUDA(cudaMallocHost(&h->size_pinned, sizeof(int64_t)));
    dev_alloc(h->stats, 1);
    LC_CUDA(cudaMemset(h->stats, 0, sizeof(lc::DevStats)));
    LC_CUDA(cudaMallocHost(&h->stats_host, sizeof(lc::DevStats)));
    for (int i = 0; i < lipcache::kTimingRing; ++i) {
      LC_CUDA(cudaEventCreate(&h->tev0[i]));
      LC_CUDA(cudaEventCreate(&h->tev1[i]));
    }
    resolve_encoder(h);
    LC_CUDA(cudaDeviceSynchronize());
  });
  if (st != LIPCACHE_OK) {
    release(h);
    return st;
  }
  *out = h;
  return st;
}

LC_API void lipcache_destroy(lipcache_t* h) { release(h); }

LC_API int64_t lipcache_size(const lipcache_t* h) {
  if (!h) return 0;
  lipcache* m = const_cast<lipcache*>(h);
  guarded([&] { sync_size(m); });  // on a CUDA error the last settled size is returned
  return m->size;
}

LC_API lipcache_status lipcache_set_head(lipcache_t* h, const float* W, const float* b, double* sigma_out,
                                         lipcache_stream_t stream) {
  return guarded([&] {
    Range nvtx_range("lipcache_set_head");
    check_handle(h);
    LC_REQUIRE(W != nullptr && b != nullptr, LIPCACHE_E_INVALID, "W and b must be device pointers");
    sync_size(h);
    LC_REQUIRE(h->size == 0, LIPCACHE_E_STATE, "set_head requires an empty cache (radii depend on W)");
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    h->head_set = false;
    h->wt_prep_ncg = 0;
    LC_CUDA(cudaMemcpyAsync(h->W, W, sizeof(float) * (size_t)h->C * h->d, cudaMemcpyDeviceToDevice, s));
    LC_CUDA(cudaMemcpyAsync(h->b, b, sizeof(float) * (size_t)h->C, cudaMemcpyDeviceToDevice, s));
    lc::spectral_norm(h, s);
    LC_CUDA(cudaMemcpyAsync(h->spec_host, h->spec, sizeof(lc::SpecResult), cudaMemcpyDeviceToHost, s));
    LC_CUDA(cudaStreamSynchronize(s));
    const lc::SpecResult r = *h->spec_host;
    h->sigma_iterations = r.iterations;
    h->sigma_residual = r.residual_rel;
    LC_REQUIRE(!r.degenerate && r.sigma > 0.0, LIPCACHE_E_DEGENERATE_HEAD,
               "sigma_max(W) <= 0: the GuardNet head is degenerate (Algorithm 1 stops construction)");
    LC_REQUIRE(r.converged, LIPCACHE_E_NOT_CONVERGED,
               "spectral power iteration reached max_iter without meeting its tolerance");
    LC_REQUIRE(std::isfinite(r.sigma), LIPCACHE_E_DEGENERATE_HEAD, "sigma_max(W) is not finite");
    h->sigma = r.sigma;
    h->head_set = true;
    if (sigma_out) *sigma_out = r.sigma;
  });
}

LC_API lipcache_status lipcache_insert(lipcache_t* h, const float* H, int64_t n, const int32_t* payload,
                                       int32_t require_consistency, int64_t* out_index, float* out_radius,
                                       int64_t* n_accepted, lipcache_stream_t stream) {
  if (n_accepted) *n_accepted = 0;
  return guarded([&] {
    Range nvtx_range("lipcache_insert");
    check_handle(h);
    LC_REQUIRE(h->head_set, LIPCACHE_E_STATE, "insert before set_head");
    LC_REQUIRE(n >= 0, LIPCACHE_E_INVALID, "n must be >= 0");
    if (n == 0) return;
    LC_REQUIRE(H != nullptr, LIPCACHE_E_INVALID, "H is NULL");
    LC_REQUIRE(((uintptr_t)H & 3) == 0, LIPCACHE_E_INVALID, "H must be 4-byte aligned");
    use_device(h);
    // unsettled asynchronous inserts grew the table by at most pending_rows
    if (n > h->capacity - h->size - h->pending_rows) lc::settle_size(h);
    LC_REQUIRE(n <= h->capacity - h->size - h->pending_rows, LIPCACHE_E_FULL, "insert would exceed the cache capacity");
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (h->size_pending && s != h->pending_stream) lc::settle_size(h);  // keep every pending insert on one stream
    lc::certify_insert(h, H, n, payload, require_consistency, out_index, out_radius, s);
    if (n_accepted == nullptr && h->policy == LIPCACHE_POLICY_CERTIFIED) {
      // asynchronous: nothing to report on the host, so no wait
      h->size_pending = true;
      h->pending_rows += n;
      h->pending_stream = s;
      return;
    }
    LC_CUDA(cudaMemcpyAsync(h->ins_total_host, h->ins_total, sizeof(int64_t), cudaMemcpyDeviceToHost, s));
    LC_CUDA(cudaMemcpyAsync(h->size_pinned, h->size_dev, sizeof(int64_t), cudaMemcpyDeviceToHost, s));
    LC_CUDA(cudaMemcpyAsync(h->stats_host, h->stats, sizeof(lc::DevStats), cudaMemcpyDeviceToHost, s));
    LC_CUDA(cudaStreamSynchronize(s));
    h->size = *h->size_pinned;  // includes earlier asynchronous inserts on this stream
    h->size_pending = false;
    h->pending_rows = 0;
    LC_REQUIRE(h->stats_host->abort_flag == 0, LIPCACHE_E_DEVICE, lc::kCertifyAbortMessage);
    const int64_t acc = *h->ins_total_host;
    const int64_t first = h->size - acc;
    if (n_accepted) *n_accepted = acc;
    if (h->policy != LIPCACHE_POLICY_CERTIFIED && acc > 0) {
      lc::policy_fill(h, first, acc, s);
      LC_CUDA(cudaStreamSynchronize(s));
    }
  });
}

LC_API lipcache_status lipcache_probe(lipcache_t* h, const float* Q, int64_t B, int64_t* out_index,
                                      int32_t* out_label, float* out_dist, lipcache_stream_t stream) {
  return guarded([&] {
    Range nvtx_range("lipcache_probe");
    check_handle(h);
    sync_size(h);  // the exact table size (after asynchronous inserts)
    LC_REQUIRE(h->head_set, LIPCACHE_E_STATE, "probe before set_head");
    LC_REQUIRE(B >= 0 && B <= (1LL << 22), LIPCACHE_E_INVALID, "B must be in [0, 2^22]");
    if (B == 0) return;
    LC_REQUIRE(Q != nullptr && out_index != nullptr, LIPCACHE_E_INVALID, "Q and out_index are required");
    LC_REQUIRE(((uintptr_t)Q & 3) == 0, LIPCACHE_E_INVALID, "Q must be 4-byte aligned");
    use_device(h);
    lc::probe(h, Q, B, out_index, out_label, out_dist, reinterpret_cast<cudaStream_t>(stream));
  });
}

LC_API lipcache_status lipcache_insert_select(lipcache_t* h, const float* H, int64_t n, const int32_t* payload,
                                              int32_t require_consistency, int32_t strategy, int64_t budget_total,
                                              int32_t budget_per_class, int64_t* out_index, float* out_radius,
                                              int64_t* n_selected, lipcache_stream_t stream) {
  if (n_selected) *n_selected = 0;
  return guarded([&] {
    Range nvtx_range("lipcache_insert_select");
    check_handle(h);
    sync_size(h);  // the exact table size (after asynchronous inserts)
    LC_REQUIRE(strategy == LIPCACHE_SELECT_ALL || strategy == LIPCACHE_SELECT_RADIUS_DEDUP ||
                   strategy == LIPCACHE_SELECT_KCENTER,
               LIPCACHE_E_INVALID, "unknown selection strategy");
    LC_REQUIRE(strategy != LIPCACHE_SELECT_KCENTER || (budget_per_class > 0 && budget_total <= 0), LIPCACHE_E_INVALID,
               "K-center takes a per-class budget and no total budget");
    if (strategy == LIPCACHE_SELECT_ALL) {
      LC_REQUIRE(budget_total <= 0 && budget_per_class <= 0, LIPCACHE_E_INVALID,
                 "LIPCACHE_SELECT_ALL takes no budget");
      const lipcache_status st = lipcache_insert(h, H, n, payload, require_consistency, out_index, out_radius,
                                                 n_selected, stream);
      if (st != LIPCACHE_OK) throw lc::Error(st, lipcache_last_error());
      return;
    }
    LC_REQUIRE(h->head_set, LIPCACHE_E_STATE, "insert before set_head");
    LC_REQUIRE(h->policy == LIPCACHE_POLICY_CERTIFIED, LIPCACHE_E_STATE,
               "selection needs the certified radius policy");
    LC_REQUIRE(n >= 0 && n < (1LL << 31), LIPCACHE_E_INVALID, "n must be in [0, 2^31)");
    if (n == 0) return;
    LC_REQUIRE(H != nullptr, LIPCACHE_E_INVALID, "H is NULL");
    LC_REQUIRE(((uintptr_t)H & 3) == 0, LIPCACHE_E_INVALID, "H must be 4-byte aligned");
    int64_t most = budget_total > 0 && budget_total < n ? budget_total : n;
    if (strategy == LIPCACHE_SELECT_KCENTER && (int64_t)budget_per_class * h->C < most)
      most = (int64_t)budget_per_class * h->C;
    LC_REQUIRE(most <= h->capacity - h->size, LIPCACHE_E_FULL, "the selection could exceed the cache capacity");
    use_device(h);
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    const int64_t kept =
        strategy == LIPCACHE_SELECT_KCENTER
            ? lc::select_kcenter(h, H, n, payload, require_consistency, budget_per_class, out_index, out_radius, s)
            : lc::select_insert(h, H, n, payload, require_consistency, budget_total, budget_per_class, out_index,
                                out_radius, s);
    LC_CUDA(cudaStreamSynchronize(s));
    if (n_selected) *n_selected = kept;
  });
}

LC_API lipcache_status lipcache_probe_writeback(lipcache_t* h, const float* Q, int64_t B, const int32_t* payload,
                                                int32_t require_consistency, int64_t* out_index, int32_t* out_label,
                                                float* out_dist, int64_t* out_inserted, int64_t* n_inserted,
                                                lipcache_stream_t stream) {
  if (n_inserted) *n_inserted = 0;
  return guarded([&] {
    Range nvtx_range("lipcache_probe_writeback");
    check_handle(h);
    sync_size(h);  // the exact table size (after asynchronous inserts)
    LC_REQUIRE(h->head_set, LIPCACHE_E_STATE, "probe before set_head");
    LC_REQUIRE(B >= 0 && B <= (1LL << 22), LIPCACHE_E_INVALID, "B must be in [0, 2^22]");
    if (B == 0) return;
    LC_REQUIRE(Q != nullptr && out_index != nullptr, LIPCACHE_E_INVALID, "Q and out_index are required");
    LC_REQUIRE(((uintptr_t)Q & 3) == 0, LIPCACHE_E_INVALID, "Q must be 4-byte aligned");
    LC_REQUIRE(B <= h->capacity - h->size, LIPCACHE_E_FULL, "write-back of B queries could exceed the capacity");
    use_device(h);
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    lc::probe(h, Q, B, out_index, out_label, out_dist, s);
    require_no_abort(h, s);  // an aborted probe reports misses: write nothing back
    lc::certify_insert(h, Q, B, payload, require_consistency, out_inserted, nullptr, s, out_index);
    LC_CUDA(cudaMemcpyAsync(h->ins_total_host, h->ins_total, sizeof(int64_t), cudaMemcpyDeviceToHost, s));
    LC_CUDA(cudaMemcpyAsync(h->stats_host, h->stats, sizeof(lc::DevStats), cudaMemcpyDeviceToHost, s));
    LC_CUDA(cudaStreamSynchronize(s));
    LC_REQUIRE(h->stats_host->abort_flag == 0, LIPCACHE_E_DEVICE, lc::kCertifyAbortMessage);
    const int64_t acc = *h->ins_total_host;
    const int64_t first = h->size;
    h->size += acc;
    if (n_inserted) *n_inserted = acc;
    if (h->policy != LIPCACHE_POLICY_CERTIFIED && acc > 0) {
      lc::policy_fill(h, first, acc, s);
      LC_CUDA(cudaStreamSynchronize(s));
    }
  });
}

LC_API lipcache_status lipcache_consistency(lipcache_t* h, const float* Q, int64_t B, const int64_t* hit_index,
                                            int8_t* out_consistent, int64_t* n_hits, int64_t* n_consistent,
                                            lipcache_stream_t stream) {
  if (n_hits) *n_hits = 0;
  if (n_consistent) *n_consistent = 0;
  return guarded([&] {
    Range nvtx_range("lipcache_consistency");
    check_handle(h);
    sync_size(h);  // the exact table size (after asynchronous inserts)
    LC_REQUIRE(h->head_set, LIPCACHE_E_STATE, "consistency check before set_head");
    LC_REQUIRE(B >= 0 && B <= (1LL << 22), LIPCACHE_E_INVALID, "B must be in [0, 2^22]");
    if (B == 0) return;
    LC_REQUIRE(Q != nullptr && hit_index != nullptr, LIPCACHE_E_INVALID, "Q and hit_index are required");
    LC_REQUIRE(((uintptr_t)Q & 3) == 0, LIPCACHE_E_INVALID, "Q must be 4-byte aligned");
    use_device(h);
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    lc::consistency_check(h, Q, B, hit_index, out_consistent, s);
    LC_CUDA(cudaMemcpyAsync(h->ins_total_host + 1, h->ins_total + 1, 3 * sizeof(int64_t), cudaMemcpyDeviceToHost, s));
    LC_CUDA(cudaMemcpyAsync(h->stats_host, h->stats, sizeof(lc::DevStats), cudaMemcpyDeviceToHost, s));
    LC_CUDA(cudaStreamSynchronize(s));
    LC_REQUIRE(h->stats_host->abort_flag == 0, LIPCACHE_E_DEVICE, lc::kCertifyAbortMessage);
    if (n_hits) *n_hits = h->ins_total_host[1];
    if (n_consistent) *n_consistent = h->ins_total_host[2];
    LC_REQUIRE(h->ins_total_host[3] == 0, LIPCACHE_E_INVALID, "hit_index holds values outside [-1, size)");
  });
}

LC_API lipcache_status lipcache_set_radius_policy(lipcache_t* h, int32_t policy, double param, double* rho_out,
                                                  lipcache_stream_t stream) {
  return guarded([&] {
    Range nvtx_range("lipcache_set_radius_policy");
    check_handle(h);
    sync_size(h);  // the exact table size (after asynchronous inserts)
    LC_REQUIRE(h->head_set, LIPCACHE_E_STATE, "set_radius_policy before set_head");
    LC_REQUIRE(policy == LIPCACHE_POLICY_CERTIFIED || policy == LIPCACHE_POLICY_GLOBAL ||
                   policy == LIPCACHE_POLICY_INTERCLASS,
               LIPCACHE_E_INVALID, "unknown radius policy");
    LC_REQUIRE(policy == LIPCACHE_POLICY_CERTIFIED || (std::isfinite(param) && param > 0.0), LIPCACHE_E_INVALID,
               "the policy parameter must be finite and > 0");
    use_device(h);
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    lc::set_radius_policy(h, policy, param, rho_out, s);
    if (rho_out && policy == LIPCACHE_POLICY_CERTIFIED)
      for (int c = 0; c < h->C; ++c) rho_out[c] = 0.0;
  });
}

LC_API lipcache_status lipcache_read_entries(lipcache_t* h, int64_t first, int64_t n, float* keys_host,
                                             float* radius_host, int32_t* label_host, int32_t* yG_host,
                                             lipcache_stream_t stream) {
  return guarded([&] {
    Range nvtx_range("lipcache_read_entries");
    check_handle(h);
    sync_size(h);  // the exact table size (after asynchronous inserts)
    LC_REQUIRE(first >= 0 && n >= 0 && first + n <= h->size, LIPCACHE_E_INVALID, "entries outside [0, size)");
    if (n == 0) return;
    use_device(h);
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (keys_host)
      LC_CUDA(cudaMemcpy2DAsync(keys_host, sizeof(float) * (size_t)h->d, h->table.keys + (size_t)first * h->dpad,
                                sizeof(float) * (size_t)h->dpad, sizeof(float) * (size_t)h->d, (size_t)n,
                                cudaMemcpyDeviceToHost, s));
    if (radius_host)
      LC_CUDA(cudaMemcpyAsync(radius_host, h->table.radius + first, sizeof(float) * (size_t)n, cudaMemcpyDeviceToHost,
                              s));
    if (label_host)
      LC_CUDA(cudaMemcpyAsync(label_host, h->table.label + first, sizeof(int32_t) * (size_t)n,
                              cudaMemcpyDeviceToHost, s));
    if (yG_host)
      LC_CUDA(cudaMemcpyAsync(yG_host, h->table.yG + first, sizeof(int32_t) * (size_t)n, cudaMemcpyDeviceToHost, s));
    LC_CUDA(cudaStreamSynchronize(s));
  });
}

LC_API lipcache_status lipcache_read_head(lipcache_t* h, float* W_host, float* b_host, lipcache_stream_t stream) {
  return guarded([&] {
    check_handle(h);
    LC_REQUIRE(h->head_set, LIPCACHE_E_STATE, "read_head before set_head");
    use_device(h);
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (W_host)
      LC_CUDA(cudaMemcpyAsync(W_host, h->W, sizeof(float) * (size_t)h->C * h->d, cudaMemcpyDeviceToHost, s));
    if (b_host) LC_CUDA(cudaMemcpyAsync(b_host, h->b, sizeof(float) * (size_t)h->C, cudaMemcpyDeviceToHost, s));
    LC_CUDA(cudaStreamSynchronize(s));
  });
}

LC_API lipcache_status lipcache_set_debug(lipcache_t* h, int32_t flags) {
  return guarded([&] {
    check_handle(h);
    LC_REQUIRE((flags & ~(LIPCACHE_DEBUG_STALL_PROBE | LIPCACHE_DEBUG_INSERT_TILE64 |
                          LIPCACHE_DEBUG_INSERT_WIDE_TILE | LIPCACHE_DEBUG_STALL_INSERT |
                          LIPCACHE_DEBUG_INSERT_FIX_STANDALONE)) == 0,
               LIPCACHE_E_INVALID,
               "unknown debug flags");
    h->debug_flags = flags;
  });
}

LC_API lipcache_status lipcache_probe_host(lipcache_t* h, const float* Q_host, int64_t B, int64_t* out_index_host,
                                           int32_t* out_label_host, float* out_dist_host, lipcache_stream_t stream) {
  return guarded([&] {
    Range nvtx_range("lipcache_probe_host");
    check_handle(h);
    sync_size(h);  // the exact table size (after asynchronous inserts)
    LC_REQUIRE(h->head_set, LIPCACHE_E_STATE, "probe before set_head");
    LC_REQUIRE(B >= 0 && B <= (1LL << 22), LIPCACHE_E_INVALID, "B must be in [0, 2^22]");
    if (B == 0) return;
    LC_REQUIRE(Q_host != nullptr && out_index_host != nullptr, LIPCACHE_E_INVALID, "Q and out_index are required");
    use_device(h);
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (B > h->hq_cap) {
      dev_free(h->hq);
      dev_free(h->hidx);
      dev_free(h->hlabel);
      dev_free(h->hdist);
      h->hq_cap = 0;
      dev_alloc(h->hq, (size_t)B * h->d);
      dev_alloc(h->hidx, (size_t)B);
      dev_alloc(h->hlabel, (size_t)B);
      dev_alloc(h->hdist, (size_t)B);
      h->hq_cap = B;
    }
    LC_CUDA(cudaMemcpyAsync(h->hq, Q_host, sizeof(float) * (size_t)B * h->d, cudaMemcpyHostToDevice, s));
    lc::probe(h, h->hq, B, h->hidx, h->hlabel, h->hdist, s);
    LC_CUDA(cudaMemcpyAsync(out_index_host, h->hidx, sizeof(int64_t) * (size_t)B, cudaMemcpyDeviceToHost, s));
    if (out_label_host)
      LC_CUDA(cudaMemcpyAsync(out_label_host, h->hlabel, sizeof(int32_t) * (size_t)B, cudaMemcpyDeviceToHost, s));
    if (out_dist_host)
      LC_CUDA(cudaMemcpyAsync(out_dist_host, h->hdist, sizeof(float) * (size_t)B, cudaMemcpyDeviceToHost, s));
    require_no_abort(h, s);
  });
}

LC_API lipcache_status lipcache_set_probe_path(lipcache_t* h, int32_t path) {
  return guarded([&] {
    check_handle(h);
    LC_REQUIRE(path >= LIPCACHE_PROBE_AUTO && path <= LIPCACHE_PROBE_TENSOR_PAIR, LIPCACHE_E_INVALID,
               "unknown probe path");
    LC_REQUIRE(path == LIPCACHE_PROBE_AUTO || path == LIPCACHE_PROBE_EXACT || lc::tensor_path_supported(h->dpad),
               LIPCACHE_E_INVALID, "the tensor probe supports d <= 256");
    h->probe_path = path;
  });
}

LC_API lipcache_status lipcache_set_radius_scale(lipcache_t* h, double kappa) {
  return guarded([&] {
    check_handle(h);
    LC_REQUIRE(kappa > 0.0 && kappa <= 1.0, LIPCACHE_E_INVALID, "kappa must be in (0, 1]");
    sync_size(h);
    LC_REQUIRE(h->size == 0, LIPCACHE_E_STATE, "the radius scale can change only while the cache is empty");
    h->radius_scale = kappa;
  });
}

LC_API lipcache_status lipcache_set_spectral_options(lipcache_t* h, int32_t squarings, int32_t max_iter) {
  return guarded([&] {
    check_handle(h);
    LC_REQUIRE(squarings >= 0 && squarings <= 60, LIPCACHE_E_INVALID, "squarings must be in [0, 60]");
    LC_REQUIRE(max_iter >= 1, LIPCACHE_E_INVALID, "max_iter must be >= 1");
    h->squarings = squarings;
    h->max_iter = max_iter;
  });
}

LC_API lipcache_status lipcache_reserve(lipcache_t* h, int64_t max_batch) {
  return guarded([&] {
    check_handle(h);
    LC_REQUIRE(max_batch >= 0 && max_batch <= (1LL << 22), LIPCACHE_E_INVALID, "max_batch must be in [0, 2^22]");
    use_device(h);
    lc::reserve_probe(h, max_batch);
  });
}

LC_API lipcache_status lipcache_enable_timing(lipcache_t* h, int32_t on) {
  return guarded([&] {
    check_handle(h);
    h->timing = on != 0;
  });
}

LC_API lipcache_status lipcache_reset_stats(lipcache_t* h) {
  return guarded([&] {
    check_handle(h);
    use_device(h);
    LC_CUDA(cudaDeviceSynchronize());
    lc::harvest_timing(h, true);
    h->t_ms_total = 0.0;
    h->t_count = 0;
    h->ti_ms_total = 0.0;
    h->ti_count = 0;
    LC_CUDA(cudaMemset(h->stats, 0, sizeof(lc::DevStats)));
    LC_CUDA(cudaDeviceSynchronize());
  });
}

LC_API lipcache_status lipcache_get_info(lipcache_t* h, lipcache_info* info) {
  return guarded([&] {
    check_handle(h);
    LC_REQUIRE(info != nullptr, LIPCACHE_E_INVALID, "info is NULL");
    sync_size(h);
    LC_CUDA(cudaDeviceSynchronize());
    LC_CUDA(cudaMemcpy(h->stats_host, h->stats, sizeof(lc::DevStats), cudaMemcpyDeviceToHost));
    lc::harvest_timing(h, true);
    std::memset(info, 0, sizeof(*info));
    info->d = h->d;
    info->C = h->C;
    info->d_pad = h->dpad;
    info->radius_mode = h->radius_mode;
    info->capacity = h->capacity;
    info->size = h->size;
    info->head_set = h->head_set ? 1 : 0;
    info->sigma_iterations = h->sigma_iterations;
    info->sigma = h->head_set ? h->sigma : 0.0;
    info->sigma_residual = h->sigma_residual;
    info->radius_scale = h->radius_scale;
    info->eps_recheck = h->eps_rc;
    info->c_screen = h->c_scr;
    info->candidates = (int64_t)h->stats_host->candidates;
    info->device_errors = (int64_t)h->stats_host->errors;
    info->insert_refined_pairs = (int64_t)h->stats_host->ins_pairs;
    info->insert_full_rows = (int64_t)h->stats_host->ins_full_rows;
    info->insert_fp64_rows = (int64_t)h->stats_host->ins_fp64_rows;
    info->probe_path = h->probe_path;
    info->last_probe_path = h->last_probe_path;
    info->last_probe_ms = h->last_ms;
    info->num_sms = h->num_sms;
    info->kernel_ms_total = h->t_ms_total;
    info->kernel_launches = h->t_count;
    info->last_grid = h->last_grid;
    info->last_cluster = h->last_cluster;
    info->radius_policy = h->policy;
    info->insert_kernel_ms_total = h->ti_ms_total;
    info->insert_kernel_launches = h->ti_count;
    info->last_insert_kernel = h->last_insert_kernel;
    info->policy_param = h->policy_param;
  });
}
