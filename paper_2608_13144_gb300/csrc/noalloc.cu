// lipcache_probe_noalloc: the batched lookup for callers that must not
// allocate device memory once they are running. Typical callers: a serving
// loop whose device memory is owned entirely by another allocator (a
// framework's caching allocator, a fixed pre-reserved pool) or whose latency
// budget cannot take a cudaMalloc/cudaFree, which may block and synchronise
// the device. lipcache_probe grows its scratch buffers with cudaMalloc when
// a batch is larger than any before; this entry point instead uses one
// fixed scratch array compiled into the library.
//
// The array is a file-scope __device__ variable: every GPU that loads the
// library holds LIPCACHE_NOALLOC_SCRATCH_BYTES of it until the process exits.
// All calls on a device share it and each call overwrites what it needs
// (padded queries, per-query screen constants, and the reduction words,
// which the prologue kernel resets to their empty value), so calls whose
// work overlaps on the GPU (different streams, handles or threads on the
// same device) race on it and must be serialised by the caller.
#include <mutex>

#include "internal.cuh"

#define LC_API extern "C" __attribute__((visibility("default")))

namespace {

static __device__ __align__(256) unsigned char g_noalloc_scratch[LIPCACHE_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of g_noalloc_scratch on the current device. In host code the
// symbol's name only stands for the variable; its device address comes from
// cudaGetSymbolAddress, resolved once per device (on the first call of that
// device) and cached.
void* scratch_address(int device) {
  LC_REQUIRE(device >= 0 && device < kMaxDevices, LIPCACHE_E_INVALID, "device ordinal out of range");
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_scratch_addr[device]) {
    void* p = nullptr;
    LC_CUDA(cudaGetSymbolAddress(&p, g_noalloc_scratch));
    LC_REQUIRE(p != nullptr, LIPCACHE_E_CUDA, "cudaGetSymbolAddress returned NULL for the scratch array");
    g_scratch_addr[device] = p;
  }
  return g_scratch_addr[device];
}

inline size_t align256(size_t x) { return (x + 255) / 256 * 256; }

}  // namespace

namespace lc {
// Scratch layout inside the static array for a batch of B queries.
struct NoallocLayout {
  size_t qpad, kappa, best, end;
};
NoallocLayout noalloc_layout(int64_t B, int dpad) {
  const size_t Bpad = (size_t)((B + 127) / 128 * 128);
  NoallocLayout L;
  L.qpad = 0;
  L.kappa = align256(L.qpad + Bpad * (size_t)dpad * sizeof(float));
  L.best = align256(L.kappa + Bpad * sizeof(float));
  L.end = L.best + Bpad * sizeof(unsigned long long);
  return L;
}
}  // namespace lc

LC_API lipcache_status lipcache_probe_noalloc(lipcache_t* h, const float* Q, int64_t B, int64_t* out_index,
                                              int32_t* out_label, float* out_dist, lipcache_stream_t stream) {
  struct Ctx {
    lipcache_t* h;
    const float* Q;
    int64_t B;
    int64_t* oi;
    int32_t* ol;
    float* od;
    lipcache_stream_t s;
  } ctx{h, Q, B, out_index, out_label, out_dist, stream};
  return lc::run_guarded(
      [](void* p) {
        Ctx& c = *static_cast<Ctx*>(p);
        LC_REQUIRE(c.h != nullptr, LIPCACHE_E_INVALID, "NULL cache handle");
        LC_REQUIRE(c.h->head_set, LIPCACHE_E_STATE, "probe before set_head");
        LC_REQUIRE(c.B >= 0, LIPCACHE_E_INVALID, "B must be >= 0");
        if (c.B == 0) return;
        LC_REQUIRE(c.Q != nullptr && c.oi != nullptr, LIPCACHE_E_INVALID, "Q and out_index are required");
        LC_REQUIRE(((uintptr_t)c.Q & 3) == 0, LIPCACHE_E_INVALID, "Q must be 4-byte aligned");
        const lc::NoallocLayout L = lc::noalloc_layout(c.B, c.h->dpad);
        LC_REQUIRE(L.end <= (size_t)LIPCACHE_NOALLOC_SCRATCH_BYTES, LIPCACHE_E_INVALID,
                   "batch too large for the fixed no-allocation scratch: need " + std::to_string(L.end) +
                       " bytes (ceil(B/128)*128 rows x (4*d_pad + 12) bytes), the array holds " +
                       std::to_string((long long)LIPCACHE_NOALLOC_SCRATCH_BYTES) + "; use lipcache_probe");
        LC_CUDA(cudaSetDevice(c.h->device));
        if (c.h->size_pending) {
          // asynchronous inserts: their size is settled by synchronising their
          // stream, which a stream being captured into a graph must not do
          cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
          LC_CUDA(cudaStreamIsCapturing(reinterpret_cast<cudaStream_t>(c.s), &cap));
          LC_REQUIRE(cap == cudaStreamCaptureStatusNone, LIPCACHE_E_STATE,
                     "asynchronous inserts are pending: settle them (lipcache_size) before capturing a probe");
          lc::settle_size(c.h);
        }
        unsigned char* base = static_cast<unsigned char*>(scratch_address(c.h->device));
        lc::probe_external_scratch(c.h, c.Q, c.B, c.oi, c.ol, c.od, reinterpret_cast<float*>(base + L.qpad),
                                   reinterpret_cast<float*>(base + L.kappa),
                                   reinterpret_cast<unsigned long long*>(base + L.best),
                                   reinterpret_cast<cudaStream_t>(c.s));
      },
      &ctx);
}
