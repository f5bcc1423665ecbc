// Allocation-free variant of the predicate + order-preserving compaction.
//
// Some callers cannot allocate device memory at the time they run a filter:
// a database worker that is handed a fixed device arena and must not grow
// the process's footprint, an operator called from inside another engine's
// allocation-free execution loop, or a latency-bound path that cannot afford
// cudaMalloc's implicit device-wide synchronisation or its failure under
// memory pressure.  aiq_filter_compact_static gives them the same kernels as
// the query path (predicate bitmask, tile-count scan, compaction), with their
// scratch (bitmask, tile counts, tile offsets) held in one file-scope device
// array instead of a context's workspace.
//
// The array is a global of this shared library: every GPU that loads the
// library keeps kStaticScratchBytes reserved on it until the process exits.
// Host code cannot pass `g_filter_scratch` itself to a kernel (in host code
// that name is a host-side shadow, not a device address): the device address
// is obtained once per device with cudaGetSymbolAddress, with that device
// current, on the first call made on that device, and cached.  A
// cudaDeviceReset in this process invalidates the cached address; the cache
// is not refreshed, so a process that resets a device must not call this
// entry point on it afterwards.
#include <mutex>
#include <string>

#include "aiq.h"
#include "aiq_ops.h"
#include "common.cuh"
#include "kernels.h"

namespace {

using namespace aiq;

constexpr int64_t kStaticMaxRows = int64_t(1) << 24;                     // 16,777,216 rows
constexpr int64_t kStaticTiles = kStaticMaxRows / kRowsPerBlock;         // 8192 tiles
constexpr size_t kBitsBytes = kStaticMaxRows / 8;                        // 2 MiB bitmask
constexpr size_t kCountBytes = kStaticTiles * sizeof(int32_t);          // 32 KiB tile counts
constexpr size_t kOffsetBytes = (kStaticTiles + 1) * sizeof(int64_t);   // 64 KiB + 8 tile offsets
constexpr size_t kOffsetAt = kBitsBytes + kCountBytes;
constexpr size_t kStaticScratchBytes = ((kOffsetAt + kOffsetBytes + 255) / 256) * 256;

static __device__ __align__(256) unsigned char g_filter_scratch[kStaticScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_setup_mu;
void* g_scratch_dev[kMaxDevices] = {};

// Failures are reported through aiq_last_error(), like every other entry point.
aiq_status static_fail(aiq_status s, const char* msg, cudaError_t e = cudaSuccess) {
  std::string m = msg;
  if (e != cudaSuccess) {
    m += ": ";
    m += cudaGetErrorString(e);
  }
  aiq::set_error_message(m.c_str());
  return s;
}

// Device address of the scratch array on the current device (set up once).
aiq_status scratch_for_current_device(unsigned char** out) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return static_fail(AIQ_ERR_CUDA, "cudaGetDevice", e);
  if (dev < 0 || dev >= kMaxDevices) return static_fail(AIQ_ERR_UNSUPPORTED, "device index above 63");
  std::lock_guard<std::mutex> lock(g_setup_mu);
  if (!g_scratch_dev[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_filter_scratch);
    if (e != cudaSuccess || !p) return static_fail(AIQ_ERR_CUDA, "cudaGetSymbolAddress(g_filter_scratch)", e);
    g_scratch_dev[dev] = p;
  }
  *out = static_cast<unsigned char*>(g_scratch_dev[dev]);
  return AIQ_OK;
}

__global__ void k_copy_count(const int64_t* src, int64_t* dst) { *dst = *src; }

}  // namespace

extern "C" {

aiq_status aiq_filter_compact_static(const aiq_term* terms, int32_t n_terms, int64_t n_rows, int32_t* ids_out,
                                     int64_t* count_out, void* stream) {
  if (n_terms < 0 || n_terms > kMaxPreds || (n_terms > 0 && !terms))
    return static_fail(AIQ_ERR_INVALID_ARG, "n_terms must be 0..8 with a term array");
  if (n_rows < 0) return static_fail(AIQ_ERR_INVALID_ARG, "n_rows must be >= 0");
  if (n_rows > kStaticMaxRows)
    return static_fail(AIQ_ERR_CAPACITY, "aiq_filter_compact_static handles at most 16,777,216 rows per call");
  if (!count_out || (n_rows > 0 && !ids_out)) return static_fail(AIQ_ERR_INVALID_ARG, "ids_out/count_out is NULL");
  PredSet ps{};
  ps.n = n_terms;
  for (int i = 0; i < n_terms; ++i) {
    const aiq_term& t = terms[i];
    if (!t.column && n_rows > 0) return static_fail(AIQ_ERR_INVALID_ARG, "a term's column is NULL");
    if (t.type < AIQ_INT32 || t.type > AIQ_FLOAT32) return static_fail(AIQ_ERR_INVALID_ARG, "term type must be INT32, INT64 or FLOAT32");
    if (t.op < AIQ_LT || t.op > AIQ_NE) return static_fail(AIQ_ERR_INVALID_ARG, "unknown comparison operator");
    if (reinterpret_cast<uintptr_t>(t.column) & 15) return static_fail(AIQ_ERR_INVALID_ARG, "columns must be 16-byte aligned");
    ps.p[i] = PredDev{t.column, t.type, t.op, t.ivalue, t.fvalue};
  }
  unsigned char* scratch = nullptr;
  aiq_status st = scratch_for_current_device(&scratch);
  if (st != AIQ_OK) return st;
  uint32_t* bits = reinterpret_cast<uint32_t*>(scratch);
  int32_t* counts = reinterpret_cast<int32_t*>(scratch + kBitsBytes);
  int64_t* offsets = reinterpret_cast<int64_t*>(scratch + kOffsetAt);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int64_t tiles = (n_rows + kRowsPerBlock - 1) / kRowsPerBlock;
  // Every scratch word the compaction reads is written earlier in this call
  // (each tile writes its whole bitmask slice and its count; the scan writes
  // offsets[0..tiles]), so nothing is carried over from the previous call.
  launch_predicate_mask(ps, ProbeSpec{}, n_rows, bits, counts, nullptr, s);
  launch_scan_counts(counts, tiles, offsets, s);
  launch_compact(bits, offsets, n_rows, ids_out, nullptr, nullptr, s);
  k_copy_count<<<1, 1, 0, s>>>(offsets + tiles, count_out);
  // A failed predicate launch is recorded (and its CUDA error consumed) by its
  // launcher; take that record here so that it is reported by this call and
  // not left behind for the next call on this host thread.
  const char* what = nullptr;
  const cudaError_t le = take_launch_error(&what);
  const cudaError_t e = cudaGetLastError();
  if (le != cudaSuccess) return static_fail(AIQ_ERR_CUDA, what, le);
  if (e != cudaSuccess) return static_fail(AIQ_ERR_CUDA, "kernel launch", e);
  return AIQ_OK;
}

}  // extern "C"
