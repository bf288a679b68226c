// Allocation-free decode attention (kvpop_attend_noalloc in include/kvpop.h).
//
// Some callers cannot allocate device memory at the point where they run the
// decode step: a serving loop whose device memory is planned up front and must
// not grow or synchronise mid-generation, or a plugin that runs inside a host
// framework and may only use the buffers that framework hands it.  For them
// this entry point runs the CUDA-core decode-attention kernel over K/V buffers
// the caller owns, with the kernel's split-K scratch (per-CTA partials and
// per-(sequence, head) counters) in the fixed array below instead of memory
// from cudaMalloc.  Nothing here calls cudaMalloc, cudaFree or any routine
// that allocates.
//
// The array lives in every GPU that loads the library until the process exits.
// All calls on a device share it and it keeps the last call's contents, so
// calls that overlap on the GPU (different streams, or different threads
// without ordering) race on it; callers must serialise them.
//
// A bounded wait inside the kernel that gives up is recorded in the library's
// device error word of the cache-free calls, which kvpop_standalone_status reads
// and clears (that word is a __device__ variable too: reading it allocates
// nothing).
#include <mutex>

#include "kvpop_internal.cuh"

namespace kvpop {
void note_error(const char* msg);
int32_t* standalone_err_word();
}

using namespace kvpop;

namespace {

constexpr size_t kScratchBytes = 2u << 20;    // 2 MiB
static __device__ __align__(256) unsigned char g_attend_scratch[kScratchBytes];

constexpr int kMaxDevices = 64;
constexpr int kMaxPairs = 12288;

struct DeviceSetup {
  bool ready = false;
  unsigned char* scratch = nullptr;   // device address of g_attend_scratch
  int32_t* err = nullptr;             // device address of the cache-free calls' error word
  int sms = 0;
  int smem_optin = 0;
};
DeviceSetup g_setup[kMaxDevices];
std::mutex g_setup_mu;

// First use on a device, with that device current: resolve the device
// addresses of the array and of the error word, and allow the attention
// kernels their dynamic shared memory.
kvpop_status setup_device(int dev, DeviceSetup** out) {
  std::lock_guard<std::mutex> lock(g_setup_mu);
  DeviceSetup& s = g_setup[dev];
  if (!s.ready) {
    void* ptr = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&ptr, g_attend_scratch);
    if (e != cudaSuccess) {
      note_error("kvpop_attend_noalloc: cudaGetSymbolAddress of the scratch array failed");
      return KVPOP_ERR_CUDA;
    }
    int32_t* err = standalone_err_word();
    if (!err) {
      note_error("kvpop_attend_noalloc: cudaGetSymbolAddress of the error word failed");
      return KVPOP_ERR_CUDA;
    }
    int sms = 0, optin = 0;
    e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    for (int dt = 0; dt < 2 && e == cudaSuccess; ++dt)
      for (int d : {64, 128})
        for (int G : {1, 2, 4}) {
          Dims dm{};
          dm.dtype = dt;
          dm.d = d;
          dm.G = G;
          AttendConfig ac;
          if (e == cudaSuccess) e = attend_config(dm, &ac);
          if (e == cudaSuccess) e = raise_smem_limit(ac.func, 0);
        }
    if (e != cudaSuccess) {
      note_error("kvpop_attend_noalloc: device set-up failed");
      return KVPOP_ERR_CUDA;
    }
    s.scratch = static_cast<unsigned char*>(ptr);
    s.err = err;
    s.sms = sms;
    s.smem_optin = optin;
    s.ready = true;
  }
  *out = &s;
  return KVPOP_OK;
}

bool al16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
bool al4(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 3u) == 0; }

}  // namespace

extern "C" kvpop_status kvpop_attend_noalloc(const void* slotK, const void* slotV, const void* ringK,
                                             const void* ringV, const int32_t* nvalid,
                                             const int32_t* len, const void* q, float* out,
                                             int32_t batch, int32_t n_kv_heads, int32_t q_per_kv,
                                             int32_t head_dim, int32_t budget_B, int32_t delay_D,
                                             kvpop_dtype kv_dtype, cudaStream_t stream) {
  if (!slotK || !slotV || !ringK || !ringV || !nvalid || !len || !q || !out)
    return KVPOP_ERR_INVALID_ARG;
  if (batch < 1 || n_kv_heads < 1 || (q_per_kv != 1 && q_per_kv != 2 && q_per_kv != 4) ||
      (head_dim != 64 && head_dim != 128) || budget_B < 1 || delay_D < 1 ||
      (kv_dtype != KVPOP_F32 && kv_dtype != KVPOP_BF16))
    return KVPOP_ERR_INVALID_ARG;
  const long long pairs = (long long)batch * n_kv_heads;
  if (pairs > kMaxPairs) {
    note_error("kvpop_attend_noalloc: batch * n_kv_heads exceeds 12288");
    return KVPOP_ERR_INVALID_ARG;
  }
  if (!al16(slotK) || !al16(slotV) || !al16(ringK) || !al16(ringV) || !al16(q) || !al16(out) ||
      !al4(nvalid) || !al4(len))
    return KVPOP_ERR_ALIGN;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return KVPOP_ERR_CUDA;
  DeviceSetup* ds = nullptr;
  kvpop_status st = setup_device(dev, &ds);
  if (st != KVPOP_OK) return st;

  Dims dm{};
  dm.batch = batch; dm.H = n_kv_heads; dm.G = q_per_kv; dm.d = head_dim;
  dm.B = budget_B; dm.D = delay_D; dm.dtype = kv_dtype; dm.pairs = (int)pairs;
  AttendConfig ac;
  if (attend_config(dm, &ac) != cudaSuccess) return KVPOP_ERR_INVALID_ARG;
  const size_t smem = ac.smem_fixed + (size_t)(pairs + 1) * 4;
  if (smem > (size_t)ds->smem_optin) {
    note_error("kvpop_attend_noalloc: too many (sequence, head) pairs for the kernel's shared memory");
    return KVPOP_ERR_INVALID_ARG;
  }
  const int grid = ds->sms;                       // one CTA per SM (the kernel's launch bounds)
  const size_t count_bytes = ((size_t)pairs * 4 + 255) & ~size_t(255);
  const size_t part_bytes = (size_t)2 * grid * (q_per_kv * head_dim + 2 * q_per_kv) * 4;
  if (count_bytes + part_bytes > kScratchBytes) {
    note_error("kvpop_attend_noalloc: split-K scratch would exceed the fixed 2 MiB array");
    return KVPOP_ERR_INVALID_ARG;
  }

  State s{};
  s.slotK = const_cast<void*>(slotK);
  s.slotV = const_cast<void*>(slotV);
  s.ringK = const_cast<void*>(ringK);
  s.ringV = const_cast<void*>(ringV);
  s.nvalid = const_cast<int32_t*>(nvalid);
  s.len = const_cast<int32_t*>(len);
  s.part_count = reinterpret_cast<int32_t*>(ds->scratch);
  s.part = reinterpret_cast<float*>(ds->scratch + count_bytes);
  s.err = ds->err;     // first error wins; kvpop_standalone_status reads and clears it
  // the counters must start at zero; the array keeps whatever the last call left
  cudaError_t e = cudaMemsetAsync(s.part_count, 0, count_bytes, stream);
  if (e == cudaSuccess) e = launch_attend(s, dm, q, out, grid, stream);
  if (e != cudaSuccess) {
    note_error("kvpop_attend_noalloc: launch failed");
    return KVPOP_ERR_CUDA;
  }
  return KVPOP_OK;
}
