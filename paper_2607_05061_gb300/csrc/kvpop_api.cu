// Host side of the C ABI declared in include/kvpop.h: argument checks, device
// memory, kernel launches.  No call throws or aborts; every failure is a status.
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <new>
#include <vector>

#include "kvpop_argmin.cuh"

using namespace kvpop;

namespace kvpop {
cudaError_t prepare_ingest(const Dims& dm);
cudaError_t prepare_prefill(const Dims& dm);
}

struct kvpop_cache {
  kvpop_config cfg;
  Dims dm;
  State st;
  int device = 0;
  int attend_grid = 0;
  size_t esz = 0;
  bool poisoned = false;
  bool has_decay = false;
  std::vector<void*> allocs;
  std::vector<unsigned char> tc_maps;   // TMA descriptors of the K/V stores (bf16 path)
  bool use_tc = false;
  bool use_fused = false;               // kvpop_decode_step as one kernel (bf16, d = 128)
  FusedBufs fb{};
  int fused_grid = 0;
  bool use_cluster = false;             // cluster ingest kernel
  float* W1s = nullptr;                 // slice-major scorer weights for it
  float* b1s = nullptr;
  float* w2s = nullptr;
  float* w1t = nullptr;                 // W1^T split for the tensor-core prompt scorer
  std::vector<unsigned char> sc_maps;   // its TMA descriptors
  bool use_tf32 = false;
  bool mlstm = false;                   // stateful mLSTM scorer instead of the MLP
  MlstmDev md{};
  // staging for kvpop_decode_step_host
  void* stage_q = nullptr;
  void* stage_k = nullptr;
  void* stage_v = nullptr;
  float* stage_out = nullptr;
  uint64_t magic = 0;
};

// First device-side error of the cache-free calls (prompt attention, causal LSE,
// future target, allocation-free attention); read and cleared by
// kvpop_standalone_status.
__device__ int32_t g_standalone_err[4];

namespace kvpop {
extern int g_debug_skip_copies;   // kvpop_attend_tc.cu
// Device address of g_standalone_err on the current device (NULL on failure).
int32_t* standalone_err_word() {
  void* p = nullptr;
  return cudaGetSymbolAddress(&p, g_standalone_err) == cudaSuccess ? static_cast<int32_t*>(p) : nullptr;
}
}  // namespace kvpop

namespace {

int32_t* standalone_err() { return kvpop::standalone_err_word(); }

constexpr uint64_t kMagic = 0x6b7670'6f70'6361ull;   // "kvpopca"
// K/V bytes per step from which kvpop_decode_step runs as one kernel: the attention then
// takes at least ~90 us, about what the scorer units need beside it on the GPU.
constexpr double kFusedMinStepBytes = 600e6;
constexpr uint64_t kStateVersion = 1;
int g_fail_after = 0;
thread_local char g_last_error[256] = "";

// Record the failing call (file-local line) for kvpop_last_error().
cudaError_t note(cudaError_t e, int line) {
  if (e != cudaSuccess)
    std::snprintf(g_last_error, sizeof(g_last_error), "kvpop_api.cu:%d: %s (%s)", line,
                  cudaGetErrorName(e), cudaGetErrorString(e));
  return e;
}
#define NOTE(expr) note((expr), __LINE__)

kvpop_status from_cuda(cudaError_t e) {
  if (e == cudaSuccess) return KVPOP_OK;
  if (e == cudaErrorMemoryAllocation) return KVPOP_ERR_OOM;
  return KVPOP_ERR_CUDA;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
bool aligned4(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 3u) == 0; }

// Device address of pinned host memory the device can address in place (NVLink-C2C /
// PCIe mapping) and 16-byte aligned there; NULL for anything else.
const void* mapped_host(const void* p) {
  cudaPointerAttributes pa{};
  const void* d = nullptr;
  if (cudaPointerGetAttributes(&pa, p) == cudaSuccess && pa.type == cudaMemoryTypeHost &&
      pa.devicePointer != nullptr && aligned16(pa.devicePointer))
    d = pa.devicePointer;
  cudaGetLastError();   // a pointer the runtime does not know is not an error here
  return d;
}

kvpop_status dev_alloc(kvpop_cache* c, void** p, size_t bytes) {
  *p = nullptr;
  if (g_fail_after > 0 && --g_fail_after == 0) return KVPOP_ERR_OOM;
  if (bytes == 0) bytes = 16;
  cudaError_t e = NOTE(cudaMalloc(p, bytes));
  if (e != cudaSuccess) {
    cudaGetLastError();   // clear the sticky-free allocation error
    *p = nullptr;
    return from_cuda(e);
  }
  try {
    c->allocs.push_back(*p);
  } catch (...) {                 // host out of memory: no exception crosses the ABI
    cudaFree(*p);
    *p = nullptr;
    return KVPOP_ERR_OOM;
  }
  return KVPOP_OK;
}

// v = n zero bytes; false when the host allocation fails
bool assign_zero(std::vector<unsigned char>& v, size_t n) {
  try {
    v.assign(n, 0);
  } catch (...) {
    return false;
  }
  return true;
}

void release(kvpop_cache* c) {
  for (void* p : c->allocs) cudaFree(p);
  c->allocs.clear();
}

// 64-byte aligned view of the stored TMA descriptors.
void* tc_map_ptr(kvpop_cache* c) {
  uintptr_t p = reinterpret_cast<uintptr_t>(c->tc_maps.data());
  return reinterpret_cast<void*>((p + 63) & ~uintptr_t(63));
}
void* sc_map_ptr(kvpop_cache* c) {
  if (!c->use_tf32) return nullptr;
  uintptr_t p = reinterpret_cast<uintptr_t>(c->sc_maps.data());
  return reinterpret_cast<void*>((p + 63) & ~uintptr_t(63));
}

kvpop_status validate(const kvpop_config* cfg) {
  if (!cfg) return KVPOP_ERR_INVALID_ARG;
  if (cfg->batch < 1 || cfg->n_kv_heads < 1) return KVPOP_ERR_INVALID_ARG;
  if (cfg->q_per_kv != 1 && cfg->q_per_kv != 2 && cfg->q_per_kv != 4) return KVPOP_ERR_INVALID_ARG;
  if (cfg->head_dim != 64 && cfg->head_dim != 128) return KVPOP_ERR_INVALID_ARG;
  if (cfg->budget_B < 1 || cfg->delay_D < 1) return KVPOP_ERR_INVALID_ARG;
  if (cfg->n_sink < 0 || cfg->n_sink >= cfg->budget_B) return KVPOP_ERR_INVALID_ARG;
  if (cfg->scorer_hidden < 1 || cfg->scorer_hidden > 1024) return KVPOP_ERR_INVALID_ARG;
  if (cfg->kv_dtype != KVPOP_F32 && cfg->kv_dtype != KVPOP_BF16) return KVPOP_ERR_INVALID_ARG;
  const long long pairs = (long long)cfg->batch * cfg->n_kv_heads;
  if (pairs > 12288) return KVPOP_ERR_INVALID_ARG;             // attention schedule in smem
  if ((long long)cfg->budget_B * pairs > (1ll << 40)) return KVPOP_ERR_INVALID_ARG;
  return KVPOP_OK;
}

kvpop_status usable(kvpop_cache* c) {
  if (!c || c->magic != kMagic) return KVPOP_ERR_INVALID_ARG;
  if (c->poisoned) return KVPOP_ERR_STATE;
  return KVPOP_OK;
}

kvpop_status poison_on(kvpop_cache* c, cudaError_t e) {
  if (e == cudaSuccess) return KVPOP_OK;
  c->poisoned = true;
  return from_cuda(e);
}

struct StateBuf {
  void* ptr;
  size_t bytes;
};
// The cache's state buffers in a fixed order (the checkpoint format); no allocation.
struct StateList {
  static constexpr int kMax = 24;     // 16 in use (13 + 3 for the mLSTM state)
  StateBuf b[kMax];
  int n = 0;
  void add(void* ptr, size_t bytes) {
    if (n < kMax) b[n++] = {ptr, bytes};
  }
  const StateBuf* begin() const { return b; }
  const StateBuf* end() const { return b + n; }
};

StateList all_state_buffers(kvpop_cache* c) {
  const Dims& dm = c->dm;
  const size_t pairs = dm.pairs;
  StateList v;
  v.add(c->st.slotK, pairs * dm.B * dm.d * c->esz);
  v.add(c->st.slotV, pairs * dm.B * dm.d * c->esz);
  v.add(c->st.ringK, pairs * dm.D * dm.d * c->esz);
  v.add(c->st.ringV, pairs * dm.D * dm.d * c->esz);
  v.add(c->st.ringQm, pairs * dm.D * dm.d * 4);
  v.add(c->st.score, pairs * dm.B * 4);
  v.add(c->st.pos, pairs * dm.B * 4);
  v.add(c->st.nvalid, pairs * 4);
  v.add(c->st.len, pairs * 4);
  v.add(c->st.min_score, pairs * 4);
  v.add(c->st.min_slot, pairs * 4);
  v.add(c->st.blk_score, pairs * min_blocks(dm.B) * 4);
  v.add(c->st.blk_slot, pairs * min_blocks(dm.B) * 4);
  if (c->mlstm) {
    const size_t d = dm.d;
    v.add(c->md.C, pairs * d * (d / 2) * 4);
    v.add(c->md.z, pairs * d * 4);
    v.add(c->md.m, pairs * 4);
  }
  return v;
}

}  // namespace

namespace kvpop {
// Message for kvpop_last_error() from other translation units of the library.
void note_error(const char* msg) { std::snprintf(g_last_error, sizeof(g_last_error), "%s", msg); }
}

extern "C" {

const char* kvpop_status_string(kvpop_status s) {
  switch (s) {
    case KVPOP_OK: return "ok";
    case KVPOP_ERR_INVALID_ARG: return "invalid argument";
    case KVPOP_ERR_ALIGN: return "device pointer not 16-byte aligned";
    case KVPOP_ERR_OOM: return "device allocation failed";
    case KVPOP_ERR_CUDA: return "CUDA runtime error";
    case KVPOP_ERR_STATE: return "cache unusable after an earlier error";
    case KVPOP_ERR_DEVICE_CHECK: return "device-side check failed";
  }
  return "unknown status";
}

void kvpop_debug_fail_alloc_after(int32_t n) { g_fail_after = n > 0 ? n : 0; }

void kvpop_debug_skip_attention_copies(int32_t on) { kvpop::g_debug_skip_copies = on ? 1 : 0; }

const char* kvpop_last_error(void) { return g_last_error; }

static kvpop_status init_cache(const kvpop_config* cfg_in, const kvpop_scorer* sc,
                               const kvpop_mlstm_scorer* ms, cudaStream_t stream, kvpop_cache** out) {
  if (!out) return KVPOP_ERR_INVALID_ARG;
  *out = nullptr;
  if (!cfg_in) return KVPOP_ERR_INVALID_ARG;
  kvpop_config cfgv = *cfg_in;
  if (ms) cfgv.scorer_hidden = 4;            // unused by the mLSTM scorer
  const kvpop_config* cfg = &cfgv;
  kvpop_status vs = validate(cfg);
  if (vs != KVPOP_OK) return vs;
  if (sc && (!sc->W1 || !sc->b1 || !sc->w2 || !sc->b2)) return KVPOP_ERR_INVALID_ARG;
  if (sc && (sc->input_kind < 0 || sc->input_kind > 1 || sc->activation < 0 || sc->activation > 2))
    return KVPOP_ERR_INVALID_ARG;
  if (ms && (!ms->Wq || !ms->Wk || !ms->Wv || !ms->wi || !ms->wf || !ms->bi || !ms->bf || !ms->a ||
             !ms->b))
    return KVPOP_ERR_INVALID_ARG;
  if (!sc && !ms) return KVPOP_ERR_INVALID_ARG;

  kvpop_cache* c = new (std::nothrow) kvpop_cache();
  if (!c) return KVPOP_ERR_OOM;
  c->cfg = *cfg;
  Dims& dm = c->dm;
  dm.batch = cfg->batch; dm.H = cfg->n_kv_heads; dm.G = cfg->q_per_kv; dm.d = cfg->head_dim;
  dm.B = cfg->budget_B; dm.D = cfg->delay_D; dm.s = cfg->n_sink; dm.F = cfg->scorer_hidden;
  dm.Fp = (dm.F + 3) & ~3;
  dm.act = sc ? sc->activation : 0;
  dm.dtype = cfg->kv_dtype;
  dm.pairs = dm.batch * dm.H;
  c->esz = cfg->kv_dtype == KVPOP_F32 ? 4 : 2;
  c->magic = kMagic;
  c->mlstm = ms != nullptr;
  if (c->mlstm && !mlstm_ok(dm)) { delete c; return KVPOP_ERR_INVALID_ARG; }
  NOTE(cudaGetDevice(&c->device));

  const size_t pairs = dm.pairs, B = dm.B, D = dm.D, d = dm.d, H = dm.H, F = dm.F, Fp = dm.Fp;
  const size_t NB = min_blocks(dm.B);
  const size_t I = 3 * d;                              // device rows of W1: [k; v; qbar]
  const size_t Isrc = (sc && sc->input_kind == 1) ? 2 * d : I;   // rows the caller gives
  AttendConfig ac;
  c->use_tc = cfg->kv_dtype == KVPOP_BF16;
  kvpop_status s = from_cuda(NOTE(c->use_tc ? tc_config(dm, &ac) : attend_config(dm, &ac)));
  void* p = nullptr;
#define ALLOC(field, type, bytes)                        \
  if (s == KVPOP_OK) {                                   \
    s = dev_alloc(c, &p, (bytes));                       \
    c->st.field = static_cast<type>(p);                  \
  }
  ALLOC(slotK, void*, pairs * B * d * c->esz)
  ALLOC(slotV, void*, pairs * B * d * c->esz)
  ALLOC(ringK, void*, pairs * D * d * c->esz)
  ALLOC(ringV, void*, pairs * D * d * c->esz)
  ALLOC(ringQm, float*, pairs * D * d * 4)
  ALLOC(score, float*, pairs * B * 4)
  ALLOC(pos, int32_t*, pairs * B * 4)
  ALLOC(nvalid, int32_t*, pairs * 4)
  ALLOC(len, int32_t*, pairs * 4)
  ALLOC(min_score, float*, pairs * 4)
  ALLOC(min_slot, int32_t*, pairs * 4)
  ALLOC(blk_score, float*, pairs * NB * 4)
  ALLOC(blk_slot, int32_t*, pairs * NB * 4)
  float* w = nullptr;
  const size_t wbytes = (H * I * Fp + 2 * H * Fp + 2 * H) * 4;
  if (s == KVPOP_OK) { s = dev_alloc(c, &p, wbytes); w = (float*)p; }
  ALLOC(part_count, int32_t*, pairs * 4)
  ALLOC(err, int32_t*, 16 * 4)
  int sms = 0, occ = 0;
  if (s == KVPOP_OK) {
    s = from_cuda(NOTE(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, c->device)));
    const size_t smem = ac.smem_fixed + (pairs + 1) * 4;
    if (s == KVPOP_OK)
      s = from_cuda(NOTE(raise_smem_limit(ac.func, smem)));
    if (s == KVPOP_OK)
      s = from_cuda(NOTE(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, ac.func, ac.threads, smem)));
    if (s == KVPOP_OK && occ < 1) s = KVPOP_ERR_INVALID_ARG;
    c->attend_grid = sms * (occ > 0 ? occ : 1);
  }
  // the one-kernel decode step, where its shape and shared memory allow it and the K/V
  // stream of a step is long enough to hide the scorer behind it (otherwise
  // kvpop_decode_step runs the ingest and the attention as two kernels)
  AttendConfig fc;
  const double step_kv_bytes = (double)pairs * (double)(B + D) * 2.0 * (double)d * (double)c->esz;
  const bool want_fused = std::getenv("KVPOP_SPLIT_STEP") == nullptr &&
                          (std::getenv("KVPOP_FUSED_STEP") != nullptr || step_kv_bytes >= kFusedMinStepBytes);
  if (s == KVPOP_OK && c->use_tc && !c->mlstm && want_fused && tc_fused_ok(dm) &&
      tc_fused_config(dm, &fc) == cudaSuccess) {
    const size_t smem = fc.smem_fixed + (pairs + 1) * 4;
    int occ_f = 0;
    if (raise_smem_limit(fc.func, smem) == cudaSuccess &&
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ_f, fc.func, fc.threads, smem) == cudaSuccess &&
        occ_f >= 1 && sms * occ_f <= tc_fused_max_grid()) {
      c->use_fused = true;
      c->fused_grid = sms * occ_f;
    }
    cudaGetLastError();   // a refused shared-memory size only disables the fused step
  }
  const size_t part_grid = c->fused_grid > c->attend_grid ? c->fused_grid : c->attend_grid;
  ALLOC(part, float*, (size_t)2 * part_grid * (dm.G * d + 2 * dm.G) * 4)
  if (s == KVPOP_OK && c->use_fused) {
    s = dev_alloc(c, &p, pairs * (dm.G * d + 2 * dm.G) * 4);
    c->fb.part_c = static_cast<float*>(p);
    if (s == KVPOP_OK) { s = dev_alloc(c, &p, pairs * 4 * 4); c->fb.meta_next = (int32_t*)p; }
    if (s == KVPOP_OK) { s = dev_alloc(c, &p, pairs * (2 * dm.G + 2 * d) * 4); c->fb.xtra = (float*)p; }
    if (s == KVPOP_OK) { s = dev_alloc(c, &p, 16); c->fb.ctr = static_cast<unsigned long long*>(p); }
    if (s == KVPOP_OK) {
      s = dev_alloc(c, &p, (size_t)c->fused_grid * sizeof(int2));
      c->fb.start_prev = static_cast<int2*>(p);
    }
  }
#undef ALLOC
  // q | k | v staging in one block, so that adjacent host buffers take a single copy
  if (s == KVPOP_OK) {
    s = dev_alloc(c, &p, pairs * (dm.G + 2) * d * c->esz);
    c->stage_q = p;
    c->stage_k = static_cast<char*>(p) + pairs * dm.G * d * c->esz;
    c->stage_v = static_cast<char*>(c->stage_k) + pairs * d * c->esz;
  }
  if (s == KVPOP_OK) { s = dev_alloc(c, &p, pairs * dm.G * d * 4); c->stage_out = (float*)p; }
  if (s == KVPOP_OK && c->use_tc) {
    s = assign_zero(c->tc_maps, tc_maps_size() + 64) ? from_cuda(NOTE(tc_make_maps(c->st, dm, tc_map_ptr(c))))
                                                     : KVPOP_ERR_OOM;
  }
  if (s == KVPOP_OK) s = from_cuda(NOTE(prepare_ingest(dm)));
  const size_t hh = d / 2, NCm = mlstm_nc(dm.d);
  if (s == KVPOP_OK && c->mlstm) {
    MlstmDev& md = c->md;
    md.NC = (int)NCm;
    s = dev_alloc(c, &p, pairs * d * hh * 4); md.C = (float*)p;
    if (s == KVPOP_OK) { s = dev_alloc(c, &p, pairs * d * 4); md.z = (float*)p; }
    if (s == KVPOP_OK) { s = dev_alloc(c, &p, pairs * 4); md.m = (float*)p; }
    if (s == KVPOP_OK) { s = dev_alloc(c, &p, H * 2 * d * NCm * 4); md.Wcat = (float*)p; }
    if (s == KVPOP_OK) { s = dev_alloc(c, &p, (4 * H + H * hh) * 4); md.bi = (float*)p; }
    if (s == KVPOP_OK) {
      md.bf = md.bi + H; md.b = md.bf + H; md.a = md.b + H;
      s = from_cuda(NOTE(prepare_mlstm(dm)));
    }
  }
  c->use_cluster = !c->mlstm && cluster_ingest_ok(dm);
  const size_t FS = cluster_ingest_fs(dm);
  if (s == KVPOP_OK && c->use_cluster) {
    s = dev_alloc(c, &p, (H * 8 * I * FS + 2 * H * 8 * FS) * 4);
    c->W1s = (float*)p;
    c->b1s = c->W1s + H * 8 * I * FS;
    c->w2s = c->b1s + H * 8 * FS;
    if (s == KVPOP_OK) s = from_cuda(NOTE(prepare_ingest_cluster(dm)));
  }
  if (s == KVPOP_OK) s = from_cuda(NOTE(prepare_prefill(dm)));
  c->use_tf32 = !c->mlstm && score_tf32_ok(dm) && std::getenv("KVPOP_PROMPT_SCORER_SIMT") == nullptr;
  if (s == KVPOP_OK && c->use_tf32) {
    s = dev_alloc(c, &p, 2 * H * dm.F * I * 4);
    c->w1t = (float*)p;
    if (s == KVPOP_OK && !assign_zero(c->sc_maps, score_tf32_maps_size() + 64)) s = KVPOP_ERR_OOM;
  }
  if (s == KVPOP_OK) {
    float* W1 = w;
    float* b1 = W1 + H * I * Fp;
    float* w2 = b1 + H * Fp;
    float* b2 = w2 + H * Fp;
    float* lg = b2 + H;
    c->st.W1 = W1; c->st.b1 = b1; c->st.w2 = w2; c->st.b2 = b2;
    // hidden units padded to Fp with zero weights: rows of F floats into rows of Fp
    cudaError_t e = NOTE(cudaMemsetAsync(w, 0, wbytes, stream));
    // a [k; v]-only scorer keeps zero weights on the qbar rows
    for (size_t h = 0; h < H && e == cudaSuccess && sc; ++h)
      e = NOTE(cudaMemcpy2DAsync(W1 + h * I * Fp, Fp * 4, sc->W1 + h * Isrc * F, F * 4, F * 4, Isrc,
                                 cudaMemcpyDefault, stream));
    if (e == cudaSuccess && sc)
      e = NOTE(cudaMemcpy2DAsync(b1, Fp * 4, sc->b1, F * 4, F * 4, H, cudaMemcpyDefault, stream));
    if (e == cudaSuccess && sc)
      e = NOTE(cudaMemcpy2DAsync(w2, Fp * 4, sc->w2, F * 4, F * 4, H, cudaMemcpyDefault, stream));
    if (e == cudaSuccess && sc) e = NOTE(cudaMemcpyAsync(b2, sc->b2, H * 4, cudaMemcpyDefault, stream));
    if (e == cudaSuccess && c->use_tf32) e = NOTE(prepare_score_tf32(dm, W1, c->w1t, sc_map_ptr(c), stream));
    if (e == cudaSuccess && c->use_fused) e = NOTE(cudaMemsetAsync(c->fb.ctr, 0, 16, stream));
    if (e == cudaSuccess && c->use_fused)
      e = NOTE(cudaMemsetAsync(c->fb.start_prev, 0, (size_t)c->fused_grid * sizeof(int2), stream));
    std::vector<float> minus_inf;
    if (c->mlstm) {
      // mLSTM weights: column blocks of Wcat [2d][NC] = [W_k | W_v | W_q | w_i | w_f | 0]
      MlstmDev& md = c->md;
      const size_t n2 = 2 * d;
      if (e == cudaSuccess) e = NOTE(cudaMemsetAsync(md.Wcat, 0, H * n2 * NCm * 4, stream));
      const float* blocks[3] = {ms->Wk, ms->Wv, ms->Wq};
      for (size_t h = 0; h < H && e == cudaSuccess; ++h) {
        float* dst = md.Wcat + h * n2 * NCm;
        for (int bidx = 0; bidx < 3 && e == cudaSuccess; ++bidx)
          e = NOTE(cudaMemcpy2DAsync(dst + bidx * hh, NCm * 4, blocks[bidx] + h * n2 * hh, hh * 4,
                                     hh * 4, n2, cudaMemcpyDefault, stream));
        if (e == cudaSuccess)
          e = NOTE(cudaMemcpy2DAsync(dst + 3 * hh, NCm * 4, ms->wi + h * n2, 4, 4, n2,
                                     cudaMemcpyDefault, stream));
        if (e == cudaSuccess)
          e = NOTE(cudaMemcpy2DAsync(dst + 3 * hh + 1, NCm * 4, ms->wf + h * n2, 4, 4, n2,
                                     cudaMemcpyDefault, stream));
      }
      if (e == cudaSuccess) e = NOTE(cudaMemcpyAsync(md.bi, ms->bi, H * 4, cudaMemcpyDefault, stream));
      if (e == cudaSuccess) e = NOTE(cudaMemcpyAsync(md.bf, ms->bf, H * 4, cudaMemcpyDefault, stream));
      if (e == cudaSuccess) e = NOTE(cudaMemcpyAsync(md.b, ms->b, H * 4, cudaMemcpyDefault, stream));
      if (e == cudaSuccess) e = NOTE(cudaMemcpyAsync(md.a, ms->a, H * hh * 4, cudaMemcpyDefault, stream));
      if (e == cudaSuccess) e = NOTE(cudaMemsetAsync(md.C, 0, pairs * d * hh * 4, stream));
      if (e == cudaSuccess) e = NOTE(cudaMemsetAsync(md.z, 0, pairs * d * 4, stream));
      try {
        minus_inf.assign(pairs, -INFINITY);
      } catch (...) {
        if (e == cudaSuccess) e = cudaErrorMemoryAllocation;
      }
      if (e == cudaSuccess)
        e = NOTE(cudaMemcpyAsync(md.m, minus_inf.data(), pairs * 4, cudaMemcpyHostToDevice, stream));
    }
    if (c->use_cluster) {
      // slice-major copy for the cluster kernel: slice r holds hidden units [r*FS, r*FS + FS)
      const size_t nW = (H * 8 * I * FS + 2 * H * 8 * FS) * 4;
      if (e == cudaSuccess) e = NOTE(cudaMemsetAsync(c->W1s, 0, nW, stream));
      for (size_t h = 0; h < H && e == cudaSuccess; ++h)
        for (size_t r = 0; r < 8 && e == cudaSuccess; ++r) {
          const size_t f0 = r * FS;
          if (f0 >= F) break;
          const size_t wcols = (F - f0 < FS) ? F - f0 : FS;
          const size_t sl = h * 8 + r;
          e = NOTE(cudaMemcpy2DAsync(c->W1s + sl * I * FS, FS * 4, sc->W1 + h * Isrc * F + f0, F * 4,
                                     wcols * 4, Isrc, cudaMemcpyDefault, stream));
          if (e == cudaSuccess)
            e = NOTE(cudaMemcpyAsync(c->b1s + sl * FS, sc->b1 + h * F + f0, wcols * 4,
                                     cudaMemcpyDefault, stream));
          if (e == cudaSuccess)
            e = NOTE(cudaMemcpyAsync(c->w2s + sl * FS, sc->w2 + h * F + f0, wcols * 4,
                                     cudaMemcpyDefault, stream));
        }
    }
    const float* lg_src = sc ? sc->log_gamma : ms->log_gamma;
    if (e == cudaSuccess && lg_src) {
      e = NOTE(cudaMemcpyAsync(lg, lg_src, H * 4, cudaMemcpyDefault, stream));
      c->st.log_gamma = lg;
      c->has_decay = true;
    } else {
      c->st.log_gamma = nullptr;
    }
    if (e == cudaSuccess) e = NOTE(cudaMemsetAsync(c->st.nvalid, 0, pairs * 4, stream));
    if (e == cudaSuccess) e = NOTE(cudaMemsetAsync(c->st.len, 0, pairs * 4, stream));
    if (e == cudaSuccess) e = NOTE(cudaMemsetAsync(c->st.part_count, 0, pairs * 4, stream));
    if (e == cudaSuccess) e = NOTE(cudaMemsetAsync(c->st.err, 0, 16 * 4, stream));
    if (e == cudaSuccess) e = NOTE(cudaMemsetAsync(c->st.pos, 0xff, pairs * B * 4, stream));
    // zeroed K/V stores: rows past the used slots are read (with weight 0) by the
    // tensor-core attention tiles and must hold finite values
    if (e == cudaSuccess) e = NOTE(cudaMemsetAsync(c->st.slotK, 0, pairs * B * d * c->esz, stream));
    if (e == cudaSuccess) e = NOTE(cudaMemsetAsync(c->st.slotV, 0, pairs * B * d * c->esz, stream));
    if (e == cudaSuccess) e = NOTE(cudaMemsetAsync(c->st.ringK, 0, pairs * D * d * c->esz, stream));
    if (e == cudaSuccess) e = NOTE(cudaMemsetAsync(c->st.ringV, 0, pairs * D * d * c->esz, stream));
    if (e == cudaSuccess) e = NOTE(cudaStreamSynchronize(stream));
    s = from_cuda(e);
  }
  if (s != KVPOP_OK) {
    release(c);
    c->magic = 0;
    delete c;
    return s;
  }
  *out = c;
  return KVPOP_OK;
}

kvpop_status kvpop_init_cache(const kvpop_config* cfg, const kvpop_scorer* sc, cudaStream_t stream,
                              kvpop_cache** out) {
  if (!sc) {
    if (out) *out = nullptr;
    return KVPOP_ERR_INVALID_ARG;
  }
  return init_cache(cfg, sc, nullptr, stream, out);
}

kvpop_status kvpop_init_cache_mlstm(const kvpop_config* cfg, const kvpop_mlstm_scorer* ms,
                                    cudaStream_t stream, kvpop_cache** out) {
  if (!ms) {
    if (out) *out = nullptr;
    return KVPOP_ERR_INVALID_ARG;
  }
  return init_cache(cfg, nullptr, ms, stream, out);
}

kvpop_status kvpop_free(kvpop_cache* c) {
  if (!c) return KVPOP_OK;
  if (c->magic != kMagic) return KVPOP_ERR_INVALID_ARG;
  cudaDeviceSynchronize();
  cudaGetLastError();
  release(c);
  c->magic = 0;
  delete c;
  return KVPOP_OK;
}

namespace {

// Prompt compression, optionally with the prompt's attention outputs under the
// running top-k mask (Y != nullptr).
kvpop_status prefill_impl(kvpop_cache* c, const void* Q, const void* K, const void* V,
                          const int32_t* plen_host, int32_t first_seq, int32_t n_seq, int32_t Pmax,
                          const float* override_, float* Y, float* lse, int32_t* rank_out,
                          int32_t* tau_out, int32_t* order_out, cudaStream_t stream) {
  kvpop_status s = usable(c);
  if (s != KVPOP_OK) return s;
  if (!plen_host || n_seq < 0 || first_seq < 0 || first_seq + (long long)n_seq > c->dm.batch ||
      Pmax < 0 || Pmax > (1 << 24))
    return KVPOP_ERR_INVALID_ARG;
  if (n_seq == 0) return KVPOP_OK;
  for (int i = 0; i < n_seq; ++i)
    if (plen_host[i] < 0 || plen_host[i] > Pmax) return KVPOP_ERR_INVALID_ARG;
  if (Pmax > 0 && (!Q || !K || !V)) return KVPOP_ERR_INVALID_ARG;
  if (!aligned16(Q) || !aligned16(K) || !aligned16(V) || !aligned4(override_))
    return KVPOP_ERR_ALIGN;
  const bool outputs = Y != nullptr;
  if (outputs) {
    if (!aligned16(Y) || !aligned4(lse) || !aligned4(rank_out) || !aligned4(tau_out))
      return KVPOP_ERR_ALIGN;
    if (Pmax > kTopkMaxS || (long long)n_seq * c->dm.H > 65535 ||
        !prompt_attend_ok(c->dm.dtype, c->dm.d, c->dm.G, c->dm.s, c->dm.D, c->dm.B - c->dm.s))
      return KVPOP_ERR_INVALID_ARG;
  }
  const size_t pairs = (size_t)n_seq * c->dm.H;
  auto al = [](size_t x) { return (x + 255) & ~size_t(255); };
  const size_t prio_bytes = al(pairs * (size_t)Pmax * 4);
  // the mLSTM prefill also needs every prompt token's features (k~, v~, q~, gates)
  const size_t feat_bytes = c->mlstm ? pairs * (size_t)Pmax * mlstm_nf(c->dm.d) * 4 : 0;
  const size_t plen_off = prio_bytes;
  const size_t feat_off = plen_off + 256;
  const size_t rank_off = al(feat_off + feat_bytes);
  const size_t tau_off = rank_off + (outputs && !rank_out ? prio_bytes : 0);
  const size_t ws_off = tau_off + (outputs && !tau_out ? prio_bytes : 0);
  const size_t ws_bytes = outputs ? topk_workspace_bytes((int)pairs, Pmax) : 0;
  void* tmp = nullptr;
  if (g_fail_after > 0 && --g_fail_after == 0) return KVPOP_ERR_OOM;
  cudaError_t e = NOTE(cudaMallocAsync(&tmp, ws_off + ws_bytes + 256, stream));
  if (e != cudaSuccess) {
    cudaGetLastError();
    return from_cuda(e);
  }
  char* base = static_cast<char*>(tmp);
  float* prio = reinterpret_cast<float*>(base);
  int32_t* plen_dev = reinterpret_cast<int32_t*>(base + plen_off);
  e = NOTE(cudaMemcpyAsync(plen_dev, plen_host, (size_t)n_seq * 4, cudaMemcpyHostToDevice, stream));
  if (e == cudaSuccess && c->mlstm) {
    float* feat = reinterpret_cast<float*>(base + feat_off);
    e = NOTE(launch_prefill_mlstm_scores(c->st, c->dm, c->md, K, V, plen_dev, first_seq, n_seq, Pmax,
                                         override_, feat, prio, stream));
    if (e == cudaSuccess)
      e = NOTE(launch_prefill_select(c->st, c->dm, Q, K, V, plen_dev, first_seq, n_seq, Pmax, prio,
                                     stream));
  } else if (e == cudaSuccess) {
    e = NOTE(launch_prefill(c->st, c->dm, Q, K, V, plen_dev, first_seq, n_seq, Pmax, override_, prio,
                            sc_map_ptr(c), stream));
  }
  if (e == cudaSuccess && outputs && Pmax > 0) {
    int32_t* rank = rank_out ? rank_out : reinterpret_cast<int32_t*>(base + rank_off);
    int32_t* tau = tau_out ? tau_out : reinterpret_cast<int32_t*>(base + tau_off);
    const int s_ = c->dm.s, D = c->dm.D, k = c->dm.B - c->dm.s;
    e = NOTE(launch_topk(prio, plen_dev, c->dm.H, D, (int)pairs, Pmax, s_, D, k, rank, tau,
                         order_out, base + ws_off, stream));
    const int32_t* order = order_out ? order_out : topk_order(base + ws_off, (int)pairs, Pmax);
    if (e == cudaSuccess)
      e = NOTE(launch_prompt_attend(Q, K, V, rank, tau, order,
                                    plen_dev, n_seq, c->dm.H, c->dm.G, c->dm.d, Pmax, s_, D, k,
                                    c->dm.dtype, Y, lse, c->st.err, stream));
  }
  // the host copy of the lengths must outlive the async copy
  if (e == cudaSuccess) e = NOTE(cudaStreamSynchronize(stream));
  cudaError_t e2 = cudaFreeAsync(tmp, stream);
  if (e == cudaSuccess) e = e2;
  return poison_on(c, e);
}

}  // namespace

kvpop_status kvpop_prefill_compress(kvpop_cache* c, const void* Q, const void* K, const void* V,
                                    const int32_t* plen_host, int32_t first_seq, int32_t n_seq,
                                    int32_t Pmax, const float* override_, cudaStream_t stream) {
  return prefill_impl(c, Q, K, V, plen_host, first_seq, n_seq, Pmax, override_, nullptr, nullptr,
                      nullptr, nullptr, nullptr, stream);
}

kvpop_status kvpop_prefill_attend(kvpop_cache* c, const void* Q, const void* K, const void* V,
                                  const int32_t* plen_host, int32_t first_seq, int32_t n_seq,
                                  int32_t Pmax, const float* override_, float* Y, float* lse,
                                  int32_t* rank_out, int32_t* tau_out, int32_t* order_out,
                                  cudaStream_t stream) {
  if (!Y) return KVPOP_ERR_INVALID_ARG;
  if (!aligned4(order_out)) return KVPOP_ERR_ALIGN;
  return prefill_impl(c, Q, K, V, plen_host, first_seq, n_seq, Pmax, override_, Y, lse, rank_out,
                      tau_out, order_out, stream);
}

size_t kvpop_topk_workspace_bytes(int32_t n_rows, int32_t S) {
  if (n_rows <= 0 || S <= 0) return 0;
  return topk_workspace_bytes(n_rows, S);
}

kvpop_status kvpop_topk_cutoff(const float* prio, const int32_t* lengths, int32_t n_rows, int32_t S,
                               int32_t n_sink, int32_t window, int32_t k, int32_t* rank, int32_t* tau,
                               int32_t* order, void* workspace, size_t workspace_bytes,
                               cudaStream_t stream) {
  if (n_rows < 0 || S < 0 || S > kTopkMaxS || n_sink < 0 || window < 1 || k < 1)
    return KVPOP_ERR_INVALID_ARG;
  if (n_rows == 0 || S == 0) return KVPOP_OK;
  if (!prio || !rank || !tau || !workspace) return KVPOP_ERR_INVALID_ARG;
  if (workspace_bytes < topk_workspace_bytes(n_rows, S)) return KVPOP_ERR_INVALID_ARG;
  if (!aligned4(prio) || !aligned4(lengths) || !aligned4(rank) || !aligned4(tau) ||
      !aligned4(order) || (reinterpret_cast<uintptr_t>(workspace) & 255u))
    return KVPOP_ERR_ALIGN;
  cudaError_t e = NOTE(launch_topk(prio, lengths, 1, 0, n_rows, S, n_sink, window, k, rank, tau,
                                   order, workspace, stream));
  return from_cuda(e);
}

kvpop_status kvpop_prompt_attention(const void* Q, const void* K, const void* V, const int32_t* rank,
                                    const int32_t* tau, const int32_t* order,
                                    const int32_t* lengths, int32_t n_seq,
                                    int32_t n_kv_heads, int32_t q_per_kv, int32_t head_dim, int32_t S,
                                    int32_t n_sink, int32_t window, int32_t k, kvpop_dtype dtype,
                                    float* Y, float* lse, cudaStream_t stream) {
  if (n_seq < 0 || n_kv_heads < 1 || S < 0 || n_sink < 0 || window < 1 || k < 1 ||
      (dtype != KVPOP_F32 && dtype != KVPOP_BF16) || (long long)n_seq * n_kv_heads > 65535 ||
      !prompt_attend_ok(dtype, head_dim, q_per_kv, n_sink, window, k))
    return KVPOP_ERR_INVALID_ARG;
  if (n_seq == 0 || S == 0) return KVPOP_OK;
  if (!Q || !K || !V || !rank || !tau || !Y) return KVPOP_ERR_INVALID_ARG;
  if (!aligned16(Q) || !aligned16(K) || !aligned16(V) || !aligned16(Y) || !aligned4(rank) ||
      !aligned4(tau) || !aligned4(order) || !aligned4(lengths) || !aligned4(lse))
    return KVPOP_ERR_ALIGN;
  cudaError_t e = NOTE(launch_prompt_attend(Q, K, V, rank, tau, order, lengths, n_seq, n_kv_heads,
                                            q_per_kv, head_dim, S, n_sink, window, k, dtype, Y, lse,
                                            standalone_err(), stream));
  return from_cuda(e);
}

kvpop_status kvpop_causal_lse(const void* Q, const void* K, const int32_t* lengths, int32_t n_seq,
                              int32_t n_kv_heads, int32_t q_per_kv, int32_t head_dim, int32_t S,
                              kvpop_dtype dtype, float* lse, cudaStream_t stream) {
  if (n_seq < 0 || n_kv_heads < 1 || S < 0 || (dtype != KVPOP_F32 && dtype != KVPOP_BF16) ||
      (long long)n_seq * n_kv_heads > 65535 || !prompt_attend_ok(dtype, head_dim, q_per_kv, 0, 1, 1))
    return KVPOP_ERR_INVALID_ARG;
  if (n_seq == 0 || S == 0) return KVPOP_OK;
  if (!Q || !K || !lse) return KVPOP_ERR_INVALID_ARG;
  if (!aligned16(Q) || !aligned16(K) || !aligned4(lse) || !aligned4(lengths)) return KVPOP_ERR_ALIGN;
  return from_cuda(NOTE(launch_causal_lse(Q, K, lengths, n_seq, n_kv_heads, q_per_kv, head_dim, S,
                                          dtype, lse, standalone_err(), stream)));
}

kvpop_status kvpop_future_target(const void* Q, const void* K, const float* lse,
                                 const int32_t* lengths, int32_t n_seq, int32_t n_kv_heads,
                                 int32_t q_per_kv, int32_t head_dim, int32_t S, int32_t window,
                                 int32_t lookahead, kvpop_dtype dtype, float* logm, float* target,
                                 int32_t agg, int32_t count_norm, float eps, cudaStream_t stream) {
  if (n_seq < 0 || n_kv_heads < 1 || S < 0 || window < 0 || lookahead < 0 ||
      (dtype != KVPOP_F32 && dtype != KVPOP_BF16) || (long long)n_seq * n_kv_heads > 65535 ||
      !prompt_attend_ok(dtype, head_dim, q_per_kv, 0, 1, 1) || (agg != 0 && agg != 1) ||
      (count_norm != 0 && count_norm != 1) || !(eps >= 0.f) || eps == INFINITY)
    return KVPOP_ERR_INVALID_ARG;
  if (n_seq == 0 || S == 0) return KVPOP_OK;
  if (!Q || !K || !lse || !logm) return KVPOP_ERR_INVALID_ARG;
  if (!aligned16(Q) || !aligned16(K) || !aligned4(lse) || !aligned4(lengths) || !aligned4(logm) ||
      !aligned4(target))
    return KVPOP_ERR_ALIGN;
  return from_cuda(NOTE(launch_future_target(Q, K, lse, lengths, n_seq, n_kv_heads, q_per_kv,
                                             head_dim, S, window, lookahead, dtype, logm, target,
                                             agg, count_norm, eps, standalone_err(), stream)));
}

kvpop_status kvpop_standalone_status(cudaStream_t stream) {
  int32_t* d = standalone_err();
  if (!d) return KVPOP_ERR_CUDA;
  int32_t h = 0;
  cudaError_t e = NOTE(cudaMemcpyAsync(&h, d, 4, cudaMemcpyDeviceToHost, stream));
  if (e == cudaSuccess) e = NOTE(cudaStreamSynchronize(stream));
  if (e != cudaSuccess) return from_cuda(e);
  if (h != 0) {
    std::snprintf(g_last_error, sizeof(g_last_error), "device error code %d", h);
    e = NOTE(cudaMemsetAsync(d, 0, 4, stream));
    if (e == cudaSuccess) e = NOTE(cudaStreamSynchronize(stream));
    return e == cudaSuccess ? KVPOP_ERR_DEVICE_CHECK : from_cuda(e);
  }
  return KVPOP_OK;
}

kvpop_status kvpop_decode_ingest(kvpop_cache* c, const void* q, const void* k, const void* v,
                                 const float* override_, int32_t* evict_info, float* score_out,
                                 cudaStream_t stream) {
  kvpop_status s = usable(c);
  if (s != KVPOP_OK) return s;
  if (!q || !k || !v) return KVPOP_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned4(override_) ||
      !aligned4(evict_info) || !aligned4(score_out))
    return KVPOP_ERR_ALIGN;
  if (c->mlstm)
    return poison_on(c, NOTE(launch_ingest_mlstm(c->st, c->dm, c->md, q, k, v, override_, evict_info,
                                                 score_out, stream)));
  if (c->use_cluster)
    return poison_on(c, NOTE(launch_ingest_cluster(c->st, c->dm, c->W1s, c->b1s, c->w2s, q, k, v,
                                                   override_, evict_info, score_out, stream)));
  return poison_on(c, NOTE(launch_ingest(c->st, c->dm, q, k, v, override_, evict_info, score_out, stream)));
}

kvpop_status kvpop_decode_attend(kvpop_cache* c, const void* q, float* out, cudaStream_t stream) {
  kvpop_status s = usable(c);
  if (s != KVPOP_OK) return s;
  if (!q || !out) return KVPOP_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(out)) return KVPOP_ERR_ALIGN;
  if (c->use_tc)
    return poison_on(c, NOTE(tc_launch(c->st, c->dm, tc_map_ptr(c), q, out, c->attend_grid, stream)));
  return poison_on(c, NOTE(launch_attend(c->st, c->dm, q, out, c->attend_grid, stream)));
}

kvpop_status kvpop_decode_step(kvpop_cache* c, const void* q, const void* k, const void* v,
                               float* out, const float* override_, int32_t* evict_info,
                               float* score_out, cudaStream_t stream) {
  kvpop_status s = usable(c);
  if (s != KVPOP_OK) return s;
  if (!out) return KVPOP_ERR_INVALID_ARG;
  if (!aligned16(out)) return KVPOP_ERR_ALIGN;
  if (c->use_fused) {
    if (!q || !k || !v) return KVPOP_ERR_INVALID_ARG;
    if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned4(override_) ||
        !aligned4(evict_info) || !aligned4(score_out))
      return KVPOP_ERR_ALIGN;
    return poison_on(c, NOTE(tc_launch_fused(c->st, c->dm, tc_map_ptr(c), c->fb, q, k, v, out,
                                             override_, evict_info, score_out, c->fused_grid,
                                             stream)));
  }
  s = kvpop_decode_ingest(c, q, k, v, override_, evict_info, score_out, stream);
  if (s != KVPOP_OK) return s;
  return kvpop_decode_attend(c, q, out, stream);
}

int32_t kvpop_step_is_fused(const kvpop_cache* c) {
  if (!c || c->magic != kMagic) return -1;
  return c->use_fused ? 1 : 0;
}

kvpop_status kvpop_decode_step_host(kvpop_cache* c, const void* q, const void* k, const void* v,
                                    float* out, cudaStream_t stream) {
  kvpop_status s = usable(c);
  if (s != KVPOP_OK) return s;
  if (!q || !k || !v || !out) return KVPOP_ERR_INVALID_ARG;
  const size_t pairs = c->dm.pairs, d = c->dm.d, G = c->dm.G;
  const size_t qb = pairs * G * d * c->esz, kb = pairs * d * c->esz;
  // pinned host memory the device can address is read (inputs) and written (output) by
  // the step's kernels in place; anything else goes through the device staging buffers
  const void* mq = mapped_host(q);
  const void* mk = mq ? mapped_host(k) : nullptr;
  const void* mv = mk ? mapped_host(v) : nullptr;
  float* direct = static_cast<float*>(const_cast<void*>(mapped_host(out)));
  const void *dq = mq, *dk = mk, *dv = mv;
  if (!mv) {
    const char* qc = static_cast<const char*>(q);
    cudaError_t e = cudaErrorInvalidValue;
    // adjacent buffers take one copy; adjacent addresses from different host allocations
    // are refused by the runtime before anything is queued, and then take three
    if (static_cast<const char*>(k) == qc + qb && static_cast<const char*>(v) == qc + qb + kb) {
      e = cudaMemcpyAsync(c->stage_q, q, qb + 2 * kb, cudaMemcpyHostToDevice, stream);
      if (e == cudaErrorInvalidValue) cudaGetLastError();
    }
    if (e == cudaErrorInvalidValue) {
      e = NOTE(cudaMemcpyAsync(c->stage_q, q, qb, cudaMemcpyHostToDevice, stream));
      if (e == cudaSuccess) e = NOTE(cudaMemcpyAsync(c->stage_k, k, kb, cudaMemcpyHostToDevice, stream));
      if (e == cudaSuccess) e = NOTE(cudaMemcpyAsync(c->stage_v, v, kb, cudaMemcpyHostToDevice, stream));
    }
    if (e != cudaSuccess) return poison_on(c, e);
    dq = c->stage_q;
    dk = c->stage_k;
    dv = c->stage_v;
  }
  s = kvpop_decode_step(c, dq, dk, dv, direct ? direct : c->stage_out, nullptr, nullptr, nullptr, stream);
  if (s != KVPOP_OK || direct) return s;
  cudaError_t e = NOTE(cudaMemcpyAsync(out, c->stage_out, pairs * G * d * 4, cudaMemcpyDeviceToHost, stream));
  return poison_on(c, e);
}

kvpop_status kvpop_check(kvpop_cache* c, cudaStream_t stream) {
  kvpop_status s = usable(c);
  if (s != KVPOP_OK) return s;
  cudaError_t e = NOTE(cudaStreamSynchronize(stream));
  if (e != cudaSuccess) return poison_on(c, e);
  int32_t err[16];
  e = NOTE(cudaMemcpy(err, c->st.err, sizeof(err), cudaMemcpyDeviceToHost));
  if (e != cudaSuccess) return poison_on(c, e);
  if (err[0] != 0) {
    cudaMemset(c->st.err, 0, sizeof(err));
    return KVPOP_ERR_DEVICE_CHECK;
  }
  return KVPOP_OK;
}

kvpop_status kvpop_export_state(kvpop_cache* c, void* host_buf, size_t* bytes, cudaStream_t stream) {
  kvpop_status s = usable(c);
  if (s != KVPOP_OK) return s;
  if (!bytes) return KVPOP_ERR_INVALID_ARG;
  auto bufs = all_state_buffers(c);
  size_t need = 4 * sizeof(uint64_t) + sizeof(kvpop_config);
  for (auto& b : bufs) need += b.bytes;
  if (!host_buf) { *bytes = need; return KVPOP_OK; }
  if (*bytes < need) { *bytes = need; return KVPOP_ERR_INVALID_ARG; }
  unsigned char* out = static_cast<unsigned char*>(host_buf);
  uint64_t hdr[4] = {kMagic, kStateVersion, (uint64_t)need, 0};
  std::memcpy(out, hdr, sizeof(hdr));
  std::memcpy(out + sizeof(hdr), &c->cfg, sizeof(kvpop_config));
  size_t off = sizeof(hdr) + sizeof(kvpop_config);
  cudaError_t e = cudaSuccess;
  for (auto& b : bufs) {
    if (e == cudaSuccess) e = NOTE(cudaMemcpyAsync(out + off, b.ptr, b.bytes, cudaMemcpyDeviceToHost, stream));
    off += b.bytes;
  }
  if (e == cudaSuccess) e = NOTE(cudaStreamSynchronize(stream));
  *bytes = need;
  return poison_on(c, e);
}

kvpop_status kvpop_import_state(kvpop_cache* c, const void* host_buf, size_t bytes, cudaStream_t stream) {
  kvpop_status s = usable(c);
  if (s != KVPOP_OK) return s;
  if (!host_buf) return KVPOP_ERR_INVALID_ARG;
  const unsigned char* in = static_cast<const unsigned char*>(host_buf);
  uint64_t hdr[4];
  if (bytes < sizeof(hdr) + sizeof(kvpop_config)) return KVPOP_ERR_INVALID_ARG;
  std::memcpy(hdr, in, sizeof(hdr));
  kvpop_config cfg;
  std::memcpy(&cfg, in + sizeof(hdr), sizeof(cfg));
  auto bufs = all_state_buffers(c);
  size_t need = sizeof(hdr) + sizeof(kvpop_config);
  for (auto& b : bufs) need += b.bytes;
  if (hdr[0] != kMagic || hdr[1] != kStateVersion || hdr[2] != need || bytes < need ||
      std::memcmp(&cfg, &c->cfg, sizeof(cfg)) != 0)
    return KVPOP_ERR_INVALID_ARG;
  size_t off = sizeof(hdr) + sizeof(kvpop_config);
  cudaError_t e = cudaSuccess;
  for (auto& b : bufs) {
    if (e == cudaSuccess) e = NOTE(cudaMemcpyAsync(b.ptr, in + off, b.bytes, cudaMemcpyHostToDevice, stream));
    off += b.bytes;
  }
  if (e == cudaSuccess) e = NOTE(cudaMemsetAsync(c->st.part_count, 0, (size_t)c->dm.pairs * 4, stream));
  if (e == cudaSuccess) e = NOTE(cudaStreamSynchronize(stream));
  return poison_on(c, e);
}

kvpop_status kvpop_get_lengths(kvpop_cache* c, int32_t* len_host, cudaStream_t stream) {
  kvpop_status s = usable(c);
  if (s != KVPOP_OK) return s;
  if (!len_host) return KVPOP_ERR_INVALID_ARG;
  std::vector<int32_t> all;
  try {
    all.resize((size_t)c->dm.pairs);
  } catch (...) {
    return KVPOP_ERR_OOM;
  }
  cudaError_t e = NOTE(cudaMemcpyAsync(all.data(), c->st.len, all.size() * 4, cudaMemcpyDeviceToHost, stream));
  if (e == cudaSuccess) e = NOTE(cudaStreamSynchronize(stream));
  if (e != cudaSuccess) return poison_on(c, e);
  for (int b = 0; b < c->dm.batch; ++b) len_host[b] = all[(size_t)b * c->dm.H];
  return KVPOP_OK;
}

kvpop_status kvpop_get_pair_state(kvpop_cache* c, int32_t seq, int32_t head, int32_t* pos_host,
                                  float* score_host, int32_t* nvalid_host, cudaStream_t stream) {
  kvpop_status s = usable(c);
  if (s != KVPOP_OK) return s;
  if (seq < 0 || seq >= c->dm.batch || head < 0 || head >= c->dm.H) return KVPOP_ERR_INVALID_ARG;
  const size_t pair = (size_t)seq * c->dm.H + head, B = c->dm.B;
  cudaError_t e = cudaSuccess;
  if (pos_host) e = NOTE(cudaMemcpyAsync(pos_host, c->st.pos + pair * B, B * 4, cudaMemcpyDeviceToHost, stream));
  if (e == cudaSuccess && score_host)
    e = NOTE(cudaMemcpyAsync(score_host, c->st.score + pair * B, B * 4, cudaMemcpyDeviceToHost, stream));
  if (e == cudaSuccess && nvalid_host)
    e = NOTE(cudaMemcpyAsync(nvalid_host, c->st.nvalid + pair, 4, cudaMemcpyDeviceToHost, stream));
  if (e == cudaSuccess) e = NOTE(cudaStreamSynchronize(stream));
  return poison_on(c, e);
}

}  // extern "C"
