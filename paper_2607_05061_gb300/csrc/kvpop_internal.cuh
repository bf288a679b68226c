// Internal declarations shared by the KVpop CUDA translation units.
// Not part of the public ABI (see include/kvpop.h).
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "../../include/kvpop.h"

namespace kvpop {

typedef __nv_bfloat16 bf16;

// Device-side error codes written to cache->err[0] (first error wins).
enum : int {
  DEVERR_NONE = 0,
  DEVERR_TIMEOUT_FULL = 1,     // consumer gave up waiting for a K/V tile
  DEVERR_TIMEOUT_EMPTY = 2,    // producer gave up waiting for a free stage
  DEVERR_TIMEOUT_DRAIN = 3,    // producer gave up draining its copies at exit
  DEVERR_BAD_SCHEDULE = 4,     // attention schedule inconsistent with the state
  DEVERR_INDEX = 5,            // an index check failed (device-check build only)
  DEVERR_TIMEOUT_SCHED = 6,    // fused step: gave up waiting for every CTA's schedule
};

// Index checks of the device-check build (compiled with -DKVPOP_DEVICE_CHECKS):
// dcheck(cond, err, code) records `code` in *err (first error wins) and returns
// false when cond fails, so the caller skips the access instead of trapping.  In
// the normal build it is `true` and compiles away.
#ifdef KVPOP_DEVICE_CHECKS
__device__ __forceinline__ bool dcheck(bool cond, int32_t* err, int code) {
  if (!cond && err) atomicCAS(err, 0, code);
  return cond;
}
#else
__device__ __forceinline__ bool dcheck(bool, int32_t*, int) { return true; }
#endif

// Used slots and window rows of a pair, clamped to the buffers they index, so that
// state the library did not write (the allocation-free entry point takes it from the
// caller) can never send a copy outside them; the device-check build also records
// any value that needed clamping.
__device__ __forceinline__ int used_slots(int nv, int B, int32_t* err) {
  dcheck(nv >= 0 && nv <= B, err, DEVERR_INDEX);
  return min(max(nv, 0), B);
}
__device__ __forceinline__ int window_rows(int len, int D, int32_t* err) {
  dcheck(len >= 0, err, DEVERR_INDEX);
  return min(max(len, 0), D);
}


// Wall-clock budget of any single mbarrier wait before a kernel gives up.
constexpr unsigned long long kWaitLimitNs = 2000000000ull;

// A kernel's dynamic shared-memory limit is one process-wide attribute.  Every
// launch path raises it to the most the device allows that kernel (the opt-in
// maximum less its static shared memory) -- the same value whoever sets it --
// so one caller's set-up never lowers the limit under another caller's launch
// (caches of different sizes, other host threads).  Returns
// cudaErrorInvalidValue when `need` exceeds that maximum.
template <typename K>
inline cudaError_t raise_smem_limit(K* func, size_t need) {
  int dev = 0, optin = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  cudaFuncAttributes fa;
  if (e == cudaSuccess) e = cudaFuncGetAttributes(&fa, reinterpret_cast<const void*>(func));
  if (e != cudaSuccess) return e;
  const long long room = (long long)optin - (long long)fa.sharedSizeBytes;
  if (room < 0 || (long long)need > room) return cudaErrorInvalidValue;
  return cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)room);
}

struct State {                 // device pointers of one cache
  void* slotK;                 // [pairs][B][d]   element type T
  void* slotV;
  void* ringK;                 // [pairs][D][d]
  void* ringV;
  float* ringQm;               // [pairs][D][d]   mean query of each window token
  float* score;                // [pairs][B]      static priority of each slot
  int32_t* pos;                // [pairs][B]      position held by each slot
  int32_t* nvalid;             // [pairs]
  int32_t* len;                // [pairs]         tokens seen (same for all heads of a sequence)
  float* min_score;            // [pairs]         argmin over slots [s, B) when full
  int32_t* min_slot;           // [pairs]
  float* blk_score;            // [pairs][NB]     per-block minima (blocks of 64 slots)
  int32_t* blk_slot;           // [pairs][NB]
  // scorer (hidden width padded to Fp = F rounded up to 4, zero weights)
  const float* W1;             // [H][3d][Fp]
  const float* b1;             // [H][Fp]
  const float* w2;             // [H][Fp]
  const float* b2;             // [H]
  const float* log_gamma;      // [H] or nullptr
  // attention workspace
  float* part;                 // [2 * grid][G*d + 2*G]
  int32_t* part_count;         // [pairs]
  int32_t* err;                // [4]
};

struct Dims {
  int batch, H, G, d, B, D, s, F, Fp;
  int act;                     // scorer hidden activation: 0 GELU (erf), 1 SiLU, 2 identity
  int dtype;                   // kvpop_dtype
  int pairs;
};

// ------------------------------------------------------------------ launchers
cudaError_t launch_ingest(const State& st, const Dims& dm, const void* q, const void* k,
                          const void* v, const float* override_, int32_t* evict_info,
                          float* score_out, cudaStream_t stream);

// Cluster ingest (8 CTAs per KV head and 16 sequences, hidden units split 8 ways).
// Weights in slice-major layout: W1s [H][8][3d][FS], b1s / w2s [H][8][FS].
bool cluster_ingest_ok(const Dims& dm);
int cluster_ingest_fs(const Dims& dm);
cudaError_t prepare_ingest_cluster(const Dims& dm);
cudaError_t launch_ingest_cluster(const State& st, const Dims& dm, const float* W1s,
                                  const float* b1s, const float* w2s, const void* q,
                                  const void* k, const void* v, const float* override_,
                                  int32_t* evict_info, float* score_out, cudaStream_t stream);

// Attention kernel resources for a (dtype, d, G) combination.
struct AttendConfig {
  int threads;
  size_t smem_fixed;           // bytes independent of the number of pairs
  int tile;                    // keys per tile
  const void* func;            // kernel symbol (for occupancy queries)
};
cudaError_t attend_config(const Dims& dm, AttendConfig* out);
cudaError_t launch_attend(const State& st, const Dims& dm, const void* q, float* out,
                          int grid, cudaStream_t stream);

// Stateful mLSTM scorer (device arrays of one cache).
struct MlstmDev {
  float* C;                    // [pairs][d][d/2]  stabilised matrix memory
  float* z;                    // [pairs][d]       normaliser
  float* m;                    // [pairs]          log-scale of the stabiliser
  float* Wcat;                 // [H][2d][NC]      columns [W_k | W_v | W_q | w_i | w_f | 0]
  float* bi;                   // [H]
  float* bf;                   // [H]
  float* a;                    // [H][d/2]
  float* b;                    // [H]
  int NC;
};
int mlstm_nc(int d);
int mlstm_nf(int d);
bool mlstm_ok(const Dims& dm);
cudaError_t prepare_mlstm(const Dims& dm);
cudaError_t launch_ingest_mlstm(const State& st, const Dims& dm, const MlstmDev& m, const void* q,
                                const void* k, const void* v, const float* override_,
                                int32_t* evict_info, float* score_out, cudaStream_t stream);
cudaError_t launch_prefill_mlstm_scores(const State& st, const Dims& dm, const MlstmDev& m,
                                        const void* K, const void* V, const int32_t* plen,
                                        int first_seq, int n_seq, int Pmax, const float* override_,
                                        float* feat, float* prio, cudaStream_t stream);
// Selection + compaction + window fill of the prefill, from precomputed priorities.
cudaError_t launch_prefill_select(const State& st, const Dims& dm, const void* Q, const void* K,
                                  const void* V, const int32_t* plen, int first_seq, int n_seq,
                                  int Pmax, const float* prio, cudaStream_t stream);

// Tensor-core attention for bf16 K/V (TMA tensor maps over the K/V stores).
size_t tc_maps_size();
cudaError_t tc_make_maps(const State& st, const Dims& dm, void* maps_out);
cudaError_t tc_config(const Dims& dm, AttendConfig* out);
cudaError_t tc_launch(const State& st, const Dims& dm, const void* maps, const void* q, float* out,
                      int grid, cudaStream_t stream);
// The whole decode step in one tensor-core kernel (bf16, d = 128, F <= 256): attention over
// the keys that cannot change this step while extra warps run the delayed scorer,
// keep-or-drop and scatter; each pair's last arrival merges.
struct FusedBufs {
  float* part_c;               // [pairs][G d + 2 G]
  int32_t* meta_next;          // [pairs][4]
  float* xtra;                 // [pairs][2 G + 2 d]
  unsigned long long* ctr;     // CTAs past their schedule over all launches (zero at init)
  int2* start_prev;            // [grid] where each CTA's range began last launch (zero at init)
};
bool tc_fused_ok(const Dims& dm);
int tc_fused_max_grid();         // largest grid the fused kernel's split table holds
cudaError_t tc_fused_config(const Dims& dm, AttendConfig* out);
cudaError_t tc_launch_fused(const State& st, const Dims& dm, const void* maps, const FusedBufs& fb,
                            const void* q, const void* k, const void* v, float* out,
                            const float* override_, int32_t* evict_info, float* score_out, int grid,
                            cudaStream_t stream);

// Prefill scores + selection; `tf32_maps` (W1^T tensor maps from prepare_score_tf32, or
// null) routes the learned scores through the tensor-core scorer.
cudaError_t launch_prefill(const State& st, const Dims& dm, const void* Q, const void* K,
                           const void* V, const int32_t* plen_dev, int first_seq, int n_seq,
                           int Pmax, const float* override_, float* tmp_prio,
                           const void* tf32_maps, cudaStream_t stream);
// Prompt scorer on the tensor cores (3xTF32 split products, fp32 accuracy): W1^T
// split into tf32 head and residual [2][H][F][3d] (w1t, 2 H F 3d floats) and two
// TMA descriptors over them (score_tf32_maps_size bytes, 64-byte aligned).
bool score_tf32_ok(const Dims& dm);
size_t score_tf32_maps_size();
cudaError_t prepare_score_tf32(const Dims& dm, const float* W1, float* w1t, void* maps_out,
                               cudaStream_t stream);
cudaError_t launch_score_tf32(const State& st, const Dims& dm, const void* maps, const void* Q,
                              const void* K, const void* V, const int32_t* plen, int n_seq, int Pmax,
                              float* prio, cudaStream_t stream);

// Running top-k over a prompt (App. C): static ranks and per-query cutoffs of
// n_rows rows of S tokens; row r has len[r / rows_per_len] tokens (S if len is
// null), the last `tail` of them without a priority.
constexpr int kTopkMaxS = 1 << 18;
size_t topk_workspace_bytes(int n_rows, int S);
// After launch_topk: the position of every rank of every row ([n_rows][S], ranks 0 .. L-1
// of a row of length L), inside the workspace.
const int32_t* topk_order(const void* workspace, int n_rows, int S);
// `order` receives the position of each rank ([n_rows][S]); null puts it in the workspace
// (topk_order).
cudaError_t launch_topk(const float* prio, const int32_t* len, int rows_per_len, int tail,
                        int n_rows, int S, int s, int w, int k, int32_t* rank, int32_t* tau,
                        int32_t* order, void* workspace, cudaStream_t stream);
// Masked causal attention over a prompt under the running top-k mask.
bool prompt_attend_ok(int dtype, int d, int G, int s, int w, int k);
// `order` (positions by rank, from topk_order, or null) lets a tile's key lists be
// built from the ranks up to its largest cutoff instead of from every eligible position.
cudaError_t launch_prompt_attend(const void* Q, const void* K, const void* V, const int32_t* rank,
                                 const int32_t* tau, const int32_t* order, const int32_t* len,
                                 int n_seq, int H, int G, int d, int S, int s, int w, int k,
                                 int dtype, float* Y, float* lse, int32_t* err, cudaStream_t stream);

// Dense causal log-normalisers of every prompt query (LSE only, no output rows).
cudaError_t launch_causal_lse(const void* Q, const void* K, const int32_t* len, int n_seq, int H,
                              int G, int d, int S, int dtype, float* lse, int32_t* err,
                              cudaStream_t stream);
// Future-attention log masses (transposed pass) and the aggregated target.
cudaError_t launch_future_target(const void* Q, const void* K, const float* lse, const int32_t* len,
                                 int n_seq, int H, int G, int d, int S, int w, int la, int dtype,
                                 float* logm, float* target, int agg, int count_norm, float eps,
                                 int32_t* err, cudaStream_t stream);

// ------------------------------------------------------------------ device helpers
__device__ __forceinline__ float to_f(float x) { return x; }
__device__ __forceinline__ float to_f(bf16 x) { return __bfloat162float(x); }

// Canonical score: NaN -> -inf, -0 -> +0 (every ranking decision uses it).
__device__ __forceinline__ float canon_score(float r) {
  if (r != r) return -INFINITY;
  return __fadd_rn(r, 0.0f);   // -0 + +0 = +0 under round-to-nearest
}

// Static priority (App. B.3, decay step n = 1) in explicit fp32 ops.
__device__ __forceinline__ float static_priority(float r, int u, const float* log_gamma, int h) {
  if (log_gamma == nullptr) return r;
  float lg = log_gamma[h];
  if (lg == 0.0f) return r;
  return canon_score(__fsub_rn(r, __fmul_rn((float)u, lg)));
}

// Exact-erf GELU.
__device__ __forceinline__ float gelu_erf(float z) {
  return 0.5f * z * (1.0f + erff(z * 0.70710678118654752440f));
}

// Hidden-layer activation of the stateless scorer (Sec. 3.3): GELU, SiLU or none.
__device__ __forceinline__ float scorer_act(float z, int act) {
  if (act == 0) return gelu_erf(z);
  if (act == 1) return z / (1.0f + expf(-z));
  return z;
}

}  // namespace kvpop
