// Two-level lowest-priority tracking over a KV head's B slots.
//
// The keep-or-drop rule compares a newly eligible token with the lowest stored
// priority among the long-range slots [s, B), ties going to the lowest slot
// index.  Slots are grouped in blocks of kMinBlock; each block keeps its own
// (priority, slot) minimum and the head keeps the minimum over blocks, so a
// replacement re-reads one block and the block minima (2 * kMinBlock / 64 ...
// a few hundred bytes) instead of all B priorities.  The lexicographic order on
// (priority, slot) makes the two-level minimum equal to the flat one.
#pragma once

#include "kvpop_ptx.cuh"

namespace kvpop {

constexpr int kMinBlock = 64;

__host__ __device__ __forceinline__ int min_blocks(int B) { return (B + kMinBlock - 1) / kMinBlock; }

// Warp-collective minimum of block k of slots; slot j_new reads as v_new.
__device__ __forceinline__ void block_min(const float* __restrict__ sc, int s, int B, int k,
                                          int j_new, float v_new, float& m, int& mi) {
  const int lane = threadIdx.x & 31;
  float best = INFINITY;
  int bi = 0x7fffffff;
  const int lo = k * kMinBlock, hi = min(B, lo + kMinBlock);
#pragma unroll
  for (int r = 0; r < kMinBlock / 32; ++r) {
    const int i = lo + r * 32 + lane;
    if (i < hi && i >= s) lex_min(best, bi, (i == j_new) ? v_new : sc[i], i);
  }
  warp_lex_min(best, bi);
  m = best;
  mi = bi;
}

// Warp-collective minimum over the NB block minima; block k_new reads as (v, vi).
__device__ __forceinline__ void blocks_min(const float* __restrict__ bs, const int32_t* __restrict__ bsl,
                                           int NB, int k_new, float v, int vi, float& m, int& mi) {
  const int lane = threadIdx.x & 31;
  float best = INFINITY;
  int bi = 0x7fffffff;
  for (int k = lane; k < NB; k += 32) {
    if (k == k_new) lex_min(best, bi, v, vi);
    else lex_min(best, bi, bs[k], bsl[k]);
  }
  warp_lex_min(best, bi);
  m = best;
  mi = bi;
}

// Warp-collective rebuild of every block minimum and of the head minimum.
__device__ __forceinline__ void rebuild_min(float* __restrict__ sc, int s, int B, int j_new,
                                            float v_new, float* __restrict__ bs,
                                            int32_t* __restrict__ bsl, float* min_score,
                                            int32_t* min_slot) {
  const int lane = threadIdx.x & 31;
  const int NB = min_blocks(B);
  for (int k = 0; k < NB; ++k) {
    float m;
    int mi;
    block_min(sc, s, B, k, j_new, v_new, m, mi);
    if (lane == 0) { bs[k] = m; bsl[k] = mi; }
  }
  __syncwarp();
  float m;
  int mi;
  blocks_min(bs, bsl, NB, -1, 0.f, 0, m, mi);
  if (lane == 0) { *min_score = m; *min_slot = mi; }
}

// Warp-collective update after slot j took priority v (the head was full).
__device__ __forceinline__ void update_min(const float* __restrict__ sc, int s, int B, int j, float v,
                                           float* __restrict__ bs, int32_t* __restrict__ bsl,
                                           float* min_score, int32_t* min_slot) {
  const int lane = threadIdx.x & 31;
  const int k = j / kMinBlock;
  float bm;
  int bmi;
  block_min(sc, s, B, k, j, v, bm, bmi);
  float m;
  int mi;
  blocks_min(bs, bsl, min_blocks(B), k, bm, bmi, m, mi);
  if (lane == 0) {
    bs[k] = bm;
    bsl[k] = bmi;
    *min_score = m;
    *min_slot = mi;
  }
}

}  // namespace kvpop
