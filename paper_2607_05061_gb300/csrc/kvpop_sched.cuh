// Split-K schedule and partial merge shared by the decode-attention kernels.
//
// The key stream of every (sequence, KV head) pair -- used slots first, then
// the window -- is cut into tiles of `tile` keys.  The concatenated tile list
// over all pairs is split into NC equal contiguous ranges, one per CTA, so the
// work per CTA is balanced whatever the per-pair lengths (ragged batches).
// A pair whose tiles span several CTAs gets one (m, l, o) partial from each;
// the last CTA to finish it (atomic counter, no waiting) merges them in CTA
// order, which keeps the result independent of arrival order.
#pragma once

#include "kvpop_internal.cuh"

namespace kvpop {

__device__ __forceinline__ int tiles_of(int nv, int np, int tile) {
  return (nv + tile - 1) / tile + (np + tile - 1) / tile;
}

// CTA whose tile range [c*T/N, (c+1)*T/N) contains tile t (requires N <= T).
__device__ __forceinline__ long long cta_of(long long t, long long T, long long N) {
  return ((t + 1) * N - 1) / T;
}
__device__ __forceinline__ long long cta_begin(long long c, long long T, long long N) {
  return c * T / N;
}

// Block-wide exclusive prefix of per-pair tile counts into prefix[0..npairs]
// (prefix[npairs] = total).  `scan` holds one int per warp.  Contains
// __syncthreads; every thread of the block must call it.
template <int NT>
__device__ __forceinline__ void build_schedule(const int32_t* __restrict__ nvalid,
                                               const int32_t* __restrict__ len, int npairs, int B,
                                               int D, int tile, int* prefix, int* scan,
                                               int32_t* err) {
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int per = (npairs + NT - 1) / NT;
  const int beg = min(tid * per, npairs), end = min(beg + per, npairs);
  int local = 0;
  for (int i = beg; i < end; ++i)
    local += tiles_of(used_slots(nvalid[i], B, err), window_rows(len[i], D, err), tile);
  int incl = local;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, incl, off);
    if (lane >= off) incl += y;
  }
  if (lane == 31) scan[warp] = incl;
  __syncthreads();
  if (tid == 0) {
    int run = 0;
    for (int w = 0; w < NT / 32; ++w) { const int x = scan[w]; scan[w] = run; run += x; }
    prefix[npairs] = run;
  }
  __syncthreads();
  int run = scan[warp] + incl - local;
  for (int i = beg; i < end; ++i) {
    prefix[i] = run;
    run += tiles_of(used_slots(nvalid[i], B, nullptr), window_rows(len[i], D, nullptr), tile);
  }
  __syncthreads();
}

// Pair p's segment in this CTA is complete; mo/ml/mm hold NW warp partials
// (log2-domain running max mm, sum ml, unnormalised output mo[w][g][d]).
// Writes the output, or this CTA's partial and -- when it is the last
// contributor -- the merged output.  Called by the NCT consumer threads
// (tid < NCT) together; `sync` is their barrier; `flag` is one shared int.
template <int G, int HD, int NW, int NCT, typename SyncFn>
__device__ __forceinline__ void finish_pair(int p, const int* prefix, long long Ttot, long long NC,
                                            long long t0, const float* mo, const float* ml,
                                            const float* mm, float* out, float* part,
                                            int32_t* part_count, int* flag, SyncFn sync) {
  constexpr int PSTRIDE = G * HD + 2 * G;
  const int tid = threadIdx.x;
  const long long ca = cta_of(prefix[p], Ttot, NC);
  const long long cb = cta_of(prefix[p + 1] - 1, Ttot, NC);
  const bool complete = (ca == cb);
  float* mypart = nullptr;
  if (!complete) {
    const int slot = (prefix[p] < t0) ? 0 : 1;
    mypart = part + ((size_t)blockIdx.x * 2 + slot) * PSTRIDE;
  }
  for (int idx = tid; idx < G * HD; idx += NCT) {
    const int g = idx / HD, i = idx - g * HD;
    float ms = -INFINITY;
#pragma unroll
    for (int w = 0; w < NW; ++w) ms = fmaxf(ms, mm[w * G + g]);
    float L = 0.f, O = 0.f;
#pragma unroll
    for (int w = 0; w < NW; ++w) {
      const float mw = mm[w * G + g];
      const float f = (mw == -INFINITY) ? 0.f : exp2f(mw - ms);
      L = fmaf(ml[w * G + g], f, L);
      O = fmaf(mo[(w * G + g) * HD + i], f, O);
    }
    if (complete) {
      out[((size_t)p * G + g) * HD + i] = O / L;
    } else {
      mypart[g * HD + i] = O;
      if (i == 0) { mypart[G * HD + g] = ms; mypart[G * HD + G + g] = L; }
    }
  }
  if (!complete) {
    __threadfence();
    sync();
    if (tid == 0) {
      const int old = atomicAdd(&part_count[p], 1);
      const int last = (old == (int)(cb - ca));
      if (last) part_count[p] = 0;
      *flag = last;
    }
    sync();
    if (*flag) {
      __threadfence();
      for (int idx = tid; idx < G * HD; idx += NCT) {
        const int g = idx / HD, i = idx - g * HD;
        float ms = -INFINITY;
        for (long long c = ca; c <= cb; ++c) {
          const int slot = (prefix[p] < cta_begin(c, Ttot, NC)) ? 0 : 1;
          const float* pc = part + ((size_t)c * 2 + slot) * PSTRIDE;
          ms = fmaxf(ms, __ldcg(pc + G * HD + g));
        }
        float L = 0.f, O = 0.f;
        for (long long c = ca; c <= cb; ++c) {
          const int slot = (prefix[p] < cta_begin(c, Ttot, NC)) ? 0 : 1;
          const float* pc = part + ((size_t)c * 2 + slot) * PSTRIDE;
          const float mc = __ldcg(pc + G * HD + g);
          const float f = (mc == -INFINITY) ? 0.f : exp2f(mc - ms);
          L = fmaf(__ldcg(pc + G * HD + G + g), f, L);
          O = fmaf(__ldcg(pc + g * HD + i), f, O);
        }
        out[((size_t)p * G + g) * HD + i] = O / L;
      }
    }
  }
  sync();
}

}  // namespace kvpop
