// Shared pieces of the prompt attention kernels (App. C.1 mask, App. C.3):
// arguments, the running top-k mask predicate and the per-tile key lists.
#pragma once

#include <climits>

#include "kvpop_internal.cuh"

namespace kvpop {
namespace prompt {

constexpr float kLn2 = 0.69314718055994530942f;

struct PromptArgs {
  const void* Q;             // [n_seq][H*G][S][d]
  const void* K;             // [n_seq][H][S][d]
  const void* V;
  const int32_t* rank;       // [n_seq*H][S]
  const int32_t* tau;        // [n_seq*H][S]
  const int32_t* order;      // [n_seq*H][S] position of each rank, or nullptr
  const int32_t* len;        // [n_seq] or nullptr (= S)
  float* Y;                  // [n_seq][H*G][S][d]
  float* lse;                // [n_seq][H*G][S] or nullptr
  int H, G, S, s, w;
  int capA, capM;
  float qscale;              // log2(e) / sqrt(d)
  int32_t* err;              // first-error word or nullptr
};

enum : int { PERR_LIST_OVERFLOW = 11 };

__device__ __forceinline__ void note_err(int32_t* err, int code) {
  if (err) atomicCAS(err, 0, code);
}

__device__ __forceinline__ bool keep_key(int q, int t, int r, int tq, int s, int w) {
  return t <= q && (t < s || q - t < w || (t <= q - w && r <= tq));
}

// Shared prologue: tile bounds, per-query cutoffs, cutoff range, key lists.
struct TileInfo {
  int seq, h, pair, q0, q1, L;
  int nA, nM;
};

template <int NT>
__device__ bool tile_setup(const PromptArgs& a, int BM, int* tauS, int* red, int32_t* posA,
                           int32_t* posM, TileInfo& ti) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  constexpr int NW = NT / 32;
  ti.pair = blockIdx.y;
  ti.seq = ti.pair / a.H;
  ti.h = ti.pair - ti.seq * a.H;
  ti.L = a.len ? max(0, min(a.len[ti.seq], a.S)) : a.S;
  ti.q0 = (gridDim.x - 1 - blockIdx.x) * BM;        // longest tiles first
  if (ti.q0 >= ti.L) return false;
  ti.q1 = min(ti.q0 + BM - 1, ti.L - 1);
  const int nq = ti.q1 - ti.q0 + 1;
  const int32_t* tau = a.tau + (size_t)ti.pair * a.S;
  const int32_t* rank = a.rank + (size_t)ti.pair * a.S;
  for (int i = tid; i < BM; i += NT) tauS[i] = i < nq ? tau[ti.q0 + i] : -1;
  __syncthreads();
  if (warp == 0) {
    int mn = INT_MAX, mx = INT_MIN;
    for (int i = lane; i < nq; i += 32) {
      mn = min(mn, tauS[i]);
      mx = max(mx, tauS[i]);
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) {
      mn = min(mn, __shfl_xor_sync(0xffffffffu, mn, o));
      mx = max(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    }
    if (lane == 0) {
      red[NW] = mn;
      red[NW + 1] = mx;
    }
  }
  __syncthreads();
  const int tmin = red[NW], tmax = red[NW + 1];
  const int s = a.s, w = a.w, q0 = ti.q0, q1 = ti.q1;
  // sinks
  const int nAs = min(s, q0 + 1);
  const int nMs = max(0, min(s, q1 + 1) - nAs);
  for (int t = tid; t < nAs && t < a.capA; t += NT) posA[t] = t;
  for (int j = tid; j < nMs && j < a.capM; j += NT) posM[j] = nAs + j;
  int nA = nAs, nM = nMs;
  // eligible for the whole tile: t in [s, q0 - w].  The candidates are the eligible
  // positions ranked within tmax: walk either the positions s .. hi (reading their ranks)
  // or, when it is shorter, the ranks 0 .. tmax (reading their positions, kept if eligible).
  const int hi = q0 - w;
  constexpr int EPT = 16;
  if (hi >= s && tmax >= 0) {
    const int32_t* order = a.order ? a.order + (size_t)ti.pair * a.S : nullptr;
    const bool by_rank = order != nullptr && tmax < hi - s;
    const int n_walk = by_rank ? tmax + 1 : hi - s + 1;
    for (int c0 = 0; c0 < n_walk; c0 += NT * EPT) {
      const int i0 = c0 + tid * EPT;
      int r[EPT], t[EPT];
#pragma unroll
      for (int e = 0; e < EPT; ++e) {
        const int i = i0 + e;
        if (i >= n_walk) {
          r[e] = INT_MAX;
          t[e] = 0;
        } else if (by_rank) {
          t[e] = __ldg(order + i);
          r[e] = (t[e] >= s && t[e] <= hi) ? i : INT_MAX;
        } else {
          t[e] = s + i;
          r[e] = __ldg(rank + s + i);
        }
      }
      int ca = 0, cm = 0;
#pragma unroll
      for (int e = 0; e < EPT; ++e) {
        ca += r[e] <= tmin;
        cm += (r[e] > tmin) & (r[e] <= tmax);
      }
      static_assert(NT * EPT < 65536, "two 16-bit counts per word");
      const int v = ca | (cm << 16);        // at most NT * EPT per field
      int x = v;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
      }
      if (lane == 31) red[warp] = x;
      __syncthreads();
      int off = 0, tot = 0;
#pragma unroll
      for (int i = 0; i < NW; ++i) {
        const int y = red[i];
        if (i < warp) off += y;
        tot += y;
      }
      const int ex = off + x - v;
      int ia = nA + (ex & 0xffff), im = nM + (ex >> 16);
#pragma unroll
      for (int e = 0; e < EPT; ++e) {
        if (r[e] <= tmin) {
          if (ia < a.capA) posA[ia] = t[e];
          ++ia;
        } else if (r[e] <= tmax) {
          if (im < a.capM) posM[im] = t[e];
          ++im;
        }
      }
      nA += tot & 0xffff;
      nM += tot >> 16;
      __syncthreads();
    }
  }
  // window and newly eligible positions
  const int c_lo = max(s, q0 - w + 1);
  for (int t = c_lo + tid; t <= q1; t += NT) {
    const int j = nM + (t - c_lo);
    if (j < a.capM) posM[j] = t;
  }
  if (q1 >= c_lo) nM += q1 - c_lo + 1;
  if (nA > a.capA || nM > a.capM) {
    if (tid == 0) note_err(a.err, PERR_LIST_OVERFLOW);
    nA = min(nA, a.capA);
    nM = min(nM, a.capM);
  }
  ti.nA = nA;
  ti.nM = nM;
  __syncthreads();
  return true;
}

// Dense causal tiles (no mask beyond causality): keys 0 .. q0 serve every query
// of the tile (list A), q0 + 1 .. q1 only the later ones (list M); a key's
// list index is its position.
__device__ __forceinline__ bool dense_setup(const PromptArgs& a, int BM, TileInfo& ti) {
  ti.pair = blockIdx.y;
  ti.seq = ti.pair / a.H;
  ti.h = ti.pair - ti.seq * a.H;
  ti.L = a.len ? max(0, min(a.len[ti.seq], a.S)) : a.S;
  ti.q0 = (gridDim.x - 1 - blockIdx.x) * BM;
  if (ti.q0 >= ti.L) return false;
  ti.q1 = min(ti.q0 + BM - 1, ti.L - 1);
  ti.nA = ti.q0 + 1;
  ti.nM = ti.q1 - ti.q0;
  return true;
}

}  // namespace prompt
}  // namespace kvpop
