// Keep-or-drop and scatter for one (sequence, KV head), warp-collective.
//
// Running top-k under the budget (Sec. 3.2, App. C.1): the token u that left the
// window takes the next free slot while fewer than B are used; afterwards it
// replaces the lowest-priority long-range slot (ties -> lowest slot index)
// iff its static priority (App. B.3) is strictly larger, else it is dropped.
#pragma once

#include "kvpop_argmin.cuh"

namespace kvpop {

// r is the raw score of u = p - D (already overridden if requested); k_u, v_u
// point at u's K/V row (any memory space readable by the warp).
template <typename T>
__device__ __forceinline__ void evict_and_scatter(const State& st, const Dims& dm, int pair, int h,
                                                  int p, float r, const T* k_u, const T* v_u,
                                                  int32_t* evict_info, float* score_out) {
  const int lane = threadIdx.x & 31;
  const int B = dm.B, d = dm.d;
  r = canon_score(r);
  const int u = p - dm.D;
  const float prio = static_priority(r, u, st.log_gamma, h);
  float* sc = st.score + (size_t)pair * B;
  int32_t* ps = st.pos + (size_t)pair * B;
  const int NB = min_blocks(B);
  float* bsc = st.blk_score + (size_t)pair * NB;
  int32_t* bsl = st.blk_slot + (size_t)pair * NB;
  const int nv = st.nvalid[pair];
  int slot = -1, evicted = -1;
  if (nv < B) {
    slot = nv;
  } else if (prio > st.min_score[pair]) {
    slot = st.min_slot[pair];
    if (!dcheck(slot >= dm.s && slot < B, st.err, DEVERR_INDEX)) slot = -1;
    else evicted = ps[slot];
  }
  if (slot >= 0 && !dcheck(nv >= 0, st.err, DEVERR_INDEX)) slot = -1;
  if (slot >= 0) {
    T* dk = static_cast<T*>(st.slotK) + ((size_t)pair * B + slot) * d;
    T* dv = static_cast<T*>(st.slotV) + ((size_t)pair * B + slot) * d;
    for (int i = lane; i < d; i += 32) {
      dk[i] = k_u[i];
      dv[i] = v_u[i];
    }
    if (nv == B)
      update_min(sc, dm.s, B, slot, prio, bsc, bsl, st.min_score + pair, st.min_slot + pair);
    else if (nv + 1 == B)
      rebuild_min(sc, dm.s, B, slot, prio, bsc, bsl, st.min_score + pair, st.min_slot + pair);
    if (lane == 0) {
      sc[slot] = prio;
      ps[slot] = u;
      st.nvalid[pair] = nv < B ? nv + 1 : nv;
    }
  }
  if (lane == 0) {
    st.len[pair] = p + 1;
    if (evict_info) { evict_info[2 * pair] = slot; evict_info[2 * pair + 1] = evicted; }
    if (score_out) score_out[pair] = r;
  }
}

}  // namespace kvpop
