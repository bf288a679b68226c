// One decode step in one kernel (bf16 K/V, d = 128): the pieces that the
// tensor-core attention kernel adds when it also ingests the new token.
//
// Which keys can change during a step is known before the step: when the
// token u = p - D leaves the window (Sec. 3.1, Eq. 4) it either takes the next
// free slot (fewer than B used) or is compared with the lowest-priority slot c
// (the cached argmin), and the new token p takes u's window row (Sec. 3.2,
// App. C.1).  Every other resident key is fixed.  So the attention streams the
// fixed keys at once -- slot c and the leaving row masked out -- while four
// extra warps per CTA run the delayed scorer (Sec. 3.3, App. E.4) on scorer
// units of 16 sequences of one KV head, keep-or-drop, scatter and the window
// update.  Each (sequence, KV head) pair counts arrivals: one per CTA that
// streamed part of it, plus one for its scorer.  The last arrival merges the
// partials and the two keys that changed (the new token's window row and
// slot c, whatever it holds after the decision; the scorer records their logits
// and V rows) into the output, then commits the pair's new length, used-slot
// count and minimum.  Those three wait in a side buffer until then because every
// CTA reads the old values for its schedule and its tiles; a grid-wide counter
// makes sure no CTA is still building its schedule when the first commit lands.
#pragma once

#include "kvpop_argmin.cuh"
#include "kvpop_sched.cuh"

namespace kvpop {

constexpr int kFusedSeqs = 16;     // sequences per scorer unit (the MMA's M)
constexpr int kFusedSW = 4;        // scorer warps per CTA
constexpr int kFusedMaxBlkLanes = 4;   // block minima held per lane (B <= 8192 slots)

struct FusedArgs {
  State st;
  const bf16* k_new;               // [b][H][d]
  const bf16* v_new;
  const float* override_;          // [b][H] or null
  int32_t* evict_info;             // [b][H][2] or null
  float* score_out;                // [b][H] or null
  float* part_c;                   // [pairs][G d + 2 G]: partial of a pair streamed by one CTA
  int32_t* meta_next;              // [pairs][4]: length, used slots, min priority (bits), min slot
  float* xtra;                     // [pairs][2 G + 2 d]: logits of the two changed keys per head
                                   // (log2 domain, -inf when absent), then their V rows
  unsigned long long* ctr;         // CTAs past their schedule, counted over all launches
  int2* start_prev;                // [grid] (pair, tile of the pair) each CTA's range began
                                   // with in the last launch
  int batch, H, F, Fp, s, act;   // Fp: W1 / b1 / w2 row length (F rounded up to 4)
};

constexpr int kMaxSplit = 256;     // CTAs of the fused grid the boundary table holds

// Smem of the scorer role, after the schedule prefix (byte offsets from its start).
struct FusedSmem {
  static constexpr int XS = 3 * 128 + 4;                 // input row stride (floats)
  static constexpr int X = 0;                            // [16][XS] fp32 scorer inputs
  static constexpr int RP = X + kFusedSeqs * XS * 4;     // [4][16] per-warp output partials
  static constexpr int SEQ = RP + kFusedSW * kFusedSeqs * 4;   // [4][16] len, nvalid, min, min slot
  static constexpr int SXC = SEQ + 4 * kFusedSeqs * 4;   // [4][2] extra-key logits (consumers)
  static constexpr int SXS = SXC + 32;                   // (spare)
  static constexpr int FLAG = SXS + kFusedSW * 32;       // [0] int: every CTA's schedule built;
                                                         // [8] u64: the count that means it
  static constexpr int BND = FLAG + 16;                  // [kMaxSplit + 1] ints: CTA ranges
  static constexpr int WBAR = BND + (kMaxSplit + 1) * 4 + 4;   // [3] mbarriers of the weight ring
  static constexpr int W1R = (WBAR + 24 + 127) & ~127;   // [3][kW1Rows][Fp] weight ring
  static constexpr int TOTAL_FIXED = W1R;                // + 3 kW1Rows Fp 4 bytes
};
constexpr int kW1Rows = 16;        // W1 rows per stage of the weight ring (one bulk copy)
constexpr int kW1Stages = 3;
__host__ __device__ inline size_t fused_smem_bytes(int Fp) {
  return (size_t)FusedSmem::TOTAL_FIXED + (size_t)kW1Stages * kW1Rows * Fp * 4;
}

__device__ __forceinline__ int ld_acquire_gpu(const int32_t* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ unsigned long long ld_acquire_gpu(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.acquire.gpu.global.b64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}
// CTA-scope release / acquire on a shared-memory flag (a fact one warp established
// passed on to the others of the CTA, with its ordering)
__device__ __forceinline__ void st_release_cta(int* p, int v) {
  asm volatile("st.release.cta.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(p)), "r"(v) : "memory");
}
__device__ __forceinline__ int ld_acquire_cta(const int* p) {
  int v;
  asm volatile("ld.acquire.cta.shared::cta.b32 %0, [%1];" : "=r"(v) : "r"(smem_u32(p)) : "memory");
  return v;
}

// The concatenated tile list of all pairs (T tiles) split into contiguous ranges over the
// N streaming CTAs: CTA c takes tiles [bnd[c], bnd[c + 1]).  The boundaries sit in shared
// memory (split_bounds), so a lookup costs a load or two, not a division.
struct Split {
  long long T, N;
  const int* bnd;              // [N + 1] in shared memory
  __device__ __forceinline__ long long begin(long long c) const { return bnd[c]; }
  // the CTA whose range holds tile t
  __device__ __forceinline__ long long of(long long t) const {
    int c = (int)(t * N / T);
    c = c < 0 ? 0 : (c >= (int)N ? (int)N - 1 : c);
    while (c + 1 < (int)N && bnd[c + 1] <= t) ++c;
    while (c > 0 && bnd[c] > t) --c;
    return c;
  }
};

// Boundaries balanced by tiles, except that the first U CTAs -- those running one scorer
// unit more than the rest -- take k/64 less: bnd[c] = T W(c) / W(N), W(c) = 64 c - k min(c, U)
// (U = 0 or k = 0: the even split c T / N).  Written by the NT threads of the block.
__device__ __forceinline__ void split_bounds(int* bnd, long long T, long long N, int U, int k,
                                             int tid, int NT) {
  const long long WN = 64 * N - (long long)k * (N < U ? N : U);
  for (long long c = tid; c <= N; c += NT) {
    const long long wc = 64 * c - (long long)k * (c < U ? c : U);
    bnd[c] = (int)(WN > 0 ? T * wc / WN : 0);
  }
}

// Pair p's contributors: CTAs [ca, cb] of the split (none when it has no tiles).
__device__ __forceinline__ int pair_ctas(int p, const int* prefix, const Split& sp, long long& ca,
                                         long long& cb) {
  if (prefix[p + 1] == prefix[p] || sp.T <= 0) { ca = 0; cb = -1; return 0; }
  ca = sp.of(prefix[p]);
  cb = sp.of(prefix[p + 1] - 1);
  return (int)(cb - ca + 1);
}

// Published partial of contributor CTA c for pair p.
template <int G, int HD>
__device__ __forceinline__ const float* pair_partial(const float* part, const float* part_c, int p,
                                                     const int* prefix, const Split& sp, long long c,
                                                     bool single) {
  constexpr int PSTRIDE = G * HD + 2 * G;
  if (single) return part_c + (size_t)p * PSTRIDE;
  const int slot = (prefix[p] < sp.begin(c)) ? 0 : 1;
  return part + ((size_t)c * 2 + slot) * PSTRIDE;
}

__device__ __forceinline__ void prefetch_l2(const void* p, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}

// Online merge of one more (max, sum, output) part into a running (M, L, O), log2 domain.
__device__ __forceinline__ void merge_part(float& M, float& L, float& O, float m, float l, float o) {
  if (m == -INFINITY) return;
  const float nm = fmaxf(M, m);
  const float fa = (M == -INFINITY) ? 0.f : exp2f(M - nm);
  const float fb = exp2f(m - nm);
  L = L * fa + l * fb;
  O = O * fa + o * fb;
  M = nm;
}

__device__ __forceinline__ void unpack_bf16x8(const uint4& u, float (&x)[8]) {
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
  for (int t = 0; t < 4; ++t) {
    x[2 * t] = __bfloat162float(h[t].x);
    x[2 * t + 1] = __bfloat162float(h[t].y);
  }
}
__device__ __forceinline__ void unpack_bf16x4(const uint2& u, float (&x)[4]) {
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
  x[0] = __bfloat162float(h[0].x);
  x[1] = __bfloat162float(h[0].y);
  x[2] = __bfloat162float(h[1].x);
  x[3] = __bfloat162float(h[1].y);
}

// Final output of pair p, by its last arrival (NTHR threads, `sync` their barrier).
// Combines: the caller's own partial (own_m/l/o, EPT elements per thread, or null), the
// published partials of the other contributors, and the scorer's record of the two keys
// that changed this step.  Then commits the pair's new metadata and re-arms its arrival
// counter.
template <int HD, int G, int NTHR>
struct MergeShape {
  static constexpr int EPT = (G * HD + NTHR - 1) / NTHR;   // output elements per thread
};

template <int HD, int G, int NTHR, typename SyncFn>
__device__ void fused_merge(const FusedArgs& f, float* out, const float* part, int32_t* part_count,
                            int p, const int* prefix, const Split& sp, long long own_cta, const float* own_m, const float* own_l,
                            const float* own_o, int tid, int* sched_seen, SyncFn sync) {
  constexpr int EPT = MergeShape<HD, G, NTHR>::EPT;
  constexpr int NE = G * HD;
  const State& st = f.st;
  // the pair's next length, used slots and minimum: written by the scorer before its
  // arrival, which the caller has acquired, so loaded now beside the partials
  int4 mt = make_int4(0, 0, 0, 0);
  if (tid == 0) mt = __ldcg(reinterpret_cast<const int4*>(f.meta_next) + p);
  long long ca, cb;
  const int nctas = pair_ctas(p, prefix, sp, ca, cb);
  const bool single = (nctas == 1);
  // the two keys that changed this step: the scorer's record of their logits and V rows
  const float* xr = f.xtra + (size_t)p * (2 * G + 2 * HD);
  // output elements idx = tid + k NTHR, in chunks of up to 4 (every load of a chunk and
  // contributor issued together)
  constexpr int CH = EPT < 4 ? EPT : 4;
  for (int k0 = 0; k0 < EPT; k0 += CH) {
    float M[CH], L[CH], O[CH];
#pragma unroll
    for (int u = 0; u < CH; ++u) {
      const int k = k0 + u;
      M[u] = (own_m && k < EPT) ? own_m[k] : -INFINITY;
      L[u] = (own_l && k < EPT) ? own_l[k] : 0.f;
      O[u] = (own_o && k < EPT) ? own_o[k] : 0.f;
    }
    float s0[CH], s1[CH], v0[CH], v1[CH];
#pragma unroll
    for (int u = 0; u < CH; ++u) {
      const int idx = tid + (k0 + u) * NTHR;
      const bool in = k0 + u < EPT && idx < NE;
      const int g = (in ? idx : 0) / HD, i = (in ? idx : 0) % HD;
      s0[u] = in ? __ldcg(xr + 2 * g) : -INFINITY;
      s1[u] = in ? __ldcg(xr + 2 * g + 1) : -INFINITY;
      v0[u] = in ? __ldcg(xr + 2 * G + i) : 0.f;
      v1[u] = in ? __ldcg(xr + 2 * G + HD + i) : 0.f;
    }
    for (long long cc = ca; cc <= cb; ++cc) {
      if (own_m && cc == own_cta) continue;
      const float* pc = pair_partial<G, HD>(part, f.part_c, p, prefix, sp, cc, single);
      float mc[CH], lc[CH], oc[CH];
#pragma unroll
      for (int u = 0; u < CH; ++u) {
        const int idx = tid + (k0 + u) * NTHR;
        const bool in = k0 + u < EPT && idx < NE;
        const int g = (in ? idx : 0) / HD;
        mc[u] = in ? __ldcg(pc + NE + g) : -INFINITY;
        lc[u] = in ? __ldcg(pc + NE + G + g) : 0.f;
        oc[u] = in ? __ldcg(pc + idx) : 0.f;
      }
#pragma unroll
      for (int u = 0; u < CH; ++u) merge_part(M[u], L[u], O[u], mc[u], lc[u], oc[u]);
    }
#pragma unroll
    for (int u = 0; u < CH; ++u) {
      const int idx = tid + (k0 + u) * NTHR;
      if (k0 + u >= EPT || idx >= NE) continue;
      merge_part(M[u], L[u], O[u], s0[u], 1.f, v0[u]);
      merge_part(M[u], L[u], O[u], s1[u], 1.f, v1[u]);
      out[(size_t)p * NE + idx] = O[u] / L[u];
    }
  }
  if (tid == 0) {
    // commit the pair's new length, used slots and minimum -- once no CTA can still be
    // reading lengths for its schedule (every CTA counts itself in after building it);
    // the first merge of this CTA to see that tells the later ones through shared memory
    const unsigned long long target = *reinterpret_cast<const unsigned long long*>(sched_seen + 2);
    bool ready = ld_acquire_cta(sched_seen) != 0;
    if (!ready) ready = ld_acquire_gpu(f.ctr) >= target;
    if (!ready) {
      const unsigned long long t0 = globaltimer();
      while (!(ready = ld_acquire_gpu(f.ctr) >= target))
        if (globaltimer() - t0 > kWaitLimitNs) {
          atomicCAS(st.err, 0, DEVERR_TIMEOUT_SCHED);
          break;
        }
    }
    if (ready) {
      st_release_cta(sched_seen, 1);
      st.len[p] = mt.x;
      st.nvalid[p] = mt.y;
      st.min_score[p] = __int_as_float(mt.z);
      st.min_slot[p] = mt.w;
    }
    part_count[p] = 0;
  }
  sync();
}

// The scorer role: NSW = 4 warps, `stid` in [0, 128).  Units u = blockIdx.x, +gridDim.x, ...
// of (KV head u % H, sequences 16 (u / H) ...): scorer inputs, hidden layer on tensor cores
// (fp32 FMAs), output layer, keep-or-drop, scatter, window update,
// arrival; the pair's merge when the scorer arrives last.  Every stage issues its loads
// together (L2 prefetch of the unit's weights and window rows first), so a unit costs a
// few memory round trips rather than one per value.
template <int HD, int G>
__device__ void fused_scorer(const FusedArgs& f, const bf16* q, float* out, const float* part,
                             int32_t* part_count, const int* prefix, const Split& sp, int D, int B,
                             float qscale, unsigned char* fsm, int stid) {
  static_assert(HD == 128, "the fused step kernel is built for d = 128");
  constexpr int XS = FusedSmem::XS;
  constexpr int I = 3 * HD, K8 = I / 8;
  static_assert(K8 % 2 == 0, "the weight loads alternate between two k-step buffers");
  const State& st = f.st;
  float* X = reinterpret_cast<float*>(fsm + FusedSmem::X);
  float* rp = reinterpret_cast<float*>(fsm + FusedSmem::RP);
  int* s_len = reinterpret_cast<int*>(fsm + FusedSmem::SEQ);
  int* s_nv = s_len + kFusedSeqs;
  float* s_ms = reinterpret_cast<float*>(s_nv + kFusedSeqs);
  int* s_msl = reinterpret_cast<int*>(s_ms + kFusedSeqs);
  const int w = stid >> 5, lane = stid & 31;
  const int H = f.H;
  const int ngroups = (f.batch + kFusedSeqs - 1) / kFusedSeqs;
  const int units = H * ngroups;
  const float inv_g = 1.0f / (float)G;
  auto ssync = [] { asm volatile("bar.sync 2, %0;" ::"r"(kFusedSW * 32) : "memory"); };
  // weight ring: stage k of a unit holds W1 rows [16 k, 16 k + 16) of its head, one bulk
  // copy; stage buffers rotate over the units of this CTA (n-th use of a buffer: parity n & 1)
  constexpr int NSTAGE = I / kW1Rows;
  static_assert(NSTAGE % kW1Stages == 0, "each unit uses every ring buffer equally often");
  uint64_t* wbar = reinterpret_cast<uint64_t*>(fsm + FusedSmem::WBAR);
  float* w1r = reinterpret_cast<float*>(fsm + FusedSmem::W1R);
  const uint32_t stage_bytes = (uint32_t)(kW1Rows * f.Fp * 4);
  if (stid == 0) {
    for (int k = 0; k < kW1Stages; ++k) mbar_init(smem_u32(&wbar[k]), 1);
    mbar_fence_init();
  }
  ssync();
  long long issued = 0, consumed = 0;   // stage copies issued / waited for by this CTA
  auto issue_w1 = [&](const float* w1h, int k) {
    const int buf = (int)(issued % kW1Stages);
    const uint32_t bar = smem_u32(&wbar[buf]);
    mbar_arrive_expect_tx(bar, stage_bytes);
    bulk_g2s(smem_u32(w1r + (size_t)buf * kW1Rows * f.Fp), w1h + (size_t)k * kW1Rows * f.Fp,
             stage_bytes, bar);
    ++issued;
  };

  for (int unit = blockIdx.x; unit < units; unit += gridDim.x) {
    const int h = unit % H, grp = unit / H;
    const int b0 = grp * kFusedSeqs;
    const float* w1h = st.W1 + (size_t)h * I * f.Fp;
    // ---- the first stages of this head's weights into the ring (the previous unit is done
    // with it), and an L2 prefetch of the window query means of the unit's sequences
    if (stid == 0)
      for (int k = 0; k < kW1Stages && k < NSTAGE; ++k) issue_w1(w1h, k);
    if (lane < kFusedSeqs / kFusedSW) {
      const int j = w * (kFusedSeqs / kFusedSW) + lane;
      if (b0 + j < f.batch)
        prefetch_l2(st.ringQm + (size_t)((b0 + j) * H + h) * D * HD, (uint32_t)(D * HD * 4));
    }
    if (stid < kFusedSeqs) {
      const int b = b0 + stid;
      if (b < f.batch) {
        const int pair = b * H + h;
        s_len[stid] = st.len[pair];
        s_nv[stid] = st.nvalid[pair];
        s_ms[stid] = st.min_score[pair];
        s_msl[stid] = st.min_slot[pair];
      } else {
        s_len[stid] = -1;
      }
    }
    ssync();
    // ---- scorer inputs x = [k_u; v_u; qbar_u], warp w rows w, w + 4, ... (zero if none)
    for (int r = 0; r < kFusedSeqs / kFusedSW; ++r) {
      const int j = w + kFusedSW * r;
      const int b = b0 + j;
      const int plen = s_len[j];
      float* xr = X + j * XS;
      if (!(b < f.batch && plen >= D)) {
        for (int e = lane; e < I; e += 32) xr[e] = 0.f;
        continue;
      }
      const int pair = b * H + h;
      const int ri = plen % D;
      // K (lanes 0-15) or V (16-31) row chunk of u, q channels 4 lane .. 4 lane + 3
      const uint4 kv = reinterpret_cast<const uint4*>(
          static_cast<const bf16*>(lane < 16 ? st.ringK : st.ringV) + ((size_t)pair * D + ri) * HD)[lane & 15];
      uint2 qv[G];
#pragma unroll
      for (int g = 0; g < G; ++g)
        qv[g] = reinterpret_cast<const uint2*>(q + ((size_t)pair * G + g) * HD)[lane];
      // window query means of u + 1 .. p - 1, summed in position order
      const float4* qm4 = reinterpret_cast<const float4*>(st.ringQm + (size_t)pair * D * HD) + lane;
      float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
      for (int jb = 1; jb < D; jb += 8) {
        float4 buf[8];
#pragma unroll
        for (int t = 0; t < 8; ++t) {
          const int jj = jb + t;
          if (jj < D) {
            int rr = ri + jj;
            rr = rr >= D ? rr - D : rr;
            buf[t] = qm4[(size_t)rr * (HD / 4)];
          }
        }
#pragma unroll
        for (int t = 0; t < 8; ++t)
          if (jb + t < D) { a0 += buf[t].x; a1 += buf[t].y; a2 += buf[t].z; a3 += buf[t].w; }
      }
      float qs[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int g = 0; g < G; ++g) {
        float qf[4];
        unpack_bf16x4(qv[g], qf);
#pragma unroll
        for (int t = 0; t < 4; ++t) qs[t] += qf[t];
      }
      a0 += qs[0] * inv_g; a1 += qs[1] * inv_g; a2 += qs[2] * inv_g; a3 += qs[3] * inv_g;
      float* xq = xr + 2 * HD + 4 * lane;
      xq[0] = a0 / (float)D; xq[1] = a1 / (float)D; xq[2] = a2 / (float)D; xq[3] = a3 / (float)D;
      float kvf[8];
      unpack_bf16x8(kv, kvf);
      float* xk = xr + (lane < 16 ? 0 : HD) + 8 * (lane & 15);
#pragma unroll
      for (int t = 0; t < 8; ++t) xk[t] = kvf[t];
    }
    ssync();
    // ---- hidden layer in fp32 FMAs: thread (half, fq) accumulates hidden units
    // 4 fq .. 4 fq + 3 of sequences 8 half .. 8 half + 7 over the 3d inputs in order
    // (W1 rows read as float4, one k-row of 4 inputs ahead)
    {
      const int half = stid >> 6, fq = stid & 63;
      const bool act_f = 4 * fq < f.F;          // threads past F compute a copy, unused
      float acc[8][4];
#pragma unroll
      for (int sq = 0; sq < 8; ++sq)
#pragma unroll
        for (int e = 0; e < 4; ++e) acc[sq][e] = 0.f;
      const int FP4 = f.Fp / 4;
      const float4* xb = reinterpret_cast<const float4*>(X) + (size_t)(8 * half) * (XS / 4);
      for (int k = 0; k < NSTAGE; ++k) {
        const int buf = (int)(consumed % kW1Stages);
        const uint32_t par = (uint32_t)((consumed / kW1Stages) & 1);
        mbar_wait(smem_u32(&wbar[buf]), par, st.err, DEVERR_TIMEOUT_FULL);
        ++consumed;
        const float4* wst = reinterpret_cast<const float4*>(w1r + (size_t)buf * kW1Rows * f.Fp) + (act_f ? fq : 0);
#pragma unroll
        for (int i4 = 0; i4 < kW1Rows / 4; ++i4) {
          float4 wc[4];
#pragma unroll
          for (int t = 0; t < 4; ++t) wc[t] = wst[(size_t)(4 * i4 + t) * FP4];
#pragma unroll
          for (int sq = 0; sq < 8; ++sq) {
            const float4 x = xb[(size_t)sq * (XS / 4) + k * (kW1Rows / 4) + i4];
            const float xv[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
            for (int t = 0; t < 4; ++t) {
              acc[sq][0] = fmaf(xv[t], wc[t].x, acc[sq][0]);
              acc[sq][1] = fmaf(xv[t], wc[t].y, acc[sq][1]);
              acc[sq][2] = fmaf(xv[t], wc[t].z, acc[sq][2]);
              acc[sq][3] = fmaf(xv[t], wc[t].w, acc[sq][3]);
            }
          }
        }
        ssync();                                  // every warp is done with this stage
        if (stid == 0 && k + kW1Stages < NSTAGE) issue_w1(w1h, k + kW1Stages);
      }
      // ---- output layer: this thread's 4 units, then the sum over the half's 64 threads
      float rs[8];
      const float* b1 = st.b1 + (size_t)h * f.Fp + 4 * fq;
      const float* w2 = st.w2 + (size_t)h * f.Fp + 4 * fq;
      float bb[4] = {0.f, 0.f, 0.f, 0.f}, ww[4] = {0.f, 0.f, 0.f, 0.f};
      if (act_f) {
#pragma unroll
        for (int e = 0; e < 4; ++e) { bb[e] = b1[e]; ww[e] = w2[e]; }
      }
#pragma unroll
      for (int sq = 0; sq < 8; ++sq) {
        float r = 0.f;
        if (act_f) {
#pragma unroll
          for (int e = 0; e < 4; ++e) r = fmaf(ww[e], scorer_act(acc[sq][e] + bb[e], f.act), r);
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) r += __shfl_xor_sync(0xffffffffu, r, off);
        rs[sq] = r;
      }
      if (lane == 0) {
#pragma unroll
        for (int sq = 0; sq < 8; ++sq) rp[w * 8 + sq] = rs[sq];   // warp w: sequences 8 (w / 2) + sq
      }
    }
    ssync();
    // ---- keep-or-drop, scatter and window update: warp w takes sequences w, w + 4, ...
    const int NB = min_blocks(B);
    const int nbl = (NB + 31) / 32;
    const bool reg_min = nbl <= kFusedMaxBlkLanes;
    for (int r = 0; r < kFusedSeqs / kFusedSW; ++r) {
      const int j = w + kFusedSW * r;
      const int b = b0 + j;
      if (b >= f.batch) continue;
      const int pair = b * H + h;
      const int plen = s_len[j];
      const int nv = s_nv[j];
      const float mn = s_ms[j];
      const int mni = s_msl[j];
      float* sc = st.score + (size_t)pair * B;
      int32_t* ps = st.pos + (size_t)pair * B;
      float* bsc = st.blk_score + (size_t)pair * NB;
      int32_t* bsl = st.blk_slot + (size_t)pair * NB;
      // every load of this pair at once: the state a replacement touches (the cached
      // minimum's block of 64 priorities, the block minima, the position it holds), the
      // new token's K / V chunk and its queries
      const bool may_replace = plen >= D && nv >= B && mni >= f.s && mni < B && reg_min;
      float blk[2] = {INFINITY, INFINITY};
      float nbv[kFusedMaxBlkLanes];
      int nbs[kFusedMaxBlkLanes];
      int ev_pos = -1;
#pragma unroll
      for (int t = 0; t < kFusedMaxBlkLanes; ++t) { nbv[t] = INFINITY; nbs[t] = 0x7fffffff; }
      if (may_replace) {
        const int lo = (mni / kMinBlock) * kMinBlock;
        blk[0] = (lo + lane < B) ? sc[lo + lane] : INFINITY;
        blk[1] = (lo + 32 + lane < B) ? sc[lo + 32 + lane] : INFINITY;
        ev_pos = ps[mni];
#pragma unroll
        for (int t = 0; t < kFusedMaxBlkLanes; ++t) {
          const int k = lane + 32 * t;
          if (t < nbl && k < NB) { nbv[t] = bsc[k]; nbs[t] = bsl[k]; }
        }
      }
      const uint4 kvn = reinterpret_cast<const uint4*>((lane < 16 ? f.k_new : f.v_new) + (size_t)pair * HD)[lane & 15];
      uint2 qv[G];
#pragma unroll
      for (int g = 0; g < G; ++g)
        qv[g] = reinterpret_cast<const uint2*>(q + ((size_t)pair * G + g) * HD)[lane];
      // channels 4 lane .. 4 lane + 3 of the new token's K / V and, when it may stay (full
      // cache), of the lowest-priority slot's
      const uint2 kn4 = reinterpret_cast<const uint2*>(f.k_new + (size_t)pair * HD)[lane];
      const uint2 vn4 = reinterpret_cast<const uint2*>(f.v_new + (size_t)pair * HD)[lane];
      uint2 ke4 = make_uint2(0u, 0u), ve4 = make_uint2(0u, 0u);
      if (plen >= D && nv >= B && mni >= 0 && mni < B) {
        ke4 = reinterpret_cast<const uint2*>(static_cast<const bf16*>(st.slotK) + ((size_t)pair * B + mni) * HD)[lane];
        ve4 = reinterpret_cast<const uint2*>(static_cast<const bf16*>(st.slotV) + ((size_t)pair * B + mni) * HD)[lane];
      }
      int slot = -1, evicted = -1, nv_post = nv;
      float r_out = __int_as_float(0x7fc00000);
      float mn_post = mn;
      int mni_post = mni;
      bool min_written = false;
      if (plen >= D) {
        const int hw = 2 * (j >> 3), sq = j & 7;
        float rr = rp[hw * 8 + sq] + rp[(hw + 1) * 8 + sq];
        rr += st.b2[h];
        if (f.override_) rr = f.override_[pair];
        rr = canon_score(rr);
        r_out = rr;
        const int u = plen - D;
        const float prio = static_priority(rr, u, st.log_gamma, h);
        if (nv < B) {
          slot = nv;
        } else if (prio > mn) {
          slot = mni;
          if (!dcheck(slot >= f.s && slot < B, st.err, DEVERR_INDEX)) slot = -1;
          else evicted = may_replace ? ev_pos : ps[slot];
        }
        if (slot >= 0 && !dcheck(nv >= 0, st.err, DEVERR_INDEX)) slot = -1;
        if (slot >= 0) {
          // u's K / V (the scorer input row, exact bf16 values) into the slot
          {
            const float* xs = X + j * XS + (lane < 16 ? 0 : HD) + 8 * (lane & 15);
            uint4 row;
            __nv_bfloat162* rh = reinterpret_cast<__nv_bfloat162*>(&row);
#pragma unroll
            for (int t = 0; t < 4; ++t) rh[t] = __floats2bfloat162_rn(xs[2 * t], xs[2 * t + 1]);
            bf16* dst = static_cast<bf16*>(lane < 16 ? st.slotK : st.slotV) + ((size_t)pair * B + slot) * HD;
            reinterpret_cast<uint4*>(dst)[lane & 15] = row;
          }
          if (nv == B && may_replace) {
            // the replaced slot's block from the loaded priorities, then the head minimum
            const int k = slot / kMinBlock, lo = k * kMinBlock;
            float bm = INFINITY;
            int bmi = 0x7fffffff;
#pragma unroll
            for (int r2 = 0; r2 < 2; ++r2) {
              const int i = lo + r2 * 32 + lane;
              if (i < B && i >= f.s) lex_min(bm, bmi, i == slot ? prio : blk[r2], i);
            }
            warp_lex_min(bm, bmi);
            float m = INFINITY;
            int mi = 0x7fffffff;
#pragma unroll
            for (int t = 0; t < kFusedMaxBlkLanes; ++t) {
              const int kk = lane + 32 * t;
              if (t < nbl && kk < NB) {
                if (kk == k) lex_min(m, mi, bm, bmi);
                else lex_min(m, mi, nbv[t], nbs[t]);
              }
            }
            warp_lex_min(m, mi);
            if (lane == 0) { bsc[k] = bm; bsl[k] = bmi; }
            mn_post = m;
            mni_post = mi;
          } else if (nv == B) {
            float* ms_out = reinterpret_cast<float*>(f.meta_next + (size_t)pair * 4 + 2);
            update_min(sc, f.s, B, slot, prio, bsc, bsl, ms_out, f.meta_next + (size_t)pair * 4 + 3);
            min_written = true;
          } else if (nv + 1 == B) {
            float* ms_out = reinterpret_cast<float*>(f.meta_next + (size_t)pair * 4 + 2);
            rebuild_min(sc, f.s, B, slot, prio, bsc, bsl, ms_out, f.meta_next + (size_t)pair * 4 + 3);
            min_written = true;
          }
          __syncwarp();
          if (lane == 0) {
            sc[slot] = prio;
            ps[slot] = u;
          }
          nv_post = nv < B ? nv + 1 : nv;
        }
      }
      // the new token into the window row it frees (u's row, consumed above)
      {
        const int ri = (plen >= 0 ? plen : 0) % D;
        bf16* dst = static_cast<bf16*>(lane < 16 ? st.ringK : st.ringV) + ((size_t)pair * D + ri) * HD;
        reinterpret_cast<uint4*>(dst)[lane & 15] = kvn;
        float qs[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int g = 0; g < G; ++g) {
          float qf[4];
          unpack_bf16x4(qv[g], qf);
#pragma unroll
          for (int t = 0; t < 4; ++t) qs[t] += qf[t];
        }
        reinterpret_cast<float4*>(st.ringQm + ((size_t)pair * D + ri) * HD)[lane] =
            make_float4(qs[0] * inv_g, qs[1] * inv_g, qs[2] * inv_g, qs[3] * inv_g);
      }
      // the record of the two keys that changed: the new token (window row) and what the
      // slot that could change holds after the decision (u, or the kept lowest-priority key)
      {
        const bool has1 = plen >= D && (slot >= 0 || (nv >= B && mni >= 0 && mni < B));
        float k0f[4], v0f[4], k1f[4] = {0.f, 0.f, 0.f, 0.f}, v1f[4] = {0.f, 0.f, 0.f, 0.f};
        unpack_bf16x4(kn4, k0f);
        unpack_bf16x4(vn4, v0f);
        if (slot >= 0) {
          const float* xu = X + j * XS;
#pragma unroll
          for (int t = 0; t < 4; ++t) { k1f[t] = xu[4 * lane + t]; v1f[t] = xu[HD + 4 * lane + t]; }
        } else if (has1) {
          unpack_bf16x4(ke4, k1f);
          unpack_bf16x4(ve4, v1f);
        }
        float* xr = f.xtra + (size_t)pair * (2 * G + 2 * HD);
#pragma unroll
        for (int g = 0; g < G; ++g) {
          float qf[4];
          unpack_bf16x4(qv[g], qf);
          float d0 = 0.f, d1 = 0.f;
#pragma unroll
          for (int t = 0; t < 4; ++t) { d0 = fmaf(qf[t], k0f[t], d0); d1 = fmaf(qf[t], k1f[t], d1); }
#pragma unroll
          for (int off = 16; off > 0; off >>= 1) {
            d0 += __shfl_xor_sync(0xffffffffu, d0, off);
            d1 += __shfl_xor_sync(0xffffffffu, d1, off);
          }
          if (lane == 0) {
            xr[2 * g] = d0 * qscale;
            xr[2 * g + 1] = has1 ? d1 * qscale : -INFINITY;
          }
        }
        reinterpret_cast<float4*>(xr + 2 * G)[lane] = make_float4(v0f[0], v0f[1], v0f[2], v0f[3]);
        reinterpret_cast<float4*>(xr + 2 * G + HD)[lane] = make_float4(v1f[0], v1f[1], v1f[2], v1f[3]);
      }
      if (lane == 0) {
        int32_t* mt = f.meta_next + (size_t)pair * 4;
        mt[0] = plen + 1;
        mt[1] = nv_post;
        if (!min_written) { mt[2] = __float_as_int(mn_post); mt[3] = mni_post; }
        if (f.evict_info) { f.evict_info[2 * pair] = slot; f.evict_info[2 * pair + 1] = evicted; }
        if (f.score_out) f.score_out[pair] = r_out;
      }
    }
    // ---- arrivals of the warp's pairs (publish, then count in); the last arrival merges
    __threadfence();
    __syncwarp();
    int last = 0;
    if (lane < kFusedSeqs / kFusedSW) {
      const int b = b0 + w + kFusedSW * lane;
      if (b < f.batch) {
        const int pair = b * H + h;
        long long ca, cb;
        const int nctas = pair_ctas(pair, prefix, sp, ca, cb);
        last = atomicAdd(part_count + pair, 1) == nctas;
      }
    }
    const unsigned lm = __ballot_sync(0xffffffffu, last);
    if (lm) __threadfence();
    for (int r = 0; r < kFusedSeqs / kFusedSW; ++r) {
      if (!((lm >> r) & 1u)) continue;
      const int pair = (b0 + w + kFusedSW * r) * H + h;
      fused_merge<HD, G, 32>(f, out, part, part_count, pair, prefix, sp, -1, nullptr, nullptr,
                             nullptr, lane, reinterpret_cast<int*>(fsm + FusedSmem::FLAG),
                             [] { __syncwarp(); });
    }
    ssync();   // X and the per-sequence state are reused by the next unit
  }
  // a wait that gave up leaves copies in flight: let them land before the CTA exits
  if (stid == 0)
    for (long long k = consumed; k < issued; ++k)
      if (!mbar_wait(smem_u32(&wbar[k % kW1Stages]), (uint32_t)((k / kW1Stages) & 1), st.err,
                     DEVERR_TIMEOUT_DRAIN))
        break;
}

}  // namespace kvpop
