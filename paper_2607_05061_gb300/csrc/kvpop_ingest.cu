// Decode steps 1-4: ingest the new token, run the delayed scorer on the token
// that leaves the window, keep or drop it under the fixed budget, scatter it.
//
// One CTA owns one KV head h and SB consecutive sequences, so the head's scorer
// weights W1 [3d][F] are read once per SB sequences.  Warp i of the CTA handles
// sequence i of the group for the per-sequence work (window ring, eviction).
//
// Paper correspondence: eligible set and the newly eligible token u = p - w
// (Sec. 3.1, Eq. 4); delayed scoring (Sec. 3.3, App. E.4) with the stateless
// MLP of Sec. 3.3 / App. E.2 on [k_u; v_u; qbar_u]; static priority
// (App. B.3); running top-k under the budget (Sec. 3.2, App. C.1).
#include "kvpop_internal.cuh"

namespace kvpop {
namespace {

constexpr int SB = 8;          // sequences per CTA (one warp each)
constexpr int NT = 256;        // threads per CTA

template <typename T>
struct IngestArgs {
  State st;
  Dims dm;
  const T* q;                  // [b][H*G][d]
  const T* k;                  // [b][H][d]
  const T* v;
  const float* override_;      // [b][H] or nullptr
  int32_t* evict_info;         // [b][H][2] or nullptr
  float* score_out;            // [b][H] or nullptr
};

// Lowest-priority slot over [s, B), ties -> lowest index.  The value of slot
// `j_new` is taken as `v_new` (it was just written by this warp).
__device__ __forceinline__ void warp_argmin(const float* __restrict__ sc, int s, int B,
                                            int j_new, float v_new, float& mval, int& midx) {
  const int lane = threadIdx.x & 31;
  float best = INFINITY;
  int bi = 0x7fffffff;
  for (int i = s + lane; i < B; i += 32) {
    float x = (i == j_new) ? v_new : sc[i];
    if (bi == 0x7fffffff || x < best) { best = x; bi = i; }
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    float ob = __shfl_xor_sync(0xffffffffu, best, off);
    int oi = __shfl_xor_sync(0xffffffffu, bi, off);
    if (oi != 0x7fffffff && (bi == 0x7fffffff || ob < best || (ob == best && oi < bi))) {
      best = ob;
      bi = oi;
    }
  }
  mval = best;
  midx = bi;
}

template <typename T>
__global__ void __launch_bounds__(NT) ingest_kernel(IngestArgs<T> a) {
  const Dims& dm = a.dm;
  const int d = dm.d, D = dm.D, G = dm.G, F = dm.F, B = dm.B, H = dm.H;
  const int h = blockIdx.y;
  const int b0 = blockIdx.x * SB;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int in_dim = 3 * d;

  extern __shared__ __align__(16) unsigned char smem[];
  float* Xt = reinterpret_cast<float*>(smem);                // [3d][SB] scorer inputs
  float* qm = Xt + SB * in_dim;                              // [SB][d]
  float* contrib = qm + SB * d;                              // [SB][F]
  T* rawk = reinterpret_cast<T*>(contrib + SB * F);          // [SB][d]
  T* rawv = rawk + SB * d;                                   // [SB][d]
  __shared__ int s_p[SB];
  __shared__ int s_active[SB];

  T* slotK = static_cast<T*>(a.st.slotK);
  T* slotV = static_cast<T*>(a.st.slotV);
  T* ringK = static_cast<T*>(a.st.ringK);
  T* ringV = static_cast<T*>(a.st.ringV);

  // ---- phase 1: per-sequence window bookkeeping and scorer input -------------------
  // X is stored transposed, Xt[i][SB], so phase 2 reads SB inputs with two 16-B loads.
  if (warp < SB) {
    const int b = b0 + warp;
    int p = -1, active = 0;
    if (b < dm.batch) {
      const int pair = b * H + h;
      p = a.st.len[pair];
      active = p >= D;
      // mean query of the new token over the G query heads of KV head h
      const T* qrow = a.q + (size_t)(pair * G) * d;
      for (int i = lane; i < d; i += 32) {
        float acc = 0.f;
        for (int g = 0; g < G; ++g) acc += to_f(qrow[g * d + i]);
        qm[warp * d + i] = acc * (1.0f / (float)G);
      }
      __syncwarp();
    }
    if (active) {
      const int pair = b * H + h;
      const int ri = p % D;          // ring slot of u = p - D
      const T* rk = ringK + ((size_t)pair * D + ri) * d;
      const T* rv = ringV + ((size_t)pair * D + ri) * d;
      const float* rq = a.st.ringQm + (size_t)pair * D * d;
      for (int i = lane; i < d; i += 32) {
        T kk = rk[i], vv = rv[i];
        rawk[warp * d + i] = kk;
        rawv[warp * d + i] = vv;
        Xt[i * SB + warp] = to_f(kk);
        Xt[(d + i) * SB + warp] = to_f(vv);
        // qbar_u: queries u+1 .. p in position order, averaged over D (and G above)
        float acc = 0.f;
        for (int j = 1; j < D; ++j) acc += rq[((ri + j) % D) * d + i];
        acc += qm[warp * d + i];
        Xt[(2 * d + i) * SB + warp] = acc / (float)D;
      }
    } else {
      for (int i = lane; i < in_dim; i += 32) Xt[i * SB + warp] = 0.f;
    }
    if (lane == 0) { s_p[warp] = p; s_active[warp] = active; }
  }
  __syncthreads();

  // ---- phase 1b: push the new token into the window (after u was read) -------------
  if (warp < SB) {
    const int b = b0 + warp;
    if (b < dm.batch) {
      const int pair = b * H + h;
      const int p = s_p[warp];
      const int wi = p % D;
      T* dk = ringK + ((size_t)pair * D + wi) * d;
      T* dv = ringV + ((size_t)pair * D + wi) * d;
      float* dq = a.st.ringQm + ((size_t)pair * D + wi) * d;
      const T* sk = a.k + (size_t)pair * d;
      const T* sv = a.v + (size_t)pair * d;
      for (int i = lane; i < d; i += 32) {
        dk[i] = sk[i];
        dv[i] = sv[i];
        dq[i] = qm[warp * d + i];
      }
    }
  }

  // ---- phase 2: scorer MLP hidden layer for the SB sequences -----------------------
  bool any_active = false;
  for (int i = 0; i < SB; ++i) any_active |= (s_active[i] != 0);
  if (any_active) {
    const float* W1 = a.st.W1 + (size_t)h * in_dim * F;
    const float* b1 = a.st.b1 + (size_t)h * F;
    const float* w2 = a.st.w2 + (size_t)h * F;
    for (int f = threadIdx.x; f < F; f += NT) {
      float acc[SB];
      const float bias = b1[f];
#pragma unroll
      for (int r = 0; r < SB; ++r) acc[r] = bias;
#pragma unroll 4
      for (int i = 0; i < in_dim; ++i) {
        const float w = __ldg(W1 + (size_t)i * F + f);
        const float4 x0 = *reinterpret_cast<const float4*>(Xt + i * SB);
        const float4 x1 = *reinterpret_cast<const float4*>(Xt + i * SB + 4);
        acc[0] = fmaf(x0.x, w, acc[0]); acc[1] = fmaf(x0.y, w, acc[1]);
        acc[2] = fmaf(x0.z, w, acc[2]); acc[3] = fmaf(x0.w, w, acc[3]);
        acc[4] = fmaf(x1.x, w, acc[4]); acc[5] = fmaf(x1.y, w, acc[5]);
        acc[6] = fmaf(x1.z, w, acc[6]); acc[7] = fmaf(x1.w, w, acc[7]);
      }
      const float wf = w2[f];
#pragma unroll
      for (int r = 0; r < SB; ++r) contrib[r * F + f] = wf * gelu_erf(acc[r]);
    }
  }
  __syncthreads();

  // ---- phase 3: score, keep-or-drop, scatter ------------------------------------------
  if (warp >= SB) return;
  const int b = b0 + warp;
  if (b >= dm.batch) return;
  const int pair = b * H + h;
  const int p = s_p[warp];
  if (!s_active[warp]) {
    if (lane == 0) {
      a.st.len[pair] = p + 1;
      if (a.evict_info) { a.evict_info[2 * pair] = -1; a.evict_info[2 * pair + 1] = -1; }
      if (a.score_out) a.score_out[pair] = __int_as_float(0x7fc00000);
    }
    return;
  }
  float r = 0.f;
  for (int f = lane; f < F; f += 32) r += contrib[warp * F + f];
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) r += __shfl_xor_sync(0xffffffffu, r, off);
  r += a.st.b2[h];
  if (a.override_) r = a.override_[pair];
  r = canon_score(r);
  const int u = p - D;
  const float prio = static_priority(r, u, a.st.log_gamma, h);

  float* sc = a.st.score + (size_t)pair * B;
  int32_t* ps = a.st.pos + (size_t)pair * B;
  const int nv = a.st.nvalid[pair];
  int slot = -1, evicted = -1;
  if (nv < B) {
    slot = nv;
  } else if (prio > a.st.min_score[pair]) {
    slot = a.st.min_slot[pair];
    evicted = ps[slot];
  }
  if (slot >= 0) {
    // scatter the token's K/V from the window copy into its slot
    T* dk = slotK + ((size_t)pair * B + slot) * d;
    T* dv = slotV + ((size_t)pair * B + slot) * d;
    for (int i = lane; i < d; i += 32) {
      dk[i] = rawk[warp * d + i];
      dv[i] = rawv[warp * d + i];
    }
    const int nv_new = nv < B ? nv + 1 : nv;
    if (nv_new == B) {                       // full: refresh the cached argmin
      float mval;
      int midx;
      warp_argmin(sc, dm.s, B, slot, prio, mval, midx);
      if (lane == 0) { a.st.min_score[pair] = mval; a.st.min_slot[pair] = midx; }
    }
    if (lane == 0) {
      sc[slot] = prio;
      ps[slot] = u;
      a.st.nvalid[pair] = nv_new;
    }
  }
  if (lane == 0) {
    a.st.len[pair] = p + 1;
    if (a.evict_info) { a.evict_info[2 * pair] = slot; a.evict_info[2 * pair + 1] = evicted; }
    if (a.score_out) a.score_out[pair] = r;
  }
}

}  // namespace

static size_t ingest_smem(const Dims& dm) {
  const size_t esz = dm.dtype == KVPOP_F32 ? 4 : 2;
  return (size_t)SB * (3 * dm.d + dm.d + dm.F) * 4 + 2 * (size_t)SB * dm.d * esz;
}

cudaError_t prepare_ingest(const Dims& dm) {
  const int smem = (int)ingest_smem(dm);
  if (dm.dtype == KVPOP_F32)
    return cudaFuncSetAttribute(ingest_kernel<float>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  return cudaFuncSetAttribute(ingest_kernel<bf16>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
}

cudaError_t launch_ingest(const State& st, const Dims& dm, const void* q, const void* k,
                          const void* v, const float* override_, int32_t* evict_info,
                          float* score_out, cudaStream_t stream) {
  dim3 grid((dm.batch + SB - 1) / SB, dm.H);
  const size_t smem = ingest_smem(dm);
  if (dm.dtype == KVPOP_F32) {
    IngestArgs<float> a{st, dm, (const float*)q, (const float*)k, (const float*)v,
                        override_, evict_info, score_out};
    ingest_kernel<float><<<grid, NT, smem, stream>>>(a);
  } else {
    IngestArgs<bf16> a{st, dm, (const bf16*)q, (const bf16*)k, (const bf16*)v,
                       override_, evict_info, score_out};
    ingest_kernel<bf16><<<grid, NT, smem, stream>>>(a);
  }
  return cudaGetLastError();
}

}  // namespace kvpop
