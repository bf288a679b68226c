// Decode steps 1-4: ingest the new token, run the delayed scorer on the token
// that leaves the window, keep or drop it under the fixed budget, scatter it.
//
// One CTA owns one KV head h and SB consecutive sequences, so each row of the
// head's scorer weights W1 [3d][F] that it streams feeds SB sequences.  W1 is
// staged through shared memory in 32 KB chunks by 1-D TMA bulk copies, the
// first ones issued before the window bookkeeping so the copy overlaps it.
// Warp i of the CTA does the per-sequence work of sequence i of the group.
//
// Paper correspondence: eligible set and the newly eligible token u = p - w
// (Sec. 3.1, Eq. 4); delayed scoring (Sec. 3.3, App. E.4) with the stateless
// MLP of Sec. 3.3 / App. E.2 on [k_u; v_u; qbar_u]; static priority
// (App. B.3); running top-k under the budget (Sec. 3.2, App. C.1).
#include "kvpop_argmin.cuh"

namespace kvpop {
namespace {

constexpr int SB = 8;               // sequences per CTA (one warp each)
constexpr int NT = 256;             // threads per CTA
constexpr int STG = 3;              // W1 chunk stages
constexpr int CHUNK = 32768;        // bytes per W1 chunk
constexpr int MAXF = 1024 / NT;     // hidden units per thread (F <= 1024)

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

__host__ __device__ inline size_t ingest_smem_bytes(int d, int Fp, int esz) {
  return (size_t)STG * CHUNK + ((size_t)3 * d * SB + (size_t)SB * d + (size_t)SB * Fp) * 4 +
         2 * (size_t)SB * d * esz;
}

template <typename T>
__global__ void __launch_bounds__(NT) ingest_kernel(IngestArgs<T> a) {
  const Dims& dm = a.dm;
  const int d = dm.d, D = dm.D, G = dm.G, F = dm.F, Fp = dm.Fp, B = dm.B, H = dm.H;
  const int h = blockIdx.y;
  const int b0 = blockIdx.x * SB;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int in_dim = 3 * d;
  const int KC = CHUNK / (Fp * 4);                 // W1 rows per chunk
  const int nchunks = (in_dim + KC - 1) / KC;

  extern __shared__ __align__(128) unsigned char smem[];
  float* Wst = reinterpret_cast<float*>(smem);                         // [STG][KC][Fp]
  float* Xt = reinterpret_cast<float*>(smem + (size_t)STG * CHUNK);    // [3d][SB]
  float* qm = Xt + SB * in_dim;                                        // [SB][d]
  float* contrib = qm + SB * d;                                        // [SB][Fp]
  T* rawk = reinterpret_cast<T*>(contrib + SB * Fp);                   // [SB][d]
  T* rawv = rawk + SB * d;
  __shared__ __align__(8) uint64_t bars[STG];
  __shared__ int s_p[SB];
  __shared__ int s_active[SB];

  const float* W1h = a.st.W1 + (size_t)h * in_dim * Fp;
  auto issue = [&](int c) {
    const int rows = min(KC, in_dim - c * KC);
    const uint32_t bytes = (uint32_t)rows * Fp * 4;
    const uint32_t bar = smem_u32(&bars[c % STG]);
    mbar_arrive_expect_tx(bar, bytes);
    bulk_g2s(smem_u32(Wst + (size_t)(c % STG) * (CHUNK / 4)), W1h + (size_t)c * KC * Fp, bytes, bar);
  };
  int issued = 0;
  if (tid == 0) {
    for (int s = 0; s < STG; ++s) mbar_init(smem_u32(&bars[s]), 1);
    mbar_fence_init();
    for (; issued < min(STG, nchunks); ++issued) issue(issued);
  }

  T* slotK = static_cast<T*>(a.st.slotK);
  T* slotV = static_cast<T*>(a.st.slotV);
  T* ringK = static_cast<T*>(a.st.ringK);
  T* ringV = static_cast<T*>(a.st.ringV);

  // ---- phase 1: per-sequence window bookkeeping and scorer input -------------------
  // X is stored transposed, Xt[i][SB], so phase 2 reads SB inputs with two 16-B loads.
  {
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
        const T kk = rk[i], vv = rv[i];
        rawk[warp * d + i] = kk;
        rawv[warp * d + i] = vv;
        Xt[i * SB + warp] = to_f(kk);
        Xt[(d + i) * SB + warp] = to_f(vv);
        // qbar_u: queries u+1 .. p in position order, averaged over D (and G above)
        float acc = 0.f;
        int j = 1;
        for (; j + 7 < D; j += 8) {
          float vals[8];
#pragma unroll
          for (int t = 0; t < 8; ++t) {
            int jj = ri + j + t;
            jj = jj >= D ? jj - D : jj;
            vals[t] = rq[(size_t)jj * d + i];
          }
#pragma unroll
          for (int t = 0; t < 8; ++t) acc += vals[t];
        }
        for (; j < D; ++j) {
          int jj = ri + j;
          jj = jj >= D ? jj - D : jj;
          acc += rq[(size_t)jj * d + i];
        }
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
  {
    const int b = b0 + warp;
    if (b < dm.batch) {
      const int pair = b * H + h;
      const int wi = s_p[warp] % D;
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

  // ---- phase 2: scorer MLP for the SB sequences, W1 streamed chunk by chunk --------
  const float* b1 = a.st.b1 + (size_t)h * Fp;
  const float* w2 = a.st.w2 + (size_t)h * Fp;
  float acc[MAXF][SB];
#pragma unroll
  for (int u = 0; u < MAXF; ++u) {
    const int f = tid + u * NT;
    const float bias = f < F ? b1[f] : 0.f;
#pragma unroll
    for (int r = 0; r < SB; ++r) acc[u][r] = bias;
  }
  bool ok = true;
  for (int c = 0; c < nchunks; ++c) {
    const int st = c % STG;
    if (ok) ok = mbar_wait(smem_u32(&bars[st]), (uint32_t)((c / STG) & 1), a.st.err, DEVERR_TIMEOUT_FULL);
    if (ok) {
      const int rows = min(KC, in_dim - c * KC);
      const float* Wc = Wst + (size_t)st * (CHUNK / 4);
      for (int r = 0; r < rows; ++r) {
        const int i = c * KC + r;
        const float4 x0 = *reinterpret_cast<const float4*>(Xt + i * SB);
        const float4 x1 = *reinterpret_cast<const float4*>(Xt + i * SB + 4);
#pragma unroll
        for (int u = 0; u < MAXF; ++u) {
          const int f = tid + u * NT;
          if (f < Fp) {
            const float w = Wc[r * Fp + f];
            acc[u][0] = fmaf(x0.x, w, acc[u][0]); acc[u][1] = fmaf(x0.y, w, acc[u][1]);
            acc[u][2] = fmaf(x0.z, w, acc[u][2]); acc[u][3] = fmaf(x0.w, w, acc[u][3]);
            acc[u][4] = fmaf(x1.x, w, acc[u][4]); acc[u][5] = fmaf(x1.y, w, acc[u][5]);
            acc[u][6] = fmaf(x1.z, w, acc[u][6]); acc[u][7] = fmaf(x1.w, w, acc[u][7]);
          }
        }
      }
    }
    __syncthreads();                  // every thread is done with stage st
    if (tid == 0 && ok && issued < nchunks) { issue(issued); ++issued; }
  }
#pragma unroll
  for (int u = 0; u < MAXF; ++u) {
    const int f = tid + u * NT;
    if (f < Fp) {
      const float wf = f < F ? w2[f] : 0.f;
#pragma unroll
      for (int r = 0; r < SB; ++r) contrib[r * Fp + f] = wf * scorer_act(acc[u][r], a.dm.act);
    }
  }
  if (tid == 0 && !ok) {
    // a wait expired: let the copies still in flight land before the CTA exits
    for (int s = 0; s < STG; ++s) {
      int last = -1;
      for (int c = s; c < issued; c += STG) last = c;
      if (last >= 0) mbar_wait(smem_u32(&bars[s]), (uint32_t)((last / STG) & 1), a.st.err, DEVERR_TIMEOUT_DRAIN);
    }
  }
  __syncthreads();

  // ---- phase 3: score, keep-or-drop, scatter ------------------------------------------
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
  for (int f = lane; f < F; f += 32) r += contrib[warp * Fp + f];
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) r += __shfl_xor_sync(0xffffffffu, r, off);
  r += a.st.b2[h];
  if (a.override_) r = a.override_[pair];
  r = canon_score(r);
  const int u = p - D;
  const float prio = static_priority(r, u, a.st.log_gamma, h);

  float* sc = a.st.score + (size_t)pair * B;
  int32_t* ps = a.st.pos + (size_t)pair * B;
  const int NB = min_blocks(B);
  float* bsc = a.st.blk_score + (size_t)pair * NB;
  int32_t* bsl = a.st.blk_slot + (size_t)pair * NB;
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
    if (nv == B)
      update_min(sc, dm.s, B, slot, prio, bsc, bsl, a.st.min_score + pair, a.st.min_slot + pair);
    else if (nv + 1 == B)
      rebuild_min(sc, dm.s, B, slot, prio, bsc, bsl, a.st.min_score + pair, a.st.min_slot + pair);
    if (lane == 0) {
      sc[slot] = prio;
      ps[slot] = u;
      a.st.nvalid[pair] = nv < B ? nv + 1 : nv;
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
  return ingest_smem_bytes(dm.d, dm.Fp, dm.dtype == KVPOP_F32 ? 4 : 2);
}

cudaError_t prepare_ingest(const Dims& dm) {
  const int smem = (int)ingest_smem(dm);
  if (dm.dtype == KVPOP_F32)
    return raise_smem_limit(ingest_kernel<float>, smem);
  return raise_smem_limit(ingest_kernel<bf16>, smem);
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
