// Stateful delayed mLSTM scorer (App. A, App. E.3, App. E.4): decode ingest and
// prompt prefill.
//
// Per KV head, x_t = [k_t; v_t]; q~ = phi(W_q x), k~ = phi(W_k x), v~ = W_v x with
// W_* in R^{2d x d/2} and the Hedgehog map phi(y) = [softmax(y); softmax(-y)];
// gates i = exp(w_i.x + b_i), f = sigmoid(w_f.x + b_f).  The state (C [d][d/2],
// z [d]) absorbs every token, kept in the stabilised form with a running
// log-scale m:  m' = max(log f + m, log i),  C' = e^{log f + m - m'} C +
// e^{log i - m'} k~ v~^T  (same for z).  At position p, after absorbing token p,
// the token u = p - D that leaves the window is read out with the current state,
// h = (q~_u^T C) / (q~_u^T z), and scored r = a . SiLU(h) + b; the keep-or-drop
// rule is the one of the MLP path (kvpop_evict.cuh).
//
// Weights are packed per head as one matrix Wcat [2d][NC] whose columns are
// [W_k | W_v | W_q | w_i | w_f | 0 pad], so one pass over x gives every
// projection.  The decode kernel loads its head's Wcat whole into shared memory
// with bulk copies (200 KB for d = 128) and serves 8 sequences per CTA.
#include "kvpop_evict.cuh"

namespace kvpop {
namespace {

constexpr int SBM = 8;             // sequences per decode CTA (one warp each)
constexpr int NTM = 256;
constexpr int UTM = 32;            // prompt tokens per projection CTA

struct MState {
  float* C;                        // [pairs][d][d/2]
  float* z;                        // [pairs][d]
  float* m;                        // [pairs]
  const float* Wcat;               // [H][2d][NC]
  const float* bi;                 // [H]
  const float* bf;                 // [H]
  const float* a;                  // [H][d/2]
  const float* b;                  // [H]
  int NC;
};

template <typename T>
struct MIngestArgs {
  State st;
  Dims dm;
  MState ms;
  const T* q;
  const T* k;
  const T* v;
  const float* override_;
  int32_t* evict_info;
  float* score_out;
};

__device__ __forceinline__ float warp_max(float x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, o));
  return x;
}
__device__ __forceinline__ float warp_sum(float x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  return x;
}
__device__ __forceinline__ float softplus(float x) {
  return fmaxf(x, 0.f) + log1pf(expf(-fabsf(x)));
}

// Hedgehog features of y[0..hh) (hh = d/2, held 32 lanes x HP values): out[0..2hh).
template <int HP>
__device__ __forceinline__ void hedgehog_warp(const float* y, float* out, int hh) {
  const int lane = threadIdx.x & 31;
  float v[HP];
  float mp = -INFINITY, mn = -INFINITY;
#pragma unroll
  for (int t = 0; t < HP; ++t) {
    const int i = lane + 32 * t;
    v[t] = i < hh ? y[i] : 0.f;
    if (i < hh) { mp = fmaxf(mp, v[t]); mn = fmaxf(mn, -v[t]); }
  }
  mp = warp_max(mp);
  mn = warp_max(mn);
  float ep[HP], en[HP], sp = 0.f, sn = 0.f;
#pragma unroll
  for (int t = 0; t < HP; ++t) {
    const int i = lane + 32 * t;
    ep[t] = i < hh ? expf(v[t] - mp) : 0.f;
    en[t] = i < hh ? expf(-v[t] - mn) : 0.f;
    sp += ep[t];
    sn += en[t];
  }
  sp = warp_sum(sp);
  sn = warp_sum(sn);
#pragma unroll
  for (int t = 0; t < HP; ++t) {
    const int i = lane + 32 * t;
    if (i < hh) { out[i] = ep[t] / sp; out[hh + i] = en[t] / sn; }
  }
}

// C <- fs C + is k~ v~^T on this lane's columns (NJ of them) and y += q~^T C, rows
// in chunks of 32 whose loads are all issued before the first store.
template <int NJ>
__device__ __forceinline__ void state_rows(float* __restrict__ C, int d, int hh, float fs, float is,
                                           const float* kt, const float* qt, const float (&vj)[2],
                                           float (&yj)[2]) {
  const int lane = threadIdx.x & 31;
  for (int i0 = 0; i0 < d; i0 += 32) {
    float c[32][NJ];
#pragma unroll
    for (int r = 0; r < 32; ++r)
#pragma unroll
      for (int t = 0; t < NJ; ++t) c[r][t] = __ldcg(C + (size_t)(i0 + r) * hh + lane + 32 * t);
#pragma unroll
    for (int r = 0; r < 32; ++r) {
      const float ki = is * kt[i0 + r], qi = qt[i0 + r];
#pragma unroll
      for (int t = 0; t < NJ; ++t) {
        const float cn = fmaf(fs, c[r][t], ki * vj[t]);
        C[(size_t)(i0 + r) * hh + lane + 32 * t] = cn;
        yj[t] = fmaf(qi, cn, yj[t]);
      }
    }
  }
}

__host__ __device__ inline size_t mlstm_ingest_smem(int d, int NC, int esz) {
  return (size_t)2 * d * NC * 4 + 2 * (size_t)2 * d * SBM * 4 + (size_t)SBM * NC * 4 +
         2 * (size_t)SBM * d * esz;
}

template <typename T>
__global__ void __launch_bounds__(NTM, 1) ingest_mlstm_kernel(MIngestArgs<T> a) {
  const Dims& dm = a.dm;
  const int d = dm.d, D = dm.D, H = dm.H, NC = a.ms.NC, hh = d / 2;
  const int in2 = 2 * d;
  const int h = blockIdx.y, b0 = blockIdx.x * SBM;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  extern __shared__ __align__(128) unsigned char smem[];
  float* Ws = reinterpret_cast<float*>(smem);                  // [2d][NC]
  float* Xp = Ws + (size_t)in2 * NC;                           // [2d][SBM]  x of the new token
  float* Xu = Xp + in2 * SBM;                                  // [2d][SBM]  x of the leaving token
  float* proj = Xu + in2 * SBM;                                // [SBM][NC]
  T* rawk = reinterpret_cast<T*>(proj + SBM * NC);             // [SBM][d]
  T* rawv = rawk + SBM * d;
  float* feat = Xp;                                            // [SBM][2][d] after the projections
  __shared__ __align__(8) uint64_t bar;
  __shared__ int s_p[SBM];

  if (tid == 0) {
    mbar_init(smem_u32(&bar), 1);
    mbar_fence_init();
    const uint32_t bytes = (uint32_t)(in2 * NC * 4);
    mbar_arrive_expect_tx(smem_u32(&bar), bytes);
    const unsigned char* src = reinterpret_cast<const unsigned char*>(a.ms.Wcat + (size_t)h * in2 * NC);
    for (uint32_t off = 0; off < bytes; off += 32768)
      bulk_g2s(smem_u32(smem + off), src + off, min(32768u, bytes - off), smem_u32(&bar));
  }
  T* ringK = static_cast<T*>(a.st.ringK);
  T* ringV = static_cast<T*>(a.st.ringV);
  {
    const int b = b0 + warp;
    int p = -1;
    if (b < dm.batch) {
      const int pair = b * H + h;
      p = a.st.len[pair];
      const int ri = p % D;
      const T* kp = a.k + (size_t)pair * d;
      const T* vp = a.v + (size_t)pair * d;
      T* rk = ringK + ((size_t)pair * D + ri) * d;
      T* rv = ringV + ((size_t)pair * D + ri) * d;
      for (int i = lane; i < d; i += 32) {
        const T ku = rk[i], vu = rv[i];
        rawk[warp * d + i] = ku;
        rawv[warp * d + i] = vu;
        Xu[i * SBM + warp] = p >= D ? to_f(ku) : 0.f;
        Xu[(d + i) * SBM + warp] = p >= D ? to_f(vu) : 0.f;
        const T kn = kp[i], vn = vp[i];
        Xp[i * SBM + warp] = to_f(kn);
        Xp[(d + i) * SBM + warp] = to_f(vn);
      }
      __syncwarp();
      for (int i = lane; i < d; i += 32) {     // the new token takes u's window slot
        rk[i] = kp[i];
        rv[i] = vp[i];
      }
    } else {
      for (int i = lane; i < in2; i += 32) { Xp[i * SBM + warp] = 0.f; Xu[i * SBM + warp] = 0.f; }
    }
    if (lane == 0) s_p[warp] = p;
  }
  __syncthreads();
  const bool ok = mbar_wait(smem_u32(&bar), 0, a.st.err, DEVERR_TIMEOUT_FULL);

  // ---- all projections of the 8 sequences: column c of Wcat per thread -------------
  for (int c = tid; c < NC; c += NTM) {
    const float* X = (c >= d && c < d + hh) ? Xu : Xp;     // W_q reads the leaving token
    float acc[SBM];
#pragma unroll
    for (int s = 0; s < SBM; ++s) acc[s] = 0.f;
    if (ok) {
#pragma unroll 4
      for (int i = 0; i < in2; ++i) {
        const float w = Ws[(size_t)i * NC + c];
        const float4 x0 = *reinterpret_cast<const float4*>(X + i * SBM);
        const float4 x1 = *reinterpret_cast<const float4*>(X + i * SBM + 4);
        acc[0] = fmaf(x0.x, w, acc[0]); acc[1] = fmaf(x0.y, w, acc[1]);
        acc[2] = fmaf(x0.z, w, acc[2]); acc[3] = fmaf(x0.w, w, acc[3]);
        acc[4] = fmaf(x1.x, w, acc[4]); acc[5] = fmaf(x1.y, w, acc[5]);
        acc[6] = fmaf(x1.z, w, acc[6]); acc[7] = fmaf(x1.w, w, acc[7]);
      }
    }
#pragma unroll
    for (int s = 0; s < SBM; ++s) proj[s * NC + c] = acc[s];
  }
  __syncthreads();

  // ---- per sequence: features, state update, delayed readout, keep-or-drop ---------
  const int b = b0 + warp;
  if (b >= dm.batch || !ok) return;
  const int pair = b * H + h;
  const int p = s_p[warp];
  const float* pr = proj + warp * NC;
  float* kt = feat + (size_t)warp * 2 * d;          // k~ [d]
  float* qt = kt + d;                                // q~ [d]
  if (hh > 32) {
    hedgehog_warp<2>(pr, kt, hh);
    hedgehog_warp<2>(pr + d, qt, hh);
  } else {
    hedgehog_warp<1>(pr, kt, hh);
    hedgehog_warp<1>(pr + d, qt, hh);
  }
  __syncwarp();
  const float ai = pr[3 * hh] + a.ms.bi[h];
  const float af = pr[3 * hh + 1] + a.ms.bf[h];
  const float lf = -softplus(-af);
  const float m_old = a.ms.m[pair];
  const float m_new = fmaxf(lf + m_old, ai);
  const float fs = (m_old == -INFINITY) ? 0.f : expf(lf + m_old - m_new);
  const float is = expf(ai - m_new);
  // columns j = lane (+32) of C and of the readout: rows are loaded 32 at a time
  // (independent loads in flight) before they are updated and stored
  float vj[2], yj[2] = {0.f, 0.f};
  const int nj = hh / 32;
  for (int t = 0; t < nj; ++t) vj[t] = pr[hh + lane + 32 * t];
  float* __restrict__ C = a.ms.C + (size_t)pair * d * hh;
  if (nj == 2) state_rows<2>(C, d, hh, fs, is, kt, qt, vj, yj);
  else         state_rows<1>(C, d, hh, fs, is, kt, qt, vj, yj);
  float den = 0.f;
  float* z = a.ms.z + (size_t)pair * d;
  for (int i = lane; i < d; i += 32) {
    const float zn = fmaf(fs, z[i], is * kt[i]);
    z[i] = zn;
    den = fmaf(qt[i], zn, den);
  }
  den = warp_sum(den);
  if (lane == 0) a.ms.m[pair] = m_new;
  if (p < D) {
    if (lane == 0) {
      a.st.len[pair] = p + 1;
      if (a.evict_info) { a.evict_info[2 * pair] = -1; a.evict_info[2 * pair + 1] = -1; }
      if (a.score_out) a.score_out[pair] = __int_as_float(0x7fc00000);
    }
    return;
  }
  float rpart = 0.f;
  for (int t = 0; t < nj; ++t) {
    const float hv = yj[t] / den;
    const float silu = hv / (1.f + expf(-hv));
    rpart = fmaf(a.ms.a[(size_t)h * hh + lane + 32 * t], silu, rpart);
  }
  float r = warp_sum(rpart) + a.ms.b[h];
  if (a.override_) r = a.override_[pair];
  evict_and_scatter<T>(a.st, dm, pair, h, p, r, rawk + warp * d, rawv + warp * d, a.evict_info,
                       a.score_out);
}

// ------------------------------------------------------------------ prefill
template <typename T>
struct MProjArgs {
  Dims dm;
  MState ms;
  const T* K;                      // [n_seq][H][Pmax][d]
  const T* V;
  const int32_t* plen;
  float* feat;                     // [n_seq*H][Pmax][NF]: k~ (d) | v~ (d/2) | q~ (d) | a_i | a_f
  int Pmax, NF;
};

template <typename T>
__global__ void __launch_bounds__(NTM) mlstm_proj_kernel(MProjArgs<T> a) {
  const Dims& dm = a.dm;
  const int d = dm.d, H = dm.H, NC = a.ms.NC, hh = d / 2, in2 = 2 * d, NF = a.NF;
  const int lp = blockIdx.y, bl = lp / H, h = lp - bl * H;
  const int P = a.plen[bl];
  const int t0 = blockIdx.x * UTM;
  if (t0 >= P) return;
  const int nrow = min(UTM, P - t0);
  extern __shared__ __align__(16) unsigned char smem[];
  float* Xt = reinterpret_cast<float*>(smem);                  // [2d][UTM]
  float* pj = Xt + in2 * UTM;                                  // [UTM][NC]
  const size_t Pm = a.Pmax;
  const T* Kp = a.K + ((size_t)bl * H + h) * Pm * d;
  const T* Vp = a.V + ((size_t)bl * H + h) * Pm * d;
  for (int idx = threadIdx.x; idx < UTM * d; idx += NTM) {
    const int r = idx / d, i = idx - r * d;
    const bool in = r < nrow;
    Xt[i * UTM + r] = in ? to_f(Kp[(size_t)(t0 + r) * d + i]) : 0.f;
    Xt[(d + i) * UTM + r] = in ? to_f(Vp[(size_t)(t0 + r) * d + i]) : 0.f;
  }
  __syncthreads();
  const float* W = a.ms.Wcat + (size_t)h * in2 * NC;
  for (int c = threadIdx.x; c < NC; c += NTM) {
    float acc[UTM];
#pragma unroll
    for (int r = 0; r < UTM; ++r) acc[r] = 0.f;
#pragma unroll 2
    for (int i = 0; i < in2; ++i) {
      const float w = __ldg(W + (size_t)i * NC + c);
      const float4* xr = reinterpret_cast<const float4*>(Xt + i * UTM);
#pragma unroll
      for (int r4 = 0; r4 < UTM / 4; ++r4) {
        const float4 x = xr[r4];
        acc[4 * r4 + 0] = fmaf(x.x, w, acc[4 * r4 + 0]);
        acc[4 * r4 + 1] = fmaf(x.y, w, acc[4 * r4 + 1]);
        acc[4 * r4 + 2] = fmaf(x.z, w, acc[4 * r4 + 2]);
        acc[4 * r4 + 3] = fmaf(x.w, w, acc[4 * r4 + 3]);
      }
    }
#pragma unroll
    for (int r = 0; r < UTM; ++r) pj[r * NC + c] = acc[r];
  }
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float* out = a.feat + ((size_t)lp * Pm) * NF;
  for (int r = warp; r < nrow; r += NTM / 32) {
    float* o = out + (size_t)(t0 + r) * NF;
    const float* pr = pj + r * NC;
    if (hh > 32) { hedgehog_warp<2>(pr, o, hh); hedgehog_warp<2>(pr + d, o + d + hh, hh); }
    else         { hedgehog_warp<1>(pr, o, hh); hedgehog_warp<1>(pr + d, o + d + hh, hh); }
    for (int j = lane; j < hh; j += 32) o[d + j] = pr[hh + j];
    if (lane == 0) {
      o[2 * d + hh] = pr[3 * hh] + a.ms.bi[h];
      o[2 * d + hh + 1] = pr[3 * hh + 1] + a.ms.bf[h];
    }
  }
}

struct MScanArgs {
  State st;
  Dims dm;
  MState ms;
  const int32_t* plen;
  const float* feat;
  const float* override_;          // [n_seq][H][Pmax] or nullptr
  float* prio;                     // [n_seq][H][Pmax]
  int first_seq, Pmax, NF;
};

// One CTA per (sequence, head): the recurrence over the prompt, scoring every
// u = t - D right after token t has been absorbed.
__global__ void __launch_bounds__(NTM) mlstm_scan_kernel(MScanArgs a) {
  const Dims& dm = a.dm;
  const int d = dm.d, D = dm.D, H = dm.H, hh = d / 2, NF = a.NF;
  const int lp = blockIdx.x, bl = lp / H, h = lp - bl * H;
  const int pair = (a.first_seq + bl) * H + h;
  const int P = a.plen[bl];
  const size_t Pm = a.Pmax;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  extern __shared__ __align__(16) unsigned char smem[];
  float* C = reinterpret_cast<float*>(smem);                   // [d][hh]
  float* z = C + d * hh;                                        // [d]
  float* ft = z + d;                                            // [NF] features of token t
  float* qu = ft + NF;                                          // [d]  q~ of token u
  float* red = qu + d;                                          // [NTM]
  __shared__ float s_den, s_r;
  for (int e = tid; e < d * hh; e += NTM) C[e] = 0.f;
  for (int e = tid; e < d; e += NTM) z[e] = 0.f;
  float m = -INFINITY;
  const float* F = a.feat + (size_t)lp * Pm * NF;
  float* prio = a.prio + (size_t)lp * Pm;
  const int groups = NTM / hh;                                  // row groups of the readout
  const int jr = tid % hh, gr = tid / hh;
  // features of the next token (and the next read-out query) are fetched into
  // registers one iteration ahead; NF <= 2 * NTM and d <= NTM
  float nf0 = 0.f, nf1 = 0.f, nq = 0.f;
  auto fetch = [&](int t) {
    if (t >= P) return;
    nf0 = tid < NF ? F[(size_t)t * NF + tid] : 0.f;
    nf1 = tid + NTM < NF ? F[(size_t)t * NF + tid + NTM] : 0.f;
    nq = (t >= D && tid < d) ? F[(size_t)(t - D) * NF + d + hh + tid] : 0.f;
  };
  fetch(0);
  for (int t = 0; t < P; ++t) {
    __syncthreads();
    if (tid < NF) ft[tid] = nf0;
    if (tid + NTM < NF) ft[tid + NTM] = nf1;
    if (t >= D && tid < d) qu[tid] = nq;
    fetch(t + 1);
    __syncthreads();    const float ai = ft[2 * d + hh], af = ft[2 * d + hh + 1];
    const float lf = -softplus(-af);
    const float m_new = fmaxf(lf + m, ai);
    const float fs = (m == -INFINITY) ? 0.f : expf(lf + m - m_new);
    const float is = expf(ai - m_new);
    m = m_new;
    for (int e = tid; e < d * hh; e += NTM) {
      const int i = e / hh, j = e - i * hh;
      C[e] = fmaf(fs, C[e], is * ft[i] * ft[d + j]);
    }
    for (int e = tid; e < d; e += NTM) z[e] = fmaf(fs, z[e], is * ft[e]);
    if (t < D) continue;
    __syncthreads();
    // readout y_j = sum_i q~_i C[i][j], den = q~ . z
    float y = 0.f;
    if (gr < groups)
      for (int i = gr; i < d; i += groups) y = fmaf(qu[i], C[i * hh + jr], y);
    red[tid] = y;
    if (warp == 0) {
      float dd = 0.f;
      for (int i = lane; i < d; i += 32) dd = fmaf(qu[i], z[i], dd);
      dd = warp_sum(dd);
      if (lane == 0) s_den = dd;
    }
    __syncthreads();
    if (warp == 0) {
      float rp = 0.f;
      for (int j = lane; j < hh; j += 32) {
        float yy = 0.f;
        for (int g = 0; g < groups; ++g) yy += red[g * hh + j];
        const float hv = yy / s_den;
        rp = fmaf(a.ms.a[(size_t)h * hh + j], hv / (1.f + expf(-hv)), rp);
      }
      rp = warp_sum(rp);
      if (lane == 0) {
        const int u = t - D;
        float r = rp + a.ms.b[h];
        if (a.override_) r = a.override_[(size_t)lp * Pm + u];
        prio[u] = static_priority(canon_score(r), u, a.st.log_gamma, h);
      }
    }
  }
  __syncthreads();
  float* Cg = a.ms.C + (size_t)pair * d * hh;
  for (int e = tid; e < d * hh; e += NTM) Cg[e] = C[e];
  for (int e = tid; e < d; e += NTM) a.ms.z[(size_t)pair * d + e] = z[e];
  if (tid == 0) a.ms.m[pair] = m;
}

}  // namespace

int mlstm_nc(int d) { return ((3 * (d / 2) + 2) + 3) & ~3; }
int mlstm_nf(int d) { return ((2 * d + d / 2 + 2) + 3) & ~3; }

static MState to_mstate(const MlstmDev& m) {
  MState s;
  s.C = m.C; s.z = m.z; s.m = m.m; s.Wcat = m.Wcat; s.bi = m.bi; s.bf = m.bf; s.a = m.a; s.b = m.b;
  s.NC = m.NC;
  return s;
}

cudaError_t prepare_mlstm(const Dims& dm) {
  const int NC = mlstm_nc(dm.d);
  const int esz = dm.dtype == KVPOP_F32 ? 4 : 2;
  const int ism = (int)mlstm_ingest_smem(dm.d, NC, esz);
  const int psm = (int)((size_t)2 * dm.d * UTM * 4 + (size_t)UTM * NC * 4);
  cudaError_t e;
  if (dm.dtype == KVPOP_F32) {
    e = raise_smem_limit(ingest_mlstm_kernel<float>, ism);
    if (e == cudaSuccess)
      e = raise_smem_limit(mlstm_proj_kernel<float>, psm);
  } else {
    e = raise_smem_limit(ingest_mlstm_kernel<bf16>, ism);
    if (e == cudaSuccess)
      e = raise_smem_limit(mlstm_proj_kernel<bf16>, psm);
  }
  return e;
}

bool mlstm_ok(const Dims& dm) {
  const int esz = dm.dtype == KVPOP_F32 ? 4 : 2;
  return mlstm_ingest_smem(dm.d, mlstm_nc(dm.d), esz) <= 227 * 1024;
}

cudaError_t launch_ingest_mlstm(const State& st, const Dims& dm, const MlstmDev& m, const void* q,
                                const void* k, const void* v, const float* override_,
                                int32_t* evict_info, float* score_out, cudaStream_t stream) {
  dim3 grid((dm.batch + SBM - 1) / SBM, dm.H);
  const int esz = dm.dtype == KVPOP_F32 ? 4 : 2;
  const size_t smem = mlstm_ingest_smem(dm.d, m.NC, esz);
  if (dm.dtype == KVPOP_F32) {
    MIngestArgs<float> a{st, dm, to_mstate(m), (const float*)q, (const float*)k, (const float*)v,
                         override_, evict_info, score_out};
    ingest_mlstm_kernel<float><<<grid, NTM, smem, stream>>>(a);
  } else {
    MIngestArgs<bf16> a{st, dm, to_mstate(m), (const bf16*)q, (const bf16*)k, (const bf16*)v,
                        override_, evict_info, score_out};
    ingest_mlstm_kernel<bf16><<<grid, NTM, smem, stream>>>(a);
  }
  return cudaGetLastError();
}

cudaError_t launch_prefill_mlstm_scores(const State& st, const Dims& dm, const MlstmDev& m,
                                        const void* K, const void* V, const int32_t* plen,
                                        int first_seq, int n_seq, int Pmax, const float* override_,
                                        float* feat, float* prio, cudaStream_t stream) {
  const int NF = mlstm_nf(dm.d);
  const int pairs = n_seq * dm.H;
  const size_t psm = (size_t)2 * dm.d * UTM * 4 + (size_t)UTM * m.NC * 4;
  dim3 g1((Pmax + UTM - 1) / UTM, pairs);
  if (Pmax > 0) {
    if (dm.dtype == KVPOP_F32) {
      MProjArgs<float> a{dm, to_mstate(m), (const float*)K, (const float*)V, plen, feat, Pmax, NF};
      mlstm_proj_kernel<float><<<g1, NTM, psm, stream>>>(a);
    } else {
      MProjArgs<bf16> a{dm, to_mstate(m), (const bf16*)K, (const bf16*)V, plen, feat, Pmax, NF};
      mlstm_proj_kernel<bf16><<<g1, NTM, psm, stream>>>(a);
    }
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  MScanArgs sa{st, dm, to_mstate(m), plen, feat, override_, prio, first_seq, Pmax, NF};
  const size_t ssm = ((size_t)dm.d * (dm.d / 2) + dm.d + NF + dm.d + NTM) * 4;
  mlstm_scan_kernel<<<pairs, NTM, ssm, stream>>>(sa);
  return cudaGetLastError();
}

}  // namespace kvpop
