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

// Chunkwise form of the same recurrence (App. A: the mLSTM as linear attention with
// gates).  Within a chunk of L tokens starting at t0, with F_s the cumulative log
// forget gate of the chunk up to token s and g_s = log i_s - F_s, the state after
// absorbing token t is, up to one common scale,
//   C(t) = e^{m - R_t} C + sum_{s <= t} e^{g_s - R_t} k~_s v~_s^T,   R_t = max(m, max_{s<=t} g_s)
// (same for z), where (C, z, m) is the stabilised state at the chunk start; the
// scale e^{F_t + R_t} cancels in the readout ratio, and at the chunk's end it is the
// new log-scale m' = F_{L-1} + R_{L-1}, which equals the token-by-token stabiliser.
// Every exponent is <= 0.  The readout of row t (token u = t0 + t - D) is
//   h = (e^{m-R_t} q~_u^T C + sum_s W_ts v~_s) / (e^{m-R_t} q~_u^T z + sum_s W_ts),
//   W_ts = e^{g_s - R_t} (q~_u . k~_s)  for s <= t,
// so a chunk costs three small dense products (q~ K^T, q~ C, W V) plus the state
// update C' = e^{m - R_{L-1}} C + K^T diag(e^{g - R_{L-1}}) V, all from shared memory
// with register tiles; chunks follow one another, the tokens of a chunk do not.
constexpr int CL = 64;             // tokens per chunk

template <int HD>
struct ChunkLayout {
  static constexpr int HH = HD / 2;
  static constexpr int QS = HD + 4;              // row strides (floats), multiples of 4
  static constexpr int VS = HH + 4;
  static constexpr int WS = CL + 4;
  static constexpr int OFF_Q = 0;                // [CL][QS]  q~ of the read-out tokens
  static constexpr int OFF_K = OFF_Q + CL * QS;  // [CL][QS]  k~ of the chunk's tokens
  static constexpr int OFF_V = OFF_K + CL * QS;  // [CL][VS]  v~
  static constexpr int OFF_C = OFF_V + CL * VS;  // [HD][VS]  state C
  static constexpr int OFF_W = OFF_C + HD * VS;  // [CL][WS]  W_ts
  static constexpr int OFF_Z = OFF_W + CL * WS;  // [HD]
  static constexpr int OFF_G = OFF_Z + HD;       // [CL] g_s
  static constexpr int OFF_R = OFF_G + CL;       // [CL] R_t
  static constexpr int OFF_QZ = OFF_R + CL;      // [CL] q~ . z
  static constexpr int OFF_SC = OFF_QZ + CL;     // [4] m, F_{L-1}
  static constexpr int FLOATS = OFF_SC + 4;
};

template <int HD>
__global__ void __launch_bounds__(NTM) mlstm_chunk_kernel(MScanArgs a) {
  using Ly = ChunkLayout<HD>;
  constexpr int HH = Ly::HH, QS = Ly::QS, VS = Ly::VS, WS = Ly::WS;
  constexpr int NB = HH / 16;                    // column blocks of q~C / num per thread
  const Dims& dm = a.dm;
  const int D = dm.D, H = dm.H, NF = a.NF;
  const int lp = blockIdx.x, bl = lp / H, h = lp - bl * H;
  const int pair = (a.first_seq + bl) * H + h;
  const int P = a.plen[bl];
  const size_t Pm = a.Pmax;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int ty = tid >> 4, tx = tid & 15;        // 16 x 16 thread grid
  extern __shared__ __align__(16) float smf[];
  float* Qs = smf + Ly::OFF_Q;
  float* Ks = smf + Ly::OFF_K;
  float* Vs = smf + Ly::OFF_V;
  float* Cs = smf + Ly::OFF_C;
  float* Ws = smf + Ly::OFF_W;
  float* zs = smf + Ly::OFF_Z;
  float* gs = smf + Ly::OFF_G;
  float* Rs = smf + Ly::OFF_R;
  float* qz = smf + Ly::OFF_QZ;
  float* sc = smf + Ly::OFF_SC;
  for (int e = tid; e < HD * VS; e += NTM) Cs[e] = 0.f;
  for (int e = tid; e < HD; e += NTM) zs[e] = 0.f;
  if (tid == 0) sc[0] = -INFINITY;
  const float* F = a.feat + (size_t)lp * Pm * NF;
  float* prio = a.prio + (size_t)lp * Pm;
  const float* av = a.ms.a + (size_t)h * HH;
  const float bsc = a.ms.b[h];
  __syncthreads();

  for (int t0 = 0; t0 < P; t0 += CL) {
    // ---- load the chunk: k~, v~ of tokens t0.., q~ of the tokens they read out ------
    for (int e = tid; e < CL * (HD / 4); e += NTM) {
      const int r = e / (HD / 4), c4 = e - r * (HD / 4);
      const int t = t0 + r, u = t - D;
      float4 kv = make_float4(0.f, 0.f, 0.f, 0.f), qv = kv;
      if (t < P) kv = *reinterpret_cast<const float4*>(F + (size_t)t * NF + 4 * c4);
      if (t < P && u >= 0) qv = *reinterpret_cast<const float4*>(F + (size_t)u * NF + HD + HH + 4 * c4);
      *reinterpret_cast<float4*>(Ks + r * QS + 4 * c4) = kv;
      *reinterpret_cast<float4*>(Qs + r * QS + 4 * c4) = qv;
    }
    for (int e = tid; e < CL * HH; e += NTM) {
      const int r = e / HH, j = e - r * HH;
      const int t = t0 + r;
      Vs[r * VS + j] = t < P ? F[(size_t)t * NF + HD + j] : 0.f;
    }
    // gates: warp 0 scans the chunk's log forget gates (two tokens per lane)
    if (warp == 0) {
      const float m = sc[0];
      float lfv[2], aiv[2];
#pragma unroll
      for (int k = 0; k < 2; ++k) {
        const int t = t0 + 2 * lane + k;
        const bool in = t < P;
        aiv[k] = in ? F[(size_t)t * NF + 2 * HD + HH] : -INFINITY;
        lfv[k] = in ? -softplus(-F[(size_t)t * NF + 2 * HD + HH + 1]) : 0.f;
      }
      float f1 = lfv[0] + lfv[1], inc = f1;          // inclusive scan over lane pairs
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const float y = __shfl_up_sync(0xffffffffu, inc, o);
        if (lane >= o) inc += y;
      }
      const float Fa = inc - f1 + lfv[0], Fb = inc;  // F of tokens 2 lane, 2 lane + 1
      const float ga = aiv[0] - Fa, gb = aiv[1] - Fb;
      float gm = fmaxf(ga, gb), run = gm;            // inclusive prefix max
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const float y = __shfl_up_sync(0xffffffffu, run, o);
        if (lane >= o) run = fmaxf(run, y);
      }
      const float prev = __shfl_up_sync(0xffffffffu, run, 1);
      const float before = lane == 0 ? -INFINITY : prev;
      gs[2 * lane] = ga;
      gs[2 * lane + 1] = gb;
      Rs[2 * lane] = fmaxf(m, fmaxf(before, ga));
      Rs[2 * lane + 1] = fmaxf(m, run);
      if (lane == 31) sc[1] = Fb;                    // F of the chunk's last token
      (void)gm;
    }
    __syncthreads();

    // ---- S = q~ K^T -> W;  q~ C -> registers;  q~ . z ----------------------------------
    {
      float acc[4][4];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
#pragma unroll 4
      for (int c = 0; c < HD; c += 4) {
        float4 qa[4], kb[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) qa[i] = *reinterpret_cast<const float4*>(Qs + (ty + 16 * i) * QS + c);
#pragma unroll
        for (int j = 0; j < 4; ++j) kb[j] = *reinterpret_cast<const float4*>(Ks + (tx + 16 * j) * QS + c);
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
          for (int j = 0; j < 4; ++j)
            acc[i][j] = fmaf(qa[i].x, kb[j].x, fmaf(qa[i].y, kb[j].y,
                        fmaf(qa[i].z, kb[j].z, fmaf(qa[i].w, kb[j].w, acc[i][j]))));
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int t = ty + 16 * i;
        const float R = Rs[t];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const int s = tx + 16 * j;
          Ws[t * WS + s] = (s <= t) ? __expf(gs[s] - R) * acc[i][j] : 0.f;
        }
      }
    }
    float num[4][NB];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < NB; ++j) num[i][j] = 0.f;
#pragma unroll 2
    for (int c = 0; c < HD; c += 4) {
      float4 qa[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) qa[i] = *reinterpret_cast<const float4*>(Qs + (ty + 16 * i) * QS + c);
#pragma unroll
      for (int j = 0; j < NB; ++j) {
        const int col = tx + 16 * j;
        const float c0 = Cs[(c + 0) * VS + col], c1 = Cs[(c + 1) * VS + col];
        const float c2 = Cs[(c + 2) * VS + col], c3 = Cs[(c + 3) * VS + col];
#pragma unroll
        for (int i = 0; i < 4; ++i)
          num[i][j] = fmaf(qa[i].x, c0, fmaf(qa[i].y, c1, fmaf(qa[i].z, c2, fmaf(qa[i].w, c3, num[i][j]))));
      }
    }
    // q~ . z: warp w takes rows 8w .. 8w + 7
#pragma unroll
    for (int rr = 0; rr < CL / 8; ++rr) {
      const int t = warp * (CL / 8) + rr;
      float s = 0.f;
      for (int c = lane; c < HD; c += 32) s = fmaf(Qs[t * QS + c], zs[c], s);
      s = warp_sum(s);
      if (lane == 0) qz[t] = s;
    }
    __syncthreads();

    // ---- readout rows: num = e^{m-R} q~C + W V, den = e^{m-R} q~.z + sum_s W ----------
    {
      const float m = sc[0];
      float den[4], coef[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int t = ty + 16 * i;
        coef[i] = __expf(m - Rs[t]);
        den[i] = 0.f;
#pragma unroll
        for (int j = 0; j < NB; ++j) num[i][j] *= coef[i];
      }
#pragma unroll 4
      for (int s = 0; s < CL; s += 4) {
        float4 wa[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          wa[i] = *reinterpret_cast<const float4*>(Ws + (ty + 16 * i) * WS + s);
          den[i] += (wa[i].x + wa[i].y) + (wa[i].z + wa[i].w);
        }
#pragma unroll
        for (int j = 0; j < NB; ++j) {
          const int col = tx + 16 * j;
          const float v0 = Vs[(s + 0) * VS + col], v1 = Vs[(s + 1) * VS + col];
          const float v2 = Vs[(s + 2) * VS + col], v3 = Vs[(s + 3) * VS + col];
#pragma unroll
          for (int i = 0; i < 4; ++i)
            num[i][j] = fmaf(wa[i].x, v0, fmaf(wa[i].y, v1, fmaf(wa[i].z, v2, fmaf(wa[i].w, v3, num[i][j]))));
        }
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int t = ty + 16 * i;
        const float dn = fmaf(coef[i], qz[t], den[i]);
        float r = 0.f;
#pragma unroll
        for (int j = 0; j < NB; ++j) {
          const float hv = num[i][j] / dn;
          r = fmaf(av[tx + 16 * j], hv / (1.f + expf(-hv)), r);
        }
#pragma unroll
        for (int o = 1; o < 16; o <<= 1) r += __shfl_xor_sync(0xffffffffu, r, o);
        const int T = t0 + t, u = T - D;
        if (tx == 0 && T < P && u >= 0) {
          float rv = r + bsc;
          if (a.override_) rv = a.override_[(size_t)lp * Pm + u];
          prio[u] = static_priority(canon_score(rv), u, a.st.log_gamma, h);
        }
      }
    }
    // ---- state update C' = e^{m-R_L} C + K^T diag(e^{g-R_L}) V;  z likewise -------------
    {
      const float RL = Rs[CL - 1];
      const float wc = __expf(sc[0] - RL);
      constexpr int NR = HD / 16;
      float acc[NR][NB];
#pragma unroll
      for (int i = 0; i < NR; ++i)
#pragma unroll
        for (int j = 0; j < NB; ++j) acc[i][j] = wc * Cs[(ty + 16 * i) * VS + tx + 16 * j];
#pragma unroll 4
      for (int s = 0; s < CL; ++s) {
        const float w = __expf(gs[s] - RL);
        float vb[NB];
#pragma unroll
        for (int j = 0; j < NB; ++j) vb[j] = w * Vs[s * VS + tx + 16 * j];
#pragma unroll
        for (int i = 0; i < NR; ++i) {
          const float kk = Ks[s * QS + ty + 16 * i];
#pragma unroll
          for (int j = 0; j < NB; ++j) acc[i][j] = fmaf(kk, vb[j], acc[i][j]);
        }
      }
      float zn = 0.f;
      if (tid < HD) {
        zn = wc * zs[tid];
        for (int s = 0; s < CL; ++s) zn = fmaf(__expf(gs[s] - RL), Ks[s * QS + tid], zn);
      }
      __syncthreads();                 // every read of C, z and the scalars is done
#pragma unroll
      for (int i = 0; i < NR; ++i)
#pragma unroll
        for (int j = 0; j < NB; ++j) Cs[(ty + 16 * i) * VS + tx + 16 * j] = acc[i][j];
      if (tid < HD) zs[tid] = zn;
      if (tid == 0) sc[0] = sc[1] + RL;
    }
    __syncthreads();
  }
  float* Cg = a.ms.C + (size_t)pair * HD * HH;
  for (int e = tid; e < HD * HH; e += NTM) Cg[e] = Cs[(e / HH) * VS + (e % HH)];
  for (int e = tid; e < HD; e += NTM) a.ms.z[(size_t)pair * HD + e] = zs[e];
  if (tid == 0) a.ms.m[pair] = sc[0];
}

template <int HD>
size_t chunk_smem() { return (size_t)ChunkLayout<HD>::FLOATS * 4; }

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
  if (e == cudaSuccess)
    e = dm.d == 128 ? raise_smem_limit(mlstm_chunk_kernel<128>, chunk_smem<128>())
                    : raise_smem_limit(mlstm_chunk_kernel<64>, chunk_smem<64>());
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
  if (dm.d == 128)
    mlstm_chunk_kernel<128><<<pairs, NTM, chunk_smem<128>(), stream>>>(sa);
  else
    mlstm_chunk_kernel<64><<<pairs, NTM, chunk_smem<64>(), stream>>>(sa);
  return cudaGetLastError();
}

}  // namespace kvpop
