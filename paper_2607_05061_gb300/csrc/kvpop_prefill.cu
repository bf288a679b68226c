// Prompt compression: the running top-k of Sec. 3.2 / App. C.1 evaluated once
// for a whole prompt.
//
// Kernel 1 scores every eligible prompt token u <= P - 1 - D with the delayed
// scorer (Sec. 3.3, App. E.4): the stateless MLP of App. E.2 on
// [k_u; v_u; qbar_u], qbar_u = mean of the queries u+1..u+D over the G query
// heads, and turns it into its static priority (App. B.3).  A CTA scores UT
// consecutive tokens of one (sequence, KV head) so each row of W1 it loads feeds
// UT rows.
//
// Kernel 2 keeps, per (sequence, KV head), the sinks u < s plus the top (B - s)
// of the rest by (priority desc, position asc) -- an exact 4-pass radix select
// on the order-preserving bit pattern of the fp32 priority, ties resolved by
// position -- writes them to slots 0.. in ascending position, and loads the
// window with the last min(P, D) tokens.
#include <algorithm>

#include "kvpop_argmin.cuh"

namespace kvpop {
namespace {

constexpr int UT = 32;          // prompt tokens scored per CTA
constexpr int NT1 = 256;
constexpr int NT2 = 512;

template <typename T>
struct ScoreArgs {
  State st;
  Dims dm;
  const T* Q;                   // [n_seq][H*G][Pmax][d]
  const T* K;                   // [n_seq][H][Pmax][d]
  const T* V;
  const int32_t* plen;          // [n_seq]
  const float* override_;       // [n_seq][H][Pmax] or nullptr
  float* prio;                  // [n_seq][H][Pmax]
  int Pmax;
};

__device__ __forceinline__ uint32_t order_key(float f) {
  const uint32_t b = __float_as_uint(f);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

template <typename T>
__global__ void __launch_bounds__(NT1) prefill_score_kernel(ScoreArgs<T> a) {
  const Dims& dm = a.dm;
  const int d = dm.d, D = dm.D, G = dm.G, F = dm.F, H = dm.H;
  const int lp = blockIdx.y;                 // local pair = b_local * H + h
  const int bl = lp / H, h = lp - bl * H;
  const int P = a.plen[bl];
  const int n_elig = max(P - D, 0);
  const int u0 = blockIdx.x * UT;
  if (u0 >= n_elig) return;
  const int nrow = min(UT, n_elig - u0);
  const size_t Pm = a.Pmax;
  float* prio_out = a.prio + (size_t)lp * Pm;

  if (a.override_) {
    const float* ov = a.override_ + (size_t)lp * Pm;
    for (int r = threadIdx.x; r < nrow; r += NT1) {
      const int u = u0 + r;
      prio_out[u] = static_priority(canon_score(ov[u]), u, a.st.log_gamma, h);
    }
    return;
  }

  extern __shared__ __align__(16) unsigned char smem[];
  const int in_dim = 3 * d;
  float* Xt = reinterpret_cast<float*>(smem);          // [3d][UT]
  float* qmc = Xt + in_dim * UT;                        // [32][d] query means of a position chunk
  float* red = qmc + 32 * d;                            // [UT][NT1]

  const T* Kp = a.K + ((size_t)bl * H + h) * Pm * d;
  const T* Vp = a.V + ((size_t)bl * H + h) * Pm * d;
  const T* Qp = a.Q + ((size_t)bl * H * G + (size_t)h * G) * Pm * d;

  // k_u, v_u rows
  for (int idx = threadIdx.x; idx < UT * d; idx += NT1) {
    const int r = idx / d, i = idx - r * d;
    float kk = 0.f, vv = 0.f;
    if (r < nrow) {
      kk = to_f(Kp[(size_t)(u0 + r) * d + i]);
      vv = to_f(Vp[(size_t)(u0 + r) * d + i]);
    }
    Xt[i * UT + r] = kk;
    Xt[(d + i) * UT + r] = vv;
  }
  // qbar_u: positions u+1..u+D in order; thread (i, row group) accumulates its rows
  {
    const int groups = NT1 / d;                // 2 (d = 128) or 4 (d = 64)
    const int i = threadIdx.x % d, rg = threadIdx.x / d;
    const int rows_per = UT / groups;
    float acc[UT / 2];
#pragma unroll
    for (int k = 0; k < UT / 2; ++k) acc[k] = 0.f;
    const int tlo = u0 + 1, thi = u0 + nrow - 1 + D;  // positions needed (inclusive)
    for (int c = tlo; c <= thi; c += 32) {
      __syncthreads();
      for (int idx = threadIdx.x; idx < 32 * d; idx += NT1) {
        const int tt = idx / d, ii = idx - tt * d;
        const int t = c + tt;
        float s = 0.f;
        if (t <= thi)
          for (int g = 0; g < G; ++g) s += to_f(Qp[((size_t)g * Pm + t) * d + ii]);
        qmc[tt * d + ii] = s * (1.0f / (float)G);
      }
      __syncthreads();
      for (int k = 0; k < rows_per; ++k) {
        const int r = rg * rows_per + k;
        const int lo = max(u0 + r + 1, c), hi = min(u0 + r + D, min(c + 31, thi));
        for (int t = lo; t <= hi; ++t) acc[k] += qmc[(t - c) * d + i];
      }
    }
    for (int k = 0; k < rows_per; ++k) {
      const int r = rg * rows_per + k;
      Xt[(2 * d + i) * UT + r] = (r < nrow) ? acc[k] / (float)D : 0.f;
    }
  }
  __syncthreads();

  // hidden layer and output projection: thread f (and f + NT1, ...) for all UT rows
  const int Fp = dm.Fp;
  const float* W1 = a.st.W1 + (size_t)h * in_dim * Fp;
  const float* b1 = a.st.b1 + (size_t)h * Fp;
  const float* w2 = a.st.w2 + (size_t)h * Fp;
  float part[UT];
#pragma unroll
  for (int r = 0; r < UT; ++r) part[r] = 0.f;
  for (int f = threadIdx.x; f < F; f += NT1) {
    float acc[UT];
    const float bias = b1[f];
#pragma unroll
    for (int r = 0; r < UT; ++r) acc[r] = bias;
#pragma unroll 2
    for (int i = 0; i < in_dim; ++i) {
      const float w = __ldg(W1 + (size_t)i * Fp + f);
      const float4* xr = reinterpret_cast<const float4*>(Xt + i * UT);
#pragma unroll
      for (int r4 = 0; r4 < UT / 4; ++r4) {
        const float4 x = xr[r4];
        acc[4 * r4 + 0] = fmaf(x.x, w, acc[4 * r4 + 0]);
        acc[4 * r4 + 1] = fmaf(x.y, w, acc[4 * r4 + 1]);
        acc[4 * r4 + 2] = fmaf(x.z, w, acc[4 * r4 + 2]);
        acc[4 * r4 + 3] = fmaf(x.w, w, acc[4 * r4 + 3]);
      }
    }
    const float wf = w2[f];
#pragma unroll
    for (int r = 0; r < UT; ++r) part[r] = fmaf(wf, scorer_act(acc[r], dm.act), part[r]);
  }
#pragma unroll
  for (int r = 0; r < UT; ++r) red[r * NT1 + threadIdx.x] = part[r];
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int r = warp; r < nrow; r += NT1 / 32) {
    float s = 0.f;
    for (int k = lane; k < NT1; k += 32) s += red[r * NT1 + k];
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
    if (lane == 0) {
      const int u = u0 + r;
      const float rr = canon_score(s + a.st.b2[h]);
      prio_out[u] = static_priority(rr, u, a.st.log_gamma, h);
    }
  }
}

// Register-tiled version for F in {128, 256}: a CTA scores UT2 = 64 consecutive
// tokens; the scorer inputs X [3d][64] sit in shared memory (fp32, rows padded
// to 68 floats), W1 streams
// through in chunks of 32 input rows (double-buffered cp.async), and each thread
// accumulates 4 tokens x NH hidden units (NH = F / 16), so every W1 row loaded
// serves 64 tokens and every shared-memory read feeds 4 NH multiply-adds.
constexpr int UT2 = 64;
constexpr int XS2 = UT2 + 4;       // row stride of X in shared memory (float4-aligned, few bank conflicts)
constexpr int KC2 = 32;
constexpr int NT3 = 256;

template <int NH>
__host__ __device__ constexpr int gemm_w_bytes() { return 2 * KC2 * 16 * NH * 4; }

template <typename T, int NH>
__global__ void __launch_bounds__(NT3) prefill_score_gemm_kernel(ScoreArgs<T> a) {
  constexpr int F = 16 * NH;
  const Dims& dm = a.dm;
  const int d = dm.d, D = dm.D, G = dm.G, H = dm.H;
  const int lp = blockIdx.y;
  const int bl = lp / H, h = lp - bl * H;
  const int P = a.plen[bl];
  const int n_elig = max(P - D, 0);
  const int u0 = blockIdx.x * UT2;
  if (u0 >= n_elig) return;
  const int nrow = min(UT2, n_elig - u0);
  const size_t Pm = a.Pmax;
  const int tid = threadIdx.x;
  const int in_dim = 3 * d;

  extern __shared__ __align__(16) unsigned char smem[];
  float* Xs = reinterpret_cast<float*>(smem);                    // [3d][XS2]
  float* Wc = Xs + (size_t)in_dim * XS2;                          // [2][KC2][F]; staging first
  const T* Kp = a.K + ((size_t)bl * H + h) * Pm * d;
  const T* Vp = a.V + ((size_t)bl * H + h) * Pm * d;
  const T* Qp = a.Q + ((size_t)bl * H * G + (size_t)h * G) * Pm * d;

  // Staging with 16-byte loads, NB items per thread issued before any is used.
  constexpr int CE = 16 / (int)sizeof(T);         // elements per 16-byte chunk
  constexpr int NB = 4;
  const int cpr = d / CE;                         // chunks per row
  auto unpack = [](const uint4& v, float (&f)[CE]) {
    const T* e = reinterpret_cast<const T*>(&v);
#pragma unroll
    for (int k = 0; k < CE; ++k) f[k] = to_f(e[k]);
  };
  // k_u, v_u -> X rows 0..2d-1 (transposed: X[channel][token])
  for (int base = tid; base < UT2 * cpr; base += NT3 * NB) {
    uint4 kk[NB], vv[NB];
#pragma unroll
    for (int b = 0; b < NB; ++b) {
      const int it = base + b * NT3;
      const int r = it / cpr, c = it - r * cpr;
      kk[b] = vv[b] = make_uint4(0u, 0u, 0u, 0u);
      if (it < UT2 * cpr && r < nrow) {
        kk[b] = __ldg(reinterpret_cast<const uint4*>(Kp + (size_t)(u0 + r) * d) + c);
        vv[b] = __ldg(reinterpret_cast<const uint4*>(Vp + (size_t)(u0 + r) * d) + c);
      }
    }
#pragma unroll
    for (int b = 0; b < NB; ++b) {
      const int it = base + b * NT3;
      if (it >= UT2 * cpr) break;
      const int r = it / cpr, c = it - r * cpr;
      float fk[CE], fv[CE];
      unpack(kk[b], fk);
      unpack(vv[b], fv);
#pragma unroll
      for (int k = 0; k < CE; ++k) {
        Xs[(c * CE + k) * XS2 + r] = fk[k];
        Xs[(d + c * CE + k) * XS2 + r] = fv[k];
      }
    }
  }
  // query means of positions u0+1 .. u0+nrow-1+D, then qbar_u = mean of the D after u
  float* qm = Wc;                                                  // [UT2 + D - 1][d]
  const int npos = nrow - 1 + D;
  for (int base = tid; base < npos * cpr; base += NT3 * NB) {
    float acc[NB][CE];
#pragma unroll
    for (int b = 0; b < NB; ++b)
#pragma unroll
      for (int k = 0; k < CE; ++k) acc[b][k] = 0.f;
    for (int g = 0; g < G; ++g) {
      uint4 qv[NB];
#pragma unroll
      for (int b = 0; b < NB; ++b) {
        const int it = base + b * NT3;
        const int tt = it / cpr, c = it - tt * cpr;
        qv[b] = make_uint4(0u, 0u, 0u, 0u);
        if (it < npos * cpr)
          qv[b] = __ldg(reinterpret_cast<const uint4*>(Qp + ((size_t)g * Pm + u0 + 1 + tt) * d) + c);
      }
#pragma unroll
      for (int b = 0; b < NB; ++b) {
        float f[CE];
        unpack(qv[b], f);
#pragma unroll
        for (int k = 0; k < CE; ++k) acc[b][k] += f[k];
      }
    }
#pragma unroll
    for (int b = 0; b < NB; ++b) {
      const int it = base + b * NT3;
      if (it >= npos * cpr) break;
      const int tt = it / cpr, c = it - tt * cpr;
#pragma unroll
      for (int k = 0; k < CE; ++k) qm[tt * d + c * CE + k] = acc[b][k] * (1.0f / (float)G);
    }
  }
  __syncthreads();
  for (int idx = tid; idx < UT2 * d; idx += NT3) {
    const int r = idx / d, i = idx - r * d;
    float acc = 0.f;
    if (r < nrow)
      for (int j = 0; j < D; ++j) acc += qm[(r + j) * d + i];
    Xs[(2 * d + i) * XS2 + r] = r < nrow ? acc / (float)D : 0.f;
  }
  __syncthreads();

  const float* W1 = a.st.W1 + (size_t)h * in_dim * dm.Fp;       // Fp == F on this path
  const uint32_t wbase = (uint32_t)__cvta_generic_to_shared(Wc);
  auto load_chunk = [&](int c, int buf) {
    const float* src = W1 + (size_t)c * KC2 * F;
    for (int i = tid; i < KC2 * F / 4; i += NT3)
      asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(wbase + (uint32_t)((buf * KC2 * F + i * 4) * 4)),
                   "l"(src + i * 4)
                   : "memory");
    asm volatile("cp.async.commit_group;" ::: "memory");
  };
  const int tm = tid & 15, tn = tid >> 4;
  float acc[4][NH];
#pragma unroll
  for (int r = 0; r < 4; ++r)
#pragma unroll
    for (int f = 0; f < NH; ++f) acc[r][f] = 0.f;
  const int nchunk = in_dim / KC2;
  load_chunk(0, 0);
  for (int c = 0; c < nchunk; ++c) {
    if (c + 1 < nchunk) {
      load_chunk(c + 1, (c + 1) & 1);
      asm volatile("cp.async.wait_group 1;" ::: "memory");
    } else {
      asm volatile("cp.async.wait_group 0;" ::: "memory");
    }
    __syncthreads();
    const float* wb = Wc + (c & 1) * KC2 * F + tn * NH;
    const float* xb = Xs + (size_t)c * KC2 * XS2 + tm * 4;
#pragma unroll 4
    for (int kk = 0; kk < KC2; ++kk) {
      const float4 x = *reinterpret_cast<const float4*>(xb + kk * XS2);
#pragma unroll
      for (int f4 = 0; f4 < NH / 4; ++f4) {
        const float4 w = *reinterpret_cast<const float4*>(wb + kk * F + f4 * 4);
        acc[0][4 * f4 + 0] = fmaf(x.x, w.x, acc[0][4 * f4 + 0]);
        acc[0][4 * f4 + 1] = fmaf(x.x, w.y, acc[0][4 * f4 + 1]);
        acc[0][4 * f4 + 2] = fmaf(x.x, w.z, acc[0][4 * f4 + 2]);
        acc[0][4 * f4 + 3] = fmaf(x.x, w.w, acc[0][4 * f4 + 3]);
        acc[1][4 * f4 + 0] = fmaf(x.y, w.x, acc[1][4 * f4 + 0]);
        acc[1][4 * f4 + 1] = fmaf(x.y, w.y, acc[1][4 * f4 + 1]);
        acc[1][4 * f4 + 2] = fmaf(x.y, w.z, acc[1][4 * f4 + 2]);
        acc[1][4 * f4 + 3] = fmaf(x.y, w.w, acc[1][4 * f4 + 3]);
        acc[2][4 * f4 + 0] = fmaf(x.z, w.x, acc[2][4 * f4 + 0]);
        acc[2][4 * f4 + 1] = fmaf(x.z, w.y, acc[2][4 * f4 + 1]);
        acc[2][4 * f4 + 2] = fmaf(x.z, w.z, acc[2][4 * f4 + 2]);
        acc[2][4 * f4 + 3] = fmaf(x.z, w.w, acc[2][4 * f4 + 3]);
        acc[3][4 * f4 + 0] = fmaf(x.w, w.x, acc[3][4 * f4 + 0]);
        acc[3][4 * f4 + 1] = fmaf(x.w, w.y, acc[3][4 * f4 + 1]);
        acc[3][4 * f4 + 2] = fmaf(x.w, w.z, acc[3][4 * f4 + 2]);
        acc[3][4 * f4 + 3] = fmaf(x.w, w.w, acc[3][4 * f4 + 3]);
      }
    }
    __syncthreads();                 // the buffer is refilled two chunks later
  }
  // hidden activation and output projection; partial sums of the 16 hidden groups
  const float* b1 = a.st.b1 + (size_t)h * dm.Fp + tn * NH;
  const float* w2 = a.st.w2 + (size_t)h * dm.Fp + tn * NH;
  float* red = Wc;                                                 // [16][UT2]
  float part[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int f = 0; f < NH; ++f) {
    const float bb = b1[f], ww = w2[f];
#pragma unroll
    for (int r = 0; r < 4; ++r) part[r] = fmaf(ww, scorer_act(acc[r][f] + bb, dm.act), part[r]);
  }
#pragma unroll
  for (int r = 0; r < 4; ++r) red[tn * UT2 + tm * 4 + r] = part[r];
  __syncthreads();
  if (tid < nrow) {
    float sum = 0.f;
    for (int g = 0; g < 16; ++g) sum += red[g * UT2 + tid];
    const int u = u0 + tid;
    float* prio_out = a.prio + (size_t)lp * Pm;
    prio_out[u] = static_priority(canon_score(sum + a.st.b2[h]), u, a.st.log_gamma, h);
  }
}

template <typename T>
struct SelectArgs {
  State st;
  Dims dm;
  const T* Q;
  const T* K;
  const T* V;
  const int32_t* plen;
  const float* prio;
  int first_seq;
  int Pmax;
};

__device__ __forceinline__ int block_excl_scan_flag(bool f, int* wsum, int& total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const unsigned bal = __ballot_sync(0xffffffffu, f);
  const int within = __popc(bal & ((1u << lane) - 1u));
  if (lane == 0) wsum[warp] = __popc(bal);
  __syncthreads();
  int before = 0, tot = 0;
  for (int w = 0; w < NT2 / 32; ++w) {
    const int x = wsum[w];
    if (w < warp) before += x;
    tot += x;
  }
  __syncthreads();
  total = tot;
  return before + within;
}

template <typename T>
__global__ void __launch_bounds__(NT2) prefill_select_kernel(SelectArgs<T> a) {
  const Dims& dm = a.dm;
  const int d = dm.d, D = dm.D, G = dm.G, H = dm.H, B = dm.B, s = dm.s;
  const int lp = blockIdx.x;
  const int bl = lp / H, h = lp - bl * H;
  const int pair = (a.first_seq + bl) * H + h;
  const int P = a.plen[bl];
  const int n_elig = max(P - D, 0);
  const int s_eff = min(s, n_elig);
  const int n_long = n_elig - s_eff;
  const int ksel = min(B - s, n_long);
  const bool selecting = n_long > ksel;
  const size_t Pm = a.Pmax;
  const float* pr = a.prio + (size_t)lp * Pm;

  __shared__ unsigned hist[256];
  __shared__ unsigned s_prefix, s_mask;
  __shared__ int s_k;
  __shared__ int wsum[NT2 / 32];

  uint32_t kth = 0;
  int need_eq = 0;
  if (selecting) {
    uint32_t prefix = 0, mask = 0;
    int k = ksel;
    for (int shift = 24; shift >= 0; shift -= 8) {
      for (int i = threadIdx.x; i < 256; i += NT2) hist[i] = 0;
      __syncthreads();
      for (int u = s_eff + threadIdx.x; u < n_elig; u += NT2) {
        const uint32_t key = order_key(pr[u]);
        if ((key & mask) == prefix) atomicAdd(&hist[(key >> shift) & 255u], 1u);
      }
      __syncthreads();
      if (threadIdx.x == 0) {
        int cum = 0;
        for (int dg = 255; dg >= 0; --dg) {
          const int c = (int)hist[dg];
          if (cum + c >= k) { s_prefix = prefix | ((uint32_t)dg << shift); s_k = k - cum; break; }
          cum += c;
        }
        s_mask = mask | (255u << shift);
      }
      __syncthreads();
      prefix = s_prefix;
      mask = s_mask;
      k = s_k;
      __syncthreads();
    }
    kth = prefix;
    need_eq = k;
  }

  float* sc = a.st.score + (size_t)pair * B;
  int32_t* ps = a.st.pos + (size_t)pair * B;
  int run_keep = 0, run_eq = 0;
  for (int base = 0; base < n_elig; base += NT2) {
    const int u = base + threadIdx.x;
    const bool in = u < n_elig;
    float pv = 0.f;
    uint32_t key = 0;
    if (in) { pv = pr[u]; key = order_key(pv); }
    const bool eq = in && selecting && u >= s_eff && key == kth;
    int tot_eq;
    const int eq_rank = run_eq + block_excl_scan_flag(eq, wsum, tot_eq);
    const bool keep = in && (u < s_eff || !selecting || key > kth || (eq && eq_rank < need_eq));
    int tot_keep;
    const int slot = run_keep + block_excl_scan_flag(keep, wsum, tot_keep);
    if (keep) { sc[slot] = pv; ps[slot] = u; }
    run_eq += tot_eq;
    run_keep += tot_keep;
  }
  __syncthreads();
  const int nkept = run_keep;

  // copy kept rows, one warp per row
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int R = d * (int)sizeof(T);
  const int chunks = R / 16;
  const unsigned char* Kp = reinterpret_cast<const unsigned char*>(a.K) + ((size_t)bl * H + h) * Pm * R;
  const unsigned char* Vp = reinterpret_cast<const unsigned char*>(a.V) + ((size_t)bl * H + h) * Pm * R;
  unsigned char* sK = static_cast<unsigned char*>(a.st.slotK) + (size_t)pair * B * R;
  unsigned char* sV = static_cast<unsigned char*>(a.st.slotV) + (size_t)pair * B * R;
  dcheck(nkept <= B, a.st.err, DEVERR_INDEX);
  for (int slot = warp; slot < min(nkept, B); slot += NT2 / 32) {
    const int u = ps[slot];
    if (!dcheck(u >= 0 && u < P, a.st.err, DEVERR_INDEX)) continue;
    for (int c = lane; c < chunks; c += 32) {
      reinterpret_cast<uint4*>(sK + (size_t)slot * R)[c] =
          reinterpret_cast<const uint4*>(Kp + (size_t)u * R)[c];
      reinterpret_cast<uint4*>(sV + (size_t)slot * R)[c] =
          reinterpret_cast<const uint4*>(Vp + (size_t)u * R)[c];
    }
  }
  // window: positions max(0, P-D) .. P-1 at ring index t % D
  unsigned char* rK = static_cast<unsigned char*>(a.st.ringK) + (size_t)pair * D * R;
  unsigned char* rV = static_cast<unsigned char*>(a.st.ringV) + (size_t)pair * D * R;
  float* rQ = a.st.ringQm + (size_t)pair * D * d;
  const T* Qp = a.Q + ((size_t)bl * H * G + (size_t)h * G) * Pm * d;
  for (int t = max(0, P - D) + warp; t < P; t += NT2 / 32) {
    const int ri = t % D;
    for (int c = lane; c < chunks; c += 32) {
      reinterpret_cast<uint4*>(rK + (size_t)ri * R)[c] = reinterpret_cast<const uint4*>(Kp + (size_t)t * R)[c];
      reinterpret_cast<uint4*>(rV + (size_t)ri * R)[c] = reinterpret_cast<const uint4*>(Vp + (size_t)t * R)[c];
    }
    for (int i = lane; i < d; i += 32) {
      float acc = 0.f;
      for (int g = 0; g < G; ++g) acc += to_f(Qp[((size_t)g * Pm + t) * d + i]);
      rQ[(size_t)ri * d + i] = acc * (1.0f / (float)G);
    }
  }
  __syncthreads();
  if (nkept == B) {
    // block minima over the long-range slots, then the head minimum
    const int NB = min_blocks(B);
    float* bsc = a.st.blk_score + (size_t)pair * NB;
    int32_t* bsl = a.st.blk_slot + (size_t)pair * NB;
    for (int k = warp; k < NB; k += NT2 / 32) {
      float m;
      int mi;
      block_min(sc, s, B, k, -1, 0.f, m, mi);
      if (lane == 0) { bsc[k] = m; bsl[k] = mi; }
    }
    __syncthreads();
    if (warp == 0) {
      float m;
      int mi;
      blocks_min(bsc, bsl, NB, -1, 0.f, 0, m, mi);
      if (lane == 0) { a.st.min_score[pair] = m; a.st.min_slot[pair] = mi; }
    }
  } else if (threadIdx.x == 0) {
    a.st.min_score[pair] = INFINITY;
    a.st.min_slot[pair] = -1;
  }
  if (threadIdx.x == 0) {
    a.st.nvalid[pair] = nkept;
    a.st.len[pair] = P;
  }
}

size_t score_smem(const Dims& dm) { return ((size_t)3 * dm.d * UT + 32 * dm.d + UT * NT1) * 4; }

// the register-tiled scorer serves F = 128 / 256 when its buffers fit
int gemm_nh(const Dims& dm) {
  if (dm.F != dm.Fp || !(dm.F == 128 || dm.F == 256)) return 0;
  return dm.F / 16;
}
size_t gemm_smem(const Dims& dm) {
  const size_t x = (size_t)3 * dm.d * XS2 * 4;
  const size_t wbytes = (size_t)2 * KC2 * dm.F * 4;
  const size_t stage = (size_t)(UT2 - 1 + dm.D) * dm.d * 4;
  const size_t red = (size_t)16 * UT2 * 4;
  return x + std::max(std::max(wbytes, stage), red);
}
bool gemm_ok(const Dims& dm) { return gemm_nh(dm) != 0 && gemm_smem(dm) <= 227 * 1024; }

}  // namespace

cudaError_t prepare_prefill(const Dims& dm) {
  const int smem = (int)score_smem(dm);
  cudaError_t e;
  if (dm.dtype == KVPOP_F32)
    e = raise_smem_limit(prefill_score_kernel<float>, smem);
  else
    e = raise_smem_limit(prefill_score_kernel<bf16>, smem);
  if (e != cudaSuccess || !gemm_ok(dm)) return e;
  const int gs = (int)gemm_smem(dm);
  if (dm.dtype == KVPOP_F32)
    return dm.F == 256 ? raise_smem_limit(prefill_score_gemm_kernel<float, 16>, gs)
                       : raise_smem_limit(prefill_score_gemm_kernel<float, 8>, gs);
  return dm.F == 256 ? raise_smem_limit(prefill_score_gemm_kernel<bf16, 16>, gs)
                     : raise_smem_limit(prefill_score_gemm_kernel<bf16, 8>, gs);
}

template <typename T>
static cudaError_t prefill_t(const State& st, const Dims& dm, const void* Q, const void* K,
                             const void* V, const int32_t* plen, int first_seq, int n_seq,
                             int Pmax, const float* override_, float* prio, const void* tf32_maps,
                             cudaStream_t stream) {
  const int pairs = n_seq * dm.H;
  ScoreArgs<T> sa{st, dm, (const T*)Q, (const T*)K, (const T*)V, plen,
                  override_ ? override_ : nullptr, prio, Pmax};
  if (Pmax > 0) {
    if (!override_ && tf32_maps) {
      cudaError_t e = launch_score_tf32(st, dm, tf32_maps, Q, K, V, plen, n_seq, Pmax, prio, stream);
      if (e != cudaSuccess) return e;
    } else if (!override_ && gemm_ok(dm)) {
      dim3 g2((Pmax + UT2 - 1) / UT2, pairs);
      if (dm.F == 256) prefill_score_gemm_kernel<T, 16><<<g2, NT3, gemm_smem(dm), stream>>>(sa);
      else prefill_score_gemm_kernel<T, 8><<<g2, NT3, gemm_smem(dm), stream>>>(sa);
    } else {
      dim3 g1((Pmax + UT - 1) / UT, pairs);
      prefill_score_kernel<T><<<g1, NT1, override_ ? 0 : score_smem(dm), stream>>>(sa);
    }
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  SelectArgs<T> sel{st, dm, (const T*)Q, (const T*)K, (const T*)V, plen, prio, first_seq, Pmax};
  prefill_select_kernel<T><<<pairs, NT2, 0, stream>>>(sel);
  return cudaGetLastError();
}

cudaError_t launch_prefill_select(const State& st, const Dims& dm, const void* Q, const void* K,
                                  const void* V, const int32_t* plen, int first_seq, int n_seq,
                                  int Pmax, const float* prio, cudaStream_t stream) {
  const int pairs = n_seq * dm.H;
  if (dm.dtype == KVPOP_F32) {
    SelectArgs<float> sel{st, dm, (const float*)Q, (const float*)K, (const float*)V, plen, prio,
                          first_seq, Pmax};
    prefill_select_kernel<float><<<pairs, NT2, 0, stream>>>(sel);
  } else {
    SelectArgs<bf16> sel{st, dm, (const bf16*)Q, (const bf16*)K, (const bf16*)V, plen, prio,
                         first_seq, Pmax};
    prefill_select_kernel<bf16><<<pairs, NT2, 0, stream>>>(sel);
  }
  return cudaGetLastError();
}

cudaError_t launch_prefill(const State& st, const Dims& dm, const void* Q, const void* K,
                           const void* V, const int32_t* plen_dev, int first_seq, int n_seq,
                           int Pmax, const float* override_, float* tmp_prio,
                           const void* tf32_maps, cudaStream_t stream) {
  if (dm.dtype == KVPOP_F32)
    return prefill_t<float>(st, dm, Q, K, V, plen_dev, first_seq, n_seq, Pmax, override_, tmp_prio,
                            tf32_maps, stream);
  return prefill_t<bf16>(st, dm, Q, K, V, plen_dev, first_seq, n_seq, Pmax, override_, tmp_prio,
                         tf32_maps, stream);
}

}  // namespace kvpop
