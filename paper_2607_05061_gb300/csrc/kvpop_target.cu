// Future-attention target for training the scorer (Sec. 3.4, App. D, App. F.1-F.2).
//
// Kernel 1, the transposed attention pass (App. D.2): for every key t of KV
// head h and every query head g of its group,
//   log mbar_t^(g) = LSE over d in [t + w, S - 1] (and d <= t + w + L with a
//                    lookahead L) of  q_d^(g) . k_t / sqrt(d_k) - LSE_d^(g),
// where LSE_d is the dense causal normaliser (exact target) or the sparse one
// returned by the prompt attention (App. D.3).  Keys play the queries: a CTA
// holds 128 keys of one (sequence, KV head) as the A operand in registers and
// streams the query rows of each head g past them in blocks of 64 (B operand,
// 16-byte cp.async into a swizzled double buffer) with the per-column LSE_d in
// shared memory; only a running max and sum are kept per (key, head) -- the
// value output of the pass is never formed.  bf16 on m16n8k16 tensor-core
// MMAs, fp32 on CUDA cores (one warp per (key, head), 32 queries per round).
//
// bf16 with d = 128 runs on the 5th-generation tensor cores (target_t5_kernel):
// a CTA holds 256 keys as two 128-row A tiles in shared memory; producer warps
// stream each head's query rows in blocks of 128 through a 4-stage cp.async ring
// and store the block's -log2(e) LSE_d beside them; one thread issues S = K Q^T
// per half into a tensor-memory double buffer; one softmax thread per (key,
// half) reads its row with 32x32b loads.  s c - log2(e) LSE_d is the query's
// log2 attention probability of the key, so the row's 2^x are summed with base 0
// and a running maximum is taken only for a 64-column half whose sum leaves
// [2^-60, 2^60].  The query rows are contiguous; the pass has no value half.
//
// Kernel 2 aggregates per KV head (Eq. 2, App. F.1-F.2):
//   r_t = log(eps + Agg_g mbar_t^(g) / N_t),  N_t = max(1, S - (t + w)),
// N_t clipped to L + 1 with a lookahead, Agg = max or mean; without count
// normalisation N_t = 1.
#include <cstdlib>

#include "kvpop_mma.cuh"
#include "kvpop_ptx.cuh"
#include "kvpop_tc05.cuh"

namespace kvpop {
namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2f = 0.69314718055994530942f;

struct TargetArgs {
  const void* Q;             // [n][H*G][S][d]
  const void* K;             // [n][H][S][d]
  const float* lse;          // [n][H*G][S] natural log
  const int32_t* len;        // [n] or nullptr
  float* logm;               // [n][H*G][S] out
  int H, G, S, w, la;
  float kscale;              // log2(e) / sqrt(d)
  int32_t* err;              // first-error word or nullptr
};

__device__ __forceinline__ int row_len(const TargetArgs& a, int seq) {
  return a.len ? max(0, min(a.len[seq], a.S)) : a.S;
}

// last query position that may attend to key t (-1 if none)
__device__ __forceinline__ int future_hi(int t, int L, int w, int la) {
  const int hi = la > 0 ? min(L - 1, t + w + la) : L - 1;
  return t + w <= hi ? hi : -1;
}

// ---------------------------------------------------------------- CUDA-core kernel
constexpr int TS_NT = 256;
constexpr int TS_BT = 32;

template <typename T, int HD>
__global__ void __launch_bounds__(TS_NT) target_simt_kernel(TargetArgs a) {
  __shared__ float kv[TS_NT / 32][HD];
  constexpr int NW = TS_NT / 32;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int pair = blockIdx.y, seq = pair / a.H, h = pair - seq * a.H;
  const int G = a.G, S = a.S, L = row_len(a, seq);
  const int t0 = blockIdx.x * TS_BT;
  if (t0 >= L) return;
  const T* Kp = static_cast<const T*>(a.K) + (size_t)pair * S * HD;
  float* k_s = kv[warp];
  for (int r = warp; r < TS_BT * G; r += NW) {
    const int tl = r / G, g = r - tl * G, t = t0 + tl;
    if (t >= L) break;
    const size_t qrow = (size_t)seq * a.H * G + (size_t)h * G + g;
    const T* Qg = static_cast<const T*>(a.Q) + qrow * S * HD;
    const float* lse = a.lse + qrow * S;
    for (int i = lane; i < HD; i += 32) k_s[i] = to_f(Kp[(size_t)t * HD + i]) * a.kscale;
    __syncwarp();
    const int hi = future_hi(t, L, a.w, a.la);
    float m = -INFINITY, l = 0.f;
    if (hi >= 0) {
      for (int d0 = t + a.w; d0 <= hi; d0 += 32) {
        const int d = d0 + lane;
        float v = -INFINITY;
        if (d <= hi) {
          const T* qr = Qg + (size_t)d * HD;
          float acc = 0.f;
#pragma unroll 8
          for (int i = 0; i < HD; ++i) acc = fmaf(k_s[i], to_f(qr[i]), acc);
          v = acc - lse[d] * kLog2e;
        }
        float mx = v;
#pragma unroll
        for (int o = 16; o; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        const float mn = fmaxf(m, mx);
        const float u = mn == -INFINITY ? 0.f : mn;
        float p = d <= hi ? exp2f(v - u) : 0.f;
#pragma unroll
        for (int o = 16; o; o >>= 1) p += __shfl_xor_sync(0xffffffffu, p, o);
        l = l * exp2f(m - u) + p;
        m = mn;
      }
    }
    if (lane == 0) a.logm[qrow * S + t] = l > 0.f ? (m + log2f(l)) * kLn2f : -INFINITY;
    __syncwarp();
  }
}

// ---------------------------------------------------------------- tensor-core kernel
template <int HD>
struct TgP {
  static constexpr int NW = 8;
  static constexpr int THREADS = NW * 32;
  static constexpr int ROWS = 16 * NW;             // keys per CTA
  static constexpr int BN = 64;                    // queries per block
  static constexpr int NKS = HD / 16;
  static constexpr int NNT = BN / 8;
  static constexpr int CH = HD / 8;
  static constexpr int ROWB = HD * 2;
  static constexpr int QB = BN * ROWB;
  static constexpr int STAGES = 2;
  static constexpr int OFF_LSE = STAGES * QB;
  static constexpr int SMEM = OFF_LSE + STAGES * BN * 4;
  static_assert(ROWS * ROWB <= STAGES * QB, "the key tile is staged in the query buffers");
};

template <int HD>
__global__ void __launch_bounds__(TgP<HD>::THREADS, 1) target_tc_kernel(TargetArgs a) {
  using P = TgP<HD>;
  extern __shared__ __align__(1024) unsigned char smem_tg[];
  float* lseS = reinterpret_cast<float*>(smem_tg + P::OFF_LSE);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int pair = blockIdx.y, seq = pair / a.H, h = pair - seq * a.H;
  const int G = a.G, S = a.S, L = row_len(a, seq), w = a.w, la = a.la;
  const int t0 = blockIdx.x * P::ROWS;
  if (t0 >= L) return;
  const int t1 = min(t0 + P::ROWS - 1, L - 1);
  const size_t qrow0 = (size_t)seq * a.H * G + (size_t)h * G;
  const int d_lo = t0 + w;
  const int d_hi = la > 0 ? min(L - 1, t1 + w + la) : L - 1;
  const int ra = 16 * warp + (lane >> 2), rb = ra + 8;
  const int ta = t0 + ra, tb = t0 + rb;
  if (d_lo > d_hi) {                               // no key of the tile has a future query
    for (int i = tid; i < (t1 - t0 + 1) * G; i += P::THREADS) {
      const int tl = i / G, g = i - tl * G;
      a.logm[(qrow0 + g) * S + t0 + tl] = -INFINITY;
    }
    return;
  }
  const int nblk = (d_hi - d_lo + P::BN) / P::BN;
  const int total = G * nblk;
  const uint32_t sbase = (uint32_t)__cvta_generic_to_shared(smem_tg);
  const bf16* Kp = static_cast<const bf16*>(a.K) + (size_t)pair * S * HD;

  // key tile -> query buffers (rows past the sequence zero-filled) -> A fragments
  for (int i = tid; i < P::ROWS * P::CH; i += P::THREADS) {
    const int r = i / P::CH, c = i - r * P::CH;
    const bool ok = t0 + r <= t1;
    cp_async16(sbase + swz(r, c, P::ROWB), Kp + (size_t)(ok ? t0 + r : t0) * HD + c * 8, ok ? 16 : 0);
  }
  cp_commit();
  cp_wait<0>();
  __syncthreads();
  uint32_t kf[P::NKS][4];
#pragma unroll
  for (int ks = 0; ks < P::NKS; ++ks) {
    const int r = 16 * warp + ((lane >> 3) & 1) * 8 + (lane & 7);
    const int c = 2 * ks + (lane >> 4);
    ldsm_x4(sbase + swz(r, c, P::ROWB), kf[ks][0], kf[ks][1], kf[ks][2], kf[ks][3]);
  }
  __syncthreads();

  auto issue = [&](int j, int st) {
    const int g = j / nblk, b = j - g * nblk;
    const int d0 = d_lo + b * P::BN;
    const bf16* Qg = static_cast<const bf16*>(a.Q) + (qrow0 + g) * S * HD;
    const uint32_t dst = sbase + st * P::QB;
    for (int i = tid; i < P::BN * P::CH; i += P::THREADS) {
      const int r = i / P::CH, c = i - r * P::CH;
      const bool ok = d0 + r <= d_hi;
      cp_async16(dst + swz(r, c, P::ROWB), Qg + (size_t)(ok ? d0 + r : d0) * HD + c * 8, ok ? 16 : 0);
    }
    if (tid < P::BN) {
      const float* lse = a.lse + (qrow0 + g) * S;
      if (d0 + tid <= d_hi)
        cp_async4(sbase + P::OFF_LSE + (st * P::BN + tid) * 4, lse + d0 + tid);
      else
        lseS[st * P::BN + tid] = 0.f;
    }
  };

  const int hia = future_hi(ta, L, w, la), hib = future_hi(tb, L, w, la);
  float ma = -INFINITY, mb = -INFINITY, la_ = 0.f, lb_ = 0.f;
  issue(0, 0);
  cp_commit();
  if (total > 1) issue(1, 1);
  cp_commit();
  for (int j = 0; j < total; ++j) {
    const int st = j & 1;
    const int g = j / nblk, b = j - g * nblk;
    const int d0 = d_lo + b * P::BN;
    cp_wait<1>();
    __syncthreads();
    const uint32_t qb = sbase + st * P::QB;
    float sc[P::NNT][4];
#pragma unroll
    for (int n = 0; n < P::NNT; ++n) sc[n][0] = sc[n][1] = sc[n][2] = sc[n][3] = 0.f;
#pragma unroll
    for (int ks = 0; ks < P::NKS; ++ks) {
#pragma unroll
      for (int np = 0; np < P::NNT / 2; ++np) {
        const int r = 8 * (2 * np + (lane >> 4)) + (lane & 7);
        const int c = 2 * ks + ((lane >> 3) & 1);
        uint32_t b0, b1, b2, b3;
        ldsm_x4(qb + swz(r, c, P::ROWB), b0, b1, b2, b3);
        mma_bf16(sc[2 * np], kf[ks][0], kf[ks][1], kf[ks][2], kf[ks][3], b0, b1);
        mma_bf16(sc[2 * np + 1], kf[ks][0], kf[ks][1], kf[ks][2], kf[ks][3], b2, b3);
      }
    }
    // rows need a mask where the block reaches below t + w, past t + w + L, or past the end
    const bool masked = d0 < t1 + w || d0 + P::BN - 1 > d_hi || (la > 0 && d0 + P::BN - 1 > t0 + w + la);
    float mxa = -INFINITY, mxb = -INFINITY;
#pragma unroll
    for (int n = 0; n < P::NNT; ++n) {
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const int col = n * 8 + 2 * (lane & 3) + (c & 1);
        const int d = d0 + col;
        float v = sc[n][c] * a.kscale - lseS[st * P::BN + col] * kLog2e;
        if (masked) {
          const int t = c < 2 ? ta : tb;
          const int hi = c < 2 ? hia : hib;
          if (d < t + w || d > hi) v = -INFINITY;
        }
        sc[n][c] = v;
      }
      mxa = fmaxf(mxa, fmaxf(sc[n][0], sc[n][1]));
      mxb = fmaxf(mxb, fmaxf(sc[n][2], sc[n][3]));
    }
#pragma unroll
    for (int o = 1; o <= 2; o <<= 1) {
      mxa = fmaxf(mxa, __shfl_xor_sync(0xffffffffu, mxa, o));
      mxb = fmaxf(mxb, __shfl_xor_sync(0xffffffffu, mxb, o));
    }
    const float mna = fmaxf(ma, mxa), mnb = fmaxf(mb, mxb);
    const float ua = mna == -INFINITY ? 0.f : mna, ub = mnb == -INFINITY ? 0.f : mnb;
    float sa = 0.f, sb = 0.f;
#pragma unroll
    for (int n = 0; n < P::NNT; ++n) {
      sa += ex2(sc[n][0] - ua) + ex2(sc[n][1] - ua);
      sb += ex2(sc[n][2] - ub) + ex2(sc[n][3] - ub);
    }
    la_ = la_ * ex2(ma - ua) + sa;
    lb_ = lb_ * ex2(mb - ub) + sb;
    ma = mna;
    mb = mnb;
    if (b == nblk - 1) {                           // head g done: write and reset
      float sa2 = la_, sb2 = lb_;
#pragma unroll
      for (int o = 1; o <= 2; o <<= 1) {
        sa2 += __shfl_xor_sync(0xffffffffu, sa2, o);
        sb2 += __shfl_xor_sync(0xffffffffu, sb2, o);
      }
      if ((lane & 3) == 0) {
        float* out = a.logm + (qrow0 + g) * S;
        if (ta <= t1) out[ta] = sa2 > 0.f ? (ma + __log2f(sa2)) * kLn2f : -INFINITY;
        if (tb <= t1) out[tb] = sb2 > 0.f ? (mb + __log2f(sb2)) * kLn2f : -INFINITY;
      }
      ma = mb = -INFINITY;
      la_ = lb_ = 0.f;
    }
    __syncthreads();
    if (j + 2 < total) issue(j + 2, st);
    cp_commit();
  }
  cp_wait<0>();
}

// ---------------------------------------------------------------- tcgen05 kernel (d = 128)
constexpr int T6_HALF = 128;
constexpr int T6_ROWS = 2 * T6_HALF;            // keys per CTA
constexpr int T6_BN = 128;                      // queries per block (MMA N)
constexpr int T6_ST = 4;                        // query-block stages
constexpr int T6_MMA_WARP = 16;                 // warps 0-15 softmax, 16 MMA, 17-19 producers
constexpr int T6_PT = 96;
constexpr int T6_THREADS = 32 * 20;
constexpr int T6_KB = T6_HALF * 256;            // key tile of one half
constexpr int T6_QB = T6_BN * 256;              // query block
constexpr int T6_OFF_Q = 2 * T6_KB;
constexpr int T6_OFF_LSE = T6_OFF_Q + T6_ST * T6_QB;
constexpr int T6_OFF_BAR = T6_OFF_LSE + T6_ST * T6_BN * 4;
constexpr int T6_OFF_TMEM = T6_OFF_BAR + 8 * 32;
constexpr int T6_OFF_PX = T6_OFF_TMEM + 16;      // [2 head parity][2 halves][128 rows][m, l, seq, -]
constexpr int T6_SMEM = T6_OFF_PX + 2 * 2 * T6_HALF * 16;
constexpr int T6_FULL = 0, T6_EMPTY = T6_ST, T6_SFULL = 2 * T6_ST, T6_PFULL = 2 * T6_ST + 4,
              T6_KFULL = 2 * T6_ST + 8;
enum : int { T6ERR_WAIT = 22 };

template <int G>
__global__ void __launch_bounds__(T6_THREADS, 1) target_t5_kernel(TargetArgs a) {
  using namespace tc05;
  extern __shared__ __align__(1024) unsigned char sm6[];
  const uint32_t sb = smem_u32(sm6);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int pair = blockIdx.y, seq = pair / a.H, h0 = pair - seq * a.H;
  const int S = a.S, L = row_len(a, seq), w = a.w, la = a.la;
  const int t0 = blockIdx.x * T6_ROWS;
  if (t0 >= L) return;
  const int t1 = min(t0 + T6_ROWS - 1, L - 1);
  const size_t qrow0 = (size_t)seq * a.H * G + (size_t)h0 * G;
  const int d_lo = t0 + w;
  const int d_hi = la > 0 ? min(L - 1, t1 + w + la) : L - 1;
  if (d_lo > d_hi) {                               // no key of the tile has a future query
    for (int i = tid; i < (t1 - t0 + 1) * G; i += T6_THREADS) {
      const int tl = i / G, g = i - tl * G;
      a.logm[(qrow0 + g) * S + t0 + tl] = -INFINITY;
    }
    return;
  }
  const int nblk = (d_hi - d_lo + T6_BN) / T6_BN;
  const int total = G * nblk;
  auto bar = [&](int i) { return sb + T6_OFF_BAR + 8u * (uint32_t)i; };
  if (tid == 0) {
    for (int i = 0; i < T6_ST; ++i) {
      mbar_init(bar(T6_FULL + i), 2 * T6_PT);            // cp.async arrivals + plain stores
      mbar_init(bar(T6_EMPTY + i), 1 + 4 * T6_HALF);   // MMA commit + every softmax thread (LSE)
    }
    for (int i = 0; i < 4; ++i) {
      mbar_init(bar(T6_SFULL + i), 1);
      mbar_init(bar(T6_PFULL + i), 2 * T6_HALF);
    }
    mbar_init(bar(T6_KFULL), T6_PT);
    mbar_fence_init();
    // the softmax halves' exchange slots start with no head done
    int* px = reinterpret_cast<int*>(sm6 + T6_OFF_PX);
    for (int i = 0; i < 2 * 2 * T6_HALF; ++i) px[4 * i + 2] = 0;
  }
  if (warp == T6_MMA_WARP) tmem_alloc(sb + T6_OFF_TMEM, 512);
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(sm6 + T6_OFF_TMEM);
  const bf16* Kp = static_cast<const bf16*>(a.K) + (size_t)pair * S * 128;
  if (warp > T6_MMA_WARP) {
    // ---------------------------------------------------------------- producers
    const int pt = tid - 32 * (T6_MMA_WARP + 1);
    for (int i = pt; i < T6_ROWS * 16; i += T6_PT) {
      const int r = i >> 4, c = i & 15;
      const bool ok = t0 + r <= t1;
      cp_async16(sb + (r >> 7) * T6_KB + tile_off(r & 127, c, T6_HALF),
                 Kp + (size_t)(ok ? t0 + r : t0) * 128 + c * 8, ok ? 16 : 0);
    }
    cp_async_arrive_noinc(bar(T6_KFULL));
    for (int j = 0; j < total; ++j) {
      const int st = j % T6_ST;
      if (j >= T6_ST && !mbar_wait(bar(T6_EMPTY + st), ((j / T6_ST) - 1) & 1, a.err, T6ERR_WAIT)) break;
      const int g = j / nblk, b = j - g * nblk;
      const int d0 = d_lo + b * T6_BN;
      const bf16* Qg = static_cast<const bf16*>(a.Q) + (qrow0 + g) * S * 128;
      const uint32_t qd = sb + T6_OFF_Q + st * T6_QB;
      for (int i = pt; i < T6_BN * 16; i += T6_PT) {
        const int r = i >> 4, c = i & 15;
        const bool ok = d0 + r <= d_hi;
        cp_async16(qd + tile_off(r, c, T6_BN), Qg + (size_t)(ok ? d0 + r : d0) * 128 + c * 8, ok ? 16 : 0);
      }
      // the block's queries' normalisers, stored once as -log2(e) LSE_d
      float* nls = reinterpret_cast<float*>(sm6 + T6_OFF_LSE) + st * T6_BN;
      const float* lse = a.lse + (qrow0 + g) * S;
      for (int i = pt; i < T6_BN; i += T6_PT) nls[i] = -kLog2e * __ldg(lse + min(d0 + i, d_hi));
      cp_async_arrive_noinc(bar(T6_FULL + st));
      mbar_arrive(bar(T6_FULL + st));
    }
    cp_wait<0>();
  } else if (warp == T6_MMA_WARP) {
    // ---------------------------------------------------------------- MMA issue
    if (lane == 0) {
      const uint32_t idS = idesc_bf16(128, T6_BN, 0);
      bool ok = mbar_wait(bar(T6_KFULL), 0, a.err, T6ERR_WAIT);
      for (int j = 0; j < total && ok; ++j) {
        const int st = j % T6_ST, b2 = j & 1;
        if (!(ok = mbar_wait(bar(T6_FULL + st), (j / T6_ST) & 1, a.err, T6ERR_WAIT))) break;
        fence_async_smem();
        fence_after();
        const uint32_t qb = sb + T6_OFF_Q + st * T6_QB;
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
          // the softmax half must be done with S_{j-2} before its buffer is rewritten
          if (j >= 2 && !(ok = mbar_wait(bar(T6_PFULL + 2 * hh + b2), ((j - 2) >> 1) & 1, a.err, T6ERR_WAIT)))
            break;
          fence_after();
          const uint32_t dS = tmem + hh * 256 + (uint32_t)b2 * T6_BN;
#pragma unroll
          for (int ks = 0; ks < 8; ++ks)
            mma_bf16(dS, kmajor_desc(sb + hh * T6_KB, T6_HALF, ks), kmajor_desc(qb, T6_BN, ks), idS, ks > 0);
          commit(bar(T6_SFULL + 2 * hh + b2));
        }
        if (!ok) break;
        commit(bar(T6_EMPTY + st));
      }
      // the last stage's release (the commit and the softmax) has landed before the CTA ends
      if (ok && total > 0)
        mbar_wait(bar(T6_EMPTY + (total - 1) % T6_ST), ((total - 1) / T6_ST) & 1, a.err, T6ERR_WAIT);
    }
    __syncwarp();
  } else {
    // ---------------------------------------------------------------- softmax rows
    // warp w: half hh = (w / 4) mod 2 of the CTA's keys, key row r = 32 (w mod 4) + lane (the
    // warp's tensor-memory lane quarter), and columns [64 cs, 64 cs + 64) of every block with
    // cs = w / 8: four warps per subpartition share the exponentials of a block.  The two
    // column halves of a row keep their own (max, sum) over a head's blocks and meet at the
    // head's end in shared memory.
    const int hh = (warp >> 2) & 1, cs = warp >> 3;
    const int r = (warp & 3) * 32 + lane;
    const int t = t0 + hh * T6_HALF + r;
    const int hi = t <= t1 ? future_hi(t, L, w, la) : -1;
    const uint32_t tS = tmem + ((uint32_t)((warp & 3) * 32) << 16) + hh * 256;
    const float* nlS = reinterpret_cast<const float*>(sm6 + T6_OFF_LSE);   // -log2(e) LSE_d per stage
    float* pxs = reinterpret_cast<float*>(sm6 + T6_OFF_PX);
    const float c2 = a.kscale;
    float m = -INFINITY, l = 0.f;
    auto uniform = [](bool x) { return __all_sync(0xffffffffu, x); };
    for (int j = 0; j < total; ++j) {
      const int st = j % T6_ST, b2 = j & 1;
      const int g = j / nblk, b = j - g * nblk;
      const int d0 = d_lo + b * T6_BN;
      if (!uniform(mbar_wait(bar(T6_SFULL + 2 * hh + b2), (j >> 1) & 1, a.err, T6ERR_WAIT))) break;
      // the stage's normalisers (complete long before S; the wait orders their reads)
      if (!uniform(mbar_wait(bar(T6_FULL + st), (j / T6_ST) & 1, a.err, T6ERR_WAIT))) break;
      fence_after();
      // this thread's 64 columns as two 32-column parts, each folded into the running sum
#pragma unroll 1
      for (int c = 0; c < 2; ++c) {
        const int col = 64 * cs + 32 * c;
        const int e0 = d0 + col;
        float s[32];
        tmem_ld32(tS + b2 * T6_BN + col, s);
        tmem_wait_ld();
        if (c == 1) {
          // the thread's part of the S buffer is in registers: the MMA may overwrite it
          fence_before();
          mbar_arrive(bar(T6_PFULL + 2 * hh + b2));
        }
        const bool masked = e0 < t1 + w || e0 + 31 > d_hi || (la > 0 && e0 + 31 > t0 + w + la);
        if (masked) {                               // on the raw logits: -inf c2 + n = -inf
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const int d = e0 + i;
            if (d < t + w || d > hi) s[i] = -INFINITY;
          }
        }
        // x = s c2 - log2(e) LSE_d is the query's log2 attention probability of the key, so
        // 2^x needs no running maximum unless the key lies outside the query's kept set
        // with a much larger logit: sum with base 0, and take the maximum only when the
        // part's sum leaves [2^-60, 2^60] (overflow, NaN, or every term tiny or masked).
        {
          const float4* l4 = reinterpret_cast<const float4*>(nlS + st * T6_BN + col);
          const uint64_t cc = f2_pack(c2, c2);
          uint64_t ps[4] = {0ull, 0ull, 0ull, 0ull};
#pragma unroll
          for (int i4 = 0; i4 < 8; ++i4) {
            const float4 v = l4[i4];
            f2_unpack(f2_fma(f2_pack(s[4 * i4], s[4 * i4 + 1]), cc, f2_pack(v.x, v.y)), s[4 * i4],
                      s[4 * i4 + 1]);
            f2_unpack(f2_fma(f2_pack(s[4 * i4 + 2], s[4 * i4 + 3]), cc, f2_pack(v.z, v.w)), s[4 * i4 + 2],
                      s[4 * i4 + 3]);
            const int k = (2 * i4) & 3;
            ps[k] = f2_add(ps[k], f2_pack(ex2(s[4 * i4]), ex2(s[4 * i4 + 1])));
            ps[k + 1] = f2_add(ps[k + 1], f2_pack(ex2(s[4 * i4 + 2]), ex2(s[4 * i4 + 3])));
          }
          // the stage's query rows and normalisers are no longer needed by this thread
          if (c == 1) mbar_arrive(bar(T6_EMPTY + st));
          float q[8];
#pragma unroll
          for (int k = 0; k < 4; ++k) f2_unpack(ps[k], q[2 * k], q[2 * k + 1]);
          const float sum = ((q[0] + q[1]) + (q[2] + q[3])) + ((q[4] + q[5]) + (q[6] + q[7]));
          if (sum >= 0x1p-60f && sum <= 0x1p60f) {
            if (m <= 0.f) {                         // new base 0
              l = (m == 0.f ? l : l * ex2(m)) + sum;
              m = 0.f;
            } else {
              l = fmaf(sum, ex2(-m), l);
            }
            continue;
          }
        }
        // part maximum: 8 chains of three-input maxima
        float pm[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) pm[k] = s[k];
#pragma unroll
        for (int k = 0; k < 8; ++k) pm[k] = fmax3(pm[k], s[8 + k], s[16 + k]);
#pragma unroll
        for (int k = 0; k < 8; ++k) pm[k] = fmaxf(pm[k], s[24 + k]);
        const float mx = fmax3(fmax3(pm[0], pm[1], pm[2]), fmax3(pm[3], pm[4], pm[5]), fmaxf(pm[6], pm[7]));
        const float mn = fmaxf(m, mx);
        const float base = mn == -INFINITY ? 0.f : mn;
        // sum of 2^(x - base), differences and partial sums packed in pairs
        const uint64_t nb = f2_pack(-base, -base);
        uint64_t ps[4] = {0ull, 0ull, 0ull, 0ull};
#pragma unroll
        for (int i = 0; i < 32; i += 8) {
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            float x0, x1;
            f2_unpack(f2_add(f2_pack(s[i + 2 * k], s[i + 2 * k + 1]), nb), x0, x1);
            ps[k] = f2_add(ps[k], f2_pack(ex2(x0), ex2(x1)));
          }
        }
        float q[8];
#pragma unroll
        for (int k = 0; k < 4; ++k) f2_unpack(ps[k], q[2 * k], q[2 * k + 1]);
        l = l * ex2(m - base) + (((q[0] + q[1]) + (q[2] + q[3])) + ((q[4] + q[5]) + (q[6] + q[7])));
        m = mn;
      }
      if (b == nblk - 1) {
        // head g done: the upper column half hands its (max, sum) to the lower, which merges
        // and writes the key's log mass (slots alternate by head; a flag names the head)
        float* px = pxs + (((size_t)(g & 1) * 2 + hh) * T6_HALF + r) * 4;
        volatile int* seq = reinterpret_cast<volatile int*>(px) + 2;
        if (cs == 1) {
          px[0] = m;
          px[1] = l;
          __threadfence_block();
          *seq = g + 1;
        } else {
          bool ready = *seq == g + 1;
          if (!ready) {
            const unsigned long long tw = globaltimer();
            while (!(ready = *seq == g + 1))
              if (globaltimer() - tw > kWaitLimitNs) { atomicCAS(a.err, 0, T6ERR_WAIT); break; }
          }
          __threadfence_block();
          const float m1 = px[0], l1 = px[1];
          const float M = fmaxf(m, m1);
          float Lr = 0.f;
          if (M != -INFINITY)
            Lr = (m == -INFINITY ? 0.f : l * ex2(m - M)) + (m1 == -INFINITY ? 0.f : l1 * ex2(m1 - M));
          if (t <= t1) a.logm[(qrow0 + g) * S + t] = Lr > 0.f ? (M + __log2f(Lr)) * kLn2f : -INFINITY;
        }
        m = -INFINITY;
        l = 0.f;
      }
    }
  }
  fence_before();
  __syncthreads();
  if (warp == T6_MMA_WARP) tmem_dealloc(tmem, 512);
}

// ---------------------------------------------------------------- aggregation
struct AggArgs {
  const float* logm;         // [n][H*G][S]
  const int32_t* len;
  float* target;             // [n][H][S]
  int n_pairs, H, G, S, w, la, agg, count_norm;
  float log_eps;             // log(eps), -inf for eps = 0
};

__global__ void aggregate_kernel(AggArgs a) {
  const size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (size_t)a.n_pairs * a.S) return;
  const int pair = (int)(i / a.S), t = (int)(i - (size_t)pair * a.S);
  const int seq = pair / a.H, h = pair - seq * a.H;
  const int L = a.len ? max(0, min(a.len[seq], a.S)) : a.S;
  if (t >= L) return;
  float logN = 0.f;
  if (a.count_norm) {
    int n = max(1, L - (t + a.w));
    if (a.la > 0) n = min(n, a.la + 1);
    logN = logf((float)n);
  }
  const float* lm = a.logm + ((size_t)seq * a.H * a.G + (size_t)h * a.G) * a.S + t;
  float x;
  if (a.agg == 0) {
    x = -INFINITY;
    for (int g = 0; g < a.G; ++g) x = fmaxf(x, lm[(size_t)g * a.S]);
  } else {
    float mx = -INFINITY;
    for (int g = 0; g < a.G; ++g) mx = fmaxf(mx, lm[(size_t)g * a.S]);
    float sum = 0.f;
    if (mx != -INFINITY)
      for (int g = 0; g < a.G; ++g) sum += expf(lm[(size_t)g * a.S] - mx);
    x = mx == -INFINITY ? -INFINITY : mx + logf(sum / (float)a.G);
  }
  x -= logN;
  // log(eps + exp(x)) without overflow
  const float hi = fmaxf(a.log_eps, x), lo = fminf(a.log_eps, x);
  a.target[i] = lo == -INFINITY ? hi : hi + log1pf(expf(lo - hi));
}

}  // namespace

cudaError_t launch_future_target(const void* Q, const void* K, const float* lse, const int32_t* len,
                                 int n_seq, int H, int G, int d, int S, int w, int la, int dtype,
                                 float* logm, float* target, int agg, int count_norm, float eps,
                                 int32_t* err, cudaStream_t stream) {
  if (n_seq <= 0 || S <= 0) return cudaSuccess;
  TargetArgs a{Q, K, lse, len, logm, H, G, S, w, la, 1.4426950408889634f / sqrtf((float)d), err};
  const int n_pairs = n_seq * H;
  static const bool mma_sync = [] {
    const char* e = getenv("KVPOP_TARGET_MMA_SYNC");
    return e && e[0] == '1';
  }();
  if (dtype == KVPOP_BF16 && d == 128 && !mma_sync) {
    dim3 grid((S + T6_ROWS - 1) / T6_ROWS, n_pairs);
    cudaError_t e = cudaSuccess;
    if (G == 4) {
      e = raise_smem_limit(target_t5_kernel<4>, T6_SMEM);
      if (e == cudaSuccess) target_t5_kernel<4><<<grid, T6_THREADS, T6_SMEM, stream>>>(a);
    } else if (G == 2) {
      e = raise_smem_limit(target_t5_kernel<2>, T6_SMEM);
      if (e == cudaSuccess) target_t5_kernel<2><<<grid, T6_THREADS, T6_SMEM, stream>>>(a);
    } else {
      e = raise_smem_limit(target_t5_kernel<1>, T6_SMEM);
      if (e == cudaSuccess) target_t5_kernel<1><<<grid, T6_THREADS, T6_SMEM, stream>>>(a);
    }
    if (e != cudaSuccess) return e;
  } else if (dtype == KVPOP_BF16) {
    const size_t smem = d == 128 ? TgP<128>::SMEM : TgP<64>::SMEM;
    dim3 grid((S + TgP<128>::ROWS - 1) / TgP<128>::ROWS, n_pairs);
    if (d == 128) {
      cudaError_t e = raise_smem_limit(target_tc_kernel<128>, smem);
      if (e != cudaSuccess) return e;
      target_tc_kernel<128><<<grid, TgP<128>::THREADS, smem, stream>>>(a);
    } else {
      cudaError_t e = raise_smem_limit(target_tc_kernel<64>, smem);
      if (e != cudaSuccess) return e;
      target_tc_kernel<64><<<grid, TgP<64>::THREADS, smem, stream>>>(a);
    }
  } else {
    dim3 grid((S + TS_BT - 1) / TS_BT, n_pairs);
    if (d == 128) target_simt_kernel<float, 128><<<grid, TS_NT, 0, stream>>>(a);
    else target_simt_kernel<float, 64><<<grid, TS_NT, 0, stream>>>(a);
  }
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess || !target) return e;
  AggArgs g{logm, len, target, n_pairs, H, G, S, w, la, agg, count_norm,
            eps > 0.f ? logf(eps) : -INFINITY};
  const size_t n = (size_t)n_pairs * S;
  aggregate_kernel<<<(unsigned)((n + 255) / 256), 256, 0, stream>>>(g);
  return cudaGetLastError();
}

}  // namespace kvpop
