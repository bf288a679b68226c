// Masked causal attention over a prompt under the running top-k mask
// (App. C.1 mask, App. C.3 use inside a fused sparse attention kernel).
//
// A CTA takes BM consecutive queries of one (sequence, KV head) with all G
// query heads of that KV head (BM * G rows), so every gathered K/V row feeds
// every head.  Instead of testing the mask on the dense causal square, it first
// gathers the tile's candidate keys into two lists (positions in shared memory):
//   A -- kept for every query of the tile: the sinks t <= q0 and the eligible
//        t <= q0 - w whose rank is within the smallest cutoff of the tile;
//   M -- kept for some queries only: later sinks, eligible keys ranked between
//        the tile's smallest and largest cutoff, and the window / newly
//        eligible positions max(s, q0 - w + 1) .. q1.
// Because the retained set of consecutive queries changes by at most one key
// per query, |A| <= s + k and |M| <= s + 2 BM + w, so the tile touches about
// s + k + w + BM keys instead of q.  Blocks of the A list run unmasked; the
// few blocks holding M entries test the mask per element:
//   t <= q and (t < s or q - t < w or (t <= q - w and rank(t) <= tau_q)).
// Outputs: y [G][q][d] in fp32 and the natural-log normaliser
// LSE = log sum_{t kept} exp(q.k_t / sqrt(d)) (the sparse LSE of App. D.3).
//
// bf16: m16n8k16 tensor-core MMAs (Q fragments in registers, K via ldmatrix,
// V via ldmatrix.trans, probabilities packed to bf16 in registers), K/V rows
// gathered by 16-byte cp.async into a 128-byte-swizzled double buffer.
// fp32: CUDA-core kernel, one warp per (query, head) row, 32 keys per round.
#include <cstdlib>

#include "kvpop_mma.cuh"
#include "kvpop_prompt.cuh"

namespace kvpop {
namespace {

using namespace prompt;

// ---------------------------------------------------------------- CUDA-core kernel
constexpr int SIMT_NT = 256;
constexpr int SIMT_BM = 32;

template <typename T, int HD, bool DENSE>
__global__ void __launch_bounds__(SIMT_NT) prompt_simt_kernel(PromptArgs a) {
  extern __shared__ __align__(16) unsigned char smem_simt[];
  unsigned char* smem = smem_simt;
  constexpr int NW = SIMT_NT / 32;
  constexpr int NC = HD / 32;
  float* qv = reinterpret_cast<float*>(smem);                 // [NW][HD]
  int* tauS = reinterpret_cast<int*>(qv + NW * HD);          // [SIMT_BM]
  int* red = tauS + SIMT_BM;                                  // [NW + 2]
  int32_t* posA = red + NW + 2;
  int32_t* posM = posA + a.capA;
  TileInfo ti;
  if (DENSE) {
    if (!dense_setup(a, SIMT_BM, ti)) return;
  } else if (!tile_setup<SIMT_NT>(a, SIMT_BM, tauS, red, posA, posM, ti)) {
    return;
  }
  const bool want_y = a.Y != nullptr;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int G = a.G, H = a.H, S = a.S;
  const int nA = ti.nA, nU = ti.nA + ti.nM;
  const T* Kp = static_cast<const T*>(a.K) + (size_t)ti.pair * S * HD;
  const T* Vp = static_cast<const T*>(a.V) + (size_t)ti.pair * S * HD;
  const int32_t* rank = DENSE ? nullptr : a.rank + (size_t)ti.pair * S;
  float* q_s = qv + warp * HD;
  for (int r = warp; r < SIMT_BM * G; r += NW) {
    const int ql = r / G, g = r - ql * G, q = ti.q0 + ql;
    if (q > ti.q1) break;
    const size_t row = ((size_t)ti.seq * H * G + (size_t)ti.h * G + g) * S + q;
    const T* qp = static_cast<const T*>(a.Q) + row * HD;
    for (int i = lane; i < HD; i += 32) q_s[i] = to_f(qp[i]) * a.qscale;
    __syncwarp();
    const int tq = DENSE ? 0 : tauS[ql];
    float m = -INFINITY, l = 0.f, o[NC];
#pragma unroll
    for (int c = 0; c < NC; ++c) o[c] = 0.f;
    for (int e0 = 0; e0 < nU; e0 += 32) {
      const int e = e0 + lane;
      int t = 0;
      bool keep = false;
      if (e < nU) {
        if (DENSE) {
          t = e;
          keep = t <= q;
        } else {
          t = e < nA ? posA[e] : posM[e - nA];
          keep = e < nA || keep_key(q, t, __ldg(rank + t), tq, a.s, a.w);
        }
      }
      float logit = -INFINITY;
      if (keep) {
        const T* kr = Kp + (size_t)t * HD;
        float acc = 0.f;
#pragma unroll 8
        for (int i = 0; i < HD; ++i) acc = fmaf(q_s[i], to_f(kr[i]), acc);
        logit = acc;
      }
      float mx = logit;
#pragma unroll
      for (int o2 = 16; o2; o2 >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o2));
      const float m_new = fmaxf(m, mx);
      const float m_use = m_new == -INFINITY ? 0.f : m_new;
      const float alpha = exp2f(m - m_use);
      const float p = keep ? exp2f(logit - m_use) : 0.f;
      float ps = p;
#pragma unroll
      for (int o2 = 16; o2; o2 >>= 1) ps += __shfl_xor_sync(0xffffffffu, ps, o2);
      l = l * alpha + ps;
      m = m_new;
      if (!want_y) continue;
#pragma unroll
      for (int c = 0; c < NC; ++c) o[c] *= alpha;
      const int nk = min(32, nU - e0);
      for (int jj = 0; jj < nk; ++jj) {
        const float pj = __shfl_sync(0xffffffffu, p, jj);
        const int tj = __shfl_sync(0xffffffffu, t, jj);
        if (pj != 0.f) {
          const T* vr = Vp + (size_t)tj * HD;
#pragma unroll
          for (int c = 0; c < NC; ++c) o[c] = fmaf(pj, to_f(vr[lane + 32 * c]), o[c]);
        }
      }
    }
    if (want_y) {
      const float inv = 1.f / l;
      float* yp = a.Y + row * HD;
#pragma unroll
      for (int c = 0; c < NC; ++c) yp[lane + 32 * c] = o[c] * inv;
    }
    if (a.lse && lane == 0) a.lse[row] = (m + log2f(l)) * kLn2;
    __syncwarp();
  }
}

// ---------------------------------------------------------------- tensor-core kernel
template <int HD, int G>
struct TcP {
  static constexpr int NW = 8;
  static constexpr int THREADS = NW * 32;
  static constexpr int ROWS = 16 * NW;             // (query, head) rows per CTA
  static constexpr int BM = ROWS / G;              // queries per CTA
  static constexpr int BN = 64;                    // keys per block
  static constexpr int NKS = HD / 16;
  static constexpr int NNT = BN / 8;
  static constexpr int NOT = HD / 8;
  static constexpr int CH = HD / 8;                // 16-byte chunks per bf16 row
  static constexpr int ROWB = HD * 2;
  static constexpr int KVB = BN * ROWB;            // K (or V) bytes of one block
  static constexpr int STAGES = 2;
  static constexpr int STAGE = 2 * KVB;
  static constexpr int OFF_POSB = STAGES * STAGE;
  static constexpr int OFF_RKB = OFF_POSB + STAGES * BN * 4;
  static constexpr int OFF_TAU = OFF_RKB + STAGES * BN * 4;
  static constexpr int OFF_RED = OFF_TAU + BM * 4;
  static constexpr int OFF_LIST = OFF_RED + (NW + 2) * 4 + 8;
  static_assert(ROWS * ROWB <= STAGE, "the Q tile is staged in the first K/V stage");
};

template <int HD, int G, bool DENSE, bool WANT_Y>
__global__ void __launch_bounds__(TcP<HD, G>::THREADS, 1) prompt_tc_kernel(PromptArgs a) {
  using P = TcP<HD, G>;
  extern __shared__ __align__(1024) unsigned char smem_tc[];
  unsigned char* smem = smem_tc;
  int32_t* posb = reinterpret_cast<int32_t*>(smem + P::OFF_POSB);
  int32_t* rkb = reinterpret_cast<int32_t*>(smem + P::OFF_RKB);
  int* tauS = reinterpret_cast<int*>(smem + P::OFF_TAU);
  int* red = reinterpret_cast<int*>(smem + P::OFF_RED);
  int32_t* posA = reinterpret_cast<int32_t*>(smem + P::OFF_LIST);
  int32_t* posM = posA + a.capA;
  TileInfo ti;
  if (DENSE) {
    if (!dense_setup(a, P::BM, ti)) return;
  } else if (!tile_setup<P::THREADS>(a, P::BM, tauS, red, posA, posM, ti)) {
    return;
  }
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int H = a.H, S = a.S;
  const int nA = ti.nA, nU = ti.nA + ti.nM;
  const uint32_t sbase = (uint32_t)__cvta_generic_to_shared(smem);
  const bf16* Kp = static_cast<const bf16*>(a.K) + (size_t)ti.pair * S * HD;
  const bf16* Vp = WANT_Y ? static_cast<const bf16*>(a.V) + (size_t)ti.pair * S * HD : nullptr;
  const int32_t* rank = DENSE ? nullptr : a.rank + (size_t)ti.pair * S;
  const bf16* Qbase = static_cast<const bf16*>(a.Q) + ((size_t)ti.seq * H * G + (size_t)ti.h * G) * S * HD;

  // Q tile -> stage 0 (rows past the prompt are zero-filled)
  for (int i = tid; i < P::ROWS * P::CH; i += P::THREADS) {
    const int r = i / P::CH, c = i - r * P::CH;
    const int q = ti.q0 + r / G, g = r % G;
    const bool ok = q <= ti.q1;
    const bf16* src = Qbase + ((size_t)g * S + (ok ? q : ti.q0)) * HD + c * 8;
    cp_async16(sbase + swz(r, c, P::ROWB), src, ok ? 16 : 0);
  }
  cp_commit();
  cp_wait<0>();
  __syncthreads();
  uint32_t qf[P::NKS][4];
#pragma unroll
  for (int ks = 0; ks < P::NKS; ++ks) {
    const int r = 16 * warp + ((lane >> 3) & 1) * 8 + (lane & 7);
    const int c = 2 * ks + (lane >> 4);
    ldsm_x4(sbase + swz(r, c, P::ROWB), qf[ks][0], qf[ks][1], qf[ks][2], qf[ks][3]);
  }
  __syncthreads();

  const int pad_t = DENSE ? 0 : (nA > 0 ? posA[0] : posM[0]);
  // position of list entry e (entries past the list gather a valid row and are masked)
  auto entry = [&](int e) {
    if (DENSE) return e < nU ? e : pad_t;
    return e < nA ? posA[e] : (e < nU ? posM[e - nA] : pad_t);
  };
  auto issue = [&](int blk, int st) {
    const uint32_t kdst = sbase + st * P::STAGE;
    const uint32_t vdst = kdst + P::KVB;
    for (int i = tid; i < P::BN * P::CH; i += P::THREADS) {
      const int key = i / P::CH, c = i - key * P::CH;
      const int t = entry(blk * P::BN + key);
      const uint32_t off = swz(key, c, P::ROWB);
      cp_async16(kdst + off, Kp + (size_t)t * HD + c * 8, 16);
      if (WANT_Y) cp_async16(vdst + off, Vp + (size_t)t * HD + c * 8, 16);
    }
    if (tid < P::BN) {
      const int e = blk * P::BN + tid;
      const int t = entry(e);
      posb[st * P::BN + tid] = e < nU ? t : INT_MAX;
      if (!DENSE) cp_async4(sbase + P::OFF_RKB + (st * P::BN + tid) * 4, rank + t);
    }
  };

  const int ra = 16 * warp + (lane >> 2), rb = ra + 8;
  const int qa = ti.q0 + ra / G, qb = ti.q0 + rb / G;
  const int ta = DENSE ? 0 : tauS[ra / G], tb = DENSE ? 0 : tauS[rb / G];
  float o[P::NOT][4];
#pragma unroll
  for (int n = 0; n < P::NOT; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.f;
  float ma = -INFINITY, mb = -INFINITY, la = 0.f, lb = 0.f;

  const int nblk = (nU + P::BN - 1) / P::BN;
  issue(0, 0);
  cp_commit();
  if (nblk > 1) issue(1, 1);
  cp_commit();
  for (int j = 0; j < nblk; ++j) {
    const int st = j & 1;
    cp_wait<1>();
    __syncthreads();
    const uint32_t kb = sbase + st * P::STAGE;
    const uint32_t vb = kb + P::KVB;
    float sc[P::NNT][4];
#pragma unroll
    for (int n = 0; n < P::NNT; ++n) sc[n][0] = sc[n][1] = sc[n][2] = sc[n][3] = 0.f;
#pragma unroll
    for (int ks = 0; ks < P::NKS; ++ks) {
#pragma unroll
      for (int np = 0; np < P::NNT / 2; ++np) {
        const int key = 8 * (2 * np + (lane >> 4)) + (lane & 7);
        const int c = 2 * ks + ((lane >> 3) & 1);
        uint32_t b0, b1, b2, b3;
        ldsm_x4(kb + swz(key, c, P::ROWB), b0, b1, b2, b3);
        mma_bf16(sc[2 * np], qf[ks][0], qf[ks][1], qf[ks][2], qf[ks][3], b0, b1);
        mma_bf16(sc[2 * np + 1], qf[ks][0], qf[ks][1], qf[ks][2], qf[ks][3], b2, b3);
      }
    }
    const bool masked = (j + 1) * P::BN > nA;
#pragma unroll
    for (int n = 0; n < P::NNT; ++n) {
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        float v = sc[n][c] * a.qscale;
        if (masked) {
          const int col = n * 8 + 2 * (lane & 3) + (c & 1);
          const int e = j * P::BN + col;
          if (e >= nA) {
            const int t = posb[st * P::BN + col];
            bool kp;
            if (DENSE) {
              kp = t <= ((c < 2) ? qa : qb);
            } else {
              const int r = rkb[st * P::BN + col];
              kp = (c < 2) ? keep_key(qa, t, r, ta, a.s, a.w) : keep_key(qb, t, r, tb, a.s, a.w);
            }
            if (e >= nU || !kp) v = -INFINITY;
          }
        }
        sc[n][c] = v;
      }
    }
    float mxa = -INFINITY, mxb = -INFINITY;
#pragma unroll
    for (int n = 0; n < P::NNT; ++n) {
      mxa = fmaxf(mxa, fmaxf(sc[n][0], sc[n][1]));
      mxb = fmaxf(mxb, fmaxf(sc[n][2], sc[n][3]));
    }
#pragma unroll
    for (int o2 = 1; o2 <= 2; o2 <<= 1) {
      mxa = fmaxf(mxa, __shfl_xor_sync(0xffffffffu, mxa, o2));
      mxb = fmaxf(mxb, __shfl_xor_sync(0xffffffffu, mxb, o2));
    }
    const float mna = fmaxf(ma, mxa), mnb = fmaxf(mb, mxb);
    const float ua = mna == -INFINITY ? 0.f : mna, ub = mnb == -INFINITY ? 0.f : mnb;
    const float aa = ex2(ma - ua), ab = ex2(mb - ub);
    ma = mna;
    mb = mnb;
    float sa = 0.f, sb = 0.f;
#pragma unroll
    for (int n = 0; n < P::NNT; ++n) {
      sc[n][0] = ex2(sc[n][0] - ua);
      sc[n][1] = ex2(sc[n][1] - ua);
      sc[n][2] = ex2(sc[n][2] - ub);
      sc[n][3] = ex2(sc[n][3] - ub);
      sa += sc[n][0] + sc[n][1];
      sb += sc[n][2] + sc[n][3];
    }
    la = la * aa + sa;
    lb = lb * ab + sb;
    if (WANT_Y) {
#pragma unroll
    for (int n = 0; n < P::NOT; ++n) {
      o[n][0] *= aa;
      o[n][1] *= aa;
      o[n][2] *= ab;
      o[n][3] *= ab;
    }
#pragma unroll
    for (int kk = 0; kk < P::BN / 16; ++kk) {
      const uint32_t p0 = pack_bf16(sc[2 * kk][0], sc[2 * kk][1]);
      const uint32_t p1 = pack_bf16(sc[2 * kk][2], sc[2 * kk][3]);
      const uint32_t p2 = pack_bf16(sc[2 * kk + 1][0], sc[2 * kk + 1][1]);
      const uint32_t p3 = pack_bf16(sc[2 * kk + 1][2], sc[2 * kk + 1][3]);
#pragma unroll
      for (int np = 0; np < P::NOT / 2; ++np) {
        const int key = 16 * kk + ((lane >> 3) & 1) * 8 + (lane & 7);
        const int c = 2 * np + (lane >> 4);
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(vb + swz(key, c, P::ROWB), b0, b1, b2, b3);
        mma_bf16(o[2 * np], p0, p1, p2, p3, b0, b1);
        mma_bf16(o[2 * np + 1], p0, p1, p2, p3, b2, b3);
      }
    }
    }
    __syncthreads();
    if (j + 2 < nblk) issue(j + 2, st);
    cp_commit();
  }
  cp_wait<0>();

#pragma unroll
  for (int o2 = 1; o2 <= 2; o2 <<= 1) {
    la += __shfl_xor_sync(0xffffffffu, la, o2);
    lb += __shfl_xor_sync(0xffffffffu, lb, o2);
  }
  const float ia = 1.f / la, ib = 1.f / lb;
  const size_t rowa = ((size_t)ti.seq * H * G + (size_t)ti.h * G + ra % G) * S + qa;
  const size_t rowb = ((size_t)ti.seq * H * G + (size_t)ti.h * G + rb % G) * S + qb;
  const int col = 2 * (lane & 3);
  if (qa <= ti.q1) {
    if (WANT_Y) {
      float* y = a.Y + rowa * HD + col;
#pragma unroll
      for (int n = 0; n < P::NOT; ++n)
        *reinterpret_cast<float2*>(y + 8 * n) = make_float2(o[n][0] * ia, o[n][1] * ia);
    }
    if (a.lse && (lane & 3) == 0) a.lse[rowa] = (ma + __log2f(la)) * kLn2;
  }
  if (qb <= ti.q1) {
    if (WANT_Y) {
      float* y = a.Y + rowb * HD + col;
#pragma unroll
      for (int n = 0; n < P::NOT; ++n)
        *reinterpret_cast<float2*>(y + 8 * n) = make_float2(o[n][2] * ib, o[n][3] * ib);
    }
    if (a.lse && (lane & 3) == 0) a.lse[rowb] = (mb + __log2f(lb)) * kLn2;
  }
}

template <typename Kern>
cudaError_t launch_cfg(Kern k, dim3 grid, int threads, size_t smem, cudaStream_t stream,
                       const PromptArgs& a) {
  if (smem > 48 * 1024) {
    cudaError_t e = raise_smem_limit(k, smem);
    if (e != cudaSuccess) return e;
  }
  k<<<grid, threads, smem, stream>>>(a);
  return cudaGetLastError();
}

template <int HD, int G>
size_t tc_smem(int capA, int capM) {
  return (size_t)TcP<HD, G>::OFF_LIST + (size_t)(capA + capM) * 4;
}

template <int HD, int G, bool DENSE, bool WANT_Y>
cudaError_t launch_tc(PromptArgs a, int n_pairs, cudaStream_t stream) {
  using P = TcP<HD, G>;
  if (DENSE) a.capA = a.capM = 0;
  else a.capM = a.s + 2 * P::BM + a.w;
  const size_t smem = tc_smem<HD, G>(a.capA, a.capM);
  if (smem > 227 * 1024) return cudaErrorInvalidValue;
  dim3 grid((a.S + P::BM - 1) / P::BM, n_pairs);
  return launch_cfg(prompt_tc_kernel<HD, G, DENSE, WANT_Y>, grid, P::THREADS, smem, stream, a);
}

template <typename T, int HD, bool DENSE>
cudaError_t launch_simt(PromptArgs a, int n_pairs, cudaStream_t stream) {
  if (DENSE) a.capA = a.capM = 0;
  else a.capM = a.s + 2 * SIMT_BM + a.w;
  const size_t smem = (size_t)(SIMT_NT / 32) * HD * 4 + (SIMT_BM + SIMT_NT / 32 + 2) * 4 +
                      (size_t)(a.capA + a.capM) * 4;
  if (smem > 227 * 1024) return cudaErrorInvalidValue;
  dim3 grid((a.S + SIMT_BM - 1) / SIMT_BM, n_pairs);
  return launch_cfg(prompt_simt_kernel<T, HD, DENSE>, grid, SIMT_NT, smem, stream, a);
}

}  // namespace

bool prompt_t5_ok(int d, int G, int s, int w, int k);
cudaError_t launch_prompt_t5(const prompt::PromptArgs& a, int n_pairs, int G, bool dense,
                             bool want_y, cudaStream_t stream);

namespace {

// tcgen05 kernel for bf16 with d = 128 (KVPOP_PROMPT_MMA_SYNC=1 selects the m16n8k16 kernel)
bool use_t5(int dtype, int d, int G, int s, int w, int k) {
  static const bool off = [] {
    const char* e = getenv("KVPOP_PROMPT_MMA_SYNC");
    return e && e[0] == '1';
  }();
  return !off && dtype == KVPOP_BF16 && prompt_t5_ok(d, G, s, w, k);
}

template <bool DENSE, bool WANT_Y>
cudaError_t dispatch(const PromptArgs& a, int n_pairs, int dtype, int d, int G, cudaStream_t stream) {
  if (use_t5(dtype, d, G, a.s, a.w, a.capA - a.s) && (DENSE || WANT_Y))
    return launch_prompt_t5(a, n_pairs, G, DENSE, WANT_Y, stream);
  if (dtype == KVPOP_BF16) {
    if (d == 128) {
      if (G == 4) return launch_tc<128, 4, DENSE, WANT_Y>(a, n_pairs, stream);
      if (G == 2) return launch_tc<128, 2, DENSE, WANT_Y>(a, n_pairs, stream);
      return launch_tc<128, 1, DENSE, WANT_Y>(a, n_pairs, stream);
    }
    if (G == 4) return launch_tc<64, 4, DENSE, WANT_Y>(a, n_pairs, stream);
    if (G == 2) return launch_tc<64, 2, DENSE, WANT_Y>(a, n_pairs, stream);
    return launch_tc<64, 1, DENSE, WANT_Y>(a, n_pairs, stream);
  }
  if (d == 128) return launch_simt<float, 128, DENSE>(a, n_pairs, stream);
  return launch_simt<float, 64, DENSE>(a, n_pairs, stream);
}

}  // namespace

bool prompt_attend_ok(int dtype, int d, int G, int s, int w, int k) {
  if (!(d == 64 || d == 128) || !(G == 1 || G == 2 || G == 4)) return false;
  const long long capA = (long long)s + k;
  const long long capM = (long long)s + 2 * 128 + w;
  const long long bytes = 4 * (capA + capM) + (dtype == KVPOP_BF16 ? 68 * 1024 : 8 * 1024);
  return bytes <= 227 * 1024;
}

cudaError_t launch_prompt_attend(const void* Q, const void* K, const void* V, const int32_t* rank,
                                 const int32_t* tau, const int32_t* order, const int32_t* len,
                                 int n_seq, int H, int G, int d, int S, int s, int w, int k,
                                 int dtype, float* Y, float* lse, int32_t* err, cudaStream_t stream) {
  if (n_seq <= 0 || S <= 0) return cudaSuccess;
  PromptArgs a{Q, K, V, rank, tau, order, len, Y, lse, H, G, S, s, w, s + k, 0,
               1.4426950408889634f / sqrtf((float)d), err};
  return dispatch<false, true>(a, n_seq * H, dtype, d, G, stream);
}

cudaError_t launch_causal_lse(const void* Q, const void* K, const int32_t* len, int n_seq, int H,
                              int G, int d, int S, int dtype, float* lse, int32_t* err,
                              cudaStream_t stream) {
  if (n_seq <= 0 || S <= 0) return cudaSuccess;
  PromptArgs a{Q, K, nullptr, nullptr, nullptr, nullptr, len, nullptr, lse, H, G, S, 0, 1, 0, 0,
               1.4426950408889634f / sqrtf((float)d), err};
  return dispatch<true, false>(a, n_seq * H, dtype, d, G, stream);
}

}  // namespace kvpop
