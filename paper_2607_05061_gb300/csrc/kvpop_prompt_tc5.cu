// Masked prompt attention on the 5th-generation tensor cores (tcgen05), bf16
// with head dimension 128 (App. C.1 mask, App. C.3; the dense causal form
// gives the normalisers of App. D.1).
//
// Same key lists as the m16n8k16 kernel (kvpop_prompt.cu), built for 256 / G
// consecutive queries of one (sequence, KV head): the CTA's 256 (query, head)
// rows form two 128-row halves that share every gathered K/V block, so each
// gathered byte feeds two M = 128 MMAs.  Roles:
//  * 3 producer warps gather the block's K and V rows by position with 16-byte
//    cp.async into 128B-swizzled tiles (2 or 3 stages, as shared memory
//    allows); completion arrives on the stage's mbarrier asynchronously
//    (cp.async.mbarrier.arrive.noinc).
//  * 1 MMA warp: one thread issues, per half, S = Q K^T (M 128, N 64, K 128;
//    Q and K K-major) into one of two tensor-memory S buffers, and O += P V
//    (M 128, N 128, K 64; P K-major from shared memory, V read MN-major straight
//    from its gathered rows) into the half's tensor-memory accumulator;
//    tcgen05.commit signals S ready, P consumed and the stage free.  Tensor
//    memory: O of both halves (256 columns) and their S double buffers (256).
//  * 2 softmax warpgroups, one per half, one thread per row: read the row of S
//    (32x32b loads), apply the mask on the few blocks that need it, keep a
//    running maximum that is only raised when a logit exceeds it by 2^8 (the
//    row of the accumulator is then rescaled in place), write the bf16
//    probabilities into the half's swizzled P tile and hand it over.
// Outputs as the other kernels: y in fp32 and the natural-log normaliser.
// Every wait is bounded; on expiry the kernel records an error code, stops
// issuing work, lets its copies drain and frees its tensor memory.  Every
// tensor-memory access, and every branch around one, is warp-uniform.
#include "kvpop_mma.cuh"
#include "kvpop_prompt.cuh"
#include "kvpop_ptx.cuh"
#include "kvpop_tc05.cuh"

namespace kvpop {
namespace {

using namespace prompt;
using namespace tc05;

constexpr int T5_HALF = 128;                     // rows per half (MMA M)
constexpr int T5_ROWS = 2 * T5_HALF;             // (query, head) rows per CTA
constexpr int T5_BN = 64;                        // keys per block
constexpr int T5_MMA_WARP = 8;                   // warps 0-7: softmax, 8: MMA, 9-11: producers
constexpr int T5_NPROD = 3;
constexpr int T5_PT = 32 * T5_NPROD;
constexpr int T5_THREADS = 32 * (T5_MMA_WARP + 1 + T5_NPROD);   // 12 warps: 168 registers fit
static_assert(T5_THREADS / 32 + 2 <= 16, "the prologue's per-warp reduction slots");
constexpr int T5_TMEM_COLS = 512;                // O_h: 128 h .. ; S_{h,b}: 256 + 128 h + 64 b
constexpr float T5_THR = 8.0f;

constexpr int QB = T5_HALF * 256;                // Q tile of one half, bytes
constexpr int KVB = T5_BN * 256;                 // K (or V) block, bytes
constexpr int PB = T5_HALF * T5_BN * 2;          // P tile of one half, bytes
constexpr int OFF_Q = 0;
constexpr int OFF_KV = OFF_Q + 2 * QB;           // stages of [K | V]
template <int ST>
struct Lay {
  static constexpr int OFF_P = OFF_KV + ST * 2 * KVB;
  static constexpr int OFF_BAR = OFF_P + 2 * PB;
  static constexpr int OFF_TMEM = OFF_BAR + 256;
  static constexpr int OFF_TAU = OFF_TMEM + 16;
  static constexpr int OFF_RED = OFF_TAU + T5_ROWS * 4;
  static constexpr int OFF_LIST = OFF_RED + 16 * 4;
};
// barrier indices
constexpr int B_FULL = 0;          // [3]  producers -> MMA
constexpr int B_EMPTY = 3;         // [3]  MMA -> producers
constexpr int B_SFULL = 6;         // [2 halves][2 buffers]  MMA -> softmax
constexpr int B_PFULL = 10;        // [2][2]  softmax -> MMA
constexpr int B_ODONE = 14;        // [2]  MMA -> softmax (one per half)
constexpr int B_QFULL = 16;
enum : int { T5ERR_WAIT = 21 };

template <int G, bool DENSE, bool WANT_Y, int ST>
__global__ void __launch_bounds__(T5_THREADS, 1) prompt_t5_kernel(PromptArgs a) {
  using L = Lay<ST>;
  constexpr int BM = T5_ROWS / G;
  extern __shared__ __align__(1024) unsigned char sm5[];
  const uint32_t sb = smem_u32(sm5);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  auto bar = [&](int i) { return sb + L::OFF_BAR + 8u * (uint32_t)i; };
  int* tauS = reinterpret_cast<int*>(sm5 + L::OFF_TAU);
  int* red = reinterpret_cast<int*>(sm5 + L::OFF_RED);
  int32_t* posA = reinterpret_cast<int32_t*>(sm5 + L::OFF_LIST);
  int32_t* posM = posA + a.capA;

  if (tid == 0) {
    for (int i = 0; i < ST; ++i) {
      mbar_init(bar(B_FULL + i), T5_PT);
      mbar_init(bar(B_EMPTY + i), 1);
    }
    for (int i = 0; i < 4; ++i) {
      mbar_init(bar(B_SFULL + i), 1);
      mbar_init(bar(B_PFULL + i), 128);
    }
    mbar_init(bar(B_ODONE + 0), 1);
    mbar_init(bar(B_ODONE + 1), 1);
    mbar_init(bar(B_QFULL), T5_PT);
    mbar_fence_init();
  }
  if (warp == T5_MMA_WARP) tmem_alloc(sb + L::OFF_TMEM, T5_TMEM_COLS);
  TileInfo ti;
  bool live;
  if (DENSE) live = dense_setup(a, BM, ti);
  else live = tile_setup<T5_THREADS>(a, BM, tauS, red, posA, posM, ti);
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(sm5 + L::OFF_TMEM);
  if (live) {
    const int H = a.H, S = a.S, nA = ti.nA, nU = ti.nA + ti.nM;
    const int nblk = (nU + T5_BN - 1) / T5_BN;
    const size_t pair_off = (size_t)ti.pair * S;
    auto entry = [&](int e) -> int {
      if (DENSE) return e < nU ? e : 0;
      if (e < nA) return posA[e];
      return e < nU ? posM[e - nA] : (nA > 0 ? posA[0] : posM[0]);
    };
    if (warp > T5_MMA_WARP) {
      // ---------------------------------------------------------------- producers
      const int pt = tid - 32 * (T5_MMA_WARP + 1);
      const bf16* Qb = static_cast<const bf16*>(a.Q) + ((size_t)ti.seq * H * G + (size_t)ti.h * G) * S * 128;
      const bf16* Kp = static_cast<const bf16*>(a.K) + pair_off * 128;
      const bf16* Vp = WANT_Y ? static_cast<const bf16*>(a.V) + pair_off * 128 : nullptr;
      for (int i = pt; i < T5_ROWS * 16; i += T5_PT) {
        const int r = i >> 4, c = i & 15;
        const int q = ti.q0 + r / G, g = r % G;
        const bool ok = q <= ti.q1;
        cp_async16(sb + OFF_Q + (r >> 7) * QB + tile_off(r & 127, c, T5_HALF),
                   Qb + ((size_t)g * S + (ok ? q : ti.q0)) * 128 + c * 8, ok ? 16 : 0);
      }
      cp_async_arrive_noinc(bar(B_QFULL));
      for (int j = 0; j < nblk; ++j) {
        const int st = j % ST;
        if (j >= ST && !mbar_wait(bar(B_EMPTY + st), ((j / ST) - 1) & 1, a.err, T5ERR_WAIT)) break;
        const uint32_t kd = sb + OFF_KV + st * 2 * KVB, vd = kd + KVB;
        // 8 threads per key row, 32 bytes (two 16-byte chunks) of K and of V each:
        // one position lookup per row and thread, rows T5_PT / 8 apart
        const int c2 = 2 * (pt & 7);
#pragma unroll 2
        for (int key = pt >> 3; key < T5_BN; key += T5_PT / 8) {
          const size_t t = (size_t)entry(j * T5_BN + key) * 128 + c2 * 8;
          const uint32_t o0 = tile_off(key, c2, T5_BN), o1 = tile_off(key, c2 + 1, T5_BN);
          cp_async16(kd + o0, Kp + t, 16);
          cp_async16(kd + o1, Kp + t + 8, 16);
          if (WANT_Y) {
            cp_async16(vd + o0, Vp + t, 16);
            cp_async16(vd + o1, Vp + t + 8, 16);
          }
        }
        cp_async_arrive_noinc(bar(B_FULL + st));
      }
      cp_wait<0>();
    } else if (warp == T5_MMA_WARP) {
      // ---------------------------------------------------------------- MMA issue
      if (lane == 0) {
        const uint32_t idS = idesc_bf16(128, T5_BN, 0);
        const uint32_t idO = idesc_bf16(128, 128, 1);
        bool ok = mbar_wait(bar(B_QFULL), 0, a.err, T5ERR_WAIT);
        if (ok) fence_async_smem();
        auto issue_s = [&](int j) {
          const int st = j % ST;
          if (!ok || !(ok = mbar_wait(bar(B_FULL + st), (j / ST) & 1, a.err, T5ERR_WAIT))) return;
          fence_async_smem();
          fence_after();
          const uint32_t kb = sb + OFF_KV + st * 2 * KVB;
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const uint32_t dS = tmem + 256 + h * 128 + (uint32_t)(j & 1) * T5_BN;
#pragma unroll
            for (int ks = 0; ks < 8; ++ks)
              mma_bf16(dS, kmajor_desc(sb + OFF_Q + h * QB, T5_HALF, ks), kmajor_desc(kb, T5_BN, ks),
                       idS, ks > 0);
            commit(bar(B_SFULL + 2 * h + (j & 1)));
          }
          if (!WANT_Y) commit(bar(B_EMPTY + st));
        };
        issue_s(0);
        if (nblk > 1) issue_s(1);
        for (int j = 0; j < nblk && ok; ++j) {
          const int st = j % ST;
          const uint32_t vb = sb + OFF_KV + st * 2 * KVB + KVB;
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            if (!(ok = mbar_wait(bar(B_PFULL + 2 * h + (j & 1)), (j >> 1) & 1, a.err, T5ERR_WAIT))) break;
            fence_after();
            if (WANT_Y) {
#pragma unroll
              for (int kk = 0; kk < 4; ++kk)
                mma_bf16(tmem + h * 128, kmajor_desc(sb + L::OFF_P + h * PB, T5_HALF, kk),
                         mnmajor_desc(vb, T5_BN, kk), idO, (j > 0 || kk > 0));
              commit(bar(B_ODONE + h));
            }
          }
          if (!ok) break;
          if (WANT_Y) commit(bar(B_EMPTY + st));
          if (j + 2 < nblk) issue_s(j + 2);
        }
      }
      __syncwarp();
    } else {
      // ---------------------------------------------------------------- softmax rows
      const int h = warp >> 2;                      // half
      const int r = (warp & 3) * 32 + lane;         // row of the half = tensor-memory lane
      const int rr = h * T5_HALF + r;               // row of the CTA tile
      const int ql = rr / G, g = rr - ql * G;
      const int q = ti.q0 + ql;
      const bool valid = q <= ti.q1;
      const int tq = DENSE ? 0 : tauS[ql];
      const uint32_t trow = (uint32_t)((warp & 3) * 32) << 16;
      const uint32_t tO = tmem + trow + h * 128, tS = tmem + trow + 256 + h * 128;
      const int32_t* rank = DENSE ? nullptr : a.rank + pair_off;
      const float c2 = a.qscale;
      float m = -INFINITY, l = 0.f;
      bool ok = true;
      auto uniform = [](bool x) { return __all_sync(0xffffffffu, x); };
      for (int j = 0; j < nblk; ++j) {
        const int b = j & 1;
        if (!(ok = uniform(mbar_wait(bar(B_SFULL + 2 * h + b), (j >> 1) & 1, a.err, T5ERR_WAIT))))
          break;
        fence_after();
        float s[64];
        tmem_ld32(tS + b * T5_BN, *reinterpret_cast<float(*)[32]>(s));
        tmem_ld32(tS + b * T5_BN + 32, *reinterpret_cast<float(*)[32]>(s + 32));
        tmem_wait_ld();
        if ((j + 1) * T5_BN > nA) {                 // block holds keys that need the mask
#pragma unroll
          for (int i = 0; i < 64; ++i) {
            const int e = j * T5_BN + i;
            if (e >= nA) {
              bool kp = false;
              if (e < nU) {
                const int t = entry(e);
                kp = DENSE ? t <= q : keep_key(q, t, __ldg(rank + t), tq, a.s, a.w);
              }
              if (!kp) s[i] = -INFINITY;
            }
          }
        }
        // 8 independent chains of three-input maxima (one 64-long chain would serialise)
        float pm[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) pm[k] = s[k];
#pragma unroll
        for (int i = 8; i < 56; i += 16)
#pragma unroll
          for (int k = 0; k < 8; ++k) pm[k] = fmax3(pm[k], s[i + k], s[i + 8 + k]);
#pragma unroll
        for (int k = 0; k < 8; ++k) pm[k] = fmaxf(pm[k], s[56 + k]);
        const float mx = fmax3(fmax3(pm[0], pm[1], pm[2]), fmax3(pm[3], pm[4], pm[5]), fmaxf(pm[6], pm[7]));
        const float mxs = mx * c2;                  // row maximum, log2 units
        float alpha = 1.f, m_new = m;
        bool resc = false;
        if (mxs > m + T5_THR) {
          m_new = mxs;
          alpha = ex2(m - m_new);
          resc = m != -INFINITY;
        }
        const float base = m_new == -INFINITY ? 0.f : m_new;
        // probabilities 2^(s c2 - base): scale-and-shift and the partial sums in packed pairs
        const uint64_t cc = f2_pack(c2, c2), nb = f2_pack(-base, -base);
        uint64_t ps2[4] = {0ull, 0ull, 0ull, 0ull};
#pragma unroll
        for (int i = 0; i < 64; i += 8) {
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            float x0, x1;
            f2_unpack(f2_fma(f2_pack(s[i + 2 * k], s[i + 2 * k + 1]), cc, nb), x0, x1);
            s[i + 2 * k] = ex2(x0);
            s[i + 2 * k + 1] = ex2(x1);
            ps2[k] = f2_add(ps2[k], f2_pack(s[i + 2 * k], s[i + 2 * k + 1]));
          }
        }
        float ps[8];
#pragma unroll
        for (int k = 0; k < 4; ++k) f2_unpack(ps2[k], ps[2 * k], ps[2 * k + 1]);
        const float sum = ((ps[0] + ps[1]) + (ps[2] + ps[3])) + ((ps[4] + ps[5]) + (ps[6] + ps[7]));
        l = l * alpha + sum;
        m = m_new;
        if (WANT_Y && j >= 1) {
          // PV_{j-1} must have consumed the P tile (and landed in O) before either changes;
          // the exponentials above overlap with it
          if (!(ok = uniform(mbar_wait(bar(B_ODONE + h), (j - 1) & 1, a.err, T5ERR_WAIT)))) break;
          if (__any_sync(0xffffffffu, resc)) {
            fence_after();
            const float f = resc ? alpha : 1.f;
#pragma unroll
            for (int c = 0; c < 4; ++c) {
              float o[32];
              tmem_ld32(tO + c * 32, o);
              tmem_wait_ld();
#pragma unroll
              for (int i = 0; i < 32; ++i) o[i] *= f;
              tmem_st32(tO + c * 32, o);
            }
            tmem_wait_st();
          }
        }
        if (WANT_Y) {
          unsigned char* prow = sm5 + L::OFF_P + h * PB;
#pragma unroll
          for (int c = 0; c < 8; ++c) {
            uint4 v;
            v.x = pack_bf16(s[8 * c + 0], s[8 * c + 1]);
            v.y = pack_bf16(s[8 * c + 2], s[8 * c + 3]);
            v.z = pack_bf16(s[8 * c + 4], s[8 * c + 5]);
            v.w = pack_bf16(s[8 * c + 6], s[8 * c + 7]);
            *reinterpret_cast<uint4*>(prow + tile_off(r, c, T5_HALF)) = v;
          }
          fence_async_smem();
        }
        fence_before();
        mbar_arrive(bar(B_PFULL + 2 * h + b));
      }
      const size_t row = ((size_t)ti.seq * H * G + (size_t)ti.h * G + g) * S + q;
      if (WANT_Y && ok && nblk > 0) {
        ok = uniform(mbar_wait(bar(B_ODONE + h), (nblk - 1) & 1, a.err, T5ERR_WAIT));
        fence_after();
        if (ok) {
          const float inv = 1.f / l;
          float4* y = reinterpret_cast<float4*>(a.Y + row * 128);
#pragma unroll
          for (int c = 0; c < 4; ++c) {
            float o[32];
            tmem_ld32(tO + c * 32, o);
            tmem_wait_ld();
            if (valid) {
#pragma unroll
              for (int i = 0; i < 8; ++i)
                y[c * 8 + i] = make_float4(o[4 * i] * inv, o[4 * i + 1] * inv, o[4 * i + 2] * inv,
                                           o[4 * i + 3] * inv);
            }
          }
        }
      }
      if (ok && valid && a.lse) a.lse[row] = l > 0.f ? (m + __log2f(l)) * kLn2 : -INFINITY;
    }
  }
  fence_before();
  __syncthreads();
  if (warp == T5_MMA_WARP) tmem_dealloc(tmem, T5_TMEM_COLS);
}

template <int ST>
size_t t5_smem(int capA, int capM) {
  return (size_t)Lay<ST>::OFF_LIST + (size_t)(capA + capM) * 4;
}

template <int G, bool DENSE, bool WANT_Y, int ST>
cudaError_t launch_t5_st(const PromptArgs& a, int n_pairs, size_t smem, cudaStream_t stream) {
  constexpr int BM = T5_ROWS / G;
  auto k = prompt_t5_kernel<G, DENSE, WANT_Y, ST>;
  cudaError_t e = raise_smem_limit(k, smem);
  if (e != cudaSuccess) return e;
  dim3 grid((a.S + BM - 1) / BM, n_pairs);
  k<<<grid, T5_THREADS, smem, stream>>>(a);
  return cudaGetLastError();
}

template <int G, bool DENSE, bool WANT_Y>
cudaError_t launch_t5_g(PromptArgs a, int n_pairs, cudaStream_t stream) {
  constexpr int BM = T5_ROWS / G;
  if (DENSE) a.capA = a.capM = 0;
  else a.capM = a.s + 2 * BM + a.w;
  const size_t s3 = t5_smem<3>(a.capA, a.capM), s2 = t5_smem<2>(a.capA, a.capM);
  if (s3 <= 227 * 1024) return launch_t5_st<G, DENSE, WANT_Y, 3>(a, n_pairs, s3, stream);
  if (s2 <= 227 * 1024) return launch_t5_st<G, DENSE, WANT_Y, 2>(a, n_pairs, s2, stream);
  return cudaErrorInvalidValue;
}

}  // namespace

bool prompt_t5_ok(int d, int G, int s, int w, int k) {
  if (d != 128 || !(G == 1 || G == 2 || G == 4)) return false;
  const long long lists = (long long)s + k + s + 2 * T5_ROWS + w;
  return Lay<2>::OFF_LIST + 4 * lists <= 227 * 1024;
}

cudaError_t launch_prompt_t5(const PromptArgs& a, int n_pairs, int G, bool dense, bool want_y,
                             cudaStream_t stream) {
  if (dense) {
    if (G == 4) return launch_t5_g<4, true, false>(a, n_pairs, stream);
    if (G == 2) return launch_t5_g<2, true, false>(a, n_pairs, stream);
    return launch_t5_g<1, true, false>(a, n_pairs, stream);
  }
  (void)want_y;
  if (G == 4) return launch_t5_g<4, false, true>(a, n_pairs, stream);
  if (G == 2) return launch_t5_g<2, false, true>(a, n_pairs, stream);
  return launch_t5_g<1, false, true>(a, n_pairs, stream);
}

}  // namespace kvpop
