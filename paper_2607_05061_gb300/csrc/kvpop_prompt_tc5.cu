// Masked prompt attention on the 5th-generation tensor cores (tcgen05), bf16
// with head dimension 128 (App. C.1 mask, App. C.3; the dense causal form
// gives the normalisers of App. D.1).
//
// Same tiling and key lists as the m16n8k16 kernel (kvpop_prompt.cu): a CTA
// owns 128 (query, head) rows -- 128 / G consecutive queries with all G heads of
// one KV head -- and walks the tile's candidate keys in blocks of 64.  Roles:
//  * 4 producer warps gather the block's K and V rows by position with 16-byte
//    cp.async into 128B-swizzled tiles (3 stages); completion arrives on the
//    stage's mbarrier asynchronously (cp.async.mbarrier.arrive.noinc).
//  * 1 MMA warp: one thread issues S = Q K^T (M 128, N 64, K 128; Q and K
//    K-major) into one of two tensor-memory S buffers, and O += P V (M 128,
//    N 128, K 64; P K-major from shared memory, V read MN-major straight from
//    its gathered rows) into the tensor-memory O accumulator; tcgen05.commit
//    signals S ready, P consumed and the stage free.
//  * 4 softmax warps, one thread per row: read the row of S from tensor memory
//    (32x32b loads), apply the mask on the few blocks that need it, keep a
//    running maximum that is only raised when a logit exceeds it by 2^8 (the
//    accumulator in tensor memory is then rescaled in place), write the bf16
//    probabilities into the swizzled P tile and hand it to the MMA warp.
// Outputs as the other kernels: y in fp32 and the natural-log normaliser.
// Every wait is bounded; on expiry the kernel records an error code, stops
// issuing work, lets its copies drain and frees its tensor memory.
#include "kvpop_mma.cuh"
#include "kvpop_prompt.cuh"
#include "kvpop_ptx.cuh"
#include "kvpop_tc05.cuh"

namespace kvpop {
namespace {

using namespace prompt;
using namespace tc05;

constexpr int T5_THREADS = 288;          // 4 softmax warps, 1 MMA warp, 4 producer warps
constexpr int T5_ROWS = 128;
constexpr int T5_BN = 64;
constexpr int T5_STAGES = 3;
constexpr int T5_TMEM_COLS = 256;        // O: 0..127, S buffers: 128..191, 192..255
constexpr float T5_THR = 8.0f;

constexpr int OFF_Q = 0;                               // 128 x 128 bf16
constexpr int OFF_K = OFF_Q + 32768;                   // 3 x (64 x 128 bf16)
constexpr int OFF_V = OFF_K + T5_STAGES * 16384;
constexpr int OFF_P = OFF_V + T5_STAGES * 16384;       // 2 x (128 x 64 bf16)
constexpr int OFF_BAR = OFF_P + 2 * 16384;
constexpr int OFF_TMEM = OFF_BAR + 128;
constexpr int OFF_TAU = OFF_TMEM + 16;
constexpr int OFF_RED = OFF_TAU + T5_ROWS * 4;
constexpr int OFF_LIST = OFF_RED + 16 * 4;
enum { B_FULL = 0, B_EMPTY = 3, B_SFULL = 6, B_PFULL = 8, B_ODONE = 10, B_QFULL = 12 };
enum : int { T5ERR_WAIT = 21 };

template <int G, bool DENSE, bool WANT_Y>
__global__ void __launch_bounds__(T5_THREADS, 1) prompt_t5_kernel(PromptArgs a) {
  constexpr int BM = T5_ROWS / G;
  extern __shared__ __align__(1024) unsigned char sm5[];
  const uint32_t sb = smem_u32(sm5);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  auto bar = [&](int i) { return sb + OFF_BAR + 8u * (uint32_t)i; };
  int* tauS = reinterpret_cast<int*>(sm5 + OFF_TAU);
  int* red = reinterpret_cast<int*>(sm5 + OFF_RED);
  int32_t* posA = reinterpret_cast<int32_t*>(sm5 + OFF_LIST);
  int32_t* posM = posA + a.capA;

  if (tid == 0) {
    for (int i = 0; i < T5_STAGES; ++i) {
      mbar_init(bar(B_FULL + i), 128);
      mbar_init(bar(B_EMPTY + i), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(bar(B_SFULL + i), 1);
      mbar_init(bar(B_PFULL + i), 128);
      mbar_init(bar(B_ODONE + i), 1);
    }
    mbar_init(bar(B_QFULL), 128);
    mbar_fence_init();
  }
  if (warp == 4) tmem_alloc(sb + OFF_TMEM, T5_TMEM_COLS);
  TileInfo ti;
  bool live;
  if (DENSE) live = dense_setup(a, BM, ti);
  else live = tile_setup<T5_THREADS>(a, BM, tauS, red, posA, posM, ti);
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(sm5 + OFF_TMEM);
  if (live) {
    const int H = a.H, S = a.S, nA = ti.nA, nU = ti.nA + ti.nM;
    const int nblk = (nU + T5_BN - 1) / T5_BN;
    const size_t pair_off = (size_t)ti.pair * S;
    auto entry = [&](int e) -> int {
      if (DENSE) return e < nU ? e : 0;
      if (e < nA) return posA[e];
      return e < nU ? posM[e - nA] : (nA > 0 ? posA[0] : posM[0]);
    };
    if (warp >= 5) {
      // ---------------------------------------------------------------- producers
      const int pt = tid - 160;
      const bf16* Qb = static_cast<const bf16*>(a.Q) + ((size_t)ti.seq * H * G + (size_t)ti.h * G) * S * 128;
      const bf16* Kp = static_cast<const bf16*>(a.K) + pair_off * 128;
      const bf16* Vp = WANT_Y ? static_cast<const bf16*>(a.V) + pair_off * 128 : nullptr;
      for (int i = pt; i < T5_ROWS * 16; i += 128) {
        const int r = i >> 4, c = i & 15;
        const int q = ti.q0 + r / G, g = r % G;
        const bool ok = q <= ti.q1;
        cp_async16(sb + OFF_Q + tile_off(r, c, T5_ROWS),
                   Qb + ((size_t)g * S + (ok ? q : ti.q0)) * 128 + c * 8, ok ? 16 : 0);
      }
      cp_async_arrive_noinc(bar(B_QFULL));
      for (int j = 0; j < nblk; ++j) {
        const int st = j % T5_STAGES;
        if (j >= T5_STAGES && !mbar_wait(bar(B_EMPTY + st), ((j / T5_STAGES) - 1) & 1, a.err, T5ERR_WAIT))
          break;
        const uint32_t kd = sb + OFF_K + st * 16384, vd = sb + OFF_V + st * 16384;
        for (int i = pt; i < T5_BN * 16; i += 128) {
          const int key = i >> 4, c = i & 15;
          const int t = entry(j * T5_BN + key);
          const uint32_t off = tile_off(key, c, T5_BN);
          cp_async16(kd + off, Kp + (size_t)t * 128 + c * 8, 16);
          if (WANT_Y) cp_async16(vd + off, Vp + (size_t)t * 128 + c * 8, 16);
        }
        cp_async_arrive_noinc(bar(B_FULL + st));
      }
      cp_wait<0>();
    } else if (warp == 4) {
      // ---------------------------------------------------------------- MMA issue
      if (lane == 0) {
        const uint32_t idS = idesc_bf16(128, T5_BN, 0);
        const uint32_t idO = idesc_bf16(128, 128, 1);
        bool ok = mbar_wait(bar(B_QFULL), 0, a.err, T5ERR_WAIT);
        auto issue_s = [&](int j) {
          const int st = j % T5_STAGES;
          if (!ok || !(ok = mbar_wait(bar(B_FULL + st), (j / T5_STAGES) & 1, a.err, T5ERR_WAIT))) return;
          fence_async_smem();
          fence_after();
          const uint32_t dS = tmem + 128 + (uint32_t)(j & 1) * T5_BN;
#pragma unroll
          for (int ks = 0; ks < 8; ++ks)
            mma_bf16(dS, kmajor_desc(sb + OFF_Q, T5_ROWS, ks),
                     kmajor_desc(sb + OFF_K + st * 16384, T5_BN, ks), idS, ks > 0);
          commit(bar(B_SFULL + (j & 1)));
          if (!WANT_Y) commit(bar(B_EMPTY + st));
        };
        if (ok) fence_async_smem();
        issue_s(0);
        if (nblk > 1) issue_s(1);
        for (int j = 0; j < nblk && ok; ++j) {
          const int st = j % T5_STAGES;
          if (!(ok = mbar_wait(bar(B_PFULL + (j & 1)), (j >> 1) & 1, a.err, T5ERR_WAIT))) break;
          fence_after();
          if (WANT_Y) {
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              mma_bf16(tmem, kmajor_desc(sb + OFF_P + (j & 1) * 16384, T5_ROWS, kk),
                       mnmajor_desc(sb + OFF_V + st * 16384, T5_BN, kk), idO, (j > 0 || kk > 0));
            commit(bar(B_ODONE + (j & 1)));
            commit(bar(B_EMPTY + st));
          }
          if (j + 2 < nblk) issue_s(j + 2);
        }
      }
      __syncwarp();
    } else {
      // ---------------------------------------------------------------- softmax rows
      const int r = tid;
      const int ql = r / G, g = r - ql * G;
      const int q = ti.q0 + ql;
      const bool valid = q <= ti.q1;
      const int tq = DENSE ? 0 : tauS[ql];
      const uint32_t trow = (uint32_t)(warp * 32) << 16;
      const int32_t* rank = DENSE ? nullptr : a.rank + pair_off;
      float m = -INFINITY, l = 0.f;
      bool ok = true;
      // tcgen05.ld / st are warp-collective: every branch around them is warp-uniform
      auto uniform = [](bool x) { return __all_sync(0xffffffffu, x); };
      for (int j = 0; j < nblk; ++j) {
        const int b = j & 1;
        if (!(ok = uniform(mbar_wait(bar(B_SFULL + b), (j >> 1) & 1, a.err, T5ERR_WAIT)))) break;
        fence_after();
        float s[64];
        {
          float* s0 = s;
          tmem_ld32(tmem + trow + 128 + b * T5_BN, *reinterpret_cast<float(*)[32]>(s0));
          tmem_ld32(tmem + trow + 128 + b * T5_BN + 32, *reinterpret_cast<float(*)[32]>(s0 + 32));
          tmem_wait_ld();
        }
#pragma unroll
        for (int i = 0; i < 64; ++i) s[i] *= a.qscale;
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
        float mx = -INFINITY;
#pragma unroll
        for (int i = 0; i < 64; ++i) mx = fmaxf(mx, s[i]);
        float alpha = 1.f, m_new = m;
        bool resc = false;
        if (mx > m + T5_THR) {
          m_new = mx;
          alpha = ex2(m - m_new);
          resc = m != -INFINITY;
        }
        const float base = m_new == -INFINITY ? 0.f : m_new;
        if (WANT_Y) {
          if (j >= 2 &&
              !(ok = uniform(mbar_wait(bar(B_ODONE + b), ((j - 2) >> 1) & 1, a.err, T5ERR_WAIT))))
            break;
          // rows whose maximum moved: rescale their accumulator once PV_{j-1} has landed
          if (j >= 1 && __any_sync(0xffffffffu, resc)) {
            if (!(ok = uniform(mbar_wait(bar(B_ODONE + ((j - 1) & 1)), ((j - 1) >> 1) & 1, a.err,
                                         T5ERR_WAIT))))
              break;
            fence_after();
            const float f = resc ? alpha : 1.f;
#pragma unroll
            for (int c = 0; c < 4; ++c) {
              float o[32];
              tmem_ld32(tmem + trow + c * 32, o);
              tmem_wait_ld();
#pragma unroll
              for (int i = 0; i < 32; ++i) o[i] *= f;
              tmem_st32(tmem + trow + c * 32, o);
            }
            tmem_wait_st();
          }
        }
        float sum = 0.f;
#pragma unroll
        for (int i = 0; i < 64; ++i) {
          s[i] = ex2(s[i] - base);
          sum += s[i];
        }
        l = l * alpha + sum;
        m = m_new;
        if (WANT_Y) {
          unsigned char* prow = sm5 + OFF_P + b * 16384;
#pragma unroll
          for (int c = 0; c < 8; ++c) {
            uint4 v;
            v.x = pack_bf16(s[8 * c + 0], s[8 * c + 1]);
            v.y = pack_bf16(s[8 * c + 2], s[8 * c + 3]);
            v.z = pack_bf16(s[8 * c + 4], s[8 * c + 5]);
            v.w = pack_bf16(s[8 * c + 6], s[8 * c + 7]);
            *reinterpret_cast<uint4*>(prow + tile_off(r, c, T5_ROWS)) = v;
          }
          fence_async_smem();
        }
        fence_before();
        mbar_arrive(bar(B_PFULL + b));
      }
      const size_t row = ((size_t)ti.seq * H * G + (size_t)ti.h * G + g) * S + q;
      if (WANT_Y && ok && nblk > 0) {
        ok = uniform(mbar_wait(bar(B_ODONE + ((nblk - 1) & 1)), ((nblk - 1) >> 1) & 1, a.err, T5ERR_WAIT));
        fence_after();
        if (ok) {
          const float inv = 1.f / l;
          float4* y = reinterpret_cast<float4*>(a.Y + row * 128);
#pragma unroll
          for (int c = 0; c < 4; ++c) {
            float o[32];
            tmem_ld32(tmem + trow + c * 32, o);
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
  if (warp == 4) tmem_dealloc(tmem, T5_TMEM_COLS);
}

template <int G, bool DENSE, bool WANT_Y>
cudaError_t launch_t5_g(PromptArgs a, int n_pairs, cudaStream_t stream) {
  constexpr int BM = T5_ROWS / G;
  if (DENSE) a.capA = a.capM = 0;
  else a.capM = a.s + 2 * BM + a.w;
  const size_t smem = (size_t)OFF_LIST + (size_t)(a.capA + a.capM) * 4;
  if (smem > 227 * 1024) return cudaErrorInvalidValue;
  auto k = prompt_t5_kernel<G, DENSE, WANT_Y>;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  dim3 grid((a.S + BM - 1) / BM, n_pairs);
  k<<<grid, T5_THREADS, smem, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace

bool prompt_t5_ok(int d, int G, int s, int w, int k) {
  if (d != 128 || !(G == 1 || G == 2 || G == 4)) return false;
  const long long lists = (long long)s + k + s + 2 * T5_ROWS + w;
  return OFF_LIST + 4 * lists <= 227 * 1024;
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
