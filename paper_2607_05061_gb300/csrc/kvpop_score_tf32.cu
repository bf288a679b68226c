// Delayed MLP scorer over every prompt token on the 5th-generation tensor cores
// with fp32 accuracy (Sec. 3.3, App. E.2, E.4: r_u = w2 . act(W1^T x_u + b1) + b2,
// x_u = [k_u; v_u; qbar_u]).
//
// The hidden pre-activations H = X W1 form an fp32 GEMM (tokens x 3d times
// 3d x F).  Each operand is split into a tf32 head and an fp32 residual,
// a = a_hi + a_lo with a_hi = tf32(a), and H = X_hi W_hi + X_hi W_lo + X_lo W_hi
// runs as three kind::tf32 tcgen05 MMAs into an fp32 tensor-memory accumulator
// (the dropped X_lo W_lo term is below fp32 rounding; measured error ~1e-6 of
// sum |x w|, like an fp32 FMA chain).  W1^T is split once when the cache is made.
//
// A CTA scores 128 consecutive tokens of one (sequence, KV head):
//  * 8 builder warps write the scorer inputs chunk by chunk (32 input dims, one
//    128-byte fp32 row per token, hi and lo parts) into 128B-swizzled shared
//    memory, two buffers deep; for the qbar chunks they first stage the query
//    means (mean over the G heads) of the positions u0+1 .. u0+126+D and then
//    average D of them per token, in the same order as the other kernels;
//  * one thread loads the matching W1^T chunk (hi and lo, F rows x 32) by TMA
//    and issues the 3 x 4 MMAs (M = 128, N = F, K = 8 each) per chunk -- 2 x 4 for
//    the k and v chunks of bf16 inputs, which are exact in tf32 (their lo is 0 and
//    is not stored);
//  * the builders finish: each thread reads half of its token's F pre-activations
//    from tensor memory, adds b1, applies the activation, dots with w2, and one
//    of the two halves writes the token's static priority.
// Every wait is bounded; an expired wait records an error code and stops the CTA.
#include <cuda.h>

#include <type_traits>

#include "kvpop_internal.cuh"
#include "kvpop_ptx.cuh"
#include "kvpop_tc05.cuh"

namespace kvpop {
namespace {

using namespace tc05;

constexpr int SC_M = 128;                 // tokens per CTA (MMA M)
constexpr int SC_KC = 32;                 // input dims per chunk (one 128-byte fp32 row)
constexpr int SC_BUILD = 256;             // builder / epilogue threads
constexpr int SC_THREADS = SC_BUILD + 32; // + the TMA / MMA warp
constexpr int SC_XB = SC_M * SC_KC * 4;   // one X part of one buffer
enum : int { SCERR_WAIT = 23 };

struct ScArgs {
  const void* Q;                          // [n][H*G][Pmax][d]
  const void* K;                          // [n][H][Pmax][d]
  const void* V;
  const int32_t* plen;                    // [n]
  float* prio;                            // [n][H][Pmax]
  const float* b1;                        // [H][F]  (cache copies, hidden padded to F)
  const float* w2;                        // [H][F]
  const float* b2;                        // [H]
  const float* log_gamma;                 // [H] or nullptr
  int H, G, d, D, Pmax, act;
  int32_t* err;
};

__device__ __forceinline__ float tf32_head(float x) {
  uint32_t t;
  asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(t) : "f"(x));
  return __uint_as_float(t);
}
__device__ __forceinline__ void mma_tf32(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc,
                                         uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a), "l"(b), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void tma_2d(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}
// barrier 1 among the builder threads; returns the AND of `v` over all of them
__device__ __forceinline__ bool builders_and(bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred pi, po;\n\tsetp.ne.u32 pi, %1, 0;\n\t"
      "barrier.cta.red.and.pred po, 1, %2, pi;\n\tselp.u32 %0, 1, 0, po;\n\t}"
      : "=r"(r)
      : "r"((uint32_t)v), "n"(SC_BUILD)
      : "memory");
  return r != 0;
}

// Input dims [dim, dim + 32) of x_u = [k; v; qbar] handled at step c: the steps run
// qbar, k, v chunks in turn so that the k / v loads of a step are issued during the one before.
__host__ __device__ inline int chunk_dim(int c, int d) {
  const int i = c / 3, r = c - 3 * i;
  return (r == 0 ? 2 * d : r == 1 ? 0 : d) + i * SC_KC;
}

struct ScOff {
  int w, qm, b1, w2, red, bar, tmem, total;
};
__host__ __device__ inline ScOff sc_offsets(int F, int D) {
  ScOff o;
  o.w = 4 * SC_XB;                                       // after [2 buffers][hi, lo] X
  o.qm = o.w + 4 * F * SC_KC * 4;                        // after [2 buffers][hi, lo] W
  o.b1 = o.qm + ((SC_M - 1 + D) * SC_KC * 4 + 15) / 16 * 16;
  o.w2 = o.b1 + F * 4;
  o.red = o.w2 + F * 4;
  o.bar = o.red + 2 * SC_M * 4;
  o.tmem = o.bar + 8 * 8;
  o.total = o.tmem + 16;
  return o;
}

template <typename T, int F, int G>
__global__ void __launch_bounds__(SC_THREADS, 1)
    score_tf32_kernel(const __grid_constant__ CUtensorMap mhi, const __grid_constant__ CUtensorMap mlo,
                      ScArgs a) {
  extern __shared__ __align__(1024) unsigned char smf[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int lp = blockIdx.y, H = a.H, bl = lp / H, h = lp - bl * H;
  const int d = a.d, D = a.D;
  const int P = a.plen[bl];
  const int n_elig = max(P - D, 0);
  const int u0 = blockIdx.x * SC_M;
  if (u0 >= n_elig) return;
  const int nrow = min(SC_M, n_elig - u0);
  const int nch = 3 * d / SC_KC;
  const size_t Pm = a.Pmax;
  const ScOff off = sc_offsets(F, D);
  const uint32_t sb = smem_u32(smf);
  auto bar = [&](int i) { return sb + off.bar + 8u * (uint32_t)i; };   // 0,1 xfull  2,3 wfull  4,5 done
  float* b1s = reinterpret_cast<float*>(smf + off.b1);
  float* w2s = reinterpret_cast<float*>(smf + off.w2);
  float* red = reinterpret_cast<float*>(smf + off.red);
  float* qm = reinterpret_cast<float*>(smf + off.qm);
  if (tid == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(bar(i), SC_BUILD);
      mbar_init(bar(2 + i), 1);
      mbar_init(bar(4 + i), 1);
    }
    mbar_fence_init();
  }
  for (int f = tid; f < F; f += SC_THREADS) {
    b1s[f] = a.b1[(size_t)h * F + f];
    w2s[f] = a.w2[(size_t)h * F + f];
  }
  if (warp == SC_BUILD / 32) tmem_alloc(sb + off.tmem, F);
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(smf + off.tmem);
  const T* Kp = static_cast<const T*>(a.K) + ((size_t)bl * H + h) * Pm * d;
  const T* Vp = static_cast<const T*>(a.V) + ((size_t)bl * H + h) * Pm * d;
  const T* Qp = static_cast<const T*>(a.Q) + ((size_t)bl * H * G + (size_t)h * G) * Pm * d;

  if (warp == SC_BUILD / 32) {
    // ------------------------------------------------------------------ TMA + MMA issue
    if (lane == 0) {
      constexpr uint32_t WB = F * SC_KC * 4;
      auto tma_w = [&](int c, int b) {
        mbar_arrive_expect_tx(bar(2 + b), 2 * WB);
        tma_2d(sb + off.w + (2 * b + 0) * WB, &mhi, chunk_dim(c, d), h * F, bar(2 + b));
        tma_2d(sb + off.w + (2 * b + 1) * WB, &mlo, chunk_dim(c, d), h * F, bar(2 + b));
      };
      int wpend[2] = {0, -1}, last = -1;     // W chunk in flight per buffer; last committed chunk
      tma_w(0, 0);
      if (nch > 1) { tma_w(1, 1); wpend[1] = 1; }
      const uint32_t idesc = (1u << 4) | (2u << 7) | (2u << 10) | ((uint32_t)(F >> 3) << 17) |
                             ((uint32_t)(SC_M >> 4) << 24);
      bool ok = true;
      for (int c = 0; c < nch && ok; ++c) {
        const int b = c & 1;
        if (!(ok = mbar_wait(bar(2 + b), (c >> 1) & 1, a.err, SCERR_WAIT))) break;
        wpend[b] = -1;
        if (!(ok = mbar_wait(bar(b), (c >> 1) & 1, a.err, SCERR_WAIT))) break;
        fence_async_smem();
        fence_after();
        const uint32_t xb = sb + 2 * b * SC_XB, wb = sb + off.w + 2 * b * WB;
        // products hi*hi, hi*lo, lo*hi; bf16 k and v are exact in tf32, so their lo is 0
        const bool x_exact = sizeof(T) == 2 && chunk_dim(c, d) < 2 * d;
#pragma unroll
        for (int p = 0; p < 3; ++p) {
          if (p == 2 && x_exact) continue;
          const uint32_t xa = xb + (p == 2 ? SC_XB : 0), wa = wb + (p == 1 ? WB : 0);
#pragma unroll
          for (int ks = 0; ks < SC_KC / 8; ++ks)
            mma_tf32(tmem, kmajor_desc(xa, SC_M, ks), kmajor_desc(wa, F, ks), idesc,
                     (c > 0 || p > 0 || ks > 0) ? 1u : 0u);
        }
        commit(bar(4 + b));
        last = c;
        // W chunk c+1 goes into the buffer chunk c-1 used, once its MMAs are done
        if (c >= 1 && c + 1 < nch) {
          if (!(ok = mbar_wait(bar(4 + (b ^ 1)), ((c - 1) >> 1) & 1, a.err, SCERR_WAIT))) break;
          tma_w(c + 1, b ^ 1);
          wpend[b ^ 1] = c + 1;
        }
      }
      if (!ok) {
        // drain what is still in flight (bounded) before the CTA releases its memory
        for (int b = 0; b < 2; ++b)
          if (wpend[b] >= 0) mbar_wait(bar(2 + b), (wpend[b] >> 1) & 1, nullptr, 0);
        if (last >= 0) mbar_wait(bar(4 + (last & 1)), (last >> 1) & 1, nullptr, 0);
      }
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------------ builders
    using Raw = typename std::conditional<sizeof(T) == 4, float4, uint2>::type;   // 4 inputs
    auto to4 = [](const Raw& u) -> float4 {
      if constexpr (sizeof(T) == 4) {
        return u;
      } else {
        const bf16* e = reinterpret_cast<const bf16*>(&u);
        return make_float4(to_f(e[0]), to_f(e[1]), to_f(e[2]), to_f(e[3]));
      }
    };
    auto ld = [](const T* p) -> Raw { return *reinterpret_cast<const Raw*>(p); };
    auto split_store = [&](uint32_t buf, int r, int g4, float4 v) {
      const float4 hi = make_float4(tf32_head(v.x), tf32_head(v.y), tf32_head(v.z), tf32_head(v.w));
      const float4 lo = make_float4(v.x - hi.x, v.y - hi.y, v.z - hi.z, v.w - hi.w);
      *reinterpret_cast<float4*>(smf + buf + tile_off(r, g4, SC_M)) = hi;
      *reinterpret_cast<float4*>(smf + buf + SC_XB + tile_off(r, g4, SC_M)) = lo;
    };
    constexpr int KVI = SC_M * (SC_KC / 4) / SC_BUILD;      // K/V items per thread per chunk
    // raw K/V inputs of step c (k or v rows of the 128 tokens, 32 dims), zero past nrow
    auto load_kv = [&](int c, Raw (&v)[KVI]) {
      const int dim0 = chunk_dim(c, d);
      const T* src = dim0 < d ? Kp + dim0 : Vp + (dim0 - d);
#pragma unroll
      for (int j = 0; j < KVI; ++j) {
        const int it = tid + j * SC_BUILD, r = it >> 3, g4 = it & 7;
        v[j] = r < nrow ? ld(src + (size_t)(u0 + r) * d + g4 * 4) : Raw{};
      }
    };
    Raw cur[KVI], nxt[KVI];
    bool ok = true;
    for (int c = 0; c < nch; ++c) {
      const int b = c & 1;
      const bool q_step = chunk_dim(c, d) >= 2 * d;
      if (c + 1 < nch && chunk_dim(c + 1, d) < 2 * d) load_kv(c + 1, nxt);   // prefetch
      if (c >= 2) ok = mbar_wait(bar(4 + b), ((c - 2) >> 1) & 1, a.err, SCERR_WAIT);
      if (!builders_and(ok)) { ok = false; break; }
      const uint32_t buf = 2 * b * SC_XB;
      if (!q_step) {
        if (c == 0) load_kv(0, cur);
#pragma unroll
        for (int j = 0; j < KVI; ++j) {
          const int it = tid + j * SC_BUILD;
          if constexpr (sizeof(T) == 2)   // exact in tf32: the head alone (no lo product runs)
            *reinterpret_cast<float4*>(smf + buf + tile_off(it >> 3, it & 7, SC_M)) = to4(cur[j]);
          else
            split_store(buf, it >> 3, it & 7, to4(cur[j]));
        }
      } else {
        const int dim0 = chunk_dim(c, d) - 2 * d;
        const int npos = nrow - 1 + D;              // positions u0+1 .. u0+nrow-1+D
        constexpr int QB = 4;                       // items per thread per pass (G QB loads in flight)
        for (int base = tid; base < npos * (SC_KC / 4); base += QB * SC_BUILD) {
          Raw v[G][QB];
#pragma unroll
          for (int g = 0; g < G; ++g)
#pragma unroll
            for (int j = 0; j < QB; ++j) {
              const int it = base + j * SC_BUILD, tt = it >> 3, g4 = it & 7;
              v[g][j] = it < npos * (SC_KC / 4) ? ld(Qp + ((size_t)g * Pm + u0 + 1 + tt) * d + dim0 + g4 * 4)
                                                : Raw{};
            }
          const float ig = 1.0f / (float)G;
#pragma unroll
          for (int j = 0; j < QB; ++j) {
            float4 s4 = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
            for (int g = 0; g < G; ++g) {
              const float4 f = to4(v[g][j]);
              s4.x += f.x; s4.y += f.y; s4.z += f.z; s4.w += f.w;
            }
            const int it = base + j * SC_BUILD;
            if (it < npos * (SC_KC / 4))
              *reinterpret_cast<float4*>(qm + (it >> 3) * SC_KC + (it & 7) * 4) =
                  make_float4(s4.x * ig, s4.y * ig, s4.z * ig, s4.w * ig);
          }
        }
        asm volatile("bar.sync 1, %0;" ::"n"(SC_BUILD) : "memory");
        for (int it = tid; it < SC_M * (SC_KC / 4); it += SC_BUILD) {
          const int r = it >> 3, g4 = it & 7;
          float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
          if (r < nrow) {
            for (int j = 0; j < D; ++j) {
              const float4 v = *reinterpret_cast<const float4*>(qm + (r + j) * SC_KC + g4 * 4);
              s.x += v.x; s.y += v.y; s.z += v.z; s.w += v.w;
            }
            const float fd = (float)D;
            s = make_float4(s.x / fd, s.y / fd, s.z / fd, s.w / fd);
          }
          split_store(buf, r, g4, s);
        }
        asm volatile("bar.sync 1, %0;" ::"n"(SC_BUILD) : "memory");   // staging reused next chunk
      }
#pragma unroll
      for (int j = 0; j < KVI; ++j) cur[j] = nxt[j];
      fence_async_smem();
      mbar_arrive(bar(b));
    }
    // ------------------------------------------------------------------ epilogue
    if (ok) ok = mbar_wait(bar(4 + ((nch - 1) & 1)), ((nch - 1) >> 1) & 1, a.err, SCERR_WAIT);
    ok = __all_sync(0xffffffffu, ok);
    const int r = (warp & 3) * 32 + lane, half = warp >> 2;
    float part = 0.f;
    if (ok) {
      fence_after();
      const uint32_t trow = tmem + ((uint32_t)((warp & 3) * 32) << 16) + half * (F / 2);
#pragma unroll 1
      for (int c0 = 0; c0 < F / 2; c0 += 32) {
        float v[32];
        tmem_ld32(trow + c0, v);
        tmem_wait_ld();
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const int f = half * (F / 2) + c0 + i;
          part = fmaf(w2s[f], scorer_act(v[i] + b1s[f], a.act), part);
        }
      }
    }
    red[half * SC_M + r] = part;
    asm volatile("bar.sync 1, %0;" ::"n"(SC_BUILD) : "memory");
    if (ok && half == 0 && r < nrow) {
      const float sum = red[r] + red[SC_M + r];
      const int u = u0 + r;
      a.prio[(size_t)lp * Pm + u] =
          static_priority(canon_score(sum + a.b2[h]), u, a.log_gamma, h);
    }
  }
  fence_before();
  __syncthreads();
  if (warp == SC_BUILD / 32) tmem_dealloc(tmem, F);
}

__global__ void split_w1_kernel(const float* W1, float* hi, float* lo, int H, int in_dim, int F,
                                int Fp) {
  const size_t n = (size_t)H * F * in_dim;
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x) {
    const int k = (int)(i % in_dim);
    const size_t hf = i / in_dim;
    const int f = (int)(hf % F), h = (int)(hf / F);
    const float w = W1[((size_t)h * in_dim + k) * Fp + f];
    const float t = tf32_head(w);
    hi[i] = t;
    lo[i] = w - t;
  }
}

typedef CUresult (*EncodeTiledFn2)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                   const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                   const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

template <typename T, int F, int G>
cudaError_t launch_g(const CUtensorMap* maps, const ScArgs& a, int n_pairs, cudaStream_t stream) {
  const ScOff off = sc_offsets(F, a.D);
  auto k = score_tf32_kernel<T, F, G>;
  cudaError_t e = raise_smem_limit(k, off.total);
  if (e != cudaSuccess) return e;
  dim3 grid((a.Pmax + SC_M - 1) / SC_M, n_pairs);
  k<<<grid, SC_THREADS, off.total, stream>>>(maps[0], maps[1], a);
  return cudaGetLastError();
}
template <typename T, int F>
cudaError_t launch_f(const CUtensorMap* maps, const ScArgs& a, int n_pairs, cudaStream_t stream) {
  if (a.G == 4) return launch_g<T, F, 4>(maps, a, n_pairs, stream);
  if (a.G == 2) return launch_g<T, F, 2>(maps, a, n_pairs, stream);
  return launch_g<T, F, 1>(maps, a, n_pairs, stream);
}

}  // namespace

bool score_tf32_ok(const Dims& dm) {
  if (dm.F != dm.Fp || !(dm.F == 128 || dm.F == 256) || dm.d % SC_KC != 0 ||
      !(dm.G == 1 || dm.G == 2 || dm.G == 4))
    return false;
  return sc_offsets(dm.F, dm.D).total <= 227 * 1024;
}

size_t score_tf32_maps_size() { return 2 * sizeof(CUtensorMap); }

cudaError_t prepare_score_tf32(const Dims& dm, const float* W1, float* w1t, void* maps_out,
                               cudaStream_t stream) {
  const int in_dim = 3 * dm.d, F = dm.F;
  const size_t n = (size_t)dm.H * F * in_dim;
  float* hi = w1t;
  float* lo = w1t + n;
  split_w1_kernel<<<(unsigned)((n + 255) / 256 < 4096 ? (n + 255) / 256 : 4096), 256, 0, stream>>>(
      W1, hi, lo, dm.H, in_dim, F, dm.Fp);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  void* fn = nullptr;
  cudaDriverEntryPointQueryResult q;
  e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
  if (e != cudaSuccess) return e;
  if (q != cudaDriverEntryPointSuccess || fn == nullptr) return cudaErrorNotSupported;
  auto enc = reinterpret_cast<EncodeTiledFn2>(fn);
  CUtensorMap* maps = static_cast<CUtensorMap*>(maps_out);
  cuuint64_t dims[2] = {(cuuint64_t)in_dim, (cuuint64_t)dm.H * F};
  cuuint64_t strides[1] = {(cuuint64_t)in_dim * 4};
  cuuint32_t box[2] = {(cuuint32_t)SC_KC, (cuuint32_t)F};
  cuuint32_t estr[2] = {1, 1};
  for (int i = 0; i < 2; ++i) {
    CUresult r = enc(&maps[i], CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, i == 0 ? hi : lo, dims, strides, box,
                     estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
  }
  return cudaSuccess;
}

cudaError_t launch_score_tf32(const State& st, const Dims& dm, const void* maps, const void* Q,
                              const void* K, const void* V, const int32_t* plen, int n_seq, int Pmax,
                              float* prio, cudaStream_t stream) {
  if (n_seq <= 0 || Pmax <= 0) return cudaSuccess;
  ScArgs a{Q, K, V, plen, prio, st.b1, st.w2, st.b2, st.log_gamma, dm.H, dm.G, dm.d, dm.D, Pmax,
           dm.act, st.err};
  const CUtensorMap* m = static_cast<const CUtensorMap*>(maps);
  const int n_pairs = n_seq * dm.H;
  if (dm.dtype == KVPOP_F32)
    return dm.F == 256 ? launch_f<float, 256>(m, a, n_pairs, stream) : launch_f<float, 128>(m, a, n_pairs, stream);
  return dm.F == 256 ? launch_f<bf16, 256>(m, a, n_pairs, stream) : launch_f<bf16, 128>(m, a, n_pairs, stream);
}

}  // namespace kvpop
