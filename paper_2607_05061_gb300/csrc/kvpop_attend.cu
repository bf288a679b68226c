// Decode step 5: GQA attention over the compact cache (kept slots + window).
//
// During decoding the cache holds only retained entries, so attention runs
// directly over them (App. C, first paragraph): for each query head g of KV
// head h, o_g = softmax(q_g K_S^T / sqrt(d)) V_S with S = slots U window.
//
// Design (one GB300, HBM-bound: every K/V byte is read once per step):
//  * Persistent grid.  The key stream of every (sequence, KV head) pair is cut
//    into tiles of TILE keys; the concatenated tile list is split evenly over
//    the CTAs (token-balanced split-K), so ragged pairs cost what they hold.
//  * One producer lane streams K and V tiles with 1-D TMA bulk copies
//    (cp.async.bulk, 16-byte granules) into a STAGES-deep shared-memory ring
//    guarded by full/empty mbarriers.
//  * NWC consumer warps.  A warp takes 4 keys at a time, 8 lanes per key, each
//    lane owning E contiguous-by-16-bytes elements of the row, with all G query
//    heads of the KV head in registers, so a K/V byte feeds G heads.  Dot
//    products reduce over the 8 lanes with xor shuffles; the online softmax
//    keeps a warp-wide running maximum that is only raised when a logit exceeds
//    it by 2^THR (exact after the final normalisation).
//  * A pair split over several CTAs leaves (m, l, o) partials in a workspace;
//    the last contributor (atomic counter, no waiting) merges them in CTA order.
//  * Every mbarrier wait is bounded in wall time; on expiry the kernel records
//    an error code and skips the remaining work without leaving a barrier.
#include <type_traits>

#include "kvpop_internal.cuh"

namespace kvpop {
namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kThr = 8.0f;           // lazy-rescale threshold (log2 units)

template <typename T, int HD, int G>
struct Traits {
  static constexpr int ESZ = (int)sizeof(T);
  static constexpr int R = HD * ESZ;             // bytes per K (or V) row
  static constexpr int CPL = R / 128;            // 16-byte chunks per lane (8 lanes / key)
  static constexpr int EPC = 16 / ESZ;           // elements per chunk
  static constexpr int E = CPL * EPC;            // elements per lane
  static constexpr int TILE = 16384 / R;         // keys per tile: 16 KB of K + 16 KB of V
  static constexpr int STAGES = 5;
  static constexpr int NWC = 8;                  // consumer warps
  static constexpr int THREADS = (NWC + 1) * 32;
  static constexpr int STAGE_BYTES = 2 * TILE * R;
  static constexpr int PSTRIDE = G * HD + 2 * G; // floats per partial
  // shared-memory carve-up (bytes)
  static constexpr int al16(int x) { return (x + 15) & ~15; }
  static constexpr int OFF_BAR = STAGES * STAGE_BYTES;
  static constexpr int OFF_META = al16(OFF_BAR + 2 * STAGES * 8);
  static constexpr int OFF_MO = al16(OFF_META + STAGES * 8);
  static constexpr int OFF_ML = OFF_MO + NWC * G * HD * 4;
  static constexpr int OFF_MM = OFF_ML + NWC * G * 4;
  static constexpr int OFF_FLAG = OFF_MM + NWC * G * 4;
  static constexpr int OFF_SCAN = OFF_FLAG + 16;
  static constexpr int OFF_PREFIX = OFF_SCAN + 16 * 4;
  static_assert(R % 128 == 0, "row must split into 8 lanes of 16-byte chunks");
  static_assert(OFF_PREFIX % 16 == 0, "alignment");
};

struct AttendArgs {
  const unsigned char* slotK;
  const unsigned char* slotV;
  const unsigned char* ringK;
  const unsigned char* ringV;
  const int32_t* nvalid;
  const int32_t* len;
  const void* q;
  float* out;
  float* part;
  int32_t* part_count;
  int32_t* err;
  int pairs, B, D;
  float qscale;                // log2(e) / sqrt(d)
};

// ------------------------------------------------------------------ PTX helpers
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.release.cta.shared::cta.b64 _, [%0], %1;" ::"r"(bar),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.release.cta.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cta.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ unsigned long long globaltimer() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
// Bounded wait: false (and an error code recorded) after kWaitLimitNs.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, int32_t* err, int code) {
  if (mbar_try_wait(bar, parity)) return true;
  const unsigned long long t0 = globaltimer();
  for (unsigned it = 1;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 63u) == 0u && globaltimer() - t0 > kWaitLimitNs) {
      atomicCAS(err, 0, code);
      return false;
    }
  }
}
__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes,
                                         uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cta.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          dst),
      "l"(src), "r"(bytes), "r"(bar)
      : "memory");
}
__device__ __forceinline__ void consumer_sync(int nthreads) {
  asm volatile("bar.sync 1, %0;" ::"r"(nthreads) : "memory");
}
__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// 16 bytes of row data -> EPC floats
__device__ __forceinline__ void unpack(const uint4& w, float (&f)[4]) {
  f[0] = __uint_as_float(w.x);
  f[1] = __uint_as_float(w.y);
  f[2] = __uint_as_float(w.z);
  f[3] = __uint_as_float(w.w);
}
__device__ __forceinline__ void unpack(const uint4& w, float (&f)[8]) {
  f[0] = __uint_as_float(w.x << 16); f[1] = __uint_as_float(w.x & 0xffff0000u);
  f[2] = __uint_as_float(w.y << 16); f[3] = __uint_as_float(w.y & 0xffff0000u);
  f[4] = __uint_as_float(w.z << 16); f[5] = __uint_as_float(w.z & 0xffff0000u);
  f[6] = __uint_as_float(w.w << 16); f[7] = __uint_as_float(w.w & 0xffff0000u);
}

__device__ __forceinline__ int tiles_of(int nv, int np, int tile) {
  return (nv + tile - 1) / tile + (np + tile - 1) / tile;
}

// CTA whose tile range [c*T/N, (c+1)*T/N) contains tile t (N <= T).
__device__ __forceinline__ int cta_of(long long t, long long T, long long N) {
  return (int)(((t + 1) * N - 1) / T);
}
__device__ __forceinline__ long long cta_begin(long long c, long long T, long long N) {
  return c * T / N;
}

template <typename T, int HD, int G>
__global__ void __launch_bounds__(Traits<T, HD, G>::THREADS, 1) attend_kernel(AttendArgs a) {
  using Tr = Traits<T, HD, G>;
  constexpr int TILE = Tr::TILE, R = Tr::R, CPL = Tr::CPL, EPC = Tr::EPC, E = Tr::E;
  constexpr int STAGES = Tr::STAGES, NWC = Tr::NWC, NT = Tr::THREADS;

  extern __shared__ __align__(128) unsigned char smem[];
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + Tr::OFF_BAR);   // full[S], empty[S]
  int2* meta = reinterpret_cast<int2*>(smem + Tr::OFF_META);
  float* mo = reinterpret_cast<float*>(smem + Tr::OFF_MO);            // [NWC][G][HD]
  float* ml = reinterpret_cast<float*>(smem + Tr::OFF_ML);            // [NWC][G]
  float* mm = reinterpret_cast<float*>(smem + Tr::OFF_MM);            // [NWC][G]
  int* flag = reinterpret_cast<int*>(smem + Tr::OFF_FLAG);
  int* scan = reinterpret_cast<int*>(smem + Tr::OFF_SCAN);
  int* prefix = reinterpret_cast<int*>(smem + Tr::OFF_PREFIX);        // [pairs + 1]

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int npairs = a.pairs;

  // ---- prologue: tile counts of every pair, exclusive prefix over pairs ------------
  {
    const int per = (npairs + NT - 1) / NT;
    const int beg = min(tid * per, npairs), end = min(beg + per, npairs);
    int local = 0;
    for (int i = beg; i < end; ++i)
      local += tiles_of(used_slots(a.nvalid[i], a.B, a.err), window_rows(a.len[i], a.D, a.err), TILE);
    int incl = local;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      int y = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += y;
    }
    if (lane == 31) scan[warp] = incl;
    if (tid == 0) {
      for (int s = 0; s < STAGES; ++s) {
        mbar_init(smem_u32(&bars[s]), 1);
        mbar_init(smem_u32(&bars[STAGES + s]), NWC);
      }
      asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
      flag[0] = 0;   // abort
      flag[1] = 0;   // last-contributor broadcast
    }
    __syncthreads();
    if (tid == 0) {
      int run = 0;
      for (int w = 0; w < NT / 32; ++w) { int x = scan[w]; scan[w] = run; run += x; }
      prefix[npairs] = run;
    }
    __syncthreads();
    int run = scan[warp] + incl - local;
    for (int i = beg; i < end; ++i) {
      prefix[i] = run;
      run += tiles_of(used_slots(a.nvalid[i], a.B, nullptr), window_rows(a.len[i], a.D, nullptr), TILE);
    }
    __syncthreads();
  }
  const long long Ttot = prefix[npairs];
  if (Ttot <= 0) return;
  const long long NC = min((long long)gridDim.x, Ttot);
  // pairs without keys (never ingested) get a zero output
  for (int p = blockIdx.x; p < npairs; p += gridDim.x)
    if (prefix[p + 1] == prefix[p])
      for (int i = tid; i < G * HD; i += NT) a.out[(size_t)p * G * HD + i] = 0.f;
  if (blockIdx.x >= NC) return;
  const long long t0 = cta_begin(blockIdx.x, Ttot, NC);
  const long long t1 = cta_begin(blockIdx.x + 1, Ttot, NC);
  int p0;
  {
    int lo = 0, hi = npairs - 1;
    while (lo < hi) {
      int mid = (lo + hi + 1) >> 1;
      if (prefix[mid] <= t0) lo = mid; else hi = mid - 1;
    }
    p0 = lo;
  }

  // ---- producer: one lane streams K/V tiles into the stage ring --------------------
  if (warp == NWC) {
    if (lane == 0) {
      int p = p0;
      long long i = 0;
      for (long long t = t0; t < t1; ++t, ++i) {
        while (t >= prefix[p + 1]) ++p;
        const int lt = (int)(t - prefix[p]);
        const int nv = used_slots(a.nvalid[p], a.B, nullptr);
        const int nvt = (nv + TILE - 1) / TILE;
        const unsigned char *sk, *sv;
        int cnt;
        if (lt < nvt) {
          const int k0 = lt * TILE;
          cnt = min(TILE, nv - k0);
          sk = a.slotK + ((size_t)p * a.B + k0) * R;
          sv = a.slotV + ((size_t)p * a.B + k0) * R;
        } else {
          const int k0 = (lt - nvt) * TILE;
          cnt = min(TILE, window_rows(a.len[p], a.D, nullptr) - k0);
          sk = a.ringK + ((size_t)p * a.D + k0) * R;
          sv = a.ringV + ((size_t)p * a.D + k0) * R;
        }
        const int s = (int)(i % STAGES);
        if (i >= STAGES) {
          if (!mbar_wait(smem_u32(&bars[STAGES + s]), (uint32_t)((i / STAGES - 1) & 1), a.err,
                         DEVERR_TIMEOUT_EMPTY)) {
            break;
          }
        }
        meta[s] = make_int2(p, cnt);
        const uint32_t fb = smem_u32(&bars[s]);
        mbar_arrive_expect_tx(fb, 2u * cnt * R);
        unsigned char* dst = smem + (size_t)s * Tr::STAGE_BYTES;
        bulk_g2s(smem_u32(dst), sk, cnt * R, fb);
        bulk_g2s(smem_u32(dst + TILE * R), sv, cnt * R, fb);
      }
      // drain: every copy this lane issued has landed before the CTA may exit
      const long long issued = i;
      for (long long k = issued > STAGES ? issued - STAGES : 0; k < issued; ++k) {
        const int s = (int)(k % STAGES);
        if (!mbar_wait(smem_u32(&bars[s]), (uint32_t)((k / STAGES) & 1), a.err,
                       DEVERR_TIMEOUT_DRAIN))
          break;
      }
    }
    return;
  }

  // ---- consumers -------------------------------------------------------------------
  const int grp = lane >> 3, j = lane & 7;
  float qf[G][E], o[G][E], l[G], m[G];
  bool ok = true;
  int cur = -1;

  auto load_q = [&](int p) {
    const unsigned char* qb = static_cast<const unsigned char*>(a.q) + (size_t)p * G * R;
#pragma unroll
    for (int g = 0; g < G; ++g) {
#pragma unroll
      for (int c = 0; c < CPL; ++c) {
        const uint4 w = __ldg(reinterpret_cast<const uint4*>(qb + (size_t)g * R + (j + 8 * c) * 16));
        float f[EPC];
        unpack(w, f);
#pragma unroll
        for (int e = 0; e < EPC; ++e) qf[g][c * EPC + e] = f[e] * a.qscale;
      }
      l[g] = 0.f;
      m[g] = -INFINITY;
#pragma unroll
      for (int e = 0; e < E; ++e) o[g][e] = 0.f;
    }
  };

  auto finalize = [&](int p) {
    // fold the 4 key groups of this warp (same d-slice, different keys)
#pragma unroll
    for (int g = 0; g < G; ++g) {
      l[g] += __shfl_xor_sync(0xffffffffu, l[g], 8);
      l[g] += __shfl_xor_sync(0xffffffffu, l[g], 16);
#pragma unroll
      for (int e = 0; e < E; ++e) {
        o[g][e] += __shfl_xor_sync(0xffffffffu, o[g][e], 8);
        o[g][e] += __shfl_xor_sync(0xffffffffu, o[g][e], 16);
      }
    }
    if (grp == 0) {
#pragma unroll
      for (int g = 0; g < G; ++g) {
#pragma unroll
        for (int c = 0; c < CPL; ++c)
#pragma unroll
          for (int e = 0; e < EPC; ++e)
            mo[(warp * G + g) * HD + (j + 8 * c) * EPC + e] = o[g][c * EPC + e];
        if (j == 0) { ml[warp * G + g] = l[g]; mm[warp * G + g] = m[g]; }
      }
    }
    consumer_sync(NWC * 32);
    const long long ca = cta_of(prefix[p], Ttot, NC);
    const long long cb = cta_of(prefix[p + 1] - 1, Ttot, NC);
    const bool complete = (ca == cb);
    float* mypart = nullptr;
    if (!complete) {
      const int slot = (prefix[p] < t0) ? 0 : 1;
      mypart = a.part + ((size_t)blockIdx.x * 2 + slot) * Tr::PSTRIDE;
    }
    for (int idx = tid; idx < G * HD; idx += NWC * 32) {
      const int g = idx / HD, i = idx - g * HD;
      float ms = -INFINITY;
#pragma unroll
      for (int w = 0; w < NWC; ++w) ms = fmaxf(ms, mm[w * G + g]);
      float L = 0.f, O = 0.f;
#pragma unroll
      for (int w = 0; w < NWC; ++w) {
        const float mw = mm[w * G + g];
        const float f = (mw == -INFINITY) ? 0.f : fast_exp2(mw - ms);
        L = fmaf(ml[w * G + g], f, L);
        O = fmaf(mo[(w * G + g) * HD + i], f, O);
      }
      if (complete) {
        a.out[((size_t)p * G + g) * HD + i] = O / L;
      } else {
        mypart[g * HD + i] = O;
        if (i == 0) { mypart[G * HD + g] = ms; mypart[G * HD + G + g] = L; }
      }
    }
    if (!complete) {
      __threadfence();
      consumer_sync(NWC * 32);
      if (tid == 0) {
        const int old = atomicAdd(&a.part_count[p], 1);
        const int last = (old == (int)(cb - ca));
        if (last) a.part_count[p] = 0;
        flag[1] = last;
      }
      consumer_sync(NWC * 32);
      if (flag[1]) {
        __threadfence();
        for (int idx = tid; idx < G * HD; idx += NWC * 32) {
          const int g = idx / HD, i = idx - g * HD;
          float ms = -INFINITY;
          for (long long c = ca; c <= cb; ++c) {
            const int slot = (prefix[p] < cta_begin(c, Ttot, NC)) ? 0 : 1;
            const float* pc = a.part + ((size_t)c * 2 + slot) * Tr::PSTRIDE;
            ms = fmaxf(ms, __ldcg(pc + G * HD + g));
          }
          float L = 0.f, O = 0.f;
          for (long long c = ca; c <= cb; ++c) {
            const int slot = (prefix[p] < cta_begin(c, Ttot, NC)) ? 0 : 1;
            const float* pc = a.part + ((size_t)c * 2 + slot) * Tr::PSTRIDE;
            const float mc = __ldcg(pc + G * HD + g);
            const float f = (mc == -INFINITY) ? 0.f : fast_exp2(mc - ms);
            L = fmaf(__ldcg(pc + G * HD + G + g), f, L);
            O = fmaf(__ldcg(pc + g * HD + i), f, O);
          }
          a.out[((size_t)p * G + g) * HD + i] = O / L;
        }
      }
    }
    consumer_sync(NWC * 32);
  };

  {
    int p = p0;
    long long i = 0;
    for (long long t = t0; t < t1; ++t, ++i) {
      while (t >= prefix[p + 1]) ++p;          // control flow from the schedule only
      if (p != cur) {
        if (cur >= 0) finalize(cur);
        cur = p;
        load_q(p);
      }
      const int s = (int)(i % STAGES);
      if (ok) ok = mbar_wait(smem_u32(&bars[s]), (uint32_t)((i / STAGES) & 1), a.err,
                             DEVERR_TIMEOUT_FULL);
      if (ok) {
        const int cnt = meta[s].y;
        const unsigned char* Ks = smem + (size_t)s * Tr::STAGE_BYTES;
        const unsigned char* Vs = Ks + TILE * R;
        for (int kb = warp * 4; kb < cnt; kb += NWC * 4) {
          const int key = kb + grp;
          const bool valid = key < cnt;
          const int kr = valid ? key : kb;     // a real row; its weight is forced to 0
          float acc0[G], acc1[G];
#pragma unroll
          for (int g = 0; g < G; ++g) { acc0[g] = 0.f; acc1[g] = 0.f; }
#pragma unroll
          for (int c = 0; c < CPL; ++c) {
            const uint4 w = *reinterpret_cast<const uint4*>(Ks + (size_t)kr * R + (j + 8 * c) * 16);
            float f[EPC];
            unpack(w, f);
#pragma unroll
            for (int g = 0; g < G; ++g)
#pragma unroll
              for (int e = 0; e < EPC; e += 2) {
                acc0[g] = fmaf(qf[g][c * EPC + e], f[e], acc0[g]);
                acc1[g] = fmaf(qf[g][c * EPC + e + 1], f[e + 1], acc1[g]);
              }
          }
          float sc[G];
#pragma unroll
          for (int g = 0; g < G; ++g) {
            float x = acc0[g] + acc1[g];
            x += __shfl_xor_sync(0xffffffffu, x, 1);
            x += __shfl_xor_sync(0xffffffffu, x, 2);
            x += __shfl_xor_sync(0xffffffffu, x, 4);
            sc[g] = x;
          }
          bool need = false;
#pragma unroll
          for (int g = 0; g < G; ++g) need |= valid && (sc[g] > m[g] + kThr);
          if (__any_sync(0xffffffffu, need)) {
#pragma unroll
            for (int g = 0; g < G; ++g) {
              float mx = valid ? sc[g] : -INFINITY;
              mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 8));
              mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
              const float mn = fmaxf(m[g], mx);
              const float f = fast_exp2(m[g] - mn);
              l[g] *= f;
#pragma unroll
              for (int e = 0; e < E; ++e) o[g][e] *= f;
              m[g] = mn;
            }
          }
          float pr[G];
#pragma unroll
          for (int g = 0; g < G; ++g) {
            pr[g] = valid ? fast_exp2(sc[g] - m[g]) : 0.f;
            l[g] += pr[g];
          }
#pragma unroll
          for (int c = 0; c < CPL; ++c) {
            const uint4 w = *reinterpret_cast<const uint4*>(Vs + (size_t)kr * R + (j + 8 * c) * 16);
            float f[EPC];
            unpack(w, f);
#pragma unroll
            for (int g = 0; g < G; ++g)
#pragma unroll
              for (int e = 0; e < EPC; ++e) o[g][c * EPC + e] = fmaf(pr[g], f[e], o[g][c * EPC + e]);
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&bars[STAGES + s]));
    }
    if (cur >= 0) finalize(cur);
  }
}

template <typename T, int HD, int G>
AttendConfig make_config() {
  using Tr = Traits<T, HD, G>;
  AttendConfig c;
  c.threads = Tr::THREADS;
  c.smem_fixed = Tr::OFF_PREFIX;
  c.tile = Tr::TILE;
  c.func = (const void*)attend_kernel<T, HD, G>;
  return c;
}

template <typename T, int HD, int G>
cudaError_t launch_t(const State& st, const Dims& dm, const void* q, float* out, int grid,
                     cudaStream_t stream) {
  using Tr = Traits<T, HD, G>;
  AttendArgs a;
  a.slotK = static_cast<const unsigned char*>(st.slotK);
  a.slotV = static_cast<const unsigned char*>(st.slotV);
  a.ringK = static_cast<const unsigned char*>(st.ringK);
  a.ringV = static_cast<const unsigned char*>(st.ringV);
  a.nvalid = st.nvalid;
  a.len = st.len;
  a.q = q;
  a.out = out;
  a.part = st.part;
  a.part_count = st.part_count;
  a.err = st.err;
  a.pairs = dm.pairs;
  a.B = dm.B;
  a.D = dm.D;
  a.qscale = kLog2e / sqrtf((float)HD);
  const size_t smem = Tr::OFF_PREFIX + (size_t)(dm.pairs + 1) * 4;
  attend_kernel<T, HD, G><<<grid, Tr::THREADS, smem, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t attend_config(const Dims& dm, AttendConfig* out) {
  const bool f = dm.dtype == KVPOP_F32;
#define CFG(T_, HD_, G_) \
  if ((f == std::is_same<T_, float>::value) && dm.d == HD_ && dm.G == G_) { *out = make_config<T_, HD_, G_>(); return cudaSuccess; }
  CFG(float, 64, 1) CFG(float, 64, 2) CFG(float, 64, 4)
  CFG(float, 128, 1) CFG(float, 128, 2) CFG(float, 128, 4)
  CFG(bf16, 64, 1) CFG(bf16, 64, 2) CFG(bf16, 64, 4)
  CFG(bf16, 128, 1) CFG(bf16, 128, 2) CFG(bf16, 128, 4)
#undef CFG
  return cudaErrorInvalidValue;
}

cudaError_t launch_attend(const State& st, const Dims& dm, const void* q, float* out, int grid,
                          cudaStream_t stream) {
  const bool f = dm.dtype == KVPOP_F32;
#define LAUNCH(T_, HD_, G_) \
  if ((f == std::is_same<T_, float>::value) && dm.d == HD_ && dm.G == G_) return launch_t<T_, HD_, G_>(st, dm, q, out, grid, stream);
  LAUNCH(float, 64, 1) LAUNCH(float, 64, 2) LAUNCH(float, 64, 4)
  LAUNCH(float, 128, 1) LAUNCH(float, 128, 2) LAUNCH(float, 128, 4)
  LAUNCH(bf16, 64, 1) LAUNCH(bf16, 64, 2) LAUNCH(bf16, 64, 4)
  LAUNCH(bf16, 128, 1) LAUNCH(bf16, 128, 2) LAUNCH(bf16, 128, 4)
#undef LAUNCH
  return cudaErrorInvalidValue;
}

}  // namespace kvpop
