// Decode step 5 for bf16 K/V: GQA attention over the compact cache on tensor
// cores (kept slots + window; App. C, first paragraph).
//
// Same persistent token-balanced split-K schedule as the CUDA-core kernel
// (kvpop_sched.cuh).  Per tile of TILE keys:
//  * K and V rows arrive by 2-D TMA tensor copies (one box per 64-column half
//    of a row) with the 128-byte swizzle, so every ldmatrix below reads eight
//    distinct bank groups.
//  * Each of the 8 consumer warps takes 16 keys of a 128-key tile (2 stages of
//    64 KB; a sweep of tile size, stage count and CTAs per SM on GB300 put this
//    shape at 0.98 of the measured copy bandwidth).  Logits S^T[16 keys x 8] =
//    K Q^T run as m16n8k16 bf16 MMAs over d (the G <= 4 query heads of the KV head padded to
//    the N = 8 of the instruction; Q^T fragments stay in registers for the
//    pair).  The fp32 accumulator is scaled by log2(e)/sqrt(d).
//  * Online softmax per head with a lazily raised running maximum (only when
//    a logit exceeds it by 2^THR; exact after the final normalisation).
//  * The probabilities are rounded to bf16 and transposed in registers
//    (movmatrix) into the B operand of O^T[d x 8] += V^T P^T, again m16n8k16
//    MMAs with V^T fragments loaded by ldmatrix.trans.  O^T stays in registers.
// Every mbarrier wait is bounded; on expiry the kernel records an error code
// and skips the remaining work while keeping every block barrier balanced.
#include <cuda.h>

#include <algorithm>
#include <cstring>

#include "kvpop_ptx.cuh"
#include "kvpop_sched.cuh"
#include "kvpop_step_fused.cuh"

namespace kvpop {
namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kThr = 8.0f;

// Pipeline shape (tuned on GB300 for the cr8x decode step).
#ifndef KVPOP_TC_NWC
#define KVPOP_TC_NWC 8
#endif
#ifndef KVPOP_TC_STAGES
#define KVPOP_TC_STAGES 2
#endif
#ifndef KVPOP_TC_MINBLOCKS
#define KVPOP_TC_MINBLOCKS 1
#endif
// Fused step: tiles (in 64ths) that a CTA with one scorer unit more than the rest gives up.
#ifndef KVPOP_FUSED_PREFETCH_TILES
#define KVPOP_FUSED_PREFETCH_TILES 4
#endif
#ifndef KVPOP_FUSED_SPLIT_K
#define KVPOP_FUSED_SPLIT_K 5
#endif

template <int HD, int G>
struct TcTraits {
  static constexpr int NH = HD / 64;               // 128-byte column halves per row
  static constexpr int NKS = HD / 16;              // k-steps of the QK contraction
  static constexpr int NMT = HD / 16;              // m-tiles of O^T
  static constexpr int NWC = KVPOP_TC_NWC;         // consumer warps, 16 keys each
  static constexpr int TILE = 16 * NWC;
  static constexpr int STAGES = KVPOP_TC_STAGES;
  static constexpr int THREADS = (NWC + 1) * 32;
  static constexpr int THREADS_F = (NWC + 1 + kFusedSW) * 32;   // with the scorer warps
  static constexpr int HALF_BYTES = TILE * 128;    // one box
  static constexpr int STAGE_BYTES = 2 * NH * HALF_BYTES;
  static constexpr int al16(int x) { return (x + 15) & ~15; }
  static constexpr int OFF_BAR = STAGES * STAGE_BYTES;
  static constexpr int OFF_MO = al16(OFF_BAR + 2 * STAGES * 8);
  static constexpr int OFF_ML = OFF_MO + NWC * G * HD * 4;
  static constexpr int OFF_MM = OFF_ML + NWC * G * 4;
  static constexpr int OFF_FLAG = al16(OFF_MM + NWC * G * 4);
  static constexpr int OFF_SCAN = OFF_FLAG + 16;
  static constexpr int OFF_PREFIX = OFF_SCAN + 16 * 4;
  static constexpr int SMEM_ALIGN = 1024;          // 128-byte swizzle atoms
};

struct TcArgs {
  const int32_t* nvalid;
  const int32_t* len;
  const bf16* q;
  float* out;
  float* part;
  int32_t* part_count;
  int32_t* err;
  int pairs, B, D;
  int ring_rows;               // rows of a window box: min(TILE, D rounded up to 8)
  float qscale;
  int skip_copies;             // testing hook: the producer issues nothing (see below)
};

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y,
                                            uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& a0, uint32_t& a1, uint32_t& a2,
                                        uint32_t& a3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(a0), "=r"(a1), "=r"(a2), "=r"(a3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& a0, uint32_t& a1, uint32_t& a2,
                                          uint32_t& a3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(a0), "=r"(a1), "=r"(a2), "=r"(a3)
               : "r"(addr));
}
__device__ __forceinline__ void mma_bf16(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7},"
      " {%8, %9}, {%0, %1, %2, %3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t movm_t(uint32_t x) {
  uint32_t y;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(y) : "r"(x));
  return y;
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ void consumer_sync() {
  asm volatile("bar.sync 1, %0;" ::"r"(KVPOP_TC_NWC * 32) : "memory");
}

// FUSED: the whole decode step (kvpop_step_fused.cuh): the consumers stream only the keys
// that cannot change this step, the scorer warps ingest the new token meanwhile, and each
// pair's last arrival merges.  Otherwise the attention alone, over the state the ingest left.
template <int HD, int G, bool FUSED>
__global__ void __launch_bounds__(FUSED ? TcTraits<HD, G>::THREADS_F : TcTraits<HD, G>::THREADS,
                                  KVPOP_TC_MINBLOCKS)
    attend_tc_kernel(const __grid_constant__ CUtensorMap mapSK, const __grid_constant__ CUtensorMap mapSV,
                     const __grid_constant__ CUtensorMap mapRK, const __grid_constant__ CUtensorMap mapRV,
                     TcArgs a, const __grid_constant__ FusedArgs f) {
  using Tr = TcTraits<HD, G>;
  constexpr int TILE = Tr::TILE, NH = Tr::NH, NKS = Tr::NKS, NMT = Tr::NMT;
  constexpr int STAGES = Tr::STAGES, NWC = Tr::NWC;
  constexpr int NT = FUSED ? Tr::THREADS_F : Tr::THREADS;

  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + Tr::SMEM_ALIGN - 1) & ~(uintptr_t)(Tr::SMEM_ALIGN - 1));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + Tr::OFF_BAR);
  float* mo = reinterpret_cast<float*>(smem + Tr::OFF_MO);
  float* ml = reinterpret_cast<float*>(smem + Tr::OFF_ML);
  float* mm = reinterpret_cast<float*>(smem + Tr::OFF_MM);
  int* flag = reinterpret_cast<int*>(smem + Tr::OFF_FLAG);
  int* scan = reinterpret_cast<int*>(smem + Tr::OFF_SCAN);
  int* prefix = reinterpret_cast<int*>(smem + Tr::OFF_PREFIX);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int npairs = a.pairs;
  if (tid == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(smem_u32(&bars[s]), 1);
      mbar_init(smem_u32(&bars[STAGES + s]), NWC);
    }
    mbar_fence_init();
  }
  if constexpr (FUSED) {
    // Where this CTA's range began last launch (the split stays the same from step to step
    // once the cache is full): its first tiles go to L2 now, while the previous step's
    // slowest CTAs still stream, so that this step starts on L2 hits.  A hint only: L2 is
    // coherent, and a stale record just prefetches something else within the slots.
    if (tid == 0 && f.start_prev != nullptr) {
      const int2 sp = __ldcg(f.start_prev + blockIdx.x);
      const bf16* sk = static_cast<const bf16*>(f.st.slotK);
      const bf16* sv = static_cast<const bf16*>(f.st.slotV);
      for (int k = 0; k < KVPOP_FUSED_PREFETCH_TILES; ++k) {
        const long long slot = (long long)(sp.y + k) * TILE;
        if (sp.x < 0 || sp.x >= npairs || sp.y < 0 || slot + TILE > a.B) break;
        const size_t row = (size_t)sp.x * a.B + (size_t)slot;
        prefetch_l2(sk + row * HD, (uint32_t)(TILE * HD * 2));
        prefetch_l2(sv + row * HD, (uint32_t)(TILE * HD * 2));
      }
    }
    // the next step's kernel may be scheduled now: it waits for this grid before reading
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  }
  // Launched as a programmatic dependent of the kernel before it (the ingest, or the
  // previous fused step): everything below reads the state it writes, so wait here for
  // it to complete (a no-op without a predecessor).
  asm volatile("griddepcontrol.wait;" ::: "memory");
  build_schedule<NT>(a.nvalid, a.len, npairs, a.B, a.D, TILE, prefix, scan, a.err);
  const long long Ttot = prefix[npairs];
  if constexpr (FUSED) {
    // lengths and used-slot counts read: their commits may start once every CTA of this
    // launch is here.  The count runs on over launches, and a launch's CTAs all start after
    // the previous launch has ended, so old / grid numbers this launch for each of its CTAs
    // and the count it must reach is the end of that epoch (kept in shared memory).
    if (tid == 0) {
      __threadfence();
      const unsigned long long old = atomicAdd(f.ctr, 1ull);
      unsigned long long* target = reinterpret_cast<unsigned long long*>(
          smem + Tr::al16(Tr::OFF_PREFIX + (npairs + 1) * 4) + FusedSmem::FLAG + 8);
      *target = (old / gridDim.x + 1) * gridDim.x;
    }
  } else {
    if (Ttot <= 0) return;
  }
  const long long NC = min((long long)gridDim.x, Ttot);
  if constexpr (!FUSED) {
    for (int p = blockIdx.x; p < npairs; p += gridDim.x)
      if (prefix[p + 1] == prefix[p])
        for (int i = tid; i < G * HD; i += NT) a.out[(size_t)p * G * HD + i] = 0.f;
    if (blockIdx.x >= NC) return;
  }
  // FUSED: a CTA without tiles (or a step without any) still runs its scorer units, and
  // the CTAs with one scorer unit more than the rest stream KVPOP_FUSED_SPLIT_K / 64 fewer
  // tiles (when every CTA has at least 4)
  int* bnd = reinterpret_cast<int*>(smem + Tr::al16(Tr::OFF_PREFIX + (npairs + 1) * 4) + FusedSmem::BND);
  int* sched_seen = reinterpret_cast<int*>(smem + Tr::al16(Tr::OFF_PREFIX + (npairs + 1) * 4) + FusedSmem::FLAG);
  Split sp{Ttot, NC, bnd};
  if constexpr (FUSED) {
    const int units = f.H * ((f.batch + kFusedSeqs - 1) / kFusedSeqs);
    const int extra = units % (int)gridDim.x;
    const bool weigh = Ttot >= 4 * NC && extra > 0;
    split_bounds(bnd, Ttot, NC, weigh ? (int)min((long long)extra, NC) : 0, weigh ? KVPOP_FUSED_SPLIT_K : 0,
                 tid, NT);
    if (tid == 0) *sched_seen = 0;
    __syncthreads();
  }
  const bool streams = Ttot > 0 && blockIdx.x < NC;
  const long long t0 = streams ? (FUSED ? sp.begin(blockIdx.x) : cta_begin(blockIdx.x, Ttot, NC)) : 0;
  const long long t1 = streams ? (FUSED ? sp.begin(blockIdx.x + 1) : cta_begin(blockIdx.x + 1, Ttot, NC)) : 0;
  int p0 = 0;
  if (streams) {
    int lo = 0, hi = npairs - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (prefix[mid] <= t0) lo = mid; else hi = mid - 1;
    }
    p0 = lo;
    if (FUSED && tid == 0 && f.start_prev != nullptr) f.start_prev[blockIdx.x] = make_int2(p0, (int)(t0 - prefix[p0]));
  }
  if constexpr (FUSED) {
    if (warp > NWC) {
      unsigned char* fsm = smem + Tr::al16(Tr::OFF_PREFIX + (npairs + 1) * 4);
      fused_scorer<HD, G>(f, a.q, a.out, a.part, a.part_count, prefix, sp, a.D, a.B, a.qscale, fsm,
                          tid - (NWC + 1) * 32);
    }
  }

  // ---- producer -------------------------------------------------------------------
  // With the testing hook on, the producer neither arms a barrier nor issues a copy:
  // every consumer's first bounded wait runs out, records DEVERR_TIMEOUT_FULL and the
  // consumers skip the rest of their work; no copy is in flight when the CTA exits.
  if (warp == NWC && streams) {
    if (lane == 0 && !a.skip_copies) {
      int p = p0;
      long long i = 0;
      for (long long t = t0; t < t1; ++t, ++i) {
        while (t >= prefix[p + 1]) ++p;
        const int lt = (int)(t - prefix[p]);
        const int nv = used_slots(a.nvalid[p], a.B, nullptr);
        const int nvt = (nv + TILE - 1) / TILE;
        const CUtensorMap *mk, *mv;
        int row;
        uint32_t bytes;
        if (lt < nvt) {
          mk = &mapSK; mv = &mapSV; row = p * a.B + lt * TILE;
          bytes = (uint32_t)Tr::STAGE_BYTES;
        } else {
          mk = &mapRK; mv = &mapRV; row = p * a.D + (lt - nvt) * TILE;
          bytes = (uint32_t)(2 * NH * a.ring_rows * 128);
        }
        const int s = (int)(i % STAGES);
        if (i >= STAGES &&
            !mbar_wait(smem_u32(&bars[STAGES + s]), (uint32_t)((i / STAGES - 1) & 1), a.err,
                       DEVERR_TIMEOUT_EMPTY))
          break;
        const uint32_t fb = smem_u32(&bars[s]);
        mbar_arrive_expect_tx(fb, bytes);
        const uint32_t dst = smem_u32(smem + (size_t)s * Tr::STAGE_BYTES);
#pragma unroll
        for (int hh = 0; hh < NH; ++hh) {
          tma_load_2d(dst + hh * Tr::HALF_BYTES, mk, hh * 64, row, fb);
          tma_load_2d(dst + (NH + hh) * Tr::HALF_BYTES, mv, hh * 64, row, fb);
        }
      }
      const long long issued = i;
      for (long long k = issued > STAGES ? issued - STAGES : 0; k < issued; ++k)
        if (!mbar_wait(smem_u32(&bars[k % STAGES]), (uint32_t)((k / STAGES) & 1), a.err,
                       DEVERR_TIMEOUT_DRAIN))
          break;
    }
    if constexpr (!FUSED) return;
  }
  if (warp < NWC && streams) {

  // ---- consumers ------------------------------------------------------------------
  const int g8 = lane >> 2, t4 = lane & 3;            // fragment row group / column pair
  uint32_t qb[NKS][2];                                 // Q^T B fragments (head g8)
  float o[NMT][4];                                     // O^T accumulators
  float m0, m1, l0, l1;                                // heads 2*t4, 2*t4 + 1
  bool ok = true;
  int cur = -1;
  // FUSED: the slot that may change this step (full cache: the cached argmin) and the
  // window row of the token leaving the window; both masked, merged by the last arrival
  int cfull = -1, wmask = -1;

  auto load_q = [&](int p) {
    if constexpr (FUSED) {
      const int plen = a.len[p];
      const int nvp = used_slots(a.nvalid[p], a.B, nullptr);
      cfull = (plen >= a.D && nvp >= a.B) ? f.st.min_slot[p] : -1;
      wmask = (plen >= a.D) ? plen % a.D : -1;
    }
    const bf16* qp = a.q + ((size_t)p * G + g8) * HD;
#pragma unroll
    for (int ks = 0; ks < NKS; ++ks) {
      if (g8 < G) {
        qb[ks][0] = *reinterpret_cast<const uint32_t*>(qp + ks * 16 + 2 * t4);
        qb[ks][1] = *reinterpret_cast<const uint32_t*>(qp + ks * 16 + 8 + 2 * t4);
      } else {
        qb[ks][0] = 0u;
        qb[ks][1] = 0u;
      }
    }
#pragma unroll
    for (int mt = 0; mt < NMT; ++mt)
#pragma unroll
      for (int e = 0; e < 4; ++e) o[mt][e] = 0.f;
    m0 = m1 = -INFINITY;
    l0 = l1 = 0.f;
  };

  auto finalize = [&](int p) {
    // sum l over the 8 row groups (lanes with the same t4)
#pragma unroll
    for (int off = 4; off < 32; off <<= 1) {
      l0 += __shfl_xor_sync(0xffffffffu, l0, off);
      l1 += __shfl_xor_sync(0xffffffffu, l1, off);
    }
    const int h0 = 2 * t4, h1 = 2 * t4 + 1;
    if (h0 < G) {
#pragma unroll
      for (int mt = 0; mt < NMT; ++mt) {
        mo[(warp * G + h0) * HD + mt * 16 + g8] = o[mt][0];
        mo[(warp * G + h0) * HD + mt * 16 + 8 + g8] = o[mt][2];
      }
      if (g8 == 0) { ml[warp * G + h0] = l0; mm[warp * G + h0] = m0; }
    }
    if (h1 < G) {
#pragma unroll
      for (int mt = 0; mt < NMT; ++mt) {
        mo[(warp * G + h1) * HD + mt * 16 + g8] = o[mt][1];
        mo[(warp * G + h1) * HD + mt * 16 + 8 + g8] = o[mt][3];
      }
      if (g8 == 0) { ml[warp * G + h1] = l1; mm[warp * G + h1] = m1; }
    }
    consumer_sync();
    if constexpr (!FUSED) {
      finish_pair<G, HD, NWC, NWC * 32>(p, prefix, Ttot, NC, t0, mo, ml, mm, a.out, a.part,
                                        a.part_count, flag, [] { consumer_sync(); });
    } else {
      constexpr int NCT = NWC * 32, PSTRIDE = G * HD + 2 * G;
      constexpr int EPT = MergeShape<HD, G, NCT>::EPT;
      float om[EPT], ol[EPT], oo[EPT];
#pragma unroll
      for (int k = 0; k < EPT; ++k) {
        const int idx = tid + k * NCT;
        om[k] = -INFINITY; ol[k] = 0.f; oo[k] = 0.f;
        if (idx >= G * HD) continue;
        const int g = idx / HD, i = idx - g * HD;
        float ms = -INFINITY;
#pragma unroll
        for (int w = 0; w < NWC; ++w) ms = fmaxf(ms, mm[w * G + g]);
        float L = 0.f, O = 0.f;
#pragma unroll
        for (int w = 0; w < NWC; ++w) {
          const float mw = mm[w * G + g];
          const float fw = (mw == -INFINITY) ? 0.f : exp2f(mw - ms);
          L = fmaf(ml[w * G + g], fw, L);
          O = fmaf(mo[(w * G + g) * HD + i], fw, O);
        }
        om[k] = ms; ol[k] = L; oo[k] = O;
      }
      long long ca, cb;
      const int nctas = pair_ctas(p, prefix, sp, ca, cb);
      // every other arrival (the other CTAs and the scorer) already in: merge from here
      // without publishing this CTA's partial
      if (tid == 0) *flag = (ld_acquire_gpu(a.part_count + p) == nctas);
      consumer_sync();
      bool last = *flag != 0;
      // seen as last by the acquire above (ordered for every consumer by the barrier), or
      // by the relaxed count below, which needs a fence before the others' data is read
      const bool acquired = last;
      if (!last) {
        float* dst = (nctas == 1) ? f.part_c + (size_t)p * PSTRIDE
                                  : a.part + ((size_t)blockIdx.x * 2 + ((prefix[p] < t0) ? 0 : 1)) * PSTRIDE;
#pragma unroll
        for (int k = 0; k < EPT; ++k) {
          const int idx = tid + k * NCT;
          if (idx >= G * HD) continue;
          const int g = idx / HD, i = idx - g * HD;
          dst[g * HD + i] = oo[k];
          if (i == 0) { dst[G * HD + g] = om[k]; dst[G * HD + G + g] = ol[k]; }
        }
        __threadfence();
        consumer_sync();
        if (tid == 0) *flag = (atomicAdd(a.part_count + p, 1) == nctas);
        consumer_sync();
        last = *flag != 0;
      }
      if (last) {
        if (!acquired) __threadfence();
        fused_merge<HD, G, NCT>(f, a.out, a.part, a.part_count, p, prefix, sp, (long long)blockIdx.x,
                                om, ol, oo, tid, sched_seen, [] { consumer_sync(); });
      }
      consumer_sync();
    }
  };

  const float qs = a.qscale;
  int p = p0;
  long long i = 0;
  for (long long t = t0; t < t1; ++t, ++i) {
    while (t >= prefix[p + 1]) ++p;                    // control flow from the schedule only
    if (p != cur) {
      if (cur >= 0) finalize(cur);
      cur = p;
      load_q(p);
    }
    const int s = (int)(i % STAGES);
    if (ok) ok = mbar_wait(smem_u32(&bars[s]), (uint32_t)((i / STAGES) & 1), a.err, DEVERR_TIMEOUT_FULL);
    const int lt = (int)(t - prefix[p]);
    const int nv = used_slots(a.nvalid[p], a.B, nullptr);
    const int nvt = (nv + TILE - 1) / TILE;
    const int cnt = lt < nvt ? min(TILE, nv - lt * TILE)
                             : min(TILE, window_rows(a.len[p], a.D, nullptr) - (lt - nvt) * TILE);
    if constexpr (!FUSED) dcheck(cnt > 0 && cnt <= TILE, a.err, DEVERR_INDEX);
    int mrow = -1;                                     // FUSED: masked row of this tile
    if constexpr (FUSED) {
      const int r = (lt < nvt) ? (cfull >= 0 ? cfull - lt * TILE : -1)
                               : (wmask >= 0 ? wmask - (lt - nvt) * TILE : -1);
      mrow = (r >= 0 && r < TILE) ? r : -1;
    }
    const int key0 = warp * 16;
    if (ok && key0 < cnt) {
      const uint32_t kbase = smem_u32(smem + (size_t)s * Tr::STAGE_BYTES);
      const uint32_t vbase = kbase + NH * Tr::HALF_BYTES;
      // ---- S^T = K Q^T over d, two accumulator chains
      float c0[4] = {0.f, 0.f, 0.f, 0.f}, c1[4] = {0.f, 0.f, 0.f, 0.f};
      {
        const int row = key0 + (lane & 7) + ((lane >> 3) & 1) * 8;
        const uint32_t rbase = kbase + row * 128;
        const int sw = row & 7;
#pragma unroll
        for (int ks = 0; ks < NKS; ++ks) {
          const int chunk = (ks & 3) * 2 + (lane >> 4);
          const uint32_t addr = rbase + (ks >> 2) * Tr::HALF_BYTES + ((chunk ^ sw) << 4);
          uint32_t x0, x1, x2, x3;
          ldsm_x4(addr, x0, x1, x2, x3);
          if (ks & 1) mma_bf16(c1, x0, x1, x2, x3, qb[ks][0], qb[ks][1]);
          else        mma_bf16(c0, x0, x1, x2, x3, qb[ks][0], qb[ks][1]);
        }
      }
      const bool va = key0 + g8 < cnt && key0 + g8 != mrow;
      const bool vb = key0 + g8 + 8 < cnt && key0 + g8 + 8 != mrow;
      float s0 = va ? (c0[0] + c1[0]) * qs : -INFINITY;   // key g8,   head 2 t4
      float s1 = va ? (c0[1] + c1[1]) * qs : -INFINITY;   // key g8,   head 2 t4 + 1
      float s2 = vb ? (c0[2] + c1[2]) * qs : -INFINITY;   // key g8+8, head 2 t4
      float s3 = vb ? (c0[3] + c1[3]) * qs : -INFINITY;   // key g8+8, head 2 t4 + 1
      const bool need = (s0 > m0 + kThr) || (s2 > m0 + kThr) || (s1 > m1 + kThr) || (s3 > m1 + kThr);
      if (__any_sync(0xffffffffu, need)) {
        float x0 = fmaxf(s0, s2), x1 = fmaxf(s1, s3);
#pragma unroll
        for (int off = 4; off < 32; off <<= 1) {
          x0 = fmaxf(x0, __shfl_xor_sync(0xffffffffu, x0, off));
          x1 = fmaxf(x1, __shfl_xor_sync(0xffffffffu, x1, off));
        }
        const float n0 = fmaxf(m0, x0), n1 = fmaxf(m1, x1);
        const float f0 = ex2(m0 - n0), f1 = ex2(m1 - n1);
        l0 *= f0;
        l1 *= f1;
#pragma unroll
        for (int mt = 0; mt < NMT; ++mt) {
          o[mt][0] *= f0; o[mt][1] *= f1; o[mt][2] *= f0; o[mt][3] *= f1;
        }
        m0 = n0;
        m1 = n1;
      }
      const float p0 = va ? ex2(s0 - m0) : 0.f;
      const float p1 = va ? ex2(s1 - m1) : 0.f;
      const float p2 = vb ? ex2(s2 - m0) : 0.f;
      const float p3 = vb ? ex2(s3 - m1) : 0.f;
      // the normaliser uses the same bf16-rounded weights as the numerator
      const uint32_t x0 = pack_bf16(p0, p1), x1 = pack_bf16(p2, p3);
      {
        const __nv_bfloat162 r0 = *reinterpret_cast<const __nv_bfloat162*>(&x0);
        const __nv_bfloat162 r1 = *reinterpret_cast<const __nv_bfloat162*>(&x1);
        l0 += __bfloat162float(r0.x) + __bfloat162float(r1.x);
        l1 += __bfloat162float(r0.y) + __bfloat162float(r1.y);
      }
      const uint32_t b0 = movm_t(x0), b1 = movm_t(x1);
      // ---- O^T += V^T P^T, one m-tile of 16 d-rows at a time
      {
        const int j = lane >> 3;
        const int key = key0 + (lane & 7) + (j >> 1) * 8;
        const uint32_t rbase = vbase + key * 128;
        const int sw = key & 7;
#pragma unroll
        for (int mt = 0; mt < NMT; ++mt) {
          const int dcol = mt * 16 + (j & 1) * 8;
          const int chunk = (dcol & 63) >> 3;
          const uint32_t addr = rbase + (dcol >> 6) * Tr::HALF_BYTES + ((chunk ^ sw) << 4);
          uint32_t y0, y1, y2, y3;
          ldsm_x4_t(addr, y0, y1, y2, y3);
          mma_bf16(o[mt], y0, y1, y2, y3, b0, b1);
        }
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(smem_u32(&bars[STAGES + s]));
  }
  if (cur >= 0) finalize(cur);
  }   // consumers
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

cudaError_t encode_rows(EncodeTiledFn fn, CUtensorMap* map, void* base, int d, long long rows,
                        int box_rows) {
  cuuint64_t dims[2] = {(cuuint64_t)d, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)d * 2};
  cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

template <int HD, int G>
size_t tc_smem(int pairs) {
  using Tr = TcTraits<HD, G>;
  return Tr::SMEM_ALIGN + Tr::OFF_PREFIX + (size_t)(pairs + 1) * 4;
}

}  // namespace

struct TcMaps {
  CUtensorMap sk, sv, rk, rv;
};

int g_debug_skip_copies = 0;   // kvpop_debug_skip_attention_copies

// Window boxes only need D rows (rounded up to a swizzle atom's 8) when D < TILE.
static int tc_ring_rows(const Dims& dm) {
  const int tile = TcTraits<128, 4>::TILE;
  const int r = (dm.D + 7) / 8 * 8;
  return r < tile ? r : tile;
}

cudaError_t tc_make_maps(const State& st, const Dims& dm, void* maps_out) {
  void* fn = nullptr;
  cudaDriverEntryPointQueryResult q;
  cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000,
                                                   cudaEnableDefault, &q);
  if (e != cudaSuccess) return e;
  if (q != cudaDriverEntryPointSuccess || fn == nullptr) return cudaErrorNotSupported;
  auto enc = reinterpret_cast<EncodeTiledFn>(fn);
  TcMaps* m = static_cast<TcMaps*>(maps_out);
  const int box = TcTraits<128, 4>::TILE;
  const int rbox = tc_ring_rows(dm);
  const long long srows = (long long)dm.pairs * dm.B, rrows = (long long)dm.pairs * dm.D;
  if ((e = encode_rows(enc, &m->sk, st.slotK, dm.d, srows, box)) != cudaSuccess) return e;
  if ((e = encode_rows(enc, &m->sv, st.slotV, dm.d, srows, box)) != cudaSuccess) return e;
  if ((e = encode_rows(enc, &m->rk, st.ringK, dm.d, rrows, rbox)) != cudaSuccess) return e;
  return encode_rows(enc, &m->rv, st.ringV, dm.d, rrows, rbox);
}

size_t tc_maps_size() { return sizeof(TcMaps); }

#define TC_CASES(X) X(64, 1) X(64, 2) X(64, 4) X(128, 1) X(128, 2) X(128, 4)
#define TC_FUSED_CASES(X) X(128, 1) X(128, 2) X(128, 4)

cudaError_t tc_config(const Dims& dm, AttendConfig* out) {
#define CFG(HD_, G_)                                                   \
  if (dm.d == HD_ && dm.G == G_) {                                     \
    out->threads = TcTraits<HD_, G_>::THREADS;                         \
    out->smem_fixed = tc_smem<HD_, G_>(0) - 4;                         \
    out->tile = TcTraits<HD_, G_>::TILE;                               \
    out->func = (const void*)attend_tc_kernel<HD_, G_, false>;         \
    return cudaSuccess;                                                \
  }
  TC_CASES(CFG)
#undef CFG
  return cudaErrorInvalidValue;
}

int tc_fused_max_grid() { return kMaxSplit; }

bool tc_fused_ok(const Dims& dm) {
  return dm.dtype == KVPOP_BF16 && dm.d == 128 && (dm.G == 1 || dm.G == 2 || dm.G == 4) &&
         dm.F <= 256;
}

// Smem of the fused kernel: the attention's, then the scorer region after the prefix.
static size_t tc_fused_smem_of(size_t attn_smem_pairs, int Fp) {
  return ((attn_smem_pairs + 15) & ~size_t(15)) + fused_smem_bytes(Fp);
}

cudaError_t tc_fused_config(const Dims& dm, AttendConfig* out) {
#define CFG(HD_, G_)                                                           \
  if (dm.d == HD_ && dm.G == G_) {                                             \
    out->threads = TcTraits<HD_, G_>::THREADS_F;                               \
    out->smem_fixed = tc_fused_smem_of(tc_smem<HD_, G_>(0) - 4, dm.Fp) + 16;   \
    out->tile = TcTraits<HD_, G_>::TILE;                                       \
    out->func = (const void*)attend_tc_kernel<HD_, G_, true>;                  \
    return cudaSuccess;                                                        \
  }
  if (tc_fused_ok(dm)) { TC_FUSED_CASES(CFG) }
#undef CFG
  return cudaErrorInvalidValue;
}

static TcArgs tc_args(const State& st, const Dims& dm, const void* q, float* out) {
  TcArgs a;
  a.nvalid = st.nvalid;
  a.len = st.len;
  a.q = static_cast<const bf16*>(q);
  a.out = out;
  a.part = st.part;
  a.part_count = st.part_count;
  a.err = st.err;
  a.pairs = dm.pairs;
  a.B = dm.B;
  a.D = dm.D;
  a.ring_rows = tc_ring_rows(dm);
  a.qscale = kLog2e / sqrtf((float)dm.d);
  a.skip_copies = g_debug_skip_copies;
  return a;
}

cudaError_t tc_launch(const State& st, const Dims& dm, const void* maps, const void* q, float* out,
                      int grid, cudaStream_t stream) {
  const TcMaps* m = static_cast<const TcMaps*>(maps);
  const TcArgs a = tc_args(st, dm, q, out);
  FusedArgs f;
  memset(&f, 0, sizeof(f));
  // programmatic stream serialisation: the grid may be scheduled while the kernel
  // before it (the ingest) finishes; the kernel waits for it before touching the state
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.gridDim = dim3(grid, 1, 1);
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
#define LAUNCH(HD_, G_)                                                                   \
  if (dm.d == HD_ && dm.G == G_) {                                                        \
    cfg.blockDim = dim3(TcTraits<HD_, G_>::THREADS, 1, 1);                                \
    cfg.dynamicSmemBytes = tc_smem<HD_, G_>(dm.pairs);                                    \
    return cudaLaunchKernelEx(&cfg, attend_tc_kernel<HD_, G_, false>, m->sk, m->sv, m->rk, \
                              m->rv, a, f);                                               \
  }
  TC_CASES(LAUNCH)
#undef LAUNCH
  return cudaErrorInvalidValue;
}

cudaError_t tc_launch_fused(const State& st, const Dims& dm, const void* maps, const FusedBufs& fb,
                            const void* q, const void* k, const void* v, float* out,
                            const float* override_, int32_t* evict_info, float* score_out, int grid,
                            cudaStream_t stream) {
  if (!tc_fused_ok(dm)) return cudaErrorInvalidValue;
  const TcMaps* m = static_cast<const TcMaps*>(maps);
  const TcArgs a = tc_args(st, dm, q, out);
  FusedArgs f;
  memset(&f, 0, sizeof(f));
  f.st = st;
  f.k_new = static_cast<const bf16*>(k);
  f.v_new = static_cast<const bf16*>(v);
  f.override_ = override_;
  f.evict_info = evict_info;
  f.score_out = score_out;
  f.part_c = fb.part_c;
  f.meta_next = fb.meta_next;
  f.xtra = fb.xtra;
  f.ctr = fb.ctr;
  f.start_prev = fb.start_prev;
  f.batch = dm.batch;
  f.H = dm.H;
  f.F = dm.F;
  f.Fp = dm.Fp;
  f.s = dm.s;
  f.act = dm.act;
  // a programmatic dependent of the step before it: scheduled while that one finishes,
  // waits for it before reading any state
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.gridDim = dim3(grid, 1, 1);
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
#define LAUNCH(HD_, G_)                                                                    \
  if (dm.d == HD_ && dm.G == G_) {                                                         \
    cfg.blockDim = dim3(TcTraits<HD_, G_>::THREADS_F, 1, 1);                               \
    cfg.dynamicSmemBytes = tc_fused_smem_of(tc_smem<HD_, G_>(dm.pairs), dm.Fp);            \
    return cudaLaunchKernelEx(&cfg, attend_tc_kernel<HD_, G_, true>, m->sk, m->sv, m->rk,  \
                              m->rv, a, f);                                                \
  }
  TC_FUSED_CASES(LAUNCH)
#undef LAUNCH
  return cudaErrorInvalidValue;
}

}  // namespace kvpop
