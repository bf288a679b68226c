// Decode steps 1-4 with one thread-block cluster per (KV head, group of 16
// sequences): ingest, delayed scorer, keep-or-drop, scatter.
//
// The 8 CTAs of a cluster split the scorer's hidden units: CTA r holds the
// slice [r*FS, (r+1)*FS) of W1 (3d x FS fp32, 48 KB for d = 128, F = 256),
// loaded in one go by bulk copies together with everything its two "owned"
// sequences need (window query means, the leaving token's K/V row, the new
// q/k/v).  Each owner builds its sequences' scorer inputs
// x = [k_u; v_u; qbar_u] (Sec. 3.3 delayed scoring, App. E.4) and writes them
// into every CTA of the cluster through distributed shared memory; after a
// cluster barrier each CTA evaluates its hidden slice for all 16 sequences and
// sends the partial output sums back to the owners; the owners add the 8
// partials in a fixed order, then run the keep-or-drop rule of Sec. 3.2 /
// App. C.1 (static priority, App. B.3) and scatter the token into its slot.
// The state the eviction reads (used slots, the cached minimum, its block) is
// loaded at kernel start so its latency hides behind the scorer.
#include "kvpop_argmin.cuh"

namespace kvpop {
namespace {

constexpr int CS = 8;          // CTAs per cluster (hidden-unit slices)
constexpr int SBC = 16;        // sequences per cluster
constexpr int OWN = SBC / CS;  // sequences owned by each CTA (2)
constexpr int NT = 256;        // threads per CTA: warp w evaluates sequences 2w, 2w+1
constexpr int kMaxBlkLanes = 8;  // block minima prefetched per lane (B <= 16384 slots)

template <typename T>
struct ClArgs {
  State st;
  Dims dm;
  const float* W1s;            // [H][CS][3d][FS]
  const float* b1s;            // [H][CS][FS]
  const float* w2s;            // [H][CS][FS]
  int FS;
  const T* q;                  // [b][H*G][d]
  const T* k;                  // [b][H][d]
  const T* v;
  const float* override_;
  int32_t* evict_info;
  float* score_out;
};

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t map_rank(uint32_t local, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(local), "r"(rank));
  return r;
}
__device__ __forceinline__ void st_cluster_v4(uint32_t addr, float4 v) {
  asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "f"(v.x), "f"(v.y),
               "f"(v.z), "f"(v.w)
               : "memory");
}
__device__ __forceinline__ void st_cluster_f32(uint32_t addr, float v) {
  asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(addr), "f"(v) : "memory");
}
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::
                   : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.expect_tx.relaxed.cta.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}

// D (16x8, fp32) += A (16x8, tf32, row) B (8x8, tf32, col), legacy tensor-core MMA
__device__ __forceinline__ void mma_tf32_16x8x8(float (&c)[4], const uint32_t (&a)[4],
                                                const uint32_t (&b)[2]) {
  asm volatile(
      "mma.sync.aligned.m16n8k8.row.col.f32.tf32.tf32.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7},"
      " {%8, %9}, {%0, %1, %2, %3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
}

struct ClLayout {              // byte offsets into dynamic shared memory
  int ws, x, qm, qrow, ring, newkv, part, total;
};
__host__ __device__ inline ClLayout cl_layout(int d, int D, int G, int FS, int esz) {
  ClLayout L;
  const int R = d * esz;
  int o = 0;
  L.ws = o;    o += 3 * d * FS * 4;                 // W1 slice, then b1, w2 slices
  o += 2 * FS * 4;
  L.x = o;     o += SBC * (3 * d + 4) * 4;          // scorer inputs of the 16 sequences (row stride 3d + 4)
  L.qm = o;    o += OWN * D * d * 4;                // window query means of the owned sequences
  L.qrow = o;  o += OWN * G * R;                    // new queries
  L.ring = o;  o += OWN * 2 * R;                    // K, V row of the leaving token
  L.newkv = o; o += OWN * 2 * R;                    // new K, V row
  L.part = o;  o += CS * OWN * 4;                   // partial scores from each CTA
  L.total = o;
  return L;
}

template <typename T>
__global__ void __launch_bounds__(NT, 1) ingest_cluster_kernel(ClArgs<T> a) {
  const Dims& dm = a.dm;
  const int d = dm.d, D = dm.D, G = dm.G, F = dm.F, B = dm.B, H = dm.H, FS = a.FS;
  const int in_dim = 3 * d;
  const int R = d * (int)sizeof(T);
  const int h = blockIdx.y;
  const uint32_t rank = cluster_rank();
  const int group = blockIdx.x / CS;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const ClLayout L = cl_layout(d, D, G, FS, (int)sizeof(T));

  extern __shared__ __align__(128) unsigned char smem[];
  float* Ws = reinterpret_cast<float*>(smem + L.ws);
  const float* b1s = Ws + in_dim * FS;
  const float* w2s = b1s + FS;
  float* X = reinterpret_cast<float*>(smem + L.x);           // [SBC][3d + 4]
  const int XS = in_dim + 4;
  float* rqm = reinterpret_cast<float*>(smem + L.qm);        // [OWN][D][d]
  T* qrow = reinterpret_cast<T*>(smem + L.qrow);             // [OWN][G][d]
  T* ring = reinterpret_cast<T*>(smem + L.ring);             // [OWN][2][d]
  T* newkv = reinterpret_cast<T*>(smem + L.newkv);           // [OWN][2][d]
  float* part = reinterpret_cast<float*>(smem + L.part);     // [CS][OWN]
  __shared__ __align__(8) uint64_t bar;
  __shared__ int s_p[OWN];

  // sequences of this cluster: group*SBC + j; CTA `rank` owns j = OWN*rank + o
  const int own_b0 = group * SBC + OWN * (int)rank;

  // the attention that follows may be scheduled now; it waits for this grid to complete
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  // ---- issue every load this CTA needs ------------------------------------------------
  if (tid == 0) {
    mbar_init(smem_u32(&bar), 1);
    mbar_fence_init();
    const uint32_t bb = smem_u32(&bar);
    const size_t slice = (size_t)h * CS + rank;
    const uint32_t wbytes = (uint32_t)(in_dim * FS * 4), vbytes = (uint32_t)(FS * 4);
    mbar_expect_tx(bb, wbytes + 2 * vbytes);
    const unsigned char* wsrc = reinterpret_cast<const unsigned char*>(a.W1s + slice * in_dim * FS);
    for (uint32_t off = 0; off < wbytes; off += 16384)
      bulk_g2s(smem_u32(smem + L.ws + off), wsrc + off, min(16384u, wbytes - off), bb);
    bulk_g2s(smem_u32(Ws + in_dim * FS), a.b1s + slice * FS, vbytes, bb);
    bulk_g2s(smem_u32(Ws + in_dim * FS + FS), a.w2s + slice * FS, vbytes, bb);
    // rows that do not depend on the sequence length first ...
    uint32_t rest = 0;
    for (int o = 0; o < OWN; ++o)
      if (own_b0 + o < dm.batch) rest += (uint32_t)(D * d * 4 + G * R + 2 * R);
    mbar_expect_tx(bb, rest);
    for (int o = 0; o < OWN; ++o) {
      const int b = own_b0 + o;
      if (b >= dm.batch) continue;
      const int pair = b * H + h;
      bulk_g2s(smem_u32(rqm + (size_t)o * D * d), a.st.ringQm + (size_t)pair * D * d, D * d * 4, bb);
      bulk_g2s(smem_u32(qrow + (size_t)o * G * d), a.q + (size_t)pair * G * d, G * R, bb);
      bulk_g2s(smem_u32(newkv + (size_t)(2 * o) * d), a.k + (size_t)pair * d, R, bb);
      bulk_g2s(smem_u32(newkv + (size_t)(2 * o + 1) * d), a.v + (size_t)pair * d, R, bb);
    }
    // ... then the leaving token's K/V row, whose window index needs the length
    int pl[OWN];
    uint32_t rows = 0;
    for (int o = 0; o < OWN; ++o) {
      const int b = own_b0 + o;
      pl[o] = b < dm.batch ? a.st.len[b * H + h] : -1;
      s_p[o] = pl[o];
      if (b < dm.batch) rows += (uint32_t)(2 * R);
    }
    mbar_arrive_expect_tx(bb, rows);
    for (int o = 0; o < OWN; ++o) {
      const int b = own_b0 + o;
      if (b >= dm.batch) continue;
      const int pair = b * H + h;
      const int ri = pl[o] % D;
      bulk_g2s(smem_u32(ring + (size_t)(2 * o) * d),
               static_cast<const T*>(a.st.ringK) + ((size_t)pair * D + ri) * d, R, bb);
      bulk_g2s(smem_u32(ring + (size_t)(2 * o + 1) * d),
               static_cast<const T*>(a.st.ringV) + ((size_t)pair * D + ri) * d, R, bb);
    }
  }
  // lengths and eviction state of the owned sequences, read now so they are ready later:
  // the cached minimum, the 64 priorities of its block, the block minima and the
  // position it holds (all that a replacement touches)
  const int NB = min_blocks(B);
  const int nbl = (NB + 31) / 32;
  const bool reg_min = nbl <= kMaxBlkLanes;
  int ev_nv = 0, ev_mslot = -1, ev_pos = -1;
  float ev_mscore = INFINITY;
  float blkv[2] = {INFINITY, INFINITY};
  float nbv[kMaxBlkLanes];
  int nbs[kMaxBlkLanes];
#pragma unroll
  for (int t = 0; t < kMaxBlkLanes; ++t) { nbv[t] = INFINITY; nbs[t] = 0x7fffffff; }
  if (warp < OWN) {
    const int b = own_b0 + warp;
    if (b < dm.batch) {
      const int pair = b * H + h;
      ev_nv = a.st.nvalid[pair];
      ev_mscore = a.st.min_score[pair];
      ev_mslot = a.st.min_slot[pair];
      if (ev_nv == B && ev_mslot >= 0 && reg_min) {
        const float* sc = a.st.score + (size_t)pair * B;
        const int lo = (ev_mslot / kMinBlock) * kMinBlock;
        blkv[0] = (lo + lane < B) ? sc[lo + lane] : INFINITY;
        blkv[1] = (lo + 32 + lane < B) ? sc[lo + 32 + lane] : INFINITY;
        ev_pos = a.st.pos[(size_t)pair * B + ev_mslot];
#pragma unroll
        for (int t = 0; t < kMaxBlkLanes; ++t) {
          const int k = lane + 32 * t;
          nbv[t] = (t < nbl && k < NB) ? a.st.blk_score[(size_t)pair * NB + k] : INFINITY;
          nbs[t] = (t < nbl && k < NB) ? a.st.blk_slot[(size_t)pair * NB + k] : 0x7fffffff;
        }
      }
    }
  }
  __syncthreads();
  const bool ok = mbar_wait(smem_u32(&bar), 0, a.st.err, DEVERR_TIMEOUT_FULL);

  // ---- scorer inputs of the owned sequences, broadcast to the cluster; window update --
  // warp w builds a quarter of the input row of owned sequence w / 4
  {
    const int o = warp >> 2, qq = warp & 3;
    const int j = OWN * (int)rank + o;       // row of X
    const int b = own_b0 + o;
    const int p = s_p[o];
    const bool active = ok && b < dm.batch && p >= D;
    const int ri = p >= 0 ? p % D : 0;
    const T* ku = ring + (size_t)(2 * o) * d;                 // the leaving token u = p - D
    const T* vu = ring + (size_t)(2 * o + 1) * d;
    const uint32_t xrow = smem_u32(X + (size_t)j * XS);
    const int nq4 = in_dim / 16;             // float4s per quarter
    if (lane < nq4) {
      const int i4 = qq * nq4 + lane;
      float4 val = make_float4(0.f, 0.f, 0.f, 0.f);
      if (active) {
        float e[4];
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          const int i = i4 * 4 + t;
          if (i < d) {
            e[t] = to_f(ku[i]);
          } else if (i < 2 * d) {
            e[t] = to_f(vu[i - d]);
          } else {
            const int c = i - 2 * d;
            float qsum = 0.f;
            for (int g = 0; g < G; ++g) qsum += to_f(qrow[(o * G + g) * d + c]);
            const float qm_p = qsum * (1.0f / (float)G);
            // qbar_u: queries u+1 .. p in position order, averaged over D
            float acc = 0.f;
            for (int jj = 1; jj < D; ++jj) {
              int w = ri + jj;
              w = w >= D ? w - D : w;
              acc += rqm[((size_t)o * D + w) * d + c];
            }
            acc += qm_p;
            e[t] = acc / (float)D;
          }
        }
        val = make_float4(e[0], e[1], e[2], e[3]);
      }
#pragma unroll
      for (int dst = 0; dst < CS; ++dst) st_cluster_v4(map_rank(xrow + i4 * 16, dst), val);
    }
    if (ok && b < dm.batch) {
      // push the new token into the window slot of u (u's copy stays in smem)
      const int pair = b * H + h;
      T* dk = static_cast<T*>(a.st.ringK) + ((size_t)pair * D + ri) * d;
      T* dv = static_cast<T*>(a.st.ringV) + ((size_t)pair * D + ri) * d;
      float* dq = a.st.ringQm + ((size_t)pair * D + ri) * d;
      for (int i = qq * 32 + lane; i < d; i += 128) {
        dk[i] = newkv[(2 * o) * d + i];
        dv[i] = newkv[(2 * o + 1) * d + i];
        float qsum = 0.f;
        for (int g = 0; g < G; ++g) qsum += to_f(qrow[(o * G + g) * d + i]);
        dq[i] = qsum * (1.0f / (float)G);
      }
    }
  }
  cluster_sync();   // every X row is in every CTA

  // ---- this CTA's hidden slice for all 16 sequences --------------------------------------
  // H[16 sequences][FS] = X W, fp32-accurate.  With FS a multiple of 8 it runs on the tensor
  // pipe: m16n8k8 tf32 MMAs, each operand split into a tf32 head and its residual and
  // X W = X_hi W_hi + X_hi W_lo + X_lo W_hi (the dropped X_lo W_lo is below fp32 rounding);
  // warp w takes k-steps [w K8 / 8, (w + 1) K8 / 8) of the 3d inputs.  Otherwise thread
  // (f, ks) accumulates unit f over input slice ks for every sequence.  Either way the
  // partial sums meet in shared memory (over the input rows, no longer needed), then warp w
  // adds b1, applies the activation and contracts with w2 for sequences 2w, 2w+1.
  {
    // (the 8 warp partials of [16][FS] must fit in the input rows: 8 FS <= 3d + 4)
    const bool tc = (FS % 8) == 0 && (in_dim % 64) == 0 && 8 * FS <= XS && FS <= 64;
    int NKS;                                          // partial sums per (sequence, unit)
    float* red = X;                                   // [NKS][SBC][FS]
    if (tc) {
      NKS = NT / 32;
      const int g = lane >> 2, tig = lane & 3;
      const int k8 = in_dim / 8, kper = k8 / NKS, kb = warp * kper;
      float acc[8][4];                                // up to FS = 64: 8 n-tiles
#pragma unroll
      for (int nt = 0; nt < 8; ++nt)
#pragma unroll
        for (int e = 0; e < 4; ++e) acc[nt][e] = 0.f;
      auto split = [](float x, uint32_t& hi, uint32_t& lo) {
        asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(hi) : "f"(x));
        lo = __float_as_uint(x - __uint_as_float(hi));
      };
      for (int kk = 0; kk < kper; ++kk) {
        const int k0 = (kb + kk) * 8;
        uint32_t ah[4], al[4];
        split(X[(size_t)g * XS + k0 + tig], ah[0], al[0]);
        split(X[(size_t)(g + 8) * XS + k0 + tig], ah[1], al[1]);
        split(X[(size_t)g * XS + k0 + tig + 4], ah[2], al[2]);
        split(X[(size_t)(g + 8) * XS + k0 + tig + 4], ah[3], al[3]);
#pragma unroll
        for (int nt = 0; nt < 8; ++nt) {
          if (nt * 8 >= FS) break;
          uint32_t bh[2], bl[2];
          split(Ws[(size_t)(k0 + tig) * FS + nt * 8 + g], bh[0], bl[0]);
          split(Ws[(size_t)(k0 + tig + 4) * FS + nt * 8 + g], bh[1], bl[1]);
          mma_tf32_16x8x8(acc[nt], ah, bh);
          mma_tf32_16x8x8(acc[nt], ah, bl);
          mma_tf32_16x8x8(acc[nt], al, bh);
        }
      }
      __syncthreads();                                // every warp is done with X
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) {
        if (nt * 8 >= FS) break;
        const int col = nt * 8 + 2 * tig;
        float* r0 = red + ((size_t)warp * SBC + g) * FS + col;
        float* r8 = red + ((size_t)warp * SBC + g + 8) * FS + col;
        r0[0] = acc[nt][0];
        r0[1] = acc[nt][1];
        r8[0] = acc[nt][2];
        r8[1] = acc[nt][3];
      }
    } else {
      // NKS * FS <= 3d keeps the partial sums inside the input rows
      NKS = min(NT / FS, in_dim / FS);
      const int SL = ((in_dim + NKS - 1) / NKS + 3) & ~3;   // inputs per slice, multiple of 4
      const int f = tid % FS, ks = tid / FS;
      float acc[SBC];
#pragma unroll
      for (int j = 0; j < SBC; ++j) acc[j] = 0.f;
      if (ks < NKS) {
        const int i_end = min(in_dim, (ks + 1) * SL);
        for (int i = ks * SL; i < i_end; i += 4) {
          const float w0 = Ws[(i + 0) * FS + f], w1 = Ws[(i + 1) * FS + f];
          const float w2 = Ws[(i + 2) * FS + f], w3 = Ws[(i + 3) * FS + f];
#pragma unroll
          for (int j = 0; j < SBC; ++j) {
            const float4 u = *reinterpret_cast<const float4*>(X + (size_t)j * XS + i);
            acc[j] = fmaf(u.x, w0, fmaf(u.y, w1, fmaf(u.z, w2, fmaf(u.w, w3, acc[j]))));
          }
        }
      }
      __syncthreads();                                // every thread is done with X
      if (ks < NKS) {
#pragma unroll
        for (int j = 0; j < SBC; ++j) red[((size_t)ks * SBC + j) * FS + f] = acc[j];
      }
    }
    __syncthreads();
    float c0 = 0.f, c1 = 0.f;
    const int j0 = 2 * warp, j1 = 2 * warp + 1;
    for (int ff = lane; ff < FS; ff += 32) {
      float a0 = b1s[ff], a1 = a0;
      for (int kk = 0; kk < NKS; ++kk) {
        a0 += red[((size_t)kk * SBC + j0) * FS + ff];
        a1 += red[((size_t)kk * SBC + j1) * FS + ff];
      }
      const float wf = w2s[ff];
      c0 = fmaf(wf, scorer_act(a0, dm.act), c0);
      c1 = fmaf(wf, scorer_act(a1, dm.act), c1);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      c0 += __shfl_xor_sync(0xffffffffu, c0, off);
      c1 += __shfl_xor_sync(0xffffffffu, c1, off);
    }
    // sequences 2w, 2w+1 are owned by CTA w (OWN = 2): part[rank][o] there
    if (lane == 0) {
      const uint32_t dst = (uint32_t)warp;
      st_cluster_f32(map_rank(smem_u32(part + rank * OWN + 0), dst), c0);
      st_cluster_f32(map_rank(smem_u32(part + rank * OWN + 1), dst), c1);
    }
  }
  cluster_sync();   // partial sums have arrived; no remote access after this point
  if (tid == 0 && !ok) {
    // a wait expired: let the copies still in flight land before the CTA exits
    mbar_wait(smem_u32(&bar), 0, a.st.err, DEVERR_TIMEOUT_DRAIN);
  }

  // ---- owners: score, keep-or-drop, scatter ------------------------------------------------
  if (warp >= OWN) return;
  const int o = warp;
  const int b = own_b0 + o;
  if (b >= dm.batch || !ok) return;
  const int pair = b * H + h;
  const int p = s_p[o];
  if (p < D) {
    if (lane == 0) {
      a.st.len[pair] = p + 1;
      if (a.evict_info) { a.evict_info[2 * pair] = -1; a.evict_info[2 * pair + 1] = -1; }
      if (a.score_out) a.score_out[pair] = __int_as_float(0x7fc00000);
    }
    return;
  }
  float r = 0.f;
  for (int src = 0; src < CS; ++src) r += part[src * OWN + o];
  r += a.st.b2[h];
  if (a.override_) r = a.override_[pair];
  r = canon_score(r);
  const int u = p - D;
  const float prio = static_priority(r, u, a.st.log_gamma, h);

  float* sc = a.st.score + (size_t)pair * B;
  int32_t* ps = a.st.pos + (size_t)pair * B;
  float* bsc = a.st.blk_score + (size_t)pair * NB;
  int32_t* bsl = a.st.blk_slot + (size_t)pair * NB;
  int slot = -1, evicted = -1;
  if (ev_nv < B) {
    slot = ev_nv;
  } else if (prio > ev_mscore) {
    slot = ev_mslot;
    evicted = reg_min ? ev_pos : ps[slot];
  }
  if (slot >= 0 && !dcheck(slot < B && ev_nv >= 0 && (ev_nv < B || slot >= dm.s), a.st.err,
                           DEVERR_INDEX))
    slot = -1;
  if (slot >= 0) {
    T* dk = static_cast<T*>(a.st.slotK) + ((size_t)pair * B + slot) * d;
    T* dv = static_cast<T*>(a.st.slotV) + ((size_t)pair * B + slot) * d;
    const T* ku = ring + (size_t)(2 * o) * d;
    const T* vu = ring + (size_t)(2 * o + 1) * d;
    for (int i = lane; i < d; i += 32) {
      dk[i] = ku[i];
      dv[i] = vu[i];
    }
    if (ev_nv == B) {
      if (reg_min) {
        // block of the replaced slot from the prefetched priorities, then the head minimum
        const int k = slot / kMinBlock, lo = k * kMinBlock;
        float bm = INFINITY;
        int bmi = 0x7fffffff;
#pragma unroll
        for (int r2 = 0; r2 < 2; ++r2) {
          const int i = lo + r2 * 32 + lane;
          if (i < B && i >= dm.s) lex_min(bm, bmi, i == slot ? prio : blkv[r2], i);
        }
        warp_lex_min(bm, bmi);
        float m = INFINITY;
        int mi = 0x7fffffff;
#pragma unroll
        for (int t = 0; t < kMaxBlkLanes; ++t) {
          const int kk = lane + 32 * t;
          if (t < nbl && kk < NB) {
            if (kk == k) lex_min(m, mi, bm, bmi);
            else lex_min(m, mi, nbv[t], nbs[t]);
          }
        }
        warp_lex_min(m, mi);
        if (lane == 0) {
          bsc[k] = bm;
          bsl[k] = bmi;
          a.st.min_score[pair] = m;
          a.st.min_slot[pair] = mi;
        }
      } else {
        update_min(sc, dm.s, B, slot, prio, bsc, bsl, a.st.min_score + pair, a.st.min_slot + pair);
      }
    } else if (ev_nv + 1 == B) {
      rebuild_min(sc, dm.s, B, slot, prio, bsc, bsl, a.st.min_score + pair, a.st.min_slot + pair);
    }
    if (lane == 0) {
      sc[slot] = prio;
      ps[slot] = u;
      a.st.nvalid[pair] = ev_nv < B ? ev_nv + 1 : ev_nv;
    }
  }
  if (lane == 0) {
    a.st.len[pair] = p + 1;
    if (a.evict_info) { a.evict_info[2 * pair] = slot; a.evict_info[2 * pair + 1] = evicted; }
    if (a.score_out) a.score_out[pair] = r;
  }
  (void)F;
}

}  // namespace

int cluster_ingest_fs(const Dims& dm) { return ((dm.F + 31) / 32 * 32) / CS; }

bool cluster_ingest_ok(const Dims& dm) {
  const int FS = cluster_ingest_fs(dm);
  const ClLayout L = cl_layout(dm.d, dm.D, dm.G, FS, dm.dtype == KVPOP_F32 ? 4 : 2);
  return FS <= 64 && L.total <= 200 * 1024;
}

size_t cluster_ingest_smem(const Dims& dm) {
  return cl_layout(dm.d, dm.D, dm.G, cluster_ingest_fs(dm), dm.dtype == KVPOP_F32 ? 4 : 2).total;
}

cudaError_t prepare_ingest_cluster(const Dims& dm) {
  const int smem = (int)cluster_ingest_smem(dm);
  if (dm.dtype == KVPOP_F32)
    return raise_smem_limit(ingest_cluster_kernel<float>, smem);
  return raise_smem_limit(ingest_cluster_kernel<bf16>, smem);
}

template <typename T>
static cudaError_t launch_cl(const State& st, const Dims& dm, const float* W1s, const float* b1s,
                             const float* w2s, const void* q, const void* k, const void* v,
                             const float* override_, int32_t* evict_info, float* score_out,
                             cudaStream_t stream) {
  ClArgs<T> a{st, dm, W1s, b1s, w2s, cluster_ingest_fs(dm), (const T*)q, (const T*)k,
              (const T*)v, override_, evict_info, score_out};
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(CS * ((dm.batch + SBC - 1) / SBC), dm.H, 1);
  cfg.blockDim = dim3(NT, 1, 1);
  cfg.dynamicSmemBytes = cluster_ingest_smem(dm);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = CS;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, ingest_cluster_kernel<T>, a);
}

cudaError_t launch_ingest_cluster(const State& st, const Dims& dm, const float* W1s,
                                  const float* b1s, const float* w2s, const void* q,
                                  const void* k, const void* v, const float* override_,
                                  int32_t* evict_info, float* score_out, cudaStream_t stream) {
  if (dm.dtype == KVPOP_F32)
    return launch_cl<float>(st, dm, W1s, b1s, w2s, q, k, v, override_, evict_info, score_out, stream);
  return launch_cl<bf16>(st, dm, W1s, b1s, w2s, q, k, v, override_, evict_info, score_out, stream);
}

}  // namespace kvpop
