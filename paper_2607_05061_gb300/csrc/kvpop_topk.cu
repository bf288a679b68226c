// Running top-k cutoffs over a prompt (App. C.1 mask, App. C.2 cutoff scan).
//
// Kernel 1 (one CTA per row) ranks the row's tokens by static priority, higher
// first, equal priorities by position: a stable least-significant-digit radix
// sort of the order-reversed fp32 bit pattern, 4 passes of 8 bits.  Within a
// round of NT tokens the stable offset of each token inside its digit bucket
// comes from a warp match on the digit plus per-warp bucket counts; one
// histogram pass up front gives every pass its bucket bases.  The last pass
// writes rank[position] directly.
//
// Kernel 2 (one CTA per row, the queries split into up to 16 chunks, one warp
// each) computes tau_q for every query position.  The paper inserts each newly
// eligible rank into a Fenwick tree and reads the k-th smallest by binary
// lifting.  Here the same value comes from the observation
// that tau_q never increases once k tokens are eligible: a bitset over ranks
// (8 KB for 65536 tokens, in shared memory) marks the inserted ranks, and when a
// newcomer ranks below the current cutoff the cutoff steps down to the next
// marked rank below it -- the warp scans 32 bitset words per ballot.  Over a
// whole row the cutoff moves down at most S ranks, so the scan is O(S) words
// plus O(1) per query.  A chunk's warp starts from the state the scan would have
// reached: it marks the ranks of the tokens already eligible and takes the
// min(k, n)-th marked rank as the cutoff (a popcount prefix over the bitset).
// While fewer than k tokens are eligible every one of them is kept, so tau_q is
// the largest inserted rank (-1 while none is).
#include <algorithm>

#include "kvpop_internal.cuh"

namespace kvpop {
namespace {

constexpr int RK_NT = 512;
constexpr int RK_NW = RK_NT / 32;
constexpr int CUT_MAX_WARPS = 16;

struct RankArgs {
  const float* prio;         // [n_rows][S]
  const int32_t* len;        // [n_rows / rows_per_len] or nullptr (every row has S tokens)
  int rows_per_len;
  int tail;                  // trailing positions of a row without a priority (-> -inf)
  int n_rows, S;
  uint32_t* ka;              // workspace: keys / positions, two buffers of [n_rows][S]
  int32_t* pa;
  uint32_t* kb;
  int32_t* pb;
  int32_t* rank;             // [n_rows][S]
  int32_t* order;            // [n_rows][S] position of each rank (inverse of rank; the pb buffer)
};

// Ascending key = descending priority; NaN -> -inf, -0 -> +0 (as the decode scores).
__device__ __forceinline__ uint32_t rank_key(float f) {
  if (f != f) f = -INFINITY;
  f = __fadd_rn(f, 0.0f);
  const uint32_t b = __float_as_uint(f);
  const uint32_t o = (b & 0x80000000u) ? ~b : (b | 0x80000000u);
  return ~o;
}

__device__ __forceinline__ int row_length(const int32_t* len, int rows_per_len, int row, int S) {
  if (!len) return S;
  return max(0, min(len[row / rows_per_len], S));
}

__global__ void __launch_bounds__(RK_NT) rank_kernel(RankArgs a) {
  __shared__ uint32_t hist[4][256];
  __shared__ uint32_t base[256];
  __shared__ uint32_t cnt[RK_NW][256];
  const int row = blockIdx.x;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int S = a.S;
  const int L = row_length(a.len, a.rows_per_len, row, S);
  const int nsc = max(L - a.tail, 0);
  const size_t ro = (size_t)row * S;
  const float* prio = a.prio + ro;
  const uint32_t lt_mask = (1u << lane) - 1u;
  const uint32_t neg_inf_key = rank_key(-INFINITY);

  for (int i = tid; i < 4 * 256; i += RK_NT) (&hist[0][0])[i] = 0;
  __syncthreads();
  // histograms of all four digits, warp-aggregated per digit value
  for (int i0 = 0; i0 < L; i0 += RK_NT) {
    const int i = i0 + tid;
    const bool ok = i < L;
    const uint32_t key = ok ? (i < nsc ? rank_key(prio[i]) : neg_inf_key) : 0u;
#pragma unroll
    for (int p = 0; p < 4; ++p) {
      const uint32_t dig = ok ? ((key >> (8 * p)) & 255u) : 256u;
      const uint32_t peers = __match_any_sync(0xffffffffu, dig);
      if (ok && (__ffs(peers) - 1) == lane) atomicAdd(&hist[p][dig], (uint32_t)__popc(peers));
    }
  }
  __syncthreads();

  for (int p = 0; p < 4; ++p) {
    // bucket bases: exclusive prefix of the digit histogram (8 warps x 32 digits)
    if (tid < 256) {
      const uint32_t h = hist[p][tid];
      uint32_t x = h;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
      }
      cnt[0][tid] = x;          // inclusive within the warp's 32 digits (scratch)
    }
    __syncthreads();
    if (tid < 256) {
      uint32_t off = 0;
      for (int w = 0; w < (tid >> 5); ++w) off += cnt[0][w * 32 + 31];
      base[tid] = off + cnt[0][tid] - hist[p][tid];
    }
    __syncthreads();
    const uint32_t* sk = (p == 1) ? a.ka + ro : (p == 2) ? a.kb + ro : (p == 3) ? a.ka + ro : nullptr;
    const int32_t* sp = (p == 1) ? a.pa + ro : (p == 2) ? a.pb + ro : (p == 3) ? a.pa + ro : nullptr;
    uint32_t* dk = (p == 0 || p == 2) ? a.ka + ro : a.kb + ro;
    int32_t* dp = (p == 0 || p == 2) ? a.pa + ro : a.pb + ro;
    for (int i0 = 0; i0 < L; i0 += RK_NT) {
      const int i = i0 + tid;
      const bool ok = i < L;
      uint32_t key = 0;
      int32_t pos = i;
      if (ok) {
        if (p == 0) {
          key = i < nsc ? rank_key(prio[i]) : neg_inf_key;
        } else {
          key = sk[i];
          pos = sp[i];
        }
      }
      const uint32_t dig = ok ? ((key >> (8 * p)) & 255u) : 256u;
      for (int j = lane; j < 256; j += 32) cnt[warp][j] = 0;
      __syncwarp();
      const uint32_t peers = __match_any_sync(0xffffffffu, dig);
      const uint32_t within = __popc(peers & lt_mask);
      if (ok && within == 0) cnt[warp][dig] = __popc(peers);
      __syncthreads();
      if (tid < 256) {
        uint32_t run = base[tid];
        for (int w = 0; w < RK_NW; ++w) {
          const uint32_t c = cnt[w][tid];
          cnt[w][tid] = run;
          run += c;
        }
        base[tid] = run;
      }
      __syncthreads();
      if (ok) {
        const uint32_t dst = cnt[warp][dig] + within;
        if (p < 3) {
          dk[dst] = key;
          dp[dst] = pos;
        } else {
          a.rank[ro + pos] = (int32_t)dst;
          a.order[ro + dst] = pos;          // pb is free in the last pass
        }
      }
      __syncwarp();
    }
    __syncthreads();     // this pass's global writes are visible to the next pass
  }
  for (int i = L + tid; i < S; i += RK_NT) a.rank[ro + i] = -1;
}

struct CutArgs {
  const int32_t* rank;       // [n_rows][S]
  const int32_t* len;
  int rows_per_len;
  int n_rows, S, s, w, k;
  int32_t* tau;              // [n_rows][S]
};

// Largest marked rank below r (one exists whenever this is called).
__device__ __forceinline__ int marked_below(const uint32_t* bits, int r, int lane) {
  const int wi = r >> 5;
  const uint32_t m = bits[wi] & ((1u << (r & 31)) - 1u);
  if (m) return (wi << 5) + 31 - __clz(m);
  for (int top = wi - 1; top >= 0; top -= 32) {
    const int idx = top - lane;
    const uint32_t v = idx >= 0 ? bits[idx] : 0u;
    const uint32_t bal = __ballot_sync(0xffffffffu, v != 0u);
    if (bal) {
      const int l = __ffs(bal) - 1;
      const uint32_t vs = __shfl_sync(0xffffffffu, v, l);
      return ((top - l) << 5) + 31 - __clz(vs);
    }
  }
  return -1;
}

// Smallest marked rank whose count of marked ranks at or below it reaches c
// (c >= 1 and at least c ranks marked); warp-collective.
__device__ __forceinline__ int kth_marked(const uint32_t* bits, int words, int c, int lane) {
  int base = 0;
  for (int w0 = 0; w0 < words; w0 += 32) {
    const int wi = w0 + lane;
    const uint32_t v = wi < words ? bits[wi] : 0u;
    const int cnt = __popc(v);
    int incl = cnt;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    const int total = __shfl_sync(0xffffffffu, incl, 31);
    if (base + total >= c) {
      const uint32_t hit = __ballot_sync(0xffffffffu, base + incl >= c);
      const int l = __ffs(hit) - 1;
      uint32_t word = __shfl_sync(0xffffffffu, v, l);
      int need = c - (base + __shfl_sync(0xffffffffu, incl - cnt, l));
      int bit = 0;
      for (; bit < 32; ++bit) {
        if ((word >> bit) & 1u) {
          if (--need == 0) break;
        }
      }
      return (w0 + l) * 32 + bit;
    }
    base += total;
  }
  return -1;
}

// One CTA per row; warp c takes the queries [c * chunk, (c + 1) * chunk).  It first
// rebuilds the state the scan has just before its first query -- the bitset of
// the ranks inserted so far and the cutoff, the min(k, n)-th smallest of them --
// then runs the same per-query update, so every chunk's cutoffs equal those of
// one scan over the whole row.
__global__ void cutoff_kernel(CutArgs a, int chunk) {
  extern __shared__ uint32_t bitsets[];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int row = blockIdx.x;
  const int S = a.S, words = (S + 31) >> 5;
  const int L = row_length(a.len, a.rows_per_len, row, S);
  const int32_t* rank = a.rank + (size_t)row * S;
  int32_t* tau_out = a.tau + (size_t)row * S;
  if (warp == 0 && blockIdx.y == 0)
    for (int i = L + lane; i < S; i += 32) tau_out[i] = -1;
  // chunk blockIdx.y * warps + warp of the row: the row's chunks are spread over
  // gridDim.y CTAs so that short batches still fill the GPU
  const int qa = (blockIdx.y * (blockDim.x >> 5) + warp) * chunk;
  if (qa >= L) return;
  const int qb = min(qa + chunk, L);
  uint32_t* bits = bitsets + (size_t)warp * words;
  for (int i = lane; i < words; i += 32) bits[i] = 0u;
  __syncwarp();
  const int s = a.s, w = a.w, k = a.k;
  // tokens inserted before query qa: positions s .. qa - 1 - w
  int cnt = 0;
  for (int t = s + lane; t <= qa - 1 - w; t += 32) {
    const int r = rank[t];
    if (r >= 0 && r < S) {
      atomicOr(&bits[r >> 5], 1u << (r & 31));
      ++cnt;
    }
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, o);
  __syncwarp();
  int n = cnt;
  int tau = n > 0 ? kth_marked(bits, words, min(k, n), lane) : -1;
  for (int q0 = qa; q0 < qb; q0 += 32) {
    const int tl = q0 + lane - w;
    int r_l = -1;
    if (tl >= s && tl < L) r_l = rank[tl];
    int mine = -1;
    const int nq = min(32, qb - q0);
    for (int j = 0; j < nq; ++j) {
      const int t = q0 + j - w;
      if (t >= s) {
        const int r = __shfl_sync(0xffffffffu, r_l, j);
        if (r >= 0 && r < S) {
          if (lane == 0) bits[r >> 5] |= 1u << (r & 31);
          __syncwarp();
          ++n;
          if (n <= k) tau = max(tau, r);
          else if (r < tau) tau = marked_below(bits, tau, lane);
        }
      }
      if (lane == j) mine = (k > 0) ? tau : -1;
    }
    if (lane < nq) tau_out[q0 + lane] = mine;
  }
}

}  // namespace

size_t topk_workspace_bytes(int n_rows, int S) {
  return (size_t)n_rows * (size_t)S * 16 + 1024;
}

const int32_t* topk_order(const void* workspace, int n_rows, int S) {
  const size_t n = (size_t)n_rows * S;
  const size_t al = (n * 4 + 255) & ~size_t(255);
  return reinterpret_cast<const int32_t*>(static_cast<const char*>(workspace) + 3 * al);
}

cudaError_t launch_topk(const float* prio, const int32_t* len, int rows_per_len, int tail,
                        int n_rows, int S, int s, int w, int k, int32_t* rank, int32_t* tau,
                        int32_t* order, void* workspace, cudaStream_t stream) {
  if (n_rows <= 0 || S <= 0) return cudaSuccess;
  const size_t n = (size_t)n_rows * S;
  char* ws = static_cast<char*>(workspace);
  auto al = [](size_t x) { return (x + 255) & ~size_t(255); };
  RankArgs ra{prio, len, rows_per_len, tail, n_rows, S,
              reinterpret_cast<uint32_t*>(ws), reinterpret_cast<int32_t*>(ws + al(n * 4)),
              reinterpret_cast<uint32_t*>(ws + 2 * al(n * 4)),
              reinterpret_cast<int32_t*>(ws + 3 * al(n * 4)), rank,
              order ? order : reinterpret_cast<int32_t*>(ws + 3 * al(n * 4))};
  rank_kernel<<<n_rows, RK_NT, 0, stream>>>(ra);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  // chunks per row: up to 16 warps, each with its own bitset of S bits in shared memory
  const size_t words_bytes = (size_t)((S + 31) / 32) * 4;
  const int nch = (int)std::max<size_t>(1, std::min<size_t>(CUT_MAX_WARPS, (200 * 1024) / words_bytes));
  // CTAs per row: enough for about two per SM, while every chunk keeps >= 512 queries
  int dev = 0, sms = 152;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int want = std::max(1, (2 * sms + n_rows - 1) / n_rows);
  const int split = std::max(1, std::min(want, S / (nch * 512)));
  const int chunk = (S + nch * split - 1) / (nch * split);
  const size_t smem = (size_t)nch * words_bytes;
  e = raise_smem_limit(cutoff_kernel, smem);
  if (e != cudaSuccess) return e;
  CutArgs ca{rank, len, rows_per_len, n_rows, S, s, w, k, tau};
  cutoff_kernel<<<dim3(n_rows, split), nch * 32, smem, stream>>>(ca, chunk);
  return cudaGetLastError();
}

}  // namespace kvpop
