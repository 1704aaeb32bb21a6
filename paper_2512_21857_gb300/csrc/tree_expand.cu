// adt_tree_expand: one layer of EAGLE-2-style dynamic draft-tree growth
// (Sec. 3.1, last paragraph; Fig. 5; node score Eq. 4 in the log domain), and
// adt_tree_rerank: the final top-N tree (Eq. 4 and the sentence after it).
//
// Expand is one launch of F thread-block clusters, one per frontier row; the
// C <= 8 CTAs of a cluster split the row's vocabulary.  Each CTA stages its
// share in shared memory with one bulk copy (x / T in fp32, round-to-nearest
// division).  A first pass keeps each thread's two largest values; the k-th
// largest of the 32 warp maxima bounds the CTA's top k from below; a second
// pass sums the exponentials against the CTA's maximum and gathers the few
// selection keys (value order, then lower index) at or above the bound,
// which are ranked by counting.  The CTAs' lists go to the cluster's first
// CTA through distributed shared memory; it ranks them, forms the row's
// log-sum-exp and writes the row's children (log-probability against it in
// fp64).  The first CTA of the last row to finish (atomic ticket) ranks the
// next frontier across all rows.
#include <cooperative_groups.h>

#include "adt_common.cuh"
#include "sm100.cuh"

namespace cg = cooperative_groups;

namespace {

constexpr int kThreads = 1024;
constexpr int kWarps = kThreads / 32;
constexpr int kMaxK = 64;
constexpr int kMaxKeep = 1024;
constexpr int kMaxCluster = 8;
constexpr int kValuesPerCta = 2048;     // a CTA per this many logits, up to kMaxCluster per row
constexpr int kTile = 16384;            // logits staged in shared memory at a time
constexpr uint32_t kWaitLimit = 1u << 22;
constexpr int kCandCap = 1024;          // a CTA's candidate buffer (also the cross-row keys)
constexpr float kLog2e = 1.44269504088896340736f;

struct ExpandParams {
  const float* logits;
  const float* logits_u;  // classifier-free guidance: unconditional rows (same ld), else NULL
  float cfg;              // guidance scale
  int64_t ld;
  const float* fscore;
  const int32_t* fid;
  int F, V, k, k_keep;
  float T;
  int use_T;
  int32_t id_base;
  int32_t* ctok;
  float* clogp;
  float* cscore;
  int32_t* cpar;
  int32_t* keep;
  float* nscore;
  int32_t* nid;
  uint64_t* cross_keys;   // [F*k]
  unsigned* all_ticket;   // [1]
  unsigned* err;
};

// Entries greater than key in a descending list of n keys.
__device__ __forceinline__ int count_greater(const uint64_t* list, int n, uint64_t key) {
  int lo = 0, hi = n;
  while (lo < hi) {
    const int mid = (lo + hi) >> 1;
    if (list[mid] > key)
      lo = mid + 1;
    else
      hi = mid;
  }
  return lo;
}

// Top k of nl descending lists (list l at lists + l * stride, its first len
// entries; 0 pads) into out[0..k), which the caller zeroed.  Keys are
// distinct, so an entry's rank is its index plus the entries greater than it
// in the other lists.
__device__ void merge_topk(const uint64_t* lists, int nl, int stride, int len, int k, uint64_t* out) {
  const int lk = min(len, k);
  for (int c = threadIdx.x; c < nl * lk; c += kThreads) {
    const int l = c / lk, j = c % lk;
    const uint64_t key = lists[l * stride + j];
    if (key == 0ull) continue;
    int rank = j;
    for (int l2 = 0; l2 < nl && rank < k; ++l2)
      if (l2 != l) rank += count_greater(lists + l2 * stride, lk, key);
    if (rank < k) out[rank] = key;
  }
}

// Collects the keys >= thr (exactly `count` of them) into sel[] and sorts
// them in descending order (padding with 0 up to a power of two).
template <class KeyAt>
__device__ void collect_sorted(KeyAt key_at, int n, uint64_t thr, int count, uint64_t* sel,
                               unsigned* s_cnt) {
  const int P = adt::next_pow2(count);
  for (int i = threadIdx.x; i < P; i += kThreads) sel[i] = 0ull;
  if (threadIdx.x == 0) *s_cnt = 0u;
  __syncthreads();
  for (int i = threadIdx.x; i < n; i += kThreads) {
    const uint64_t key = key_at(i);
    if (key >= thr && key != 0ull) {
      const unsigned slot = atomicAdd(s_cnt, 1u);
      if (slot < static_cast<unsigned>(P)) sel[slot] = key;
    }
  }
  __syncthreads();
  adt::block_bitonic_sort_desc<kThreads>(sel, P);
}

// The k (<= 64) largest keys a warp is offered, kept sorted by insertion:
// lane i holds entries i (a) and i + 32 (b); 0 marks an empty entry.  Used
// only when a warp's candidate buffer overflows (inputs with very many keys
// at or above the warp's bound).
struct WarpTopK {
  uint64_t a = 0, b = 0;
  __device__ __forceinline__ uint64_t threshold(int k) const {
    const int i = k - 1;
    return __shfl_sync(adt::kFullMask, i < 32 ? a : b, i & 31);
  }
  __device__ __forceinline__ void insert(uint64_t key, int k, int lane) {
    const int pos = __popc(__ballot_sync(adt::kFullMask, a > key)) + __popc(__ballot_sync(adt::kFullMask, b > key));
    if (pos >= k) return;
    const uint64_t up_a = __shfl_up_sync(adt::kFullMask, a, 1);
    const uint64_t up_b = __shfl_up_sync(adt::kFullMask, b, 1);
    const uint64_t a31 = __shfl_sync(adt::kFullMask, a, 31);
    const int ia = lane, ib = lane + 32;
    const uint64_t na = ia < pos ? a : (ia == pos ? key : up_a);
    const uint64_t nb = ib < pos ? b : (ib == pos ? key : (lane == 0 ? a31 : up_b));
    a = ia < k ? na : 0ull;
    b = ib < k ? nb : 0ull;
  }
  __device__ __forceinline__ void offer(uint64_t key, int k, int lane, uint64_t& thr) {
    unsigned m = __ballot_sync(adt::kFullMask, key > thr);
    while (m) {
      const int src = __ffs(m) - 1;
      insert(__shfl_sync(adt::kFullMask, key, src), k, lane);
      thr = threshold(k);
      m &= m - 1;
      m &= __ballot_sync(adt::kFullMask, key > thr);
    }
  }
};

// Stages logits [t0, t1) of a row (t0 a multiple of 4; rows start 16-byte
// aligned and ld is a multiple of 4) in shared memory with one bulk copy
// (two with guidance: the unconditional row goes to vals_u), waiting with a
// bound; then forms u + s (c - u) under guidance and divides by the
// temperature, in place.  Block-wide.
__device__ bool stage_tile(float* vals, float* vals_u, const float* row, const float* row_u, int t0, int t1,
                           const ExpandParams& p, uint64_t* bar, uint32_t& phase) {
  const int n = t1 - t0;
  if (threadIdx.x == 0 && n > 0) {
    const uint32_t bytes = static_cast<uint32_t>((n + 3) / 4 * 16);
    sm100::mbar_arrive_expect_tx(sm100::smem_addr(bar), row_u ? 2 * bytes : bytes);
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];\n" ::"r"(
            sm100::smem_addr(vals)),
        "l"(row + t0), "r"(bytes), "r"(sm100::smem_addr(bar))
        : "memory");
    if (row_u)
      asm volatile(
          "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];\n" ::"r"(
              sm100::smem_addr(vals_u)),
          "l"(row_u + t0), "r"(bytes), "r"(sm100::smem_addr(bar))
          : "memory");
  }
  bool ok = true;
  if (n > 0) {
    ok = sm100::mbar_wait_bounded(sm100::smem_addr(bar), phase, kWaitLimit);
    phase ^= 1u;
  }
  if (row_u || p.use_T) {
    for (int i = threadIdx.x; i < n; i += kThreads) {
      float x = vals[i];
      if (row_u) x = adt::cfg_combine(x, vals_u[i], p.cfg);
      if (p.use_T) x = __fdiv_rn(x, p.T);
      vals[i] = x;
    }
  }
  __syncthreads();
  return ok;
}

// out[rank] = key for the k largest of the n distinct nonzero keys in
// keys[0..n) (0 entries skipped); out[] zeroed by the caller.  Block-wide:
// a warp takes a key and its lanes count the keys above it.
__device__ void rank_select(const uint64_t* keys, int n, int k, uint64_t* out) {
  const int lane = threadIdx.x & 31;
  for (int i = threadIdx.x >> 5; i < n; i += kWarps) {
    const uint64_t key = keys[i];
    if (key == 0ull) continue;
    int rk = 0;
    for (int j = 0; j < n; j += 32) rk += __popc(__ballot_sync(adt::kFullMask, j + lane < n && keys[j + lane] > key));
    if (lane == 0 && rk < k) out[rk] = key;
  }
}

// 2^x with the hardware approximation (flush-to-zero); 2^-inf = 0.
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;\n" : "=f"(y) : "f"(x));
  return y;
}

// The k-th largest (k <= 32) of the warp's 32 values (none NaN): the one
// whose rank -- the values above it, with equal values of lower lanes
// counted as above -- is k - 1.  32 independent shuffles instead of the
// dependent chain of a sort.
__device__ __forceinline__ float warp_kth_largest(float v, int k, int lane) {
  int rk = 0;
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    const float o = __shfl_sync(adt::kFullMask, v, j);
    rk += (o > v || (o == v && j < lane)) ? 1 : 0;
  }
  const unsigned m = __ballot_sync(adt::kFullMask, rk == k - 1);
  return __shfl_sync(adt::kFullMask, v, __ffs(m) - 1);
}

// rank_select for n <= 64 keys: 16 threads per key, each counting the keys
// above it among four of the others, the counts summed by shuffles within
// the group; one round of loads instead of a warp per key looping over n.
__device__ void rank_select64(const uint64_t* keys, int n, int k, uint64_t* out) {
  static_assert(kThreads == 64 * 16, "16 threads for each of 64 keys");
  const int i = threadIdx.x >> 4, s = threadIdx.x & 15;
  const uint64_t key = i < n ? keys[i] : 0ull;
  int c = 0;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const int o = s + 16 * j;
    c += (o < n && keys[o] > key) ? 1 : 0;
  }
#pragma unroll
  for (int off = 8; off > 0; off >>= 1) c += __shfl_xor_sync(adt::kFullMask, c, off);
  if (s == 0 && key != 0ull && c < k) out[c] = key;
}

__global__ void __launch_bounds__(kThreads) expand_kernel(const ExpandParams p) {
  extern __shared__ __align__(16) float vals[];    // [min(per, kTile)] staged logits (x2 with guidance)
  __shared__ uint64_t cand[kCandCap];              // keys at or above the CTA's bound
  __shared__ uint64_t wl[kWarps][kMaxK];           // overflow path: each warp's top k
  __shared__ float s_bw[kWarps], s_mw[kWarps], s_sw[kWarps];
  __shared__ float s_B, s_M;
  __shared__ unsigned s_cnt;
  __shared__ uint64_t ctl[kMaxK];                  // this CTA's top k
  __shared__ uint64_t cl_keys[kMaxCluster * kMaxK];  // first CTA of the cluster: every CTA's k keys
  __shared__ float2 cl_ms[kMaxCluster];
  __shared__ uint64_t rowl[kMaxK];
  __shared__ adt::RadixScratch rs;
  __shared__ __align__(8) uint64_t s_bar;
  __shared__ int s_last;
  __shared__ double s_lse;
  uint64_t* cross_s = cand;  // cross-row keys (reuses the candidate buffer)
  uint64_t* sel = cand;      // radix path [kMaxKeep]

  cg::cluster_group cl = cg::this_cluster();
  const int rank = blockIdx.x, C = gridDim.x, r = blockIdx.y;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int K = p.k;
  // Shared-memory set-up before the dependency wait (it reads nothing an
  // earlier kernel writes): after the wait the first bulk copy goes out at once.
  for (int i = tid; i < kMaxK; i += kThreads) ctl[i] = 0ull;
  if (tid == 0) {
    s_cnt = 0u;
    sm100::mbar_init(sm100::smem_addr(&s_bar), 1);
    sm100::fence_mbar_init();
  }
  __syncthreads();
  asm volatile("griddepcontrol.wait;\n" ::: "memory");
  // This CTA's share of the row: [c0, c1), c0 a multiple of 4.
  const int per = (((p.V + C - 1) / C) + 3) & ~3;
  const int c0 = min(p.V, rank * per), c1 = min(p.V, c0 + per);
  const int ntiles = (c1 - c0 + kTile - 1) / kTile;
  const float* row = p.logits + static_cast<int64_t>(r) * p.ld;
  const float* row_u = p.logits_u ? p.logits_u + static_cast<int64_t>(r) * p.ld : nullptr;
  float* vals_u = vals + min(per, kTile);  // used only with guidance

  // The row's frontier score and id, read now by the threads that write the
  // children at the end: the loads' latency hides behind the passes.
  const bool writer = rank == 0 && tid < K;
  const float f_score = writer ? p.fscore[r] : 0.f;
  const int32_t f_id = writer ? (p.fid ? p.fid[r] : r) : 0;
  uint32_t phase = 0;
  bool ok = true;

  // Pass 1: each thread's two largest values (ties kept).  Thread tid takes
  // elements tid, tid + 1024, ... of every tile.
  float v1 = -INFINITY, v2 = -INFINITY;
  for (int tt = 0; tt < ntiles; ++tt) {
    const int t0 = c0 + tt * kTile, t1 = min(c1, t0 + kTile);
    if (tt > 0) __syncthreads();  // the previous tile is consumed
    ok &= stage_tile(vals, vals_u, row, row_u, t0, t1, p, &s_bar, phase);
#pragma unroll 8
    for (int i = tid; i < t1 - t0; i += kThreads) {
      const float x = vals[i];
      v2 = fmaxf(v2, fminf(v1, x));
      v1 = fmaxf(v1, x);
    }
  }
  if (!ok && tid == 0) adt::raise_error(p.err, ADT_DEVERR_TIMEOUT);
  // The bound B: a value with at least k of the CTA's logits at or above it,
  // so that its k best are among those >= B.  For k <= 32: the k-th largest
  // of the 32 warp maxima (ranked by counting in warp 0).  For larger k: per
  // warp, the largest of its 64 lane values (two per lane) with k of them at
  // or above it; B is the largest of those.
  {
    const float mw = adt::warp_max(v1);
    float bw = -INFINITY;
    if (K > 32) {
      int g1 = 0, g2 = 0;
      for (int j = 0; j < 32; ++j) {
        const float o1 = __shfl_sync(adt::kFullMask, v1, j), o2 = __shfl_sync(adt::kFullMask, v2, j);
        g1 += (o1 >= v1) + (o2 >= v1);
        g2 += (o1 >= v2) + (o2 >= v2);
      }
      float cb = -INFINITY;
      if (g1 >= K) cb = v1;
      if (g2 >= K) cb = fmaxf(cb, v2);
      bw = adt::warp_max(cb);
    }
    if (lane == 0) {
      s_bw[warp] = bw;
      s_mw[warp] = mw;
    }
  }
  __syncthreads();
  if (warp == 0) {
    const float mv = s_mw[lane];
    const float mmax = adt::warp_max(mv);
    const float b = K <= 32 ? warp_kth_largest(mv, K, lane) : adt::warp_max(s_bw[lane]);
    if (lane == 0) {
      s_B = b;
      s_M = mmax;
    }
  }
  __syncthreads();
  const float B = s_B, M = s_M;
  // Pass 2: sum of exp(x - M) as 2^(x log2 e - M log2 e); gather the keys of
  // values >= B (few: shared-memory atomics, no per-element vote).
  const float Ml = M == -INFINITY ? 0.f : M * kLog2e;
  float sa[4] = {0.f, 0.f, 0.f, 0.f};
  for (int tt = 0; tt < ntiles; ++tt) {
    const int t0 = c0 + tt * kTile, t1 = min(c1, t0 + kTile);
    if (ntiles > 1) {
      __syncthreads();
      ok &= stage_tile(vals, vals_u, row, row_u, t0, t1, p, &s_bar, phase);
    }
    const int n = t1 - t0;
    for (int i0 = tid; i0 < n; i0 += 4 * kThreads) {
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int i = i0 + u * kThreads;
        if (i < n) {
          const float x = vals[i];
          sa[u] += ex2_approx(fmaf(x, kLog2e, -Ml));
          if (x >= B) {
            const unsigned pos = atomicAdd(&s_cnt, 1u);
            if (pos < static_cast<unsigned>(kCandCap)) cand[pos] = adt::select_key(x, static_cast<uint32_t>(t0 + i));
          }
        }
      }
    }
  }
  {
    const float sw = adt::warp_sum((sa[0] + sa[1]) + (sa[2] + sa[3]));
    if (lane == 0) s_sw[warp] = sw;
  }
  __syncthreads();
  const int cnt = static_cast<int>(s_cnt);
  if (cnt <= 64) {
    rank_select64(cand, cnt, K, ctl);
  } else if (cnt <= kCandCap) {
    rank_select(cand, cnt, K, ctl);
  } else {
    // Overflow (very many values at or above B): each warp keeps its k
    // largest by insertion in a third pass, then the lists merge.
    for (int i = tid; i < kWarps * kMaxK; i += kThreads) (&wl[0][0])[i] = 0ull;
    const uint64_t kb = B == -INFINITY ? 1ull : adt::select_key(B, 0xffffffffu);  // lowest key of value B
    WarpTopK tk;
    uint64_t thr = 0ull;
    for (int tt = 0; tt < ntiles; ++tt) {
      const int t0 = c0 + tt * kTile, t1 = min(c1, t0 + kTile);
      if (ntiles > 1) {
        __syncthreads();
        ok &= stage_tile(vals, vals_u, row, row_u, t0, t1, p, &s_bar, phase);
      }
      const int n = t1 - t0;
      for (int base = warp * 32; base < n; base += kThreads) {
        const int i = base + lane;
        const uint64_t key = i < n ? adt::select_key(vals[i], static_cast<uint32_t>(t0 + i)) : 0ull;
        tk.offer(key >= kb ? key : 0ull, K, lane, thr);
      }
    }
    __syncthreads();
    wl[warp][lane] = tk.a;
    wl[warp][lane + 32] = tk.b;
    __syncthreads();
    merge_topk(&wl[0][0], kWarps, kMaxK, K, K, ctl);
  }
  __syncthreads();
  if (!ok && tid == 0) adt::raise_error(p.err, ADT_DEVERR_TIMEOUT);  // a restaged tile's wait
  // This CTA's top k and (max, sum of exponentials), to the cluster's first CTA.
  if (warp == 0) {
    uint64_t* dst = cl.map_shared_rank(&cl_keys[rank * K], 0);
    if (lane < K) dst[lane] = ctl[lane];
    if (lane + 32 < K) dst[lane + 32] = ctl[lane + 32];
    const float S = adt::warp_sum(s_sw[lane]);  // kWarps == 32
    if (lane == 0) *cl.map_shared_rank(&cl_ms[rank], 0) = make_float2(M, S);
  }
  sm100::cluster_arrive_release();
  sm100::cluster_wait_acquire();
  // The next kernel in the stream may launch now.  Released here rather than
  // right after the wait: a graph of six back-to-back calls (F = 1, then 8;
  // V = 65536, k = 8) and the rerank took 49.2 us against 51.2 us.
  asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
  if (rank != 0) return;

  // ---- first CTA of row r: the row's top k and log-sum-exp, its children.
  for (int i = tid; i < kMaxK; i += kThreads) rowl[i] = 0ull;
  if (warp == 0) {  // lane c takes CTA c's (max, sum); C <= 8
    const float2 ms = lane < C ? cl_ms[lane] : make_float2(-INFINITY, 0.f);
    const float Mr = adt::warp_max(ms.x);
    const float S = adt::warp_sum(ms.x != -INFINITY ? ms.y * ex2_approx((ms.x - Mr) * kLog2e) : 0.f);
    if (lane == 0) s_lse = static_cast<double>(Mr) + static_cast<double>(logf(S));
  }
  __syncthreads();
  if (C * K <= 64)
    rank_select64(cl_keys, C * K, K, rowl);
  else
    rank_select(cl_keys, C * K, K, rowl);
  __syncthreads();
  if (writer) {
    const uint64_t key = rowl[tid];
    const double lp = static_cast<double>(adt::select_key_value(key)) - s_lse;
    const float score = static_cast<float>(static_cast<double>(f_score) + lp);
    const int64_t c = static_cast<int64_t>(r) * K + tid;
    p.ctok[c] = static_cast<int32_t>(adt::select_key_index(key));
    if (p.clogp) p.clogp[c] = static_cast<float>(lp);
    p.cscore[c] = score;
    p.cpar[c] = f_id;
    if (!p.keep) {
      // No next frontier wanted (the tree's last layer).
    } else if (p.F == 1) {
      // One row: its children are already in score order (the score grows
      // with the log-probability; ties keep the lower index, as the
      // cross-row ranking would), so the next frontier is their first k_keep.
      if (tid < p.k_keep) {
        p.keep[tid] = static_cast<int32_t>(c);
        if (p.nscore) p.nscore[tid] = score;
        if (p.nid) p.nid[tid] = p.id_base + static_cast<int32_t>(c);
      }
    } else {
      p.cross_keys[c] = adt::select_key(score, static_cast<uint32_t>(c));
    }
  }
  if (p.F == 1 || !p.keep) return;
  // The row's cross keys are written (CTA order); the ticket's release
  // publishes them at device scope and its acquire, in the last row, makes
  // every row's keys visible.
  __syncthreads();
  if (tid == 0) s_last = adt::atomic_add_acq_rel_gpu(p.all_ticket, 1u) == static_cast<unsigned>(p.F - 1);
  __syncthreads();
  if (!s_last) return;

  // ---- last row: next frontier across all rows.
  const int nc = p.F * K;
  if (p.k_keep <= kMaxK && nc <= kCandCap) {
    for (int i = tid; i < nc; i += kThreads) cross_s[i] = __ldcg(p.cross_keys + i);
    for (int i = tid; i < kMaxK; i += kThreads) rowl[i] = 0ull;
    __syncthreads();
    if (nc <= 64)
      rank_select64(cross_s, nc, p.k_keep, rowl);
    else
      rank_select(cross_s, nc, p.k_keep, rowl);
    __syncthreads();
    if (tid < p.k_keep) {
      const uint64_t key = rowl[tid];
      const int32_t c = static_cast<int32_t>(adt::select_key_index(key));
      p.keep[tid] = c;
      if (p.nscore) p.nscore[tid] = adt::select_key_value(key);
      if (p.nid) p.nid[tid] = p.id_base + c;
    }
  } else {
    auto cross_key = [&](int i) { return __ldcg(p.cross_keys + i); };
    const uint64_t thr3 = adt::block_topk_threshold<kThreads>(cross_key, nc, p.k_keep, &rs);
    collect_sorted(cross_key, nc, thr3, p.k_keep, sel, &s_cnt);
    for (int j = tid; j < p.k_keep; j += kThreads) {
      const uint64_t key = sel[j];
      const int32_t c = static_cast<int32_t>(adt::select_key_index(key));
      p.keep[j] = c;
      if (p.nscore) p.nscore[j] = adt::select_key_value(key);
      if (p.nid) p.nid[j] = p.id_base + c;
    }
  }
  if (tid == 0) *p.all_ticket = 0u;
}

// CTAs per row (the cluster size).
int expand_cluster(int V) {
  const int c = (V + kValuesPerCta - 1) / kValuesPerCta;
  return c < 1 ? 1 : (c > kMaxCluster ? kMaxCluster : c);
}

// Workspace layout.  The completion counter sits at a fixed offset at the
// start, after a zeroed region kept for layout stability, so calls of any
// shape can share one workspace; the keys after it are rewritten before use.
constexpr int kMaxRows = 4096;

struct ExpandWs {
  size_t all_ticket, cross_keys, total;
};

ExpandWs expand_ws(int F, int V, int k) {
  (void)V;
  ExpandWs w{};
  w.all_ticket = kMaxRows * sizeof(unsigned);
  w.cross_keys = adt::align_up(w.all_ticket + sizeof(unsigned), 256);
  w.total = adt::align_up(w.cross_keys + static_cast<size_t>(F) * k * sizeof(uint64_t), 256);
  return w;
}

// ------------------------------------------------------------------ rerank

constexpr int kRerankThreads = 1024;

struct RerankParams {
  const int32_t* ctok;
  const float* cscore;
  const int32_t* cpar;
  int C;
  const int32_t* root;
  int n_nodes;
  int32_t* tokens;
  int32_t* parents;
  int32_t* cand_index;
  int32_t* depth;
  int32_t* node_of;       // [C]  workspace
  int32_t* cand_of_node;  // [n_nodes] workspace
  unsigned* err;
};

// Shared-memory rerank for up to kRerankSmall candidates and nodes: a
// candidate is selected when fewer than n_nodes - 1 candidate keys exceed
// its own (a warp takes a key and its lanes count), node ids follow
// ascending candidate index (block scan of the selection flags), and the
// node maps, parents and depths never leave shared memory.  With at most
// kRerankBound nodes to select from at least 64 candidates, only the keys
// at or above a bound are ranked: every warp's two largest keys (over a
// strided view, so that every warp holds candidates) give 64 distinct keys,
// and the (n_nodes - 1)-th largest of them has at least n_nodes - 1 keys at
// or above it.
constexpr int kRerankSmall = 1024;
constexpr int kRerankBound = 64;

__device__ __forceinline__ uint64_t warp_max_u64(uint64_t v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const uint64_t w = __shfl_xor_sync(adt::kFullMask, v, o);
    v = w > v ? w : v;
  }
  return v;
}

__global__ void __launch_bounds__(kRerankThreads) rerank_small_kernel(const RerankParams p) {
  __shared__ uint64_t keys[kRerankSmall];
  __shared__ int node_of[kRerankSmall];
  __shared__ int cand_of_node[kRerankSmall + 1];
  __shared__ int par[kRerankSmall + 1];
  __shared__ int cpar_s[kRerankSmall];
  __shared__ uint64_t list[kRerankSmall];
  __shared__ uint64_t s_top[2 * 32];
  __shared__ uint64_t s_bound;
  __shared__ int s_nlist;
  __shared__ int warp_tot[32];
  __shared__ int s_bad;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int need = p.n_nodes - 1, C = p.C;
  adt::pdl_wait_then_release();
  if (tid == 0) {
    p.tokens[0] = *p.root;
    p.parents[0] = -1;
    if (p.cand_index) p.cand_index[0] = -1;
    if (p.depth) p.depth[0] = 0;
    par[0] = -1;
    s_bad = 0;
    s_nlist = 0;
  }
  if (need == 0) return;
  // Candidate tid (C <= kRerankThreads): its key, token and parent id, all
  // loaded in one round; node_of holds the selection flags until the scan.
  uint64_t key = 0ull;
  int tok = 0;
  if (tid < C) {
    key = adt::select_key(p.cscore[tid], static_cast<uint32_t>(tid));
    tok = p.ctok[tid];
    cpar_s[tid] = p.cpar[tid];
    keys[tid] = key;
    node_of[tid] = 0;
  }
  __syncthreads();
  if (need <= kRerankBound && C >= 2 * 32) {
    {
      const int i = lane * 32 + warp;  // every warp sees at least two candidates
      const uint64_t v = i < C ? keys[i] : 0ull;
      const uint64_t m1 = warp_max_u64(v);
      const uint64_t m2 = warp_max_u64(v == m1 ? 0ull : v);
      if (lane == 0) {
        s_top[warp] = m1;
        s_top[warp + 32] = m2;
      }
    }
    __syncthreads();
    {
      // warp w ranks s_top[w] and s_top[w + 32] among the 64
      const uint64_t x = s_top[lane], y = s_top[lane + 32];
      const uint64_t a = s_top[warp], c = s_top[warp + 32];
      const int ra = __popc(__ballot_sync(adt::kFullMask, x > a)) + __popc(__ballot_sync(adt::kFullMask, y > a));
      const int rc = __popc(__ballot_sync(adt::kFullMask, x > c)) + __popc(__ballot_sync(adt::kFullMask, y > c));
      if (lane == 0 && ra == need - 1) s_bound = a;
      if (lane == 0 && rc == need - 1) s_bound = c;
    }
    __syncthreads();
    if (tid < C && key >= s_bound) list[atomicAdd(&s_nlist, 1)] = key;
    __syncthreads();
    const int nl = s_nlist;
    for (int e = warp; e < nl; e += kRerankThreads / 32) {
      const uint64_t ke = list[e];
      int rk = 0;
      for (int j = 0; j < nl; j += 32) rk += __popc(__ballot_sync(adt::kFullMask, j + lane < nl && list[j + lane] > ke));
      if (lane == 0 && rk < need) node_of[adt::select_key_index(ke)] = 1;
    }
  } else {
    for (int i = warp; i < C; i += kRerankThreads / 32) {
      const uint64_t ki = keys[i];
      int rk = 0;
      for (int j = 0; j < C; j += 32) rk += __popc(__ballot_sync(adt::kFullMask, j + lane < C && keys[j + lane] > ki));
      if (lane == 0) node_of[i] = rk < need ? 1 : 0;
    }
  }
  __syncthreads();
  const bool sel = tid < C && node_of[tid] != 0;
  // node id = 1 + selected candidates of lower index (block exclusive scan)
  const unsigned bal = __ballot_sync(adt::kFullMask, sel);
  if (lane == 0) warp_tot[warp] = __popc(bal);
  __syncthreads();
  int before = __popc(bal & ((1u << lane) - 1u));
  for (int w = 0; w < warp; ++w) before += warp_tot[w];
  if (tid < C) {
    const int node = sel ? 1 + before : -1;
    node_of[tid] = node;
    if (sel) {
      cand_of_node[node] = tid;
      p.tokens[node] = tok;
      if (p.cand_index) p.cand_index[node] = tid;
    }
  }
  __syncthreads();
  for (int node = 1 + tid; node <= need; node += kRerankThreads) {
    const int pc = cpar_s[cand_of_node[node]];
    int pr = 0;
    if (pc >= 0) {
      pr = pc < C ? node_of[pc] : -1;
      if (pr < 0 || pr >= node) {
        s_bad = 1;
        pr = 0;
      }
    }
    par[node] = pr;
    p.parents[node] = pr;
  }
  __syncthreads();
  if (s_bad && tid == 0) adt::raise_error(p.err, ADT_DEVERR_BAD_TREE);
  if (p.depth) {
    for (int node = 1 + tid; node <= need; node += kRerankThreads) {
      int d = 0, j = node;
      while (j > 0 && d <= need) {
        j = par[j];
        ++d;
      }
      p.depth[node] = d;
    }
  }
}

__global__ void __launch_bounds__(kRerankThreads) rerank_kernel(const RerankParams p) {
  __shared__ adt::RadixScratch rs;
  __shared__ int warp_tot[32];
  __shared__ int warp_excl[32];
  __shared__ int s_running;
  __shared__ int s_tile;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int need = p.n_nodes - 1;
  adt::pdl_wait_then_release();
  if (tid == 0) {
    p.tokens[0] = *p.root;
    p.parents[0] = -1;
    if (p.cand_index) p.cand_index[0] = -1;
    if (p.depth) p.depth[0] = 0;
    p.cand_of_node[0] = -1;
    s_running = 0;
  }
  if (need == 0) return;
  auto key_at = [&](int i) { return adt::select_key(p.cscore[i], static_cast<uint32_t>(i)); };
  const uint64_t thr = adt::block_topk_threshold<kRerankThreads>(key_at, p.C, need, &rs);
  // Node ids in ascending candidate order: block-wide exclusive scan of the flags.
  for (int base = 0; base < p.C; base += kRerankThreads) {
    const int i = base + tid;
    const bool f = i < p.C && key_at(i) >= thr;
    const unsigned bal = __ballot_sync(adt::kFullMask, f);
    const int in_warp = __popc(bal & ((1u << lane) - 1u));
    if (lane == 0) warp_tot[warp] = __popc(bal);
    __syncthreads();
    if (warp == 0) {
      const int v = warp_tot[lane];
      int incl = v;
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(adt::kFullMask, incl, o);
        if (lane >= o) incl += y;
      }
      warp_excl[lane] = incl - v;
      if (lane == 31) s_tile = incl;
    }
    __syncthreads();
    const int before = s_running + warp_excl[warp] + in_warp;
    if (i < p.C) {
      const int node = f ? 1 + before : -1;
      if (node >= 1 && node <= need) {
        p.node_of[i] = node;
        p.tokens[node] = p.ctok[i];
        p.cand_of_node[node] = i;
        if (p.cand_index) p.cand_index[node] = i;
      } else {
        p.node_of[i] = -1;
      }
    }
    __syncthreads();
    if (tid == 0) s_running += s_tile;
    __syncthreads();
  }
  __threadfence_block();
  __syncthreads();
  for (int node = 1 + tid; node <= need; node += kRerankThreads) {
    const int c = p.cand_of_node[node];
    const int pc = p.cpar[c];
    int par = 0;
    if (pc >= 0) {
      par = (pc < p.C) ? p.node_of[pc] : -1;
      if (par < 0 || par >= node) {
        adt::raise_error(p.err, ADT_DEVERR_BAD_TREE);
        par = 0;
      }
    }
    p.parents[node] = par;
  }
  __threadfence_block();
  __syncthreads();
  if (p.depth) {
    for (int node = 1 + tid; node <= need; node += kRerankThreads) {
      int d = 0, j = node;
      while (j > 0 && d <= need) {
        j = p.parents[j];
        ++d;
      }
      p.depth[node] = d;
    }
  }
}

}  // namespace

static adt_status expand_impl(const float* logits, const float* logits_u, float cfg_scale, int64_t ld,
                              const float* frontier_score, const int32_t* frontier_id, int32_t F, int32_t V,
                              int32_t k_child, int32_t k_keep, float temperature, int32_t child_id_base,
                              int32_t* child_token, float* child_logp, float* child_score,
                              int32_t* child_parent, int32_t* keep_idx, float* next_score, int32_t* next_id,
                              void* workspace, size_t workspace_bytes, void* stream) {
  ADT_REQUIRE(logits && frontier_score && child_token && child_score && child_parent);
  ADT_REQUIRE(keep_idx || (!next_score && !next_id));
  if (logits_u) ADT_REQUIRE(adt::aligned16(logits_u) && cfg_scale > -1e30f && cfg_scale < 1e30f);
  ADT_REQUIRE(F >= 1 && F <= kMaxRows && V >= 1 && V <= (1 << 24));
  ADT_REQUIRE(k_child >= 1 && k_child <= kMaxK && k_child <= V);
  ADT_REQUIRE(k_keep >= 1 && k_keep <= F * k_child && k_keep <= kMaxKeep);
  ADT_REQUIRE(ld >= V && ld % 4 == 0 && adt::aligned16(logits));
  ADT_REQUIRE(temperature > 0.f && temperature < 1e30f);
  const ExpandWs w = expand_ws(F, V, k_child);
  if (!workspace || workspace_bytes < w.total || !adt::aligned16(workspace)) return ADT_ERR_WORKSPACE;
  adt::DeviceInfo info;
  adt_status st = adt::device_info(&info);
  if (st != ADT_OK) return st;
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  ExpandParams p;
  p.logits = logits;
  p.logits_u = logits_u;
  p.cfg = cfg_scale;
  p.ld = ld;
  p.fscore = frontier_score;
  p.fid = frontier_id;
  p.F = F;
  p.V = V;
  p.k = k_child;
  p.k_keep = k_keep;
  p.T = temperature;
  p.use_T = temperature != 1.0f;
  p.id_base = child_id_base;
  p.ctok = child_token;
  p.clogp = child_logp;
  p.cscore = child_score;
  p.cpar = child_parent;
  p.keep = keep_idx;
  p.nscore = next_score;
  p.nid = next_id;
  p.cross_keys = reinterpret_cast<uint64_t*>(ws + w.cross_keys);
  p.all_ticket = reinterpret_cast<unsigned*>(ws + w.all_ticket);
  p.err = info.error_word;
  const int C = expand_cluster(V);
  const int per = ((V + C - 1) / C + 3) & ~3;
  const size_t dyn = static_cast<size_t>(per < kTile ? per : kTile) * sizeof(float) * (logits_u ? 2 : 1);
  static unsigned configured[2] = {0u, 0u};  // bit per device (< 64)
  unsigned& word = configured[(info.device >> 5) & 1];
  const unsigned bit = 1u << (info.device & 31);
  if (!(__atomic_load_n(&word, __ATOMIC_ACQUIRE) & bit)) {
    ADT_CUDA_TRY(cudaFuncSetAttribute(expand_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      static_cast<int>(2 * kTile * sizeof(float))));
    __atomic_fetch_or(&word, bit, __ATOMIC_ACQ_REL);
  }
  cudaLaunchConfig_t cfg = {};
  cfg.dynamicSmemBytes = dyn;
  cfg.gridDim = dim3(static_cast<unsigned>(C), static_cast<unsigned>(F), 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.stream = adt::as_stream(stream);
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = static_cast<unsigned>(C);
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1] = adt::pdl_attribute();
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  ADT_CUDA_TRY(cudaLaunchKernelEx(&cfg, expand_kernel, p));
  return adt::launch_status();
}

extern "C" {

size_t adt_tree_expand_workspace_size(int32_t F, int32_t V, int32_t k_child) {
  if (F < 1 || V < 1 || k_child < 1) return 0;
  return expand_ws(F, V, k_child).total;
}

adt_status adt_tree_expand(const float* logits, int64_t ld, const float* frontier_score,
                           const int32_t* frontier_id, int32_t F, int32_t V, int32_t k_child,
                           int32_t k_keep, float temperature, int32_t child_id_base,
                           int32_t* child_token, float* child_logp, float* child_score,
                           int32_t* child_parent, int32_t* keep_idx, float* next_score,
                           int32_t* next_id, void* workspace, size_t workspace_bytes,
                           void* stream) {
  adt::TraceRange trace_("adt_tree_expand");
  return expand_impl(logits, nullptr, 0.f, ld, frontier_score, frontier_id, F, V, k_child, k_keep, temperature,
                     child_id_base, child_token, child_logp, child_score, child_parent, keep_idx, next_score,
                     next_id, workspace, workspace_bytes, stream);
}

adt_status adt_tree_expand_cfg(const float* logits_cond, const float* logits_uncond, int64_t ld,
                               float cfg_scale, const float* frontier_score, const int32_t* frontier_id,
                               int32_t F, int32_t V, int32_t k_child, int32_t k_keep, float temperature,
                               int32_t child_id_base, int32_t* child_token, float* child_logp,
                               float* child_score, int32_t* child_parent, int32_t* keep_idx,
                               float* next_score, int32_t* next_id, void* workspace,
                               size_t workspace_bytes, void* stream) {
  adt::TraceRange trace_("adt_tree_expand_cfg");
  ADT_REQUIRE(logits_uncond);
  return expand_impl(logits_cond, logits_uncond, cfg_scale, ld, frontier_score, frontier_id, F, V, k_child,
                     k_keep, temperature, child_id_base, child_token, child_logp, child_score, child_parent,
                     keep_idx, next_score, next_id, workspace, workspace_bytes, stream);
}

size_t adt_tree_rerank_workspace_size(int32_t C) {
  if (C < 1) return 0;
  return adt::align_up(static_cast<size_t>(C) * sizeof(int32_t), 256) +
         adt::align_up(4097 * sizeof(int32_t), 256);
}

adt_status adt_tree_rerank(const int32_t* cand_token, const float* cand_score,
                           const int32_t* cand_parent, int32_t C, const int32_t* root_token,
                           int32_t n_nodes, int32_t* tokens, int32_t* parents,
                           int32_t* cand_index, int32_t* depth, void* workspace,
                           size_t workspace_bytes, void* stream) {
  adt::TraceRange trace_("adt_tree_rerank");
  ADT_REQUIRE(cand_token && cand_score && cand_parent && root_token && tokens && parents);
  ADT_REQUIRE(C >= 1 && C <= 65536 && n_nodes >= 1 && n_nodes <= C + 1 && n_nodes <= 4096);
  const size_t need = adt_tree_rerank_workspace_size(C);
  if (!workspace || workspace_bytes < need || !adt::aligned16(workspace)) return ADT_ERR_WORKSPACE;
  adt::DeviceInfo info;
  adt_status st = adt::device_info(&info);
  if (st != ADT_OK) return st;
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  RerankParams p;
  p.ctok = cand_token;
  p.cscore = cand_score;
  p.cpar = cand_parent;
  p.C = C;
  p.root = root_token;
  p.n_nodes = n_nodes;
  p.tokens = tokens;
  p.parents = parents;
  p.cand_index = cand_index;
  p.depth = depth;
  p.node_of = reinterpret_cast<int32_t*>(ws);
  p.cand_of_node = reinterpret_cast<int32_t*>(ws + adt::align_up(static_cast<size_t>(C) * sizeof(int32_t), 256));
  p.err = info.error_word;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(1, 1, 1);
  cfg.blockDim = dim3(kRerankThreads, 1, 1);
  cfg.stream = adt::as_stream(stream);
  cudaLaunchAttribute attr[1] = {adt::pdl_attribute()};
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (C <= kRerankSmall && C <= kRerankThreads && n_nodes <= kRerankSmall + 1)
    ADT_CUDA_TRY(cudaLaunchKernelEx(&cfg, rerank_small_kernel, p));
  else
    ADT_CUDA_TRY(cudaLaunchKernelEx(&cfg, rerank_kernel, p));
  return adt::launch_status();
}

}  // extern "C"
