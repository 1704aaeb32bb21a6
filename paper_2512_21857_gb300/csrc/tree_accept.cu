// adt_tree_accept: the verification walk (Sec. 3.1, Eq. 1; greedy T = 0 and
// sampling T = 1 as in Sec. 5.1).
//
// One thread-block cluster per tree.  The vocabulary is split into equal
// slices, one per CTA of the cluster; a CTA keeps its slice of the current
// node's target (and draft) row in shared memory.  Vocabulary-wide
// quantities (argmax, max, sum of exponentials, residual mass, the CDF
// offset of each slice) are block reductions whose per-CTA results are
// published in shared memory and read by every CTA of the cluster through
// distributed shared memory after a cluster barrier.  Every CTA sums the
// published values in the same order, so all CTAs take identical decisions
// without further communication.  p(x), q(x) of a child's token are read
// from the owning CTA's slice.  The walk itself (children in ascending
// index, one accept test each) is sequential, as the method defines it.
#include <cooperative_groups.h>

#include "adt_common.cuh"
#include "dfloat.cuh"

namespace cg = cooperative_groups;

namespace {

constexpr int kThreads = 512;
constexpr int kMaxNodes = 1024;

struct AcceptParams {
  const float* target;
  int64_t ldt;
  const float* draft;
  int64_t ldd;
  const float* target_u;  // classifier-free guidance: unconditional rows (same layout), else NULL
  const float* draft_u;
  float cfg;              // guidance scale
  const int32_t* drow;
  const int32_t* tokens;
  const int32_t* parents;
  const int32_t* offs;
  int B, V, max_nodes;
  const float* ua;
  const float* us;
  int mode;
  float T;
  int use_T;
  int32_t* path;
  int max_path;
  int32_t* alen;
  int32_t* bonus;
  unsigned* err;
  int Vs;  // vocabulary slice per CTA (multiple of 4)
};

// Values a CTA publishes to its cluster; two copies alternate so that one
// barrier per exchange suffices.
struct Slot {
  float2 g[2];  // double-float values (hi, lo)
  float f[2];
  int i[2];
};

struct Shared {
  Slot slot[2];
  int par[kMaxNodes];
  int tok[kMaxNodes];
  int kids[kMaxNodes];
  int path[kMaxNodes];
  int rejected[kMaxNodes];
  float fred[32];
  int ired[32];
  float2 exptab[64];  // 2^(j/64) as double-floats (the double-float exponential's table)
  float2 dfred[32];   // double-float block reductions
  float2 dfpre[32];   // exclusive prefix of the warps' double-float totals
  // Scalars thread 0 derives from the cluster's published values (in
  // double-float, once per CTA) and hands to the block.
  float2 bf[4];
  int bi[4];
  int nkids;
  int bad;
  int found;
  int last_pos;
};

struct Walker {
  cg::cluster_group cl;
  Shared* sh;
  int rank, csize, parity;
  __device__ Slot* publish_slot() { return &sh->slot[parity]; }
  // Barrier, then return the published slot of CTA c (same parity).
  __device__ const Slot* peer(int c) { return cl.map_shared_rank(&sh->slot[parity], c); }
  __device__ void exchange() {
    cl.sync();
  }
  __device__ void flip() { parity ^= 1; }
};

__device__ __forceinline__ bool better(float v, int i, float bv, int bi) {
  return v > bv || (v == bv && i < bi);
}

// The cluster's published double-float values g[k] summed over its CTAs:
// lane c (< csize) of the calling warp reads CTA c's slot, so the reads go
// out together instead of one after another, and the lanes combine them by
// shuffles.  Every CTA runs the same operations on the same values, so all
// get the same sum; lane 0's is the one used.
__device__ __forceinline__ dfl::df warp_cluster_sum(Walker& w, int k) {
  const int lane = threadIdx.x & 31;
  dfl::df v{0.f, 0.f};
  if (lane < w.csize) {
    const float2 g = w.peer(lane)->g[k];
    v = dfl::df{g.x, g.y};
  }
  for (int o = 16; o > 0; o >>= 1)
    v = dfl::df_add(v, dfl::df{__shfl_xor_sync(adt::kFullMask, v.hi, o), __shfl_xor_sync(adt::kFullMask, v.lo, o)});
  return v;
}

// The sampling modes' slices of p and q.  Slice<true>: double-float
// entries (hi, lo), exponentials and every update in double-float, so the
// decisions the walk takes from them (u q(x) < p(x), the inverse-CDF draw)
// agree with fp64 arithmetic to about 1e-11 relative; used where the slices
// fit in shared memory.  Slice<false>: fp32 entries and fp32 exponentials
// (relative error about 1e-7), for larger vocabularies.
template <bool kDF>
struct Slice;

template <>
struct Slice<false> {
  using E = float;
  static __device__ __forceinline__ E logit(float x) { return x; }
  static __device__ __forceinline__ float value_hi(E v) { return v; }
  static __device__ __forceinline__ E exp_diff(float x, float M, const float2*) { return expf(x - M); }
  static __device__ __forceinline__ bool pos(E v) { return v > 0.f; }
  static __device__ __forceinline__ E zero() { return 0.f; }
  static __device__ __forceinline__ dfl::df as_df(E v) { return dfl::df{v, 0.f}; }
  using F = float;  // a scale factor, converted once per pass
  static __device__ __forceinline__ F factor(float2 s) { return s.x; }
  static __device__ __forceinline__ E scale(E v, F f) { return v * f; }
  static __device__ __forceinline__ E resid(E p, E q) { return fmaxf(p - q, 0.f); }
  struct Acc {
    float a = 0.f;
    __device__ __forceinline__ void add(E v) { a += v; }
    __device__ __forceinline__ dfl::df value_df() const { return dfl::df{a, 0.f}; }
  };
};

template <>
struct Slice<true> {
  using E = float2;
  static __device__ __forceinline__ E logit(float x) { return make_float2(x, 0.f); }
  static __device__ __forceinline__ float value_hi(E v) { return v.x; }
  static __device__ __forceinline__ E exp_diff(float x, float M, const float2* tab) {
    const dfl::df e = dfl::df_exp_diff(x, M, tab);
    return make_float2(e.hi, e.lo);
  }
  static __device__ __forceinline__ bool pos(E v) { return v.x > 0.f; }
  static __device__ __forceinline__ E zero() { return make_float2(0.f, 0.f); }
  static __device__ __forceinline__ dfl::df as_df(E v) { return dfl::df{v.x, v.y}; }
  using F = dfl::df;
  static __device__ __forceinline__ F factor(float2 s) { return dfl::df{s.x, s.y}; }
  static __device__ __forceinline__ E scale(E v, F f) {
    const dfl::df r = dfl::df_mul(dfl::df{v.x, v.y}, f);
    return make_float2(r.hi, r.lo);
  }
  static __device__ __forceinline__ E resid(E p, E q) {
    const dfl::df r = dfl::df_max0(dfl::df_add(dfl::df{p.x, p.y}, dfl::df{-q.x, -q.y}));
    return make_float2(r.hi, r.lo);
  }
  struct Acc {
    dfl::Acc a;
    __device__ __forceinline__ void add(E v) { a.add(dfl::df{v.x, v.y}); }
    __device__ __forceinline__ dfl::df value_df() const { return a.value_df(); }
  };
};

// Block argmax over (value desc, index asc); all threads get the result.
__device__ void block_argmax(float& v, int& idx, Shared* sh) {
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(adt::kFullMask, v, o);
    const int oi = __shfl_xor_sync(adt::kFullMask, idx, o);
    if (better(ov, oi, v, idx)) {
      v = ov;
      idx = oi;
    }
  }
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  __syncthreads();
  if (lane == 0) {
    sh->fred[warp] = v;
    sh->ired[warp] = idx;
  }
  __syncthreads();
  v = lane < kThreads / 32 ? sh->fred[lane] : -INFINITY;
  idx = lane < kThreads / 32 ? sh->ired[lane] : 0x7fffffff;
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(adt::kFullMask, v, o);
    const int oi = __shfl_xor_sync(adt::kFullMask, idx, o);
    if (better(ov, oi, v, idx)) {
      v = ov;
      idx = oi;
    }
  }
}

// Loads this CTA's slice of a logit row (under guidance u + s (c - u) with
// the unconditional row row_u; then divided by T) into buf; entries past V
// are -inf.
template <bool kDF>
__device__ void load_slice(const float* row, const float* row_u, int lo, int cnt, int Vs,
                           typename Slice<kDF>::E* buf, const AcceptParams& p) {
  for (int i = threadIdx.x * 4; i < Vs; i += kThreads * 4) {
    float x[4];
    if (i + 3 < cnt) {
      const float4 v = __ldg(reinterpret_cast<const float4*>(row + lo + i));
      x[0] = v.x; x[1] = v.y; x[2] = v.z; x[3] = v.w;
      if (row_u) {
        const float4 w = __ldg(reinterpret_cast<const float4*>(row_u + lo + i));
        x[0] = adt::cfg_combine(x[0], w.x, p.cfg);
        x[1] = adt::cfg_combine(x[1], w.y, p.cfg);
        x[2] = adt::cfg_combine(x[2], w.z, p.cfg);
        x[3] = adt::cfg_combine(x[3], w.w, p.cfg);
      }
    } else {
      for (int e = 0; e < 4; ++e)
        x[e] = (i + e < cnt) ? (row_u ? adt::cfg_combine(__ldg(row + lo + i + e), __ldg(row_u + lo + i + e), p.cfg)
                                      : __ldg(row + lo + i + e))
                             : -INFINITY;
    }
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      float y = x[e];
      if (p.use_T && i + e < cnt) y = __fdiv_rn(y, p.T);
      buf[i + e] = Slice<kDF>::logit(y);
    }
  }
}

// Sum over the block in double-float (fp32 operations only); every thread
// gets the result.
__device__ dfl::df block_sum_df(dfl::df v, Shared* sh) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int o = 16; o > 0; o >>= 1)
    v = dfl::df_add(v, dfl::df{__shfl_xor_sync(adt::kFullMask, v.hi, o), __shfl_xor_sync(adt::kFullMask, v.lo, o)});
  __syncthreads();
  if (lane == 0) sh->dfred[warp] = make_float2(v.hi, v.lo);
  __syncthreads();
  dfl::df r = lane < kThreads / 32 ? dfl::df{sh->dfred[lane].x, sh->dfred[lane].y} : dfl::df{0.f, 0.f};
  for (int o = 16; o > 0; o >>= 1)
    r = dfl::df_add(r, dfl::df{__shfl_xor_sync(adt::kFullMask, r.hi, o), __shfl_xor_sync(adt::kFullMask, r.lo, o)});
  return r;
}

// exp(x - M) in place over the slice (the logits M is the row maximum of);
// returns the block's sum.
template <bool kDF>
__device__ dfl::df exp_in_place(typename Slice<kDF>::E* buf, int Vs, float M, Shared* sh) {
  typename Slice<kDF>::Acc acc;
  for (int i = threadIdx.x; i < Vs; i += kThreads) {
    const typename Slice<kDF>::E e = Slice<kDF>::exp_diff(Slice<kDF>::value_hi(buf[i]), M, sh->exptab);
    buf[i] = e;
    acc.add(e);
  }
  return block_sum_df(acc.value_df(), sh);
}

template <bool kDF>
__device__ float slice_max(const typename Slice<kDF>::E* buf, int Vs, Shared* sh) {
  float m = -INFINITY;
  for (int i = threadIdx.x; i < Vs; i += kThreads) m = fmaxf(m, Slice<kDF>::value_hi(buf[i]));
  return adt::block_max<kThreads>(m, sh->fred);
}

// Inverse-CDF draw over the (unnormalised, non-negative) distribution held
// in the cluster's slices: smallest t with sum_{j<=t} w_j > u * sum_j w_j.
// Returns the token id on every CTA.
template <bool kDF>
__device__ int cluster_sample(Walker& w, const typename Slice<kDF>::E* buf, int lo, int cnt, float u, Shared* sh) {
  // 1. per-CTA slice totals (each thread owns a contiguous run), published.
  // A thread reads its run starting at offset tid mod len, wrapping around:
  // at the same step the threads of a half-warp then touch different banks
  // (in index order every thread would hit the same bank).
  const int per = (cnt + kThreads - 1) / kThreads;
  const int b0 = min(cnt, static_cast<int>(threadIdx.x) * per), b1 = min(cnt, b0 + per);
  typename Slice<kDF>::Acc racc;
  int last_pos = -1;
  {
    const int len = b1 - b0;
    int j = len > 0 ? static_cast<int>(threadIdx.x) % len : 0;
    for (int k = 0; k < len; ++k) {
      const int i = b0 + j;
      racc.add(buf[i]);
      if (Slice<kDF>::pos(buf[i])) last_pos = max(last_pos, i);
      if (++j == len) j = 0;
    }
  }
  const dfl::df run = racc.value_df();
  const dfl::df tot = block_sum_df(run, sh);
  if (threadIdx.x == 0) w.publish_slot()->g[0] = make_float2(tot.hi, tot.lo);
  w.exchange();
  if (threadIdx.x < 32) {
    // Lane c reads CTA c's total; an inclusive scan over the lanes gives
    // every CTA's cumulative total (the grand total in lane csize - 1).
    const int lane = threadIdx.x;
    dfl::df t{0.f, 0.f};
    if (lane < w.csize) {
      const float2 g = w.peer(lane)->g[0];
      t = dfl::df{g.x, g.y};
    }
    dfl::df incl = t;
    for (int o = 1; o < 32; o <<= 1) {
      const dfl::df y{__shfl_up_sync(adt::kFullMask, incl.hi, o), __shfl_up_sync(adt::kFullMask, incl.lo, o)};
      if (lane >= o) incl = dfl::df_add(incl, y);
    }
    const dfl::df grand{__shfl_sync(adt::kFullMask, incl.hi, w.csize - 1),
                        __shfl_sync(adt::kFullMask, incl.lo, w.csize - 1)};
    const int br = w.rank > 0 ? w.rank - 1 : 0;
    const dfl::df before{__shfl_sync(adt::kFullMask, incl.hi, br), __shfl_sync(adt::kFullMask, incl.lo, br)};
    const dfl::df base = w.rank > 0 ? before : dfl::df{0.f, 0.f};
    const dfl::df target = dfl::df_mul_f(grand, u);
    // Owner: first CTA whose cumulative total passes the target; else the
    // last CTA with mass.
    const unsigned pass = __ballot_sync(adt::kFullMask, lane < w.csize && dfl::df_less(target, incl));
    const unsigned mass = __ballot_sync(adt::kFullMask, lane < w.csize && t.hi > 0.f);
    if (lane == 0) {
      sh->bi[0] = pass ? __ffs(pass) - 1 : (mass ? 31 - __clz(mass) : 0);
      sh->bf[0] = make_float2(base.hi, base.lo);
      sh->bf[1] = make_float2(-target.hi, -target.lo);
    }
  }
  __syncthreads();
  const int owner = sh->bi[0];
  const dfl::df base = dfl::df{sh->bf[0].x, sh->bf[0].y}, ntgt = dfl::df{sh->bf[1].x, sh->bf[1].y};
  w.flip();
  int result_local = -1;
  if (w.rank == owner) {
    // exclusive scan of the per-thread runs, in double-float
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    dfl::df incl = run;
    for (int o = 1; o < 32; o <<= 1) {
      const dfl::df y{__shfl_up_sync(adt::kFullMask, incl.hi, o), __shfl_up_sync(adt::kFullMask, incl.lo, o)};
      if (lane >= o) incl = dfl::df_add(incl, y);
    }
    __syncthreads();
    if (lane == 31) sh->dfred[warp] = make_float2(incl.hi, incl.lo);
    if (threadIdx.x == 0) {
      sh->found = 0x7fffffff;
      sh->last_pos = -1;
    }
    __syncthreads();
    if (warp == 0) {
      // exclusive prefix of the warps' totals, one scan in warp 0
      dfl::df wt = lane < kThreads / 32 ? dfl::df{sh->dfred[lane].x, sh->dfred[lane].y} : dfl::df{0.f, 0.f};
      for (int o = 1; o < 32; o <<= 1) {
        const dfl::df y{__shfl_up_sync(adt::kFullMask, wt.hi, o), __shfl_up_sync(adt::kFullMask, wt.lo, o)};
        if (lane >= o) wt = dfl::df_add(wt, y);
      }
      const dfl::df prev{__shfl_up_sync(adt::kFullMask, wt.hi, 1), __shfl_up_sync(adt::kFullMask, wt.lo, 1)};
      if (lane < kThreads / 32) sh->dfpre[lane] = lane == 0 ? make_float2(0.f, 0.f) : make_float2(prev.hi, prev.lo);
    }
    __syncthreads();
    // The running CDF in double-float, compared with the target through the
    // sign of their difference.  A run whose end does not pass the target
    // cannot hold the draw and is not walked.
    dfl::df acc = dfl::df_add(base, dfl::df{sh->dfpre[warp].x, sh->dfpre[warp].y});
    acc = dfl::df_add(acc, dfl::df_add(incl, dfl::df_neg(run)));
    if (last_pos >= 0) atomicMax(&sh->last_pos, last_pos);
    if (dfl::df_add(dfl::df_add(acc, run), ntgt).hi > 0.f) {
      for (int i = b0; i < b1; ++i) {
        acc = dfl::df_add(acc, Slice<kDF>::as_df(buf[i]));
        if (Slice<kDF>::pos(buf[i]) && dfl::df_add(acc, ntgt).hi > 0.f) {
          atomicMin(&sh->found, i);
          break;
        }
      }
    }
    __syncthreads();
    int t = sh->found;
    if (t == 0x7fffffff) t = sh->last_pos < 0 ? 0 : sh->last_pos;
    result_local = lo + t;
    if (threadIdx.x == 0) w.publish_slot()->i[0] = result_local;
  }
  w.exchange();
  const int res = w.peer(owner)->i[0];
  w.flip();
  return res;
}

template <bool kDF>
__global__ void __launch_bounds__(kThreads) accept_kernel(const AcceptParams p) {
  using SL = Slice<kDF>;
  using E = typename SL::E;
  extern __shared__ __align__(16) float dyn[];
  __shared__ Shared sh;
  if (kDF) dfl::exp_table_to_smem(sh.exptab);  // read after the __syncthreads below
  adt::pdl_wait_then_release();
  cg::cluster_group cl = cg::this_cluster();
  Walker w{cl, &sh, static_cast<int>(cl.block_rank()), static_cast<int>(cl.num_blocks()), 0};
  const int b = blockIdx.x / w.csize;
  const int tid = threadIdx.x;
  E* pbuf = reinterpret_cast<E*>(dyn);
  E* qbuf = pbuf + p.Vs;
  const int lo = w.rank * p.Vs;
  const int cnt = max(0, min(p.Vs, p.V - lo));

  const int node0 = p.offs[b];
  const int n = p.offs[b + 1] - node0;
  if (tid == 0) sh.bad = (n < 1 || n > p.max_nodes) ? 1 : 0;
  __syncthreads();
  if (!sh.bad) {
    for (int i = tid; i < n; i += kThreads) {
      const int pr = p.parents[node0 + i];
      sh.par[i] = pr;
      sh.tok[i] = p.tokens[node0 + i];
      if ((i == 0) != (pr < 0) || pr >= i) sh.bad = 1;
    }
  }
  __syncthreads();
  if (sh.bad) {
    if (w.rank == 0 && tid == 0) {
      adt::raise_error(p.err, ADT_DEVERR_BAD_TREE);
      p.alen[b] = 0;
      p.bonus[b] = 0;
      for (int i = 0; i < p.max_path; ++i) p.path[static_cast<int64_t>(b) * p.max_path + i] = i == 0 ? 0 : -1;
    }
    cl.sync();
    return;
  }

  int v = 0, plen = 1;
  if (tid == 0) sh.path[0] = 0;
  int bonus = 0;
  for (int step = 0; step < n; ++step) {
    // children of v, ascending
    __syncthreads();
    if (tid == 0) sh.nkids = 0;
    __syncthreads();
    for (int base = 0; base < n; base += kThreads) {
      const int i = base + tid;
      const bool f = i < n && sh.par[i] == v;
      const unsigned bal = __ballot_sync(adt::kFullMask, f);
      const int lane = tid & 31, warp = tid >> 5;
      if (lane == 0) sh.ired[warp] = __popc(bal);
      __syncthreads();
      int before = 0;
      for (int j = 0; j < warp; ++j) before += sh.ired[j];
      if (f) sh.kids[sh.nkids + before + __popc(bal & ((1u << lane) - 1u))] = i;
      __syncthreads();
      if (tid == 0) {
        int t = 0;
        for (int j = 0; j < kThreads / 32; ++j) t += sh.ired[j];
        sh.nkids += t;
      }
      __syncthreads();
    }
    int nk = sh.nkids;
    const int gv = node0 + v;
    const float* trow = p.target + static_cast<int64_t>(gv) * p.ldt;
    const float* trow_u = p.target_u ? p.target_u + static_cast<int64_t>(gv) * p.ldt : nullptr;

    if (p.mode == ADT_ACCEPT_GREEDY) {
      float bv = -INFINITY;
      int bi = 0x7fffffff;
      // 16-byte loads (the row start and lo are multiples of 4 floats), a
      // thread's kU loads all issued before any value is compared.
      constexpr int kU = 4;
      const int c4 = cnt >> 2;
      const float4* t4 = reinterpret_cast<const float4*>(trow + lo);
      const float4* u4 = trow_u ? reinterpret_cast<const float4*>(trow_u + lo) : nullptr;
      for (int g0 = tid; g0 < c4; g0 += kU * kThreads) {
        float4 x[kU];
#pragma unroll
        for (int u = 0; u < kU; ++u) {
          const int g = g0 + u * kThreads;
          x[u] = g < c4 ? __ldg(t4 + g) : make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
        }
        if (u4) {
#pragma unroll
          for (int u = 0; u < kU; ++u) {
            const int g = g0 + u * kThreads;
            if (g < c4) {
              const float4 y = __ldg(u4 + g);
              x[u].x = adt::cfg_combine(x[u].x, y.x, p.cfg);
              x[u].y = adt::cfg_combine(x[u].y, y.y, p.cfg);
              x[u].z = adt::cfg_combine(x[u].z, y.z, p.cfg);
              x[u].w = adt::cfg_combine(x[u].w, y.w, p.cfg);
            }
          }
        }
#pragma unroll
        for (int u = 0; u < kU; ++u) {
          const int g = g0 + u * kThreads;
          if (g >= c4) continue;
          const int i = lo + 4 * g;
          const float e[4] = {x[u].x, x[u].y, x[u].z, x[u].w};
#pragma unroll
          for (int j = 0; j < 4; ++j)
            if (better(e[j], i + j, bv, bi)) {
              bv = e[j];
              bi = i + j;
            }
        }
      }
      for (int i = 4 * c4 + tid; i < cnt; i += kThreads) {  // the last slice's final cnt % 4 values
        float x = __ldg(trow + lo + i);
        if (trow_u) x = adt::cfg_combine(x, __ldg(trow_u + lo + i), p.cfg);
        if (better(x, lo + i, bv, bi)) {
          bv = x;
          bi = lo + i;
        }
      }
      block_argmax(bv, bi, &sh);
      if (tid == 0) {
        w.publish_slot()->f[0] = bv;
        w.publish_slot()->i[0] = bi;
      }
      w.exchange();
      // lane c reads CTA c's candidate; the warp's argmax over the lanes
      float gvv = -INFINITY;
      int g = 0x7fffffff;
      if ((tid & 31) < w.csize) {
        const Slot* s = w.peer(tid & 31);
        gvv = s->f[0];
        g = s->i[0];
      }
      for (int o = 16; o > 0; o >>= 1) {
        const float ov = __shfl_xor_sync(adt::kFullMask, gvv, o);
        const int oi = __shfl_xor_sync(adt::kFullMask, g, o);
        if (better(ov, oi, gvv, g)) {
          gvv = ov;
          g = oi;
        }
      }
      w.flip();
      int nxt = -1;
      for (int j = 0; j < nk; ++j) {
        if (sh.tok[sh.kids[j]] == g) {
          nxt = sh.kids[j];
          break;
        }
      }
      if (nxt < 0) {
        bonus = g;
        break;
      }
      if (tid == 0) sh.path[plen] = nxt;
      ++plen;
      v = nxt;
      continue;
    }

    // ---- sampling modes: p = softmax(target row / T) in the slices.
    const bool spec = p.mode == ADT_ACCEPT_SPEC;
    // The draft row of v (the same value in every thread of the cluster).  A
    // node with children but no draft row (negative index) is an error; its
    // children are then not considered and the bonus comes from p.
    const int64_t dr = spec && nk > 0 && p.drow ? static_cast<int64_t>(p.drow[gv]) : gv;
    if (dr < 0) {
      if (w.rank == 0 && tid == 0) adt::raise_error(p.err, ADT_DEVERR_BAD_INDEX);
      nk = 0;
    }
    const bool need_q = spec && nk > 0;
    load_slice<kDF>(trow, trow_u, lo, cnt, p.Vs, pbuf, p);
    if (need_q)
      load_slice<kDF>(p.draft + dr * p.ldd, p.draft_u ? p.draft_u + dr * p.ldd : nullptr, lo, cnt, p.Vs, qbuf, p);
    __syncthreads();
    const float mp = slice_max<kDF>(pbuf, p.Vs, &sh);
    const float mq = need_q ? slice_max<kDF>(qbuf, p.Vs, &sh) : 0.f;
    if (tid == 0) {
      w.publish_slot()->f[0] = mp;
      w.publish_slot()->f[1] = mq;
    }
    w.exchange();
    float Mp = -INFINITY, Mq = -INFINITY;
    if ((tid & 31) < w.csize) {  // lane c reads CTA c's maxima
      Mp = w.peer(tid & 31)->f[0];
      Mq = w.peer(tid & 31)->f[1];
    }
    Mp = adt::warp_max(Mp);
    Mq = adt::warp_max(Mq);
    w.flip();
    const dfl::df sp_loc = exp_in_place<kDF>(pbuf, p.Vs, Mp, &sh);
    const dfl::df sq_loc = need_q ? exp_in_place<kDF>(qbuf, p.Vs, Mq, &sh) : dfl::df{0.f, 0.f};
    if (tid == 0) {
      w.publish_slot()->g[0] = make_float2(sp_loc.hi, sp_loc.lo);
      w.publish_slot()->g[1] = make_float2(sq_loc.hi, sq_loc.lo);
    }
    w.exchange();
    // The row totals, formed once (thread 0 keeps them for the decisions) and
    // handed to the block as double-float reciprocals.
    dfl::df Sp{0.f, 0.f}, Sq{0.f, 0.f};
    if (tid < 32) {
      Sp = warp_cluster_sum(w, 0);
      Sq = warp_cluster_sum(w, 1);
    }
    if (tid == 0) {
      const dfl::df ip = dfl::df_recip(Sp), iq = Sq.hi > 0.f ? dfl::df_recip(Sq) : dfl::df{0.f, 0.f};
      sh.bf[0] = make_float2(ip.hi, ip.lo);
      sh.bf[1] = make_float2(iq.hi, iq.lo);
    }
    __syncthreads();
    w.flip();
    if (spec && need_q) {
      // normalise both slices
      const typename SL::F ip = SL::factor(sh.bf[0]), iq = SL::factor(sh.bf[1]);
      for (int i = tid; i < p.Vs; i += kThreads) {
        pbuf[i] = SL::scale(pbuf[i], ip);
        qbuf[i] = SL::scale(qbuf[i], iq);
      }
      w.exchange();  // slices final before any peer reads them
      w.flip();
    }

    // The children in ascending index.  Thread 0 reads p(x), q(x) from the
    // owning CTA, takes the decision in double-float and hands it to the
    // block.
    int nxt = -1;
    dfl::df e_rej{0.f, 0.f};  // SPEC_DET, thread 0: rejected unnormalised mass
    int nrej = 0;        // SPEC_DET: rejected tokens (in sh.rejected)
    for (int j = 0; j < nk; ++j) {
      const int c = sh.kids[j];
      const int x = sh.tok[c];
      if (x < 0 || x >= p.V) {
        if (w.rank == 0 && tid == 0) adt::raise_error(p.err, ADT_DEVERR_BAD_INDEX);
        continue;
      }
      const int owner = x / p.Vs, off = x - owner * p.Vs;
      if (tid == 0) {
        // u < p(x) / denom is taken as u denom < p(x): no division.
        const float u = p.ua[node0 + c];
        if (!spec) {
          bool dup = false;
          for (int r = 0; r < nrej; ++r) dup |= sh.rejected[r] == x;
          const dfl::df ex = dup ? dfl::df{0.f, 0.f} : SL::as_df(*cl.map_shared_rank(pbuf + off, owner));
          const dfl::df denom = dfl::df_add(Sp, dfl::df_neg(e_rej));
          const bool a = denom.hi > 0.f && dfl::df_less(dfl::df_mul_f(denom, u), ex);
          sh.bi[1] = a;
          sh.bi[2] = !a && !dup;  // a new rejected token
          if (!a && !dup) {
            e_rej = dfl::df_add(e_rej, ex);
            sh.rejected[nrej] = x;
          }
        } else {
          const dfl::df px = SL::as_df(*cl.map_shared_rank(pbuf + off, owner));
          const dfl::df qx = SL::as_df(*cl.map_shared_rank(qbuf + off, owner));
          sh.bi[1] = dfl::df_less(dfl::df_mul_f(qx, u), px);
          sh.bi[2] = 0;
        }
      }
      __syncthreads();
      const bool acc = sh.bi[1] != 0;
      nrej += sh.bi[2];
      __syncthreads();  // sh.bi is rewritten for the next child
      if (!acc && spec) {
        // residual: p <- max(0, p - q)/Z (kept if Z = 0); q(x) <- 0, q <- q/sum
        typename SL::Acc zl, ql;
        for (int i = tid; i < p.Vs; i += kThreads) {
          zl.add(SL::resid(pbuf[i], qbuf[i]));
          if (lo + i != x) ql.add(qbuf[i]);
        }
        const dfl::df zb = block_sum_df(zl.value_df(), &sh);
        const dfl::df qb = block_sum_df(ql.value_df(), &sh);
        if (tid == 0) {
          w.publish_slot()->g[0] = make_float2(zb.hi, zb.lo);
          w.publish_slot()->g[1] = make_float2(qb.hi, qb.lo);
        }
        w.exchange();  // also: every peer has finished reading px, qx
        dfl::df Z{0.f, 0.f}, Qs{0.f, 0.f};
        if (tid < 32) {
          Z = warp_cluster_sum(w, 0);
          Qs = warp_cluster_sum(w, 1);
        }
        if (tid == 0) {
          const dfl::df iz = Z.hi > 0.f ? dfl::df_recip(Z) : dfl::df{0.f, 0.f};
          const dfl::df iqs = Qs.hi > 0.f ? dfl::df_recip(Qs) : dfl::df{0.f, 0.f};
          sh.bf[0] = make_float2(iz.hi, iz.lo);
          sh.bf[1] = make_float2(iqs.hi, iqs.lo);
          sh.bi[0] = Z.hi > 0.f;
        }
        __syncthreads();
        w.flip();
        const typename SL::F iz = SL::factor(sh.bf[0]), iqs = SL::factor(sh.bf[1]);
        const bool zpos = sh.bi[0] != 0;
        for (int i = tid; i < p.Vs; i += kThreads) {
          const E pi = pbuf[i], qi = qbuf[i];
          if (zpos) pbuf[i] = SL::scale(SL::resid(pi, qi), iz);
          qbuf[i] = (lo + i == x) ? SL::zero() : SL::scale(qi, iqs);
        }
        w.exchange();  // updated slices visible before the next read
        w.flip();
      }
      if (acc) {
        nxt = c;
        break;
      }
    }
    if (nxt >= 0) {
      if (tid == 0) sh.path[plen] = nxt;
      ++plen;
      v = nxt;
      continue;
    }
    // bonus from the current (residual) p
    if (!spec && nrej > 0) {
      __syncthreads();
      for (int r = 0; r < nrej; ++r) {
        const int x = sh.rejected[r];
        if (x >= lo && x < lo + cnt && tid == 0) pbuf[x - lo] = SL::zero();
      }
    }
    __syncthreads();
    bonus = cluster_sample<kDF>(w, pbuf, lo, cnt, p.us[gv], &sh);
    break;
  }

  __syncthreads();
  if (w.rank == 0 && tid == 0) {
    int64_t o = static_cast<int64_t>(b) * p.max_path;
    if (plen > p.max_path) adt::raise_error(p.err, ADT_DEVERR_BAD_PATH);
    for (int i = 0; i < p.max_path; ++i) p.path[o + i] = i < plen ? sh.path[i] : -1;
    p.alen[b] = min(plen, p.max_path) - 1;
    p.bonus[b] = bonus;
  }
  cl.sync();  // no CTA leaves while a peer may still read its shared memory
}

// 8 CTAs up to 131072 entries for the greedy walk (it keeps no slices);
// the sampling modes keep slices in shared memory and take 16 CTAs past
// 65536 entries, so that double-float slices fit up to about 200000 (SPEC)
// and 262144 (SPEC_DET) entries.
int cluster_size_for(int V, adt_accept_mode mode) {
  if (mode == ADT_ACCEPT_GREEDY) return V <= 131072 ? 8 : 16;
  return V <= 65536 ? 8 : 16;
}

int slice_for(int V, int cs) {
  int vs = (V + cs - 1) / cs;
  return (vs + 3) / 4 * 4;
}

}  // namespace

static adt_status accept_impl(const float* target_logits, const float* target_u, int64_t ld_target,
                              const float* draft_logits, const float* draft_u, int64_t ld_draft,
                              const int32_t* draft_row, float cfg_scale, const int32_t* tokens,
                              const int32_t* parents, const int32_t* node_offsets, int32_t B, int32_t V,
                              int32_t max_nodes, const float* u_accept, const float* u_sample,
                              adt_accept_mode mode, float temperature, int32_t* path, int32_t max_path,
                              int32_t* accept_len, int32_t* bonus_token, void* workspace,
                              size_t workspace_bytes, void* stream) {
  (void)workspace;
  (void)workspace_bytes;
  ADT_REQUIRE(target_logits && tokens && parents && node_offsets && path && accept_len && bonus_token);
  ADT_REQUIRE(mode == ADT_ACCEPT_GREEDY || mode == ADT_ACCEPT_SPEC || mode == ADT_ACCEPT_SPEC_DET);
  ADT_REQUIRE(B >= 1 && V >= 1 && V <= 262144 && max_nodes >= 1 && max_path >= 1);
  if (max_nodes > kMaxNodes) return ADT_ERR_UNSUPPORTED;
  ADT_REQUIRE(ld_target >= V && ld_target % 4 == 0 && adt::aligned16(target_logits));
  if (mode != ADT_ACCEPT_GREEDY) {
    ADT_REQUIRE(u_accept && u_sample);
    ADT_REQUIRE(temperature > 0.f && temperature < 1e30f);
  }
  if (mode == ADT_ACCEPT_SPEC) {
    ADT_REQUIRE(draft_logits && ld_draft >= V && ld_draft % 4 == 0 && adt::aligned16(draft_logits));
  }
  if (target_u) {
    ADT_REQUIRE(adt::aligned16(target_u) && cfg_scale > -1e30f && cfg_scale < 1e30f);
    if (mode == ADT_ACCEPT_SPEC) ADT_REQUIRE(draft_u && adt::aligned16(draft_u));
  }
  adt::DeviceInfo info;
  adt_status st = adt::device_info(&info);
  if (st != ADT_OK) return st;
  const int cs = cluster_size_for(V, mode);
  const int vs = slice_for(V, cs);
  const int nbuf = mode == ADT_ACCEPT_SPEC ? 2 : 1;
  // Double-float slices where they fit, fp32 slices otherwise.
  const size_t smem_df = static_cast<size_t>(vs) * sizeof(float2) * nbuf;
  const bool use_df = mode != ADT_ACCEPT_GREEDY && smem_df + sizeof(Shared) <= static_cast<size_t>(info.max_smem_optin);
  const size_t smem = mode == ADT_ACCEPT_GREEDY ? 0 : use_df ? smem_df : static_cast<size_t>(vs) * sizeof(float) * nbuf;
  if (smem + sizeof(Shared) > static_cast<size_t>(info.max_smem_optin)) return ADT_ERR_UNSUPPORTED;
  static int configured_smem[64][2];  // largest dynamic smem already allowed, per device and instantiation
  static int configured_np[64][2];
  const int dev = info.device & 63;
  auto kern = use_df ? accept_kernel<true> : accept_kernel<false>;
  if (configured_smem[dev][use_df] < static_cast<int>(smem)) {
    ADT_CUDA_TRY(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem)));
    configured_smem[dev][use_df] = static_cast<int>(smem);
  }
  if (cs > 8 && !configured_np[dev][use_df]) {
    ADT_CUDA_TRY(cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1));
    configured_np[dev][use_df] = 1;
  }
  AcceptParams p;
  p.target = target_logits;
  p.ldt = ld_target;
  p.draft = draft_logits;
  p.ldd = ld_draft;
  p.drow = draft_row;
  p.target_u = target_u;
  p.draft_u = target_u ? draft_u : nullptr;
  p.cfg = cfg_scale;
  p.tokens = tokens;
  p.parents = parents;
  p.offs = node_offsets;
  p.B = B;
  p.V = V;
  p.max_nodes = max_nodes;
  p.ua = u_accept;
  p.us = u_sample;
  p.mode = static_cast<int>(mode);
  p.T = temperature;
  p.use_T = mode != ADT_ACCEPT_GREEDY && temperature != 1.0f;
  p.path = path;
  p.max_path = max_path;
  p.alen = accept_len;
  p.bonus = bonus_token;
  p.err = info.error_word;
  p.Vs = vs;

  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(cs * B), 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = adt::as_stream(stream);
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = cs;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1] = adt::pdl_attribute();
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  ADT_CUDA_TRY(cudaLaunchKernelEx(&cfg, kern, p));
  return adt::launch_status();
}

namespace {

__global__ void exp_diff_probe_kernel(const float* a, const float* b, int n, double* out) {
  __shared__ float2 tab[64];
  dfl::exp_table_to_smem(tab);
  __syncthreads();
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x)
    out[i] = dfl::to_double(dfl::df_exp_diff(a[i], b[i], tab));
}

}  // namespace

extern "C" {

adt_status adt_testing_exp_diff(const float* a, const float* b, int32_t n, double* out, void* stream) {
  ADT_REQUIRE(a && b && out && n >= 0);
  if (n == 0) return ADT_OK;
  exp_diff_probe_kernel<<<(n + 255) / 256 < 1024 ? (n + 255) / 256 : 1024, 256, 0, adt::as_stream(stream)>>>(a, b, n,
                                                                                                         out);
  return adt::launch_status();
}

size_t adt_tree_accept_workspace_size(int32_t B, int32_t V) {
  (void)B;
  (void)V;
  return 0;
}

adt_status adt_tree_accept(const float* target_logits, int64_t ld_target,
                           const float* draft_logits, int64_t ld_draft, const int32_t* draft_row,
                           const int32_t* tokens, const int32_t* parents,
                           const int32_t* node_offsets, int32_t B, int32_t V, int32_t max_nodes,
                           const float* u_accept, const float* u_sample, adt_accept_mode mode,
                           float temperature, int32_t* path, int32_t max_path,
                           int32_t* accept_len, int32_t* bonus_token, void* workspace,
                           size_t workspace_bytes, void* stream) {
  adt::TraceRange trace_("adt_tree_accept");
  return accept_impl(target_logits, nullptr, ld_target, draft_logits, nullptr, ld_draft, draft_row, 0.f, tokens,
                     parents, node_offsets, B, V, max_nodes, u_accept, u_sample, mode, temperature, path, max_path,
                     accept_len, bonus_token, workspace, workspace_bytes, stream);
}

adt_status adt_tree_accept_cfg(const float* target_cond, const float* target_uncond, int64_t ld_target,
                               const float* draft_cond, const float* draft_uncond, int64_t ld_draft,
                               const int32_t* draft_row, float cfg_scale, const int32_t* tokens,
                               const int32_t* parents, const int32_t* node_offsets, int32_t B, int32_t V,
                               int32_t max_nodes, const float* u_accept, const float* u_sample,
                               adt_accept_mode mode, float temperature, int32_t* path, int32_t max_path,
                               int32_t* accept_len, int32_t* bonus_token, void* workspace,
                               size_t workspace_bytes, void* stream) {
  adt::TraceRange trace_("adt_tree_accept_cfg");
  ADT_REQUIRE(target_uncond);
  return accept_impl(target_cond, target_uncond, ld_target, draft_cond, draft_uncond, ld_draft, draft_row,
                     cfg_scale, tokens, parents, node_offsets, B, V, max_nodes, u_accept, u_sample, mode,
                     temperature, path, max_path, accept_len, bonus_token, workspace, workspace_bytes, stream);
}

}  // extern "C"
