// adt_tree_attn: tree-masked attention of the draft-tree nodes over the
// prefix KV cache and their own ancestors (Sec. 3.1: every node is verified
// conditioned on s_{1:t} and ans(t) under the tree mask; the mask is the
// T_N term of Eq. 5).
//
// Split-KV flash decoding on the 5th-generation tensor cores.  The keys a
// tree sees are cut into units of 64: ceil(L/64) prefix units plus one tree
// unit (its <= 64 nodes, masked per query row by an ancestor bitmask built
// from the parent pointers).  Grid = (splits, H, B), one CTA per SM; a CTA
// handles one (tree, head) and a contiguous share of the units.
//
// Warp roles inside a CTA (192 threads):
//   warp 4    producer: TMA tensor loads of prefix K/V chunks (128-byte
//             swizzle) into a ring of stages; the tree unit (rows of
//             k_tree / v_tree that TMA cannot bound) with cp.async;
//   warp 5    one elected thread issues tcgen05.mma: S = Q K^T into a
//             double-buffered tensor-memory tile (M = 64 queries, N = 64
//             keys), then O += P V (N = head_dim, V read MN-major);
//   warps 0-3 softmax: warp w owns query rows 16w .. 16w+15 (tensor-memory
//             lanes 32w .. 32w+15 for M = 64), read with the 16x256b shape so
//             that each thread holds two rows x 16 columns of a chunk; masks
//             branch-free, exponentiates against a lazily raised running
//             maximum (O is rescaled only when a row maximum grows by more
//             than 2^8), writes P (bf16) to shared memory for the PV
//             product; at the end they read O and l and emit the partial.
// mbarriers connect the roles; every wait is bounded and a timeout sets
// ADT_DEVERR_TIMEOUT.  The splits of one (tree, head) form a thread-block
// cluster (<= 8) and merge their partials through distributed shared
// memory; with more splits they merge through the workspace.
#include <cooperative_groups.h>
#include <cuda.h>

#include <mutex>

#include "adt_common.cuh"
#include "sm100.cuh"

namespace cg = cooperative_groups;

namespace {

constexpr int kUnit = 64;               // keys per pipeline unit
constexpr int kMaxNodes = 64;           // tree nodes (query rows) per (tree, head)
constexpr int kSoftmaxWarps = 4;
constexpr int kProducerWarp = 4;
constexpr int kMmaWarp = 5;
constexpr int kThreads = 6 * 32;
constexpr int kMaxClusterSplits = 8;    // portable cluster size
constexpr int kMaxSplits = 96;          // workspace merge: weights fit in shared memory
constexpr int kMaxStages = 8;
constexpr uint32_t kWaitLimit = 1u << 20;
constexpr uint32_t kTmemCols = 256;     // S double buffer (2 x 64 columns) + O (<= 128 columns)
constexpr uint32_t kOCol = 128;
constexpr float kLn2 = 0.69314718055994530942f;
constexpr float kLog2e = 1.44269504088896340736f;
constexpr float kRescaleThreshold = 8.0f;  // log2 units

template <int D>
struct Cfg {
  static constexpr int kBlocks = D / 64;             // 128-byte column blocks per row
  static constexpr int kBlockBytes = kUnit * 128;    // one column block of 64 rows
  static constexpr int kTileBytes = kBlocks * kBlockBytes;  // 64 rows x D bf16
  static constexpr int kStages = D == 128 ? 4 : 8;
  static constexpr int kQOff = 0;
  static constexpr int kPOff = kTileBytes;                  // two P buffers (64 x 64 bf16)
  static constexpr int kTreeOff = kPOff + 2 * kBlockBytes;    // tree unit: K tile, then V tile
  static constexpr int kStageOff = kTreeOff + 2 * kTileBytes;
  static constexpr int kStageBytes = 2 * kTileBytes;        // K tile, then V tile
  static constexpr int kDynSmem = kStageOff + kStages * kStageBytes + 1024;  // + alignment slack
  static constexpr uint32_t kIdescS = sm100::idesc_bf16_f32(64, 64, 0, 0);
  static constexpr uint32_t kIdescO = sm100::idesc_bf16_f32(64, D, 0, 1);
  static constexpr int kMergeStride = D + 4;                // fp32 per row of a parked partial
};

struct TcParams {
  const __nv_bfloat16* q;
  const __nv_bfloat16* kt;
  const __nv_bfloat16* vt;
  const int32_t* kv_len;
  const int32_t* parents;
  const int32_t* offs;
  int B, H, Hkv, group, max_kv, splits;
  int cluster_merge;
  float scale_log2;
  __nv_bfloat16* out;
  float* lse;
  float* part_o;      // [B][H][splits][64][D]   (workspace merge only)
  float2* part_ml;    // [B][H][splits][64]
  unsigned* tickets;  // [B][H]
  unsigned* err;
};

// Byte offset of 16-byte chunk `ch` (0 .. D/8-1) of row `row` in a tile of
// 128-byte column blocks with the 128-byte swizzle (the layout TMA writes).
__device__ __forceinline__ uint32_t sw128_off(int row, int ch) {
  return static_cast<uint32_t>((ch >> 3) * (kUnit * 128) + row * 128 + (((ch & 7) ^ (row & 7)) << 4));
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, int src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;\n" ::: "memory"); }

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}


// tcgen05.ld / st, shape 16x256b, 8 repetitions: for an M = 64 accumulator
// (rows 16w .. 16w+15 in lanes 32w .. 32w+15), thread (g = lane / 4,
// t = lane % 4) of warp w gets, for each 8-column block b = 0..7 starting at
// the address's column: r[4b + 0, 1] = row 16w + g, columns 8b + 2t, 8b + 2t + 1
// and r[4b + 2, 3] = the same columns of row 16w + g + 8.
__device__ __forceinline__ void tmem_ld_16x256b_x8(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.16x256b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr)
      : "memory");
}
__device__ __forceinline__ void tmem_st_16x256b_x8(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.16x256b.x8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
      "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};\n" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
      "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]),
      "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]),
      "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}

// x masked to -inf where the keep bit is 0, without branching.
__device__ __forceinline__ float mask_or_neg_inf(float x, uint32_t keep_bit) {
  const uint32_t keep = 0u - keep_bit;
  return __uint_as_float((__float_as_uint(x) & keep) | (0xFF800000u & ~keep));
}

struct Barriers {
  uint64_t q_full;
  uint64_t kv_full[kMaxStages];
  uint64_t kv_empty[kMaxStages];
  uint64_t s_full[2];
  uint64_t s_free[2];
  uint64_t p_full[2];
  uint64_t pv_done[2];
  uint64_t o_full;
};

// Bounded wait that also gives up when another role has aborted.
__device__ __forceinline__ bool wait_bar(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                         unsigned* err) {
  const uint32_t a = sm100::smem_addr(bar);
  for (uint32_t i = 0; i < kWaitLimit; ++i) {
    if (sm100::mbar_try_wait(a, parity)) return true;
    if ((i & 255u) == 255u && *abort_flag) return false;
  }
  *abort_flag = 1;
  adt::raise_error(err, ADT_DEVERR_TIMEOUT);
  return false;
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    tree_attn_tc_kernel(const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_v,
                        const TcParams p) {
  using C = Cfg<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ Barriers bars;
  __shared__ uint64_t anc[kMaxNodes];
  __shared__ uint32_t tmem_slot;
  __shared__ int s_bad;
  __shared__ int s_last;
  __shared__ volatile int s_abort;

  const int split = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int g = h / p.group;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  const int node0 = p.offs[b];
  const int n = p.offs[b + 1] - node0;
  const int L = p.kv_len[b];

  if (tid == 0) {
    s_bad = 0;
    s_abort = 0;
  }
  __syncthreads();
  // Conditions that hold for every CTA of this (tree, head): all leave here.
  if (n < 1 || n > kMaxNodes) {
    if (split == 0 && h == 0 && tid == 0) adt::raise_error(p.err, ADT_DEVERR_BAD_TREE);
    return;
  }
  if (L < 0 || L > p.max_kv) {
    if (split == 0 && h == 0 && tid == 0) adt::raise_error(p.err, ADT_DEVERR_KV_RANGE);
    return;
  }
  // Ancestor bitmask of every node: bit j of anc[t] <=> j in ans(t) or j == t.
  if (tid < kMaxNodes) {
    uint64_t m = 0;
    if (tid < n) {
      int j = tid;
      int par = p.parents[node0 + j];
      m = 1ull << j;
      if ((j == 0) != (par < 0)) s_bad = 1;
      while (par >= 0) {
        if (par >= j) {
          s_bad = 1;
          break;
        }
        m |= 1ull << par;
        j = par;
        par = p.parents[node0 + j];
        if ((j == 0) != (par < 0)) {
          s_bad = 1;
          break;
        }
      }
    }
    anc[tid] = m;
  }
  __syncthreads();
  if (s_bad) {
    if (split == 0 && h == 0 && tid == 0) adt::raise_error(p.err, ADT_DEVERR_BAD_TREE);
    return;
  }

  const int U = (L + kUnit - 1) / kUnit + 1;  // prefix units + the tree unit
  const int S = p.splits;
  const int u_begin = static_cast<int>(static_cast<int64_t>(split) * U / S);
  const int u_end = static_cast<int>(static_cast<int64_t>(split + 1) * U / S);
  const int nu = u_end - u_begin;
  // The CTA whose share ends with the tree unit processes it first (its K/V
  // are loaded with Q at the start); prefix units follow in order through
  // the TMA ring.  Iteration j handles unit unit_of(j).
  const int has_tree = (u_end == U && nu > 0) ? 1 : 0;
  const int np = nu - has_tree;  // prefix units of this CTA
  auto unit_of = [&](int j) { return has_tree ? (j == 0 ? U - 1 : u_begin + j - 1) : u_begin + j; };
  const int NS = C::kStages;

  uint8_t* sQ = smem + C::kQOff;
  uint8_t* sP = smem + C::kPOff;
  uint8_t* sStage = smem + C::kStageOff;
  uint8_t* sTree = smem + C::kTreeOff;

  if (tid == 0) {
    sm100::mbar_init(sm100::smem_addr(&bars.q_full), kSoftmaxWarps);
    for (int s = 0; s < NS; ++s) {
      sm100::mbar_init(sm100::smem_addr(&bars.kv_full[s]), 1);
      sm100::mbar_init(sm100::smem_addr(&bars.kv_empty[s]), 1);
    }
    for (int s = 0; s < 2; ++s) {
      sm100::mbar_init(sm100::smem_addr(&bars.s_full[s]), 1);
      sm100::mbar_init(sm100::smem_addr(&bars.s_free[s]), kSoftmaxWarps);
      sm100::mbar_init(sm100::smem_addr(&bars.p_full[s]), kSoftmaxWarps);
      sm100::mbar_init(sm100::smem_addr(&bars.pv_done[s]), 1);
    }
    sm100::mbar_init(sm100::smem_addr(&bars.o_full), 1);
    sm100::fence_mbar_init();
  }
  if (warp == 0) {
    sm100::tmem_alloc(sm100::smem_addr(&tmem_slot), kTmemCols);
    sm100::tmem_relinquish();
  }
  sm100::tc_fence_before();
  __syncthreads();
  sm100::tc_fence_after();
  const uint32_t tmem = tmem_slot;

  // Final row statistics of the softmax threads' two rows (a, b).
  float m_ra = -INFINITY, l_ra = 0.f, m_rb = -INFINITY, l_rb = 0.f;

  if (warp == kProducerWarp) {
    // ------------------------------------------------------------ producer
    int issued = 0;
    for (int jp = 0; jp < np; ++jp) {
      const int st = jp % NS;
      if (jp >= NS &&
          !__all_sync(adt::kFullMask, wait_bar(&bars.kv_empty[st], ((jp / NS) - 1) & 1, &s_abort, p.err)))
        break;
      if (lane == 0) {
        uint8_t* kdst = sStage + st * C::kStageBytes;
        uint8_t* vdst = kdst + C::kTileBytes;
        const uint32_t bar = sm100::smem_addr(&bars.kv_full[st]);
        sm100::mbar_arrive_expect_tx(bar, 2 * C::kTileBytes);
        const int key0 = (u_begin + jp) * kUnit;
        for (int blk = 0; blk < C::kBlocks; ++blk) {
          sm100::tma_load_4d(sm100::smem_addr(kdst + blk * C::kBlockBytes), &tm_k, blk * 64, key0, g, b, bar);
          sm100::tma_load_4d(sm100::smem_addr(vdst + blk * C::kBlockBytes), &tm_v, blk * 64, key0, g, b, bar);
        }
      }
      __syncwarp();
      ++issued;
    }
    if (s_abort && lane == 0) {
      // let every copy still in flight land before the CTA can exit
      for (int jp = (issued > NS ? issued - NS : 0); jp < issued; ++jp)
        (void)sm100::mbar_wait_bounded(sm100::smem_addr(&bars.kv_full[jp % NS]), (jp / NS) & 1, kWaitLimit);
    }
  } else if (warp == kMmaWarp) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      bool ok = wait_bar(&bars.q_full, 0, &s_abort, p.err);
      const uint32_t q_addr = sm100::smem_addr(sQ);
      const uint32_t p_addr = sm100::smem_addr(sP);
      auto issue_pv = [&](int i) -> bool {
        const int pb = i & 1;
        if (!wait_bar(&bars.p_full[pb], (i >> 1) & 1, &s_abort, p.err)) return false;
        sm100::tc_fence_after();
        const bool tree_i = has_tree && i == 0;
        const int ip = i - has_tree;
        const uint32_t v_addr = tree_i ? sm100::smem_addr(sTree + C::kTileBytes)
                                       : sm100::smem_addr(sStage + (ip % NS) * C::kStageBytes + C::kTileBytes);
#pragma unroll
        for (int kk = 0; kk < kUnit / 16; ++kk) {
          const uint64_t da = sm100::smem_desc_sw128(p_addr + pb * C::kBlockBytes + kk * 32, 16, 1024);
          const uint64_t db = sm100::smem_desc_sw128(v_addr + kk * 2048, C::kBlockBytes, 1024);
          sm100::mma_bf16_ss(tmem + kOCol, da, db, C::kIdescO, (i > 0 || kk > 0) ? 1u : 0u);
        }
        if (!tree_i) sm100::mma_commit(sm100::smem_addr(&bars.kv_empty[ip % NS]));
        sm100::mma_commit(sm100::smem_addr(&bars.pv_done[pb]));
        return true;
      };
      for (int j = 0; ok && j < nu; ++j) {
        const bool tree_j = has_tree && j == 0;
        const int jp = j - has_tree;
        const int st = jp % NS, sb = j & 1;
        if (!tree_j && !wait_bar(&bars.kv_full[st], (jp / NS) & 1, &s_abort, p.err)) break;
        if (j >= 2 && !wait_bar(&bars.s_free[sb], ((j >> 1) - 1) & 1, &s_abort, p.err)) break;
        sm100::tc_fence_after();
        const uint32_t k_addr = tree_j ? sm100::smem_addr(sTree) : sm100::smem_addr(sStage + st * C::kStageBytes);
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t off = (kk >> 2) * C::kBlockBytes + (kk & 3) * 32;
          const uint64_t da = sm100::smem_desc_sw128(q_addr + off, 16, 1024);
          const uint64_t db = sm100::smem_desc_sw128(k_addr + off, 16, 1024);
          sm100::mma_bf16_ss(tmem + sb * 64, da, db, C::kIdescS, kk > 0 ? 1u : 0u);
        }
        sm100::mma_commit(sm100::smem_addr(&bars.s_full[sb]));
        if (j >= 1 && !issue_pv(j - 1)) break;
        if (j == nu - 1 && issue_pv(j)) sm100::mma_commit(sm100::smem_addr(&bars.o_full));
      }
      if (s_abort) {
        // wait for the tensor core to finish whatever was issued
        sm100::mma_commit(sm100::smem_addr(&bars.o_full));
        (void)sm100::mbar_wait_bounded(sm100::smem_addr(&bars.o_full), 0, kWaitLimit);
      }
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ softmax warps 0-3
    // Q tile: rows node0 .. node0+63 (rows past the tree zero-filled).
    for (int i = tid; i < kUnit * (D / 8); i += kSoftmaxWarps * 32) {
      const int r = i / (D / 8), ch = i % (D / 8);
      const bool valid = r < n;
      const __nv_bfloat16* src = p.q + (static_cast<int64_t>(node0 + (valid ? r : 0)) * p.H + h) * D + ch * 8;
      cp_async16(sm100::smem_addr(sQ) + sw128_off(r, ch), src, valid ? 16 : 0);
    }
    if (has_tree) {
      // Tree unit: rows node0 .. node0+63 of k_tree / v_tree for kv head g;
      // rows past this tree are zero-filled, never read out of bounds.
      for (int i = tid; i < kUnit * (D / 8); i += kSoftmaxWarps * 32) {
        const int r = i / (D / 8), ch = i % (D / 8);
        const bool valid = r < n;
        const int64_t off = (static_cast<int64_t>(node0 + (valid ? r : 0)) * p.Hkv + g) * D + ch * 8;
        cp_async16(sm100::smem_addr(sTree) + sw128_off(r, ch), p.kt + off, valid ? 16 : 0);
        cp_async16(sm100::smem_addr(sTree + C::kTileBytes) + sw128_off(r, ch), p.vt + off, valid ? 16 : 0);
      }
    }
    cp_async_wait_all();
    sm100::fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) sm100::mbar_arrive(sm100::smem_addr(&bars.q_full));

    // Thread (g, t) = (lane / 4, lane % 4) of warp w owns rows ra = 16w + g
    // and rb = ra + 8 of the tile, columns 8b + 2t, 8b + 2t + 1 of every
    // 8-column block b (the 16x256b tensor-memory layout); the four threads
    // of a quad share a row and combine row statistics with two shuffles.
    const int g8 = lane >> 2, t4 = lane & 3;
    const int ra = warp * 16 + g8, rb = ra + 8;
    const uint64_t ama = ra < n ? anc[ra] : 0ull;
    const uint64_t amb = rb < n ? anc[rb] : 0ull;
    const uint32_t lane_base = static_cast<uint32_t>(warp * 32) << 16;
    float mua = -INFINITY, mub = -INFINITY;  // running maxima used for the exponentials
    float la = 0.f, lb = 0.f;                // this thread's share of the row sums
    for (int j = 0; j < nu; ++j) {
      const int sb = j & 1;
      if (!__all_sync(adt::kFullMask, wait_bar(&bars.s_full[sb], (j >> 1) & 1, &s_abort, p.err))) break;
      sm100::tc_fence_after();
      uint32_t r[32];
      tmem_ld_16x256b_x8(tmem + lane_base + sb * 64, r);
      sm100::tmem_wait_ld();
      // S is in registers: hand the tensor-memory buffer back to the MMA warp.
      sm100::tc_fence_before();
      __syncwarp();
      if (lane == 0) sm100::mbar_arrive(sm100::smem_addr(&bars.s_free[sb]));

      const int u = unit_of(j);
      // Which of the chunk's 64 keys a row sees (the prefix up to L, or the
      // row's ancestors and itself in the tree unit), applied with bit
      // operations so no lane branches on it.
      uint64_t vma, vmb;
      if (u == U - 1) {
        vma = ama;
        vmb = amb;
      } else {
        const int kl = L - u * kUnit;  // >= 1 for every prefix unit
        vma = vmb = kl >= 64 ? ~0ull : ((1ull << kl) - 1ull);
      }
      const float scale = p.scale_log2;
      float xa[16], xb[16];
      float mxa = -INFINITY, mxb = -INFINITY;
#pragma unroll
      for (int bk = 0; bk < 8; ++bk) {
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const int c = 8 * bk + 2 * t4 + e;
          xa[2 * bk + e] = mask_or_neg_inf(__uint_as_float(r[4 * bk + e]) * scale,
                                           static_cast<uint32_t>(vma >> c) & 1u);
          xb[2 * bk + e] = mask_or_neg_inf(__uint_as_float(r[4 * bk + 2 + e]) * scale,
                                           static_cast<uint32_t>(vmb >> c) & 1u);
          mxa = fmaxf(mxa, xa[2 * bk + e]);
          mxb = fmaxf(mxb, xb[2 * bk + e]);
        }
      }
      mxa = fmaxf(mxa, __shfl_xor_sync(adt::kFullMask, mxa, 1));
      mxa = fmaxf(mxa, __shfl_xor_sync(adt::kFullMask, mxa, 2));
      mxb = fmaxf(mxb, __shfl_xor_sync(adt::kFullMask, mxb, 1));
      mxb = fmaxf(mxb, __shfl_xor_sync(adt::kFullMask, mxb, 2));
      // Lazily raised maximum: O is rescaled only when a row's maximum grows
      // by more than 2^8 over the one its exponentials were taken against.
      const bool needa = mxa > mua + kRescaleThreshold, needb = mxb > mub + kRescaleThreshold;
      const float nma = needa ? mxa : mua, nmb = needb ? mxb : mub;
      const float alpha_a = needa ? exp2f(mua - nma) : 1.f, alpha_b = needb ? exp2f(mub - nmb) : 1.f;
      const float base_a = nma == -INFINITY ? 0.f : nma, base_b = nmb == -INFINITY ? 0.f : nmb;
      float rsa = 0.f, rsb = 0.f;
      uint32_t pa[8], pb[8];
#pragma unroll
      for (int bk = 0; bk < 8; ++bk) {
        const float a0 = exp2f(xa[2 * bk] - base_a), a1 = exp2f(xa[2 * bk + 1] - base_a);
        const float b0 = exp2f(xb[2 * bk] - base_b), b1 = exp2f(xb[2 * bk + 1] - base_b);
        rsa += a0 + a1;
        rsb += b0 + b1;
        pa[bk] = pack_bf16x2(a0, a1);
        pb[bk] = pack_bf16x2(b0, b1);
      }
      la = la * alpha_a + rsa;
      lb = lb * alpha_b + rsb;
      // P buffer sb was last read by the PV product of chunk j - 2.
      if (j >= 2 &&
          !__all_sync(adt::kFullMask, wait_bar(&bars.pv_done[sb], ((j >> 1) - 1) & 1, &s_abort, p.err)))
        break;
      {
        const uint32_t pbase = sm100::smem_addr(sP + sb * C::kBlockBytes);
        const uint32_t rowa = pbase + ra * 128 + t4 * 4, rowb = pbase + rb * 128 + t4 * 4;
#pragma unroll
        for (int bk = 0; bk < 8; ++bk) {
          asm volatile("st.shared.b32 [%0], %1;\n" ::"r"(rowa + (((bk ^ ra) & 7) << 4)), "r"(pa[bk]) : "memory");
          asm volatile("st.shared.b32 [%0], %1;\n" ::"r"(rowb + (((bk ^ rb) & 7) << 4)), "r"(pb[bk]) : "memory");
        }
      }
      sm100::fence_proxy_async_smem();
      // Raise O to the new maxima (rare): needs the previous PV product done.
      if (j > 0 && __any_sync(adt::kFullMask, needa || needb)) {
        if (!__all_sync(adt::kFullMask,
                        wait_bar(&bars.pv_done[(j - 1) & 1], ((j - 1) >> 1) & 1, &s_abort, p.err)))
          break;
        sm100::tc_fence_after();
#pragma unroll 1
        for (int c0 = 0; c0 < D; c0 += 64) {
          uint32_t o[32];
          tmem_ld_16x256b_x8(tmem + lane_base + kOCol + c0, o);
          sm100::tmem_wait_ld();
#pragma unroll
          for (int bk = 0; bk < 8; ++bk) {
            o[4 * bk + 0] = __float_as_uint(__uint_as_float(o[4 * bk + 0]) * alpha_a);
            o[4 * bk + 1] = __float_as_uint(__uint_as_float(o[4 * bk + 1]) * alpha_a);
            o[4 * bk + 2] = __float_as_uint(__uint_as_float(o[4 * bk + 2]) * alpha_b);
            o[4 * bk + 3] = __float_as_uint(__uint_as_float(o[4 * bk + 3]) * alpha_b);
          }
          tmem_st_16x256b_x8(tmem + lane_base + kOCol + c0, o);
        }
        sm100::tmem_wait_st();
      }
      mua = nma;
      mub = nmb;
      sm100::tc_fence_before();
      __syncwarp();
      if (lane == 0) sm100::mbar_arrive(sm100::smem_addr(&bars.p_full[sb]));
    }
    // Full row sums: add the four shares of each quad.
    la += __shfl_xor_sync(adt::kFullMask, la, 1);
    la += __shfl_xor_sync(adt::kFullMask, la, 2);
    lb += __shfl_xor_sync(adt::kFullMask, lb, 1);
    lb += __shfl_xor_sync(adt::kFullMask, lb, 2);
    m_ra = mua;
    l_ra = la;
    m_rb = mub;
    l_rb = lb;
  }

  // ------------------------------------------------------------ epilogue
  // Park this split's partial (O unnormalised, m, l) in shared memory (the
  // stage ring is idle once O is complete), then merge.
  constexpr int MS = C::kMergeStride;
  float* so = reinterpret_cast<float*>(sStage);                         // [64][MS]
  float2* sml = reinterpret_cast<float2*>(sStage + kMaxNodes * MS * 4);  // [64]
  float* sw = reinterpret_cast<float*>(sStage + kMaxNodes * MS * 4 + kMaxNodes * 8);  // weights
  if (warp < kSoftmaxWarps) {
    const int g8 = lane >> 2, t4 = lane & 3;
    const int ra = warp * 16 + g8, rb = ra + 8;
    // A split without key units (kv_len shorter than max_kv) contributes
    // nothing: weight 0, zero partial.
    const bool ok = nu > 0 && !s_abort && __all_sync(adt::kFullMask, wait_bar(&bars.o_full, 0, &s_abort, p.err));
    if (ok) {
      sm100::tc_fence_after();
      const uint32_t lane_base = static_cast<uint32_t>(warp * 32) << 16;
#pragma unroll 1
      for (int c0 = 0; c0 < D; c0 += 64) {
        uint32_t o[32];
        tmem_ld_16x256b_x8(tmem + lane_base + kOCol + c0, o);
        sm100::tmem_wait_ld();
#pragma unroll
        for (int bk = 0; bk < 8; ++bk) {
          const int c = c0 + 8 * bk + 2 * t4;
          if (ra < n)
            *reinterpret_cast<float2*>(so + ra * MS + c) = make_float2(__uint_as_float(o[4 * bk]), __uint_as_float(o[4 * bk + 1]));
          if (rb < n)
            *reinterpret_cast<float2*>(so + rb * MS + c) =
                make_float2(__uint_as_float(o[4 * bk + 2]), __uint_as_float(o[4 * bk + 3]));
        }
      }
      if (t4 == 0) {
        if (ra < n) sml[ra] = make_float2(m_ra, l_ra);
        if (rb < n) sml[rb] = make_float2(m_rb, l_rb);
      }
    } else if (t4 == 0) {
      for (int half = 0; half < 2; ++half) {
        const int rr = half ? rb : ra;
        if (rr < n) {
          for (int c = 0; c < D; c += 4) *reinterpret_cast<float4*>(so + rr * MS + c) = make_float4(0.f, 0.f, 0.f, 0.f);
          sml[rr] = make_float2(-INFINITY, 0.f);
        }
      }
    }
  }
  sm100::tc_fence_before();
  __syncthreads();
  if (warp == 0) sm100::tmem_dealloc(tmem, kTmemCols);

  const int64_t bh = static_cast<int64_t>(b) * p.H + h;
  constexpr int kC4 = D / 4;
  if (p.cluster_merge) {
    // CTA r of the cluster merges rows r, r + S, ... from every peer's partial.
    cg::cluster_group cl = cg::this_cluster();
    cl.sync();
    const int rank = static_cast<int>(cl.block_rank());
    const int rows_mine = rank < n ? (n - rank + S - 1) / S : 0;
    if (tid < rows_mine) {
      const int rr = rank + S * tid;
      float M = -INFINITY;
      for (int c = 0; c < S; ++c) M = fmaxf(M, cl.map_shared_rank(sml, c)[rr].x);
      float lt = 0.f;
      for (int c = 0; c < S; ++c) {
        const float2 ml = cl.map_shared_rank(sml, c)[rr];
        const float w = ml.x == -INFINITY ? 0.f : exp2f(ml.x - M);
        sw[tid * S + c] = w;
        lt += w * ml.y;
      }
      const float inv = 1.f / lt;
      for (int c = 0; c < S; ++c) sw[tid * S + c] *= inv;
      if (p.lse) p.lse[static_cast<int64_t>(node0 + rr) * p.H + h] = (M + log2f(lt)) * kLn2;
    }
    __syncthreads();
    for (int idx = tid; idx < rows_mine * kC4; idx += kThreads) {
      const int i = idx / kC4, c4 = idx % kC4;
      const int rr = rank + S * i;
      // Issue every peer's load before combining (latency, not bandwidth, bound).
      float4 v[kMaxClusterSplits];
#pragma unroll
      for (int c = 0; c < kMaxClusterSplits; ++c) {
        v[c] = make_float4(0.f, 0.f, 0.f, 0.f);
        if (c < S && sw[i * S + c] != 0.f)
          v[c] = *reinterpret_cast<const float4*>(cl.map_shared_rank(so, c) + rr * MS + c4 * 4);
      }
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
      for (int c = 0; c < kMaxClusterSplits; ++c) {
        const float w = c < S ? sw[i * S + c] : 0.f;
        acc.x += w * v[c].x;
        acc.y += w * v[c].y;
        acc.z += w * v[c].z;
        acc.w += w * v[c].w;
      }
      __nv_bfloat16* dst = p.out + (static_cast<int64_t>(node0 + rr) * p.H + h) * D + c4 * 4;
      uint2 pk;
      pk.x = pack_bf16x2(acc.x, acc.y);
      pk.y = pack_bf16x2(acc.z, acc.w);
      *reinterpret_cast<uint2*>(dst) = pk;
    }
    cl.sync();  // peers may still be reading this CTA's partial
    return;
  }

  // More splits than a portable cluster holds: partials go to the workspace
  // and the CTA that finishes a (tree, head) last merges them.
  float* po = p.part_o + (bh * S + split) * kMaxNodes * D;
  float2* pml = p.part_ml + (bh * S + split) * kMaxNodes;
  for (int idx = tid; idx < n * kC4; idx += kThreads) {
    const int rr = idx / kC4, c4 = idx % kC4;
    *reinterpret_cast<float4*>(po + rr * D + c4 * 4) = *reinterpret_cast<const float4*>(so + rr * MS + c4 * 4);
  }
  if (tid < n) pml[tid] = sml[tid];
  __threadfence();
  __syncthreads();
  if (tid == 0) s_last = atomicAdd(p.tickets + bh, 1u) == static_cast<unsigned>(S - 1);
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  const float* po_bh = p.part_o + bh * S * kMaxNodes * D;
  const float2* pml_bh = p.part_ml + bh * S * kMaxNodes;
  float* wsm = reinterpret_cast<float*>(sStage);  // [64][S]; the parked partial is in global now
  __syncthreads();
  if (tid < n) {
    float M = -INFINITY;
    for (int sp = 0; sp < S; ++sp) M = fmaxf(M, __ldcg(&pml_bh[sp * kMaxNodes + tid]).x);
    float lt = 0.f;
    for (int sp = 0; sp < S; ++sp) {
      const float2 ml = __ldcg(&pml_bh[sp * kMaxNodes + tid]);
      const float w = ml.x == -INFINITY ? 0.f : exp2f(ml.x - M);
      wsm[tid * S + sp] = w;
      lt += w * ml.y;
    }
    const float inv = 1.f / lt;
    for (int sp = 0; sp < S; ++sp) wsm[tid * S + sp] *= inv;
    if (p.lse) p.lse[static_cast<int64_t>(node0 + tid) * p.H + h] = (M + log2f(lt)) * kLn2;
  }
  __syncthreads();
  constexpr int kStride4 = kMaxNodes * D / 4;
  for (int idx = tid; idx < n * kC4; idx += kThreads) {
    const int rr = idx / kC4, c4 = idx % kC4;
    const float4* src = reinterpret_cast<const float4*>(po_bh + rr * D) + c4;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    int sp = 0;
    for (; sp + 4 <= S; sp += 4) {
      float4 v[4];
#pragma unroll
      for (int q4 = 0; q4 < 4; ++q4) v[q4] = __ldcg(src + (sp + q4) * kStride4);
#pragma unroll
      for (int q4 = 0; q4 < 4; ++q4) {
        const float w = wsm[rr * S + sp + q4];
        acc.x += w * v[q4].x;
        acc.y += w * v[q4].y;
        acc.z += w * v[q4].z;
        acc.w += w * v[q4].w;
      }
    }
    for (; sp < S; ++sp) {
      const float4 v = __ldcg(src + sp * kStride4);
      const float w = wsm[rr * S + sp];
      acc.x += w * v.x;
      acc.y += w * v.y;
      acc.z += w * v.z;
      acc.w += w * v.w;
    }
    __nv_bfloat16* dst = p.out + (static_cast<int64_t>(node0 + rr) * p.H + h) * D + c4 * 4;
    uint2 pk;
    pk.x = pack_bf16x2(acc.x, acc.y);
    pk.y = pack_bf16x2(acc.z, acc.w);
    *reinterpret_cast<uint2*>(dst) = pk;
  }
  if (tid == 0) p.tickets[bh] = 0u;
}

// ---------------------------------------------------------------- host side

// Splits per (tree, head): about one CTA per SM, at most one split per unit
// of keys.  Up to kMaxClusterSplits splits form a cluster; the count is
// lowered until all B*H clusters are co-resident (GPC sizes decide how many
// clusters of a given size fit at once).  Many splits (small B*H, long
// prefixes) merge through the workspace instead.
int max_active_clusters(int D, int cluster, int dev);

int choose_splits(int sm_count, int B, int H, int D, int max_kv, int dev) {
  const int units = (max_kv + kUnit - 1) / kUnit + 1;
  const int bh = B * H;
  int s = sm_count / bh;
  if (s < 1) s = 1;
  if (s > units) s = units;
  if (s >= 2 * kMaxClusterSplits) return s > kMaxSplits ? kMaxSplits : s;
  if (s > kMaxClusterSplits) s = kMaxClusterSplits;
  while (s > 1 && max_active_clusters(D, s, dev) < bh) --s;
  return s;
}

// Workspace layout.  The per-(tree, head) completion tickets sit at fixed
// offsets at the start (room for kMaxBH pairs), so calls of any shape can
// share one workspace; the partials after them are rewritten before use.
constexpr int kMaxBH = 65536;

struct WsLayout {
  size_t tickets, part_ml, part_o, total;
};

WsLayout ws_layout(int B, int H, int D, int splits) {
  WsLayout w{};
  const size_t bhs = static_cast<size_t>(B) * H * splits;
  w.tickets = 0;
  w.part_ml = adt::align_up(static_cast<size_t>(kMaxBH) * sizeof(unsigned), 256);
  w.part_o = adt::align_up(w.part_ml + bhs * kMaxNodes * sizeof(float2), 256);
  w.total = adt::align_up(w.part_o + bhs * kMaxNodes * D * sizeof(float), 256);
  return w;
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

std::once_flag g_encode_once;
EncodeTiledFn g_encode = nullptr;

void load_encode() {
  void* fn = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
          cudaSuccess &&
      q == cudaDriverEntryPointSuccess)
    g_encode = reinterpret_cast<EncodeTiledFn>(fn);
}

// 4-D map of a cache (d, pos, kv head, tree) with the 128-byte swizzle and
// 64 x 64 boxes; positions at or past max_kv read as zero.
adt_status make_cache_map(CUtensorMap* map, const void* base, int D, int max_kv, int Hkv, int B, int64_t sh,
                          int64_t sb) {
  std::call_once(g_encode_once, load_encode);
  if (!g_encode) return ADT_ERR_CUDA;
  const int64_t span = static_cast<int64_t>(max_kv > 0 ? max_kv : 1);
  cuuint64_t dims[4] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(span), static_cast<cuuint64_t>(Hkv),
                        static_cast<cuuint64_t>(B)};
  cuuint64_t strides[3] = {static_cast<cuuint64_t>(D) * 2, static_cast<cuuint64_t>(sh > 0 ? sh : span * D) * 2,
                           static_cast<cuuint64_t>(sb > 0 ? sb : span * D * Hkv) * 2};
  cuuint32_t box[4] = {64, kUnit, 1, 1};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? ADT_OK : ADT_ERR_INVALID_ARG;
}

int max_active_clusters(int D, int cluster, int dev) {
  static int cache[64][2][kMaxClusterSplits + 1];  // 0 = not queried yet
  int& slot = cache[dev & 63][D == 128 ? 1 : 0][cluster];
  int v = __atomic_load_n(&slot, __ATOMIC_ACQUIRE);
  if (v) return v - 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(cluster), 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = static_cast<unsigned>(cluster);
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int num = 0;
  cudaError_t e;
  if (D == 128) {
    cudaFuncSetAttribute(tree_attn_tc_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg<128>::kDynSmem);
    cfg.dynamicSmemBytes = Cfg<128>::kDynSmem;
    e = cudaOccupancyMaxActiveClusters(&num, tree_attn_tc_kernel<128>, &cfg);
  } else {
    cudaFuncSetAttribute(tree_attn_tc_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg<64>::kDynSmem);
    cfg.dynamicSmemBytes = Cfg<64>::kDynSmem;
    e = cudaOccupancyMaxActiveClusters(&num, tree_attn_tc_kernel<64>, &cfg);
  }
  if (e != cudaSuccess) {
    (void)cudaGetLastError();
    num = 0;
  }
  __atomic_store_n(&slot, num + 1, __ATOMIC_RELEASE);
  return num;
}

template <int D>
adt_status launch(TcParams prm, const void* k_cache, const void* v_cache, int64_t sb, int64_t sh, cudaStream_t st,
                  int dev) {
  static unsigned configured[2] = {0u, 0u};  // bit per device (< 64)
  const unsigned bit = 1u << (dev & 31);
  unsigned& word = configured[dev >> 5];
  if (!(__atomic_load_n(&word, __ATOMIC_ACQUIRE) & bit)) {
    ADT_CUDA_TRY(cudaFuncSetAttribute(tree_attn_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      Cfg<D>::kDynSmem));
    __atomic_fetch_or(&word, bit, __ATOMIC_ACQ_REL);
  }
  CUtensorMap tm_k, tm_v;
  adt_status s1 = make_cache_map(&tm_k, k_cache, D, prm.max_kv, prm.Hkv, prm.B, sh, sb);
  if (s1 != ADT_OK) return s1;
  s1 = make_cache_map(&tm_v, v_cache, D, prm.max_kv, prm.Hkv, prm.B, sh, sb);
  if (s1 != ADT_OK) return s1;
  prm.cluster_merge = prm.splits <= kMaxClusterSplits ? 1 : 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(prm.splits), static_cast<unsigned>(prm.H), static_cast<unsigned>(prm.B));
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = Cfg<D>::kDynSmem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = prm.cluster_merge ? static_cast<unsigned>(prm.splits) : 1u;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  ADT_CUDA_TRY(cudaLaunchKernelEx(&cfg, tree_attn_tc_kernel<D>, tm_k, tm_v, prm));
  return adt::launch_status();
}

// Shared host checks of both entry points.
adt_status check_args(const adt_bf16* q, const adt_bf16* k_cache, const adt_bf16* v_cache, const int32_t* kv_len,
                      int64_t sb, int64_t sh, const adt_bf16* k_tree, const adt_bf16* v_tree,
                      const int32_t* parents, const int32_t* node_offsets, int32_t B, int32_t H, int32_t Hkv,
                      int32_t D, int32_t max_nodes, int32_t max_kv, float scale, const adt_bf16* out) {
  ADT_REQUIRE(q && k_cache && v_cache && kv_len && k_tree && v_tree && parents && node_offsets && out);
  ADT_REQUIRE(B >= 1 && H >= 1 && Hkv >= 1 && H % Hkv == 0);
  ADT_REQUIRE(static_cast<int64_t>(B) * H <= kMaxBH && B <= 65535 && H <= 65535);
  ADT_REQUIRE(max_nodes >= 1 && max_kv >= 0 && max_kv < (1 << 30));
  ADT_REQUIRE(scale > 0.f && scale < 1e30f);
  if (D != 64 && D != 128) return ADT_ERR_UNSUPPORTED;
  if (max_nodes > kMaxNodes) return ADT_ERR_UNSUPPORTED;
  ADT_REQUIRE(sb >= 0 && sh >= 0 && sb % 8 == 0 && sh % 8 == 0);
  ADT_REQUIRE(Hkv == 1 || sh >= static_cast<int64_t>(max_kv) * D);
  ADT_REQUIRE(B == 1 || sb >= static_cast<int64_t>(max_kv) * D);
  ADT_REQUIRE(adt::aligned16(q) && adt::aligned16(k_cache) && adt::aligned16(v_cache) && adt::aligned16(k_tree) &&
              adt::aligned16(v_tree) && adt::aligned16(out));
  return ADT_OK;
}

TcParams make_params(const adt_bf16* q, const int32_t* kv_len, const adt_bf16* k_tree, const adt_bf16* v_tree,
                     const int32_t* parents, const int32_t* node_offsets, int B, int H, int Hkv, int max_kv,
                     int splits, float scale, adt_bf16* out, float* lse, unsigned* err) {
  TcParams prm{};
  prm.q = reinterpret_cast<const __nv_bfloat16*>(q);
  prm.kt = reinterpret_cast<const __nv_bfloat16*>(k_tree);
  prm.vt = reinterpret_cast<const __nv_bfloat16*>(v_tree);
  prm.kv_len = kv_len;
  prm.parents = parents;
  prm.offs = node_offsets;
  prm.B = B;
  prm.H = H;
  prm.Hkv = Hkv;
  prm.group = H / Hkv;
  prm.max_kv = max_kv;
  prm.splits = splits;
  prm.scale_log2 = scale * kLog2e;
  prm.out = reinterpret_cast<__nv_bfloat16*>(out);
  prm.lse = lse;
  prm.err = err;
  return prm;
}

}  // namespace

extern "C" {

size_t adt_tree_attn_workspace_size(int32_t B, int32_t H, int32_t D, int32_t max_nodes,
                                    int32_t max_kv) {
  (void)max_nodes;
  if (B < 1 || H < 1 || (D != 64 && D != 128) || max_kv < 0 || static_cast<int64_t>(B) * H > kMaxBH) return 0;
  adt::DeviceInfo info;
  if (adt::device_info(&info) != ADT_OK) return 0;
  return ws_layout(B, H, D, choose_splits(info.sm_count, B, H, D, max_kv, info.device)).total;
}

adt_status adt_tree_attn(const adt_bf16* q, const adt_bf16* k_cache, const adt_bf16* v_cache,
                         const int32_t* kv_len, int64_t cache_stride_b, int64_t cache_stride_h,
                         const adt_bf16* k_tree, const adt_bf16* v_tree, const int32_t* parents,
                         const int32_t* node_offsets, int32_t B, int32_t H, int32_t Hkv, int32_t D,
                         int32_t max_nodes, int32_t max_kv, float softmax_scale, adt_bf16* out,
                         float* lse, void* workspace, size_t workspace_bytes, void* stream) {
  adt_status st = check_args(q, k_cache, v_cache, kv_len, cache_stride_b, cache_stride_h, k_tree, v_tree, parents,
                             node_offsets, B, H, Hkv, D, max_nodes, max_kv, softmax_scale, out);
  if (st != ADT_OK) return st;
  adt::DeviceInfo info;
  st = adt::device_info(&info);
  if (st != ADT_OK) return st;
  const int splits = choose_splits(info.sm_count, B, H, D, max_kv, info.device);
  const WsLayout w = ws_layout(B, H, D, splits);
  if (!workspace || workspace_bytes < w.total || !adt::aligned16(workspace)) return ADT_ERR_WORKSPACE;
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  TcParams prm = make_params(q, kv_len, k_tree, v_tree, parents, node_offsets, B, H, Hkv, max_kv, splits,
                             softmax_scale, out, lse, info.error_word);
  prm.part_o = reinterpret_cast<float*>(ws + w.part_o);
  prm.part_ml = reinterpret_cast<float2*>(ws + w.part_ml);
  prm.tickets = reinterpret_cast<unsigned*>(ws + w.tickets);
  cudaStream_t s = adt::as_stream(stream);
  return D == 128 ? launch<128>(prm, k_cache, v_cache, cache_stride_b, cache_stride_h, s, info.device)
                  : launch<64>(prm, k_cache, v_cache, cache_stride_b, cache_stride_h, s, info.device);
}

}  // extern "C"

// ---------------------------------------------------------------------------
// adt_tree_attn_noalloc: the same tree attention for callers that cannot
// allocate device memory themselves, for example a plugin inside a serving
// engine whose host owns every device allocation, or code on a latency-
// critical thread that must not call cudaMalloc (it can synchronise the
// device).  The scratch that adt_tree_attn takes as a workspace (split
// partials and completion tickets) lives in one fixed, per-device static
// array instead.
// ---------------------------------------------------------------------------

// 8 MiB of scratch, held by every GPU that loads the library until the
// process exits.  Shared by all calls on a device: calls that overlap on the
// GPU (different streams, or different host threads) race on it.
static constexpr size_t kNoAllocScratchBytes = size_t(8) << 20;
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

namespace {

constexpr int kNoAllocMaxDevices = 64;
std::once_flag g_noalloc_once[kNoAllocMaxDevices];
void* g_noalloc_ptr[kNoAllocMaxDevices];
cudaError_t g_noalloc_status[kNoAllocMaxDevices];

// Runs once per device, with that device current: the array's name is a
// host-side stand-in in host code, so the kernel needs its device address.
void noalloc_setup(int dev) {
  void* p = nullptr;
  g_noalloc_status[dev] = cudaGetSymbolAddress(&p, g_noalloc_scratch);
  g_noalloc_ptr[dev] = p;
}

struct NoAllocLayout {
  size_t tickets, part_ml, part_o, total;
};

NoAllocLayout noalloc_layout(int B, int H, int D, int splits) {
  NoAllocLayout w{};
  const size_t bh = static_cast<size_t>(B) * H;
  const size_t bhs = bh * splits;
  w.tickets = 0;
  w.part_ml = adt::align_up(bh * sizeof(unsigned), 256);
  w.part_o = adt::align_up(w.part_ml + bhs * kMaxNodes * sizeof(float2), 256);
  w.total = adt::align_up(w.part_o + bhs * kMaxNodes * D * sizeof(float), 256);
  return w;
}

}  // namespace

extern "C" adt_status adt_tree_attn_noalloc(const adt_bf16* q, const adt_bf16* k_cache,
                                            const adt_bf16* v_cache, const int32_t* kv_len,
                                            int64_t cache_stride_b, int64_t cache_stride_h,
                                            const adt_bf16* k_tree, const adt_bf16* v_tree,
                                            const int32_t* parents, const int32_t* node_offsets,
                                            int32_t B, int32_t H, int32_t Hkv, int32_t D,
                                            int32_t max_nodes, int32_t max_kv, float softmax_scale,
                                            adt_bf16* out, float* lse, void* stream) {
  adt_status st = check_args(q, k_cache, v_cache, kv_len, cache_stride_b, cache_stride_h, k_tree, v_tree, parents,
                             node_offsets, B, H, Hkv, D, max_nodes, max_kv, softmax_scale, out);
  if (st != ADT_OK) return st;
  adt::DeviceInfo info;
  st = adt::device_info(&info);
  if (st != ADT_OK) return st;
  if (info.device < 0 || info.device >= kNoAllocMaxDevices) return ADT_ERR_UNSUPPORTED;
  std::call_once(g_noalloc_once[info.device], noalloc_setup, info.device);
  if (g_noalloc_status[info.device] != cudaSuccess || !g_noalloc_ptr[info.device]) return ADT_ERR_CUDA;
  // As many splits as the usual heuristic picks, fewer if the partials would
  // not fit; a shape that does not fit even unsplit is rejected.
  int splits = choose_splits(info.sm_count, B, H, D, max_kv, info.device);
  while (splits > 1 && noalloc_layout(B, H, D, splits).total > kNoAllocScratchBytes) --splits;
  const NoAllocLayout w = noalloc_layout(B, H, D, splits);
  if (w.total > kNoAllocScratchBytes) return ADT_ERR_WORKSPACE;
  uint8_t* ws = static_cast<uint8_t*>(g_noalloc_ptr[info.device]);
  cudaStream_t s = adt::as_stream(stream);
  // The array keeps the previous call's contents: the tickets must start at zero.
  ADT_CUDA_TRY(cudaMemsetAsync(ws + w.tickets, 0, static_cast<size_t>(B) * H * sizeof(unsigned), s));
  TcParams prm = make_params(q, kv_len, k_tree, v_tree, parents, node_offsets, B, H, Hkv, max_kv, splits,
                             softmax_scale, out, lse, info.error_word);
  prm.part_o = reinterpret_cast<float*>(ws + w.part_o);
  prm.part_ml = reinterpret_cast<float2*>(ws + w.part_ml);
  prm.tickets = reinterpret_cast<unsigned*>(ws + w.tickets);
  return D == 128 ? launch<128>(prm, k_cache, v_cache, cache_stride_b, cache_stride_h, s, info.device)
                  : launch<64>(prm, k_cache, v_cache, cache_stride_b, cache_stride_h, s, info.device);
}
