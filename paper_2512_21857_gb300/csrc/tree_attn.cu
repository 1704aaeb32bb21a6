// adt_tree_attn: tree-masked attention of the draft-tree nodes over the
// prefix KV cache and their own ancestors (Sec. 3.1: every node is verified
// conditioned on s_{1:t} and ans(t) under the tree mask; the mask is the
// T_N term of Eq. 5).
//
// Split-KV flash decoding on the 5th-generation tensor cores.  A tree's
// nodes (<= 256) are cut into query tiles of 64 rows; the keys a tile sees
// are cut into units of 64: ceil(L/64) prefix units plus the tree units up
// to its own (a node's ancestors come before it), masked per query row by an
// ancestor bitmask, one 64-bit word per tree unit, built from the parent
// pointers.  Grid = (splits, H, B x tiles), one CTA per SM; a CTA handles one
// (tree, head, tile) and a contiguous share of the units, which it walks in
// chunks of two units (128 keys): its tree chunks first (their K/V are
// loaded with Q), then its prefix chunks.
//
// Warp roles inside a CTA (256 threads; one thread of each of warps 4-7):
//   warp 4    TMA tensor loads of prefix K (boxes of 128 keys x 64 columns,
//             128-byte swizzle) into a ring of 128-key stages;
//   warp 5    tcgen05.mma S = Q K^T into one of two tensor-memory tiles
//             (M = 64 queries, N = 128 keys), back to back (softmax warp 0
//             frees each K tile once it sees its S product done);
//   warp 6    TMA loads of prefix V into the same stages;
//   warp 7    tcgen05.mma O += P V (N = head_dim, V read MN-major);
//   warps 0-3 softmax: warp w owns query rows 16w .. 16w+15 (tensor-memory
//             lanes 32w .. 32w+15 for M = 64), read with the 16x256b shape so
//             that each thread holds two rows; exponentiates against a lazily
//             raised running maximum (O is rescaled only when a row maximum
//             grows by more than 2^8), writes P (bf16) with stmatrix for the
//             PV product, and at the end reads O and l for the merge.
// K and V of a stage are released separately (K when S is done, V and the P
// buffer when PV is done), and S and PV are issued by different threads, so
// loads of later chunks never queue behind the softmax of earlier ones.
// Every mbarrier wait is bounded; a timeout sets ADT_DEVERR_TIMEOUT.
//
// The splits of one (tree, head) form a thread-block cluster (<= 8).  Each
// split pushes its partial rows (O, running max, row sum) into the shared
// memory of the split that owns those rows, which then merges them locally;
// at D = 128 a row travels as O / l in fp16 with a power-of-two scale (half
// the bytes of fp32, which the copies between SMs are bound by).  With more
// splits they merge through the workspace.
#include <cooperative_groups.h>
#include <cuda.h>
#include <cuda_fp16.h>

#include <mutex>

#include "adt_common.cuh"
#include "sm100.cuh"

namespace cg = cooperative_groups;

namespace {

constexpr int kUnit = 64;               // keys per split unit; the tree unit
constexpr int kChunk = 128;             // keys per pipeline chunk
constexpr int kMaxNodes = 64;           // query rows per CTA: one tile of a tree's nodes
constexpr int kMaxTreeNodes = 256;      // nodes per tree: up to four query tiles
constexpr int kMaxTreeUnits = kMaxTreeNodes / kUnit;
static_assert(kMaxTreeUnits == 4, "the ancestor walk keeps four mask words");
constexpr int kSoftmaxWarps = 4;
constexpr int kKLoadWarp = 4;
constexpr int kSMmaWarp = 5;
constexpr int kVLoadWarp = 6;
constexpr int kPvMmaWarp = 7;
constexpr int kThreads = 8 * 32;
constexpr int kMaxClusterSplits = 8;    // portable cluster size
constexpr int kMaxSplits = 96;          // workspace merge: weights fit in shared memory
constexpr int kMaxStages = 4;
constexpr uint32_t kWaitLimit = 1u << 20;
constexpr int kTmaRows = 1 << 24;       // node extent of the Q / tree tensor maps (boxes are kept inside the buffers)
constexpr uint32_t kTmemCols = 512;     // two S tiles of 128 columns, O (<= 128 columns), row sums
constexpr uint32_t kSCols = 128;
constexpr uint32_t kOCol = 256;
constexpr uint32_t kLCols = 16;         // P times a tile of ones: every column holds the row sum
constexpr float kLn2 = 0.69314718055994530942f;
constexpr float kLog2e = 1.44269504088896340736f;
constexpr float kRescaleThreshold = 8.0f;  // log2 units

template <int D>
struct Cfg {
  static constexpr int kBlocks = D / 64;                 // 128-byte column blocks per row
  static constexpr int kBlock64 = kUnit * 128;           // one column block of 64 rows
  static constexpr int kBlock128 = kChunk * 128;         // one column block of 128 rows
  static constexpr int kTreeTile = kBlocks * kBlock64;   // 64 rows x D
  static constexpr int kStageTile = kBlocks * kBlock128; // 128 rows x D
  static constexpr int kStageBytes = 2 * kStageTile;     // K tile, then V tile
  static constexpr int kPBytes = 2 * kBlock64;           // 64 query rows x 128 keys
  static constexpr int kStages = D == 128 ? 2 : 4;
  // A partial row of the cluster merge, in 32-bit words.  D = 128: D fp16
  // values (O / l scaled by 2^-e), then m, l (fp32) and e (int32), padded to
  // 16 bytes; D = 64: D fp32 values (O), m, l, padding (distributed shared
  // memory moves its rows fast enough that the conversions would cost more
  // than the halved bytes save).
  static constexpr bool kHalfRows = D == 128;
  static constexpr int kRowStride = kHalfRows ? D / 2 + 4 : D + 8;
  static constexpr int kQOff = 0;
  static constexpr int kPOff = kTreeTile;                // Q is 64 rows x D, like a tree tile
  static constexpr int kStageOff = kPOff + 2 * kPBytes;  // the tree unit's K/V go to slot 0
  static constexpr int kSlotOff = kStageOff + kStages * kStageBytes;  // incoming rows of the merge
  static constexpr int kSlotBytes = (kMaxNodes + kMaxClusterSplits) * kRowStride * 4;
  static constexpr int kOnesOff = (kSlotOff + kSlotBytes + 1023) / 1024 * 1024;  // 16 rows of ones (bf16)
  static constexpr int kOnesBytes = 16 * 128;
  static constexpr int kDynSmem = kOnesOff + kOnesBytes + 1024;  // + alignment slack
  static constexpr uint32_t kLCol = kOCol + D;
  static constexpr uint32_t kIdescS128 = sm100::idesc_bf16_f32(64, 128, 0, 0);
  static constexpr uint32_t kIdescS64 = sm100::idesc_bf16_f32(64, 64, 0, 0);
  static constexpr uint32_t kIdescO = sm100::idesc_bf16_f32(64, D, 0, 1);
  static constexpr uint32_t kIdescL = sm100::idesc_bf16_f32(64, kLCols, 0, 1);
  static_assert(kLCol + kLCols <= kTmemCols, "tensor memory");
  static_assert(kStages <= kMaxStages, "stage ring");
};

struct TcParams {
  const __nv_bfloat16* q;
  const __nv_bfloat16* kt;
  const __nv_bfloat16* vt;
  const int32_t* kv_len;
  const int32_t* parents;
  const int32_t* offs;
  int B, H, Hkv, group, max_kv, splits;
  int qtiles;         // 64-row query tiles per tree: ceil(max_nodes / 64)
  int cluster_merge;
  float scale_log2;
  __nv_bfloat16* out;
  float* lse;
  float* part_o;      // [B][H][splits][64][D]   (workspace merge only)
  float2* part_ml;    // [B][H][splits][64]
  unsigned* tickets;  // [B][H]
  unsigned* err;
  uint32_t wait_limit;  // polls before a pipeline wait gives up (kWaitLimit unless a test lowers it)
};

// Byte offset of 16-byte chunk `ch` (0 .. D/8-1) of row `row` in a tile of
// 128-byte column blocks of `block_rows` rows with the 128-byte swizzle (the
// layout TMA writes).
__device__ __forceinline__ uint32_t sw128_off(int row, int ch, int block_rows) {
  return static_cast<uint32_t>((ch >> 3) * block_rows * 128 + row * 128 + (((ch & 7) ^ (row & 7)) << 4));
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, int src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
__device__ __forceinline__ void cp_async4(uint32_t dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;\n" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;\n" ::: "memory"); }

// Named barrier over the four softmax warps.
__device__ __forceinline__ void softmax_warps_sync() { asm volatile("bar.sync 1, 128;\n" ::: "memory"); }

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// 2^x with the hardware approximation (flush-to-zero); 2^-inf = 0.
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;\n" : "=f"(y) : "f"(x));
  return y;
}

// Four 8x8 bf16 tiles to shared memory; thread l supplies the address of row
// l % 8 of tile l / 8 and holds, in register i, row lane / 4, columns
// 2 (lane % 4) .. +1 of tile i.
__device__ __forceinline__ void stmatrix_x4(uint32_t addr, uint32_t r0, uint32_t r1, uint32_t r2, uint32_t r3) {
  asm volatile("stmatrix.sync.aligned.m8n8.x4.shared.b16 [%0], {%1, %2, %3, %4};\n" ::"r"(addr), "r"(r0), "r"(r1),
               "r"(r2), "r"(r3)
               : "memory");
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

// The same shape, one 8-column block: r[0, 1] row 16w + g, r[2, 3] row 16w + g + 8.
__device__ __forceinline__ void tmem_ld_16x256b_x1(uint32_t taddr, uint32_t (&r)[4]) {
  asm volatile("tcgen05.ld.sync.aligned.16x256b.x1.b32 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(taddr)
               : "memory");
}
__device__ __forceinline__ void tmem_st_16x256b_x1(uint32_t taddr, const uint32_t (&r)[4]) {
  asm volatile("tcgen05.st.sync.aligned.16x256b.x1.b32 [%0], {%1,%2,%3,%4};\n" ::"r"(taddr), "r"(r[0]), "r"(r[1]),
               "r"(r[2]), "r"(r[3])
               : "memory");
}

// x masked to -inf where the keep bit is 0, without branching (a NaN score
// at a masked position also becomes -inf).
__device__ __forceinline__ float mask_or_neg_inf(float x, uint32_t keep_bit) {
  const uint32_t keep = 0u - keep_bit;
  return __uint_as_float((__float_as_uint(x) & keep) | (0xFF800000u & ~keep));
}

// Softmax of one chunk for the two rows (a, b) a thread holds: NB 8-column
// blocks (8 for 64 keys, 16 for 128), scores in sa / sb (raw Q.K), keep
// masks (bit c = column c) applied only when `masked`.  Updates the lazily
// raised maxima mu (log2 units), returns the rescale factors of O (and of
// the row sums, which the tensor core accumulates from the same bf16
// probabilities) and the probabilities packed in column pairs.
template <int NB>
__device__ __forceinline__ void chunk_softmax(float (&sa)[32], float (&sb)[32], bool masked, uint64_t ka0,
                                              uint64_t ka1, uint64_t kb0, uint64_t kb1, int t4, float scale,
                                              float& mu_a, float& mu_b, float& alpha_a,
                                              float& alpha_b, uint32_t (&pa)[16], uint32_t (&pb)[16]) {
  if (masked) {
    const int sh = 2 * t4;
    const uint64_t a0 = ka0 >> sh, a1 = ka1 >> sh, b0 = kb0 >> sh, b1 = kb1 >> sh;
#pragma unroll
    for (int bk = 0; bk < NB; ++bk) {
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int c = 8 * (bk & 7) + e;
        const uint64_t ma = bk < 8 ? a0 : a1, mb = bk < 8 ? b0 : b1;
        sa[2 * bk + e] = mask_or_neg_inf(sa[2 * bk + e], static_cast<uint32_t>(ma >> c) & 1u);
        sb[2 * bk + e] = mask_or_neg_inf(sb[2 * bk + e], static_cast<uint32_t>(mb >> c) & 1u);
      }
    }
  }
  float mxa = sa[0], mxb = sb[0];
#pragma unroll
  for (int i = 1; i < 2 * NB; ++i) {
    mxa = fmaxf(mxa, sa[i]);
    mxb = fmaxf(mxb, sb[i]);
  }
  mxa = fmaxf(mxa, __shfl_xor_sync(adt::kFullMask, mxa, 1));
  mxa = fmaxf(mxa, __shfl_xor_sync(adt::kFullMask, mxa, 2));
  mxb = fmaxf(mxb, __shfl_xor_sync(adt::kFullMask, mxb, 1));
  mxb = fmaxf(mxb, __shfl_xor_sync(adt::kFullMask, mxb, 2));
  mxa *= scale;  // scale > 0: the maximum of the scaled scores
  mxb *= scale;
  const bool needa = mxa > mu_a + kRescaleThreshold, needb = mxb > mu_b + kRescaleThreshold;
  const float nma = needa ? mxa : mu_a, nmb = needb ? mxb : mu_b;
  alpha_a = needa ? ex2_approx(mu_a - nma) : 1.f;
  alpha_b = needb ? ex2_approx(mu_b - nmb) : 1.f;
  const float base_a = nma == -INFINITY ? 0.f : nma, base_b = nmb == -INFINITY ? 0.f : nmb;
#pragma unroll
  for (int bk = 0; bk < NB; ++bk) {
    pa[bk] = pack_bf16x2(ex2_approx(fmaf(sa[2 * bk], scale, -base_a)), ex2_approx(fmaf(sa[2 * bk + 1], scale, -base_a)));
    pb[bk] = pack_bf16x2(ex2_approx(fmaf(sb[2 * bk], scale, -base_b)), ex2_approx(fmaf(sb[2 * bk + 1], scale, -base_b)));
  }
  mu_a = nma;
  mu_b = nmb;
}

struct Barriers {
  uint64_t q_full;                 // Q and the tree unit's K/V are in shared memory (softmax warps' copies)
  uint64_t q_tma;                  // the same, when they come as tensor copies: those copies landed
  uint64_t k_full[kMaxStages];     // a stage's K tile has landed
  uint64_t v_full[kMaxStages];     // a stage's V tile has landed
  uint64_t k_free[kMaxStages];     // the S product of the chunk in that slot finished
  uint64_t done[kMaxStages];       // the PV product of the chunk in that slot finished
  uint64_t s_full[2];
  uint64_t s_free[2];
  uint64_t p_full[2];
  uint64_t drain[2];               // abort path: every MMA a thread issued finished
  uint64_t recv;                   // cluster merge: every split's rows for this owner landed
};

// Bounded wait of the pipeline that also gives up when another role has
// aborted.  (The waits that let in-flight copies and products land before a
// CTA leaves always keep the full kWaitLimit.)
__device__ __forceinline__ bool wait_bar(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                         unsigned* err, uint32_t limit) {
  const uint32_t a = sm100::smem_addr(bar);
  for (uint32_t i = 0; i < limit; ++i) {
    if (sm100::mbar_try_wait(a, parity)) return true;
    if ((i & 255u) == 255u && *abort_flag) return false;
  }
  *abort_flag = 1;
  adt::raise_error(err, ADT_DEVERR_TIMEOUT);
  return false;
}

// kLarge: trees of more than 64 nodes (query tiles, one mask word per tree
// unit); otherwise one tile and one word, kept in registers.

template <int D, bool kLarge>
__global__ void __launch_bounds__(kThreads, 1)
    tree_attn_tc_kernel(const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_v,
                        const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_kt,
                        const __grid_constant__ CUtensorMap tm_vt, const TcParams p) {
  using C = Cfg<D>;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  // 1024-byte aligned for the 128-byte swizzle; pointer arithmetic on the
  // shared array keeps accesses in the shared address space.
  uint8_t* smem = smem_raw + ((1024u - (sm100::smem_addr(smem_raw) & 1023u)) & 1023u);
  __shared__ Barriers bars;
  constexpr int kUnits = kLarge ? kMaxTreeUnits : 1;
  __shared__ uint64_t anc[kMaxNodes][kUnits];
  __shared__ int s_par[kLarge ? kMaxTreeNodes : kMaxNodes];
  __shared__ uint32_t tmem_slot;
  __shared__ int s_bad;
  __shared__ int s_last;
  __shared__ volatile int s_abort;

  const int split = blockIdx.x, h = blockIdx.y;
  const int slot = kLarge ? static_cast<int>(blockIdx.z) / p.qtiles : static_cast<int>(blockIdx.z);
  const int qt = kLarge ? static_cast<int>(blockIdx.z) % p.qtiles : 0;
  const int g = h / p.group;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int NS = C::kStages;

  // Set-up that touches no memory the previous kernel writes: the
  // mbarriers, the tensor memory and the tensor maps' descriptors.  It runs
  // before the dependency wait, so a CTA that is resident early (on an SM
  // the previous launch leaves idle) has it done when the wait releases.
  if (tid == 0) {
    s_bad = 0;
    s_abort = 0;
    sm100::mbar_init(sm100::smem_addr(&bars.q_full), kSoftmaxWarps);
    sm100::mbar_init(sm100::smem_addr(&bars.q_tma), 1);
    for (int s = 0; s < NS; ++s) {
      sm100::mbar_init(sm100::smem_addr(&bars.k_full[s]), 1);
      sm100::mbar_init(sm100::smem_addr(&bars.v_full[s]), 1);
      sm100::mbar_init(sm100::smem_addr(&bars.k_free[s]), 1);
      sm100::mbar_init(sm100::smem_addr(&bars.done[s]), 1);
    }
    for (int s = 0; s < 2; ++s) {
      sm100::mbar_init(sm100::smem_addr(&bars.s_full[s]), 1);
      sm100::mbar_init(sm100::smem_addr(&bars.s_free[s]), kSoftmaxWarps);
      sm100::mbar_init(sm100::smem_addr(&bars.p_full[s]), kSoftmaxWarps);
    }
    sm100::mbar_init(sm100::smem_addr(&bars.drain[0]), 1);
    sm100::mbar_init(sm100::smem_addr(&bars.drain[1]), 1);
    sm100::mbar_init(sm100::smem_addr(&bars.recv), 1);
    sm100::fence_mbar_init();
  }
  if (warp == 0) {
    sm100::tmem_alloc(sm100::smem_addr(&tmem_slot), kTmemCols);
    sm100::tmem_relinquish();
  }
  if (warp == kKLoadWarp && lane < 4)
    sm100::prefetch_tensormap(lane == 0 ? &tm_k : lane == 1 ? &tm_q : lane == 2 ? &tm_kt : &tm_vt);
  if (warp == kVLoadWarp && lane == 0) sm100::prefetch_tensormap(&tm_v);
  sm100::tc_fence_before();
  __syncthreads();
  sm100::tc_fence_after();
  const uint32_t tmem = tmem_slot;

  // Programmatic dependent launch: every global-memory access comes after
  // the previous kernel in the stream has completed (immediate when this
  // launch does not overlap one).
  asm volatile("griddepcontrol.wait;\n" ::: "memory");
  // The tree of this CTA.  With several trees (up to 32) the launch slots
  // go to the trees by decreasing prefix length (ties: lower index): the
  // CTAs are dispatched in slot order, so the longest streams start first
  // and the short ones fill in behind them instead of a late long tree
  // ending the launch.  Every warp ranks the trees itself (one lane per
  // tree), from the same single round of loads the one-tree path makes.
  int b, node0, n, total_nodes, L;
  if (p.B > 1 && p.B <= 32) {
    const bool mine = lane < p.B;
    const int kl = mine ? p.kv_len[lane] : 0;
    const int off = mine ? p.offs[lane] : 0;
    total_nodes = p.offs[p.B];
    int rank = 0;
    for (int i = 0; i < p.B; ++i) {
      const int o = __shfl_sync(adt::kFullMask, kl, i);
      rank += (o > kl || (o == kl && i < lane)) ? 1 : 0;
    }
    const unsigned hit = __ballot_sync(adt::kFullMask, mine && rank == slot);
    b = hit ? __ffs(hit) - 1 : slot;
    L = __shfl_sync(adt::kFullMask, kl, b);
    node0 = __shfl_sync(adt::kFullMask, off, b);
    const int next = __shfl_sync(adt::kFullMask, off, (b + 1) & 31);
    n = (b + 1 < p.B ? next : total_nodes) - node0;
  } else {
    b = slot;
    node0 = p.offs[b];
    n = p.offs[b + 1] - node0;
    total_nodes = p.offs[p.B];
    L = p.kv_len[b];
  }

  // Conditions that hold for every CTA of this (tree, head, tile): all
  // leave here, handing back the tensor memory.  A tile past the end of its
  // tree has no rows.
  const int row0 = qt * kMaxNodes;  // first node (query row) of this tile
  const bool bad_tree = n < 1 || n > kMaxNodes * (kLarge ? p.qtiles : 1) || node0 < 0 || node0 + n > total_nodes;
  const bool bad_kv = L < 0 || L > p.max_kv;
  if (bad_tree || bad_kv || n - row0 <= 0) {
    if (split == 0 && h == 0 && qt == 0 && tid == 0 && (bad_tree || bad_kv))
      adt::raise_error(p.err, bad_tree ? ADT_DEVERR_BAD_TREE : ADT_DEVERR_KV_RANGE);
    if (warp == 0) sm100::tmem_dealloc(tmem, kTmemCols);
    return;
  }
  const int nq = min(n - row0, kMaxNodes);

  // The keys are cut into chunks of two 64-key units: ceil(P / 2) prefix
  // chunks (P = ceil(L / 64); the last holds one unit when P is odd), then
  // the tree units the tile's rows can see, 0 .. qt (a node's ancestors come
  // before it), two to a chunk.  Split s takes chunks [s T / S, (s + 1) T / S)
  // of the T and processes its tree chunks first.
  const int P = (L + kUnit - 1) / kUnit;
  const int Pc = (P + 1) / 2;
  const int Tc = kLarge ? (qt + 2) / 2 : 1;  // tree chunks of this tile
  const int T = Pc + Tc;
  const int S = p.splits;
  // (32-bit: T < 2^24 chunks and S <= 96 splits; 64-bit division is slow)
  const int c_begin = split * T / S;
  const int c_end = (split + 1) * T / S;
  const int nch = c_end - c_begin;
  const int tc0 = max(c_begin, Pc) - Pc;         // first tree chunk of this split
  const int n_tc = max(0, c_end - max(c_begin, Pc));  // its tree chunks, in slots 0 .. n_tc-1
  auto chunk_keys = [&](int j) -> int {
    if (j < n_tc) return (kLarge && 2 * (tc0 + j) + 1 <= qt ? 2 : 1) * kUnit;
    const int pc = c_begin + j - n_tc;
    return (2 * pc + 1 < P ? 2 : 1) * kUnit;
  };
  auto chunk_key0 = [&](int j) -> int { return (c_begin + j - n_tc) * kChunk; };

  // Q (and the one tree unit's K/V) as 64-row tensor copies when the whole
  // box lies inside the node_offsets[B] rows the caller's buffers hold;
  // otherwise (the last tree of a batch with fewer than 64 nodes after its
  // first, or trees of more than 64 nodes) the softmax warps copy the rows
  // of the tree alone, 16 bytes at a time.
  const bool q_tma = !kLarge && node0 + kMaxNodes <= total_nodes && total_nodes < kTmaRows;
  uint8_t* sQ = smem + C::kQOff;
  uint8_t* sP = smem + C::kPOff;
  uint8_t* sStage = smem + C::kStageOff;
  float* slots = reinterpret_cast<float*>(smem + C::kSlotOff);  // merge: [S][rows_per][kRowStride]

  if (warp < kSoftmaxWarps) {
    // Q tile: rows row0 .. row0+63 of the tree (rows past it zero-filled);
    // this split's tree chunks (K/V of kv head g, nodes past the tree
    // zero-filled) into stage slots 0 .. n_tc-1; the parent pointers.
    for (int i = tid; !q_tma && i < kUnit * (D / 8); i += kSoftmaxWarps * 32) {
      const int r = i / (D / 8), ch = i % (D / 8);
      const bool valid = r < nq;
      const int row = node0 + row0 + (valid ? r : 0);
      cp_async16(sm100::smem_addr(sQ) + sw128_off(r, ch, kUnit),
                 p.q + (static_cast<int64_t>(row) * p.H + h) * D + ch * 8, valid ? 16 : 0);
      if (!kLarge && n_tc) {  // the one tree unit: the same rows
        const int64_t off = (static_cast<int64_t>(row) * p.Hkv + g) * D + ch * 8;
        cp_async16(sm100::smem_addr(sStage) + sw128_off(r, ch, kChunk), p.kt + off, valid ? 16 : 0);
        cp_async16(sm100::smem_addr(sStage + C::kStageTile) + sw128_off(r, ch, kChunk), p.vt + off, valid ? 16 : 0);
      }
    }
    for (int jt = 0; kLarge && jt < n_tc; ++jt) {
      uint8_t* st = sStage + jt * C::kStageBytes;
      for (int i = tid; i < chunk_keys(jt) * (D / 8); i += kSoftmaxWarps * 32) {
        const int r = i / (D / 8), ch = i % (D / 8);
        const int t = (tc0 + jt) * kChunk + r;  // tree node
        const bool valid = t < n;
        const int64_t off = (static_cast<int64_t>(node0 + (valid ? t : 0)) * p.Hkv + g) * D + ch * 8;
        cp_async16(sm100::smem_addr(st) + sw128_off(r, ch, kChunk), p.kt + off, valid ? 16 : 0);
        cp_async16(sm100::smem_addr(st + C::kStageTile) + sw128_off(r, ch, kChunk), p.vt + off, valid ? 16 : 0);
      }
    }
    for (int t = tid; t < n; t += kSoftmaxWarps * 32) cp_async4(sm100::smem_addr(&s_par[t]), p.parents + node0 + t);
    // The ones tile (bf16 1.0) of the row-sum product.
    static_assert(C::kOnesBytes == kSoftmaxWarps * 32 * 16, "one 16-byte store per softmax thread");
    reinterpret_cast<uint4*>(smem + C::kOnesOff)[tid] = make_uint4(0x3F803F80u, 0x3F803F80u, 0x3F803F80u, 0x3F803F80u);
  }
  // Stage loads: chunk j goes to slot j % NS, K tile by warp 4 and V tile by
  // warp 6.  A tree chunk loads nothing (its K/V came with Q) but still
  // completes its slot's phases, so that every slot's phases advance once
  // per chunk.
  const bool is_loader = (warp == kKLoadWarp || warp == kVLoadWarp) && lane == 0;
  const bool load_v = warp == kVLoadWarp;
  auto issue_tile = [&](int j) {
    const int st = j % NS;
    const uint32_t bar = sm100::smem_addr(load_v ? &bars.v_full[st] : &bars.k_full[st]);
    if (j < n_tc) {
      sm100::mbar_arrive(bar);
      return;
    }
    // One 128-key box per column block (a chunk of one unit loads the next
    // 64 rows too; nothing reads them: its products stop at 64 keys).
    const int key0 = chunk_key0(j);
    uint8_t* dst = sStage + st * C::kStageBytes + (load_v ? C::kStageTile : 0);
    const CUtensorMap* map = load_v ? &tm_v : &tm_k;
    sm100::mbar_arrive_expect_tx(bar, C::kBlocks * C::kBlock128);
    for (int blk = 0; blk < C::kBlocks; ++blk)
      sm100::tma_load_4d(sm100::smem_addr(dst + blk * C::kBlock128), map, blk * 64, key0, g, b, bar);
  };
  const int first_issue = nch < NS ? nch : NS;
  if (q_tma) {
    // Q and the tree unit go out first, from the thread that then requests
    // the first K stages; nothing waits for the softmax warps' set-up.
    if (warp == kKLoadWarp && lane == 0) {
      const uint32_t bar = sm100::smem_addr(&bars.q_tma);
      sm100::mbar_arrive_expect_tx(bar, C::kBlocks * C::kBlock64 * (n_tc ? 3 : 1));
      for (int blk = 0; blk < C::kBlocks; ++blk)
        sm100::tma_load_3d(sm100::smem_addr(sQ + blk * C::kBlock64), &tm_q, blk * 64, h, node0, bar);
      for (int blk = 0; n_tc && blk < C::kBlocks; ++blk) {
        sm100::tma_load_3d(sm100::smem_addr(sStage + blk * C::kBlock128), &tm_kt, blk * 64, g, node0, bar);
        sm100::tma_load_3d(sm100::smem_addr(sStage + C::kStageTile + blk * C::kBlock128), &tm_vt, blk * 64, g, node0,
                           bar);
      }
    }
    if (is_loader) {
      for (int j = 0; j < first_issue; ++j) issue_tile(j);
    }
  }
  // Q's copies (when the softmax warps make them) are requested before the
  // stage loads: a CTA's first stages are 128 KB, and Q queued behind them
  // would hold back the first S.
  __syncthreads();
  // The mbarriers are initialised: tell the cluster (the merge's bulk copies
  // complete on a peer's barrier; every thread waits on this before one).
  sm100::cluster_arrive_relaxed();
  if (!q_tma && is_loader) {
    for (int j = 0; j < first_issue; ++j) issue_tile(j);
  }
  if (warp < kSoftmaxWarps) {
    cp_async_wait_all();
    softmax_warps_sync();
    // Ancestor bitmask of every row r of the tile (node t = row0 + r), one
    // 64-bit word per tree unit: bit j of anc[r][u] <=> node 64u + j is in
    // ans(t) or is t.  Parents precede their children, so the walk visits
    // decreasing indices; anything else marks the tree malformed.
    if (!kLarge && tid < kMaxNodes) {
      uint64_t m = 0;
      if (tid < nq) {
        int j = tid;
        int par = s_par[j];
        m = 1ull << j;
        bool bad = (j == 0) != (par < 0);
        while (!bad && par >= 0) {
          if (par >= j) {
            bad = true;
            break;
          }
          m |= 1ull << par;
          j = par;
          par = s_par[j];
          bad = (j == 0) != (par < 0);
        }
        if (bad) s_bad = 1;
      }
      anc[tid][0] = m;
    }
    if (kLarge && tid < kMaxNodes) {
      uint64_t m0 = 0, m1 = 0, m2 = 0, m3 = 0;
      auto set_bit = [&](int j) {
        const uint64_t bit = 1ull << (j & 63);
        const int u = j >> 6;
        m0 |= u == 0 ? bit : 0ull;
        m1 |= u == 1 ? bit : 0ull;
        m2 |= u == 2 ? bit : 0ull;
        m3 |= u == 3 ? bit : 0ull;
      };
      if (tid < nq) {
        int j = row0 + tid;
        int par = s_par[j];
        set_bit(j);
        bool bad = (j == 0) != (par < 0);
        while (!bad && par >= 0) {
          if (par >= j) {
            bad = true;
            break;
          }
          set_bit(par);
          j = par;
          par = s_par[j];
          bad = (j == 0) != (par < 0);
        }
        if (bad) s_bad = 1;
      }
      uint64_t* w = anc[tid];
      w[0] = m0;
      if constexpr (kUnits > 1) {
        w[1] = m1;
        w[2] = m2;
        w[3] = m3;
      }
    }
  }
  __syncthreads();
  if (s_bad) {
    // Same tree for every CTA of the cluster: all leave here, after the
    // loads already issued have landed.
    if (split == 0 && h == 0 && tid == 0) adt::raise_error(p.err, ADT_DEVERR_BAD_TREE);
    if (is_loader) {
      for (int j = 0; j < first_issue; ++j)
        (void)sm100::mbar_wait_bounded(sm100::smem_addr(load_v ? &bars.v_full[j % NS] : &bars.k_full[j % NS]), 0,
                                       kWaitLimit);
      if (q_tma && !load_v) (void)sm100::mbar_wait_bounded(sm100::smem_addr(&bars.q_tma), 0, kWaitLimit);
    }
    sm100::tc_fence_before();
    __syncthreads();
    if (warp == 0) sm100::tmem_dealloc(tmem, kTmemCols);
    return;
  }

  // Final row statistics of the softmax threads' two rows (a, b).
  float m_ra = -INFINITY, l_ra = 0.f, m_rb = -INFINITY, l_rb = 0.f;

  if (warp == kKLoadWarp || warp == kVLoadWarp) {
    // ------------------------------------------------------------ K / V loads
    if (lane == 0) {
      int issued = first_issue;
      for (int j = first_issue; j < nch; ++j) {
        const int st = j % NS;
        // slot st was last used by chunk j - NS: its K is free once its S is
        // done, its V once its PV is done
        if (!wait_bar(load_v ? &bars.done[st] : &bars.k_free[st], ((j / NS) - 1) & 1, &s_abort, p.err, p.wait_limit)) break;
        issue_tile(j);
        ++issued;
      }
      // Every copy issued lands before the CTA goes on: after an abort
      // elsewhere its consumer may never have waited for it (on the normal
      // path these waits return at once).
      for (int j = (issued > NS ? issued - NS : 0); j < issued; ++j)
        (void)sm100::mbar_wait_bounded(sm100::smem_addr(load_v ? &bars.v_full[j % NS] : &bars.k_full[j % NS]),
                                       (j / NS) & 1, kWaitLimit);
      if (q_tma && !load_v) (void)sm100::mbar_wait_bounded(sm100::smem_addr(&bars.q_tma), 0, kWaitLimit);
    }
    __syncwarp();
  } else if (warp == kSMmaWarp) {
    // ------------------------------------------------------------ S = Q K^T
    if (lane == 0) {
      bool ok = wait_bar(&bars.q_full, 0, &s_abort, p.err, p.wait_limit) &&
                (!q_tma || wait_bar(&bars.q_tma, 0, &s_abort, p.err, p.wait_limit));
      const uint32_t q_addr = sm100::smem_addr(sQ);
      for (int j = 0; ok && j < nch; ++j) {
        const int st = j % NS, sb = j & 1;
        if (!wait_bar(&bars.k_full[st], (j / NS) & 1, &s_abort, p.err, p.wait_limit) ||
            (j >= 2 && !wait_bar(&bars.s_free[sb], ((j >> 1) - 1) & 1, &s_abort, p.err, p.wait_limit)))
          break;
        sm100::tc_fence_after();
        const uint32_t k_addr = sm100::smem_addr(sStage + st * C::kStageBytes);
        const uint32_t idesc = chunk_keys(j) == kChunk ? C::kIdescS128 : C::kIdescS64;
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint64_t da = sm100::smem_desc_sw128(q_addr + (kk >> 2) * C::kBlock64 + (kk & 3) * 32, 16, 1024);
          const uint64_t db = sm100::smem_desc_sw128(k_addr + (kk >> 2) * C::kBlock128 + (kk & 3) * 32, 16, 1024);
          sm100::mma_bf16_ss(tmem + sb * kSCols, da, db, idesc, kk > 0 ? 1u : 0u);
        }
        sm100::mma_commit(sm100::smem_addr(&bars.s_full[sb]));
      }
      // The tensor core finishes whatever was issued before this thread goes
      // on, also when a consumer aborted after the last product was issued.
      sm100::mma_commit(sm100::smem_addr(&bars.drain[0]));
      (void)sm100::mbar_wait_bounded(sm100::smem_addr(&bars.drain[0]), 0, kWaitLimit);
    }
    __syncwarp();
  } else if (warp == kPvMmaWarp) {
    // ------------------------------------------------------------ O += P V
    if (lane == 0) {
      const uint32_t p_addr = sm100::smem_addr(sP);
      // Any 16 K-rows of the ones tile are the same: one descriptor serves
      // every k step.
      const uint64_t ones_desc = sm100::smem_desc_sw128(sm100::smem_addr(smem + C::kOnesOff), C::kBlock128, 1024);
      for (int i = 0; i < nch; ++i) {
        if (!wait_bar(&bars.p_full[i & 1], (i >> 1) & 1, &s_abort, p.err, p.wait_limit) ||
            !wait_bar(&bars.v_full[i % NS], (i / NS) & 1, &s_abort, p.err, p.wait_limit))
          break;
        sm100::tc_fence_after();
        const uint32_t v_addr = sm100::smem_addr(sStage + (i % NS) * C::kStageBytes + C::kStageTile);
        const uint32_t pb = p_addr + (i & 1) * C::kPBytes;
        const int ksteps = chunk_keys(i) / 16;
        for (int kk = 0; kk < ksteps; ++kk) {
          const uint64_t da = sm100::smem_desc_sw128(pb + (kk >> 2) * C::kBlock64 + (kk & 3) * 32, 16, 1024);
          const uint64_t db = sm100::smem_desc_sw128(v_addr + kk * 2048, C::kBlock128, 1024);  // LBO: d blocks
          sm100::mma_bf16_ss(tmem + kOCol, da, db, C::kIdescO, (i > 0 || kk > 0) ? 1u : 0u);
          // row sums of the same bf16 P: P times a 16-column tile of ones
          sm100::mma_bf16_ss(tmem + C::kLCol, da, ones_desc, C::kIdescL, (i > 0 || kk > 0) ? 1u : 0u);
        }
        sm100::mma_commit(sm100::smem_addr(&bars.done[i % NS]));
      }
      sm100::mma_commit(sm100::smem_addr(&bars.drain[1]));
      (void)sm100::mbar_wait_bounded(sm100::smem_addr(&bars.drain[1]), 0, kWaitLimit);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ softmax warps 0-3
    if (q_tma && n_tc && n < kUnit) {
      // The tree unit came as a 64-row box: V rows past the tree (another
      // tree's nodes) are zeroed, so that P = 0 there meets finite values.
      if (__all_sync(adt::kFullMask, wait_bar(&bars.q_tma, 0, &s_abort, p.err, p.wait_limit))) {
        uint8_t* vt = sStage + C::kStageTile;
        const int per_row = C::kBlocks * 8;
        for (int i = tid; i < (kUnit - n) * per_row; i += kSoftmaxWarps * 32) {
          const int rr = n + i / per_row, rem = i % per_row;
          *reinterpret_cast<uint4*>(vt + (rem >> 3) * C::kBlock128 + rr * 128 + (rem & 7) * 16) =
              make_uint4(0u, 0u, 0u, 0u);
        }
      }
    }
    sm100::fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) sm100::mbar_arrive(sm100::smem_addr(&bars.q_full));

    // Thread (g, t) = (lane / 4, lane % 4) of warp w owns rows ra = 16w + g
    // and rb = ra + 8 of the tile, columns 8b + 2t, 8b + 2t + 1 of every
    // 8-column block b (the 16x256b tensor-memory layout); the four threads
    // of a quad share a row and combine row statistics with two shuffles.
    const int g8 = lane >> 2, t4 = lane & 3;
    const int ra = warp * 16 + g8, rb = ra + 8;
    const uint32_t lane_base = static_cast<uint32_t>(warp * 32) << 16;
    // stmatrix addressing: lane l writes row (l / 8 odd ? 8 : 0) + l % 8 of
    // the warp's rows, in column block (l / 16) of each pair of blocks.
    const int st_row = warp * 16 + ((lane >> 3) & 1) * 8 + (lane & 7);
    const int st_blk = lane >> 4;
    const float scale = p.scale_log2;
    const uint64_t ama = anc[ra][0], amb = anc[rb][0];  // the one tree unit (kLarge: unused)
    float mua = -INFINITY, mub = -INFINITY;  // running maxima used for the exponentials
    for (int j = 0; j < nch; ++j) {
      const int sb = j & 1;
      if (!__all_sync(adt::kFullMask, wait_bar(&bars.s_full[sb], (j >> 1) & 1, &s_abort, p.err, p.wait_limit))) break;
      // S(j) is complete, so its K tile can be refilled (the S issuer goes
      // straight on to the next S product).
      if (warp == 0 && lane == 0) sm100::mbar_arrive(sm100::smem_addr(&bars.k_free[j % NS]));
      sm100::tc_fence_after();
      const int keys = chunk_keys(j);
      uint32_t r0[32], r1[32];
      tmem_ld_16x256b_x8(tmem + lane_base + sb * kSCols, r0);
      if (keys == kChunk) tmem_ld_16x256b_x8(tmem + lane_base + sb * kSCols + 64, r1);
      sm100::tmem_wait_ld();
      // S is in registers: hand the tensor-memory tile back to the MMA warp.
      sm100::tc_fence_before();
      __syncwarp();
      if (lane == 0) sm100::mbar_arrive(sm100::smem_addr(&bars.s_free[sb]));

      // Which keys a row sees: its ancestors and itself in the tree unit,
      // the prefix up to L otherwise.  Only the tree chunk and a chunk that
      // holds the end of the prefix need a mask.
      const bool tree_j = j < n_tc;
      const int kl = tree_j ? keys : L - chunk_key0(j);
      const bool masked = tree_j || kl < keys;
      uint64_t ka0 = ~0ull, ka1 = ~0ull, kb0 = ~0ull, kb1 = ~0ull;
      if (tree_j) {
        if constexpr (kLarge) {
          // units 2u and 2u + 1 of the tree (rows past the tile have no bits)
          const int u = 2 * (tc0 + j);
          ka0 = anc[ra][u];
          kb0 = anc[rb][u];
          ka1 = u + 1 < kUnits ? anc[ra][u + 1] : 0ull;
          kb1 = u + 1 < kUnits ? anc[rb][u + 1] : 0ull;
        } else {
          ka0 = ama;
          kb0 = amb;
        }
      } else if (kl < keys) {
        ka0 = kb0 = kl >= 64 ? ~0ull : ((1ull << kl) - 1ull);
        ka1 = kb1 = kl >= 128 ? ~0ull : (kl > 64 ? ((1ull << (kl - 64)) - 1ull) : 0ull);
      }
      float sa[32], sbv[32];
#pragma unroll
      for (int bk = 0; bk < 8; ++bk) {
        sa[2 * bk] = __uint_as_float(r0[4 * bk]);
        sa[2 * bk + 1] = __uint_as_float(r0[4 * bk + 1]);
        sbv[2 * bk] = __uint_as_float(r0[4 * bk + 2]);
        sbv[2 * bk + 1] = __uint_as_float(r0[4 * bk + 3]);
        sa[16 + 2 * bk] = __uint_as_float(r1[4 * bk]);
        sa[16 + 2 * bk + 1] = __uint_as_float(r1[4 * bk + 1]);
        sbv[16 + 2 * bk] = __uint_as_float(r1[4 * bk + 2]);
        sbv[16 + 2 * bk + 1] = __uint_as_float(r1[4 * bk + 3]);
      }
      uint32_t pa[16], pb[16];
      float alpha_a, alpha_b;
      if (keys == kChunk)
        chunk_softmax<16>(sa, sbv, masked, ka0, ka1, kb0, kb1, t4, scale, mua, mub, alpha_a, alpha_b, pa, pb);
      else
        chunk_softmax<8>(sa, sbv, masked, ka0, ka1, kb0, kb1, t4, scale, mua, mub, alpha_a, alpha_b, pa, pb);

      // P buffer sb was last read by the PV product of chunk j - 2.
      if (j >= 2 && !__all_sync(adt::kFullMask,
                                wait_bar(&bars.done[(j - 2) % NS], ((j - 2) / NS) & 1, &s_abort, p.err, p.wait_limit)))
        break;
      {
        const uint32_t pbase = sm100::smem_addr(sP) + sb * C::kPBytes + st_row * 128;
        const int nb = keys / 8;
#pragma unroll
        for (int bb = 0; bb < 16; bb += 2) {
          if (bb < nb) {
            const int blk = bb + st_blk;
            const uint32_t addr = pbase + (blk >> 3) * C::kBlock64 + (((blk & 7) ^ (st_row & 7)) << 4);
            stmatrix_x4(addr, pa[bb], pb[bb], pa[bb + 1], pb[bb + 1]);
          }
        }
      }
      // Cache rows at or past L in this chunk (the end of the prefix) can
      // hold anything, NaN included, and P is 0 there: zero their V rows.
      if (!tree_j && kl < keys) {
        if (!__all_sync(adt::kFullMask, wait_bar(&bars.v_full[j % NS], (j / NS) & 1, &s_abort, p.err, p.wait_limit))) break;
        uint8_t* vt = sStage + (j % NS) * C::kStageBytes + C::kStageTile;
        const int per_row = C::kBlocks * 8;
        for (int i = tid; i < (keys - kl) * per_row; i += kSoftmaxWarps * 32) {
          const int rr = kl + i / per_row, rem = i % per_row;
          *reinterpret_cast<uint4*>(vt + (rem >> 3) * C::kBlock128 + rr * 128 + (rem & 7) * 16) =
              make_uint4(0u, 0u, 0u, 0u);
        }
      }
      sm100::fence_proxy_async_smem();
      // Raise O to the new maxima (rare): needs the previous PV product done.
      if (j > 0 && __any_sync(adt::kFullMask, alpha_a != 1.f || alpha_b != 1.f)) {
        if (!__all_sync(adt::kFullMask,
                        wait_bar(&bars.done[(j - 1) % NS], ((j - 1) / NS) & 1, &s_abort, p.err, p.wait_limit)))
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
        {
          uint32_t l4[4];
          tmem_ld_16x256b_x1(tmem + lane_base + C::kLCol, l4);
          sm100::tmem_wait_ld();
          l4[0] = __float_as_uint(__uint_as_float(l4[0]) * alpha_a);
          l4[1] = __float_as_uint(__uint_as_float(l4[1]) * alpha_a);
          l4[2] = __float_as_uint(__uint_as_float(l4[2]) * alpha_b);
          l4[3] = __float_as_uint(__uint_as_float(l4[3]) * alpha_b);
          tmem_st_16x256b_x1(tmem + lane_base + C::kLCol, l4);
        }
        sm100::tmem_wait_st();
      }
      sm100::tc_fence_before();
      __syncwarp();
      if (lane == 0) sm100::mbar_arrive(sm100::smem_addr(&bars.p_full[sb]));
    }
    m_ra = mua;
    m_rb = mub;
  }

  // ------------------------------------------------------------ epilogue
  // The next kernel in the stream may start its set-up now.
  asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
  // The softmax threads take their rows of O (unnormalised) into registers.
  constexpr int kOB = D / 64;
  uint32_t o[kOB][32];
  bool have_o = false;
  if (warp < kSoftmaxWarps) {
    const int last = nch - 1;
    // s_abort can change under the warp: decide once, by a vote.
    if (__all_sync(adt::kFullMask, nch > 0 && !s_abort))
      have_o = __all_sync(adt::kFullMask, wait_bar(&bars.done[last % NS], (last / NS) & 1, &s_abort, p.err, p.wait_limit));
    if (have_o) {
      sm100::tc_fence_after();
      const uint32_t lane_base = static_cast<uint32_t>(warp * 32) << 16;
#pragma unroll
      for (int c = 0; c < kOB; ++c) tmem_ld_16x256b_x8(tmem + lane_base + kOCol + c * 64, o[c]);
      uint32_t l4[4];
      tmem_ld_16x256b_x1(tmem + lane_base + C::kLCol, l4);  // every column holds the row sum
      sm100::tmem_wait_ld();
      l_ra = __uint_as_float(l4[0]);
      l_rb = __uint_as_float(l4[2]);
    } else {
      // A split without key units (kv_len shorter than max_kv) contributes
      // nothing: weight 0.
      m_ra = m_rb = -INFINITY;
      l_ra = l_rb = 0.f;
    }
  }
  sm100::tc_fence_before();

  const int g8 = lane >> 2, t4 = lane & 3;
  const int ra = warp * 16 + g8, rb = ra + 8;
  const int64_t bh = static_cast<int64_t>(blockIdx.z) * p.H + h;  // (tree, tile, head)
  constexpr int kC4 = D / 4;
  if (p.cluster_merge) {
    // Row r of the (tree, head, tile) is merged by split r / rows_per, its owner.
    // Each split writes its partial rows (O unnormalised, then m and l) into
    // its own stage ring, idle now, in row order; one thread sends every
    // owner its rows with bulk shared-to-shared copies into the owner's slot
    // region, completing on the owner's mbarrier; each owner merges locally.
    constexpr int RS = C::kRowStride;
    const int rows_per = (nq + S - 1) / S;
    const int r_lo = split * rows_per;
    const int rows_mine = max(0, min(nq, r_lo + rows_per) - r_lo);
    float* rows_out = reinterpret_cast<float*>(sStage);
    if (tid == 0)
      sm100::mbar_arrive_expect_tx(sm100::smem_addr(&bars.recv), static_cast<uint32_t>(S * rows_mine * RS * 4));
    if (warp < kSoftmaxWarps) {
      if constexpr (C::kHalfRows) {
        // The row normalised by its sum, O / l, goes out in fp16: half the
        // bytes through distributed shared memory.  It is a convex
        // combination of V rows, scaled by 2^-e (e from the row's largest
        // magnitude, over the quad) into [2^14, 2^15): no overflow, and full
        // fp16 precision relative to that magnitude whatever V's range; the
        // owner undoes the scale.
#pragma unroll
        for (int half = 0; half < 2; ++half) {
          const int r = half ? rb : ra;
          const float l = half ? l_rb : l_ra;
          const float inv = have_o && l > 0.f ? __fdividef(1.f, l) : 0.f;
          float amax = 0.f;
#pragma unroll
          for (int c = 0; c < kOB; ++c)
#pragma unroll
            for (int bk = 0; bk < 8; ++bk)
              if (have_o)
                amax = fmaxf(amax, fmaxf(fabsf(__uint_as_float(o[c][4 * bk + 2 * half])),
                                         fabsf(__uint_as_float(o[c][4 * bk + 2 * half + 1]))));
          amax = fmaxf(amax, __shfl_xor_sync(adt::kFullMask, amax, 1));
          amax = fmaxf(amax, __shfl_xor_sync(adt::kFullMask, amax, 2));
          amax *= inv;
          const int ex = static_cast<int>((__float_as_uint(amax) >> 23) & 0xFFu);  // biased exponent
          const int e = amax > 0.f ? min(max(ex - 127 - 14, -110), 110) : 0;
          const float sc = inv * __uint_as_float(static_cast<uint32_t>(127 - e) << 23);  // inv * 2^-e
          if (r < nq) {
            float* dst = rows_out + r * RS;
            if (t4 == 0) {
              *reinterpret_cast<float2*>(dst + D / 2) =
                  make_float2(have_o ? (half ? m_rb : m_ra) : -INFINITY, have_o ? l : 0.f);
              reinterpret_cast<int*>(dst)[D / 2 + 2] = e;
            }
#pragma unroll
            for (int c = 0; c < kOB; ++c) {
#pragma unroll
              for (int bk = 0; bk < 8; ++bk)
                reinterpret_cast<__half2*>(dst)[(c * 64 + 8 * bk + 2 * t4) / 2] =
                    have_o ? __floats2half2_rn(__uint_as_float(o[c][4 * bk + 2 * half]) * sc,
                                               __uint_as_float(o[c][4 * bk + 2 * half + 1]) * sc)
                           : __floats2half2_rn(0.f, 0.f);
            }
          }
        }
      } else {
#pragma unroll
        for (int half = 0; half < 2; ++half) {
          const int r = half ? rb : ra;
          if (r < nq) {
            float* dst = rows_out + r * RS;
            if (t4 == 0) *reinterpret_cast<float2*>(dst + D) = half ? make_float2(m_rb, l_rb) : make_float2(m_ra, l_ra);
#pragma unroll
            for (int c = 0; c < kOB; ++c) {
#pragma unroll
              for (int bk = 0; bk < 8; ++bk)
                *reinterpret_cast<float2*>(dst + c * 64 + 8 * bk + 2 * t4) =
                    have_o ? make_float2(__uint_as_float(o[c][4 * bk + 2 * half]),
                                         __uint_as_float(o[c][4 * bk + 2 * half + 1]))
                           : make_float2(0.f, 0.f);
            }
          }
        }
      }
      sm100::fence_proxy_async_smem();
      softmax_warps_sync();
    }
    // Pairs with the arrive after the prologue: every peer's receive barrier
    // is initialised.
    sm100::cluster_wait_acquire();
    if (tid == 0) {
      for (int c = 0; c < S; ++c) {
        const int rc = max(0, min(nq, (c + 1) * rows_per) - c * rows_per);
        if (rc > 0)
          sm100::bulk_copy_to_cluster(sm100::mapa_shared(sm100::smem_addr(slots + split * rows_per * RS), c),
                                      sm100::smem_addr(rows_out + c * rows_per * RS),
                                      static_cast<uint32_t>(rc * RS * 4),
                                      sm100::mapa_shared(sm100::smem_addr(&bars.recv), c));
      }
    }
    // Not abandoned on an abort elsewhere: copies into this CTA's shared
    // memory must have landed before it exits.
    if (!sm100::mbar_wait_bounded(sm100::smem_addr(&bars.recv), 0, kWaitLimit) && tid == 0)
      adt::raise_error(p.err, ADT_DEVERR_TIMEOUT);
    // This owner has its rows, so the copies it was sent are complete.
    sm100::cluster_arrive_relaxed();
    if constexpr (C::kHalfRows) {
      // Thread (row i, 8-column group c8) combines the S normalised partials
      // of that row: weights 2^(m_c - M) l_c / sum (times 2^e_c, the scale the
      // partial was stored at).  A split without keys sent m = -inf (weight 0).
      constexpr int kC8 = D / 8;
      for (int idx = tid; idx < rows_mine * kC8; idx += kThreads) {
        const int i = idx / kC8, c8 = idx % kC8;
        float2 ml[kMaxClusterSplits];
        int ec[kMaxClusterSplits];
        uint4 v[kMaxClusterSplits];
  #pragma unroll
        for (int c = 0; c < kMaxClusterSplits; ++c) {
          if (c < S) {
            const float* row = slots + (c * rows_per + i) * RS;
            ml[c] = *reinterpret_cast<const float2*>(row + D / 2);
            ec[c] = reinterpret_cast<const int*>(row)[D / 2 + 2];
            v[c] = *reinterpret_cast<const uint4*>(row + c8 * 4);
          }
        }
        float M = -INFINITY;
  #pragma unroll
        for (int c = 0; c < kMaxClusterSplits; ++c)
          if (c < S) M = fmaxf(M, ml[c].x);
        float lt = 0.f;
        float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  #pragma unroll
        for (int c = 0; c < kMaxClusterSplits; ++c) {
          if (c < S) {
            const float w = ml[c].x == -INFINITY ? 0.f : ex2_approx(ml[c].x - M) * ml[c].y;
            lt += w;
            const float ws = w * __uint_as_float(static_cast<uint32_t>(127 + ec[c]) << 23);  // w * 2^e_c
            const __half2* hv = reinterpret_cast<const __half2*>(&v[c]);
  #pragma unroll
            for (int e = 0; e < 4; ++e) {
              const float2 f = __half22float2(hv[e]);
              acc[2 * e] += ws * f.x;
              acc[2 * e + 1] += ws * f.y;
            }
          }
        }
        const float inv = __fdividef(1.f, lt);
        __nv_bfloat16* dst = p.out + (static_cast<int64_t>(node0 + row0 + r_lo + i) * p.H + h) * D + c8 * 8;
        uint4 pk;
        pk.x = pack_bf16x2(acc[0] * inv, acc[1] * inv);
        pk.y = pack_bf16x2(acc[2] * inv, acc[3] * inv);
        pk.z = pack_bf16x2(acc[4] * inv, acc[5] * inv);
        pk.w = pack_bf16x2(acc[6] * inv, acc[7] * inv);
        *reinterpret_cast<uint4*>(dst) = pk;
        if (c8 == 0 && p.lse) p.lse[static_cast<int64_t>(node0 + row0 + r_lo + i) * p.H + h] = (M + __log2f(lt)) * kLn2;
      }
    } else {
      // Thread (row i, column group c4) combines the S partials of that row:
      // weights 2^(m_c - M) l_c / sum.  A thread takes two items per pass and
      // loads every split's values of both before combining either.
      // A split without keys sent zeros with m = -inf (weight 0).
      auto merge_item = [&](int idx, float2 (&ml)[kMaxClusterSplits], float4 (&v)[kMaxClusterSplits]) {
        const int i = idx / kC4, c4 = idx % kC4;
        float M = ml[0].x;
  #pragma unroll
        for (int c = 1; c < kMaxClusterSplits; ++c) M = fmaxf(M, ml[c].x);
        float lt = 0.f;
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  #pragma unroll
        for (int c = 0; c < kMaxClusterSplits; ++c) {
          const float w = ml[c].x == -INFINITY ? 0.f : ex2_approx(ml[c].x - M);
          lt += w * ml[c].y;
          acc.x += w * v[c].x;
          acc.y += w * v[c].y;
          acc.z += w * v[c].z;
          acc.w += w * v[c].w;
        }
        const float inv = __fdividef(1.f, lt);
        __nv_bfloat16* dst = p.out + (static_cast<int64_t>(node0 + row0 + r_lo + i) * p.H + h) * D + c4 * 4;
        uint2 pk;
        pk.x = pack_bf16x2(acc.x * inv, acc.y * inv);
        pk.y = pack_bf16x2(acc.z * inv, acc.w * inv);
        *reinterpret_cast<uint2*>(dst) = pk;
        if (c4 == 0 && p.lse) p.lse[static_cast<int64_t>(node0 + row0 + r_lo + i) * p.H + h] = (M + __log2f(lt)) * kLn2;
      };
      auto load_item = [&](int idx, float2 (&ml)[kMaxClusterSplits], float4 (&v)[kMaxClusterSplits]) {
        const int i = idx / kC4, c4 = idx % kC4;
  #pragma unroll
        for (int c = 0; c < kMaxClusterSplits; ++c) {
          if (c < S) {
            const float* row = slots + (c * rows_per + i) * RS;
            ml[c] = *reinterpret_cast<const float2*>(row + D);
            v[c] = *reinterpret_cast<const float4*>(row + c4 * 4);
          } else {
            ml[c] = make_float2(-INFINITY, 0.f);
            v[c] = make_float4(0.f, 0.f, 0.f, 0.f);
          }
        }
      };
      for (int idx = tid; idx < rows_mine * kC4; idx += 2 * kThreads) {
        float2 ml0[kMaxClusterSplits], ml1[kMaxClusterSplits];
        float4 v0[kMaxClusterSplits], v1[kMaxClusterSplits];
        const bool two = idx + kThreads < rows_mine * kC4;
        load_item(idx, ml0, v0);
        if (two) load_item(idx + kThreads, ml1, v1);
        merge_item(idx, ml0, v0);
        if (two) merge_item(idx + kThreads, ml1, v1);
      }
    }
    // Every owner has its rows: this CTA's outgoing copies are complete.
    sm100::cluster_wait_acquire();
    sm100::tc_fence_after();
    if (warp == 0) sm100::tmem_dealloc(tmem, kTmemCols);
    return;
  }

  // More splits than a portable cluster holds: partials go to the workspace
  // and the CTA that finishes a (tree, head) last merges them.
  float* po = p.part_o + (bh * S + split) * kMaxNodes * D;
  float2* pml = p.part_ml + (bh * S + split) * kMaxNodes;
  if (warp < kSoftmaxWarps) {
#pragma unroll
    for (int half = 0; half < 2; ++half) {
      const int r = half ? rb : ra;
      if (r < nq) {
        if (t4 == 0) pml[r] = half ? make_float2(m_rb, l_rb) : make_float2(m_ra, l_ra);
#pragma unroll
        for (int c = 0; c < kOB; ++c) {
#pragma unroll
          for (int bk = 0; bk < 8; ++bk) {
            const float2 v = have_o ? make_float2(__uint_as_float(o[c][4 * bk + 2 * half]),
                                                  __uint_as_float(o[c][4 * bk + 2 * half + 1]))
                                    : make_float2(0.f, 0.f);
            *reinterpret_cast<float2*>(po + r * D + c * 64 + 8 * bk + 2 * t4) = v;
          }
        }
      }
    }
  }
  sm100::cluster_wait_acquire();  // pairs with the prologue's arrive (a cluster of one CTA here)
  __syncthreads();
  sm100::tc_fence_after();
  if (warp == 0) sm100::tmem_dealloc(tmem, kTmemCols);
  // The ticket's release publishes this split's partials (ordered before it
  // by the barrier); its acquire, in the last split, makes all of them visible.
  if (tid == 0) s_last = adt::atomic_add_acq_rel_gpu(p.tickets + bh, 1u) == static_cast<unsigned>(S - 1);
  __syncthreads();
  if (!s_last) return;
  const float* po_bh = p.part_o + bh * S * kMaxNodes * D;
  const float2* pml_bh = p.part_ml + bh * S * kMaxNodes;
  float* wsm = reinterpret_cast<float*>(sStage);  // [64][S]
  if (tid < nq) {
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
    if (p.lse) p.lse[static_cast<int64_t>(node0 + row0 + tid) * p.H + h] = (M + log2f(lt)) * kLn2;
  }
  __syncthreads();
  constexpr int kStride4 = kMaxNodes * D / 4;
  for (int idx = tid; idx < nq * kC4; idx += kThreads) {
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
    __nv_bfloat16* dst = p.out + (static_cast<int64_t>(node0 + row0 + rr) * p.H + h) * D + c4 * 4;
    uint2 pk;
    pk.x = pack_bf16x2(acc.x, acc.y);
    pk.y = pack_bf16x2(acc.z, acc.w);
    *reinterpret_cast<uint2*>(dst) = pk;
  }
  if (tid == 0) p.tickets[bh] = 0u;
}

// ---------------------------------------------------------------- host side

// Splits per (tree, head): about one CTA per SM, at most one split per chunk
// of keys.  Up to kMaxClusterSplits splits form a cluster; the count is
// lowered until all B*H clusters are co-resident (GPC sizes decide how many
// clusters of a given size fit at once).  Many splits (small B*H, long
// prefixes) merge through the workspace instead.
int max_active_clusters(int D, bool large, int cluster, int dev);

int qtiles_for(int max_nodes) { return (max_nodes + kMaxNodes - 1) / kMaxNodes; }

// Bq = trees x query tiles.
int choose_splits(int sm_count, int Bq, int H, int D, int max_kv, int dev, bool large) {
  const int units = ((max_kv + kUnit - 1) / kUnit + 1) / 2 + 1;  // chunks, the tree unit included
  const int bh = Bq * H;
  int s = sm_count / bh;
  if (s < 1) s = 1;
  if (s > units) s = units;
  if (s >= 2 * kMaxClusterSplits) return s > kMaxSplits ? kMaxSplits : s;
  if (s > kMaxClusterSplits) s = kMaxClusterSplits;
  while (s > 1 && max_active_clusters(D, large, s, dev) < bh) --s;
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
// boxes of 64 columns x 128 positions; positions at or past max_kv read as
// zero.
adt_status make_cache_map(CUtensorMap* map, const void* base, int D, int max_kv, int Hkv, int B, int64_t sh,
                          int64_t sb) {
  std::call_once(g_encode_once, load_encode);
  if (!g_encode) return ADT_ERR_CUDA;
  const int64_t span = static_cast<int64_t>(max_kv > 0 ? max_kv : 1);
  cuuint64_t dims[4] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(span), static_cast<cuuint64_t>(Hkv),
                        static_cast<cuuint64_t>(B)};
  cuuint64_t strides[3] = {static_cast<cuuint64_t>(D) * 2, static_cast<cuuint64_t>(sh > 0 ? sh : span * D) * 2,
                           static_cast<cuuint64_t>(sb > 0 ? sb : span * D * Hkv) * 2};
  cuuint32_t box[4] = {64, kChunk, 1, 1};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? ADT_OK : ADT_ERR_INVALID_ARG;
}

// 3-D map of a node-major tensor [nodes][heads][D] (Q or the tree's K / V)
// with the 128-byte swizzle and boxes of 64 nodes x 64 columns of one head.
// The node extent is nominal: the kernel only requests boxes that lie inside
// the node_offsets[B] rows the caller's buffer holds.
adt_status make_rows_map(CUtensorMap* map, const void* base, int D, int heads) {
  std::call_once(g_encode_once, load_encode);
  if (!g_encode) return ADT_ERR_CUDA;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(heads), static_cast<cuuint64_t>(kTmaRows)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(D) * 2, static_cast<cuuint64_t>(heads) * D * 2};
  cuuint32_t box[3] = {64, 1, kUnit};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? ADT_OK : ADT_ERR_INVALID_ARG;
}

template <int D, bool kLarge>
int occupancy_clusters(cudaLaunchConfig_t* cfg) {
  int num = 0;
  cudaFuncSetAttribute(tree_attn_tc_kernel<D, kLarge>, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg<D>::kDynSmem);
  cfg->dynamicSmemBytes = Cfg<D>::kDynSmem;
  if (cudaOccupancyMaxActiveClusters(&num, tree_attn_tc_kernel<D, kLarge>, cfg) != cudaSuccess) {
    (void)cudaGetLastError();
    num = 0;
  }
  return num;
}

int max_active_clusters(int D, bool large, int cluster, int dev) {
  static int cache[64][2][2][kMaxClusterSplits + 1];  // 0 = not queried yet
  int& slot = cache[dev & 63][D == 128 ? 1 : 0][large ? 1 : 0][cluster];
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
  const int num = D == 128 ? (large ? occupancy_clusters<128, true>(&cfg) : occupancy_clusters<128, false>(&cfg))
                           : (large ? occupancy_clusters<64, true>(&cfg) : occupancy_clusters<64, false>(&cfg));
  __atomic_store_n(&slot, num + 1, __ATOMIC_RELEASE);
  return num;
}

template <int D, bool kLarge>
adt_status launch(TcParams prm, const void* k_cache, const void* v_cache, int64_t sb, int64_t sh, cudaStream_t st,
                  int dev, bool overlap_previous) {
  static unsigned configured[2] = {0u, 0u};  // bit per device (< 64), per instantiation
  const unsigned bit = 1u << (dev & 31);
  unsigned& word = configured[dev >> 5];
  if (!(__atomic_load_n(&word, __ATOMIC_ACQUIRE) & bit)) {
    ADT_CUDA_TRY(cudaFuncSetAttribute(tree_attn_tc_kernel<D, kLarge>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      Cfg<D>::kDynSmem));
    __atomic_fetch_or(&word, bit, __ATOMIC_ACQ_REL);
  }
  CUtensorMap tm_k, tm_v, tm_q, tm_kt, tm_vt;
  adt_status s1 = make_cache_map(&tm_k, k_cache, D, prm.max_kv, prm.Hkv, prm.B, sh, sb);
  if (s1 != ADT_OK) return s1;
  s1 = make_cache_map(&tm_v, v_cache, D, prm.max_kv, prm.Hkv, prm.B, sh, sb);
  if (s1 != ADT_OK) return s1;
  if ((s1 = make_rows_map(&tm_q, prm.q, D, prm.H)) != ADT_OK) return s1;
  if ((s1 = make_rows_map(&tm_kt, prm.kt, D, prm.Hkv)) != ADT_OK) return s1;
  if ((s1 = make_rows_map(&tm_vt, prm.vt, D, prm.Hkv)) != ADT_OK) return s1;
  prm.cluster_merge = prm.splits <= kMaxClusterSplits ? 1 : 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(prm.splits), static_cast<unsigned>(prm.H),
                     static_cast<unsigned>(prm.B * prm.qtiles));
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = Cfg<D>::kDynSmem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = prm.cluster_merge ? static_cast<unsigned>(prm.splits) : 1u;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  // Programmatic dependent launch: the launch and the set-up before the
  // kernel's griddepcontrol.wait may overlap the tail of the previous kernel.
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = overlap_previous ? 2 : 1;
  ADT_CUDA_TRY(cudaLaunchKernelEx(&cfg, tree_attn_tc_kernel<D, kLarge>, tm_k, tm_v, tm_q, tm_kt, tm_vt, prm));
  return adt::launch_status();
}

// Trees of more than 64 nodes take the query-tiled instantiation.
adt_status launch_any(const TcParams& prm, int D, const void* k_cache, const void* v_cache, int64_t sb, int64_t sh,
                      cudaStream_t st, int dev, bool overlap_previous) {
  const bool large = prm.qtiles > 1;
  if (D == 128)
    return large ? launch<128, true>(prm, k_cache, v_cache, sb, sh, st, dev, overlap_previous)
                 : launch<128, false>(prm, k_cache, v_cache, sb, sh, st, dev, overlap_previous);
  return large ? launch<64, true>(prm, k_cache, v_cache, sb, sh, st, dev, overlap_previous)
               : launch<64, false>(prm, k_cache, v_cache, sb, sh, st, dev, overlap_previous);
}

// Shared host checks of both entry points.
adt_status check_args(const adt_bf16* q, const adt_bf16* k_cache, const adt_bf16* v_cache, const int32_t* kv_len,
                      int64_t sb, int64_t sh, const adt_bf16* k_tree, const adt_bf16* v_tree,
                      const int32_t* parents, const int32_t* node_offsets, int32_t B, int32_t H, int32_t Hkv,
                      int32_t D, int32_t max_nodes, int32_t max_kv, float scale, const adt_bf16* out) {
  ADT_REQUIRE(q && k_cache && v_cache && kv_len && k_tree && v_tree && parents && node_offsets && out);
  ADT_REQUIRE(B >= 1 && H >= 1 && Hkv >= 1 && H % Hkv == 0);
  ADT_REQUIRE(max_nodes >= 1 && max_kv >= 0 && max_kv < (1 << 30));
  if (max_nodes > kMaxTreeNodes) return ADT_ERR_UNSUPPORTED;
  const int64_t bq = static_cast<int64_t>(B) * qtiles_for(max_nodes);
  ADT_REQUIRE(bq * H <= kMaxBH && bq <= 65535 && H <= 65535);
  ADT_REQUIRE(scale > 0.f && scale < 1e30f);
  if (D != 64 && D != 128) return ADT_ERR_UNSUPPORTED;
  ADT_REQUIRE(sb >= 0 && sh >= 0 && sb % 8 == 0 && sh % 8 == 0);
  ADT_REQUIRE(Hkv == 1 || sh >= static_cast<int64_t>(max_kv) * D);
  ADT_REQUIRE(B == 1 || sb >= static_cast<int64_t>(max_kv) * D);
  ADT_REQUIRE(adt::aligned16(q) && adt::aligned16(k_cache) && adt::aligned16(v_cache) && adt::aligned16(k_tree) &&
              adt::aligned16(v_tree) && adt::aligned16(out));
  return ADT_OK;
}

// Polls before a pipeline wait gives up; 0 = kWaitLimit.  Set only by
// adt_testing_set_wait_limit.
uint32_t g_wait_limit = 0;

TcParams make_params(const adt_bf16* q, const int32_t* kv_len, const adt_bf16* k_tree, const adt_bf16* v_tree,
                     const int32_t* parents, const int32_t* node_offsets, int B, int H, int Hkv, int max_kv,
                     int max_nodes, int splits, float scale, adt_bf16* out, float* lse, unsigned* err) {
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
  prm.qtiles = qtiles_for(max_nodes);
  prm.scale_log2 = scale * kLog2e;
  prm.out = reinterpret_cast<__nv_bfloat16*>(out);
  prm.lse = lse;
  prm.err = err;
  const uint32_t lim = __atomic_load_n(&g_wait_limit, __ATOMIC_RELAXED);
  prm.wait_limit = lim ? lim : kWaitLimit;
  return prm;
}

}  // namespace

extern "C" {

adt_status adt_testing_set_wait_limit(uint32_t polls) {
  __atomic_store_n(&g_wait_limit, polls, __ATOMIC_RELAXED);
  return ADT_OK;
}

size_t adt_tree_attn_workspace_size(int32_t B, int32_t H, int32_t D, int32_t max_nodes,
                                    int32_t max_kv) {
  if (B < 1 || H < 1 || (D != 64 && D != 128) || max_kv < 0 || max_nodes < 1 || max_nodes > kMaxTreeNodes) return 0;
  const int Bq = B * qtiles_for(max_nodes);
  if (static_cast<int64_t>(Bq) * H > kMaxBH) return 0;
  adt::DeviceInfo info;
  if (adt::device_info(&info) != ADT_OK) return 0;
  return ws_layout(Bq, H, D, choose_splits(info.sm_count, Bq, H, D, max_kv, info.device, max_nodes > kMaxNodes)).total;
}

adt_status adt_tree_attn(const adt_bf16* q, const adt_bf16* k_cache, const adt_bf16* v_cache,
                         const int32_t* kv_len, int64_t cache_stride_b, int64_t cache_stride_h,
                         const adt_bf16* k_tree, const adt_bf16* v_tree, const int32_t* parents,
                         const int32_t* node_offsets, int32_t B, int32_t H, int32_t Hkv, int32_t D,
                         int32_t max_nodes, int32_t max_kv, float softmax_scale, adt_bf16* out,
                         float* lse, void* workspace, size_t workspace_bytes, void* stream) {
  adt::TraceRange trace_("adt_tree_attn");
  adt_status st = check_args(q, k_cache, v_cache, kv_len, cache_stride_b, cache_stride_h, k_tree, v_tree, parents,
                             node_offsets, B, H, Hkv, D, max_nodes, max_kv, softmax_scale, out);
  if (st != ADT_OK) return st;
  adt::DeviceInfo info;
  st = adt::device_info(&info);
  if (st != ADT_OK) return st;
  const int Bq = B * qtiles_for(max_nodes);
  const int splits = choose_splits(info.sm_count, Bq, H, D, max_kv, info.device, max_nodes > kMaxNodes);
  const WsLayout w = ws_layout(Bq, H, D, splits);
  if (!workspace || workspace_bytes < w.total || !adt::aligned16(workspace)) return ADT_ERR_WORKSPACE;
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  TcParams prm = make_params(q, kv_len, k_tree, v_tree, parents, node_offsets, B, H, Hkv, max_kv, max_nodes, splits,
                             softmax_scale, out, lse, info.error_word);
  prm.part_o = reinterpret_cast<float*>(ws + w.part_o);
  prm.part_ml = reinterpret_cast<float2*>(ws + w.part_ml);
  prm.tickets = reinterpret_cast<unsigned*>(ws + w.tickets);
  cudaStream_t s = adt::as_stream(stream);
  return launch_any(prm, D, k_cache, v_cache, cache_stride_b, cache_stride_h, s, info.device, true);
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

// 4 MiB of scratch, held by every GPU that loads the library until the
// process exits.  Shared by all calls on a device: calls that overlap on the
// GPU (different streams, or different host threads) race on it.
static constexpr size_t kNoAllocScratchBytes = size_t(4) << 20;
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

// What a launch with `splits` key splits uses: nothing when the splits merge
// inside their cluster (splits <= kMaxClusterSplits, the kernel returns
// before it touches tickets or partials); otherwise Bq*H tickets, then
// Bq*H*splits partial rows (m, l) and partial outputs of 64 rows x D.
struct NoAllocLayout {
  size_t tickets, part_ml, part_o, total;
};

NoAllocLayout noalloc_layout(int Bq, int H, int D, int splits) {
  NoAllocLayout w{};
  if (splits <= kMaxClusterSplits) return w;
  const size_t bh = static_cast<size_t>(Bq) * H;
  const size_t bhs = bh * splits;
  w.tickets = 0;
  w.part_ml = adt::align_up(bh * sizeof(unsigned), 256);
  w.part_o = adt::align_up(w.part_ml + bhs * kMaxNodes * sizeof(float2), 256);
  w.total = adt::align_up(w.part_o + bhs * kMaxNodes * D * sizeof(float), 256);
  return w;
}

// The split count of a no-allocation launch: the usual heuristic's, lowered
// while a workspace merge's partials would not fit the scratch; once it is
// down to a cluster's size the splits merge in their cluster and need no
// scratch, and the count is lowered further until all clusters are
// co-resident, as the heuristic does for its own cluster-sized counts.
int noalloc_splits(int sm_count, int Bq, int H, int D, int max_kv, int dev, bool large) {
  int s = choose_splits(sm_count, Bq, H, D, max_kv, dev, large);
  while (s > kMaxClusterSplits && noalloc_layout(Bq, H, D, s).total > kNoAllocScratchBytes) --s;
  if (s <= kMaxClusterSplits) {
    const int bh = Bq * H;
    while (s > 1 && max_active_clusters(D, large, s, dev) < bh) --s;
  }
  return s;
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
  adt::TraceRange trace_("adt_tree_attn_noalloc");
  adt_status st = check_args(q, k_cache, v_cache, kv_len, cache_stride_b, cache_stride_h, k_tree, v_tree, parents,
                             node_offsets, B, H, Hkv, D, max_nodes, max_kv, softmax_scale, out);
  if (st != ADT_OK) return st;
  adt::DeviceInfo info;
  st = adt::device_info(&info);
  if (st != ADT_OK) return st;
  if (info.device < 0 || info.device >= kNoAllocMaxDevices) return ADT_ERR_UNSUPPORTED;
  std::call_once(g_noalloc_once[info.device], noalloc_setup, info.device);
  if (g_noalloc_status[info.device] != cudaSuccess || !g_noalloc_ptr[info.device]) return ADT_ERR_CUDA;
  const int Bq = B * qtiles_for(max_nodes);
  const int splits = noalloc_splits(info.sm_count, Bq, H, D, max_kv, info.device, max_nodes > kMaxNodes);
  const NoAllocLayout w = noalloc_layout(Bq, H, D, splits);
  // Unreachable for the shapes check_args accepts (a workspace merge is
  // chosen only when its partials fit); kept as the guard of the array.
  if (w.total > kNoAllocScratchBytes) return ADT_ERR_WORKSPACE;
  uint8_t* ws = static_cast<uint8_t*>(g_noalloc_ptr[info.device]);
  cudaStream_t s = adt::as_stream(stream);
  // A workspace merge counts finished splits in tickets that start at zero.
  // A completed call leaves them at zero, but one that a bounded wait ended
  // (ADT_DEVERR_TIMEOUT) can leave them set, so they are cleared here, on
  // the caller's stream.  Cluster merges use no tickets.
  if (splits > kMaxClusterSplits)
    ADT_CUDA_TRY(cudaMemsetAsync(ws + w.tickets, 0, static_cast<size_t>(Bq) * H * sizeof(unsigned), s));
  TcParams prm = make_params(q, kv_len, k_tree, v_tree, parents, node_offsets, B, H, Hkv, max_kv, max_nodes, splits,
                             softmax_scale, out, lse, info.error_word);
  prm.part_o = reinterpret_cast<float*>(ws + w.part_o);
  prm.part_ml = reinterpret_cast<float2*>(ws + w.part_ml);
  prm.tickets = reinterpret_cast<unsigned*>(ws + w.tickets);
  return launch_any(prm, D, k_cache, v_cache, cache_stride_b, cache_stride_h, s, info.device, false);
}

