// adt_tree_attn: tree-masked attention of the draft-tree nodes over the
// prefix KV cache and their own ancestors (Sec. 3.1: every node is verified
// conditioned on s_{1:t} and ans(t) under the tree mask; the mask is the
// T_N term of Eq. 5).
//
// Split-KV flash decoding.  The keys a tree sees are cut into units of 64:
// ceil(L/64) prefix units plus one tree unit (the <= 64 tree nodes, masked
// per row by an ancestor bitmask built from the parent pointers).  Grid =
// (splits, H, B); a CTA streams its share of units for one (tree, head)
// through a 3-stage cp.async pipeline into XOR-swizzled shared memory and
// runs QK^T and PV on bf16 mma.sync tiles (m16n8k16, fp32 accumulation) with
// an online softmax in registers.  Each warp owns 16 query rows.  The CTA
// that finishes a (tree, head) last (atomic ticket) merges the split
// partials (m, l, unnormalised O) and writes bf16 O and the natural-log LSE.
#include "adt_common.cuh"

namespace {

constexpr int kKeys = 64;
constexpr int kStages = 3;
constexpr int kWarps = 4;
constexpr int kThreads = kWarps * 32;
constexpr int kMaxNodes = 64;
constexpr float kLn2 = 0.69314718055994530942f;
constexpr float kLog2e = 1.44269504088896340736f;

template <int D>
struct Cfg {
  static constexpr int kRowBytes = D * 2;
  static constexpr int kChunks = kRowBytes / 16;  // 16-byte chunks per key row
  static constexpr int kTileBytes = kKeys * kRowBytes;
  static constexpr int kStageBytes = 2 * kTileBytes;  // K tile + V tile
  static constexpr int kSmemBytes = kStages * kStageBytes + kMaxNodes * 8;
  static constexpr int kKSteps = D / 16;  // k-steps of QK^T
  static constexpr int kNTiles = D / 8;   // n-tiles of O
};

struct AttnParams {
  const __nv_bfloat16* q;
  const __nv_bfloat16* kc;
  const __nv_bfloat16* vc;
  const int32_t* kv_len;
  int64_t sb, sh;
  const __nv_bfloat16* kt;
  const __nv_bfloat16* vt;
  const int32_t* parents;
  const int32_t* offs;
  int B, H, Hkv, group, max_kv, splits;
  float scale_log2;
  __nv_bfloat16* out;
  float* lse;
  float* part_o;   // [B][H][splits][64][D]
  float2* part_ml; // [B][H][splits][64]
  unsigned* tickets;  // [B][H]
  unsigned* err;
};

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, int src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src), "r"(src_bytes));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;\n" ::"n"(N));
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_trans(uint32_t addr, uint32_t& r0, uint32_t& r1,
                                              uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                               uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// Byte offset of 16-byte chunk `ch` of key row `row` inside a swizzled tile.
template <int D>
__device__ __forceinline__ uint32_t tile_off(int row, int ch) {
  return static_cast<uint32_t>(row * Cfg<D>::kRowBytes + ((ch ^ (row & 7)) << 4));
}

template <int D>
__global__ void __launch_bounds__(kThreads) tree_attn_kernel(const AttnParams p) {
  using C = Cfg<D>;
  extern __shared__ __align__(128) uint8_t smem[];
  uint64_t* anc = reinterpret_cast<uint64_t*>(smem + kStages * C::kStageBytes);
  __shared__ int s_bad;
  __shared__ int s_last;

  const int split = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int g = h / p.group;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int grp = lane >> 2, tig = lane & 3;

  const int node0 = p.offs[b];
  const int n = p.offs[b + 1] - node0;
  const int L = p.kv_len[b];

  if (tid == 0) s_bad = 0;
  __syncthreads();
  if (n < 1 || n > kMaxNodes) {
    if (split == 0 && h == 0) adt::raise_error(p.err, ADT_DEVERR_BAD_TREE);
    return;  // uniform over the CTA and over every split of this (b, h)
  }
  if (L < 0 || L > p.max_kv) {
    if (split == 0 && h == 0) adt::raise_error(p.err, ADT_DEVERR_KV_RANGE);
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
    if (split == 0 && h == 0) adt::raise_error(p.err, ADT_DEVERR_BAD_TREE);
    return;
  }

  const int U = (L + kKeys - 1) / kKeys + 1;  // prefix units + the tree unit
  const int S = p.splits;
  const int u_begin = static_cast<int>(static_cast<int64_t>(split) * U / S);
  const int u_end = static_cast<int>(static_cast<int64_t>(split + 1) * U / S);
  const int nu = u_end - u_begin;

  const __nv_bfloat16* kc_bh = p.kc + b * p.sb + g * p.sh;
  const __nv_bfloat16* vc_bh = p.vc + b * p.sb + g * p.sh;

  auto load_unit = [&](int u, int stage) {
    const uint32_t ks = smem_u32(smem + stage * C::kStageBytes);
    const bool tree = (u == U - 1);
    for (int i = tid; i < kKeys * C::kChunks; i += kThreads) {
      const int row = i / C::kChunks, ch = i % C::kChunks;
      const __nv_bfloat16* ksrc;
      const __nv_bfloat16* vsrc;
      bool valid;
      if (!tree) {
        const int key = u * kKeys + row;
        valid = key < L;
        const int64_t off = static_cast<int64_t>(valid ? key : 0) * D + ch * 8;
        ksrc = kc_bh + off;
        vsrc = vc_bh + off;
      } else {
        valid = row < n;
        const int64_t off = (static_cast<int64_t>(node0 + (valid ? row : 0)) * p.Hkv + g) * D + ch * 8;
        ksrc = p.kt + off;
        vsrc = p.vt + off;
      }
      const uint32_t dst = ks + tile_off<D>(row, ch);
      cp_async16(dst, ksrc, valid ? 16 : 0);
      cp_async16(dst + C::kTileBytes, vsrc, valid ? 16 : 0);
    }
  };

  // Query fragments (A operand of QK^T) for rows r0 = 16*warp + grp and r0 + 8.
  const int r0 = warp * 16 + grp, r1 = r0 + 8;
  const bool warp_active = warp * 16 < n;
  uint32_t qa[C::kKSteps][4];
  {
    const __nv_bfloat16* q0 = p.q + (static_cast<int64_t>(node0 + r0) * p.H + h) * D;
    const __nv_bfloat16* q1 = p.q + (static_cast<int64_t>(node0 + r1) * p.H + h) * D;
#pragma unroll
    for (int kk = 0; kk < C::kKSteps; ++kk) {
      const int d0 = kk * 16 + tig * 2;
      qa[kk][0] = r0 < n ? *reinterpret_cast<const uint32_t*>(q0 + d0) : 0u;
      qa[kk][1] = r1 < n ? *reinterpret_cast<const uint32_t*>(q1 + d0) : 0u;
      qa[kk][2] = r0 < n ? *reinterpret_cast<const uint32_t*>(q0 + d0 + 8) : 0u;
      qa[kk][3] = r1 < n ? *reinterpret_cast<const uint32_t*>(q1 + d0 + 8) : 0u;
    }
  }

  float o[C::kNTiles][4];
#pragma unroll
  for (int t = 0; t < C::kNTiles; ++t) o[t][0] = o[t][1] = o[t][2] = o[t][3] = 0.f;
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
  const uint64_t anc0 = r0 < n ? anc[r0] : 0ull;
  const uint64_t anc1 = r1 < n ? anc[r1] : 0ull;

#pragma unroll
  for (int s = 0; s < kStages - 1; ++s) {
    if (s < nu) load_unit(u_begin + s, s);
    cp_async_commit();
  }

  for (int it = 0; it < nu; ++it) {
    cp_async_wait<kStages - 2>();
    __syncthreads();
    {
      const int nx = it + kStages - 1;
      if (nx < nu) load_unit(u_begin + nx, nx % kStages);
      cp_async_commit();
    }
    if (!warp_active) continue;
    const int u = u_begin + it;
    const uint32_t ks = smem_u32(smem + (it % kStages) * C::kStageBytes);
    const uint32_t vs = ks + C::kTileBytes;
    const bool tree = (u == U - 1);

    float s[8][4];
#pragma unroll
    for (int j = 0; j < 8; ++j) s[j][0] = s[j][1] = s[j][2] = s[j][3] = 0.f;
    const int mat = lane >> 3, mr = lane & 7;
#pragma unroll
    for (int kk = 0; kk < C::kKSteps; ++kk) {
#pragma unroll
      for (int j = 0; j < 8; j += 2) {
        const int row = (j + (mat >> 1)) * 8 + mr;
        const int ch = 2 * kk + (mat & 1);
        uint32_t b0, b1, b2, b3;
        ldsm_x4(ks + tile_off<D>(row, ch), b0, b1, b2, b3);
        mma_bf16_16816(s[j], qa[kk], b0, b1);
        mma_bf16_16816(s[j + 1], qa[kk], b2, b3);
      }
    }
    // Mask, scale to the log2 domain, online softmax.
    float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int key = j * 8 + tig * 2 + (e & 1);
        bool ok;
        if (tree) {
          ok = ((e < 2 ? anc0 : anc1) >> key) & 1ull;
        } else {
          ok = u * kKeys + key < L;
        }
        const float v = ok ? s[j][e] * p.scale_log2 : -INFINITY;
        s[j][e] = v;
        if (e < 2) mx0 = fmaxf(mx0, v); else mx1 = fmaxf(mx1, v);
      }
    }
    mx0 = fmaxf(mx0, __shfl_xor_sync(adt::kFullMask, mx0, 1));
    mx0 = fmaxf(mx0, __shfl_xor_sync(adt::kFullMask, mx0, 2));
    mx1 = fmaxf(mx1, __shfl_xor_sync(adt::kFullMask, mx1, 1));
    mx1 = fmaxf(mx1, __shfl_xor_sync(adt::kFullMask, mx1, 2));
    const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
    const float base0 = mn0 == -INFINITY ? 0.f : mn0;
    const float base1 = mn1 == -INFINITY ? 0.f : mn1;
    const float a0 = exp2f(m0 - base0), a1 = exp2f(m1 - base1);
    m0 = mn0;
    m1 = mn1;
    float rs0 = 0.f, rs1 = 0.f;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      s[j][0] = exp2f(s[j][0] - base0);
      s[j][1] = exp2f(s[j][1] - base0);
      s[j][2] = exp2f(s[j][2] - base1);
      s[j][3] = exp2f(s[j][3] - base1);
      rs0 += s[j][0] + s[j][1];
      rs1 += s[j][2] + s[j][3];
    }
    l0 = l0 * a0 + rs0;
    l1 = l1 * a1 + rs1;
#pragma unroll
    for (int t = 0; t < C::kNTiles; ++t) {
      o[t][0] *= a0;
      o[t][1] *= a0;
      o[t][2] *= a1;
      o[t][3] *= a1;
    }
    // O += P V
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      uint32_t pa[4];
      pa[0] = pack_bf16x2(s[2 * kk][0], s[2 * kk][1]);
      pa[1] = pack_bf16x2(s[2 * kk][2], s[2 * kk][3]);
      pa[2] = pack_bf16x2(s[2 * kk + 1][0], s[2 * kk + 1][1]);
      pa[3] = pack_bf16x2(s[2 * kk + 1][2], s[2 * kk + 1][3]);
#pragma unroll
      for (int t = 0; t < C::kNTiles; t += 2) {
        const int key = kk * 16 + (mat & 1) * 8 + mr;
        const int ch = t + (mat >> 1);
        uint32_t b0, b1, b2, b3;
        ldsm_x4_trans(vs + tile_off<D>(key, ch), b0, b1, b2, b3);
        mma_bf16_16816(o[t], pa, b0, b1);
        mma_bf16_16816(o[t + 1], pa, b2, b3);
      }
    }
  }
  cp_async_wait<0>();

  // Partial (m, l, O) of this split.
  l0 += __shfl_xor_sync(adt::kFullMask, l0, 1);
  l0 += __shfl_xor_sync(adt::kFullMask, l0, 2);
  l1 += __shfl_xor_sync(adt::kFullMask, l1, 1);
  l1 += __shfl_xor_sync(adt::kFullMask, l1, 2);
  const int64_t bh = static_cast<int64_t>(b) * p.H + h;
  float* po = p.part_o + (bh * S + split) * kMaxNodes * D;
  float2* pml = p.part_ml + (bh * S + split) * kMaxNodes;
  if (warp_active) {
#pragma unroll
    for (int t = 0; t < C::kNTiles; ++t) {
      const int d = t * 8 + tig * 2;
      if (r0 < n) *reinterpret_cast<float2*>(po + r0 * D + d) = make_float2(o[t][0], o[t][1]);
      if (r1 < n) *reinterpret_cast<float2*>(po + r1 * D + d) = make_float2(o[t][2], o[t][3]);
    }
    if (tig == 0) {
      if (r0 < n) pml[r0] = make_float2(m0, l0);
      if (r1 < n) pml[r1] = make_float2(m1, l1);
    }
  }
  __threadfence();
  __syncthreads();
  if (tid == 0) {
    const unsigned prev = atomicAdd(p.tickets + bh, 1u);
    s_last = (prev == static_cast<unsigned>(S - 1));
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();

  // Merge the splits of this (tree, head).
  const float* po_bh = p.part_o + bh * S * kMaxNodes * D;
  const float2* pml_bh = p.part_ml + bh * S * kMaxNodes;
  constexpr int kC4 = D / 4;
  for (int idx = tid; idx < n * kC4; idx += kThreads) {
    const int row = idx / kC4, c4 = idx % kC4;
    float M = -INFINITY;
    for (int sp = 0; sp < S; ++sp) M = fmaxf(M, __ldcg(&pml_bh[sp * kMaxNodes + row]).x);
    float lt = 0.f;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int sp = 0; sp < S; ++sp) {
      const float2 ml = __ldcg(&pml_bh[sp * kMaxNodes + row]);
      if (ml.x == -INFINITY) continue;
      const float w = exp2f(ml.x - M);
      lt += w * ml.y;
      const float4 v = __ldcg(reinterpret_cast<const float4*>(po_bh + (sp * kMaxNodes + row) * D) + c4);
      acc.x += w * v.x;
      acc.y += w * v.y;
      acc.z += w * v.z;
      acc.w += w * v.w;
    }
    const float inv = 1.f / lt;
    __nv_bfloat16* dst = p.out + (static_cast<int64_t>(node0 + row) * p.H + h) * D + c4 * 4;
    __nv_bfloat162 lo = __floats2bfloat162_rn(acc.x * inv, acc.y * inv);
    __nv_bfloat162 hi = __floats2bfloat162_rn(acc.z * inv, acc.w * inv);
    uint2 pk;
    pk.x = *reinterpret_cast<uint32_t*>(&lo);
    pk.y = *reinterpret_cast<uint32_t*>(&hi);
    *reinterpret_cast<uint2*>(dst) = pk;
    if (c4 == 0 && p.lse) p.lse[static_cast<int64_t>(node0 + row) * p.H + h] = (M + log2f(lt)) * kLn2;
  }
  if (tid == 0) p.tickets[bh] = 0u;
}

int choose_splits(int sm_count, int B, int H, int D, int max_kv) {
  const int units = (max_kv + kKeys - 1) / kKeys + 1;
  const int per_sm = D == 128 ? 2 : 4;
  const int target = sm_count * per_sm;
  int s = target / (B * H);
  if (s < 1) s = 1;
  if (s > units) s = units;
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

template <int D>
adt_status launch(const AttnParams& prm, cudaStream_t st, int dev) {
  static unsigned configured[2] = {0u, 0u};  // bit per device (< 64)
  const unsigned bit = 1u << (dev & 31);
  unsigned& word = configured[dev >> 5];
  if (!(__atomic_load_n(&word, __ATOMIC_ACQUIRE) & bit)) {
    ADT_CUDA_TRY(cudaFuncSetAttribute(tree_attn_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      Cfg<D>::kSmemBytes));
    __atomic_fetch_or(&word, bit, __ATOMIC_ACQ_REL);
  }
  dim3 grid(prm.splits, prm.H, prm.B);
  tree_attn_kernel<D><<<grid, kThreads, Cfg<D>::kSmemBytes, st>>>(prm);
  return adt::launch_status();
}

}  // namespace

extern "C" {

size_t adt_tree_attn_workspace_size(int32_t B, int32_t H, int32_t D, int32_t max_nodes,
                                    int32_t max_kv) {
  (void)max_nodes;
  if (B < 1 || H < 1 || (D != 64 && D != 128) || max_kv < 0 || static_cast<int64_t>(B) * H > kMaxBH) return 0;
  adt::DeviceInfo info;
  if (adt::device_info(&info) != ADT_OK) return 0;
  return ws_layout(B, H, D, choose_splits(info.sm_count, B, H, D, max_kv)).total;
}

adt_status adt_tree_attn(const adt_bf16* q, const adt_bf16* k_cache, const adt_bf16* v_cache,
                         const int32_t* kv_len, int64_t cache_stride_b, int64_t cache_stride_h,
                         const adt_bf16* k_tree, const adt_bf16* v_tree, const int32_t* parents,
                         const int32_t* node_offsets, int32_t B, int32_t H, int32_t Hkv, int32_t D,
                         int32_t max_nodes, int32_t max_kv, float softmax_scale, adt_bf16* out,
                         float* lse, void* workspace, size_t workspace_bytes, void* stream) {
  ADT_REQUIRE(q && k_cache && v_cache && kv_len && k_tree && v_tree && parents && node_offsets && out);
  ADT_REQUIRE(B >= 1 && H >= 1 && Hkv >= 1 && H % Hkv == 0);
  ADT_REQUIRE(static_cast<int64_t>(B) * H <= kMaxBH && B <= 65535 && H <= 65535);
  ADT_REQUIRE(max_nodes >= 1 && max_kv >= 0);
  ADT_REQUIRE(softmax_scale > 0.f && softmax_scale < 1e30f);
  if (D != 64 && D != 128) return ADT_ERR_UNSUPPORTED;
  if (max_nodes > kMaxNodes) return ADT_ERR_UNSUPPORTED;
  ADT_REQUIRE(cache_stride_b >= 0 && cache_stride_h >= 0 && cache_stride_b % 8 == 0 &&
              cache_stride_h % 8 == 0);
  ADT_REQUIRE(adt::aligned16(q) && adt::aligned16(k_cache) && adt::aligned16(v_cache) &&
              adt::aligned16(k_tree) && adt::aligned16(v_tree) && adt::aligned16(out));
  adt::DeviceInfo info;
  adt_status st = adt::device_info(&info);
  if (st != ADT_OK) return st;
  const int splits = choose_splits(info.sm_count, B, H, D, max_kv);
  const WsLayout w = ws_layout(B, H, D, splits);
  if (!workspace || workspace_bytes < w.total || !adt::aligned16(workspace)) return ADT_ERR_WORKSPACE;
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  AttnParams prm;
  prm.q = reinterpret_cast<const __nv_bfloat16*>(q);
  prm.kc = reinterpret_cast<const __nv_bfloat16*>(k_cache);
  prm.vc = reinterpret_cast<const __nv_bfloat16*>(v_cache);
  prm.kv_len = kv_len;
  prm.sb = cache_stride_b;
  prm.sh = cache_stride_h;
  prm.kt = reinterpret_cast<const __nv_bfloat16*>(k_tree);
  prm.vt = reinterpret_cast<const __nv_bfloat16*>(v_tree);
  prm.parents = parents;
  prm.offs = node_offsets;
  prm.B = B;
  prm.H = H;
  prm.Hkv = Hkv;
  prm.group = H / Hkv;
  prm.max_kv = max_kv;
  prm.splits = splits;
  prm.scale_log2 = softmax_scale * kLog2e;
  prm.out = reinterpret_cast<__nv_bfloat16*>(out);
  prm.lse = lse;
  prm.part_o = reinterpret_cast<float*>(ws + w.part_o);
  prm.part_ml = reinterpret_cast<float2*>(ws + w.part_ml);
  prm.tickets = reinterpret_cast<unsigned*>(ws + w.tickets);
  prm.err = info.error_word;
  cudaStream_t s = adt::as_stream(stream);
  return D == 128 ? launch<128>(prm, s, info.device) : launch<64>(prm, s, info.device);
}

}  // extern "C"

// ---------------------------------------------------------------------------
// adt_tree_attn_noalloc: the same tree attention for callers that cannot
// allocate device memory themselves, for example a plugin inside a serving
// engine whose host owns every device allocation, or code on a latency-
// critical thread that must not call cudaMalloc (it can synchronise the
// device).  The split partials and completion tickets live in one fixed,
// per-device static array instead of a caller-provided workspace.
// ---------------------------------------------------------------------------

#include <mutex>

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
  ADT_REQUIRE(q && k_cache && v_cache && kv_len && k_tree && v_tree && parents && node_offsets && out);
  ADT_REQUIRE(B >= 1 && H >= 1 && Hkv >= 1 && H % Hkv == 0);
  ADT_REQUIRE(B <= 65535 && H <= 65535);
  ADT_REQUIRE(max_nodes >= 1 && max_kv >= 0);
  ADT_REQUIRE(softmax_scale > 0.f && softmax_scale < 1e30f);
  if (D != 64 && D != 128) return ADT_ERR_UNSUPPORTED;
  if (max_nodes > kMaxNodes) return ADT_ERR_UNSUPPORTED;
  ADT_REQUIRE(cache_stride_b >= 0 && cache_stride_h >= 0 && cache_stride_b % 8 == 0 &&
              cache_stride_h % 8 == 0);
  ADT_REQUIRE(adt::aligned16(q) && adt::aligned16(k_cache) && adt::aligned16(v_cache) &&
              adt::aligned16(k_tree) && adt::aligned16(v_tree) && adt::aligned16(out));
  adt::DeviceInfo info;
  adt_status st = adt::device_info(&info);
  if (st != ADT_OK) return st;
  if (info.device < 0 || info.device >= kNoAllocMaxDevices) return ADT_ERR_UNSUPPORTED;
  std::call_once(g_noalloc_once[info.device], noalloc_setup, info.device);
  if (g_noalloc_status[info.device] != cudaSuccess || !g_noalloc_ptr[info.device]) return ADT_ERR_CUDA;
  // As many splits as the usual heuristic picks, fewer if the partials would
  // not fit; a shape that does not fit even unsplit is rejected.
  int splits = choose_splits(info.sm_count, B, H, D, max_kv);
  while (splits > 1 && noalloc_layout(B, H, D, splits).total > kNoAllocScratchBytes) --splits;
  const NoAllocLayout w = noalloc_layout(B, H, D, splits);
  if (w.total > kNoAllocScratchBytes) return ADT_ERR_WORKSPACE;
  uint8_t* ws = static_cast<uint8_t*>(g_noalloc_ptr[info.device]);
  cudaStream_t s = adt::as_stream(stream);
  // The array keeps the previous call's contents: the tickets must start at zero.
  ADT_CUDA_TRY(cudaMemsetAsync(ws + w.tickets, 0, static_cast<size_t>(B) * H * sizeof(unsigned), s));
  AttnParams prm;
  prm.q = reinterpret_cast<const __nv_bfloat16*>(q);
  prm.kc = reinterpret_cast<const __nv_bfloat16*>(k_cache);
  prm.vc = reinterpret_cast<const __nv_bfloat16*>(v_cache);
  prm.kv_len = kv_len;
  prm.sb = cache_stride_b;
  prm.sh = cache_stride_h;
  prm.kt = reinterpret_cast<const __nv_bfloat16*>(k_tree);
  prm.vt = reinterpret_cast<const __nv_bfloat16*>(v_tree);
  prm.parents = parents;
  prm.offs = node_offsets;
  prm.B = B;
  prm.H = H;
  prm.Hkv = Hkv;
  prm.group = H / Hkv;
  prm.max_kv = max_kv;
  prm.splits = splits;
  prm.scale_log2 = softmax_scale * kLog2e;
  prm.out = reinterpret_cast<__nv_bfloat16*>(out);
  prm.lse = lse;
  prm.part_o = reinterpret_cast<float*>(ws + w.part_o);
  prm.part_ml = reinterpret_cast<float2*>(ws + w.part_ml);
  prm.tickets = reinterpret_cast<unsigned*>(ws + w.tickets);
  prm.err = info.error_word;
  return D == 128 ? launch<128>(prm, s, info.device) : launch<64>(prm, s, info.device);
}
