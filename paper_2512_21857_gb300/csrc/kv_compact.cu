// adt_kv_compact: commit the accepted path's K/V to the cache (the accepted
// draft tokens extend the prefix s_{1:t}, Sec. 3.1), all layers in one launch.
//
// Grid (path slot i, tree b, layer l).  A CTA first checks the whole path of
// tree b (so a malformed path skips the tree entirely), then copies node
// path[b][i]'s K and V rows of every kv head with 16-byte vector moves to
// cache position kv_len[b] + i.  The source (tree buffer) and destination
// (cache) must not overlap, so no ordering between CTAs is needed.
#include "adt_common.cuh"

namespace {

constexpr int kThreads = 256;
constexpr int kMaxInplacePath = 256;  // staged rows per CTA: 128 KB at D = 128

struct CompactParams {
  uint4* kc;
  uint4* vc;
  const int32_t* kv_len;
  int32_t* kv_len_out;
  const uint4* kt;
  const uint4* vt;
  const int32_t* offs;
  const int32_t* path;
  int max_path;
  const int32_t* alen;
  int Hkv, D, max_kv;
  int64_t cls, sb, sh, tls;  // strides in elements
  unsigned* err;
};

// Warp 0: checks path entries 0 .. a of one tree at once (lane j reads
// entries j, j + 32, ...): each a node of the tree (0 <= node < n), the first
// the root.  Entry `want` goes to *want_node, and with keep_all every entry
// to keep[j].  Returns the same verdict in every lane.
__device__ __forceinline__ bool warp_check_path(const int32_t* path, int a, int n, int want, int* want_node,
                                                int* keep) {
  const int lane = threadIdx.x & 31;
  bool bad = false;
  for (int j = lane; j <= a; j += 32) {
    const int node = path[j];
    bad |= node < 0 || node >= n || (j == 0 && node != 0);
    if (j == want) *want_node = node;
    if (keep) keep[j] = node;
  }
  return !__any_sync(adt::kFullMask, bad);
}

__global__ void __launch_bounds__(kThreads) kv_compact_kernel(const CompactParams p) {
  __shared__ int s_ok, s_node;
  adt::pdl_wait_then_release();
  const int i = blockIdx.x, b = blockIdx.y, l = blockIdx.z, tid = threadIdx.x;
  const int a = p.alen[b];
  const int L = p.kv_len[b];
  const int node0 = p.offs[b];
  const int n = p.offs[b + 1] - node0;
  if (tid < 32) {
    int ok = (a >= 0 && a < p.max_path && L >= 0 && static_cast<int64_t>(L) + a + 1 <= p.max_kv) ? 1 : 0;
    unsigned bits = ok ? 0u : ADT_DEVERR_KV_RANGE;
    if (ok && !warp_check_path(p.path + static_cast<int64_t>(b) * p.max_path, a, n, i, &s_node, nullptr)) {
      ok = 0;
      bits = ADT_DEVERR_BAD_PATH;
    }
    if (tid == 0) {
      s_ok = ok;
      if (i == 0 && l == 0) {
        if (!ok) adt::raise_error(p.err, bits);
        if (p.kv_len_out) p.kv_len_out[b] = ok ? L + a + 1 : L;
      }
    }
  }
  __syncthreads();
  if (!s_ok || i > a) return;
  const int node = node0 + s_node;
  const int vec_per_head = p.D / 8;  // 16-byte vectors of bf16
  const int nvec = p.Hkv * vec_per_head;
  const int64_t src = (static_cast<int64_t>(l) * p.tls + static_cast<int64_t>(node) * p.Hkv * p.D) / 8;
  for (int v = tid; v < nvec; v += kThreads) {
    const int g = v / vec_per_head, c = v % vec_per_head;
    const int64_t dst = (static_cast<int64_t>(l) * p.cls + static_cast<int64_t>(b) * p.sb +
                         static_cast<int64_t>(g) * p.sh + static_cast<int64_t>(L + i) * p.D) / 8 + c;
    p.kc[dst] = p.kt[src + v];
    p.vc[dst] = p.vt[src + v];
  }
}

// In-place variant: the tree's K/V rows sit in the cache itself, right
// after the prefix (row kv_len[b] + t holds node t), and the accepted rows
// move down to kv_len[b] + i.  A destination row can be the source of a
// later path entry (path [0, 2, 5]: row L + 2 is written from L + 5 and read
// for i = 1), so each CTA, one (layer, tree, kv head), stages every row it
// moves in shared memory before it writes any.
struct InplaceParams {
  uint4* kc;
  uint4* vc;
  const int32_t* kv_len;
  int32_t* kv_len_out;
  const int32_t* offs;
  const int32_t* path;
  int max_path;
  const int32_t* alen;
  int D, max_kv;
  int64_t cls, sb, sh;  // strides in elements
  unsigned* err;
};

__global__ void __launch_bounds__(kThreads) kv_compact_inplace_kernel(const InplaceParams p) {
  extern __shared__ uint4 stage[];  // [row i][K, V][D / 8]
  __shared__ int s_ok, s_unused;
  __shared__ int path[kMaxInplacePath];  // the tree's path entries 0 .. a
  adt::pdl_wait_then_release();
  const int g = blockIdx.x, b = blockIdx.y, l = blockIdx.z, tid = threadIdx.x;
  const int a = p.alen[b];
  const int L = p.kv_len[b];
  const int n = p.offs[b + 1] - p.offs[b];
  if (tid < 32) {
    // the tree's rows L .. L+n-1 and the path's destinations must fit
    int ok = (a >= 0 && a < p.max_path && L >= 0 && n >= 1 && a < n &&
              static_cast<int64_t>(L) + n <= p.max_kv) ? 1 : 0;
    unsigned bits = ok ? 0u : ADT_DEVERR_KV_RANGE;
    if (ok && !warp_check_path(p.path + static_cast<int64_t>(b) * p.max_path, a, n, -1, &s_unused, path)) {
      ok = 0;
      bits = ADT_DEVERR_BAD_PATH;
    }
    if (tid == 0) {
      s_ok = ok;
      if (g == 0 && l == 0) {
        if (!ok) adt::raise_error(p.err, bits);
        if (p.kv_len_out) p.kv_len_out[b] = ok ? L + a + 1 : L;
      }
    }
  }
  __syncthreads();
  if (!s_ok) return;
  const int vpr = p.D / 8;  // 16-byte vectors per row
  const int64_t base = (static_cast<int64_t>(l) * p.cls + static_cast<int64_t>(b) * p.sb +
                        static_cast<int64_t>(g) * p.sh) / 8;
  const int nv = (a + 1) * vpr;
  for (int v = tid; v < nv; v += kThreads) {
    const int i = v / vpr, c = v % vpr;
    const int64_t src = base + static_cast<int64_t>(L + path[i]) * vpr + c;
    stage[(2 * i) * vpr + c] = p.kc[src];
    stage[(2 * i + 1) * vpr + c] = p.vc[src];
  }
  __syncthreads();
  for (int v = tid; v < nv; v += kThreads) {
    const int i = v / vpr, c = v % vpr;
    if (path[i] == i) continue;  // already in place (the root always is)
    const int64_t dst = base + static_cast<int64_t>(L + i) * vpr + c;
    p.kc[dst] = stage[(2 * i) * vpr + c];
    p.vc[dst] = stage[(2 * i + 1) * vpr + c];
  }
}

}  // namespace

extern "C" {

adt_status adt_kv_compact(adt_bf16* k_cache, adt_bf16* v_cache, const int32_t* kv_len,
                          int32_t* kv_len_out, const adt_bf16* k_tree, const adt_bf16* v_tree,
                          const int32_t* node_offsets, const int32_t* path, int32_t max_path,
                          const int32_t* accept_len, int32_t B, int32_t Hkv, int32_t D,
                          int32_t num_layers, int32_t max_kv, int64_t cache_layer_stride,
                          int64_t cache_stride_b, int64_t cache_stride_h,
                          int64_t tree_layer_stride, void* stream) {
  adt::TraceRange trace_("adt_kv_compact");
  ADT_REQUIRE(k_cache && v_cache && kv_len && k_tree && v_tree && node_offsets && path && accept_len);
  ADT_REQUIRE(B >= 1 && B <= 65535 && Hkv >= 1 && num_layers >= 1 && num_layers <= 65535);
  ADT_REQUIRE(max_path >= 1 && max_path <= (1 << 20) && max_kv >= 1);
  ADT_REQUIRE(kv_len_out != kv_len);
  if (D != 64 && D != 128) return ADT_ERR_UNSUPPORTED;
  ADT_REQUIRE(cache_layer_stride >= 0 && cache_stride_b >= 0 && cache_stride_h >= 0 && tree_layer_stride >= 0);
  ADT_REQUIRE(cache_layer_stride % 8 == 0 && cache_stride_b % 8 == 0 && cache_stride_h % 8 == 0 &&
              tree_layer_stride % 8 == 0);
  ADT_REQUIRE(adt::aligned16(k_cache) && adt::aligned16(v_cache) && adt::aligned16(k_tree) &&
              adt::aligned16(v_tree));
  adt::DeviceInfo info;
  adt_status st = adt::device_info(&info);
  if (st != ADT_OK) return st;
  CompactParams p;
  p.kc = reinterpret_cast<uint4*>(k_cache);
  p.vc = reinterpret_cast<uint4*>(v_cache);
  p.kv_len = kv_len;
  p.kv_len_out = kv_len_out;
  p.kt = reinterpret_cast<const uint4*>(k_tree);
  p.vt = reinterpret_cast<const uint4*>(v_tree);
  p.offs = node_offsets;
  p.path = path;
  p.max_path = max_path;
  p.alen = accept_len;
  p.Hkv = Hkv;
  p.D = D;
  p.max_kv = max_kv;
  p.cls = cache_layer_stride;
  p.sb = cache_stride_b;
  p.sh = cache_stride_h;
  p.tls = tree_layer_stride;
  p.err = info.error_word;
  dim3 grid(static_cast<unsigned>(max_path), static_cast<unsigned>(B), static_cast<unsigned>(num_layers));
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.stream = adt::as_stream(stream);
  cudaLaunchAttribute attr[1] = {adt::pdl_attribute()};
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  ADT_CUDA_TRY(cudaLaunchKernelEx(&cfg, kv_compact_kernel, p));
  return adt::launch_status();
}

adt_status adt_kv_compact_inplace(adt_bf16* k_cache, adt_bf16* v_cache, const int32_t* kv_len,
                                  int32_t* kv_len_out, const int32_t* node_offsets, const int32_t* path,
                                  int32_t max_path, const int32_t* accept_len, int32_t B, int32_t Hkv, int32_t D,
                                  int32_t num_layers, int32_t max_kv, int64_t cache_layer_stride,
                                  int64_t cache_stride_b, int64_t cache_stride_h, void* stream) {
  adt::TraceRange trace_("adt_kv_compact_inplace");
  ADT_REQUIRE(k_cache && v_cache && kv_len && node_offsets && path && accept_len);
  ADT_REQUIRE(B >= 1 && B <= 65535 && Hkv >= 1 && Hkv <= 65535 && num_layers >= 1 && num_layers <= 65535);
  ADT_REQUIRE(max_path >= 1 && max_kv >= 1);
  ADT_REQUIRE(kv_len_out != kv_len);
  if (D != 64 && D != 128) return ADT_ERR_UNSUPPORTED;
  if (max_path > kMaxInplacePath) return ADT_ERR_UNSUPPORTED;
  ADT_REQUIRE(cache_layer_stride >= 0 && cache_stride_b >= 0 && cache_stride_h >= 0);
  ADT_REQUIRE(cache_layer_stride % 8 == 0 && cache_stride_b % 8 == 0 && cache_stride_h % 8 == 0);
  ADT_REQUIRE(adt::aligned16(k_cache) && adt::aligned16(v_cache));
  adt::DeviceInfo info;
  adt_status st = adt::device_info(&info);
  if (st != ADT_OK) return st;
  InplaceParams p;
  p.kc = reinterpret_cast<uint4*>(k_cache);
  p.vc = reinterpret_cast<uint4*>(v_cache);
  p.kv_len = kv_len;
  p.kv_len_out = kv_len_out;
  p.offs = node_offsets;
  p.path = path;
  p.max_path = max_path;
  p.alen = accept_len;
  p.D = D;
  p.max_kv = max_kv;
  p.cls = cache_layer_stride;
  p.sb = cache_stride_b;
  p.sh = cache_stride_h;
  p.err = info.error_word;
  const size_t smem = static_cast<size_t>(max_path) * D * 2 * sizeof(adt_bf16);
  if (smem > 48 * 1024) {
    static unsigned configured[2] = {0u, 0u};  // bit per device (< 64)
    const unsigned bit = 1u << (info.device & 31);
    unsigned& word = configured[(info.device >> 5) & 1];
    if (!(__atomic_load_n(&word, __ATOMIC_ACQUIRE) & bit)) {
      ADT_CUDA_TRY(cudaFuncSetAttribute(kv_compact_inplace_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                        static_cast<int>(kMaxInplacePath) * 128 * 2 * 2));
      __atomic_fetch_or(&word, bit, __ATOMIC_ACQ_REL);
    }
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(Hkv), static_cast<unsigned>(B), static_cast<unsigned>(num_layers));
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = adt::as_stream(stream);
  cudaLaunchAttribute attr[1] = {adt::pdl_attribute()};
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  ADT_CUDA_TRY(cudaLaunchKernelEx(&cfg, kv_compact_inplace_kernel, p));
  return adt::launch_status();
}

}  // extern "C"
