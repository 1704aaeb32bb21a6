// adt_tree_expand: one layer of EAGLE-2-style dynamic draft-tree growth
// (Sec. 3.1, last paragraph; Fig. 5; node score Eq. 4 in the log domain), and
// adt_tree_rerank: the final top-N tree (Eq. 4 and the sentence after it).
//
// Expand is one launch over (vocab chunk, frontier row).  Each CTA stages a
// 4096-logit chunk in shared memory, computes the chunk's max and sum of
// exponentials and its exact top-k by radix selection on 64-bit keys
// (value order, then lower index), and writes them to the workspace.  The
// last CTA of a row (atomic ticket) merges the chunk results into the row's
// top-k and log-sum-exp and writes the children; the last row to finish
// selects the next frontier across all rows the same way.
#include "adt_common.cuh"

namespace {

constexpr int kThreads = 256;
constexpr int kChunk = 4096;
constexpr int kMaxK = 64;
constexpr int kMaxKeep = 1024;

struct ExpandParams {
  const float* logits;
  int64_t ld;
  const float* fscore;
  const int32_t* fid;
  int F, V, k, k_keep, S;
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
  uint64_t* part_keys;  // [F][S][k]
  float* part_max;      // [F][S]
  double* part_sum;     // [F][S]
  uint64_t* cross_keys; // [F*k]
  unsigned* row_tickets;  // [F]
  unsigned* all_ticket;   // [1]
};

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

__global__ void __launch_bounds__(kThreads) expand_kernel(const ExpandParams p) {
  __shared__ float vals[kChunk];
  __shared__ uint64_t sel[kMaxKeep];
  __shared__ adt::RadixScratch rs;
  __shared__ double dred[32];
  __shared__ float fred[32];
  __shared__ unsigned s_cnt;
  __shared__ int s_last;
  __shared__ double s_lse;

  const int s = blockIdx.x, r = blockIdx.y, tid = threadIdx.x;
  const int t0 = s * kChunk;
  const int len = min(kChunk, p.V - t0);
  const float* row = p.logits + static_cast<int64_t>(r) * p.ld;

  // Stage the chunk (x / T in fp32, round-to-nearest division).
  for (int i = tid * 4; i < len; i += kThreads * 4) {
    float x[4];
    if (i + 3 < len) {
      const float4 v = __ldg(reinterpret_cast<const float4*>(row + t0 + i));
      x[0] = v.x; x[1] = v.y; x[2] = v.z; x[3] = v.w;
    } else {
      for (int e = 0; e < 4; ++e) x[e] = (i + e < len) ? __ldg(row + t0 + i + e) : 0.f;
    }
    for (int e = 0; e < 4 && i + e < len; ++e) vals[i + e] = p.use_T ? __fdiv_rn(x[e], p.T) : x[e];
  }
  __syncthreads();

  float m = -INFINITY;
  for (int i = tid; i < len; i += kThreads) m = fmaxf(m, vals[i]);
  m = adt::block_max<kThreads>(m, fred);
  float acc = 0.f;
  for (int i = tid; i < len; i += kThreads) acc += expf(vals[i] - m);
  const double tot = adt::block_sum<kThreads, double>(static_cast<double>(acc), dred);

  const int kk = min(p.k, len);
  auto chunk_key = [&](int i) { return adt::select_key(vals[i], static_cast<uint32_t>(t0 + i)); };
  const uint64_t thr = adt::block_topk_threshold<kThreads>(chunk_key, len, kk, &rs);
  collect_sorted(chunk_key, len, thr, kk, sel, &s_cnt);

  const int64_t rs_idx = static_cast<int64_t>(r) * p.S + s;
  for (int j = tid; j < p.k; j += kThreads) p.part_keys[rs_idx * p.k + j] = j < kk ? sel[j] : 0ull;
  if (tid == 0) {
    p.part_max[rs_idx] = m;
    p.part_sum[rs_idx] = tot;
  }
  __threadfence();
  __syncthreads();
  if (tid == 0) s_last = atomicAdd(p.row_tickets + r, 1u) == static_cast<unsigned>(p.S - 1);
  __syncthreads();
  if (!s_last) return;
  __threadfence();

  // ---- last CTA of row r: merge chunk results.
  const uint64_t* rk = p.part_keys + static_cast<int64_t>(r) * p.S * p.k;
  auto row_key = [&](int i) { return __ldcg(rk + i); };
  const uint64_t thr2 = adt::block_topk_threshold<kThreads>(row_key, p.S * p.k, p.k, &rs);
  collect_sorted(row_key, p.S * p.k, thr2, p.k, sel, &s_cnt);
  if (tid < 32) {
    double M = -INFINITY;
    for (int c = tid; c < p.S; c += 32) M = fmax(M, static_cast<double>(__ldcg(p.part_max + r * p.S + c)));
    for (int o = 16; o > 0; o >>= 1) M = fmax(M, __shfl_xor_sync(adt::kFullMask, M, o));
    double sum = 0.0;
    for (int c = tid; c < p.S; c += 32) {
      const double mc = __ldcg(p.part_max + r * p.S + c);
      sum += __ldcg(p.part_sum + r * p.S + c) * exp(mc - M);
    }
    sum = adt::warp_sum(sum);
    if (tid == 0) s_lse = M + log(sum);
  }
  __syncthreads();
  const double lse = s_lse;
  const float ps = p.fscore[r];
  const int32_t parent = p.fid ? p.fid[r] : r;
  for (int j = tid; j < p.k; j += kThreads) {
    const uint64_t key = sel[j];
    const float x = adt::select_key_value(key);
    const double lp = static_cast<double>(x) - lse;
    const float score = static_cast<float>(static_cast<double>(ps) + lp);
    const int64_t c = static_cast<int64_t>(r) * p.k + j;
    p.ctok[c] = static_cast<int32_t>(adt::select_key_index(key));
    if (p.clogp) p.clogp[c] = static_cast<float>(lp);
    p.cscore[c] = score;
    p.cpar[c] = parent;
    p.cross_keys[c] = adt::select_key(score, static_cast<uint32_t>(c));
  }
  if (tid == 0) p.row_tickets[r] = 0u;
  __threadfence();
  __syncthreads();
  if (tid == 0) s_last = atomicAdd(p.all_ticket, 1u) == static_cast<unsigned>(p.F - 1);
  __syncthreads();
  if (!s_last) return;
  __threadfence();

  // ---- last row: next frontier across all rows.
  const int nc = p.F * p.k;
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
  if (tid == 0) *p.all_ticket = 0u;
}

// Workspace layout.  The completion counters sit at fixed offsets at the
// start (room for the largest F), so calls of any shape can share one
// workspace; the data regions after them are rewritten before being read.
constexpr int kMaxRows = 4096;

struct ExpandWs {
  size_t row_tickets, all_ticket, part_keys, part_max, part_sum, cross_keys, total;
};

ExpandWs expand_ws(int F, int V, int k) {
  const size_t S = (static_cast<size_t>(V) + kChunk - 1) / kChunk;
  ExpandWs w{};
  w.row_tickets = 0;
  w.all_ticket = kMaxRows * sizeof(unsigned);
  w.part_keys = adt::align_up(w.all_ticket + sizeof(unsigned), 256);
  w.part_max = adt::align_up(w.part_keys + F * S * k * sizeof(uint64_t), 256);
  w.part_sum = adt::align_up(w.part_max + F * S * sizeof(float), 256);
  w.cross_keys = adt::align_up(w.part_sum + F * S * sizeof(double), 256);
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

__global__ void __launch_bounds__(kRerankThreads) rerank_kernel(const RerankParams p) {
  __shared__ adt::RadixScratch rs;
  __shared__ int warp_tot[32];
  __shared__ int warp_excl[32];
  __shared__ int s_running;
  __shared__ int s_tile;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int need = p.n_nodes - 1;
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
  ADT_REQUIRE(logits && frontier_score && child_token && child_score && child_parent && keep_idx);
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
  p.ld = ld;
  p.fscore = frontier_score;
  p.fid = frontier_id;
  p.F = F;
  p.V = V;
  p.k = k_child;
  p.k_keep = k_keep;
  p.S = (V + kChunk - 1) / kChunk;
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
  p.part_keys = reinterpret_cast<uint64_t*>(ws + w.part_keys);
  p.part_max = reinterpret_cast<float*>(ws + w.part_max);
  p.part_sum = reinterpret_cast<double*>(ws + w.part_sum);
  p.cross_keys = reinterpret_cast<uint64_t*>(ws + w.cross_keys);
  p.row_tickets = reinterpret_cast<unsigned*>(ws + w.row_tickets);
  p.all_ticket = reinterpret_cast<unsigned*>(ws + w.all_ticket);
  dim3 grid(p.S, F);
  expand_kernel<<<grid, kThreads, 0, adt::as_stream(stream)>>>(p);
  return adt::launch_status();
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
  rerank_kernel<<<1, kRerankThreads, 0, adt::as_stream(stream)>>>(p);
  return adt::launch_status();
}

}  // extern "C"
