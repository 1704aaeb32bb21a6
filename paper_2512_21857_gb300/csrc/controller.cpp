// Host-side depth / width controller of ADT-Tree (Sec. 4.1 adjacent
// initialisation, Eq. 2 bisectional adaptation, the bounds at the end of
// Sec. 4.2, hyper-parameters of Sec. 5.1).  One object per image; no GPU.
#include <cstdint>
#include <cstring>
#include <new>
#include <vector>

#include "adt.h"

struct adt_ctrl {
  adt_ctrl_params p;
  int32_t h, w;
  std::vector<int32_t> d_grid, k_grid;  // (d, k) of the tree that emitted each position; 0 = not yet
  bool have_alpha = false;
  double alpha_prev = 0.0;
  bool have_cur = false;
  int32_t cur_d = 0, cur_k = 0;
};

namespace {

constexpr uint64_t kGamma = 0x9E3779B97F4A7C15ull;

// SplitMix64 (Steele, Lea, Flood 2014): one output for a state.
uint64_t splitmix64(uint64_t state) {
  uint64_t z = state + kGamma;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

uint64_t counter_draw(uint64_t seed, uint64_t counter) { return splitmix64(seed + counter * kGamma); }

int32_t clamp(int32_t x, int32_t lo, int32_t hi) { return x < lo ? lo : (x > hi ? hi : x); }

// TokenFlock initialisation (the alternative of Table 3): the generated
// positions within Euclidean distance delta of (row i, column j) that come
// before it, each weighted by delta + 1 - (rows above); returns false when
// there are none.  Integer weights make the mean an exact fraction, rounded
// half up.
bool flock_init(const adt_ctrl* c, int32_t i, int32_t j, int32_t* d, int32_t* k) {
  const int32_t delta = c->p.flock_delta;
  int64_t wsum = 0, dsum = 0, ksum = 0;
  for (int32_t dy = delta; dy >= 0; --dy) {
    const int32_t r = i - dy;
    if (r < 0) continue;
    for (int32_t dx = -delta; dx <= delta; ++dx) {
      const int32_t col = j + dx;
      if (col < 0 || col >= c->w) continue;
      if (dy == 0 && dx >= 0) break;  // only positions before (i, j)
      if (dx * dx + dy * dy > delta * delta) continue;
      const int32_t q = r * c->w + col;
      if (c->d_grid[q] <= 0) continue;
      const int64_t wgt = delta + 1 - dy;
      wsum += wgt;
      dsum += wgt * c->d_grid[q];
      ksum += wgt * c->k_grid[q];
    }
  }
  if (wsum == 0) return false;
  *d = static_cast<int32_t>((2 * dsum + wsum) / (2 * wsum));
  *k = static_cast<int32_t>((2 * ksum + wsum) / (2 * wsum));
  return true;
}

}  // namespace

extern "C" {

adt_status adt_ctrl_create(const adt_ctrl_params* params, int32_t grid_h, int32_t grid_w,
                           adt_ctrl** out) {
  if (!params || !out || grid_h < 1 || grid_w < 1) return ADT_ERR_INVALID_ARG;
  const adt_ctrl_params& p = *params;
  if (p.d_lo < 1 || p.d_hi < p.d_lo || p.k_lo < 1 || p.k_hi < p.k_lo || p.k_cap < p.k_hi) return ADT_ERR_INVALID_ARG;
  if (p.l_d < 0 || p.l_k < 0 || p.d0 < 1 || p.k0 < 1 || p.fix_d < 0 || p.fix_k < 0) return ADT_ERR_INVALID_ARG;
  if (p.init_mode != ADT_INIT_HORIZONTAL && p.init_mode != ADT_INIT_VERTICAL && p.init_mode != ADT_INIT_RANDOM &&
      p.init_mode != ADT_INIT_TOKENFLOCK)
    return ADT_ERR_INVALID_ARG;
  if (p.init_mode == ADT_INIT_TOKENFLOCK && (p.flock_delta < 1 || p.flock_delta > 64)) return ADT_ERR_INVALID_ARG;
  if (static_cast<int64_t>(grid_h) * grid_w > (int64_t{1} << 28)) return ADT_ERR_INVALID_ARG;
  adt_ctrl* c = new (std::nothrow) adt_ctrl;
  if (!c) return ADT_ERR_INVALID_ARG;
  c->p = p;
  c->h = grid_h;
  c->w = grid_w;
  try {
    c->d_grid.assign(static_cast<size_t>(grid_h) * grid_w, 0);
    c->k_grid.assign(static_cast<size_t>(grid_h) * grid_w, 0);
  } catch (...) {
    delete c;
    return ADT_ERR_INVALID_ARG;
  }
  *out = c;
  return ADT_OK;
}

void adt_ctrl_destroy(adt_ctrl* ctrl) { delete ctrl; }

adt_status adt_ctrl_next(adt_ctrl* c, int32_t pos, int32_t* depth, int32_t* width) {
  if (!c || !depth || !width) return ADT_ERR_INVALID_ARG;
  const int32_t n = c->h * c->w;
  if (pos < 0 || pos >= n) return ADT_ERR_INVALID_ARG;
  const adt_ctrl_params& P = c->p;
  const int32_t i = pos / c->w;
  int32_t d, k;
  // Adjacent initialisation (Sec. 4.1).
  if (P.init_mode == ADT_INIT_TOKENFLOCK) {
    if (!flock_init(c, i, pos % c->w, &d, &k)) {
      d = P.d0;
      k = P.k0;
    }
  } else if (P.init_mode == ADT_INIT_RANDOM) {
    d = P.d_lo + static_cast<int32_t>(counter_draw(P.seed, 2ull * static_cast<uint64_t>(pos)) %
                                      static_cast<uint64_t>(P.d_hi - P.d_lo + 1));
    k = P.k_lo + static_cast<int32_t>(counter_draw(P.seed, 2ull * static_cast<uint64_t>(pos) + 1) %
                                      static_cast<uint64_t>(P.k_hi - P.k_lo + 1));
  } else if (P.init_mode == ADT_INIT_VERTICAL && i >= 1 && c->d_grid[pos - c->w] > 0) {
    d = c->d_grid[pos - c->w];
    k = c->k_grid[pos - c->w];
  } else if (pos >= 1 && c->d_grid[pos - 1] > 0) {
    d = c->d_grid[pos - 1];
    k = c->k_grid[pos - 1];
  } else {
    d = P.d0;
    k = P.k0;
  }
  if (P.fix_d > 0) d = P.fix_d;
  if (P.fix_k > 0) k = P.fix_k;
  // Bisectional dynamic adaptation (Eq. 2).
  if (c->have_alpha) {
    if (c->alpha_prev >= P.beta) {
      d += P.l_d;
      k -= P.l_k;
    } else {
      d -= P.l_d;
      k += P.l_k;
    }
  }
  // Bounds (end of Sec. 4.2): width is restricted only when the adapted depth exceeds 1.
  const bool restrict_k = P.clamp_k_always != 0 || d > 1;
  d = clamp(d, P.d_lo, P.d_hi);
  k = restrict_k ? clamp(k, P.k_lo, P.k_hi) : clamp(k, 1, P.k_cap);
  c->cur_d = d;
  c->cur_k = k;
  c->have_cur = true;
  *depth = d;
  *width = k;
  return ADT_OK;
}

adt_status adt_ctrl_update(adt_ctrl* c, int32_t pos, int32_t accept_len, int32_t* next_pos) {
  if (!c || !c->have_cur) return ADT_ERR_INVALID_ARG;
  const int32_t n = c->h * c->w;
  if (pos < 0 || pos >= n || accept_len < 0 || accept_len > c->cur_d) return ADT_ERR_INVALID_ARG;
  // alpha = accepted draft nodes / tree depth (Sec. 3.2 defines alpha = tau / d).
  c->alpha_prev = static_cast<double>(accept_len) / static_cast<double>(c->cur_d);
  c->have_alpha = true;
  const int32_t end = pos + accept_len + 1 < n ? pos + accept_len + 1 : n;
  for (int32_t t = pos; t < end; ++t) {
    c->d_grid[t] = c->cur_d;
    c->k_grid[t] = c->cur_k;
  }
  if (next_pos) *next_pos = pos + accept_len + 1;
  return ADT_OK;
}

// Saved state: a header, the parameters, the adaptation state and the two
// grids, in host byte order (a checkpoint for the same build, not an
// interchange format).
namespace {
constexpr uint32_t kStateMagic = 0x41445443u;  // "ADTC"
constexpr uint32_t kStateVersion = 1u;
struct StateHeader {
  uint32_t magic, version;
  int32_t h, w;
  adt_ctrl_params p;
  double alpha_prev;
  int32_t have_alpha, have_cur, cur_d, cur_k;
};
}  // namespace

size_t adt_ctrl_state_size(const adt_ctrl* c) {
  if (!c) return 0;
  return sizeof(StateHeader) + 2 * c->d_grid.size() * sizeof(int32_t);
}

adt_status adt_ctrl_save(const adt_ctrl* c, void* buf, size_t bytes) {
  if (!c || !buf || bytes < adt_ctrl_state_size(c)) return ADT_ERR_INVALID_ARG;
  StateHeader hd;
  std::memset(&hd, 0, sizeof(hd));
  hd.magic = kStateMagic;
  hd.version = kStateVersion;
  hd.h = c->h;
  hd.w = c->w;
  hd.p = c->p;
  hd.alpha_prev = c->alpha_prev;
  hd.have_alpha = c->have_alpha ? 1 : 0;
  hd.have_cur = c->have_cur ? 1 : 0;
  hd.cur_d = c->cur_d;
  hd.cur_k = c->cur_k;
  uint8_t* out = static_cast<uint8_t*>(buf);
  std::memcpy(out, &hd, sizeof(hd));
  const size_t g = c->d_grid.size() * sizeof(int32_t);
  std::memcpy(out + sizeof(hd), c->d_grid.data(), g);
  std::memcpy(out + sizeof(hd) + g, c->k_grid.data(), g);
  return ADT_OK;
}

adt_status adt_ctrl_load(const void* buf, size_t bytes, adt_ctrl** out) {
  if (!buf || !out || bytes < sizeof(StateHeader)) return ADT_ERR_INVALID_ARG;
  StateHeader hd;
  std::memcpy(&hd, buf, sizeof(hd));
  if (hd.magic != kStateMagic || hd.version != kStateVersion || hd.h < 1 || hd.w < 1 ||
      static_cast<int64_t>(hd.h) * hd.w > (int64_t{1} << 28))
    return ADT_ERR_INVALID_ARG;
  const size_t g = static_cast<size_t>(hd.h) * hd.w * sizeof(int32_t);
  if (bytes < sizeof(hd) + 2 * g) return ADT_ERR_INVALID_ARG;
  adt_ctrl* c = nullptr;
  adt_status st = adt_ctrl_create(&hd.p, hd.h, hd.w, &c);  // validates the parameters
  if (st != ADT_OK) return st;
  const uint8_t* in = static_cast<const uint8_t*>(buf);
  std::memcpy(c->d_grid.data(), in + sizeof(hd), g);
  std::memcpy(c->k_grid.data(), in + sizeof(hd) + g, g);
  c->alpha_prev = hd.alpha_prev;
  c->have_alpha = hd.have_alpha != 0;
  c->have_cur = hd.have_cur != 0;
  c->cur_d = hd.cur_d;
  c->cur_k = hd.cur_k;
  *out = c;
  return ADT_OK;
}

adt_status adt_ctrl_get(const adt_ctrl* c, int32_t pos, int32_t* depth, int32_t* width) {
  if (!c || !depth || !width || pos < 0 || pos >= c->h * c->w) return ADT_ERR_INVALID_ARG;
  *depth = c->d_grid[pos];
  *width = c->k_grid[pos];
  return ADT_OK;
}

}  // extern "C"
