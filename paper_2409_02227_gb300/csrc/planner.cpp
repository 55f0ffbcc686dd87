// Host-side dynamic logic: lookup table, bucketing and planning.
//
// The paper's command-processor logic (Sec. 4.3, Sec. 4.4) inspects the
// independent GEMMs waiting at the queue heads, predicts the concurrency
// degree (CD) worth running, and rewrites each GEMM's kernel pointer to the
// GO-Kernel tuned for that CD.  NVIDIA exposes no programmable command
// processor, so this runs on the host right before launch: integer work over
// at most 64 descriptors, no CUDA call, a pure function of its inputs.
//
// Rules (Sec. 4.3: CD = min(preferred CD, GEMMs available); Sec. 6.7: a
// heterogeneous set runs at once only when every distinct GEMM prefers that
// many, otherwise homogeneous groups each with its own CD):
//   key      = (floor log2 M, floor log2 N, floor log2 K, C dtype)
//   lookup   = exact key, else nearest stored key (L1 over the log2 sizes,
//              +16 for a differing dtype), ties to the smallest key
//   blocks   = one per distinct key, in decreasing total FLOPs (ties: smaller
//              key), merged greedily with the next block while every key in
//              the merged group prefers at least the merged size
//   group CD = min(pref, size) for one key, size for a merged group
//   slots    = member j of a group -> slot j mod CD
//   kernel   = table's variant for the smallest CD class >= the group's CD
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <fstream>
#include <iterator>
#include <new>
#include <string>
#include <vector>

#include "goldy_internal.h"

namespace goldy {


static thread_local std::string g_last_error;

goldy_status fail(goldy_status st, const std::string& msg) {
  g_last_error = msg;
  return st;
}
goldy_status ok() {
  g_last_error.clear();
  return GOLDY_OK;
}

goldy_status check_desc(const goldy_gemm_desc& d, int i) {
  const std::string at = "gemm " + std::to_string(i) + ": ";
  if (d.trans_a != 0 || d.trans_b != 0)
    return fail(GOLDY_ERR_UNSUPPORTED, at + "transposed operands are not supported");
  if (d.a_dtype != GOLDY_BF16 || d.b_dtype != GOLDY_BF16)
    return fail(GOLDY_ERR_UNSUPPORTED, at + "A and B must be bf16");
  if (d.c_dtype != GOLDY_BF16 && d.c_dtype != GOLDY_F32)
    return fail(GOLDY_ERR_UNSUPPORTED, at + "C must be bf16 or fp32");
  if (d.reserved != 0) return fail(GOLDY_ERR_INVALID_ARG, at + "reserved field must be 0");
  if (d.M < 0 || d.N < 0 || d.K < 0) return fail(GOLDY_ERR_INVALID_ARG, at + "negative size");
  const int64_t lim = int64_t(1) << 31;
  if (d.M >= lim || d.N >= lim || d.K >= lim)
    return fail(GOLDY_ERR_INVALID_ARG, at + "size does not fit 31 bits");
  if (d.lda < std::max<int64_t>(d.K, 1) || d.ldb < std::max<int64_t>(d.N, 1) ||
      d.ldc < std::max<int64_t>(d.N, 1))
    return fail(GOLDY_ERR_INVALID_ARG, at + "leading dimension smaller than the row");
  if (d.lda % 8 != 0 || d.ldb % 8 != 0)
    return fail(GOLDY_ERR_INVALID_ARG, at + "lda and ldb must be multiples of 8 (16-byte rows)");
  if (d.lda >= (int64_t(1) << 36) || d.ldb >= (int64_t(1) << 36))
    return fail(GOLDY_ERR_INVALID_ARG, at + "leading dimension too large");
  if (d.batch < 1 || d.batch >= lim) return fail(GOLDY_ERR_INVALID_ARG, at + "batch must be in 1 .. 2^31-1");
  if (d.batch > 1) {
    if (d.stride_a < d.M * d.lda || d.stride_b < d.K * d.ldb || d.stride_c < d.M * d.ldc)
      return fail(GOLDY_ERR_INVALID_ARG, at + "batch entries overlap (stride smaller than one entry)");
    if (d.stride_a % 8 != 0 || d.stride_b % 8 != 0)
      return fail(GOLDY_ERR_INVALID_ARG, at + "stride_a and stride_b must be multiples of 8 (16 bytes)");
    if (d.stride_a >= (int64_t(1) << 36) || d.stride_b >= (int64_t(1) << 36) || d.stride_c >= (int64_t(1) << 36))
      return fail(GOLDY_ERR_INVALID_ARG, at + "batch stride too large");
  }
  return GOLDY_OK;
}

static uint8_t floor_log2_u8(int64_t x) {
  if (x <= 0) return 0;
  int b = 0;
  while ((x >> 1) > 0) {
    x >>= 1;
    ++b;
  }
  return (uint8_t)std::min(b, 255);
}

}  // namespace goldy

using namespace goldy;

// ---------------------------------------------------------------------------
// Lookup table
// ---------------------------------------------------------------------------
namespace {
struct LutEntry {
  uint8_t lm, ln, lk, out;
  uint8_t pref_cd;
  uint8_t flags;   // co-run with an element-wise op: bit 0 at once, bit 1 CD-2 kernel, bits 2-3 add cap
  uint16_t variant[5];
  uint32_t key() const { return (uint32_t(lm) << 24) | (uint32_t(ln) << 16) | (uint32_t(lk) << 8) | out; }
};
constexpr int kCdClasses[5] = {1, 2, 4, 8, 16};

uint32_t rd32(const uint8_t* p) { return uint32_t(p[0]) | (uint32_t(p[1]) << 8) | (uint32_t(p[2]) << 16) | (uint32_t(p[3]) << 24); }
uint16_t rd16(const uint8_t* p) { return uint16_t(p[0] | (p[1] << 8)); }

int cd_class_index(int cd) {
  for (int i = 0; i < 5; ++i)
    if (cd <= kCdClasses[i]) return i;
  return 4;
}
}  // namespace

struct goldy_lut {
  std::vector<LutEntry> entries;
  uint32_t n_variants = 0;
  uint32_t sm_count = 0;
};

extern "C" goldy_status goldy_lut_from_memory(const void* data, size_t bytes, goldy_lut** out) {
  if (!data || !out) return fail(GOLDY_ERR_INVALID_ARG, "null argument");
  *out = nullptr;
  const uint8_t* p = static_cast<const uint8_t*>(data);
  if (bytes < 32 || std::memcmp(p, "GOLDYLUT", 8) != 0) return fail(GOLDY_ERR_LUT, "lut: bad magic");
  const uint32_t version = rd32(p + 8), n = rd32(p + 12), nv = rd32(p + 16), sm = rd32(p + 20);
  if (version != 1) return fail(GOLDY_ERR_LUT, "lut: unsupported version");
  if (uint64_t(bytes) != 32 + 16 * uint64_t(n)) return fail(GOLDY_ERR_LUT, "lut: size does not match entry count");
  if (n == 0) return fail(GOLDY_ERR_LUT, "lut: empty table");
  if (nv == 0 || nv > uint32_t(kNumVariants))
    return fail(GOLDY_ERR_LUT, "lut: variant-id bound does not match this library");
  goldy_lut* lut = new (std::nothrow) goldy_lut();
  if (!lut) return fail(GOLDY_ERR_NOMEM, "lut: out of host memory");
  lut->n_variants = nv;
  lut->sm_count = sm;
  lut->entries.resize(n);
  for (uint32_t e = 0; e < n; ++e) {
    const uint8_t* q = p + 32 + 16 * size_t(e);
    LutEntry& x = lut->entries[e];
    x.lm = q[0];
    x.ln = q[1];
    x.lk = q[2];
    x.out = q[3];
    x.pref_cd = q[4];
    x.flags = q[5];
    for (int c = 0; c < 5; ++c) x.variant[c] = rd16(q + 6 + 2 * c);
    bool bad = (x.out != GOLDY_BF16 && x.out != GOLDY_F32) || (x.flags & ~0x0Fu) != 0 || ((x.flags >> 2) & 3u) == 3u;
    bool pref_ok = false;
    for (int c : kCdClasses) pref_ok |= (x.pref_cd == c);
    bad |= !pref_ok;
    for (int c = 0; c < 5; ++c) bad |= (x.variant[c] >= nv);
    if (e > 0) bad |= (x.key() <= lut->entries[e - 1].key());
    if (bad) {
      delete lut;
      return fail(GOLDY_ERR_LUT, "lut: malformed entry " + std::to_string(e));
    }
  }
  *out = lut;
  return ok();
}

extern "C" goldy_status goldy_lut_load(const char* path, goldy_lut** out) {
  if (!path || !out) return fail(GOLDY_ERR_INVALID_ARG, "null argument");
  *out = nullptr;
  std::ifstream f(path, std::ios::binary);
  if (!f) return fail(GOLDY_ERR_LUT, std::string("lut: cannot open ") + path);
  std::vector<char> buf((std::istreambuf_iterator<char>(f)), std::istreambuf_iterator<char>());
  return goldy_lut_from_memory(buf.data(), buf.size(), out);
}

extern "C" void goldy_lut_free(goldy_lut* lut) { delete lut; }

// ---------------------------------------------------------------------------
// Logistic-regression CD predictor (Sec. 4.3, Eq. 1)
// ---------------------------------------------------------------------------
struct goldy_predictor {
  double lo[GOLDY_LR_FEATURES], hi[GOLDY_LR_FEATURES];
  double W[5][GOLDY_LR_FEATURES], b[5];
  uint32_t sm_count = 0;
};

static double rd_f64(const uint8_t* p) {
  uint64_t u = 0;
  for (int i = 7; i >= 0; --i) u = (u << 8) | p[i];
  double d;
  std::memcpy(&d, &u, sizeof d);
  return d;
}

extern "C" goldy_status goldy_predictor_from_memory(const void* data, size_t bytes, goldy_predictor** out) {
  if (!data || !out) return fail(GOLDY_ERR_INVALID_ARG, "null argument");
  *out = nullptr;
  constexpr int nf = GOLDY_LR_FEATURES, nc = 5;
  const uint8_t* p = static_cast<const uint8_t*>(data);
  if (bytes < 32 || std::memcmp(p, "GOLDYLRM", 8) != 0) return fail(GOLDY_ERR_LUT, "predictor: bad magic");
  if (rd32(p + 8) != 1 || rd32(p + 12) != uint32_t(nf) || rd32(p + 16) != uint32_t(nc))
    return fail(GOLDY_ERR_LUT, "predictor: unsupported version or shape");
  const uint32_t sm = rd32(p + 20);
  if (sm == 0) return fail(GOLDY_ERR_LUT, "predictor: SM count is zero");
  if (bytes != 32 + 8 * size_t(2 * nf + nc * nf + nc)) return fail(GOLDY_ERR_LUT, "predictor: bad size");
  goldy_predictor* m = new (std::nothrow) goldy_predictor();
  if (!m) return fail(GOLDY_ERR_NOMEM, "predictor: out of host memory");
  m->sm_count = sm;
  const uint8_t* q = p + 32;
  bool bad = false;
  auto next = [&]() {
    const double v = rd_f64(q);
    q += 8;
    bad |= !std::isfinite(v);
    return v;
  };
  for (int j = 0; j < nf; ++j) m->lo[j] = next();
  for (int j = 0; j < nf; ++j) m->hi[j] = next();
  for (int c = 0; c < nc; ++c)
    for (int j = 0; j < nf; ++j) m->W[c][j] = next();
  for (int c = 0; c < nc; ++c) m->b[c] = next();
  for (int j = 0; j < nf && !bad; ++j) bad |= (m->hi[j] < m->lo[j]);
  if (bad) {
    delete m;
    return fail(GOLDY_ERR_LUT, "predictor: non-finite value or hi below lo");
  }
  *out = m;
  return ok();
}

extern "C" goldy_status goldy_predictor_load(const char* path, goldy_predictor** out) {
  if (!path || !out) return fail(GOLDY_ERR_INVALID_ARG, "null argument");
  *out = nullptr;
  std::ifstream f(path, std::ios::binary);
  if (!f) return fail(GOLDY_ERR_LUT, std::string("predictor: cannot open ") + path);
  std::vector<char> buf((std::istreambuf_iterator<char>(f)), std::istreambuf_iterator<char>());
  return goldy_predictor_from_memory(buf.data(), buf.size(), out);
}

extern "C" void goldy_predictor_free(goldy_predictor* m) { delete m; }

static uint32_t bucket_key(const goldy_gemm_desc& d) {
  return (uint32_t(floor_log2_u8(d.M * std::max<int64_t>(d.batch, 1))) << 24) |
         (uint32_t(floor_log2_u8(d.N)) << 16) |
         (uint32_t(floor_log2_u8(d.K)) << 8) | uint32_t(d.c_dtype & 0xFF);
}

extern "C" goldy_status goldy_bucket_key(const goldy_gemm_desc* d, uint32_t* key) {
  if (!d || !key) return fail(GOLDY_ERR_INVALID_ARG, "null argument");
  *key = bucket_key(*d);
  return ok();
}

static const LutEntry& lookup(const goldy_lut& lut, uint32_t key) {
  const int lm = key >> 24, ln = (key >> 16) & 0xFF, lk = (key >> 8) & 0xFF, out = key & 0xFF;
  size_t best = 0;
  int best_d = -1;
  for (size_t e = 0; e < lut.entries.size(); ++e) {   // sorted ascending: first minimum wins ties
    const LutEntry& x = lut.entries[e];
    int d = std::abs(int(x.lm) - lm) + std::abs(int(x.ln) - ln) + std::abs(int(x.lk) - lk) +
            (int(x.out) != out ? 16 : 0);
    if (best_d < 0 || d < best_d) {
      best_d = d;
      best = e;
    }
  }
  return lut.entries[best];
}

extern "C" goldy_status goldy_lut_lookup(const goldy_lut* lut, const goldy_gemm_desc* d, int* pref_cd,
                                         int variants[5]) {
  if (!lut || !d || !pref_cd || !variants) return fail(GOLDY_ERR_INVALID_ARG, "null argument");
  const LutEntry& e = lookup(*lut, bucket_key(*d));
  *pref_cd = e.pref_cd;
  for (int c = 0; c < 5; ++c) variants[c] = e.variant[c];
  return ok();
}

// Features of one GEMM for the predictor (Sec. 4.3): M (times the batch), N,
// K, then for each CD class the table's GO-Kernel's CTAs of work (tiles over
// all batch entries x split-K slices, two CTAs per tile for a CTA pair), CTAs
// resident per SM, and waves (CTAs of work over the capped persistent grid,
// rounded up).
static void lr_features(const goldy_gemm_desc& d, const LutEntry& e, int64_t sm_count,
                        double x[GOLDY_LR_FEATURES]) {
  x[0] = double(d.M * d.batch);
  x[1] = double(d.N);
  x[2] = double(d.K);
  for (int c = 0; c < 5; ++c) {
    const Variant v = variant_of(e.variant[c]);
    const KindInfo& k = kKinds[v.kind];
    const int64_t per_tile = k.pair ? 2 : 1;
    const int64_t split = v.split;
    const int64_t ctas = d.batch * ceil_div(d.M, tile_rows(k)) * ceil_div(d.N, tile_cols(k)) * split * per_tile;
    const int64_t cap = std::max<int64_t>(per_tile, int64_t(k.ctas_per_sm) * sm_count / v.rc_div);
    x[3 + 3 * c] = double(ctas);
    x[4 + 3 * c] = double(k.ctas_per_sm);
    x[5 + 3 * c] = double(ceil_div(ctas, cap));
  }
}

extern "C" goldy_status goldy_lr_features(const goldy_gemm_desc* d, const goldy_lut* lut, int sm_count,
                                          double out[GOLDY_LR_FEATURES]) {
  if (!d || !lut || !out) return fail(GOLDY_ERR_INVALID_ARG, "null argument");
  if (sm_count < 1) return fail(GOLDY_ERR_INVALID_ARG, "SM count must be positive");
  goldy_status st = check_desc(*d, 0);
  if (st != GOLDY_OK) return st;
  lr_features(*d, lookup(*lut, bucket_key(*d)), sm_count, out);
  return ok();
}

// Class index (0..4 for CD 1, 2, 4, 8, 16) of largest score; scores are
// accumulated in a fixed order without contraction so that the decision is
// reproducible bit for bit.
static int lr_predict(const goldy_predictor& m, const double x[GOLDY_LR_FEATURES], double s[5]) {
  int best = 0;
  for (int c = 0; c < 5; ++c) {
    double acc = m.b[c];
    for (int j = 0; j < GOLDY_LR_FEATURES; ++j) {
      const double xn = m.hi[j] > m.lo[j] ? (x[j] - m.lo[j]) / (m.hi[j] - m.lo[j]) : 0.0;
      const double t = m.W[c][j] * xn;
      acc = acc + t;
    }
    s[c] = acc;
    if (c > 0 && s[c] > s[best]) best = c;
  }
  return best;
}

extern "C" goldy_status goldy_predict_cd(const goldy_predictor* m, const goldy_lut* lut, const goldy_gemm_desc* d,
                                         int* cd, double probs[5]) {
  if (!m || !lut || !d || !cd) return fail(GOLDY_ERR_INVALID_ARG, "null argument");
  goldy_status st = check_desc(*d, 0);
  if (st != GOLDY_OK) return st;
  double x[GOLDY_LR_FEATURES], s[5];
  lr_features(*d, lookup(*lut, bucket_key(*d)), m->sm_count, x);
  const int best = lr_predict(*m, x, s);
  *cd = kCdClasses[best];
  if (probs) {   // Eq. 1
    double tot = 0.0;
    for (int c = 0; c < 5; ++c) tot += (probs[c] = std::exp(s[c] - s[best]));
    for (int c = 0; c < 5; ++c) probs[c] /= tot;
  }
  return ok();
}

// ---------------------------------------------------------------------------
// Schedule construction
// ---------------------------------------------------------------------------
namespace goldy {

void finalize_schedule(goldy_schedule* s) {
  size_t off = 0;
  auto align = [](size_t x) { return (x + 255) & ~size_t(255); };
  int max_streams = 1;
  for (auto& g : s->groups) max_streams = std::max(max_streams, g.cd);
  s->max_streams = max_streams;
  for (auto& gp : s->gemms) {
    const Variant v = variant_of(gp.variant);
    const KindInfo& k = kKinds[v.kind];
    gp.kind = v.kind;
    gp.tiles_m = ceil_div(gp.desc.M, tile_rows(k));
    gp.tiles_n = ceil_div(gp.desc.N, tile_cols(k));
    gp.k_blocks = ceil_div(gp.desc.K, kBlockK);
    gp.split = int(std::max<int64_t>(1, std::min<int64_t>(v.split, gp.k_blocks)));
    const int64_t tiles = gp.tiles_m * gp.tiles_n * gp.desc.batch;   // over all batch entries
    gp.units = (gp.desc.K > 0) ? tiles * gp.split : 0;
    gp.ws_part_off = gp.ws_cnt_off = gp.ws_bytes = 0;
    if (gp.split > 1 && tiles > 0) {
      // a partial tile per unit (a CTA pair: one per CTA, 128 rows each) and
      // an arrival counter per tile (per tile half for a pair)
      const size_t halves = k.pair ? 2 : 1;
      gp.ws_part_off = off;
      off = align(off + size_t(gp.units) * halves * kMmaM * k.mma_n * sizeof(float));
      gp.ws_cnt_off = off;
      off = align(off + size_t(tiles) * halves * sizeof(uint32_t));
      gp.ws_bytes = off - gp.ws_part_off;
    }
  }
  // fused schedules of several GEMMs: a pair of unit counters per GEMM (a
  // fused launch uses its first member's); zero like the split-K counters
  if ((s->flags & GOLDY_PLAN_FUSED) && s->gemms.size() > 1) {
    for (size_t i = 0; i < s->gemms.size(); ++i) s->gemms[i].ws_dyn_off = off + 8 * i;
    off = align(off + 8 * s->gemms.size());
  } else {
    for (auto& gp : s->gemms) gp.ws_dyn_off = ~size_t(0);
  }
  s->workspace_bytes = off;
}

}  // namespace goldy

// A wave of a group (its members taken CD at a time, in launch order) that
// mixes kernel kinds runs one launch per kind side by side in the fused
// launch mode, and its smaller launches mostly wait for SMs in the largest
// one's tail.  Under the automatic policy a GEMM of a wave therefore takes
// the kernel kind of the wave's largest GEMM (most FLOPs; ties: the first in
// launch order) — without K split, at that kernel's grid-cap constraint —
// when that kind suits it: the same output dtype, K no longer than the
// largest GEMM's (no longer units than the launch's own), and M within the
// kind's reach (a CTA-pair kind: M >= 128; a transposed skinny-M kind:
// M <= 2 x its tile's rows; the others: M >= 64).  The wave then runs as
// fewer, larger launches.  (This build's rule for its fused launches; the
// paper runs one kernel per GEMM.)
static void one_kind_per_wave(goldy_schedule* s) {
  auto flops = [&](int i) {
    const goldy_gemm_desc& d = s->gemms[i].desc;
    return (unsigned __int128)2 * uint64_t(d.M) * uint64_t(d.N) * uint64_t(d.K) * uint64_t(d.batch);
  };
  for (const Group& grp : s->groups) {
    const size_t size = grp.members.size();
    const size_t cd = size_t(std::max(1, grp.cd));
    for (size_t w0 = 0; w0 < size; w0 += cd) {
      const size_t w1 = std::min(size, w0 + cd);
      int dom = grp.members[w0];
      for (size_t j = w0 + 1; j < w1; ++j)
        if (flops(grp.members[j]) > flops(dom)) dom = grp.members[j];
      const Variant vd = variant_of(s->gemms[dom].variant);
      const KindInfo& kd = kKinds[vd.kind];
      const goldy_gemm_desc& dd = s->gemms[dom].desc;
      for (size_t j = w0; j < w1; ++j) {
        const int i = grp.members[j];
        const goldy_gemm_desc& di = s->gemms[i].desc;
        if (i == dom || variant_of(s->gemms[i].variant).kind == vd.kind) continue;
        if (di.c_dtype != dd.c_dtype || di.K > dd.K) continue;
        const bool fits = kd.pair ? di.M >= 128 : (kd.swap_ab ? di.M <= 2 * kd.mma_n : di.M >= 64);
        if (!fits) continue;
        s->gemms[i].variant = variant_id(vd.kind, 0, vd.id % 3);
      }
    }
  }
}

static goldy_status new_schedule(const goldy_gemm_desc* descs, int n, goldy_schedule** out) {
  if (!descs || !out) return fail(GOLDY_ERR_INVALID_ARG, "null argument");
  *out = nullptr;
  if (n < 1 || n > GOLDY_MAX_GEMMS) return fail(GOLDY_ERR_INVALID_ARG, "number of GEMMs out of range");
  for (int i = 0; i < n; ++i) {
    goldy_status st = check_desc(descs[i], i);
    if (st != GOLDY_OK) return st;
  }
  goldy_schedule* s = new (std::nothrow) goldy_schedule();
  if (!s) return fail(GOLDY_ERR_NOMEM, "out of host memory");
  s->gemms.resize(n);
  for (int i = 0; i < n; ++i) s->gemms[i].desc = descs[i];
  *out = s;
  return GOLDY_OK;
}

extern "C" goldy_status goldy_plan(const goldy_gemm_desc* descs, int n, const goldy_lut* lut,
                                   int flags, goldy_schedule** out) {
  return goldy_plan_ex(descs, n, lut, nullptr, flags, out);
}

extern "C" goldy_status goldy_plan_ex(const goldy_gemm_desc* descs, int n, const goldy_lut* lut,
                                      const goldy_predictor* predictor, int flags, goldy_schedule** out) {
  if (!lut) return fail(GOLDY_ERR_LUT, "no lookup table");
  const int policy = flags & 0xF;
  const int forced = (flags >> 8) & 0xFF;
  if ((flags & ~0xFF1F) != 0 || policy > GOLDY_PLAN_FORCE_CD ||
      (policy == GOLDY_PLAN_FORCE_CD && forced < 1))
    return fail(GOLDY_ERR_INVALID_ARG, "bad flags");
  goldy_schedule* s = nullptr;
  goldy_status st = new_schedule(descs, n, &s);
  if (st != GOLDY_OK) return st;
  s->flags = flags;

  std::vector<uint32_t> keys(n);
  std::vector<const LutEntry*> ent(n);
  std::vector<int> pref(n);
  for (int i = 0; i < n; ++i) {
    keys[i] = bucket_key(descs[i]);
    ent[i] = &lookup(*lut, keys[i]);
    pref[i] = ent[i]->pref_cd;
    if (predictor && policy == GOLDY_PLAN_AUTO) {   // the trained model replaces the table's preference
      double x[GOLDY_LR_FEATURES], sc[5];
      lr_features(descs[i], *ent[i], predictor->sm_count, x);
      pref[i] = kCdClasses[lr_predict(*predictor, x, sc)];
    }
  }

  // (cd, members, class-cd override) triples; class-cd 0 means "use cd"
  struct G {
    int cd;
    std::vector<int> members;
    int class_cd;
  };
  std::vector<G> groups;
  auto all_members = [n]() {
    std::vector<int> m(n);
    for (int i = 0; i < n; ++i) m[i] = i;
    return m;
  };
  auto clamp_cd = [n](int cd) { return std::max(1, std::min({cd, n, GOLDY_MAX_STREAMS})); };

  switch (policy) {
    case GOLDY_PLAN_SEQUENTIAL: groups.push_back({1, all_members(), 1}); break;
    case GOLDY_PLAN_DEFAULT: groups.push_back({clamp_cd(n), all_members(), 1}); break;
    case GOLDY_PLAN_GO: groups.push_back({clamp_cd(n), all_members(), 0}); break;
    case GOLDY_PLAN_FORCE_CD: groups.push_back({clamp_cd(forced), all_members(), 0}); break;
    default: {
      struct Block {
        uint32_t key;
        unsigned __int128 flops;
        std::vector<int> members;
        int pref;
      };
      std::vector<Block> blocks;
      for (int i = 0; i < n; ++i) {
        auto it = std::find_if(blocks.begin(), blocks.end(), [&](const Block& b) { return b.key == keys[i]; });
        const unsigned __int128 f = (unsigned __int128)2 * uint64_t(descs[i].M) * uint64_t(descs[i].N) *
                                    uint64_t(descs[i].K) * uint64_t(descs[i].batch);
        if (it == blocks.end()) {
          blocks.push_back({keys[i], f, {i}, pref[i]});
        } else {
          it->flops += f;
          it->members.push_back(i);
          it->pref = std::min(it->pref, pref[i]);
        }
      }
      std::sort(blocks.begin(), blocks.end(), [](const Block& a, const Block& b) {
        if (a.flops != b.flops) return a.flops > b.flops;
        return a.key < b.key;
      });
      struct Merged {
        std::vector<int> members;
        int min_pref;
        int n_keys;
      };
      std::vector<Merged> merged;
      for (const Block& b : blocks) {
        if (!merged.empty()) {
          Merged& cur = merged.back();
          const int size = int(cur.members.size() + b.members.size());
          const int mp = std::min(cur.min_pref, b.pref);
          if (mp >= size) {
            cur.members.insert(cur.members.end(), b.members.begin(), b.members.end());
            cur.min_pref = mp;
            cur.n_keys += 1;
            continue;
          }
        }
        merged.push_back({b.members, b.pref, 1});
      }
      for (Merged& m : merged) {
        const int size = int(m.members.size());
        int cd = (m.n_keys > 1) ? size : std::min(m.min_pref, size);
        cd = std::max(1, std::min(cd, GOLDY_MAX_STREAMS));
        groups.push_back({cd, m.members, 0});
      }
    }
  }

  s->groups.resize(groups.size());
  for (size_t g = 0; g < groups.size(); ++g) {
    s->groups[g].cd = groups[g].cd;
    s->groups[g].members = groups[g].members;
    const int ci = cd_class_index(groups[g].class_cd ? groups[g].class_cd : groups[g].cd);
    for (size_t j = 0; j < groups[g].members.size(); ++j) {
      const int i = groups[g].members[j];
      s->gemms[i].group = int(g);
      s->gemms[i].variant = ent[i]->variant[ci];
      s->gemms[i].slot = int(j % size_t(groups[g].cd));
    }
  }
  if (policy == GOLDY_PLAN_AUTO) one_kind_per_wave(s);
  finalize_schedule(s);
  *out = s;
  return ok();
}

extern "C" goldy_status goldy_schedule_build(const goldy_gemm_desc* descs, int n, const int* group_of,
                                             const int* variant_of, const int* slot_of, int flags,
                                             goldy_schedule** out) {
  if (!group_of || !variant_of || !slot_of) return fail(GOLDY_ERR_INVALID_ARG, "null argument");
  if ((flags & ~GOLDY_PLAN_FUSED) != 0) return fail(GOLDY_ERR_INVALID_ARG, "bad flags");
  goldy_schedule* s = nullptr;
  goldy_status st = new_schedule(descs, n, &s);
  if (st != GOLDY_OK) return st;
  s->flags = flags;
  int n_groups = 0;
  for (int i = 0; i < n; ++i) {
    if (group_of[i] < 0 || group_of[i] >= n || variant_of[i] < 0 || variant_of[i] >= kNumVariants ||
        slot_of[i] < 0 || slot_of[i] >= GOLDY_MAX_STREAMS) {
      delete s;
      return fail(GOLDY_ERR_INVALID_ARG, "gemm " + std::to_string(i) + ": group, variant or slot out of range");
    }
    n_groups = std::max(n_groups, group_of[i] + 1);
  }
  s->groups.resize(n_groups);
  for (int i = 0; i < n; ++i) {
    s->gemms[i].group = group_of[i];
    s->gemms[i].variant = variant_of[i];
    s->gemms[i].slot = slot_of[i];
    s->groups[group_of[i]].members.push_back(i);
  }
  for (int g = 0; g < n_groups; ++g) {
    if (s->groups[g].members.empty()) {
      delete s;
      return fail(GOLDY_ERR_INVALID_ARG, "group ids must be 0 .. n_groups-1 with none empty");
    }
    uint32_t used = 0;
    for (int i : s->groups[g].members) used |= 1u << s->gemms[i].slot;
    s->groups[g].cd = __builtin_popcount(used);
  }
  finalize_schedule(s);
  // max_streams counts slot ids, which need not be dense in an explicit schedule
  for (auto& gp : s->gemms) s->max_streams = std::max(s->max_streams, gp.slot + 1);
  *out = s;
  return ok();
}

extern "C" goldy_status goldy_schedule_query(const goldy_schedule* s, int* n_gemms, int* n_groups,
                                             int* max_streams, size_t* workspace_bytes) {
  if (!s) return fail(GOLDY_ERR_INVALID_ARG, "null schedule");
  if (n_gemms) *n_gemms = int(s->gemms.size());
  if (n_groups) *n_groups = int(s->groups.size());
  if (max_streams) *max_streams = s->max_streams;
  if (workspace_bytes) *workspace_bytes = s->workspace_bytes;
  return ok();
}

extern "C" goldy_status goldy_schedule_entry(const goldy_schedule* s, int gemm, int* group, int* variant,
                                             int* slot, int* cd) {
  if (!s) return fail(GOLDY_ERR_INVALID_ARG, "null schedule");
  if (gemm < 0 || gemm >= int(s->gemms.size())) return fail(GOLDY_ERR_INVALID_ARG, "gemm index out of range");
  const GemmPlan& gp = s->gemms[gemm];
  if (group) *group = gp.group;
  if (variant) *variant = gp.variant;
  if (slot) *slot = gp.slot;
  if (cd) *cd = s->groups[gp.group].cd;
  return ok();
}

extern "C" goldy_status goldy_schedule_serialize(const goldy_schedule* s, void* buf, size_t cap, size_t* size) {
  if (!s || !size) return fail(GOLDY_ERR_INVALID_ARG, "null argument");
  std::vector<uint32_t> w = {0x48435347u, 1u, uint32_t(s->gemms.size()), uint32_t(s->groups.size()),
                             uint32_t(s->max_streams), uint32_t(s->flags)};
  for (const Group& g : s->groups) {
    w.push_back(uint32_t(g.cd));
    w.push_back(uint32_t(g.members.size()));
    for (int m : g.members) w.push_back(uint32_t(m));
  }
  for (const GemmPlan& gp : s->gemms) {
    w.push_back(uint32_t(gp.group));
    w.push_back(uint32_t(gp.variant));
    w.push_back(uint32_t(gp.slot));
  }
  *size = w.size() * 4;
  if (!buf || cap < *size) return fail(GOLDY_ERR_NOMEM, "buffer too small");
  uint8_t* o = static_cast<uint8_t*>(buf);
  for (size_t i = 0; i < w.size(); ++i)
    for (int b = 0; b < 4; ++b) o[4 * i + b] = uint8_t(w[i] >> (8 * b));
  return ok();
}

extern "C" void goldy_schedule_free(goldy_schedule* s) {
  if (!s) return;
  runtime_release(s->rt);
  delete s;
}

// ---------------------------------------------------------------------------
// Misc
// ---------------------------------------------------------------------------
extern "C" int goldy_abi_version(void) { return GOLDY_ABI_VERSION; }
extern "C" const char* goldy_last_error(void) { return g_last_error.c_str(); }
extern "C" int goldy_variant_count(void) { return kNumVariants; }

extern "C" goldy_status goldy_variant_info_get(int id, goldy_variant_info* out) {
  if (!out || id < 0 || id >= kNumVariants) return fail(GOLDY_ERR_INVALID_ARG, "variant id out of range");
  const Variant v = variant_of(id);
  const KindInfo& k = kKinds[v.kind];
  std::memset(out, 0, sizeof(*out));
  out->id = id;
  out->kind = v.kind;
  out->mma_m = k.pair ? 2 * kMmaM : kMmaM;
  out->mma_n = k.mma_n;
  out->swap_ab = k.swap_ab;
  out->stages = k.stages;
  out->acc_stages = k.acc_stages;
  out->tmem_cols = tmem_cols(k);
  out->smem_bytes = smem_bytes(k);
  out->split_k = v.split;
  out->rc_div = v.rc_div;
  out->ctas_per_sm = k.ctas_per_sm;
  out->cta_pair = k.pair ? 2 : 1;
  std::snprintf(out->name, sizeof(out->name), "%s_s%d_rc%d", k.name, v.split, v.rc_div);
  return ok();
}

// ---------------------------------------------------------------------------
// A GEMM co-scheduled with an element-wise add (Sec. 7.1)
// ---------------------------------------------------------------------------
extern "C" goldy_status goldy_corun_plan(const goldy_gemm_desc* gemm, const goldy_ewise_desc* ew,
                                         const goldy_lut* lut, int policy, goldy_corun** out) {
  if (!gemm || !ew || !out) return fail(GOLDY_ERR_INVALID_ARG, "null argument");
  *out = nullptr;
  if (!lut) return fail(GOLDY_ERR_LUT, "no lookup table");
  if (policy != GOLDY_PLAN_AUTO && policy != GOLDY_PLAN_SEQUENTIAL && policy != GOLDY_PLAN_DEFAULT &&
      policy != GOLDY_PLAN_GO)
    return fail(GOLDY_ERR_INVALID_ARG, "bad policy");
  if (ew->n < 0 || ew->reserved != 0 || (ew->dtype != GOLDY_BF16 && ew->dtype != GOLDY_F32))
    return fail(GOLDY_ERR_INVALID_ARG, "bad element-wise descriptor");
  goldy_status st = check_desc(*gemm, 0);
  if (st != GOLDY_OK) return st;
  const LutEntry& e = lookup(*lut, bucket_key(*gemm));
  bool concurrent = false;
  int variant = e.variant[0], add_rc_div = 1;
  switch (policy) {
    case GOLDY_PLAN_SEQUENTIAL: break;
    case GOLDY_PLAN_DEFAULT: concurrent = true; break;
    case GOLDY_PLAN_GO:
      concurrent = true;
      variant = e.variant[1];
      add_rc_div = 2;
      break;
    default:   // the table's profiled configuration
      if (e.flags & 1u) {
        concurrent = true;
        variant = (e.flags & 2u) ? e.variant[1] : e.variant[0];
        add_rc_div = 1 << ((e.flags >> 2) & 3u);
      }
  }
  const int group = 0, slot = 0;
  goldy_schedule* s = nullptr;
  st = goldy_schedule_build(gemm, 1, &group, &variant, &slot, 0, &s);
  if (st != GOLDY_OK) return st;
  goldy_corun* c = new (std::nothrow) goldy_corun();
  if (!c) {
    goldy_schedule_free(s);
    return fail(GOLDY_ERR_NOMEM, "out of host memory");
  }
  c->gemm = s;
  c->ew = *ew;
  c->policy = policy;
  c->concurrent = concurrent ? 1 : 0;
  c->add_rc_div = add_rc_div;
  *out = c;
  return ok();
}

extern "C" goldy_status goldy_corun_query(const goldy_corun* c, int* concurrent, int* gemm_variant, int* add_rc_div,
                                          size_t* workspace_bytes) {
  if (!c) return fail(GOLDY_ERR_INVALID_ARG, "null argument");
  if (concurrent) *concurrent = c->concurrent;
  if (gemm_variant) *gemm_variant = c->gemm->gemms[0].variant;
  if (add_rc_div) *add_rc_div = c->add_rc_div;
  if (workspace_bytes) *workspace_bytes = c->gemm->workspace_bytes;
  return ok();
}

extern "C" void goldy_corun_free(goldy_corun* c) {
  if (!c) return;
  goldy_schedule_free(c->gemm);
  goldy::runtime_release(c->rt);
  delete c;
}
