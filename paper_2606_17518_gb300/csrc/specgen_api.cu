// C ABI of the fork-decode attention library: argument checks, the host
// planner that turns ragged lengths into a work list, and the launches.
//
// Planning runs on the host from host copies of the lengths, so a call needs
// no device->host copy.  The work list and the per-fork partial-slot map are
// copied into the caller's workspace; the kernels read them from there.
#include <cuda_runtime.h>
#include <math.h>
#include <string.h>

#include <algorithm>
#include <climits>
#include <map>
#include <tuple>
#include <queue>
#include <utility>
#include <vector>

#include "../../include/specgen.h"
#include "append_kv.h"
#include "pack_pages.h"
#include "lse_merge.h"
#include "plan.h"
#include "fork_tc.h"
#include "mla_tc.h"
#include "split_decode.h"
#include "suffix_stage.h"

using namespace specgen;

namespace {

constexpr size_t kAlign = 256;
constexpr size_t kHeaderBytes = 256;  // status word + reserved
constexpr int kTileTokens = 64;       // split-kernel tile; chunk sizes are multiples of it
constexpr int kRowBlock = 16;         // split-kernel rows per item

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

int device_sm_count() {
  static thread_local int cached_dev = -1, cached_sms = 0;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 148;
  if (dev != cached_dev) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
      n = 148;
    cached_dev = dev;
    cached_sms = n;
  }
  return cached_sms;
}

struct Shape {
  int T, F, hq, hkv, G, dqk, dv, B, num_pages;
  bool latent;
};

// Checks of the scalar arguments shared by decode and prefill; fills s (F = the
// query rows, args->total_forks).
specgen_status check_common(const specgen_fork_attn_args* a, Shape* s) {
  if (a->num_traces < 1 || a->total_forks < 1 || a->hq < 1 || a->hkv < 1 || a->page_size < 1 ||
      a->num_pages < 0 || a->head_dim_qk < 1 || a->head_dim_v < 1)
    return SPECGEN_ERR_SHAPE;
  if (a->hq % a->hkv != 0) return SPECGEN_ERR_SHAPE;
  if (!isfinite(a->scale) || !(a->scale > 0.f)) return SPECGEN_ERR_SHAPE;
  const bool latent = a->v_pages == nullptr;
  if (latent && a->head_dim_v > a->head_dim_qk) return SPECGEN_ERR_SHAPE;
  if (!split_variant_supported(a->head_dim_qk, a->head_dim_v, latent))
    return SPECGEN_ERR_UNSUPPORTED;
  if (a->page_size > 1024 || (a->page_size & (a->page_size - 1)) != 0)
    return SPECGEN_ERR_UNSUPPORTED;
  if (a->kv_layout != SPECGEN_KV_ROWS && a->kv_layout != SPECGEN_KV_TILED) return SPECGEN_ERR_SHAPE;
  if (a->kv_layout == SPECGEN_KV_TILED &&
      !fork_tc_supported(a->head_dim_qk, a->head_dim_v, latent, a->page_size, a->hq / a->hkv))
    return SPECGEN_ERR_UNSUPPORTED;
  s->T = a->num_traces;
  s->F = a->total_forks;
  s->hq = a->hq;
  s->hkv = a->hkv;
  s->G = a->hq / a->hkv;
  s->dqk = a->head_dim_qk;
  s->dv = a->head_dim_v;
  s->B = a->page_size;
  s->num_pages = a->num_pages;
  s->latent = latent;
  return SPECGEN_OK;
}

specgen_status check_shape(const specgen_fork_attn_args* a, const specgen_host_lens* lens,
                           Shape* s) {
  if (!a || !lens || !lens->prefix_lens || !lens->fork_offsets || !lens->suffix_lens)
    return SPECGEN_ERR_NULL;
  const specgen_status st = check_common(a, s);
  if (st != SPECGEN_OK) return st;
  const int32_t* fo = lens->fork_offsets;
  if (fo[0] != 0 || fo[a->num_traces] != a->total_forks) return SPECGEN_ERR_SHAPE;
  for (int t = 0; t < a->num_traces; ++t) {
    if (fo[t + 1] < fo[t] || lens->prefix_lens[t] < 0) return SPECGEN_ERR_SHAPE;
  }
  for (int f = 0; f < a->total_forks; ++f)
    if (lens->suffix_lens[f] < 0) return SPECGEN_ERR_SHAPE;
  return SPECGEN_OK;
}

// Prefill: args->total_forks counts query rows (the sum of the chunk lengths);
// the forks themselves are lens->fork_offsets[num_traces].
specgen_status check_prefill(const specgen_fork_attn_args* a, const specgen_prefill_lens* lens,
                             Shape* s) {
  if (!a || !lens || !lens->prefix_lens || !lens->fork_offsets || !lens->suffix_lens ||
      !lens->chunk_lens)
    return SPECGEN_ERR_NULL;
  const specgen_status st = check_common(a, s);
  if (st != SPECGEN_OK) return st;
  if (a->suffix_lens != nullptr) return SPECGEN_ERR_SHAPE;  // device lengths: decode only
  const int32_t* fo = lens->fork_offsets;
  if (fo[0] != 0) return SPECGEN_ERR_SHAPE;
  for (int t = 0; t < a->num_traces; ++t)
    if (fo[t + 1] < fo[t] || lens->prefix_lens[t] < 0) return SPECGEN_ERR_SHAPE;
  long long rows = 0;
  for (int f = 0; f < fo[a->num_traces]; ++f) {
    if (lens->suffix_lens[f] < 0 || lens->chunk_lens[f] < 0) return SPECGEN_ERR_SHAPE;
    if ((long long)lens->suffix_lens[f] + lens->chunk_lens[f] > INT32_MAX) return SPECGEN_ERR_SHAPE;
    rows += lens->chunk_lens[f];
  }
  if (rows != a->total_forks) return SPECGEN_ERR_SHAPE;
  return SPECGEN_OK;
}

specgen_status check_pointers(const specgen_fork_attn_args* a) {
  if (!a->q || !a->k_pages || !a->prefix_block_table || !a->prefix_bt_offsets ||
      !a->suffix_block_table || !a->suffix_bt_offsets || !a->out || !a->lse || !a->workspace)
    return SPECGEN_ERR_NULL;
  if (reinterpret_cast<uintptr_t>(a->workspace) % kAlign != 0) return SPECGEN_ERR_WORKSPACE;
  // queries and pools move in 16-byte pieces and bulk copies
  const void* rows16[3] = {a->q, a->k_pages, a->v_pages};
  for (const void* r : rows16)
    if (reinterpret_cast<uintptr_t>(r) % 16 != 0) return SPECGEN_ERR_SHAPE;
  return SPECGEN_OK;
}

// The host-side plan: work items, their CTA assignment, and the partial-slot map.
struct HostPlan {
  std::vector<SplitItem> split;
  std::vector<TcItem> tc;
  std::vector<int32_t> cta_items, cta_offsets;
  // suffix-stage items in worker order, worker w taking [sfx_offsets[w], [w+1])
  std::vector<TcItem> sfx;
  std::vector<int32_t> sfx_offsets;
  int n_sfx_ctas = 0;
  std::vector<int32_t> part_base;
  std::vector<int32_t> n_parts;  // [forks][n_groups]: partial slots used by each head group
  int n_groups = 1;
  int total_slots = 0;
};

// A shared prefix segment: `len` tokens in prefix table `index` (its token 0 at
// slot 0 of the table's first page), attended to by the query rows
// [row_begin, row_end).  Decode and prefill have one segment per trace; a
// cascade (repeated fork events at growing prefixes) has nested segments.
struct Segment {
  int len, row_begin, row_end;
};

// The query rows a plan serves.  Decode: one row per fork.  Prefill: one row per
// new token of every fork; row j of fork f attends to the fork's first
// S_f + j + 1 suffix tokens (its earlier tokens and, causally, the chunk up to
// itself).  A row reads the suffix table of fork `seq`.
struct Rows {
  std::vector<Segment> segs;
  std::vector<int32_t> seq;                    // [R]
  std::vector<int32_t> len;                    // [R]
  const int32_t* prefix_bt_offsets = nullptr;  // optional host copies of the table offsets
  const int32_t* suffix_bt_offsets = nullptr;
  // Derived by order_segments: enclosing segments before enclosed ones, each
  // segment's enclosing chain (outermost first) and its outermost segment.
  std::vector<int> order, root;
  std::vector<std::vector<int>> anc;
};

// Segment ranges must be laminar (any two nested or disjoint); checked by the
// callers that accept nested segments.
void order_segments(Rows* r) {
  const int n = (int)r->segs.size();
  r->order.resize(n);
  for (int i = 0; i < n; ++i) r->order[i] = i;
  std::stable_sort(r->order.begin(), r->order.end(), [&](int x, int y) {
    const Segment &a = r->segs[x], &b = r->segs[y];
    return a.row_begin < b.row_begin || (a.row_begin == b.row_begin && a.row_end > b.row_end);
  });
  r->root.assign(n, 0);
  r->anc.assign(n, std::vector<int>());
  std::vector<int> stack;
  for (int s : r->order) {
    const Segment& g = r->segs[s];
    while (!stack.empty() && r->segs[stack.back()].row_end <= g.row_begin) stack.pop_back();
    while (!stack.empty() && r->segs[stack.back()].row_end < g.row_end) stack.pop_back();
    r->anc[s] = stack;
    r->root[s] = stack.empty() ? s : stack.front();
    stack.push_back(s);
  }
}

bool laminar(const std::vector<Segment>& segs) {
  for (size_t i = 0; i < segs.size(); ++i)
    for (size_t j = i + 1; j < segs.size(); ++j) {
      const Segment &a = segs[i], &b = segs[j];
      const bool disjoint = a.row_end <= b.row_begin || b.row_end <= a.row_begin;
      const bool nested = (a.row_begin <= b.row_begin && b.row_end <= a.row_end) ||
                          (b.row_begin <= a.row_begin && a.row_end <= b.row_end);
      if (!disjoint && !nested) return false;
    }
  return true;
}

Rows rows_for_decode(const specgen_host_lens* lens, int T, int F) {
  Rows r;
  for (int t = 0; t < T; ++t)
    r.segs.push_back(Segment{lens->prefix_lens[t], lens->fork_offsets[t], lens->fork_offsets[t + 1]});
  r.seq.resize(F);
  r.len.assign(lens->suffix_lens, lens->suffix_lens + F);
  for (int f = 0; f < F; ++f) r.seq[f] = f;
  if (lens->prefix_bt_offsets && lens->suffix_bt_offsets) {
    r.prefix_bt_offsets = lens->prefix_bt_offsets;
    r.suffix_bt_offsets = lens->suffix_bt_offsets;
  }
  order_segments(&r);
  return r;
}

Rows rows_for_prefill(const specgen_prefill_lens* lens, int T) {
  Rows r;
  const int32_t* fo = lens->fork_offsets;
  for (int t = 0; t < T; ++t) {
    const int begin = (int)r.seq.size();
    for (int f = fo[t]; f < fo[t + 1]; ++f)
      for (int j = 0; j < lens->chunk_lens[f]; ++j) {
        r.seq.push_back(f);
        r.len.push_back(lens->suffix_lens[f] + j + 1);  // causal within the chunk
      }
    r.segs.push_back(Segment{lens->prefix_lens[t], begin, (int)r.seq.size()});
  }
  if (lens->prefix_bt_offsets && lens->suffix_bt_offsets) {
    r.prefix_bt_offsets = lens->prefix_bt_offsets;
    r.suffix_bt_offsets = lens->suffix_bt_offsets;
  }
  order_segments(&r);
  return r;
}

specgen_status check_cascade(const specgen_fork_attn_args* a, const specgen_cascade_lens* lens,
                             Shape* s) {
  if (!a || !lens || !lens->segment_lens || !lens->segment_rows || !lens->suffix_lens)
    return SPECGEN_ERR_NULL;
  const specgen_status st = check_common(a, s);
  if (st != SPECGEN_OK) return st;
  if (lens->num_segments != a->num_traces) return SPECGEN_ERR_SHAPE;
  std::vector<Segment> segs;
  for (int i = 0; i < lens->num_segments; ++i) {
    const Segment g{lens->segment_lens[i], lens->segment_rows[2 * i], lens->segment_rows[2 * i + 1]};
    if (g.len < 0 || g.row_begin < 0 || g.row_end < g.row_begin || g.row_end > a->total_forks)
      return SPECGEN_ERR_SHAPE;
    segs.push_back(g);
  }
  if (!laminar(segs)) return SPECGEN_ERR_SHAPE;
  for (int f = 0; f < a->total_forks; ++f)
    if (lens->suffix_lens[f] < 0) return SPECGEN_ERR_SHAPE;
  return SPECGEN_OK;
}

Rows rows_for_cascade(const specgen_cascade_lens* lens, int F) {
  Rows r;
  for (int s = 0; s < lens->num_segments; ++s)
    r.segs.push_back(Segment{lens->segment_lens[s], lens->segment_rows[2 * s],
                             lens->segment_rows[2 * s + 1]});
  r.seq.resize(F);
  r.len.assign(lens->suffix_lens, lens->suffix_lens + F);
  for (int f = 0; f < F; ++f) r.seq[f] = f;
  if (lens->segment_bt_offsets && lens->suffix_bt_offsets) {
    r.prefix_bt_offsets = lens->segment_bt_offsets;
    r.suffix_bt_offsets = lens->suffix_bt_offsets;
  }
  order_segments(&r);
  return r;
}

// Longest-processing-time-first assignment of items to `n_cta` persistent CTAs:
// items in decreasing cost, each to the currently least-loaded CTA.
void assign_lpt(const std::vector<long long>& cost, int n_cta, std::vector<int32_t>* cta_items,
                std::vector<int32_t>* cta_offsets) {
  const int n = (int)cost.size();
  std::vector<int> order(n);
  for (int i = 0; i < n; ++i) order[i] = i;
  std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return cost[a] > cost[b]; });
  typedef std::pair<long long, int> Load;  // (load, cta)
  std::priority_queue<Load, std::vector<Load>, std::greater<Load>> heap;
  for (int c = 0; c < n_cta; ++c) heap.push(Load(0, c));
  std::vector<std::vector<int32_t>> lists(n_cta);
  for (int i : order) {
    Load top = heap.top();
    heap.pop();
    lists[top.second].push_back(i);
    heap.push(Load(top.first + cost[i], top.second));
  }
  cta_items->clear();
  cta_offsets->assign(1, 0);
  for (int c = 0; c < n_cta; ++c) {
    cta_items->insert(cta_items->end(), lists[c].begin(), lists[c].end());
    cta_offsets->push_back((int32_t)cta_items->size());
  }
}

// Assign tensor-core items to CTAs (longest first), store them in CTA order so
// that CTA c walks items [cta_offsets[c], cta_offsets[c+1]), and resolve each
// item's block-table start on the host when the host table offsets are given.
void finish_tc_plan(HostPlan* hp, const std::vector<long long>& cost, int n_sm,
                    const Rows& rows) {
  const int n_cta = (int)std::min<size_t>((size_t)n_sm, hp->tc.size());
  std::vector<int32_t> order;
  assign_lpt(cost, n_cta, &order, &hp->cta_offsets);
  std::vector<TcItem> sorted;
  sorted.reserve(hp->tc.size());
  const bool host_off = rows.prefix_bt_offsets && rows.suffix_bt_offsets;
  for (int32_t i : order) {
    TcItem it = hp->tc[i];
    it.table_off = host_off ? (it.table_kind == 0 ? rows.prefix_bt_offsets[it.seq]
                                                  : rows.suffix_bt_offsets[it.seq])
                            : -1;
    sorted.push_back(it);
  }
  hp->tc.swap(sorted);
  hp->cta_items.clear();
}

// Budget packing of the tensor-core work.  A unit is one kv head of either a
// fork's suffix (cut only when it alone exceeds the budget) or a group of forks'
// shared prefix (cut freely at tile boundaries).  Under a per-CTA budget T, in
// token-equivalents with kItemCost per item, one pass deals the suffix pieces
// (longest first) over the CTAs in snake order, then visits the CTAs from the
// least loaded up and fills each one's spare budget with prefix chunks.  The
// plan takes the smallest budget for which the prefix fits.  An item costs its
// whole tiles: a partial tile takes the pipeline as long as a full one.
constexpr long long kItemCost = 256;  // fixed cost of an item (Q staging, merge, pipeline refill)
static_assert(kItemCost % 128 == 0, "item cost in whole tiles of every tile size");
constexpr int kMinChunk = 128;        // smallest prefix chunk carved into a CTA's spare budget
// Suffix stage (its own kernel beside the prefix CTAs, kSuffixWarps workers per
// CTA): an item's fixed cost in pages (query rows in, partial out), and the
// smallest load in pages worth a worker, which bounds the suffix CTAs of small
// calls.
constexpr long long kSfxItemPages = 3;
constexpr long long kSfxMinWorkerPages = 2;
constexpr long long kSfxMinPiecePages = 2;
constexpr long long kSfxSplitMinPages = 8;  // beside a prefix: the least worker load that pays
// beside a prefix: the largest mean suffix (in pages) for which the split pays;
// longer suffixes stream as well on the tensor-core kernel, which then keeps
// every SM and one kernel less in the chain
constexpr long long kSfxSplitMaxUnitPages = 48;
// weight of a suffix page against a prefix token-page in the SM split (percent)
constexpr long long kSfxWeightPct = 80;

struct TcUnit {
  int kind, seq, g, fork0, nforks, len;
  int row_limit0;  // causal rows (a prefill chunk): row i of the unit sees row_limit0 + i tokens
};

struct TcPlacement {
  int cta;
  TcItem item;
};

// One packing pass under budget T.  `load` and `order` are caller-owned
// scratch; `out` (when given) receives the items with their CTAs.
bool pack_tc(const std::vector<TcUnit>& sfx, const std::vector<TcUnit>& pfx, int n_cta,
             long long T, int tt, std::vector<long long>* load, std::vector<long long>* order,
             std::vector<TcPlacement>* out) {
  load->assign(n_cta, 0);
  if (out) out->clear();
  // tt (64 or 128 tokens) is a power of two: whole tiles by shifts (this runs a
  // few times per plan)
  int sh = 0;
  while ((1 << sh) < tt) ++sh;
  if (T - kItemCost < tt) return false;
  const long long lmax = (T - kItemCost) >> sh << sh;
  auto tiles = [&](long long n) { return (n + tt - 1) >> sh << sh; };  // tokens of whole tiles
  auto place = [&](int cta, const TcUnit& u, int b, int e, int part) {
    (*load)[cta] += tiles(e - b) + kItemCost;
    if (!out) return;
    TcPlacement pl;
    pl.cta = cta;
    TcItem& it = pl.item;
    it.table_kind = u.kind;
    it.seq = u.seq;
    it.kv_head = u.g;
    it.fork0 = u.fork0;
    it.nforks = u.nforks;
    it.tok_begin = b;
    it.tok_end = e;
    it.part = part;
    it.dv0 = 0;
    it.table_off = -1;
    it.row_limit0 = u.row_limit0;
    out->push_back(pl);
  };
  // suffix pieces in snake order over the CTAs: piece i of a round goes to CTA
  // i, or to CTA n_cta - 1 - i in odd rounds
  int i_snake = 0;
  bool odd = false;
  for (const TcUnit& u : sfx) {
    const long long k = (u.len + lmax - 1) / lmax;
    const int piece = (int)tiles((u.len + k - 1) / k);
    for (int c = 0, pos = 0; pos < u.len; ++c, pos += piece) {
      place(odd ? n_cta - 1 - i_snake : i_snake, u, pos, std::min(u.len, pos + piece), c);
      if (++i_snake == n_cta) {
        i_snake = 0;
        odd = !odd;
      }
    }
  }
  // CTAs from the least loaded up (ties by index): a stable counting sort of
  // the loads, which are whole tiles (tiles and kItemCost are multiples of tt)
  static thread_local std::vector<int> count;
  long long most = 0;
  for (int c = 0; c < n_cta; ++c) most = std::max(most, (*load)[c]);
  count.assign((size_t)(most >> sh) + 2, 0);
  for (int c = 0; c < n_cta; ++c) ++count[(size_t)((*load)[c] >> sh) + 1];
  for (size_t b = 1; b < count.size(); ++b) count[b] += count[b - 1];
  order->resize(n_cta);
  for (int c = 0; c < n_cta; ++c) (*order)[count[(size_t)((*load)[c] >> sh)]++] = c;
  size_t ui = 0;
  int pos = 0, part = 0;
  for (int oc = 0; oc < n_cta && ui < pfx.size(); ++oc) {
    const int cta = (int)(*order)[oc];
    while (ui < pfx.size()) {
      const TcUnit& u = pfx[ui];
      const int rem = u.len - pos;
      const long long room = T - (*load)[cta] - kItemCost;
      if (room < std::min(kMinChunk, rem)) break;  // this CTA is full
      const long long spare = room >> sh << sh;
      if (spare < std::min(kMinChunk, rem)) break;
      long long len = std::min<long long>(rem, spare);
      if (rem - len < kMinChunk / 2) len = rem;  // leave no sliver behind
      place(cta, u, pos, pos + (int)len, part);
      pos += (int)len;
      ++part;
      if (pos == u.len) {
        ++ui;
        pos = 0;
        part = 0;
      }
    }
  }
  return ui == pfx.size();
}

// The suffix units over n_workers suffix-stage workers (cta = -1 - worker), in
// one pass.  Every unit is laid on a ribbon as its item cost (kSfxItemPages)
// followed by its pages, the units end to end; the ribbon of length T is cut
// into n_workers runs of equal length (worker w takes positions
// [T w / n, T (w+1) / n)), so the loads differ by at most a page or two.  A
// unit is cut at page boundaries where a run ends, and no piece is shorter
// than kSfxMinPiecePages unless its unit is.
void place_suffix_stage(const std::vector<TcUnit>& units, int n_workers, int page,
                        std::vector<TcPlacement>* placed) {
  // in row order (fork, then kv head): every run then holds suffixes of mixed
  // lengths, and no worker is left with all the short ones (whose item costs
  // are real time on the GPU)
  static thread_local std::vector<TcUnit> sfx;
  sfx.assign(units.begin(), units.end());
  std::sort(sfx.begin(), sfx.end(), [](const TcUnit& a, const TcUnit& b) {
    return a.fork0 < b.fork0 || (a.fork0 == b.fork0 && a.g < b.g);
  });
  auto pages = [&](long long n) { return (n + page - 1) / page; };
  long long T = 0;
  for (const TcUnit& u : sfx) T += kSfxItemPages + pages(u.len);
  auto bound = [&](long long w) { return T * w / n_workers; };  // first position of run w
  long long g = 0;  // position on the ribbon
  int w = 0;        // the worker whose run holds g
  for (const TcUnit& u : sfx) {
    const long long p0 = g + kSfxItemPages, end = p0 + pages(u.len);  // the unit's pages
    int part = 0;
    while (g < end) {
      while (w + 1 < n_workers && bound(w + 1) <= g) ++w;
      long long stop = std::min(end, w + 1 < n_workers ? bound(w + 1) : end);
      // no piece shorter than kSfxMinPiecePages (or the rest of the unit), and
      // no shorter remainder left behind at the unit's end
      stop = std::max(stop, std::min(end, std::max(g, p0) + kSfxMinPiecePages));
      if (end - stop < kSfxMinPiecePages) stop = end;
      TcPlacement pl;
      pl.cta = -1 - w;
      TcItem& it = pl.item;
      it.table_kind = 1;
      it.seq = u.seq;
      it.kv_head = u.g;
      it.fork0 = u.fork0;
      it.nforks = 1;
      it.tok_begin = (int)((std::max(g, p0) - p0) * page);
      it.tok_end = (int)std::min<long long>(u.len, (stop - p0) * page);
      it.part = part++;
      it.dv0 = 0;
      it.table_off = -1;
      it.row_limit0 = 0;
      placed->push_back(pl);
      g = stop;
    }
  }
}

void build_tc_plan(const Shape& s, const Rows& rows, int n_sm, HostPlan* hp) {
  const int tt = fork_tc_tile_tokens(s.dqk);
  const int forks_per_item = std::max(1, 128 / s.G);
  const int R = (int)rows.seq.size();
  // Prefix units: the rows of a segment in groups of forks_per_item, on the grid
  // of its outermost enclosing segment, so that every row of a group sees the
  // same groups (and chunk counts) in the segments that enclose this one.
  auto group_of = [&](int seg, int f) {
    return (f - rows.segs[rows.root[seg]].row_begin) / forks_per_item;
  };
  // scratch kept across calls (planning runs on every decode call)
  static thread_local std::vector<TcUnit> sfx, pfx, unit_tmp;
  static thread_local std::vector<uint64_t> unit_keys;
  static thread_local std::vector<int> group_id;
  static thread_local std::vector<TcPlacement> placed, trial;
  sfx.clear();
  pfx.clear();
  long long total = 0;
  for (int sg = 0; sg < (int)rows.segs.size(); ++sg) {
    const Segment& seg = rows.segs[sg];
    if (seg.len <= 0) continue;
    const int r0 = rows.segs[rows.root[sg]].row_begin;
    for (int g = 0; g < s.hkv; ++g)
      for (int f0 = seg.row_begin; f0 < seg.row_end;) {
        const int f1 = std::min(seg.row_end, r0 + (group_of(sg, f0) + 1) * forks_per_item);
        pfx.push_back(TcUnit{0, sg, g, f0, f1 - f0, seg.len, 0});
        f0 = f1;
      }
  }
  // Suffix units: a row's own suffix, or -- for consecutive rows of one fork whose
  // lengths grow by one (the tokens of a prefill chunk, causal) -- one unit for up
  // to forks_per_item of them inside one prefix row group: the fork's suffix
  // pages are then read once for the whole group, each row masked at its own
  // length.
  group_id.assign(R, -1);  // prefix row group of each row
  for (int sg = 0; sg < (int)rows.segs.size(); ++sg)
    if (rows.root[sg] == sg)
      for (int f = rows.segs[sg].row_begin; f < rows.segs[sg].row_end; ++f)
        group_id[f] = sg * (R / forks_per_item + 2) + group_of(sg, f);
  for (int g = 0; g < s.hkv; ++g)
    for (int f = 0; f < R;) {
      int f1 = f + 1;
      while (f1 < R && f1 - f < forks_per_item && rows.seq[f1] == rows.seq[f] &&
             rows.len[f1] == rows.len[f1 - 1] + 1 && group_id[f1] == group_id[f] &&
             group_id[f] >= 0)
        ++f1;
      if (rows.len[f1 - 1] > 0)
        sfx.push_back(TcUnit{1, rows.seq[f], g, f, f1 - f, rows.len[f1 - 1],
                             f1 - f > 1 ? rows.len[f] : 0});
      f = f1;
    }
  // The suffix stage takes the suffix units when each serves one query row
  // (decode and cascade; prefill only when no chunk shares an item) and the
  // group fits its n-tiles.  The grid is then split between the prefix CTAs
  // and the suffix-stage CTAs in proportion to their work.
  bool use_sfx = !sfx.empty() && suffix_stage_supported(s.dqk, s.dv, s.latent, s.B, s.G);
  for (const TcUnit& u : sfx) use_sfx = use_sfx && u.nforks == 1 && u.row_limit0 == 0;
  int n_sfx_sm = 0;
  if (use_sfx) {
    const int pg = fork_tc_page_size();
    long long ws = 0, wp = 0, sfx_pages = 0;
    for (const TcUnit& u : sfx) {
      sfx_pages += (u.len + pg - 1) / pg;
      ws += ((u.len + pg - 1) / pg + kSfxItemPages) * pg;
    }
    for (const TcUnit& u : pfx) wp += (u.len + tt - 1) / tt * tt + kItemCost;
    const int n_all = std::max(1, n_sm);
    constexpr long long kWorkersPerSm = kSuffixWarps * kSuffixCtasPerSm;
    const long long most = std::max<long long>(
        1, (sfx_pages + kWorkersPerSm * kSfxMinWorkerPages - 1) / (kWorkersPerSm * kSfxMinWorkerPages));
    if (wp == 0) {
      n_sfx_sm = (int)std::min<long long>(n_all, most);
    } else if (n_all < 2) {
      use_sfx = false;
    } else {
      const double wsw = (double)ws * kSfxWeightPct / 100.0;
      long long n = (long long)llround((double)n_all * wsw / (wsw + (double)wp));
      n = std::max<long long>(1, std::min<long long>(std::min<long long>(n, n_all - 1), most));
      n_sfx_sm = (int)n;
      // a kernel of its own pays (one more launch in the chain, more partials to
      // merge) only when each worker streams enough pages
      if (sfx_pages < n * kWorkersPerSm * kSfxSplitMinPages ||
          sfx_pages > (long long)sfx.size() * kSfxSplitMaxUnitPages) {
        use_sfx = false;
        n_sfx_sm = 0;
      }
    }
  }
  static thread_local std::vector<TcUnit> no_units;
  std::vector<TcUnit>& tc_sfx = use_sfx ? no_units : sfx;
  for (const TcUnit& u : tc_sfx) total += (u.len + tt - 1) / tt * tt;
  for (const TcUnit& u : pfx) total += u.len;
  // longest first, ties in their present order (a sort of (length, index) keys)
  auto longest_first = [](std::vector<TcUnit>& v) {
    unit_keys.resize(v.size());
    for (size_t i = 0; i < v.size(); ++i)
      unit_keys[i] = ((uint64_t)(0x7fffffff - v[i].len) << 32) | (uint64_t)i;
    std::sort(unit_keys.begin(), unit_keys.end());
    unit_tmp.resize(v.size());
    for (size_t i = 0; i < v.size(); ++i) unit_tmp[i] = v[unit_keys[i] & 0xffffffffu];
    v.swap(unit_tmp);
  };
  longest_first(sfx);
  longest_first(pfx);
  placed.clear();
  const int n_units = (int)(tc_sfx.size() + pfx.size());
  const int n_cta = std::max(1, n_sm - n_sfx_sm);
  if (n_units > 0) {
    // Budget search.  Loads and item costs are whole tiles, so feasibility only
    // changes at multiples of the tile: search the budget in tiles.  Start
    // from the average load with one item per suffix unit and about one prefix
    // chunk per CTA, step up by 1/16 until the packing fits, then bisect the
    // last step (a few linear passes in all).
    // Every pass records its placements; `placed` keeps those of the pass that
    // last fitted, which is the one at the final budget.
    static thread_local std::vector<long long> load, order;
    const long long n_items = (long long)tc_sfx.size() + std::max<long long>((long long)pfx.size(), n_cta);
    long long lo = std::max<long long>(kItemCost + tt, (total + kItemCost * n_items) / n_cta) / tt;
    long long hi = lo;
    while (!pack_tc(tc_sfx, pfx, n_cta, hi * tt, tt, &load, &order, &trial)) {
      lo = hi;
      hi += std::max<long long>(1, hi / 16);
    }
    placed.swap(trial);
    while (hi - lo > 1) {
      const long long mid = (lo + hi) / 2;
      if (pack_tc(tc_sfx, pfx, n_cta, mid * tt, tt, &load, &order, &trial)) {
        hi = mid;
        placed.swap(trial);
      } else {
        lo = mid;
      }
    }
  }
  // the suffix-stage grid has kSuffixCtasPerSm CTAs on each of its n_sfx_sm SMs
  if (use_sfx)
    place_suffix_stage(sfx, n_sfx_sm * kSuffixCtasPerSm * kSuffixWarps, fork_tc_page_size(),
                       &placed);
  // Partial slots: per (row, head group) the prefix chunks come first (segment
  // by segment, enclosing segments first), then the suffix pieces; a row owns
  // as many slots as its busiest head group.  A prefix chunk's part is the
  // chunk index plus the chunks of the enclosing segments' same-row groups.
  hp->n_groups = s.hkv;
  hp->n_parts.assign((size_t)s.F * s.hkv, 0);
  const int n_grp = (R + forks_per_item - 1) / forks_per_item;
  static thread_local std::vector<int> chunks, per_cta, next;
  static thread_local std::vector<int32_t> n_pre, n_suf;
  static thread_local std::vector<TcItem> by_cta;
  chunks.assign(rows.segs.size() * s.hkv * std::max(1, n_grp), 0);  // (segment, head, group)
  auto chunk_at = [&](int seg, int g, int grp) -> int& {
    return chunks[((size_t)seg * s.hkv + g) * std::max(1, n_grp) + grp];
  };
  n_pre.assign((size_t)s.F * s.hkv, 0);
  n_suf.assign((size_t)s.F * s.hkv, 0);
  for (const TcPlacement& pl : placed) {
    const TcItem& it = pl.item;
    if (it.table_kind == 0) {
      int& c = chunk_at(it.seq, it.kv_head, group_of(it.seq, it.fork0));
      c = std::max(c, it.part + 1);
    } else {
      for (int f = it.fork0; f < it.fork0 + it.nforks; ++f) {
        int32_t& n = n_suf[(size_t)f * s.hkv + it.kv_head];
        n = std::max(n, it.part + 1);
      }
    }
  }
  auto base_of = [&](int seg, int g, int f) {  // chunks of the enclosing segments for row f
    int b = 0;
    for (int a : rows.anc[seg]) b += chunk_at(a, g, group_of(a, f));
    return b;
  };
  for (const TcUnit& u : pfx) {
    const int c = chunk_at(u.seq, u.g, group_of(u.seq, u.fork0));
    for (int f = u.fork0; f < u.fork0 + u.nforks; ++f) n_pre[(size_t)f * s.hkv + u.g] += c;
  }
  int slot = 0;
  for (int f = 0; f < s.F; ++f) {
    int most = 0;
    for (int g = 0; g < s.hkv; ++g) {
      const size_t i = (size_t)f * s.hkv + g;
      hp->n_parts[i] = n_pre[i] + n_suf[i];
      most = std::max(most, hp->n_parts[i]);
    }
    hp->part_base[f] = slot;
    slot += most;
  }
  hp->total_slots = slot;
  // items in CTA order (empty CTAs dropped), suffix parts after the prefix ones,
  // block-table starts resolved on the host when the host offsets are given
  const bool host_off = rows.prefix_bt_offsets && rows.suffix_bt_offsets;
  hp->tc.clear();
  hp->cta_offsets.assign(1, 0);
  // lists 0 .. n_cta-1: the prefix CTAs; then one per suffix-stage worker
  const int n_workers = n_sfx_sm * kSuffixCtasPerSm * kSuffixWarps;
  const int n_lists = n_cta + n_workers;
  auto list_of = [&](const TcPlacement& pl) { return pl.cta >= 0 ? pl.cta : n_cta + (-1 - pl.cta); };
  per_cta.assign(n_lists + 1, 0);  // counting sort of the placements by list
  for (const TcPlacement& pl : placed) ++per_cta[list_of(pl) + 1];
  for (int c = 0; c < n_lists; ++c) per_cta[c + 1] += per_cta[c];
  by_cta.resize(placed.size());
  next.assign(per_cta.begin(), per_cta.end() - 1);
  for (const TcPlacement& pl : placed) by_cta[next[list_of(pl)]++] = pl.item;
  auto finish = [&](TcItem it) {
    if (it.table_kind == 1)
      it.part += n_pre[(size_t)it.fork0 * s.hkv + it.kv_head];
    else
      it.part += base_of(it.seq, it.kv_head, it.fork0);
    it.table_off = host_off ? (it.table_kind == 0 ? rows.prefix_bt_offsets[it.seq]
                                                  : rows.suffix_bt_offsets[it.seq])
                            : -1;
    return it;
  };
  for (int c = 0; c < n_cta; ++c) {
    if (per_cta[c + 1] == per_cta[c]) continue;  // empty CTAs are dropped
    for (int i = per_cta[c]; i < per_cta[c + 1]; ++i) hp->tc.push_back(finish(by_cta[i]));
    hp->cta_offsets.push_back((int32_t)hp->tc.size());
  }
  // every worker keeps its place (worker w is warp w % kSuffixWarps of CTA
  // w / kSuffixWarps), empty or not
  hp->sfx.clear();
  hp->sfx_offsets.assign(1, 0);
  for (int w = 0; w < n_workers; ++w) {
    for (int i = per_cta[n_cta + w]; i < per_cta[n_cta + w + 1]; ++i)
      hp->sfx.push_back(finish(by_cta[i]));
    hp->sfx_offsets.push_back((int32_t)hp->sfx.size());
  }
  hp->n_sfx_ctas = n_sfx_sm * kSuffixCtasPerSm;
  hp->cta_items.clear();
}

void build_plan(const Shape& s, const Rows& rows, HostPlan* hp) {
  const int n_sm = device_sm_count();
  const bool tc = fork_tc_supported(s.dqk, s.dv, s.latent, s.B, s.G);
  const int R = (int)rows.seq.size();
  hp->split.clear();
  hp->tc.clear();
  hp->sfx.clear();
  hp->sfx_offsets.assign(1, 0);
  hp->n_sfx_ctas = 0;
  hp->cta_items.clear();
  hp->cta_offsets.assign(1, 0);
  hp->part_base.assign(s.F, 0);
  hp->n_parts.assign(s.F, 0);
  hp->n_groups = 1;
  int slot = 0;

  if (tc) {
    build_tc_plan(s, rows, n_sm, hp);
    return;
  }

  // The non-tensor-core planners give every row its own items: the segments
  // that serve a row (enclosing ones first), then its suffix.
  std::vector<std::vector<int>> serving(R);
  for (int sg : rows.order)
    if (rows.segs[sg].len > 0)
      for (int f = rows.segs[sg].row_begin; f < rows.segs[sg].row_end; ++f) serving[f].push_back(sg);

  if (mla_tc_supported(s.dqk, s.dv, s.latent, s.B, s.hq, s.hkv)) {
    // Latent-KV tensor-core path: one item = one row's 128 heads x one value
    // half x a chunk of a prefix segment or of its suffix; chunks are whole tiles.
    const int tt = mla_tc_tile_tokens();
    long long work = 0;
    for (int f = 0; f < R; ++f) {
      long long keys = rows.len[f];
      for (int sg : serving[f]) keys += rows.segs[sg].len;
      work += 2LL * keys;
    }
    const long long item_overhead = 128;
    // Chunk length: near work / n_sm, chosen among whole-tile lengths for the
    // smallest longest-CTA load under the longest-first assignment (one CTA
    // with a second item would otherwise set the kernel's end).
    // Longest-first assignment of every item cost (two per chunk, one per value
    // half) to n_sm CTAs; its largest load.  All whole chunks cost the same and
    // are the longest items, so they come first and leave the loads at q or q + 1
    // times their cost; only the shorter last chunks of the sequences go through
    // the heap.
    static thread_local std::vector<long long> costs, heap;
    const int m = std::max(1, n_sm);
    // `bound`: a candidate whose lower bound (the largest item, or the average
    // CTA load) already exceeds it cannot be chosen, and is not simulated
    auto makespan = [&](long long c, long long bound) {
      const long long full = c + item_overhead;  // c is whole tiles
      long long n_full = 0;
      costs.clear();
      auto add = [&](long long len) {
        n_full += 2 * (len / c);
        const long long rest = len % c;
        if (rest > 0) {
          const long long n = (rest + tt - 1) / tt * tt + item_overhead;
          costs.push_back(n);
          costs.push_back(n);
        }
      };
      for (int f = 0; f < R; ++f) {
        add(rows.len[f]);
        for (int sg : serving[f]) add(rows.segs[sg].len);
      }
      long long total = n_full * full, largest = n_full > 0 ? full : 0;
      for (long long x : costs) {
        total += x;
        largest = std::max(largest, x);
      }
      const long long lower = std::max(largest, (total + m - 1) / m);
      if (lower > bound) return lower;
      std::sort(costs.begin(), costs.end(), std::greater<long long>());
      const long long q = n_full / m, r = n_full % m;
      heap.assign(m, q * full);
      for (long long i = 0; i < r; ++i) heap[i] += full;
      std::make_heap(heap.begin(), heap.end(), std::greater<long long>());
      long long worst = (r > 0 ? q + 1 : q) * full;
      for (long long x : costs) {
        std::pop_heap(heap.begin(), heap.end(), std::greater<long long>());
        heap.back() += x;
        worst = std::max(worst, heap.back());
        std::push_heap(heap.begin(), heap.end(), std::greater<long long>());
      }
      return worst;
    };
    const long long c0 = std::max<long long>(4 * tt, ((work + n_sm - 1) / std::max(1, n_sm) + tt - 1) / tt * tt);
    // candidates: every whole-tile length between half and one and a half
    // times the average, and the lengths at which a prefix segment's chunk
    // count changes in that range
    std::vector<long long> cand;
    for (long long c = std::max<long long>(4 * tt, c0 / 2 / tt * tt); c <= c0 * 3 / 2; c += tt)
      cand.push_back(c);
    for (const Segment& sg : rows.segs) {
      if (sg.len <= 0) continue;
      const long long k0 = std::max<long long>(1, (sg.len + c0 * 3 / 2 - 1) / (c0 * 3 / 2));
      for (long long k = k0; k <= k0 + 16; ++k) {
        const long long c = ((sg.len + k - 1) / k + tt - 1) / tt * tt;
        if (c < std::max<long long>(4 * tt, c0 / 2)) break;
        cand.push_back(c);
      }
    }
    std::sort(cand.begin(), cand.end());
    cand.erase(std::unique(cand.begin(), cand.end()), cand.end());
    long long chunk = c0, best = makespan(c0, LLONG_MAX);
    for (long long c : cand) {
      const long long m = makespan(c, best);
      if (m < best || (m == best && c > chunk)) {
        best = m;
        chunk = c;
      }
    }
    std::vector<long long> cost;
    auto emit = [&](int kind, int seq, int f, int len, int part0) {
      const int n = (int)((len + chunk - 1) / chunk);
      for (int c = 0; c < n; ++c)
        for (int half = 0; half < 2; ++half) {
          TcItem it;
          it.table_kind = kind;
          it.seq = seq;
          it.kv_head = 0;
          it.fork0 = f;
          it.nforks = 1;
          it.tok_begin = (int)(c * chunk);
          it.tok_end = (int)std::min<long long>(len, (c + 1) * chunk);
          it.part = part0 + c;
          it.dv0 = half * 256;
          it.row_limit0 = 0;
          hp->tc.push_back(it);
          cost.push_back(it.tok_end - it.tok_begin + item_overhead);
        }
      return n;
    };
    for (int f = 0; f < R; ++f) {
      int parts = 0;
      for (int sg : serving[f]) parts += emit(0, sg, f, rows.segs[sg].len, parts);
      parts += emit(1, rows.seq[f], f, rows.len[f], parts);
      hp->part_base[f] = slot;
      hp->n_parts[f] = parts;
      slot += parts;
    }
    finish_tc_plan(hp, cost, n_sm, rows);
    hp->total_slots = slot;
    return;
  }

  // Split-K path (shapes the tensor-core kernels do not cover): every row reads
  // its prefix segments and its own suffix in chunks of whole tiles.
  const int dvt = split_dv_tile(s.dqk, s.dv, s.latent);
  const int row_blocks = (s.G + kRowBlock - 1) / kRowBlock;
  const int dv_blocks = s.dv / dvt;
  const long long units = (long long)s.hkv * row_blocks * dv_blocks;
  long long split_tokens = 0;
  for (int f = 0; f < R; ++f) {
    split_tokens += rows.len[f];
    for (int sg : serving[f]) split_tokens += rows.segs[sg].len;
  }
  const long long target_items = (long long)n_sm * 4;
  long long chunk = (split_tokens * units + target_items - 1) / std::max(1LL, target_items);
  chunk = std::max<long long>(kTileTokens, (chunk + kTileTokens - 1) / kTileTokens * kTileTokens);
  chunk = std::min<long long>(chunk, 1 << 20);
  for (int f = 0; f < R; ++f) {
    // (kind, table, length) of every key range of this row, in slot order
    std::vector<std::tuple<int, int, int>> ranges;
    for (int sg : serving[f]) ranges.push_back(std::make_tuple(0, sg, rows.segs[sg].len));
    ranges.push_back(std::make_tuple(1, (int)rows.seq[f], (int)rows.len[f]));
    int parts = 0;
    for (auto& r : ranges) parts += (int)((std::get<2>(r) + chunk - 1) / chunk);
    hp->part_base[f] = slot;
    hp->n_parts[f] = parts;
    for (int g = 0; g < s.hkv; ++g)
      for (int rb = 0; rb < row_blocks; ++rb)
        for (int db = 0; db < dv_blocks; ++db) {
          SplitItem it;
          it.fork = f;
          it.kv_head = g;
          it.h0 = g * s.G + rb * kRowBlock;
          it.nrows = std::min(kRowBlock, s.G - rb * kRowBlock);
          it.dv0 = db * dvt;
          int part = 0;
          for (auto& r : ranges) {
            const int len = std::get<2>(r);
            for (long long c = 0; c * chunk < len; ++c, ++part) {
              it.table_kind = std::get<0>(r);
              it.seq = std::get<1>(r);
              it.tok_begin = (int)(c * chunk);
              it.tok_end = (int)std::min<long long>(len, (c + 1) * chunk);
              it.slot = slot + part;
              hp->split.push_back(it);
            }
          }
        }
    slot += parts;
  }
  hp->total_slots = slot;
}

struct Layout {
  size_t split_off, tc_off, cta_items_off, cta_offsets_off, part_base_off, n_parts_off, plan_bytes;
  size_t sfx_off, sfx_offsets_off;
  size_t ws_plan, ws_part_o, ws_part_lse, ws_end;
};

Layout layout_of(const Shape& s, const HostPlan& hp) {
  Layout L;
  L.split_off = align_up(sizeof(PlanHeader), 16);
  L.tc_off = align_up(L.split_off + hp.split.size() * sizeof(SplitItem), 16);
  L.cta_items_off = align_up(L.tc_off + hp.tc.size() * sizeof(TcItem), 16);
  L.cta_offsets_off = align_up(L.cta_items_off + hp.cta_items.size() * 4, 16);
  L.sfx_off = align_up(L.cta_offsets_off + hp.cta_offsets.size() * 4, 16);
  L.sfx_offsets_off = align_up(L.sfx_off + hp.sfx.size() * sizeof(TcItem), 16);
  L.part_base_off = align_up(L.sfx_offsets_off + hp.sfx_offsets.size() * 4, 16);
  L.n_parts_off = align_up(L.part_base_off + (size_t)s.F * 4, 16);
  L.plan_bytes = L.n_parts_off + hp.n_parts.size() * 4;
  L.ws_plan = kHeaderBytes;
  L.ws_part_o = align_up(L.ws_plan + L.plan_bytes, kAlign);
  L.ws_part_lse =
      align_up(L.ws_part_o + (size_t)hp.total_slots * s.hq * s.dv * sizeof(float), kAlign);
  L.ws_end = align_up(L.ws_part_lse + (size_t)hp.total_slots * s.hq * sizeof(float), kAlign);
  return L;
}

thread_local HostPlan t_plan;
thread_local std::vector<unsigned char> t_plan_bytes;


// Plans one call on the host: the plan region (zeroed header, then the work
// list) into t_plan_bytes and the launch shapes into *plan.  No CUDA call;
// SPECGEN_ERR_WORKSPACE when args->workspace_bytes is below what the call needs.
specgen_status plan_build(const specgen_fork_attn_args* args, const Shape& s, const Rows& rows,
                          specgen_plan* plan);

// plan_build, then: host_dst == nullptr uploads the plan region to the workspace
// on cuda_stream (from this thread's page-locked ring when `pinned`, else from
// the pageable buffer); otherwise it is copied into host_dst (host_bytes long)
// and no CUDA call is made.
specgen_status plan_impl(const specgen_fork_attn_args* args, const Shape& s, const Rows& rows,
                         specgen_plan* plan, void* cuda_stream, void* host_dst = nullptr,
                         size_t host_bytes = 0, bool pinned = false);

}  // namespace

extern "C" {

size_t specgen_fork_attn_workspace_size(const specgen_fork_attn_args* args,
                                        const specgen_host_lens* lens) {
  Shape s;
  if (check_shape(args, lens, &s) != SPECGEN_OK) return 0;
  HostPlan hp;
  build_plan(s, rows_for_decode(lens, s.T, s.F), &hp);
  return layout_of(s, hp).ws_end;
}

specgen_status specgen_fork_attn_plan(const specgen_fork_attn_args* args,
                                      const specgen_host_lens* lens, specgen_plan* plan,
                                      void* cuda_stream) {
  if (!plan) return SPECGEN_ERR_NULL;
  memset(plan, 0, sizeof(*plan));
  Shape s;
  specgen_status st = check_shape(args, lens, &s);
  if (st != SPECGEN_OK) return st;
  return plan_impl(args, s, rows_for_decode(lens, s.T, s.F), plan, cuda_stream);
}

specgen_status specgen_fork_attn_plan_host(const specgen_fork_attn_args* args,
                                           const specgen_host_lens* lens, void* host_dst,
                                           size_t host_bytes, specgen_plan* plan) {
  if (!plan || !host_dst) return SPECGEN_ERR_NULL;
  memset(plan, 0, sizeof(*plan));
  Shape s;
  specgen_status st = check_shape(args, lens, &s);
  if (st != SPECGEN_OK) return st;
  return plan_impl(args, s, rows_for_decode(lens, s.T, s.F), plan, nullptr, host_dst, host_bytes);
}

size_t specgen_fork_cascade_workspace_size(const specgen_fork_attn_args* args,
                                           const specgen_cascade_lens* lens) {
  Shape s;
  if (check_cascade(args, lens, &s) != SPECGEN_OK) return 0;
  HostPlan hp;
  build_plan(s, rows_for_cascade(lens, s.F), &hp);
  return layout_of(s, hp).ws_end;
}

specgen_status specgen_fork_cascade_plan(const specgen_fork_attn_args* args,
                                         const specgen_cascade_lens* lens, specgen_plan* plan,
                                         void* cuda_stream) {
  if (!plan) return SPECGEN_ERR_NULL;
  memset(plan, 0, sizeof(*plan));
  Shape s;
  specgen_status st = check_cascade(args, lens, &s);
  if (st != SPECGEN_OK) return st;
  return plan_impl(args, s, rows_for_cascade(lens, s.F), plan, cuda_stream);
}

specgen_status specgen_fork_cascade_plan_host(const specgen_fork_attn_args* args,
                                              const specgen_cascade_lens* lens, void* host_dst,
                                              size_t host_bytes, specgen_plan* plan) {
  if (!plan || !host_dst) return SPECGEN_ERR_NULL;
  memset(plan, 0, sizeof(*plan));
  Shape s;
  specgen_status st = check_cascade(args, lens, &s);
  if (st != SPECGEN_OK) return st;
  return plan_impl(args, s, rows_for_cascade(lens, s.F), plan, nullptr, host_dst, host_bytes);
}

size_t specgen_fork_prefill_workspace_size(const specgen_fork_attn_args* args,
                                           const specgen_prefill_lens* lens) {
  Shape s;
  if (check_prefill(args, lens, &s) != SPECGEN_OK) return 0;
  HostPlan hp;
  build_plan(s, rows_for_prefill(lens, s.T), &hp);
  return layout_of(s, hp).ws_end;
}

specgen_status specgen_fork_prefill_plan(const specgen_fork_attn_args* args,
                                         const specgen_prefill_lens* lens, specgen_plan* plan,
                                         void* cuda_stream) {
  if (!plan) return SPECGEN_ERR_NULL;
  memset(plan, 0, sizeof(*plan));
  Shape s;
  specgen_status st = check_prefill(args, lens, &s);
  if (st != SPECGEN_OK) return st;
  return plan_impl(args, s, rows_for_prefill(lens, s.T), plan, cuda_stream);
}

specgen_status specgen_fork_prefill_plan_host(const specgen_fork_attn_args* args,
                                              const specgen_prefill_lens* lens, void* host_dst,
                                              size_t host_bytes, specgen_plan* plan) {
  if (!plan || !host_dst) return SPECGEN_ERR_NULL;
  memset(plan, 0, sizeof(*plan));
  Shape s;
  specgen_status st = check_prefill(args, lens, &s);
  if (st != SPECGEN_OK) return st;
  return plan_impl(args, s, rows_for_prefill(lens, s.T), plan, nullptr, host_dst, host_bytes);
}

}  // extern "C"

namespace {

specgen_status plan_build(const specgen_fork_attn_args* args, const Shape& s, const Rows& rows,
                          specgen_plan* plan) {
  build_plan(s, rows, &t_plan);
  const Layout L = layout_of(s, t_plan);
  if (args->workspace_bytes < L.ws_end) return SPECGEN_ERR_WORKSPACE;

  t_plan_bytes.assign(L.ws_plan + L.plan_bytes, 0);  // zeroed header, then the plan
  PlanHeader h;
  h.n_split = (int32_t)t_plan.split.size();
  h.n_tc = (int32_t)t_plan.tc.size();
  h.n_tc_ctas = (int32_t)t_plan.cta_offsets.size() - 1;
  h.n_forks = s.F;
  h.split_off = (int32_t)L.split_off;
  h.tc_off = (int32_t)L.tc_off;
  h.cta_items_off = (int32_t)L.cta_items_off;
  h.cta_offsets_off = (int32_t)L.cta_offsets_off;
  h.part_base_off = (int32_t)L.part_base_off;
  h.n_parts_off = (int32_t)L.n_parts_off;
  h.n_sfx = (int32_t)t_plan.sfx.size();
  h.n_sfx_ctas = t_plan.n_sfx_ctas;
  h.sfx_off = (int32_t)L.sfx_off;
  h.sfx_offsets_off = (int32_t)L.sfx_offsets_off;
  unsigned char* b = t_plan_bytes.data() + L.ws_plan;
  memcpy(b, &h, sizeof(h));
  auto put = [&](size_t off, const void* src, size_t bytes) {
    if (bytes) memcpy(b + off, src, bytes);
  };
  put(L.split_off, t_plan.split.data(), t_plan.split.size() * sizeof(SplitItem));
  put(L.tc_off, t_plan.tc.data(), t_plan.tc.size() * sizeof(TcItem));
  put(L.cta_items_off, t_plan.cta_items.data(), t_plan.cta_items.size() * 4);
  put(L.cta_offsets_off, t_plan.cta_offsets.data(), t_plan.cta_offsets.size() * 4);
  put(L.sfx_off, t_plan.sfx.data(), t_plan.sfx.size() * sizeof(TcItem));
  put(L.sfx_offsets_off, t_plan.sfx_offsets.data(), t_plan.sfx_offsets.size() * 4);
  put(L.part_base_off, t_plan.part_base.data(), (size_t)s.F * 4);
  put(L.n_parts_off, t_plan.n_parts.data(), t_plan.n_parts.size() * 4);

  plan->valid = 1;
  plan->n_tc_items = h.n_tc;
  plan->n_tc_ctas = h.n_tc_ctas;
  plan->n_split_items = h.n_split;
  plan->n_rows = s.F * s.hq;
  plan->total_slots = t_plan.total_slots;
  plan->n_part_groups = t_plan.n_groups;
  bool causal = false;  // causal suffix items (prefill chunks) need the per-row limit
  for (const TcItem& it : t_plan.tc) causal = causal || it.row_limit0 > 0;
  plan->flags = (s.latent ? 1 : 0) | (args->kv_layout == SPECGEN_KV_TILED ? 2 : 0) |
                (causal ? 4 : 0);
  plan->plan_bytes = (int64_t)L.plan_bytes;
  plan->ws_plan_off = (int64_t)L.ws_plan;
  plan->ws_part_o_off = (int64_t)L.ws_part_o;
  plan->ws_part_lse_off = (int64_t)L.ws_part_lse;
  plan->ws_end = (int64_t)L.ws_end;
  plan->offsets[0] = (int64_t)L.split_off;
  plan->offsets[1] = (int64_t)L.tc_off;
  plan->offsets[2] = (int64_t)L.cta_items_off;
  plan->offsets[3] = (int64_t)L.cta_offsets_off;
  plan->offsets[4] = (int64_t)L.part_base_off;
  plan->offsets[5] = (int64_t)L.n_parts_off;
  plan->offsets[6] = t_plan.n_parts.empty() ? 0 : (int64_t)*std::max_element(t_plan.n_parts.begin(), t_plan.n_parts.end());
  plan->n_sfx_items = h.n_sfx;
  plan->n_sfx_ctas = h.n_sfx_ctas;
  plan->sfx_offsets[0] = (int64_t)L.sfx_off;
  plan->sfx_offsets[1] = (int64_t)L.sfx_offsets_off;
  return SPECGEN_OK;
}

// One upload of the plan region built last on this thread: the zeroed header
// (status word), then the plan.
specgen_status upload_plan(void* workspace, void* cuda_stream) {
  if (cudaMemcpyAsync(workspace, t_plan_bytes.data(), t_plan_bytes.size(), cudaMemcpyHostToDevice,
                      static_cast<cudaStream_t>(cuda_stream)) != cudaSuccess)
    return SPECGEN_ERR_CUDA;
  return SPECGEN_OK;
}

// Page-locked staging for the plan uploads of the one-call step
// (specgen_fork_attn_decode_staged): a ring of kRing host slots per host
// thread.  A copy from page-locked memory is queued without the host staging
// it first, so the call returns as soon as its work is queued.  A slot is
// written again only after the copy that last read it has run (an event
// recorded behind that copy), which lets the host run up to kRing calls ahead
// of the GPU and holds it there.  A slot grows, to the next power of two, when
// a plan does not fit; the slots are kept until the process exits.  If
// page-locked memory cannot be had, the upload goes from the pageable buffer.
struct PinnedRing {
  static constexpr int kRing = 4;
  void* buf[kRing] = {};
  size_t cap[kRing] = {};
  cudaEvent_t read[kRing] = {};
  int dev = -1;
  int next = 0;
};
thread_local PinnedRing t_ring;

specgen_status upload_plan_pinned(void* workspace, void* cuda_stream) {
  PinnedRing& r = t_ring;
  cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return SPECGEN_ERR_CUDA;
  if (dev != r.dev) {  // an event belongs to the device it was made on
    for (int i = 0; i < PinnedRing::kRing; ++i) {
      if (!r.read[i]) continue;
      if (cudaEventSynchronize(r.read[i]) != cudaSuccess) return SPECGEN_ERR_CUDA;
      cudaEventDestroy(r.read[i]);
      r.read[i] = nullptr;
    }
    r.dev = dev;
  }
  const int k = r.next;
  r.next = (k + 1) % PinnedRing::kRing;
  if (r.read[k]) {
    if (cudaEventSynchronize(r.read[k]) != cudaSuccess) return SPECGEN_ERR_CUDA;
  } else if (cudaEventCreateWithFlags(&r.read[k], cudaEventDisableTiming) != cudaSuccess) {
    r.read[k] = nullptr;
    return SPECGEN_ERR_CUDA;
  }
  const size_t n = t_plan_bytes.size();
  if (r.cap[k] < n) {
    size_t c = 4096;
    while (c < n) c <<= 1;
    if (r.buf[k]) cudaFreeHost(r.buf[k]);
    r.buf[k] = nullptr;
    r.cap[k] = 0;
    if (cudaHostAlloc(&r.buf[k], c, cudaHostAllocPortable) != cudaSuccess) {
      (void)cudaGetLastError();
      r.buf[k] = nullptr;
      return upload_plan(workspace, cuda_stream);
    }
    r.cap[k] = c;
  }
  memcpy(r.buf[k], t_plan_bytes.data(), n);
  if (cudaMemcpyAsync(workspace, r.buf[k], n, cudaMemcpyHostToDevice, stream) != cudaSuccess ||
      cudaEventRecord(r.read[k], stream) != cudaSuccess)
    return SPECGEN_ERR_CUDA;
  return SPECGEN_OK;
}

specgen_status plan_impl(const specgen_fork_attn_args* args, const Shape& s, const Rows& rows,
                         specgen_plan* plan, void* cuda_stream, void* host_dst,
                         size_t host_bytes, bool pinned) {
  specgen_status st;
  if ((st = check_pointers(args)) != SPECGEN_OK) return st;
  if ((st = plan_build(args, s, rows, plan)) != SPECGEN_OK) {
    memset(plan, 0, sizeof(*plan));
    return st;
  }
  if (host_dst) {
    if (host_bytes < t_plan_bytes.size()) {
      memset(plan, 0, sizeof(*plan));
      return SPECGEN_ERR_WORKSPACE;
    }
    memcpy(host_dst, t_plan_bytes.data(), t_plan_bytes.size());
    return SPECGEN_OK;
  }
  st = pinned ? upload_plan_pinned(args->workspace, cuda_stream)
              : upload_plan(args->workspace, cuda_stream);
  if (st != SPECGEN_OK) memset(plan, 0, sizeof(*plan));
  return st;
}

}  // namespace

extern "C" {

}  // extern "C"

namespace {

// Records mark `i` of the caller's event list (if there is one) on `stream`.
struct Marks {
  void* const* events;
  int n;
  int launches = 0;
  bool mark(cudaStream_t stream, int i) {
    if (!events || i >= n || !events[i]) return true;
    // inside a stream capture the mark must be an external event-record node so
    // that it still records a time stamp when the graph is replayed
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(stream, &cs) != cudaSuccess) return false;
    if (cs == cudaStreamCaptureStatusActive)
      return cudaEventRecordWithFlags(static_cast<cudaEvent_t>(events[i]), stream,
                                      cudaEventRecordExternal) == cudaSuccess;
    return cudaEventRecord(static_cast<cudaEvent_t>(events[i]), stream) == cudaSuccess;
  }
};

// stages: bit 0 the partial-attention kernels, bit 1 the merge.
// region: where the plan region (status header, then the plan) was uploaded,
// when not at the start of args->workspace (the partials stay there)
specgen_status run_impl(const specgen_fork_attn_args* args, const specgen_plan* plan,
                        void* cuda_stream, Marks& marks, int stages = 3,
                        unsigned char* region = nullptr);

}  // namespace

extern "C" {

specgen_status specgen_fork_attn_run(const specgen_fork_attn_args* args, const specgen_plan* plan,
                                     void* cuda_stream) {
  Marks marks{nullptr, 0};
  return run_impl(args, plan, cuda_stream, marks);
}

specgen_status specgen_fork_attn_run_partials(const specgen_fork_attn_args* args,
                                              const specgen_plan* plan, void* cuda_stream) {
  Marks marks{nullptr, 0};
  return run_impl(args, plan, cuda_stream, marks, 1);
}

specgen_status specgen_fork_attn_run_merge(const specgen_fork_attn_args* args,
                                           const specgen_plan* plan, void* cuda_stream) {
  Marks marks{nullptr, 0};
  return run_impl(args, plan, cuda_stream, marks, 2);
}

specgen_status specgen_fork_attn_run_profiled(const specgen_fork_attn_args* args,
                                              const specgen_plan* plan, void* cuda_stream,
                                              void* const* events, int n_events,
                                              int* n_launches) {
  Marks marks{events, n_events};
  specgen_status st = run_impl(args, plan, cuda_stream, marks);
  if (n_launches) *n_launches = marks.launches;
  return st;
}

}  // extern "C"

namespace {

specgen_status run_impl(const specgen_fork_attn_args* args, const specgen_plan* plan,
                        void* cuda_stream, Marks& marks, int stages, unsigned char* region) {
  if (!args || !plan) return SPECGEN_ERR_NULL;
  if (!plan->valid) return SPECGEN_ERR_SHAPE;
  specgen_status st = check_pointers(args);
  if (st != SPECGEN_OK) return st;
  if ((int64_t)args->workspace_bytes < plan->ws_end) return SPECGEN_ERR_WORKSPACE;
  if ((args->v_pages == nullptr) != (plan->flags & 1)) return SPECGEN_ERR_SHAPE;
  if ((args->kv_layout == SPECGEN_KV_TILED) != ((plan->flags & 2) != 0)) return SPECGEN_ERR_SHAPE;
  cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
  unsigned char* ws = static_cast<unsigned char*>(args->workspace);
  unsigned char* hdr = region ? region : ws;  // status word, then the plan
  unsigned char* pl = hdr + plan->ws_plan_off;
  float* part_o = reinterpret_cast<float*>(ws + plan->ws_part_o_off);
  float* part_lse = reinterpret_cast<float*>(ws + plan->ws_part_lse_off);

  SplitParams sp;
  sp.q = static_cast<const __nv_bfloat16*>(args->q);
  sp.k_pages = static_cast<const __nv_bfloat16*>(args->k_pages);
  sp.v_pages = static_cast<const __nv_bfloat16*>(args->v_pages);
  sp.prefix_bt = args->prefix_block_table;
  sp.prefix_bt_off = args->prefix_bt_offsets;
  sp.suffix_bt = args->suffix_block_table;
  sp.suffix_bt_off = args->suffix_bt_offsets;
  sp.items = reinterpret_cast<const SplitItem*>(pl + plan->offsets[0]);
  sp.part_o = part_o;
  sp.part_lse = part_lse;
  sp.status = reinterpret_cast<uint32_t*>(hdr);
  sp.hq = args->hq;
  sp.hkv = args->hkv;
  sp.dqk = args->head_dim_qk;
  sp.dv = args->head_dim_v;
  sp.page_size = args->page_size;
  sp.num_pages = args->num_pages;
  sp.scale_log2 = args->scale * 1.4426950408889634f;
  sp.suffix_lens = args->suffix_lens;
  if (!marks.mark(stream, 0)) return SPECGEN_ERR_CUDA;
  // With both partial kernels the suffix stage goes first: it waits for the
  // stream's previous kernel, then lets the prefix kernel launch beside it on
  // the SMs it leaves free; the prefix kernel, which usually ends last, waits
  // for the suffix-stage grid only at its end, and the merge waits for the
  // prefix kernel.  (The other order makes the suffix stage hold its CTAs
  // until the prefix kernel completes: two grid completions in a row at the
  // end of every call.)
  const bool both = (stages & 1) && plan->n_tc_ctas > 0 && plan->n_sfx_ctas > 0;
  auto launch_tc = [&]() -> specgen_status {
    TcParams tp;
    tp.q = sp.q;
    tp.prefix_bt = args->prefix_block_table;
    tp.prefix_bt_off = args->prefix_bt_offsets;
    tp.suffix_bt = args->suffix_block_table;
    tp.suffix_bt_off = args->suffix_bt_offsets;
    tp.items = reinterpret_cast<const TcItem*>(pl + plan->offsets[1]);
    tp.cta_offsets = reinterpret_cast<const int32_t*>(pl + plan->offsets[3]);
    tp.part_base = reinterpret_cast<const int32_t*>(pl + plan->offsets[4]);
    tp.part_o = part_o;
    tp.part_lse = part_lse;
    tp.status = sp.status;
    tp.hq = args->hq;
    tp.hkv = args->hkv;
    tp.G = args->hq / args->hkv;
    tp.dv = args->head_dim_v;
    tp.num_pages = args->num_pages;
    tp.scale_log2 = sp.scale_log2;
    tp.suffix_lens = args->suffix_lens;
    tp.wait_at_end = both ? 1 : 0;
    cudaError_t e;
    if (args->v_pages == nullptr) {
      MlaParams mp;
      mp.q = tp.q;
      mp.prefix_bt = tp.prefix_bt;
      mp.prefix_bt_off = tp.prefix_bt_off;
      mp.suffix_bt = tp.suffix_bt;
      mp.suffix_bt_off = tp.suffix_bt_off;
      mp.items = tp.items;
      mp.cta_offsets = tp.cta_offsets;
      mp.part_base = tp.part_base;
      mp.part_o = part_o;
      mp.part_lse = part_lse;
      mp.status = tp.status;
      mp.hq = args->hq;
      mp.num_pages = args->num_pages;
      mp.scale_log2 = tp.scale_log2;
      mp.suffix_lens = args->suffix_lens;
      e = launch_mla_tc(mp, args->k_pages, plan->n_tc_ctas, stream);
    } else {
      tp.k_pages = static_cast<const __nv_bfloat16*>(args->k_pages);
      tp.v_pages = static_cast<const __nv_bfloat16*>(args->v_pages);
      e = launch_fork_tc(tp, args->k_pages, args->v_pages, plan->n_tc_ctas, args->head_dim_qk,
                         args->kv_layout == SPECGEN_KV_TILED, (plan->flags & 4) != 0, stream);
    }
    if (e != cudaSuccess) return SPECGEN_ERR_CUDA;
    if (!marks.mark(stream, ++marks.launches)) return SPECGEN_ERR_CUDA;
    return SPECGEN_OK;
  };
  auto launch_sfx = [&]() -> specgen_status {
    SfxParams xp;
    xp.q = sp.q;
    xp.k_pages = static_cast<const __nv_bfloat16*>(args->k_pages);
    xp.v_pages = static_cast<const __nv_bfloat16*>(args->v_pages);
    xp.suffix_bt = args->suffix_block_table;
    xp.suffix_bt_off = args->suffix_bt_offsets;
    xp.items = reinterpret_cast<const TcItem*>(pl + plan->sfx_offsets[0]);
    xp.worker_offsets = reinterpret_cast<const int32_t*>(pl + plan->sfx_offsets[1]);
    xp.part_base = reinterpret_cast<const int32_t*>(pl + plan->offsets[4]);
    xp.part_o = part_o;
    xp.part_lse = part_lse;
    xp.status = sp.status;
    xp.suffix_lens = args->suffix_lens;
    xp.hq = args->hq;
    xp.hkv = args->hkv;
    xp.G = args->hq / args->hkv;
    xp.dv = args->head_dim_v;
    xp.num_pages = args->num_pages;
    xp.scale_log2 = sp.scale_log2;
    xp.late_trigger = both ? 1 : 0;
    if (launch_suffix_stage(xp, args->k_pages, args->v_pages, plan->n_sfx_ctas, args->head_dim_qk,
                            args->kv_layout == SPECGEN_KV_TILED, stream) != cudaSuccess)
      return SPECGEN_ERR_CUDA;
    if (!marks.mark(stream, ++marks.launches)) return SPECGEN_ERR_CUDA;
    return SPECGEN_OK;
  };
  if ((stages & 1) && plan->n_sfx_ctas > 0) {
    const specgen_status st = launch_sfx();
    if (st != SPECGEN_OK) return st;
  }
  if ((stages & 1) && plan->n_tc_ctas > 0) {
    const specgen_status st = launch_tc();
    if (st != SPECGEN_OK) return st;
  }
  if ((stages & 1) && plan->n_split_items > 0) {
    if (launch_split_decode(sp, plan->n_split_items, args->v_pages == nullptr, stream) !=
        cudaSuccess)
      return SPECGEN_ERR_CUDA;
    if (!marks.mark(stream, ++marks.launches)) return SPECGEN_ERR_CUDA;
  }

  if (stages & 2) {  // merge pass: combine every row's partials
    MergeParams mp;
    mp.part_o = part_o;
    mp.part_lse = part_lse;
    mp.part_base = reinterpret_cast<const int32_t*>(pl + plan->offsets[4]);
    mp.n_parts = reinterpret_cast<const int32_t*>(pl + plan->offsets[5]);
    mp.max_parts = (int)plan->offsets[6];
    mp.out = static_cast<__nv_bfloat16*>(args->out);
    mp.lse = args->lse;
    mp.n_rows = plan->n_rows;
    mp.n_groups = plan->n_part_groups;
    mp.hq = args->hq;
    mp.dv = args->head_dim_v;
    if (launch_merge_parts(mp, stream,
                           (plan->n_tc_ctas > 0 || plan->n_sfx_ctas > 0) && plan->n_split_items == 0) !=
        cudaSuccess)
      return SPECGEN_ERR_CUDA;
    if (!marks.mark(stream, ++marks.launches)) return SPECGEN_ERR_CUDA;
  }
  return SPECGEN_OK;
}

}  // namespace

extern "C" {

specgen_status specgen_fork_attn_decode(const specgen_fork_attn_args* args,
                                        const specgen_host_lens* lens, void* cuda_stream) {
  specgen_plan plan;
  specgen_status st = specgen_fork_attn_plan(args, lens, &plan, cuda_stream);
  if (st != SPECGEN_OK) return st;
  return specgen_fork_attn_run(args, &plan, cuda_stream);
}

specgen_status specgen_fork_attn_decode_staged(const specgen_fork_attn_args* args,
                                               const specgen_host_lens* lens,
                                               const void* host_in, void* dev_in,
                                               size_t in_bytes, const void* dev_out,
                                               void* host_out, size_t out_bytes,
                                               void* cuda_stream) {
  if (!args || !lens) return SPECGEN_ERR_NULL;
  if ((in_bytes > 0 && (!host_in || !dev_in)) || (out_bytes > 0 && (!dev_out || !host_out)))
    return SPECGEN_ERR_NULL;
  cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
  // shapes first: a call refused here queues nothing
  Shape s;
  specgen_status st = check_shape(args, lens, &s);
  if (st != SPECGEN_OK) return st;
  if (in_bytes > 0 &&
      cudaMemcpyAsync(dev_in, host_in, in_bytes, cudaMemcpyHostToDevice, stream) != cudaSuccess)
    return SPECGEN_ERR_CUDA;
  specgen_plan plan;
  memset(&plan, 0, sizeof(plan));
  st = plan_impl(args, s, rows_for_decode(lens, s.T, s.F), &plan, cuda_stream, nullptr, 0, true);
  if (st != SPECGEN_OK) return st;
  if ((st = specgen_fork_attn_run(args, &plan, cuda_stream)) != SPECGEN_OK) return st;
  if (out_bytes > 0 &&
      cudaMemcpyAsync(host_out, dev_out, out_bytes, cudaMemcpyDeviceToHost, stream) != cudaSuccess)
    return SPECGEN_ERR_CUDA;
  return SPECGEN_OK;
}

specgen_status specgen_fork_attn_decode_staged_inline(const specgen_fork_attn_args* args,
                                                      const specgen_host_lens* lens,
                                                      void* host_in, void* dev_in,
                                                      size_t in_bytes, size_t in_capacity,
                                                      const void* dev_out, void* host_out,
                                                      size_t out_bytes, void* cuda_stream) {
  if (!args || !lens || !host_in || !dev_in) return SPECGEN_ERR_NULL;
  if (out_bytes > 0 && (!dev_out || !host_out)) return SPECGEN_ERR_NULL;
  if (reinterpret_cast<uintptr_t>(dev_in) % 256 != 0) return SPECGEN_ERR_SHAPE;
  // everything that can refuse the call is checked before anything is queued
  Shape s;
  specgen_status st = check_shape(args, lens, &s);
  if (st != SPECGEN_OK) return st;
  if ((st = check_pointers(args)) != SPECGEN_OK) return st;
  const size_t off = align_up(in_bytes, 256);
  if (off > in_capacity) return SPECGEN_ERR_WORKSPACE;
  cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
  unsigned char* hin = static_cast<unsigned char*>(host_in);
  unsigned char* din = static_cast<unsigned char*>(dev_in);
  // A stream with nothing left to run is waiting for this host: its inputs
  // then go up at once, overlapping the planning, and the plan follows in a
  // second copy.  A busy stream gets inputs and plan in one copy after the
  // planning (the copy would wait behind the queued work anyway).  A stream
  // that cannot be queried counts as busy (its copy then reports the error).
  const cudaError_t q = cudaStreamQuery(stream);
  if (q != cudaSuccess) (void)cudaGetLastError();  // "not ready" is not an error
  const bool idle = q == cudaSuccess;
  if (idle && in_bytes > 0 &&
      cudaMemcpyAsync(dev_in, host_in, in_bytes, cudaMemcpyHostToDevice, stream) != cudaSuccess)
    return SPECGEN_ERR_CUDA;
  specgen_plan plan;
  memset(&plan, 0, sizeof(plan));
  if ((st = plan_build(args, s, rows_for_decode(lens, s.T, s.F), &plan)) != SPECGEN_OK) return st;
  const size_t region = t_plan_bytes.size();
  if (off + region > in_capacity) return SPECGEN_ERR_WORKSPACE;
  memcpy(hin + off, t_plan_bytes.data(), region);
  const cudaError_t e =
      idle ? cudaMemcpyAsync(din + off, hin + off, region, cudaMemcpyHostToDevice, stream)
           : cudaMemcpyAsync(dev_in, host_in, off + region, cudaMemcpyHostToDevice, stream);
  if (e != cudaSuccess) return SPECGEN_ERR_CUDA;
  Marks marks{nullptr, 0};
  if ((st = run_impl(args, &plan, cuda_stream, marks, 3,
                     static_cast<unsigned char*>(dev_in) + off)) != SPECGEN_OK)
    return st;
  if (out_bytes > 0 &&
      cudaMemcpyAsync(host_out, dev_out, out_bytes, cudaMemcpyDeviceToHost, stream) != cudaSuccess)
    return SPECGEN_ERR_CUDA;
  return SPECGEN_OK;
}

specgen_status specgen_append_kv(const specgen_append_args* a, void* cuda_stream) {
  if (!a) return SPECGEN_ERR_NULL;
  if (a->total_forks < 0 || a->hkv < 1 || a->page_size < 1 || a->num_pages < 0 || a->num_free < 0)
    return SPECGEN_ERR_SHAPE;
  if (a->head_dim_qk < 8 || a->head_dim_qk % 8 != 0) return SPECGEN_ERR_UNSUPPORTED;
  const bool latent = a->v_pages == nullptr;
  if (latent != (a->v_new == nullptr)) return SPECGEN_ERR_SHAPE;
  if (!latent && (a->head_dim_v < 8 || a->head_dim_v % 8 != 0)) return SPECGEN_ERR_UNSUPPORTED;
  if (a->page_size > 1024 || (a->page_size & (a->page_size - 1)) != 0)
    return SPECGEN_ERR_UNSUPPORTED;
  if (a->kv_layout != SPECGEN_KV_ROWS && a->kv_layout != SPECGEN_KV_TILED) return SPECGEN_ERR_SHAPE;
  if (a->kv_layout == SPECGEN_KV_TILED && (latent || a->page_size % 8 != 0))
    return SPECGEN_ERR_UNSUPPORTED;
  if (a->total_forks == 0) return SPECGEN_OK;
  if (!a->k_new || !a->k_pages || !a->suffix_block_table || !a->suffix_bt_offsets ||
      !a->suffix_lens || (a->num_free > 0 && !a->free_pages))
    return SPECGEN_ERR_NULL;
  if (a->suffix_lens_next != nullptr && a->suffix_lens_next == a->suffix_lens)
    return SPECGEN_ERR_UNSUPPORTED;
  const void* rows[4] = {a->k_new, a->v_new, a->k_pages, a->v_pages};
  for (const void* r : rows)
    if (reinterpret_cast<uintptr_t>(r) % 16 != 0) return SPECGEN_ERR_SHAPE;
  AppendParams p;
  p.k_new = static_cast<const __nv_bfloat16*>(a->k_new);
  p.v_new = static_cast<const __nv_bfloat16*>(a->v_new);
  p.k_pages = static_cast<__nv_bfloat16*>(a->k_pages);
  p.v_pages = static_cast<__nv_bfloat16*>(a->v_pages);
  p.table = a->suffix_block_table;
  p.offs = a->suffix_bt_offsets;
  p.lens = a->suffix_lens;
  p.lens_next = a->suffix_lens_next;
  p.free_pages = a->free_pages;
  p.status = a->status;
  p.F = a->total_forks;
  p.hkv = a->hkv;
  p.dqk = a->head_dim_qk;
  p.dv = latent ? 0 : a->head_dim_v;
  p.B = a->page_size;
  p.num_pages = a->num_pages;
  p.num_free = a->num_free;
  p.tiled = a->kv_layout == SPECGEN_KV_TILED;
  if (launch_append_kv(p, static_cast<cudaStream_t>(cuda_stream)) != cudaSuccess)
    return SPECGEN_ERR_CUDA;
  return SPECGEN_OK;
}

namespace {

// Checks a pool description; fills the 16-byte words per page of each pool.
specgen_status check_pool(const specgen_pool_desc* d, size_t* k16, size_t* v16) {
  if (!d) return SPECGEN_ERR_NULL;
  if (d->hkv < 1 || d->page_size < 1 || d->num_pages < 0 || d->head_dim_qk < 1)
    return SPECGEN_ERR_SHAPE;
  if (d->v_pages && d->head_dim_v < 1) return SPECGEN_ERR_SHAPE;
  const size_t kb = (size_t)d->hkv * d->page_size * d->head_dim_qk * 2;
  const size_t vb = d->v_pages ? (size_t)d->hkv * d->page_size * d->head_dim_v * 2 : 0;
  if (kb % 16 != 0 || vb % 16 != 0) return SPECGEN_ERR_UNSUPPORTED;
  *k16 = kb / 16;
  *v16 = vb / 16;
  return SPECGEN_OK;
}

specgen_status pack_impl(const specgen_pool_desc* d, const int32_t* table, int n_pages,
                         void* packed, bool unpack, void* cuda_stream) {
  size_t k16 = 0, v16 = 0;
  specgen_status st = check_pool(d, &k16, &v16);
  if (st != SPECGEN_OK) return st;
  if (n_pages < 0) return SPECGEN_ERR_SHAPE;
  if (n_pages == 0) return SPECGEN_OK;
  if (!table || !packed || !d->k_pages) return SPECGEN_ERR_NULL;
  const void* ptrs[3] = {packed, d->k_pages, d->v_pages};
  for (const void* q : ptrs)
    if (reinterpret_cast<uintptr_t>(q) % 16 != 0) return SPECGEN_ERR_SHAPE;
  PackParams p;
  p.k_pages = static_cast<uint4*>(d->k_pages);
  p.v_pages = static_cast<uint4*>(d->v_pages);
  p.packed = static_cast<uint4*>(packed);
  p.table = table;
  p.status = d->status;
  p.k_block16 = k16;
  p.v_block16 = v16;
  p.n_pages = n_pages;
  p.num_pages = d->num_pages;
  p.unpack = unpack;
  if (launch_pack_pages(p, device_sm_count(), static_cast<cudaStream_t>(cuda_stream)) !=
      cudaSuccess)
    return SPECGEN_ERR_CUDA;
  return SPECGEN_OK;
}

}  // namespace

size_t specgen_packed_bytes(const specgen_pool_desc* pool, int n_pages) {
  size_t k16 = 0, v16 = 0;
  if (n_pages < 0 || check_pool(pool, &k16, &v16) != SPECGEN_OK) return 0;
  return (size_t)n_pages * (k16 + v16) * 16;
}

specgen_status specgen_pack_pages(const specgen_pool_desc* pool, const int32_t* table,
                                  int n_pages, void* packed, void* cuda_stream) {
  return pack_impl(pool, table, n_pages, packed, false, cuda_stream);
}

specgen_status specgen_unpack_pages(const specgen_pool_desc* pool, const int32_t* table,
                                    int n_pages, const void* packed, void* cuda_stream) {
  return pack_impl(pool, table, n_pages, const_cast<void*>(packed), true, cuda_stream);
}

specgen_status specgen_lse_merge(const void* out_a, const float* lse_a, const void* out_b,
                                 const float* lse_b, void* out, float* lse, int rows, int dv,
                                 int dtype, void* cuda_stream) {
  if (rows < 0 || dv < 0) return SPECGEN_ERR_SHAPE;
  if (dtype != 0 && dtype != 1) return SPECGEN_ERR_UNSUPPORTED;
  if (rows == 0) return SPECGEN_OK;
  if (!out_a || !lse_a || !out_b || !lse_b || !out || !lse) return SPECGEN_ERR_NULL;
  if (launch_lse_merge2(out_a, lse_a, out_b, lse_b, out, lse, rows, dv, dtype,
                        static_cast<cudaStream_t>(cuda_stream)) != cudaSuccess)
    return SPECGEN_ERR_CUDA;
  return SPECGEN_OK;
}

specgen_status specgen_workspace_status(const void* workspace, void* cuda_stream) {
  if (!workspace) return SPECGEN_ERR_NULL;
  uint32_t word = 0;
  cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
  if (cudaMemcpyAsync(&word, workspace, sizeof(word), cudaMemcpyDeviceToHost, stream) !=
      cudaSuccess)
    return SPECGEN_ERR_CUDA;
  if (cudaStreamSynchronize(stream) != cudaSuccess) return SPECGEN_ERR_CUDA;
  if (word & kStatusTimeout) return SPECGEN_ERR_TIMEOUT;
  if (word & kStatusIndex) return SPECGEN_ERR_INDEX;
  return SPECGEN_OK;
}

const char* specgen_status_string(specgen_status status) {
  switch (status) {
    case SPECGEN_OK: return "ok";
    case SPECGEN_ERR_NULL: return "null pointer argument";
    case SPECGEN_ERR_SHAPE: return "inconsistent shape or length";
    case SPECGEN_ERR_UNSUPPORTED: return "unsupported head dims, page size or group size";
    case SPECGEN_ERR_WORKSPACE: return "workspace too small or misaligned";
    case SPECGEN_ERR_INDEX: return "page id outside [0, num_pages)";
    case SPECGEN_ERR_CUDA: return "CUDA error";
    case SPECGEN_ERR_TIMEOUT: return "device wait exceeded its iteration limit";
  }
  return "unknown status";
}

int specgen_version(void) { return 100; }

}  // extern "C"

// ---------------------------------------------------------------------------
// Allocation-free variant of specgen_fork_attn_decode.
//
// Some callers cannot allocate device memory at all: a plugin that runs inside
// a host engine which owns the whole device memory pool, or code on a
// latency-critical path where cudaMalloc (which can synchronise the device) is
// not allowed.  They cannot provide the workspace the other entry points take,
// so this variant uses a fixed, library-owned scratch array instead.  The
// array is a file-scope device variable: every GPU that loads this library
// holds kStaticWorkspaceBytes of it until the process exits.
namespace {

constexpr size_t kStaticWorkspaceBytes = 16u << 20;  // 16 MiB
static __device__ __align__(256) unsigned char g_static_workspace[kStaticWorkspaceBytes];

// Device address of the scratch array on the current device.  In host code
// the symbol names a host-side stand-in, not device memory, so the address is
// asked of the runtime with the device current, on every call: it is a host
// query, and an address kept from an earlier call could belong to a context
// that has since been torn down and created again.
specgen_status static_workspace(void** ptr) {
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_static_workspace) != cudaSuccess || !p) return SPECGEN_ERR_CUDA;
  *ptr = p;
  return SPECGEN_OK;
}

}  // namespace

extern "C" {

specgen_status specgen_fork_attn_decode_static(const specgen_fork_attn_args* args,
                                               const specgen_host_lens* lens,
                                               void* cuda_stream) {
  if (!args) return SPECGEN_ERR_NULL;
  Shape s;
  specgen_status st = check_shape(args, lens, &s);
  if (st != SPECGEN_OK) return st;
  specgen_fork_attn_args a = *args;
  a.workspace_bytes = kStaticWorkspaceBytes;
  // the other pointers are checked as for every call; the workspace is ours
  a.workspace = reinterpret_cast<void*>(kAlign);
  if ((st = check_pointers(&a)) != SPECGEN_OK) return st;
  // planned once, on the host: a call that needs more than the array is
  // refused here, before any CUDA call
  specgen_plan plan;
  memset(&plan, 0, sizeof(plan));
  if ((st = plan_build(&a, s, rows_for_decode(lens, s.T, s.F), &plan)) != SPECGEN_OK) return st;
  void* ws = nullptr;
  if ((st = static_workspace(&ws)) != SPECGEN_OK) return st;
  a.workspace = ws;
  if ((st = upload_plan(ws, cuda_stream)) != SPECGEN_OK) return st;
  return specgen_fork_attn_run(&a, &plan, cuda_stream);
}

specgen_status specgen_static_workspace_status(void* cuda_stream) {
  void* ws = nullptr;
  const specgen_status st = static_workspace(&ws);
  if (st != SPECGEN_OK) return st;
  return specgen_workspace_status(ws, cuda_stream);
}

}  // extern "C"
