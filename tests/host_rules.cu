// host_rules.cu -- the launch code's host-side rules, checked exhaustively on
// the CPU (no device is touched): the backward team shapes, the ragged
// workspace offsets, the ragged norm backward's bucket covers and partial-row
// segments, the longest ragged norm row, and the stripe design's stripes,
// element counts, partial-row columns and workspace.  Built and run by
// tests/test_host_rules.py; prints "ok" and exits 0 when every check holds.
#include <cstdio>
#include <initializer_list>

#include "bwd_launch.cuh"
#include "launchers.cuh"

using namespace rowop;

static int g_fails = 0;
#define CHECK(cond, fmt, ...)                                                   \
  do {                                                                          \
    if (!(cond)) {                                                              \
      if (g_fails++ < 20)                                                       \
        std::printf("FAIL line %d: %s | " fmt "\n", __LINE__, #cond, __VA_ARGS__); \
    }                                                                           \
  } while (0)

static bool pow2(int64_t v) { return v > 0 && (v & (v - 1)) == 0; }

// Team shapes: a team (tpr threads of each of cs CTAs, cpt slots a thread)
// covers the row's units; lane groups are powers of two filling a CTA of
// small_cta threads; warp teams are whole warps; CTAs stay within 512
// threads; clusters are powers of two up to 16; a forced split is honoured
// whenever its CTAs fit; the rule refuses only rows no 16-CTA team can hold.
static void check_shapes() {
  for (int cpt : {2, 4, 8})
    for (int small : {128, 256})
      for (int force : {0, 2, 4, 8, 16})
        for (int64_t units = 1; units <= 8192LL * cpt + 64; units += units < 4096 ? 1 : 29) {
          BwdShape s{};
          const bool ok = bwd_shape(units, cpt, force, small, s);
          const int64_t need = (units + cpt - 1) / cpt;
          CHECK(ok == (need <= 8192), "units %lld cpt %d force %d", (long long)units, cpt, force);
          if (!ok) continue;
          CHECK(s.cs >= 1 && s.cs <= kMaxCluster && pow2(s.cs), "cs %d", s.cs);
          CHECK(s.nt >= 1 && s.nt <= kBwdMaxThreads && s.nt % s.tpr == 0, "nt %d tpr %d", s.nt,
                s.tpr);
          if (s.tpr < 32) {
            CHECK(pow2(s.tpr) && s.nt == small && s.cs == 1, "tpr %d nt %d cs %d", s.tpr, s.nt,
                  s.cs);
          } else {
            CHECK(s.tpr % 32 == 0 && s.tpr <= kBwdMaxThreads, "tpr %d", s.tpr);
          }
          if (s.cs > 1) CHECK(s.nt == s.tpr, "a cluster CTA is one team: nt %d tpr %d", s.nt, s.tpr);
          CHECK(static_cast<int64_t>(s.tpr) * s.cs * cpt >= units, "units %lld tpr %d cs %d",
                (long long)units, s.tpr, s.cs);
          const int64_t per = (need + force - 1) / (force > 0 ? force : 1);
          if (force >= 2 && per <= kBwdMaxThreads)
            CHECK(s.cs == force, "forced %d got %d", force, s.cs);
        }
}

// Ragged workspace: the regions follow each other, 256-byte aligned, each
// large enough; the classify blocks cover every row.
static void check_ragged_workspace() {
  for (int64_t rows : {0LL, 1LL, 7LL, 1023LL, 1024LL, 1025LL, 16384LL, 262144LL, 262145LL,
                       1000000LL, 2147483646LL}) {
    const int64_t blocks = ragged_blocks(rows), rpb = ragged_rows_per_block(rows);
    CHECK(blocks >= 1 && blocks <= kClassifyMaxBlocks, "rows %lld blocks %lld", (long long)rows,
          (long long)blocks);
    CHECK(blocks * rpb >= rows, "rows %lld", (long long)rows);
    const size_t co = ragged_counts_offset(rows), lo = ragged_lists_offset(rows);
    CHECK(co % 256 == 0 && co >= kWsBuckets + static_cast<size_t>(rows), "rows %lld",
          (long long)rows);
    CHECK(lo % 256 == 0 && lo >= co + 12 * static_cast<size_t>(blocks), "rows %lld",
          (long long)rows);
    CHECK(ragged_ws_bytes(rows) >= lo + 3 * kWsRecordBytes * static_cast<size_t>(rows),
          "rows %lld", (long long)rows);
  }
}

// Ragged norm backward: every row of every bucket fits its bucket's cover;
// the covers' segments follow the classify plan, 256-byte aligned, disjoint,
// each with room for the partial rows the launch may write.
static void check_ragged_norm_layout() {
  for (int es : {2, 4})
    for (int64_t max_len : {0LL, 1LL, 40LL, 1024LL, 1025LL, 2048LL, 2049LL, 8192LL, 8193LL,
                            16384LL, 16385LL, 70000LL, 131072LL})
      for (int nacc : {1, 2})
        for (int sm : {1, 148, 152}) {
          int64_t cover[3];
          bwd_ragged_covers(max_len, es, cover);
          CHECK(cover[kSmall] >= 1, "max_len %lld", (long long)max_len);
          for (int64_t n : std::initializer_list<int64_t>{1, max_len / 3, max_len / 2, max_len - 1,
                                                          max_len}) {
            if (n < 1 || n > max_len) continue;
            CHECK(cover[bucket_of(n, es)] >= n, "row %lld of max_len %lld es %d", (long long)n,
                  (long long)max_len, es);
          }
          CHECK(cover[kLarge] == (max_len * es > kMediumMaxBytes ? max_len : 0), "max_len %lld",
                (long long)max_len);
          for (int64_t rows : {1LL, 1000LL, 16384LL}) {
            size_t seg[3];
            const size_t total = bwd_ragged_layout(rows, max_len, es, nacc, sm, seg);
            CHECK(seg[0] >= ragged_ws_bytes(rows), "rows %lld", (long long)rows);
            for (int b = 0; b < 3; ++b) {
              const size_t need = static_cast<size_t>(kBwdMaxPartsPerSm) * sm * nacc *
                                  static_cast<size_t>(cover[b]) * sizeof(float);
              const size_t next = b < 2 ? seg[b + 1] : total;
              CHECK(seg[b] % 256 == 0 && seg[b] + need <= next, "bucket %d rows %lld", b,
                    (long long)rows);
            }
            CHECK(total == bwd_ragged_layout(rows, max_len, es, nacc, sm, nullptr), "%s", "");
          }
        }
}

// The longest ragged norm row is the longest row a team of half-slot
// threads can hold; one element more is refused by the shape rule.
static void check_ragged_norm_limit() {
  for (int es : {2, 4}) {
    const int e = 16 / es;
    const int cpt = kBwdSlots / e / 2;
    BwdShape s{};
    CHECK(bwd_shape((kBwdMaxColsNormRagged + e - 1) / e, cpt, 0, 128, s), "es %d", es);
    CHECK(!bwd_shape((kBwdMaxColsNormRagged + 1 + e - 1) / e, cpt, 0, 128, s), "es %d", es);
  }
}

// Forward tile design: the longest accepted row fits the largest cluster's
// portions at every head offset (one element more does not at the last
// offset), and the cluster chosen for a K-tile row is the smallest power of
// two whose portions hold at most `cap` tiles.
static void check_forward_rules() {
  for (int es : {2, 4}) {
    const int64_t e = 16 / es;
    const int64_t n = max_row_len_elems(es);
    const int64_t capacity = static_cast<int64_t>(kMaxPortionTiles) * kMaxCluster;
    for (int64_t h = 0; h < e; ++h) {
      const int64_t k = ((h + n + e - 1) / e + kTileChunks - 1) / kTileChunks;
      CHECK(k <= capacity, "es %d head %lld tiles %lld", es, (long long)h, (long long)k);
    }
    const int64_t k1 = ((e - 1 + n + 1 + e - 1) / e + kTileChunks - 1) / kTileChunks;
    CHECK(k1 > capacity, "es %d: one element more still fits", es);
  }
  for (int64_t cap : {1LL, 12LL, 96LL, 192LL})
    for (int64_t k = 1; k <= cap * kMaxCluster; ++k) {
      const int cs = pick_cluster(k, cap, 0);
      CHECK(pow2(cs) && cs >= 2 && cs <= kMaxCluster, "cs %d", cs);
      CHECK(ceil_div(k, cs) <= cap, "k %lld cap %lld cs %d", (long long)k, (long long)cap, cs);
      CHECK(cs == 2 || ceil_div(k, cs / 2) > cap, "k %lld cap %lld cs %d not smallest",
            (long long)k, (long long)cap, cs);
    }
  for (int w : {1, 2, 4, 8})
    for (int64_t tiles : {1LL, 4LL, 16LL, 17LL, 32LL, 64LL, 72LL, 192LL}) {
      const int g = kConsumerWarps / w;
      const int st = pick_stages(tiles, w, 0);
      CHECK(st >= g, "stages %d for %d groups", st, g);
      if (static_cast<int64_t>(g) * tiles * kTileBytes <= kStageBudgetBytes)
        CHECK(static_cast<int64_t>(st) * tiles * kTileBytes <= kStageBudgetBytes,
              "stages %d of %lld tiles over the budget", st, (long long)tiles);
    }
}

// Stripe design of the ragged norm backward: for every head class c and
// row length, the stats stripes cover the row's window positions and their
// element counts (the stats kernel's per-warp counts, the dx kernel's
// per-stripe counts) add up to the row; every column a dx stripe of any
// head class writes lands at an entry the finalize reads, and no other
// stripe writes it; the workspace parts are aligned, disjoint and large
// enough, and within the size the call asks for.
static void check_stripe_layout() {
  for (int es : {2, 4}) {
    const int e = 16 / es;
    const int64_t w1 = stripe_stat_width(es), w2 = stripe_dx_width(es);
    CHECK(w1 == static_cast<int64_t>(e) * kStatThreads * kStatChunks && w2 == static_cast<int64_t>(e) * kDxThreads,
          "es %d", es);
    for (int64_t max_len : {1LL, 7LL, 8LL, 2047LL, 2048LL, 4095LL, 4096LL, 4097LL, 32768LL,
                            70000LL, 131072LL}) {
      const StripeLayout L = stripe_layout(1000, max_len, es, 2);
      for (int c = 0; c < e; ++c) {
        for (int64_t len : std::initializer_list<int64_t>{1, 2, e - 1, e, e + 1, w2 - 1, w2,
                                                          w2 + 1, w1 - 1, w1, w1 + 1,
                                                          2 * w1 + 3, max_len - 1, max_len}) {
          if (len < 1 || len > max_len) continue;
          const int n = static_cast<int>(len);
          const int64_t nst = (len + c + w1 - 1) / w1;
          CHECK(nst <= L.ns1, "es %d c %d len %lld nst %lld ns1 %lld", es, c, (long long)len,
                (long long)nst, (long long)L.ns1);
          int64_t total = 0;
          for (int64_t q = 0; q < nst; ++q) {
            const int nq = static_cast<int>(std::min<int64_t>(len, w1 * (q + 1) - c) -
                                            std::max<int64_t>(0, w1 * q - c));
            int warps = 0;
            for (int w = 0; w < kStatThreads / 32; ++w)
              warps += e == 8 ? stat_warp_count<8>(static_cast<int>(w1 * q), n, c, w)
                              : stat_warp_count<4>(static_cast<int>(w1 * q), n, c, w);
            CHECK(nq > 0 && nq == warps, "es %d c %d len %lld stripe %lld: %d vs %d", es, c,
                  (long long)len, (long long)q, nq, warps);
            total += nq;
          }
          CHECK(total == len, "es %d c %d len %lld", es, c, (long long)len);
          CHECK((len + c + w2 - 1) / w2 <= L.ns2, "es %d c %d len %lld", es, c, (long long)len);
        }
        // a column j of head class c is in dx stripe (j + c) / w2, at entry
        // j - (w2 s - e); the finalize reads stripe j / w2 at j - w2 sa + e
        // and, when that entry is at least w2, stripe sa + 1 at that minus w2
        for (int64_t j = 0; j < std::min<int64_t>(max_len, 3 * w2 + 17); ++j) {
          const int64_t s = (j + c) / w2, l = j - (w2 * s - e);
          const int64_t sa = j / w2, ia = j - w2 * sa + e, ib = ia - w2;
          CHECK(s < L.ns2 && l >= 0 && l < w2 + e, "es %d c %d j %lld", es, c, (long long)j);
          const bool read = (s == sa && l == ia) || (s == sa + 1 && sa + 1 < L.ns2 && ib >= 0 && l == ib);
          CHECK(read, "es %d c %d column %lld (stripe %lld entry %lld) not read", es, c,
                (long long)j, (long long)s, (long long)l);
        }
      }
      for (int64_t rows : {1LL, 31LL, 32LL, 33LL, 4095LL, 16384LL, 33000LL, 1000000LL})
        for (int nacc : {1, 2}) {
          const StripeLayout R = stripe_layout(rows, max_len, es, nacc);
          CHECK(R.ng2 >= 1 && R.ng2 <= kDxMaxGroups && R.g2 >= 1 && R.ng2 * R.g2 >= rows,
                "rows %lld ng2 %lld g2 %lld", (long long)rows, (long long)R.ng2, (long long)R.g2);
          CHECK(R.ng1 * kStatRows >= rows && (R.ng1 - 1) * kStatRows < rows, "rows %lld",
                (long long)rows);
          CHECK(R.psum % 256 == 0 && R.part % 256 == 0 &&
                    R.part >= R.psum + static_cast<size_t>(rows) * R.ns1 * 16,
                "rows %lld", (long long)rows);
          CHECK(R.total >= R.part + static_cast<size_t>(R.ng2) * R.ns2 * nacc * (w2 + e) * 4,
                "rows %lld", (long long)rows);
          CHECK(bwd_ragged_norm_ws(rows, max_len, es, nacc, 152) >= R.total, "rows %lld",
                (long long)rows);
        }
    }
  }
}

int main() {
  check_stripe_layout();
  check_forward_rules();
  check_shapes();
  check_ragged_workspace();
  check_ragged_norm_layout();
  check_ragged_norm_limit();
  if (g_fails) {
    std::printf("%d checks failed\n", g_fails);
    return 1;
  }
  std::printf("ok\n");
  return 0;
}
