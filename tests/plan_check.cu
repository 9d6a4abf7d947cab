// Host-side check of the weight-stream stage planner (plan_stages, stage_desc)
// that decides every bulk copy of the decode kernel and of tvl_gemv: for each
// matrix of each workload and several SM counts, every element is copied
// exactly once, every copy stays inside its matrix, holds at most one stage,
// starts on a 16-byte boundary and has a size that is a multiple of 16 bytes
// (the bulk-copy rules), row pairs stay whole within one CTA, and deferred
// partials fit the shared scratch. Also the attention split (att_split): the
// chunks of every position cover positions 0..pos exactly, none is empty or
// longer than the score scratch, and with B sequences no head gets more
// chunks than the record buffer holds. Prints "ok <plans>" or FAIL lines.
#include <algorithm>
#include <cstdio>
#include <utility>
#include <vector>

#include "../paper_2601_03324_gb300/csrc/decode_kernel.cuh"

using namespace tvl;

static int fails = 0;
static long long nplans = 0;
#define CHECK(c, ...)                                            \
  do {                                                           \
    if (!(c)) {                                                  \
      if (fails++ < 20) {                                        \
        printf("FAIL line %d: ", __LINE__);                      \
        printf(__VA_ARGS__);                                     \
        printf("\n");                                            \
      }                                                          \
    }                                                            \
  } while (0)

// An [M x K] matrix of 4-byte words streamed by G CTAs with row granule gran;
// B input vectors share the deferred-partial scratch.
static void check(const char* what, long long M, int K, int G, int gran, int B) {
  std::vector<std::vector<std::pair<int, int>>> cols((size_t)M);
  long long expect_r0 = 0;
  for (int c = 0; c < G; ++c) {
    const StagePlan p = plan_stages(M, K, G, c, gran);
    ++nplans;
    CHECK(p.r0 == expect_r0, "%s G=%d c=%d: r0 %d, expected %lld", what, G, c, p.r0, expect_r0);
    CHECK(p.r1 >= p.r0 && p.r1 <= M, "%s G=%d c=%d: rows [%d, %d)", what, G, c, p.r0, p.r1);
    expect_r0 = p.r1;
    if (gran == 2) CHECK(p.r0 % 2 == 0 && p.r1 % 2 == 0, "%s: pair split across CTAs", what);
    if (p.defer)
      CHECK((long long)(p.r1 - p.r0) * p.spr * B <= kMaxSegParts,
            "%s G=%d c=%d B=%d: %d deferred partials > %d", what, G, c, B,
            (p.r1 - p.r0) * p.spr * B, kMaxSegParts);
    long long rows_seen = 0;
    for (int j = 0; j < p.nstages; ++j) {
      const StageDesc s = stage_desc(p, j);
      const long long bytes = 4LL * s.nrows * (s.c1 - s.c0);
      const long long src = 4LL * ((long long)s.row * K + s.c0);
      CHECK(s.nrows >= 1 && s.row >= p.r0 && s.row + s.nrows <= p.r1,
            "%s G=%d c=%d j=%d: rows [%d, %d) outside [%d, %d)", what, G, c, j, s.row,
            s.row + s.nrows, p.r0, p.r1);
      CHECK(s.c0 >= 0 && s.c0 < s.c1 && s.c1 <= K, "%s: columns [%d, %d) of %d", what, s.c0, s.c1,
            K);
      CHECK(bytes <= kStageBytes, "%s: %lld bytes in one stage", what, bytes);
      CHECK(bytes % 16 == 0 && src % 16 == 0, "%s G=%d c=%d j=%d: copy at %lld of %lld bytes",
            what, G, c, j, src, bytes);
      if (s.nrows > 1) CHECK(s.c0 == 0 && s.c1 == K, "%s: several rows, part of a row", what);
      if (gran == 2 && !p.defer)
        CHECK(s.row % 2 == 0 && s.nrows % 2 == 0, "%s: a stage splits a row pair", what);
      for (int r = s.row; r < s.row + s.nrows; ++r) cols[(size_t)r].push_back({s.c0, s.c1});
      if (s.c0 == 0) rows_seen += s.nrows;
    }
    CHECK(rows_seen == p.r1 - p.r0, "%s G=%d c=%d: %lld rows started, %d owned", what, G, c,
          rows_seen, p.r1 - p.r0);
  }
  CHECK(expect_r0 == M, "%s G=%d: rows end at %lld of %lld", what, G, expect_r0, M);
  for (long long r = 0; r < M; ++r) {
    auto& v = cols[(size_t)r];
    std::sort(v.begin(), v.end());
    int at = 0;
    for (auto& iv : v) {
      CHECK(iv.first == at, "%s: row %lld columns from %d, expected %d", what, r, iv.first, at);
      at = iv.second;
    }
    CHECK(at == K, "%s: row %lld covered to %d of %d", what, r, at, K);
  }
}

struct Shape {
  const char* name;
  int d, F, H, Hkv, V;
};

// tvl_gemv's K split for short-and-wide matrices (same rule as gemv.cu).
static int split_for(int M, int K, int G) {
  int S = 1;
  while ((long long)M * S < G && K % (8 * S) == 0 && K / (2 * S) >= 128) S *= 2;
  return S;
}

// The record buffer holds, per (sequence, head), the most chunks one sequence's
// head gets at any position (the arena's rule).
static int nch_cap_for(int S, int H, int G) {
  int cap = 1;
  for (int pos = 0; pos < S; ++pos) {
    int nch, clen;
    att_split(pos, H, G, &nch, &clen);
    cap = std::max(cap, nch);
  }
  return cap;
}

static void check_attention(int S, int H, int G) {
  const int cap = nch_cap_for(S, H, G);
  for (int B = 1; B <= 4; ++B)
    for (int pos = 0; pos < S; ++pos) {
      int nch, clen;
      att_split(pos, H * B, G, &nch, &clen);
      CHECK(nch >= 1 && nch <= cap, "S=%d H=%d G=%d B=%d pos=%d: %d chunks, capacity %d", S, H, G,
            B, pos, nch, cap);
      CHECK(clen >= 1 && clen <= kAttMaxChunk, "pos=%d: chunk of %d positions", pos, clen);
      int covered = 0;
      for (int c = 0; c < nch; ++c) {
        const int t0 = c * clen, t1 = std::min(t0 + clen, pos + 1);
        CHECK(t0 == covered && t1 > t0, "S=%d H=%d G=%d B=%d pos=%d chunk %d: [%d, %d)", S, H, G,
              B, pos, c, t0, t1);
        covered = t1;
      }
      CHECK(covered == pos + 1, "pos=%d: chunks end at %d", pos, covered);
      ++nplans;
    }
}

int main() {
  const Shape shapes[] = {{"tiny", 288, 768, 6, 6, 32000},     {"110m", 768, 2048, 12, 12, 32000},
                          {"7b", 4096, 11008, 32, 32, 32000},  {"small", 64, 96, 4, 4, 1000},
                          {"small_gqa", 64, 96, 4, 2, 1000},    {"hd128", 128, 256, 1, 1, 1000}};
  const int Gs[] = {152, 148, 132, 8};
  char what[160];
  for (const Shape& sh : shapes) {
    const int kvd = sh.Hkv * (sh.d / sh.H);
    // float32 rows, then 8-bit rows (4 + K/4 words), then 4-bit rows (4 + K/8 words)
    for (int fmt = 0; fmt < 3; ++fmt) {
      if (fmt == 1 && (sh.d % 16 || sh.F % 16)) continue;
      if (fmt == 2 && (sh.d % 32 || sh.F % 32)) continue;
      const int kd = fmt == 0 ? sh.d : fmt == 1 ? 4 + sh.d / 4 : 4 + sh.d / 8;
      const int kf = fmt == 0 ? sh.F : fmt == 1 ? 4 + sh.F / 4 : 4 + sh.F / 8;
      const long long Ms[5] = {sh.d + 2LL * kvd, sh.d, 2LL * sh.F, sh.d, sh.V};
      const int Ks[5] = {kd, kd, kd, kf, kd};
      for (int G : Gs)
        for (int B = 1; B <= (fmt == 0 ? 4 : 1); ++B) {
          // tvl_load refuses a model whose deferred partials could overflow the
          // scratch (its bound: one row more than a CTA's share); skip those
          bool accepted = true;
          for (int i = 0; i < 5; ++i) {
            const StagePlan pl = plan_stages(Ms[i], Ks[i], G, 0, i == 2 ? 2 : 1);
            if (pl.defer && ((Ms[i] + G - 1) / G + 1) * pl.spr * B > kMaxSegParts) accepted = false;
          }
          if (!accepted) continue;
          for (int i = 0; i < 5; ++i) {
            snprintf(what, sizeof what, "%s fmt%d phase%d B%d", sh.name, fmt, i, B);
            check(what, Ms[i], Ks[i], G, i == 2 ? 2 : 1, B);
          }
        }
    }
  }
  // standalone GEMV shapes (sweep and tests), with the K split of tvl_gemv
  const int gm[][2] = {{768, 768},  {2048, 768},   {768, 2048},  {32000, 768}, {11008, 4096},
                       {4096, 11008}, {32000, 4096}, {300, 288},   {5, 4096},    {3, 16},
                       {1, 16384},  {7, 128},      {33, 4096},   {4096, 32}};
  for (auto& mk : gm)
    for (int sms : Gs) {
      const int S = split_for(mk[0], mk[1], sms);
      const long long nv = (long long)mk[0] * S;
      const int G = (int)(nv < sms ? nv : sms);
      snprintf(what, sizeof what, "gemv %dx%d S=%d", mk[0], mk[1], S);
      const StagePlan p0 = plan_stages(nv, mk[1] / S, G, 0);
      if (p0.spr > 1 && ((nv + G - 1) / G) * p0.spr > kMaxSegParts) continue;  // per-row kernel
      check(what, nv, mk[1] / S, G, 1, 1);
    }
  const int att[][2] = {{256, 6}, {1024, 12}, {2048, 32}, {64, 4}, {64, 1}, {4096, 2}};
  for (auto& sh : att)
    for (int G : Gs) check_attention(sh[0], sh[1], G);
  if (fails) {
    printf("%d failures\n", fails);
    return 1;
  }
  printf("ok %lld plans\n", nplans);
  return 0;
}
