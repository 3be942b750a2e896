// Host check of the stage-1 candidate packing (the same __host__ __device__ functions the kernels use): unsigned
// order of packed candidates is the lookup's candidate order (score descending, then entry id ascending), equal
// scores including -0.0 and +0.0 pack alike, and score and id come back out unchanged. Exits non-zero on a failure.
#include <math.h>
#include <stdio.h>

#include "internal.cuh"

static int failures = 0;
#define CHECK(cond)                                                  \
  do {                                                               \
    if (!(cond)) {                                                   \
      fprintf(stderr, "check failed at line %d: %s\n", __LINE__, #cond); \
      ++failures;                                                    \
    }                                                                \
  } while (0)

int main() {
  using namespace lc;
  // ascending scores, the two zeros equal
  const float s[] = {-INFINITY, -1.0f, -0.5f, -1e-30f, -0.0f, 0.0f, 1e-30f, 0.5f, 0.9f, 0.90000004f, 1.0f, INFINITY};
  const int n = (int)(sizeof s / sizeof s[0]);
  for (int i = 0; i + 1 < n; ++i) {
    if (s[i] == s[i + 1])
      CHECK(score_order(s[i]) == score_order(s[i + 1]));
    else
      CHECK(score_order(s[i]) < score_order(s[i + 1]));
  }
  CHECK(score_order(-0.0f) == score_order(0.0f));
  for (int i = 0; i < n; ++i) {
    for (uint32_t j : {0u, 1u, 7u, 123456u, 0x7FFFFFFEu}) {
      const uint64_t c = pack_cand(s[i], j);
      CHECK(c != 0);                                  // 0 marks an empty slot
      CHECK(cand_id(c) == j);
      const float back = cand_score(c);
      CHECK(back == s[i]);                            // -0.0 comes back as +0.0, which compares equal
      CHECK(pack_cand(s[i], j) > pack_cand(s[i], j + 1));   // equal scores: the lower id first
      if (i + 1 < n && s[i] < s[i + 1]) CHECK(pack_cand(s[i + 1], 0x7FFFFFFEu) > pack_cand(s[i], 0u));
    }
  }
  CHECK(pack_cand(-0.0f, 5) == pack_cand(0.0f, 5));
  CHECK(pack_cand(-0.0f, 4) > pack_cand(0.0f, 5));
  if (failures) return 1;
  printf("candidate packing: ok\n");
  return 0;
}
