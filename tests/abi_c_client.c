/* A plain C99 client of include/chameleon.h: the header compiles as C, the library links from C,
 * and the host-only entry points (no GPU needed) answer as the header documents.  Built and run
 * by tests/test_abi_c.py; prints "ok" and exits 0, or names the first failed check and exits 1. */
#include <stdio.h>
#include <string.h>

#include "chameleon.h"

static int failures = 0;

#define CHECK(cond)                                          \
  do {                                                       \
    if (!(cond)) {                                           \
      printf("failed: %s (line %d)\n", #cond, __LINE__);     \
      ++failures;                                            \
    }                                                        \
  } while (0)

int main(void) {
  /* layouts shared with the Python binding */
  CHECK(sizeof(cham_wpack_desc) == 256);
  CHECK(sizeof(cham_qparams) == 16);
  CHECK(chameleon_version() == 3);
  CHECK(chameleon_status_string(CHAM_ERR_WORKSPACE) != NULL);

  /* Alg. 2 / Alg. 3 bucket: b = min(floor(t / (T/B)), B-1) */
  CHECK(chameleon_bucket(0, 1000, 10) == 0);
  CHECK(chameleon_bucket(99, 1000, 10) == 0);
  CHECK(chameleon_bucket(100, 1000, 10) == 1);
  CHECK(chameleon_bucket(999, 1000, 10) == 9);
  CHECK(chameleon_bucket(-1, 1000, 10) == -1);

  /* SNR(t) of the scaled-linear schedule falls monotonically with t */
  {
    static double snr[1000];
    int t, monotone = 1;
    CHECK(chameleon_snr(CHAM_SCHEDULE_SCALED_LINEAR, 1000, snr) == CHAM_OK);
    for (t = 1; t < 1000; ++t) monotone &= snr[t] < snr[t - 1];
    CHECK(monotone);
    CHECK(snr[999] > 0.0);
  }

  /* ScaleZP: E4M3 takes s = amax / 448 with z = 0; a reversed range is rejected */
  {
    cham_qparams p;
    const float s = 4.0f / 448.0f;
    memset(&p, 0, sizeof p);
    CHECK(chameleon_scale_zp(CHAM_A_E4M3, -2.0f, 4.0f, &p) == CHAM_OK);
    CHECK(p.s == s && p.z == 0 && p.fmt == CHAM_A_E4M3);
    CHECK(chameleon_scale_zp(CHAM_A_INT8_ASYM, 1.0f, -1.0f, &p) == CHAM_ERR_INVALID_ARG);
    CHECK(chameleon_last_error_detail() != NULL);
  }

  /* pack plan of 256 x 320 INT8-sym weights: one MMA class, two 128-channel tiles */
  {
    static uint8_t fmt[256];
    cham_wpack_desc d;
    memset(fmt, CHAM_W_INT8_SYM, sizeof fmt);
    CHECK(chameleon_pack_plan(256, 320, fmt, &d) == CHAM_OK);
    CHECK(d.magic == 0x574D4843u && d.version == 3 && d.N == 256 && d.K == 320 && d.Kp == 320);
    CHECK(d.bits == 8 && d.n_tiles[0] + d.n_tiles[1] == 2 && d.n_fmt[CHAM_W_INT8_SYM] == 256);
    CHECK(d.bytes > (uint64_t)256 * 320 && d.off_codes % 256 == 0);
  }

  /* size queries */
  {
    size_t q = 0, w = 0;
    CHECK(chameleon_act_quant_size(16, 64, CHAM_A_E4M3, &q, &w) == CHAM_OK);
    CHECK(q >= 16 * 64);
    CHECK(chameleon_act_quant_size(16, 48, CHAM_A_E4M3, &q, &w) == CHAM_ERR_INVALID_ARG);
  }

  if (failures == 0) printf("ok\n");
  return failures == 0 ? 0 : 1;
}
