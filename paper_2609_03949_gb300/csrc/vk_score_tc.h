// vk_score_tc.h -- arguments of the tcgen05 scoring kernel (host and device).
#pragma once
#include <stdint.h>

namespace vk {

struct ScoreTcArgs {
  // filled by the launcher
  int B, H, N, n_rows, tiles_per_seq, n_pages;
  int64_t total_tiles;
  uint32_t tmem_cols;
  // epilogue mode: 0 dense scores, 1 threshold candidates, 2 trigger
  int mode;
  // mode 0: scores[(b*H + h) * scores_ld + row], fp32; or, with scores_bf16, bf16 (rounded to nearest even)
  float* scores;
  int64_t scores_ld;
  int scores_bf16;
  // modes 1, 2: archive [arch_lo, arch_hi) in positions
  int arch_lo, arch_hi;
  // mode 1: emit rows with a >= theta[b*H + h]
  const float* theta;
  // modes 1, 2 (top_j > 0): candidate lists cand[(b*H + h) * capc + i] = (u, score bits), counts cand_cnt[b*H + h]
  int* cand_cnt;
  int2* cand;
  int capc;
  // mode 2: trigger T = lam * (a + qrn * page_res[page] + z * qcn * eta[u]) > smax1, u not in selbm
  const float *qcn, *qrn, *eta, *page_res, *smax1;
  float lam, z;
  const uint32_t* selbm;
  uint32_t* firebm;
  int64_t nw;
  int top_j;
  // mode 2 page skip (when page_knorm != NULL): a 128-row tile is neither loaded nor multiplied when, for every head
  // and both of its pages, lam * (qrf * page_knorm + z * qcn * page_eta) cannot reach smax1 (page_may_fire)
  const float *qrf, *page_knorm, *page_eta;
  // mode 2 content sketch (r_sk in {16, 32, 64}, r = 64, H <= 128): sketch rows [B][N][r_sk] bf16 and the query's bf16
  // high and low parts of p = V^T Qc, [B][2][H][r_sk]; qcn then holds the sketch residual norms of the queries
  int r_sk;
  const void *sketch, *sketch_q;
  // mode 2, set by the launcher: the producer stages each tile's eta rows in shared memory by TMA (N % 4 == 0)
  int eta_tma;
  int* status;
};

}  // namespace vk
