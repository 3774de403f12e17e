"""Planted mistakes for the mutation test of the oracle's pins
(tests/test_pins_mutants.py). Each entry is one plausible mistake in the
oracle (oracle/awsrc_oracle.c), written as text edits: every (old, new) pair
replaces one occurrence of `old` in the oracle's source with `new`. The
mutation test applies the edits to a copy of the source, builds that copy and
requires the pin files to fail against it. The oracle itself carries none of
them."""


MUTANTS = {
    1: ('Gram off-diagonal sums with the sign of the atom product flipped', [
        ("""        sv += (negmask[p * C + j] ^ negmask[q * C + j]) ? -(int64_t)Dq[j] : (int64_t)Dq[j];
""",
         """        sv += (negmask[p * C + j] ^ negmask[q * C + j]) ? (int64_t)Dq[j] : -(int64_t)Dq[j];
"""),
    ]),
    2: ('Gram off-diagonal sums taking a wrong atom index', [
        ("""        sv += (negmask[p * C + j] ^ negmask[q * C + j]) ? -(int64_t)Dq[j] : (int64_t)Dq[j];
""",
         """        sv += (negmask[p * C + j] ^ negmask[p * C + (j ^ 1)]) ? -(int64_t)Dq[j] : (int64_t)Dq[j];
"""),
    ]),
    3: ('b = B^T D r without the C^-1/2 normalisation', [
        ("""    bvec[p] = c * u;
""",
         """    bvec[p] = u;
"""),
    ]),
    4: ('power-of-two scale exponent one too large', [
        ("""    int e = e0 + (amax > ldexpf((float)qmax, e0) ? 1 : 0);
""",
         """    int e = e0 + (amax > ldexpf((float)qmax, e0) ? 1 : 0) + 1;
"""),
    ]),
    5: ('ridge eps absolute instead of relative to mean(d)', [
        ("""  float eps = prm->ridge_rel * gd;
""",
         """  float eps = prm->ridge_rel;
"""),
    ]),
    6: ('Eq. 4 gain without the factor 2 on alpha^T b', [
        ("""  float g = sc * (2.0f * Aq - t);
""",
         """  float g = sc * (Aq - t);
"""),
    ]),
    7: ('seed ties keep the larger selector', [
        ("""        if (g > best.gain) {
""",
         """        if (g >= best.gain) {
"""),
    ]),
    8: ('records with equal gains ordered by tile descending', [
        ("""  return (x->tile > y->tile) - (x->tile < y->tile);  /* ties: tile ascending */
""",
         """  return (x->tile < y->tile) - (x->tile > y->tile);
"""),
    ]),
    9: ('progressive prefix one record longer than the budget allows', [
        ("""      int64_t K = (B - h) / L;
""",
         """      int64_t K = (B - h) / L + 1;
"""),
    ]),
    10: ('record width rounded up one byte too far', [
        ("""  return (bits + 7) / 8;
""",
         """  return (bits + 8) / 8;
"""),
    ]),
    11: ('decoder adds half the correction', [
        ("""      float rh = ((float)kj * c) * sc;
""",
         """      float rh = ((float)kj * c) * (0.5f * sc);
"""),
    ]),
    12: ('Fisher-Yates permutation draw range one short', [
        ("""      int k = (int)((x * (uint64_t)(i + 1)) >> 32);
""",
         """      int k = (int)((x * (uint64_t)i) >> 32);
"""),
    ]),
    13: ('Hadamard entry sign from OR instead of AND', [
        ("""      negmask[p * C + j] = (uint8_t)((sign[j] + orc_popcount((uint32_t)(perm[j] & cols[p]))) & 1);
""",
         """      negmask[p * C + j] = (uint8_t)((sign[j] + orc_popcount((uint32_t)(perm[j] | cols[p]))) & 1);
"""),
    ]),
    14: ('RTN group scale max|w| / 8 instead of / 7', [
        ("""    const uint16_t h = orc_f32_to_f16(amax / 7.0f);
""",
         """    const uint16_t h = orc_f32_to_f16(amax / 8.0f);
"""),
    ]),
    15: ('SDQ step max deviation / 128 instead of / 127', [
        ("""      const float step = a / 127.0f;
""",
         """      const float step = a / 128.0f;
"""),
    ]),
    16: ('forward substitution dropping its last term', [
        ("""    for (int i = 0; i < k; ++i) v = fmaf(-L[k][i], z[i], v);
""",
         """    for (int i = 0; i < k - 1; ++i) v = fmaf(-L[k][i], z[i], v);
"""),
    ]),
    17: ('fixed-point grid one bit coarser', [
        ("""  int q = ilogbf(m) - 20;
""",
         """  int q = ilogbf(m) - 19;
"""),
    ]),
    18: ('record fields packed seed before tile', [
        ("""  orc_put_bits(rec, &pos, (uint64_t)tile, orc_ceil_log2((uint64_t)T));
  orc_put_bits(rec, &pos, cd->seed, orc_ceil_log2((uint64_t)prm->S));
""",
         """  orc_put_bits(rec, &pos, cd->seed, orc_ceil_log2((uint64_t)prm->S));
  orc_put_bits(rec, &pos, (uint64_t)tile, orc_ceil_log2((uint64_t)T));
"""),
    ]),
    19: ('packed GEMV subtracting the sidecar correction', [
        ("""      Rt[base + j] = (double)kj * c * sc;  /* a later record of the tile replaces it */
""",
         """      Rt[base + j] = -(double)kj * c * sc;  /* a later record of the tile replaces it */
"""),
    ]),
    20: ('sign word bits read most-significant first', [
        ("""    for (int j = w * 64; j < C && j < w * 64 + 64; ++j) sign[j] = (uint8_t)((word >> (j - w * 64)) & 1u);
""",
         """    for (int j = w * 64; j < C && j < w * 64 + 64; ++j) sign[j] = (uint8_t)((word >> (63 - (j - w * 64))) & 1u);
"""),
    ]),
    21: ('P_F Fisher term read without the column block offset', [
        ("""    else d[j] = w_act * a + w_fisher * fisher[idx];
""",
         """    else d[j] = w_act * a + w_fisher * fisher[row * cols + j];
"""),
    ]),
    22: ('residual taken as W0 - W', [
        ("""    r[j] = W[idx] - W0[idx];
""",
         """    r[j] = W0[idx] - W[idx];
"""),
    ]),
    23: ('codes clamped to [-qmax - 1, qmax] when the exponent field clips', [
        ("""      float q = rintf(alpha[p] * inv);
      if (q > (float)qmax) q = (float)qmax;
      if (q < (float)-qmax) q = (float)-qmax;
""",
         """      float q = rintf(alpha[p] * inv);
      if (q > (float)qmax) q = (float)qmax;
      if (q < (float)(-qmax - 1)) q = (float)(-qmax - 1);
"""),
    ]),
    24: ('U quotas shared out of B instead of B - h', [
        ("""      unsigned __int128 q = (unsigned __int128)(uint64_t)(B - h) * (uint64_t)mod_weights[m];
""",
         """      unsigned __int128 q = (unsigned __int128)(uint64_t)B * (uint64_t)mod_weights[m];
"""),
    ]),
    25: ('binary16 scale max|alpha| / (qmax + 1)', [
        ("""    uint16_t h = orc_f32_to_f16(amax / (float)qmax);
""",
         """    uint16_t h = orc_f32_to_f16(amax / (float)(qmax + 1));
"""),
    ]),
    26: ('SDQ mean of a short last block divided by the full block size', [
        ("""      const float mu = (float)(sum / (double)n);
""",
         """      const float mu = (float)(sum / (double)block);
"""),
    ]),
    27: ('fixed-point grid values truncated instead of rounded', [
        ("""  for (int j = 0; j < C; ++j) X[j] = (int32_t)rintf(ldexpf(x[j], -q));
""",
         """  for (int j = 0; j < C; ++j) X[j] = (int32_t)ldexpf(x[j], -q);
"""),
    ]),
    28: ('P_F prefixes taken out of B instead of B - h', [
        ("""      int64_t K = (B - h) / L;
""",
         """      int64_t K = B / L;
"""),
    ]),
    29: ('Eq. 4 gain with the ridge in G', [
        ("""    Qq = fmaf((float)(codes[p] * codes[p]), G[p][p], Qq);
""",
         """    Qq = fmaf((float)(codes[p] * codes[p]), A[p][p], Qq);
"""),
    ]),
    30: ('decoder normalising by 1/C instead of C^-1/2', [
        ("""  const float c = (float)(1.0 / sqrt((double)C));
""",
         """  const float c = (float)(1.0 / (double)C);
"""),
    ]),
    31: ('scale field holding e + e_bias', [
        ("""  if (prm->scale_mode == 0) sf = (uint64_t)(int64_t)(cd->scale - prm->e_bias);
""",
         """  if (prm->scale_mode == 0) sf = (uint64_t)(int64_t)(cd->scale + prm->e_bias);
"""),
    ]),
    32: ('decoder adding a record to the next column block', [
        ("""    int64_t base = (lt / n_cb) * mod_cols[m] + (lt % n_cb) * C;
""",
         """    int64_t base = (lt / n_cb) * mod_cols[m] + ((lt + 1) % n_cb) * C;
"""),
    ]),
    33: ('byte budget rounded up', [
        ("""  return (int64_t)floor(rate_bpw * (double)n_scope / 8.0);
""",
         """  return (int64_t)ceil(rate_bpw * (double)n_scope / 8.0);
"""),
    ]),
    34: ('SDQ step from the largest deviation above the mean only', [
        ("""        const float d = fabsf(s_eff[g] - mu);
""",
         """        const float d = s_eff[g] - mu;
"""),
    ]),
    35: ('seed key taken from stream output s instead of s + 1', [
        ("""  uint64_t key = orc_splitmix64_output(gen_seed, (uint64_t)s + 1);
""",
         """  uint64_t key = orc_splitmix64_output(gen_seed, (uint64_t)s);
"""),
    ]),
    36: ('coordinate permutation applied inverted', [
        ("""  /* B_s[j][p] = C^-1/2 * sigma_j * H[pi(j), c_p],  H[i][k] = (-1)^popcount(i & k) */
""",
         """  /* B_s[j][p] = C^-1/2 * sigma_j * H[pi(j), c_p],  H[i][k] = (-1)^popcount(i & k) */
  {
    int32_t inv[256];
    for (int j = 0; j < C; ++j) inv[perm[j]] = j;
    for (int j = 0; j < C; ++j) perm[j] = inv[j];
  }
"""),
    ]),
    37: ('Hadamard columns drawn with replacement', [
        ("""    int k = p + (int)((x * (uint64_t)(C - p)) >> 32);
    int32_t t = pool[p]; pool[p] = pool[k]; pool[k] = t;
    cols[p] = pool[p];
""",
         """    cols[p] = (int)((x * (uint64_t)C) >> 32);
    (void)pool;
"""),
    ]),
    38: ('candidates with a zero gain kept', [
        ("""    if (cands[t].gain > 0.0f && cands[t].gain <= FLT_MAX) { keys[npos].gain = cands[t].gain; keys[npos].tile = t; ++npos; }
""",
         """    if (cands[t].gain >= 0.0f && cands[t].gain <= FLT_MAX) { keys[npos].gain = cands[t].gain; keys[npos].tile = t; ++npos; }
"""),
    ]),
    39: ('decoder dropping the last of its K records', [
        ("""  int32_t perm[256], cols[8];
  int bad = 0;
  for (int64_t k = 0; k < K; ++k) {
""",
         """  int32_t perm[256], cols[8];
  int bad = 0;
  for (int64_t k = 0; k < K - 1; ++k) {
"""),
    ]),
    40: ('BF16 output truncated instead of rounded to nearest even', [
        ("""  uint32_t lsb = (x >> 16) & 1u;
  return (uint16_t)((x + 0x7fffu + lsb) >> 16);
""",
         """  return (uint16_t)(x >> 16);
"""),
    ]),
    41: ('U quotas rounded up', [
        ("""      int64_t quota = (int64_t)(q / (uint64_t)Nscope);
""",
         """      int64_t quota = (int64_t)((q + (uint64_t)Nscope - 1) / (uint64_t)Nscope);
"""),
    ]),
    42: ('RTN codes from the product with the rounded reciprocal of the scale', [
        ("""        v = rintf(w[j] / s);
""",
         """        v = rintf(w[j] * (1.0f / s));
"""),
    ]),
    43: ('packed GEMV adding both records of a tile named twice', [
        ("""      Rt[base + j] = (double)kj * c * sc;  /* a later record of the tile replaces it */
""",
         """      Rt[base + j] += (double)kj * c * sc;  /* a later record of the tile replaces it */
"""),
    ]),
    44: ('packed GEMV magnitude of the summed weight instead of its two terms', [
        ("""        aabs += fabs(Wt[i * cols + j] * xj) + fabs(Rt[i * cols + j] * xj);
""",
         """        aabs += fabs((Wt[i * cols + j] + Rt[i * cols + j]) * xj);
"""),
    ]),
}
