"""The C ABI used from C alone (no Python, no PyTorch): a program linked against
liblv.so and the CUDA runtime creates a pool over its own cudaMalloc'd KV arrays,
ranks, swaps out, commits, checks the bytes in the host pool, reloads and checks
the bytes in HBM; then frees pages with lv_evict and runs one lv_turn whose load
keys set the reload order."""
import os
import subprocess

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PKG = os.path.join(ROOT, "paper_2606_22983_gb300")

PROGRAM = r'''
#include <stdio.h>
#include <stdint.h>
#include <string.h>
#include <cuda_runtime_api.h>
#include "lv.h"

#define CHECK(x) do { lv_status s_ = (x); if (s_ != LV_OK) { \
  printf("%s failed: %s\n", #x, lv_status_str(s_)); return 1; } } while (0)
#define CUDA(x) do { if ((x) != cudaSuccess) { printf("%s failed\n", #x); return 1; } } while (0)

enum { L = 1, J = 2, T = 16, H = 1, D = 64, PAGES = 64, SLOTS = 64, S = 2, MAXB = 8 };
static const size_t P = (size_t)T * H * D * 2;   /* 2048-byte sub-pages */

int main(void) {
  uint8_t* kv[J];
  for (int j = 0; j < J; ++j) {
    CUDA(cudaMalloc((void**)&kv[j], PAGES * P));
    /* every byte of sub-page j of page p is (p * 2 + j + 1) mod 256 */
    for (int p = 0; p < PAGES; ++p) CUDA(cudaMemset(kv[j] + p * P, (p * 2 + j + 1) & 255, P));
  }
  lv_pool_desc d;
  memset(&d, 0, sizeof d);
  d.num_layers = L; d.num_kv_heads = H; d.head_dim = D; d.page_tokens = T; d.elem_bytes = 2;
  d.max_sessions = S; d.max_blocks = MAXB; d.within_order = LV_SUFFIX_FIRST;
  d.hbm_pages = PAGES; d.hbm_budget_pages = PAGES; d.host_pages = SLOTS;
  d.hbm_kv = (void* const*)kv; d.host_kv = NULL;
  d.reply_prior_us = 3000000; d.protect_us = 2000000; d.unit_us = 80000;
  d.t_play_mode = LV_PLAY_PLAYBACK; d.policy = LV_POLICY_NEXT_USE; d.tiers = LV_TIERS_EXCLUSIVE;
  lv_pool* pool = NULL;
  CHECK(lv_pool_create(&d, NULL, &pool));

  /* session 0: 4 blocks on pages 10..13; session 1: 2 blocks on pages 20, 21 */
  int32_t placement[S * MAXB], ctx[S] = {64, 32};
  for (int i = 0; i < S * MAXB; ++i) placement[i] = -1;
  for (int b = 0; b < 4; ++b) placement[b] = 10 + b;
  placement[MAXB + 0] = 20; placement[MAXB + 1] = 21;
  CHECK(lv_pool_import(pool, placement, ctx, NULL));
  /* session 1 is running: only session 0 is a candidate */
  lv_session_state st[S];
  memset(st, 0, sizeof st);
  st[1].flags = LV_RUNNING;
  CHECK(lv_session_set(pool, st, 0, S, NULL));

  lv_victim v[3];
  int64_t n = 0;
  CHECK(lv_select_victims(pool, 0, 3, 0, v, 3, &n, NULL));
  CHECK(lv_sync(pool, NULL));
  if (n != 3) { printf("victims %lld\n", (long long)n); return 1; }
  /* suffix first: blocks 3, 2, 1 of session 0 */
  for (int i = 0; i < 3; ++i)
    if (v[i].sid != 0 || v[i].blk != 3 - i || v[i].page != 13 - i) { printf("victim %d\n", i); return 1; }

  int32_t slots[3];
  lv_remap_entry commit[3];
  CHECK(lv_swap_out(pool, v, 3, slots, commit, LV_MODE_AUTO, NULL));
  CHECK(lv_remap(pool, commit, 3, NULL));
  CHECK(lv_sync(pool, NULL));
  const uint8_t* host = (const uint8_t*)lv_pool_host_ptr(pool);
  for (int i = 0; i < 3; ++i) {
    if (slots[i] != i) { printf("slot %d = %d\n", i, slots[i]); return 1; }
    for (int j = 0; j < J; ++j) {
      const uint8_t* sub = host + ((size_t)slots[i] * J + j) * P;
      const uint8_t want = (uint8_t)((v[i].page * 2 + j + 1) & 255);
      for (size_t b = 0; b < P; ++b)
        if (sub[b] != want) { printf("host byte %d/%d/%zu\n", i, j, b); return 1; }
    }
  }
  lv_stats stats;
  CHECK(lv_get_stats(pool, &stats, NULL));
  if (stats.pages_out != 3 || stats.host_allocated != 3 || stats.hbm_allocated != 3) {
    printf("stats %lld %lld %lld\n", (long long)stats.pages_out, (long long)stats.host_allocated,
           (long long)stats.hbm_allocated);
    return 1;
  }

  /* reload the three blocks (ascending) into fresh pages; their bytes come back */
  int32_t blks[3] = {1, 2, 3}, pages[3];
  CHECK(lv_swap_in(pool, 0, blks, 3, pages, commit, LV_MODE_AUTO, NULL));
  CHECK(lv_remap(pool, commit, 3, NULL));
  CHECK(lv_sync(pool, NULL));
  uint8_t sub[2048];
  for (int i = 0; i < 3; ++i) {
    if (pages[i] != i) { printf("page %d = %d\n", i, pages[i]); return 1; }
    for (int j = 0; j < J; ++j) {
      CUDA(cudaMemcpy(sub, kv[j] + (size_t)pages[i] * P, P, cudaMemcpyDeviceToHost));
      const uint8_t want = (uint8_t)(((11 + i) * 2 + j + 1) & 255);   /* block 1+i was on page 11+i */
      for (size_t b = 0; b < P; ++b)
        if (sub[b] != want) { printf("hbm byte %d/%d/%zu\n", i, j, b); return 1; }
    }
  }
  int32_t tables[S * MAXB];
  CHECK(lv_read_tables(pool, tables, NULL, NULL, NULL));
  CHECK(lv_sync(pool, NULL));
  if (tables[0] != 10 || tables[1] != 0 || tables[2] != 1 || tables[3] != 2) { printf("tables\n"); return 1; }

  /* free 2 pages now on the device: the suffix of session 0 (session 1 runs) */
  static lv_victim ev[PAGES];
  static int32_t evs[PAGES];
  lv_resident_result res;
  CHECK(lv_evict(pool, 0, 2, 0, ev, evs, &res, NULL));
  CHECK(lv_sync(pool, NULL));
  if (res.status != LV_RESIDENT_DONE || res.n_victims != 2 || ev[0].sid != 0 || ev[0].blk != 3 ||
      ev[1].blk != 2 || evs[0] != 0 || evs[1] != 1) { printf("evict\n"); return 1; }

  /* one turn of session 0 whose load keys reverse its host blocks: block 3 loads first and
     takes the lowest free page (1), block 2 the next (2) */
  static uint64_t keys[MAXB];
  for (int b = 0; b < MAXB; ++b) keys[b] = (uint64_t)(MAXB - b);
  lv_turn_desc td;
  memset(&td, 0, sizeof td);
  td.sid = 0; td.now_us = 10; td.reply_audio_us = 1000; td.reply_units = 1; td.load_keys = keys;
  int32_t tblocks[MAXB], tpages[MAXB];
  CHECK(lv_turn(pool, &td, NULL, NULL, tblocks, tpages, NULL, &res, NULL));
  CHECK(lv_sync(pool, NULL));
  if (res.status != LV_RESIDENT_DONE || res.n_loaded != 2 || res.sid != 0 || tblocks[0] != 3 ||
      tblocks[1] != 2 || tpages[0] != 1 || tpages[1] != 2) { printf("turn\n"); return 1; }
  for (int i = 0; i < 2; ++i) {
    for (int j = 0; j < J; ++j) {
      CUDA(cudaMemcpy(sub, kv[j] + (size_t)tpages[i] * P, P, cudaMemcpyDeviceToHost));
      const uint8_t want = (uint8_t)(((10 + tblocks[i]) * 2 + j + 1) & 255);   /* block b began on page 10+b */
      for (size_t b = 0; b < P; ++b)
        if (sub[b] != want) { printf("turn byte %d/%d/%zu\n", i, j, b); return 1; }
    }
  }
  CHECK(lv_read_tables(pool, tables, NULL, NULL, NULL));
  CHECK(lv_sync(pool, NULL));
  if (tables[0] != 10 || tables[1] != 0 || tables[2] != 2 || tables[3] != 1) { printf("tables 2\n"); return 1; }
  CHECK(lv_pool_destroy(pool, NULL));
  for (int j = 0; j < J; ++j) CUDA(cudaFree(kv[j]));
  printf("ok\n");
  return 0;
}
'''


def test_c_program_drives_the_abi(tmp_path):
    from paper_2606_22983_gb300 import LIB  # noqa: F401  (builds / locates liblv.so)
    cuda = os.environ.get("CUDA_HOME", "/usr/local/cuda")
    src = tmp_path / "abi_user.c"
    src.write_text(PROGRAM)
    exe = tmp_path / "abi_user"
    subprocess.run(["gcc", "-std=c99", "-Wall", "-Werror", "-I", os.path.join(ROOT, "include"),
                    "-I", os.path.join(cuda, "include"), str(src), "-o", str(exe),
                    "-L", PKG, "-llv", "-L", os.path.join(cuda, "lib64"), "-lcudart",
                    f"-Wl,-rpath,{PKG}", f"-Wl,-rpath,{os.path.join(cuda, 'lib64')}"], check=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True, timeout=120)
    assert out.returncode == 0 and out.stdout.strip().endswith("ok"), out.stdout + out.stderr
