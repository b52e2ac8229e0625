"""GPU parity of intent / advance / pull / push / sync against the CPU oracle.

Every test drives the CUDA path through the C ABI (ctypes binding) and the
oracle with the same seeded call sequence and compares:
  * bit-exact: replica key sets (the logical slot map), intent refcounts,
    pulled rows, and - with dyadic deltas, whose sums are exact in any
    order - replica values, pending updates and the main store;
  * with gaussian deltas: |gpu - oracle| <= 1e-5 * M + 1e-30 per element,
    M = the same quantity computed on |init| and |deltas| (the sum of the
    magnitudes of every contribution to that element).
Sizes span several sort sub-tiles, many push chunks and ragged tails.
"""
import numpy as np
import pytest
import torch

from oracle import ParameterManagerOracle
from tests.golden_util import load_scenarios
from tests.seqgen import dyadic_init, random_sequence

pytestmark = pytest.mark.gpu

RTOL = 1e-5


def make_pair(gpu_lib, K, D, W, init, capacity=0):
    pm = gpu_lib.ParameterManager(K, D, W, replica_capacity=capacity,
                                  init_values=torch.from_numpy(init).cuda())
    ref = ParameterManagerOracle(K, D, W, init)
    return pm, ref


def dev(keys):
    return torch.as_tensor(np.asarray(keys, dtype=np.int64), device="cuda")


def apply_gpu(pm, op):
    kind = op["op"]
    if kind == "intent":
        pm.intent(op["w"], dev(op["keys"]), op["start"], op["end"])
    elif kind == "advance":
        pm.advance_clock(op["w"])
    elif kind == "pull":
        out = pm.pull(op["w"], dev(op["keys"]))
        torch.cuda.synchronize()
        return out.cpu().numpy()
    elif kind == "push":
        pm.push(op["w"], dev(op["keys"]), torch.from_numpy(np.ascontiguousarray(op["deltas"])).cuda())
    elif kind == "sync":
        pm.sync()
    return None


def apply_ref(ref, op):
    kind = op["op"]
    if kind == "intent":
        ref.intent(op["w"], op["keys"], op["start"], op["end"])
    elif kind == "advance":
        ref.advance_clock(op["w"])
    elif kind == "pull":
        return ref.pull(op["w"], op["keys"])
    elif kind == "push":
        ref.push(op["w"], op["keys"], op["deltas"])
    elif kind == "sync":
        ref.sync()
    return None


def compare_full_state(pm, ref, K, W, exact=True, mag=None):
    keys = np.arange(K)
    pm.wait()
    for w in range(W):
        assert np.array_equal(pm.replica_keys(w), ref.replica_keys(w)), f"replica set of worker {w}"
        assert np.array_equal(pm.refcounts(w, keys), ref.refcounts(w, keys)), f"refcounts of worker {w}"
        val, acc, has = pm.replica_rows(w, keys)
        rk, rval, racc = ref.replica_values(w)
        assert np.array_equal(np.nonzero(has)[0], rk)
        if exact:
            assert np.array_equal(val[rk], rval) and np.array_equal(acc[rk], racc)
        else:
            mv, ma = mag.replica_values(w)[1:]
            assert np.all(np.abs(val[rk] - rval) <= RTOL * mv + 1e-30)
            assert np.all(np.abs(acc[rk] - racc) <= RTOL * ma + 1e-30)
    main = pm.read_main(keys)
    if exact:
        assert np.array_equal(main, ref.main)
    else:
        assert np.all(np.abs(main - ref.main) <= RTOL * mag.main + 1e-30)


CASES = [
    # K, D, W, max_batch, n_ops
    (40, 4, 3, 12, 160),
    (300, 16, 4, 700, 60),
    (5000, 64, 3, 6000, 40),      # several sort sub-tiles, ragged tails, many push chunks
    (900, 200, 2, 2500, 30),
    (700, 300, 2, 1500, 25),
    (500, 512, 2, 1200, 25),
    (200, 1024, 2, 600, 20),
]


@pytest.mark.parametrize("K,D,W,max_batch,n_ops", CASES)
@pytest.mark.parametrize("seed", [0, 1])
def test_random_sequences_dyadic_bit_exact(gpu_lib, K, D, W, max_batch, n_ops, seed):
    init = dyadic_init(K, D, seed)
    pm, ref = make_pair(gpu_lib, K, D, W, init)
    ops = random_sequence(seed * 31 + K, K, D, W, n_ops, max_batch=max_batch)
    for i, op in enumerate(ops):
        got = apply_gpu(pm, op)
        want = apply_ref(ref, op)
        if op["op"] == "pull":
            assert np.array_equal(got, want), f"pull {i}"
        if op["op"] in ("intent", "advance") and K <= 300:
            w = op["w"]
            assert np.array_equal(pm.replica_keys(w), ref.replica_keys(w)), f"op {i}"
    compare_full_state(pm, ref, K, W)
    pm.sync()
    ref.sync()
    compare_full_state(pm, ref, K, W)
    pm.close()


@pytest.mark.parametrize("K,D,W", [(64, 8, 3), (2000, 64, 4)])
def test_random_sequences_gaussian_within_tolerance(gpu_lib, K, D, W):
    rng = np.random.default_rng(K)
    init = rng.normal(0, 0.1, size=(K, D)).astype(np.float32)
    pm, ref = make_pair(gpu_lib, K, D, W, init)
    mag = ParameterManagerOracle(K, D, W, np.abs(init))
    ops = random_sequence(K + 7, K, D, W, 80, max_batch=3000, gaussian=True)
    for op in ops:
        got = apply_gpu(pm, op)
        want = apply_ref(ref, op)
        mop = dict(op)
        if op["op"] == "push":
            mop["deltas"] = np.abs(op["deltas"])
        m = apply_ref(mag, mop)
        if op["op"] == "pull":
            assert np.all(np.abs(got - want) <= RTOL * m + 1e-30)
    compare_full_state(pm, ref, K, W, exact=False, mag=mag)
    pm.close()


def test_golden_scenarios_on_gpu(gpu_lib):
    g, scenarios = load_scenarios()
    for sc in scenarios:
        init = np.array(g["init"], dtype=np.float32)
        pm = gpu_lib.ParameterManager(g["num_keys"], 4, g["num_workers"], replica_capacity=16,
                                      init_values=torch.from_numpy(np.pad(init, ((0, 0), (0, 2)))).cuda())
        for i, st in enumerate(sc["steps"]):
            where = f"{sc['name']} step {i}"
            op = st["op"]
            if op == "intent":
                pm.intent(st["w"], dev(st["keys"]), st["start"], st["end"])
            elif op == "advance":
                pm.advance_clock(st["w"])
            elif op == "push":
                d = np.pad(np.array(st["deltas"], dtype=np.float32), ((0, 0), (0, 2)))
                pm.push(st["w"], dev(st["keys"]), torch.from_numpy(d).cuda())
            elif op == "sync":
                pm.sync()
            elif op == "pull":
                out = pm.pull(st["w"], dev(st["keys"])).cpu().numpy()[:, :2]
                assert out.tolist() == st["expect"], where
            elif op == "main":
                assert pm.read_main(st["keys"])[:, :2].tolist() == st["expect"], where
            elif op == "replica_keys":
                assert pm.replica_keys(st["w"]).tolist() == st["expect"], where
            elif op == "refcounts":
                assert pm.refcounts(st["w"], st["keys"]).tolist() == st["expect"], where
        pm.wait()
        pm.close()


def test_hot_key_spanning_many_chunks_and_determinism(gpu_lib):
    # one key is 40% of a 60k batch: its segment spans hundreds of push chunks
    K, D, W, n = 5000, 16, 2, 60000
    rng = np.random.default_rng(3)
    init = dyadic_init(K, D, 3)
    keys = rng.integers(0, K, size=n)
    keys[rng.random(n) < 0.4] = 1234
    d = (rng.integers(-64, 65, size=(n, D)) * 2.0 ** -10).astype(np.float32)
    for with_replica in (False, True):
        pm, ref = make_pair(gpu_lib, K, D, W, init)
        if with_replica:
            for api in (pm, ref):
                api.intent(1, np.unique(keys)[::2], 0, 3)
        for api in (pm, ref):
            api.push(1, keys, d)
        compare_full_state(pm, ref, K, W)
        pm.close()
    # gaussian deltas: two identical pushes give identical bits
    g = rng.normal(0, 1e-3, size=(n, D)).astype(np.float32)
    outs = []
    for _ in range(2):
        pm = gpu_lib.ParameterManager(K, D, W, init_values=torch.from_numpy(init).cuda())
        pm.push(0, dev(keys), torch.from_numpy(g).cuda())
        outs.append(pm.read_main(np.arange(K)))
        pm.close()
    assert np.array_equal(outs[0], outs[1])


@pytest.mark.parametrize("n", [200_000, 400_000, 1_600_000])
def test_push_sizes_across_the_sort_layouts(gpu_lib, n):
    # the push's sort at 200k rows: 1024-key sub-tiles, digit rows scanned by
    # four warps; 400k: 2048-key sub-tiles, four warps; 1.6M: more than one
    # sub-tile per block (at most 152 SMs x 4 blocks resident); a hot key
    K, D, W = 200_000, 4, 2
    rng = np.random.default_rng(11)
    init = dyadic_init(K, D, 5)
    keys = rng.integers(0, K, size=n)
    keys[rng.random(n) < 0.05] = 777
    d = (rng.integers(-64, 65, size=(n, D)) * 2.0 ** -12).astype(np.float32)
    pm, ref = make_pair(gpu_lib, K, D, W, init)
    for api in (pm, ref):
        api.intent(0, np.arange(0, K, 3), 0, 2)
        api.push(0, keys, d)
    compare_full_state(pm, ref, K, W)
    pm.close()


def test_host_and_device_arguments_agree(gpu_lib):
    K, D, W = 3000, 32, 2
    init = dyadic_init(K, D, 9)
    rng = np.random.default_rng(9)
    keys = rng.integers(0, K, size=4000)
    d = (rng.integers(-64, 65, size=(4000, D)) * 2.0 ** -10).astype(np.float32)
    results = []
    for mode in ("device", "numpy", "pinned"):
        pm = gpu_lib.ParameterManager(K, D, W, init_values=init if mode == "numpy" else torch.from_numpy(init).cuda())
        if mode == "device":
            kk, dd = dev(keys), torch.from_numpy(d).cuda()
        elif mode == "numpy":
            kk, dd = keys, d
        else:
            kk = torch.from_numpy(keys.astype(np.int32)).pin_memory()
            dd = torch.from_numpy(d).pin_memory()
        pm.intent(0, kk, 0, 2)
        pm.push(0, kk, dd)
        pm.push(1, kk, dd)
        out = pm.pull(0, kk)
        pm.wait()
        results.append((np.asarray(out.cpu() if hasattr(out, "cpu") else out), pm.read_main(np.arange(K))))
        pm.close()
    for r in results[1:]:
        assert np.array_equal(r[0], results[0][0]) and np.array_equal(r[1], results[0][1])


def test_pinned_inputs_copied_ahead_of_the_kernels(gpu_lib):
    # pinned host inputs are copied on a stream of their own that runs ahead of the kernels: a long
    # sequence enqueued without waits must give exactly the state of the same calls with device arrays
    K, D, W = 20000, 16, 4
    init = dyadic_init(K, D, 12)
    rng = np.random.default_rng(12)
    calls = []
    for c in range(30):
        for w in range(W):
            k = rng.integers(0, K, size=3000)
            calls.append((w, c, k, (rng.integers(-64, 65, size=(3000, D)) * 2.0 ** -10).astype(np.float32)))
    states = []
    for pinned in (False, True):
        pm = gpu_lib.ParameterManager(K, D, W, init_values=torch.from_numpy(init).cuda())
        conv = ((lambda a: torch.from_numpy(np.ascontiguousarray(a)).pin_memory()) if pinned
                else (lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()))
        args = [(w, c, conv(k.astype(np.int32)), conv(d)) for w, c, k, d in calls]   # kept alive until wait
        outs = []
        for w, c, kk, dd in args:
            pm.intent(w, kk, c + 1, c + 2)
            outs.append(pm.pull(w, kk))
            pm.push(w, kk, dd)
            pm.advance_clock(w)
            if w == W - 1:
                pm.sync()
        pm.wait()
        states.append(([o.cpu().numpy() for o in outs], pm.read_main(np.arange(K))))
        pm.close()
    assert all(np.array_equal(a, b) for a, b in zip(states[0][0], states[1][0]))
    assert np.array_equal(states[0][1], states[1][1])


def test_errors_and_degenerate_inputs(gpu_lib):
    A = gpu_lib
    K, D, W = 50, 8, 2
    init = dyadic_init(K, D, 1)
    pm, ref = make_pair(A, K, D, W, init, capacity=10)
    # argument errors are synchronous and change nothing
    with pytest.raises(A.AdaPMError) as e:
        pm.advance_clock(2)
    assert e.value.status == A.EINVAL
    with pytest.raises(A.AdaPMError):
        pm.pull(5, dev([1]))
    assert pm.clock(0) == 0
    # empty calls
    pm.intent(0, dev([]), 0, 3)
    pm.push(0, dev([]), torch.zeros((0, D), device="cuda"))
    assert pm.pull(0, dev([])).shape == (0, D)
    pm.wait()
    # key out of range: pull row zero, push skips it, sticky ERANGE at wait
    out = pm.pull(0, dev([3, K + 5]))
    with pytest.raises(A.AdaPMError) as e:
        pm.wait()
    assert e.value.status == A.ERANGE
    assert np.array_equal(out.cpu().numpy()[0], init[3]) and not out.cpu().numpy()[1].any()
    pm.push(1, dev([4, K]), torch.ones((2, D), device="cuda"))
    with pytest.raises(A.AdaPMError):
        pm.wait()
    ref.push(1, [4], np.ones((1, D), np.float32))
    pm.wait()   # error was cleared by the previous wait
    assert np.array_equal(pm.read_main(np.arange(K)), ref.main)
    # replica capacity 10: an intent for 12 keys exhausts it -> ENOMEM, reads fall back to main
    pm.intent(1, dev(np.arange(12)), 0, 2)
    with pytest.raises(A.AdaPMError) as e:
        pm.wait()
    assert e.value.status == A.ENOMEM
    assert len(pm.replica_keys(1)) == 0
    assert np.array_equal(pm.pull(1, dev(np.arange(12))).cpu().numpy(), ref.main[:12])
    pm.close()


@pytest.mark.parametrize("K,W", [(1, 1), (7, 32)])
def test_tiny_key_spaces_and_max_workers(gpu_lib, K, W):
    D = 4
    init = dyadic_init(K, D, K)
    pm, ref = make_pair(gpu_lib, K, D, W, init)
    ops = random_sequence(K * 101 + W, K, D, W, 200, max_batch=9)
    for op in ops:
        got = apply_gpu(pm, op)
        want = apply_ref(ref, op)
        if op["op"] == "pull":
            assert np.array_equal(got, want)
    compare_full_state(pm, ref, K, W)
    pm.close()
