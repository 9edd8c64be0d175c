"""Training a small model through the library with real gradients.

Four workers, each with its own slice of a synthetic classification task
(heterogeneous data: every worker sees three of the eight classes), train a
two-layer MLP with Algorithm 1: at each local step every worker's gradient
comes from an autograd backward pass evaluated at that worker's model
(dsm_replica_ptr, Eq. (base-sgd)) and is written into the library's gradient
buffer (dsm_grad_ptr).  The oracle, fed the same gradients, must agree bit for
bit, and the global model's loss over all classes must fall.
"""

import numpy as np
import pytest

import workloads as W
from gpu_common import compare_state

torch = pytest.importorskip("torch")
pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")]

from oracle import dsm_oracle as O  # noqa: E402
from paper_2411_17866_gb300 import dsm  # noqa: E402

IN, HID, OUT, N, TAU, BATCH = 32, 64, 8, 4, 4, 64
TENSORS = (W.Tensor("fc1.w", IN * HID, W.KIND_WEIGHT, 0.0), W.Tensor("fc1.b", HID, W.KIND_BIAS, 0.0, wd=0),
           W.Tensor("fc2.w", HID * OUT, W.KIND_WEIGHT, 0.0), W.Tensor("fc2.b", OUT, W.KIND_BIAS, 0.0, wd=0))
OFFS = np.cumsum([0] + [t.numel for t in TENSORS])
WORKER_CLASSES = [[0, 1, 2], [2, 3, 4], [4, 5, 6], [6, 7, 0]]


def _params(flat):
    """The model's tensors as views of a flat parameter vector (torch, any device)."""
    return [flat[OFFS[0]:OFFS[1]].view(IN, HID), flat[OFFS[1]:OFFS[2]],
            flat[OFFS[2]:OFFS[3]].view(HID, OUT), flat[OFFS[3]:OFFS[4]]]


def _loss(p, X, y):
    h = torch.relu(X @ p[0] + p[1])
    return torch.nn.functional.cross_entropy(h @ p[2] + p[3], y)


def _batch(centers, classes, gen):
    y = torch.tensor(classes)[torch.randint(len(classes), (BATCH,), generator=gen)]
    return centers[y] + 0.7 * torch.randn(BATCH, IN, generator=gen), y


@pytest.mark.parametrize("fused", [False, True], ids=["unfused", "fused"])
def test_training_with_autograd_gradients(fused):
    torch.backends.cuda.matmul.allow_tf32 = False
    hp = W.HParams(lr=1e-2, wd=0.0, g_eta=1.0, g_b1=0.95, g_b2=0.98, g_wd=0.0,
                   flags=W.FLAG_FUSED_ROUND if fused else 0)
    run = dsm.DistributedSignMomentum(TENSORS, N, TAU, hp)
    ora = O.OracleRun(TENSORS, N, TAU, hp)
    g = torch.Generator().manual_seed(0)
    centers = torch.randn(OUT, IN, generator=g)
    X_eval, y_eval = _batch(centers, list(range(OUT)), torch.Generator().manual_seed(99))
    X_eval, y_eval = X_eval.cuda(), y_eval.cuda()
    gens = [torch.Generator().manual_seed(10 + i) for i in range(N)]

    def eval_loss():
        return float(_loss(_params(run.read(dsm.BUF_X).cuda()), X_eval, y_eval))

    loss0 = eval_loss()
    for t in range(40):
        for k in range(TAU):
            grads = []
            for i in range(N):
                # the worker's current model (x itself while a fused round's reset is pending)
                p = [q.detach().requires_grad_() for q in _params(run.replica_view(i))]
                X, y = _batch(centers, WORKER_CLASSES[i], gens[i])
                gr = torch.autograd.grad(_loss(p, X.cuda(), y.cuda()), p)
                flat = torch.cat([q.reshape(-1) for q in gr])
                run.grad_view(i).copy_(flat)
                grads.append(flat.cpu().numpy())
            run.local_step()
            ora.local_step(grads)
        run.global_step()
        ora.global_step()
        if t == 0:
            compare_state(run, ora)
    torch.cuda.synchronize()
    compare_state(run, ora)
    loss1 = eval_loss()
    assert loss1 < 0.6 * loss0, (loss0, loss1)
    run.close()


def test_replica_view_follows_the_lazy_reset():
    """In the fused round the first local step's replica is x itself; after a local step it is the
    worker's own buffer, holding that worker's new model."""
    hp = W.HParams(flags=W.FLAG_FUSED_ROUND)
    run = dsm.DistributedSignMomentum(TENSORS, 2, 2, hp)
    ora = O.OracleRun(TENSORS, 2, 2, hp)
    run.synthetic_round()
    ora.run_round()
    x = run.read(dsm.BUF_X).cuda()
    for i in range(2):
        assert torch.equal(run.replica_view(i), x)
        assert run.replica_view(i).data_ptr() == run.replica_view(1 - i).data_ptr()   # both alias x
    run.fill_synthetic_grads(2)
    run.local_step()
    ora.local_step()
    for i in range(2):
        assert np.array_equal(run.replica_view(i).cpu().numpy().view(np.uint32), ora.X[i].view(np.uint32))
    assert run.replica_view(0).data_ptr() != run.replica_view(1).data_ptr()
    with pytest.raises(dsm.DsmError) as e:
        dsm.dsm_replica_ptr(run.h, 2)
    assert e.value.code == dsm.DSM_ERANGE
    run.close()


def test_training_a_module_built_from_its_parameters():
    """DistributedSignMomentum.from_tensors over a torch module's parameters (its current values are x0),
    unflatten for the per-worker parameter views: 20 rounds, bit-exact against the oracle started from
    the same x0, and the loss falls."""
    torch.backends.cuda.matmul.allow_tf32 = False
    torch.manual_seed(3)
    model = torch.nn.Sequential(torch.nn.Linear(IN, HID), torch.nn.ReLU(), torch.nn.Linear(HID, OUT))
    params = list(model.parameters())
    hp = W.HParams(lr=1e-2, wd=0.0, g_eta=1.0, g_b1=0.95, g_b2=0.98, g_wd=0.0, flags=W.FLAG_FUSED_ROUND)
    run = dsm.DistributedSignMomentum.from_tensors(params, N, TAU, hp)
    assert run.shapes == [tuple(p.shape) for p in params]
    x0 = torch.cat([p.detach().reshape(-1) for p in params]).numpy()
    tensors = tuple(W.Tensor(f"p{i}", p.numel(), W.KIND_WEIGHT if p.dim() > 1 else W.KIND_BIAS, 0.0)
                    for i, p in enumerate(params))
    ora = O.OracleRun(tensors, N, TAU, hp, x0=x0)

    def forward(p, X):
        return torch.nn.functional.linear(torch.relu(torch.nn.functional.linear(X, p[0], p[1])), p[2], p[3])

    centers = torch.randn(OUT, IN, generator=torch.Generator().manual_seed(0))
    X_eval, y_eval = _batch(centers, list(range(OUT)), torch.Generator().manual_seed(99))
    X_eval, y_eval = X_eval.cuda(), y_eval.cuda()
    gens = [torch.Generator().manual_seed(40 + i) for i in range(N)]

    def eval_loss():
        return float(torch.nn.functional.cross_entropy(forward(run.unflatten(run.read(dsm.BUF_X).cuda()), X_eval),
                                                       y_eval))

    loss0 = eval_loss()
    for t in range(20):
        for k in range(TAU):
            grads = []
            for i in range(N):
                p = [q.detach().requires_grad_() for q in run.unflatten(run.replica_view(i))]
                X, y = _batch(centers, WORKER_CLASSES[i], gens[i])
                gr = torch.autograd.grad(torch.nn.functional.cross_entropy(forward(p, X.cuda()), y.cuda()), p)
                flat = torch.cat([q.reshape(-1) for q in gr])
                run.grad_view(i).copy_(flat)
                grads.append(flat.cpu().numpy())
            run.local_step()
            ora.local_step(grads)
        run.global_step()
        ora.global_step()
    torch.cuda.synchronize()
    compare_state(run, ora)
    assert eval_loss() < 0.8 * loss0
    run.close()
